// RIS sparse attention, bf16 inputs, gather design (paper, Methods, "Hybrid Anchor and
// Pre-Fusion Unified Softmax (PFUS)": one softmax over each row's whole sampled key set).
//
// One warp owns one task (row i, KV head g, output set s) and walks the row's ascending key
// list 16 keys at a time. The G query heads that share KV head g (GQA) ride in the N
// dimension of the tensor-core tile, so every gathered K/V row is fetched once and used by
// all of them:
//
//   S^T[16 keys x 8 heads] = K~[16 keys x D] . Q~^T          (mma m16n8k16, keys in M)
//   online softmax per head in fp32 (exp2 domain, scale log2(e)/sqrt(D) applied in fp32)
//   O^T[D x 8 heads]     += V^T[D x 16 keys] . P^T           (mma m16n8k16, head dim in M)
//
// Gathered rows go straight from L2 into registers, with no shared-memory staging. The head
// dimension is permuted (the same permutation on K~ and Q~, undone when O is stored) so
// that every 16-byte-per-lane load instruction reads whole, fully used 32-byte sectors in
// long runs: for K the four lanes that share a key row read 64 contiguous bytes of it, for
// V the eight lanes that share a row read 128 contiguous bytes. Scattered gathers are
// bounded by the L1 data pipe's wavefronts per instruction, not by L2 bandwidth, so the
// fewer sectors and lines an instruction touches the better. P^T moves from the
// accumulator layout of the first product into the operand layout of the second with
// movmatrix (an 8x8 transpose in registers).
//
// Lane (p = lane/4, q = lane%4). K row: lane q holds elements 32u + 8q + [0, 8), u < D/32;
// k-step t takes elements 32(t/2) + 8q + 4(t%2) + [0, 4). V row: lane p holds elements
// 64u + 8p + [0, 8), u < D/64; word j of that run (d, d+1) feeds m-tile j.
//
// Precision. With activation outlier channels (|v| up to ~30) a max-abs error of 1e-2 needs
// ~12+ significant bits in the scores and in P, more than bf16 (8) or fp16 (11) carry. So:
//   - rotated queries arrive in fp32 and are split into bf16 hi + lo in registers;
//   - rotated keys arrive as a bf16 hi + lo pair (written by the RoPE kernel);
//   - S^T = K_hi Q_hi + K_hi Q_lo + K_lo Q_hi (the lo*lo term is below 2^-16);
//   - P is split into bf16 hi + lo and O^T += V^T P_hi + V^T P_lo.
// V is an exact bf16 input. Unrotated bf16 q/k are exact and take one product each.
#include <cuda_bf16.h>

#include <cstdint>

#include "attn_common.cuh"

namespace ris {
namespace {

__device__ __forceinline__ void mma16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t transpose8x8(uint32_t x)
{
    uint32_t y;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;\n" : "=r"(y) : "r"(x));
    return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t *>(&v);
}

__device__ __forceinline__ uint4 ldg16(const void *p)
{
    return __ldg(reinterpret_cast<const uint4 *>(p));
}

template <typename TOut>
__device__ __forceinline__ void store_run(TOut *dst, const float *x, int n);

template <>
__device__ __forceinline__ void store_run<float>(float *dst, const float *x, int n)
{
    for (int e = 0; e < n; e += 4)
        *reinterpret_cast<float4 *>(dst + e) = make_float4(x[e], x[e + 1], x[e + 2], x[e + 3]);
}

template <>
__device__ __forceinline__ void store_run<__nv_bfloat16>(__nv_bfloat16 *dst, const float *x, int n)
{
    for (int e = 0; e < n; e += 8) {
        uint4 w;
        w.x = pack_bf16(x[e], x[e + 1]);
        w.y = pack_bf16(x[e + 2], x[e + 3]);
        w.z = pack_bf16(x[e + 4], x[e + 5]);
        w.w = pack_bf16(x[e + 6], x[e + 7]);
        *reinterpret_cast<uint4 *>(dst + e) = w;
    }
}

// D: head dim (64 or 128). QSPLIT: q is fp32 (split hi + lo); else q is bf16.
// KSPLIT: keys come as a bf16 hi (a.k) + lo (a.k_lo) pair.
#ifndef RIS_ATTN_MIN_BLOCKS
#define RIS_ATTN_MIN_BLOCKS 1
#endif

template <int D, bool QSPLIT, bool KSPLIT, typename TIdx, bool DENSE, typename TOut>
__global__ void __launch_bounds__(kAttnWarps * 32, RIS_ATTN_MIN_BLOCKS) k_attn_bf16(const AttnArgs a)
{
    constexpr int KSTEPS = D / 16;  // k-steps of the score product
    constexpr int KU = D / 32;      // 16-byte loads per K row per lane (D/2 bytes)
    constexpr int VU = D / 64;      // 16-byte loads per V row per lane (D/8 elements)
    constexpr int MT = D / 16;      // m-tiles of the value product (head dim)

    const int lane = threadIdx.x & 31;
    const int64_t tid = (int64_t)blockIdx.x * kAttnWarps + (threadIdx.x >> 5);
    if (tid >= a.n_tasks) return;
    const int p = lane >> 2, q = lane & 3;
    const Task t = decode_task(a, tid);
    int64_t beg, n;
    key_range<DENSE>(a, t, beg, n);
    const TIdx *cols = DENSE ? nullptr : reinterpret_cast<const TIdx *>(a.col) + beg;

    // ---- query fragments (B operand of the score product), head p of this KV group
    uint32_t qh[KSTEPS][2], ql[KSTEPS][2];
    {
        const bool hv = p < a.G;
        const int64_t qrow = (t.i * a.Hq + (int64_t)t.g * a.G + (hv ? p : 0)) * D;
#pragma unroll
        for (int ks = 0; ks < KSTEPS; ++ks) {
            const int d0 = 32 * (ks >> 1) + 8 * q + 4 * (ks & 1);
            if (QSPLIT) {
                float4 x = hv ? *reinterpret_cast<const float4 *>(reinterpret_cast<const float *>(a.q) + qrow + d0)
                              : make_float4(0.f, 0.f, 0.f, 0.f);
                const float h0 = __bfloat162float(__float2bfloat16_rn(x.x));
                const float h1 = __bfloat162float(__float2bfloat16_rn(x.y));
                const float h2 = __bfloat162float(__float2bfloat16_rn(x.z));
                const float h3 = __bfloat162float(__float2bfloat16_rn(x.w));
                qh[ks][0] = pack_bf16(h0, h1);
                qh[ks][1] = pack_bf16(h2, h3);
                ql[ks][0] = pack_bf16(x.x - h0, x.y - h1);
                ql[ks][1] = pack_bf16(x.z - h2, x.w - h3);
            } else {
                uint2 w = hv ? *reinterpret_cast<const uint2 *>(reinterpret_cast<const __nv_bfloat16 *>(a.q) + qrow + d0)
                             : make_uint2(0u, 0u);
                qh[ks][0] = w.x;
                qh[ks][1] = w.y;
                ql[ks][0] = ql[ks][1] = 0u;
            }
        }
    }

    const size_t row_bytes = (size_t)a.Hkv * D * sizeof(__nv_bfloat16);
    const char *kb = reinterpret_cast<const char *>(a.k) + (size_t)t.g * D * sizeof(__nv_bfloat16) + 16 * q;
    const char *kbl = KSPLIT ? reinterpret_cast<const char *>(a.k_lo) + (size_t)t.g * D * sizeof(__nv_bfloat16) + 16 * q
                             : nullptr;
    const char *vb = reinterpret_cast<const char *>(a.v) + (size_t)t.g * D * sizeof(__nv_bfloat16) + 16 * p;

    float o[MT][4];
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
    const float sc = a.scale_log2;

    // ---- key indices, prefetched 64 keys (4 groups) ahead: lane holds positions
    //      64c + lane and 64c + 32 + lane of chunk c; slots past the row read the row itself
    int cur[2], nxt[2];
    auto load_chunk = [&](int64_t cbase, int (&dst)[2]) {
#pragma unroll
        for (int w = 0; w < 2; ++w) {
            const int64_t pos = cbase + 32 * w + lane;
            dst[w] = pos < n ? key_at<DENSE, TIdx>(cols, pos) : (int)t.i;
        }
    };
    load_chunk(0, cur);
    load_chunk(64, nxt);
    // index of slot r (0..15) of group slot gs (0..3) of a chunk held in (c0, c1)
    auto slot = [&](int c0, int c1, int gs, int r) -> int {
        return __shfl_sync(0xFFFFFFFFu, (gs >> 1) ? c1 : c0, (16 * gs + r) & 31);
    };

    // ---- gathered rows of one group: K rows p and p+8 (D/2 bytes each of hi and lo),
    //      V rows 2q, 2q+1, 2q+8, 2q+9 (D/8 elements each)
    uint4 k0[KU], k1[KU], kl0[KSPLIT ? KU : 1], kl1[KSPLIT ? KU : 1], v0[VU], v1[VU], v2[VU], v3[VU];
    auto issue_k = [&](int c0, int c1, int gs) {
        const int ik0 = slot(c0, c1, gs, p), ik1 = slot(c0, c1, gs, p + 8);
#pragma unroll
        for (int u = 0; u < KU; ++u) {
            k0[u] = ldg16(kb + (size_t)ik0 * row_bytes + 64 * u);
            k1[u] = ldg16(kb + (size_t)ik1 * row_bytes + 64 * u);
            if (KSPLIT) {
                kl0[u % (KSPLIT ? KU : 1)] = ldg16(kbl + (size_t)ik0 * row_bytes + 64 * u);
                kl1[u % (KSPLIT ? KU : 1)] = ldg16(kbl + (size_t)ik1 * row_bytes + 64 * u);
            }
        }
    };
    auto issue_v = [&](int c0, int c1, int gs) {
        const int iv0 = slot(c0, c1, gs, 2 * q), iv1 = slot(c0, c1, gs, 2 * q + 1);
        const int iv2 = slot(c0, c1, gs, 2 * q + 8), iv3 = slot(c0, c1, gs, 2 * q + 9);
#pragma unroll
        for (int u = 0; u < VU; ++u) {
            v0[u] = ldg16(vb + (size_t)iv0 * row_bytes + 128 * u);
            v1[u] = ldg16(vb + (size_t)iv1 * row_bytes + 128 * u);
            v2[u] = ldg16(vb + (size_t)iv2 * row_bytes + 128 * u);
            v3[u] = ldg16(vb + (size_t)iv3 * row_bytes + 128 * u);
        }
    };

    // Phase-shifted pipeline: the next group's K rows are requested as soon as this group's
    // scores are formed, its V rows as soon as this group's values are accumulated.
    issue_k(cur[0], cur[1], 0);
    issue_v(cur[0], cur[1], 0);
    const int64_t ngroups = (n + 15) / 16;
    for (int64_t g = 0; g < ngroups; ++g) {
        const int64_t base = 16 * g;
        const int gs = (int)(g & 3), gs1 = (gs + 1) & 3;
        const bool more = g + 1 < ngroups;
        const int n0 = gs1 == 0 ? nxt[0] : cur[0], n1 = gs1 == 0 ? nxt[1] : cur[1];
        const bool val0 = base + p < n, val1 = base + p + 8 < n;

        // ---- S^T = K~ Q~^T: independent accumulator chains (hi*hi, hi*lo, lo*hi, and even/odd
        //      k-steps) so the tensor-core latencies overlap instead of forming one serial chain
        float sa[2][4], sb[2][4], sl[2][4];
#pragma unroll
        for (int c = 0; c < 2; ++c)
#pragma unroll
            for (int e = 0; e < 4; ++e) sa[c][e] = sb[c][e] = sl[c][e] = 0.f;
#pragma unroll
        for (int ks = 0; ks < KSTEPS; ++ks) {
            const uint4 &x0 = k0[ks >> 1], &x1 = k1[ks >> 1];
            const uint32_t a0 = (ks & 1) ? x0.z : x0.x;
            const uint32_t a1 = (ks & 1) ? x1.z : x1.x;
            const uint32_t a2 = (ks & 1) ? x0.w : x0.y;
            const uint32_t a3 = (ks & 1) ? x1.w : x1.y;
            mma16816(sa[ks & 1], a0, a1, a2, a3, qh[ks][0], qh[ks][1]);
            if (QSPLIT) mma16816(sb[ks & 1], a0, a1, a2, a3, ql[ks][0], ql[ks][1]);
            if (KSPLIT) {
                const uint4 &y0 = kl0[(ks >> 1) % (KSPLIT ? KU : 1)], &y1 = kl1[(ks >> 1) % (KSPLIT ? KU : 1)];
                mma16816(sl[ks & 1], (ks & 1) ? y0.z : y0.x, (ks & 1) ? y1.z : y1.x, (ks & 1) ? y0.w : y0.y,
                         (ks & 1) ? y1.w : y1.y, qh[ks][0], qh[ks][1]);
            }
        }
        float s[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) s[e] = ((sa[0][e] + sa[1][e]) + (sb[0][e] + sb[1][e])) + (sl[0][e] + sl[1][e]);
        if (more) issue_k(n0, n1, gs1);

        // ---- online softmax; lane holds keys p, p+8 x heads 2q, 2q+1
        float s0 = val0 ? s[0] * sc : -INFINITY, s1 = val0 ? s[1] * sc : -INFINITY;
        float s2 = val1 ? s[2] * sc : -INFINITY, s3 = val1 ? s[3] * sc : -INFINITY;
        float mx0 = fmaxf(s0, s2), mx1 = fmaxf(s1, s3);
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
            mx0 = fmaxf(mx0, __shfl_xor_sync(0xFFFFFFFFu, mx0, off));
            mx1 = fmaxf(mx1, __shfl_xor_sync(0xFFFFFFFFu, mx1, off));
        }
        const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
        const float mu0 = (mn0 == -INFINITY) ? 0.f : mn0, mu1 = (mn1 == -INFINITY) ? 0.f : mn1;
        const float al0 = exp2f(m0 - mu0), al1 = exp2f(m1 - mu1);
        m0 = mn0;
        m1 = mn1;
        const float p0 = exp2f(s0 - mu0), p1 = exp2f(s1 - mu1);
        const float p2 = exp2f(s2 - mu0), p3 = exp2f(s3 - mu1);
        l0 = l0 * al0 + (p0 + p2);
        l1 = l1 * al1 + (p1 + p3);
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
            o[mt][0] *= al0;
            o[mt][1] *= al1;
            o[mt][2] *= al0;
            o[mt][3] *= al1;
        }
        // P = P_hi + P_lo in bf16; transposed into the B operand P[head p][keys 2q.., 2q+8..]
        const float h0 = __bfloat162float(__float2bfloat16_rn(p0)), h1 = __bfloat162float(__float2bfloat16_rn(p1));
        const float h2 = __bfloat162float(__float2bfloat16_rn(p2)), h3 = __bfloat162float(__float2bfloat16_rn(p3));
        const uint32_t pb0 = transpose8x8(pack_bf16(h0, h1));
        const uint32_t pb1 = transpose8x8(pack_bf16(h2, h3));
        const uint32_t pl0 = transpose8x8(pack_bf16(p0 - h0, p1 - h1));
        const uint32_t pl1 = transpose8x8(pack_bf16(p2 - h2, p3 - h3));

        // ---- O^T += V^T P^T
        const uint32_t *w0 = reinterpret_cast<const uint32_t *>(v0);
        const uint32_t *w1 = reinterpret_cast<const uint32_t *>(v1);
        const uint32_t *w2 = reinterpret_cast<const uint32_t *>(v2);
        const uint32_t *w3 = reinterpret_cast<const uint32_t *>(v3);
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
            const uint32_t a0 = __byte_perm(w0[mt], w1[mt], 0x5410);
            const uint32_t a1 = __byte_perm(w0[mt], w1[mt], 0x7632);
            const uint32_t a2 = __byte_perm(w2[mt], w3[mt], 0x5410);
            const uint32_t a3 = __byte_perm(w2[mt], w3[mt], 0x7632);
            mma16816(o[mt], a0, a1, a2, a3, pb0, pb1);
            mma16816(o[mt], a0, a1, a2, a3, pl0, pl1);
        }
        if (more) issue_v(n0, n1, gs1);
        if (gs == 3) {  // the next group starts the prefetched chunk; fetch the one after it
            cur[0] = nxt[0];
            cur[1] = nxt[1];
            load_chunk(base + 16 + 64, nxt);
        }
    }

    // ---- epilogue: full row sums, normalise, undo the head-dim permutation
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
        l0 += __shfl_xor_sync(0xFFFFFFFFu, l0, off);
        l1 += __shfl_xor_sync(0xFFFFFFFFu, l1, off);
    }
    const float inv0 = 1.f / l0, inv1 = 1.f / l1;
    const int h0 = 2 * q, h1 = 2 * q + 1;
    TOut *out = reinterpret_cast<TOut *>(a.out) + (((int64_t)t.s * a.N + t.i) * a.Hq + (int64_t)t.g * a.G) * D + 8 * p;
    float run[8];
#pragma unroll
    for (int u = 0; u < VU; ++u) {
        if (h0 < a.G) {
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                run[2 * j] = o[4 * u + j][0] * inv0;
                run[2 * j + 1] = o[4 * u + j][2] * inv0;
            }
            store_run<TOut>(out + (int64_t)h0 * D + 64 * u, run, 8);
        }
        if (h1 < a.G) {
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                run[2 * j] = o[4 * u + j][1] * inv1;
                run[2 * j + 1] = o[4 * u + j][3] * inv1;
            }
            store_run<TOut>(out + (int64_t)h1 * D + 64 * u, run, 8);
        }
    }
    if (a.lse != nullptr && p == 0) {
        float *lse = a.lse + ((int64_t)t.s * a.Hq + (int64_t)t.g * a.G) * a.N + t.i;
        if (h0 < a.G) lse[(int64_t)h0 * a.N] = (m0 + __log2f(l0)) * kLn2;
        if (h1 < a.G) lse[(int64_t)h1 * a.N] = (m1 + __log2f(l1)) * kLn2;
    }
}

template <int D, bool QSPLIT, typename TOut>
cudaError_t launch_d(const AttnArgs &a, int col_bytes, bool dense, cudaStream_t s)
{
    // rotated inputs: fp32 queries and hi + lo keys; as given: bf16 queries and keys
    constexpr bool KSPLIT = QSPLIT;
    const unsigned grid = (unsigned)((a.n_tasks + kAttnWarps - 1) / kAttnWarps);
    const dim3 block(kAttnWarps * 32);
    if (dense)
        k_attn_bf16<D, QSPLIT, KSPLIT, uint32_t, true, TOut><<<grid, block, 0, s>>>(a);
    else if (col_bytes == 2)
        k_attn_bf16<D, QSPLIT, KSPLIT, uint16_t, false, TOut><<<grid, block, 0, s>>>(a);
    else
        k_attn_bf16<D, QSPLIT, KSPLIT, uint32_t, false, TOut><<<grid, block, 0, s>>>(a);
    note_launch();
    return cudaGetLastError();
}

template <bool QSPLIT, typename TOut>
cudaError_t launch_q(const AttnArgs &a, int D, int col_bytes, bool dense, cudaStream_t s)
{
    return D == 64 ? launch_d<64, QSPLIT, TOut>(a, col_bytes, dense, s)
                   : launch_d<128, QSPLIT, TOut>(a, col_bytes, dense, s);
}

}  // namespace

cudaError_t launch_attention_bf16(const AttnArgs &a, int D, int out_dtype, bool q_split,
                                  int col_bytes, bool dense, cudaStream_t s)
{
    if (out_dtype == RIS_F32)
        return q_split ? launch_q<true, float>(a, D, col_bytes, dense, s)
                       : launch_q<false, float>(a, D, col_bytes, dense, s);
    return q_split ? launch_q<true, __nv_bfloat16>(a, D, col_bytes, dense, s)
                   : launch_q<false, __nv_bfloat16>(a, D, col_bytes, dense, s);
}

}  // namespace ris
