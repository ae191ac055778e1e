// RIS sparse attention, bf16 inputs, TMA-gather design (paper, Methods, "Hybrid Anchor and
// Pre-Fusion Unified Softmax (PFUS)": one softmax over each row's whole sampled key set).
//
// Same arithmetic as k_attn_bf16 (one warp per (row i, KV head g, set s), 16 keys per group,
// S^T = K~ Q~^T and O^T += V^T P^T on m16n8k16 tensor-core products, fp32 online softmax,
// hi + lo splits for the precision bar), but the sampled K/V rows no longer pass through
// the load/store unit. One lane per warp issues TMA `tile::gather4` copies (four arbitrary
// rows per instruction, 128-byte swizzled) of the next groups' rows of K~ hi, K~ lo and V
// into a per-warp ring of shared-memory stages, completing on an mbarrier; the warp reads
// the operand fragments back with ldmatrix, conflict-free thanks to the swizzle. The copy
// engine fetches whole 128-byte row halves from L2, so the L1 data pipe only carries the
// ldmatrix traffic (4 wavefronts per 512 bytes) instead of the scattered global loads.
//
// Every mbarrier wait is bounded (about 2^31 cycles); a wait that gives up sets bit 0 of
// g_ris_device_error, waits (bounded) for the copies still in flight and returns, and the host
// reads the flag with ris_device_status.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>

#include <cstdint>
#include <mutex>

#include "attn_common.cuh"

namespace ris {

__device__ unsigned int g_ris_device_error;

namespace {

constexpr int kTmaWarps = 4;   // tasks per CTA
constexpr int kStages = 2;     // groups in flight per warp
constexpr int kHalf = 16 * 128;  // one 64-column half of a 16-row array (bytes)

__device__ __forceinline__ uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait for the phase with the given parity; false if it did not complete in time.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity)
{
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity)) {
        if (clock64() - t0 > (1LL << 31)) return false;
    }
    return true;
}

__device__ __forceinline__ void tma_gather4(uint32_t dst, const CUtensorMap *map, int col, int r0, int r1, int r2,
                                            int r3, uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cta.global.tile::gather4.mbarrier::complete_tx::bytes "
        "[%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(col), "r"(r0), "r"(r1), "r"(r2), "r"(r3), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void ldsm4(uint32_t addr, uint32_t &a0, uint32_t &a1, uint32_t &a2, uint32_t &a3)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(a0), "=r"(a1), "=r"(a2), "=r"(a3)
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm4_t(uint32_t addr, uint32_t &a0, uint32_t &a1, uint32_t &a2, uint32_t &a3)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(a0), "=r"(a1), "=r"(a2), "=r"(a3)
                 : "r"(addr));
}

__device__ __forceinline__ void mma16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1)
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

// Byte offset of 16-byte chunk c of row r in a 16-row x 128-byte half written by TMA with
// the 128-byte swizzle (chunk index xor row mod 8; the half starts on a 1 KB boundary).
__device__ __forceinline__ uint32_t swz(int r, int c) { return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4)); }

template <typename TOut>
__device__ __forceinline__ void st_out(TOut *p, float x);
template <>
__device__ __forceinline__ void st_out<float>(float *p, float x) { *p = x; }
template <>
__device__ __forceinline__ void st_out<__nv_bfloat16>(__nv_bfloat16 *p, float x) { *p = __float2bfloat16_rn(x); }

// D: head dim (64 or 128). SPLIT: fp32 queries split hi + lo and keys given as hi + lo maps.
template <int D, bool SPLIT, typename TIdx, bool DENSE, typename TOut>
__global__ void __launch_bounds__(kTmaWarps * 32, 1)
    k_attn_tma(const AttnArgs a, const __grid_constant__ CUtensorMap tk, const __grid_constant__ CUtensorMap tkl,
               const __grid_constant__ CUtensorMap tv)
{
    constexpr int HALVES = D / 64;
    constexpr int KSTEPS = D / 16;
    constexpr int MT = D / 16;
    constexpr int ARR = HALVES * kHalf;           // one 16-row array
    constexpr int NARR = SPLIT ? 3 : 2;           // K hi, (K lo), V
    constexpr int STAGE = NARR * ARR;
    constexpr uint32_t STAGE_TX = (uint32_t)STAGE;  // bytes each stage's copies deliver

    extern __shared__ unsigned char smem_raw[];
    __shared__ __align__(8) uint64_t bars[kTmaWarps][kStages];
    unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                            ~uintptr_t(1023));
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t tid = (int64_t)blockIdx.x * kTmaWarps + warp;
    if (tid >= a.n_tasks) return;
    // once any warp has given up on a copy, the rest of the grid leaves at once
    if (*reinterpret_cast<volatile unsigned int *>(&g_ris_device_error) != 0u) return;
    const uint32_t wbase = smem_u32(smem + (size_t)warp * kStages * STAGE);
    const int p = lane >> 2, q = lane & 3;
    const Task t = decode_task(a, tid);
    int64_t beg, n;
    key_range<DENSE>(a, t, beg, n);
    const TIdx *cols = DENSE ? nullptr : reinterpret_cast<const TIdx *>(a.col) + beg;
    const int64_t ngroups = (n + 15) / 16;

    if (lane == 0) {
#pragma unroll
        for (int st = 0; st < kStages; ++st) mbar_init(smem_u32(&bars[warp][st]), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    __syncwarp();

    // ---- key indices, prefetched 64 keys ahead (lane holds positions 64c + lane, 64c + 32 + lane)
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
    int64_t cur_base = 0;  // first position held in cur

    // Issue the copies of group gi into stage st (all lanes gather the 16 row coordinates,
    // lane 0 issues). Group gi lies in cur (gi < cur_base/16 + 4) or nxt.
    auto issue = [&](int64_t gi, int st) {
        const int64_t pos0 = 16 * gi - cur_base;  // 0..127
        const int w = (int)(pos0 >> 5);           // 0..3 over (cur[0], cur[1], nxt[0], nxt[1])
        const int src = w == 0 ? cur[0] : w == 1 ? cur[1] : w == 2 ? nxt[0] : nxt[1];
        const int my = __shfl_sync(0xFFFFFFFFu, src, (int)(pos0 & 31) + (lane & 15));
        const int crd = my * a.Hkv + t.g;  // tensor-map row of (token, KV head)
        int rc[16];
#pragma unroll
        for (int r = 0; r < 16; ++r) rc[r] = __shfl_sync(0xFFFFFFFFu, crd, r);
        if (lane == 0) {
            const uint32_t bar = smem_u32(&bars[warp][st]);
            const uint32_t dst = wbase + (uint32_t)st * STAGE;
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            mbar_arrive_expect_tx(bar, STAGE_TX);
#pragma unroll
            for (int arr = 0; arr < NARR; ++arr) {
                const CUtensorMap *map = arr == 0 ? &tk : (SPLIT && arr == 1) ? &tkl : &tv;
#pragma unroll
                for (int h = 0; h < HALVES; ++h)
#pragma unroll
                    for (int g4 = 0; g4 < 4; ++g4)
                        tma_gather4(dst + arr * ARR + h * kHalf + g4 * 512, map, 64 * h, rc[4 * g4], rc[4 * g4 + 1],
                                    rc[4 * g4 + 2], rc[4 * g4 + 3], bar);
            }
        }
    };

    // ---- query fragments (natural head-dim order), head p of this KV group
    uint32_t qh[KSTEPS][2], ql[KSTEPS][2];
    {
        const bool hv = p < a.G;
        const int64_t qrow = (t.i * a.Hq + (int64_t)t.g * a.G + (hv ? p : 0)) * D;
#pragma unroll
        for (int ks = 0; ks < KSTEPS; ++ks) {
#pragma unroll
            for (int hw = 0; hw < 2; ++hw) {
                const int d0 = 16 * ks + 8 * hw + 2 * q;
                if (SPLIT) {
                    const float2 x = hv ? *reinterpret_cast<const float2 *>(reinterpret_cast<const float *>(a.q) + qrow + d0)
                                        : make_float2(0.f, 0.f);
                    const float h0 = __bfloat162float(__float2bfloat16_rn(x.x));
                    const float h1 = __bfloat162float(__float2bfloat16_rn(x.y));
                    qh[ks][hw] = pack_bf16(h0, h1);
                    ql[ks][hw] = pack_bf16(x.x - h0, x.y - h1);
                } else {
                    qh[ks][hw] = hv ? *reinterpret_cast<const uint32_t *>(reinterpret_cast<const __nv_bfloat16 *>(a.q) +
                                                                          qrow + d0)
                                    : 0u;
                    ql[ks][hw] = 0u;
                }
            }
        }
    }

    // prologue: fill the ring
#pragma unroll
    for (int st = 0; st < kStages; ++st)
        if (st < ngroups) issue(st, st);

    float o[MT][4];
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
    const float sc = a.scale_log2;
    bool ok = true;

    // ldmatrix lane roles: matrix m = lane / 8 of an x4 load, row lane % 8 of it
    const int lm = lane >> 3, lr = lane & 7;

    for (int64_t g = 0; g < ngroups; ++g) {
        const int st = (int)(g % kStages);
        const uint32_t parity = (uint32_t)((g / kStages) & 1);
        const bool got = mbar_wait(smem_u32(&bars[warp][st]), parity);
        if (!__all_sync(0xFFFFFFFFu, got)) {
            ok = false;
            break;
        }
        const uint32_t sb = wbase + (uint32_t)st * STAGE;
        const int64_t base = 16 * g;
        const bool val0 = base + p < n, val1 = base + p + 8 < n;

        // ---- S^T = K~ Q~^T from the stage (rows = keys): matrices (rows 0-7 | 8-15) x (k 0-7 | 8-15)
        float sa[2][4], sbb[2][4], sl[2][4];
#pragma unroll
        for (int c = 0; c < 2; ++c)
#pragma unroll
            for (int e = 0; e < 4; ++e) sa[c][e] = sbb[c][e] = sl[c][e] = 0.f;
#pragma unroll
        for (int ks = 0; ks < KSTEPS; ++ks) {
            const int h = ks >> 2, c0 = 2 * (ks & 3);
            const int r = ((lm & 1) << 3) + lr, c = c0 + (lm >> 1);
            const uint32_t off = (uint32_t)(h * kHalf) + swz(r, c);
            uint32_t a0, a1, a2, a3;
            ldsm4(sb + off, a0, a1, a2, a3);
            mma16816(sa[ks & 1], a0, a1, a2, a3, qh[ks][0], qh[ks][1]);
            if (SPLIT) {
                mma16816(sbb[ks & 1], a0, a1, a2, a3, ql[ks][0], ql[ks][1]);
                uint32_t b0, b1, b2, b3;
                ldsm4(sb + ARR + off, b0, b1, b2, b3);
                mma16816(sl[ks & 1], b0, b1, b2, b3, qh[ks][0], qh[ks][1]);
            }
        }
        float s[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) s[e] = ((sa[0][e] + sa[1][e]) + (sbb[0][e] + sbb[1][e])) + (sl[0][e] + sl[1][e]);

        // ---- online softmax; lane holds keys p, p+8 x heads 2q, 2q+1
        const float s0 = val0 ? s[0] * sc : -INFINITY, s1 = val0 ? s[1] * sc : -INFINITY;
        const float s2 = val1 ? s[2] * sc : -INFINITY, s3 = val1 ? s[3] * sc : -INFINITY;
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
        const float h0 = __bfloat162float(__float2bfloat16_rn(p0)), h1 = __bfloat162float(__float2bfloat16_rn(p1));
        const float h2 = __bfloat162float(__float2bfloat16_rn(p2)), h3 = __bfloat162float(__float2bfloat16_rn(p3));
        const uint32_t pb0 = transpose8x8(pack_bf16(h0, h1));
        const uint32_t pb1 = transpose8x8(pack_bf16(h2, h3));
        const uint32_t pl0 = transpose8x8(pack_bf16(p0 - h0, p1 - h1));
        const uint32_t pl1 = transpose8x8(pack_bf16(p2 - h2, p3 - h3));

        // ---- O^T += V^T P^T; V^T fragments by transposing loads of key rows
        const uint32_t vsb = sb + (uint32_t)((NARR - 1) * ARR);
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
            const int h = mt >> 2, c = 2 * (mt & 3) + (lm & 1), r = ((lm >> 1) << 3) + lr;
            uint32_t a0, a1, a2, a3;
            ldsm4_t(vsb + (uint32_t)(h * kHalf) + swz(r, c), a0, a1, a2, a3);
            mma16816(o[mt], a0, a1, a2, a3, pb0, pb1);
            mma16816(o[mt], a0, a1, a2, a3, pl0, pl1);
        }

        // ---- refill this stage with group g + kStages; the chunk window slides every 4 groups
        __syncwarp();
        const int64_t gn = g + kStages;
        if (gn < ngroups) {
            if (16 * gn >= cur_base + 64) {  // the group lives in the next chunk: slide the window
                cur[0] = nxt[0];
                cur[1] = nxt[1];
                cur_base += 64;
                load_chunk(cur_base + 64, nxt);
            }
            issue(gn, st);
        }
    }

    if (!ok) {
        // a copy never completed: flag it, give in-flight copies a bounded chance to land, return
        if (lane == 0) atomicOr(&g_ris_device_error, 1u);
        for (int st = 0; st < kStages; ++st) mbar_wait(smem_u32(&bars[warp][st]), 0);
        return;
    }

    // ---- epilogue: full row sums, normalise, store (head dim in natural order)
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
        l0 += __shfl_xor_sync(0xFFFFFFFFu, l0, off);
        l1 += __shfl_xor_sync(0xFFFFFFFFu, l1, off);
    }
    const float inv0 = 1.f / l0, inv1 = 1.f / l1;
    const int e0 = 2 * q, e1 = 2 * q + 1;
    TOut *out = reinterpret_cast<TOut *>(a.out) + (((int64_t)t.s * a.N + t.i) * a.Hq + (int64_t)t.g * a.G) * D;
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
        const int d = 16 * mt + p;
        if (e0 < a.G) {
            st_out<TOut>(out + (int64_t)e0 * D + d, o[mt][0] * inv0);
            st_out<TOut>(out + (int64_t)e0 * D + d + 8, o[mt][2] * inv0);
        }
        if (e1 < a.G) {
            st_out<TOut>(out + (int64_t)e1 * D + d, o[mt][1] * inv1);
            st_out<TOut>(out + (int64_t)e1 * D + d + 8, o[mt][3] * inv1);
        }
    }
    if (a.lse != nullptr && p == 0) {
        float *lse = a.lse + ((int64_t)t.s * a.Hq + (int64_t)t.g * a.G) * a.N + t.i;
        if (e0 < a.G) lse[(int64_t)e0 * a.N] = (m0 + __log2f(l0)) * kLn2;
        if (e1 < a.G) lse[(int64_t)e1 * a.N] = (m1 + __log2f(l1)) * kLn2;
    }
}

// ---------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static std::once_flag once;
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// Rows of (token, KV head) of a [N][Hkv][D] bf16 tensor; box = one row x 64 columns.
bool make_map(CUtensorMap *m, const void *base, int64_t rows, int D)
{
    auto fn = encode_fn();
    if (fn == nullptr) return false;
    cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)D * 2};
    cuuint32_t box[2] = {64, 1};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D, bool SPLIT, typename TIdx, bool DENSE, typename TOut>
cudaError_t launch_one(const AttnArgs &a, const CUtensorMap &tk, const CUtensorMap &tkl, const CUtensorMap &tv,
                       cudaStream_t s)
{
    constexpr int NARR = SPLIT ? 3 : 2;
    constexpr size_t smem = (size_t)kTmaWarps * kStages * NARR * (D / 64) * kHalf + 1024;
    auto kern = k_attn_tma<D, SPLIT, TIdx, DENSE, TOut>;
    static bool attr_set = false;  // per instantiation
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const unsigned grid = (unsigned)((a.n_tasks + kTmaWarps - 1) / kTmaWarps);
    kern<<<grid, kTmaWarps * 32, smem, s>>>(a, tk, tkl, tv);
    note_launch();
    return cudaGetLastError();
}

template <int D, bool SPLIT, typename TOut>
cudaError_t launch_d(const AttnArgs &a, const CUtensorMap &tk, const CUtensorMap &tkl, const CUtensorMap &tv,
                     int col_bytes, bool dense, cudaStream_t s)
{
    if (dense) return launch_one<D, SPLIT, uint32_t, true, TOut>(a, tk, tkl, tv, s);
    if (col_bytes == 2) return launch_one<D, SPLIT, uint16_t, false, TOut>(a, tk, tkl, tv, s);
    return launch_one<D, SPLIT, uint32_t, false, TOut>(a, tk, tkl, tv, s);
}

template <bool SPLIT, typename TOut>
cudaError_t launch_s(const AttnArgs &a, int D, const CUtensorMap &tk, const CUtensorMap &tkl, const CUtensorMap &tv,
                     int col_bytes, bool dense, cudaStream_t s)
{
    return D == 64 ? launch_d<64, SPLIT, TOut>(a, tk, tkl, tv, col_bytes, dense, s)
                   : launch_d<128, SPLIT, TOut>(a, tk, tkl, tv, col_bytes, dense, s);
}

}  // namespace

bool tma_gather_available()
{
    return encode_fn() != nullptr;
}

// Read and clear the device error word (bit 0: a bounded mbarrier wait gave up).
cudaError_t read_device_error(unsigned int *out, cudaStream_t s)
{
    cudaError_t e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return e;
    e = cudaMemcpyFromSymbol(out, g_ris_device_error, sizeof(unsigned int));
    if (e != cudaSuccess) return e;
    if (*out != 0u) {
        const unsigned int zero = 0u;
        e = cudaMemcpyToSymbol(g_ris_device_error, &zero, sizeof(unsigned int));
    }
    return e;
}

cudaError_t launch_attention_tma(const AttnArgs &a, int D, int out_dtype, bool split, int col_bytes, bool dense,
                                 cudaStream_t s)
{
    static std::mutex mu;  // the per-instantiation attribute flags
    std::lock_guard<std::mutex> lk(mu);
    alignas(64) CUtensorMap tk, tkl, tv;
    const int64_t rows = a.N * a.Hkv;
    if (!make_map(&tk, a.k, rows, D) || !make_map(&tv, a.v, rows, D)) return cudaErrorInvalidValue;
    if (split) {
        if (!make_map(&tkl, a.k_lo, rows, D)) return cudaErrorInvalidValue;
    } else {
        tkl = tk;
    }
    if (out_dtype == RIS_F32)
        return split ? launch_s<true, float>(a, D, tk, tkl, tv, col_bytes, dense, s)
                     : launch_s<false, float>(a, D, tk, tkl, tv, col_bytes, dense, s);
    return split ? launch_s<true, __nv_bfloat16>(a, D, tk, tkl, tv, col_bytes, dense, s)
                 : launch_s<false, __nv_bfloat16>(a, D, tk, tkl, tv, col_bytes, dense, s);
}

}  // namespace ris
