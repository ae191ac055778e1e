// RIS sparse attention, bf16 inputs, gather design (paper, Methods, "Hybrid Anchor and
// Pre-Fusion Unified Softmax (PFUS)": one softmax over each row's whole sampled key set).
//
// One warp owns one task (row i, KV head g, output set s) and walks the row's ascending key
// list 16 keys at a time (per-seed outputs: one warp walks the sets of (i, g) one after the
// other, see SEEDS below). The G query heads that share KV head g (GQA) ride in the N
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
//   - rotated queries arrive in fp32 and are split into bf16 hi + lo in registers, or as a
//     bf16 hi + lo pair;
//   - rotated keys arrive as a bf16 hi + lo pair (written by the RoPE kernel);
//   - S^T = K_hi Q_hi + K_hi Q_lo + K_lo Q_hi (the lo*lo term is below 2^-16);
//   - or, at head dim 128 with rotated bf16 inputs, fp16 hi parts with e4m3 lo parts (E8
//     below);
//   - P is split into bf16 hi + lo and O^T += V^T P_hi + V^T P_lo against the exact bf16 V;
//   - E8: P as one fp16 against the values' fp16 copy (exact after a power-of-two scale), the
//     row sums adding P as rounded, as the tile kernel does.
// Unrotated bf16 q/k are exact and take one product each.
//
// Residency. The gather is bound by the gathered rows it keeps in flight, hence by how many
// warps fit on an SM. In the fp8 form each thread parks its query fragments
// and output accumulators in its own lane of tensor memory (128 columns per CTA) and reloads
// them around the products that use them: 168 registers, three CTAs per SM instead of two.
// The loads that feed one product share one wait, and a store of the accumulators is waited
// for only before their next load.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_fp8.h>

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

__device__ __forceinline__ void mma16816_f16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                             uint32_t a3, uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// e4m3 x e4m3 -> fp32, m16n8k32: four e4m3 values per 32-bit register, lowest byte first. A:
// a0 / a2 row lane/4 at columns 4(lane%4) + [0, 4) / 16 + 4(lane%4) + [0, 4), a1 / a3 the same
// of row lane/4 + 8; B: b0 / b1 rows 4(lane%4) + [0, 4) / 16 + 4(lane%4) + [0, 4) of column
// lane/4; C as for m16n8k16.
__device__ __forceinline__ void mma16832_e4m3(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                              uint32_t a3, uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.f32.e4m3.e4m3.f32 "
        "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// two e4m3 values (lowest byte first) times s, as an fp16 pair
__device__ __forceinline__ uint32_t e4m3x2_to_f16x2(uint32_t two, float s)
{
    const __half2_raw hr = __nv_cvt_fp8x2_to_halfraw2((__nv_fp8x2_storage_t)(two & 0xFFFFu), __NV_E4M3);
    const float2 f = __half22float2(*reinterpret_cast<const __half2 *>(&hr));
    const __half2 h = __floats2half2_rn(f.x * s, f.y * s);
    return *reinterpret_cast<const uint32_t *>(&h);
}

// Per-thread private storage in tensor memory: thread l of warp w owns TMEM lane 32 (w % 4) + l,
// and a 32x32b access moves N consecutive 32-bit columns of that lane (warp-collective).
template <int N>
__device__ __forceinline__ void tm_st(uint32_t taddr, const uint32_t *v);
template <>
__device__ __forceinline__ void tm_st<8>(uint32_t taddr, const uint32_t *v)
{
    asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr), "r"(v[0]),
                 "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7])
                 : "memory");
}
template <>
__device__ __forceinline__ void tm_st<16>(uint32_t taddr, const uint32_t *v)
{
    asm volatile("tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};"
                 ::"r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
                 "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
                 : "memory");
}
__device__ __forceinline__ void tm_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
// loads that share one wait: issue them with tm_issue<N>, then tm_wait_ld, then tm_pin<N> on
// each destination (an empty asm that redefines the registers, so that no use of them is
// scheduled before the wait)
template <int N>
__device__ __forceinline__ void tm_issue(uint32_t taddr, uint32_t *v);
template <>
__device__ __forceinline__ void tm_issue<8>(uint32_t taddr, uint32_t *v)
{
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7])
                 : "r"(taddr)
                 : "memory");
}
template <>
__device__ __forceinline__ void tm_issue<16>(uint32_t taddr, uint32_t *v)
{
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
                 : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
                   "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
                 : "r"(taddr)
                 : "memory");
}
__device__ __forceinline__ void tm_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void tm_pin(uint32_t *v)
{
#pragma unroll
    for (int i = 0; i < N; i += 8)
        asm volatile("" : "+r"(v[i]), "+r"(v[i + 1]), "+r"(v[i + 2]), "+r"(v[i + 3]), "+r"(v[i + 4]), "+r"(v[i + 5]),
                     "+r"(v[i + 6]), "+r"(v[i + 7]));
}
// the output accumulators o[8][4] <-> 32 columns; a store is not waited for here, the next
// load of the same columns (tm_ld_o) waits for it
__device__ __forceinline__ void tm_st_o(uint32_t taddr, float (&o)[8][4])
{
    uint32_t w[16];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
#pragma unroll
        for (int i = 0; i < 16; ++i) w[i] = __float_as_uint(o[4 * h + i / 4][i % 4]);
        tm_st<16>(taddr + 16 * h, w);
    }
}
__device__ __forceinline__ void tm_ld_o(uint32_t taddr, float (&o)[8][4])
{
    uint32_t w[2][16];
    tm_wait_st();  // the previous store of these columns
    tm_issue<16>(taddr, w[0]);
    tm_issue<16>(taddr + 16, w[1]);
    tm_wait_ld();
    tm_pin<16>(w[0]);
    tm_pin<16>(w[1]);
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int i = 0; i < 16; ++i) o[4 * h + i / 4][i % 4] = __uint_as_float(w[h][i]);
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

// 32-byte load that does not allocate in L1: each gathered sector is consumed whole by the
// one instruction that loads it, so caching it in L1 only costs data-pipe bandwidth.
__device__ __forceinline__ void ldg32(const void *p, uint32_t *w)
{
    asm volatile("ld.global.nc.L1::no_allocate.v8.u32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(w[0]), "=r"(w[1]), "=r"(w[2]), "=r"(w[3]), "=r"(w[4]), "=r"(w[5]), "=r"(w[6]), "=r"(w[7])
                 : "l"(p));
}

__device__ __forceinline__ void ldg16w(const void *p, uint32_t *w)
{
    const uint4 x = ldg16(p);
    w[0] = x.x;
    w[1] = x.y;
    w[2] = x.z;
    w[3] = x.w;
}

// Head-dim layout of one lane's share of a gathered row (lane p = lane/4, q = lane%4).
//   K row, WIDE (32-byte loads): lane q holds elements 64u + 16q + [0, 16), u < D/64, and the
//     four lanes of a row read 128 contiguous bytes per load; narrow (16-byte loads): lane q
//     holds 32u + 8q + [0, 8), u < D/32 (64 contiguous bytes per row per load).
//   Either way word 2t / 2t+1 of the lane's K words is the A operand of k-step t, and the
//   query takes the same elements (kelem below).
//   V row, WIDE and D = 128: lane p holds 16p + [0, 16) (eight lanes read the whole 256-byte
//     row); otherwise 64u + 8p + [0, 8), u < D/64. Word j (elements d, d+1) feeds m-tile j.
template <int D, bool WIDE>
__device__ __forceinline__ int kelem(int t, int q)
{
    return WIDE ? 64 * (t >> 2) + 16 * q + 4 * (t & 3) : 32 * (t >> 1) + 8 * q + 4 * (t & 1);
}

template <int D, bool WIDE>
__device__ __forceinline__ int velem(int j, int p)
{
    return (WIDE && D == 128) ? 16 * p + 2 * j : 64 * (j >> 2) + 8 * p + 2 * (j & 3);
}

constexpr float kLazyLog2 = 8.f;  // rescale O only when the row maximum grows by more than 2^8

#ifndef RIS_ATTN_MIN_BLOCKS
#define RIS_ATTN_MIN_BLOCKS 1
#endif

// D: head dim (64 or 128). QSPLIT: q is fp32 (split hi + lo); else q is bf16.
// KSPLIT: keys come as a bf16 hi (a.k) + lo (a.k_lo) pair. WIDE: 32-byte loads (K, K lo and
// V pointers 32-byte aligned).
// SEEDS (per-seed masks, n_sets > 1): a warp owns (row i, KV head g) and walks the sets one
// after the other, requesting the next set's key range and first keys while the current set
// runs and its first K/V rows during the current set's last group, so the load pipeline
// never drains between sets; a.n_tasks counts (row, KV head) pairs.
// E8 (head dim 128, rotated bf16 inputs, 32-byte loads): the operands of the tile kernel's
// fp8-correction scheme, written by launch_fp8_prep (see fp8_score_scales): keys as fp16 hi
// parts (a.k) and, in each (token, head)'s 2D-byte record of a.k_lo, e4m3(k_h 2^-eb) at bytes
// [0, D) and e4m3(k_l 2^(12+ea)) at [D, 2D); queries likewise (a.q, a.q_lo; 2^-ea and
// 2^(12+eb)). The gather fetches only the fp16 hi part and the e4m3 lo part of a key row (384
// bytes instead of 512) and forms
//   S^T = K_h Q_h + K_h Q_l + 2^-12 e4m3(K_l) e4m3(Q_h)
// with Q_l taken back to fp16 from its e4m3 operand: two fp16 products and one e4m3 product of
// half the k-steps (m16n8k32) instead of three bf16 products. Each of the two approximated
// terms is within about 2^-15 of |q||k| per channel, as in the tile kernel's scheme. (Widening
// the e4m3 lo part to fp16 in registers for a third fp16 product instead measured slower than
// the bf16 pairs: the conversions cost more than the bytes saved.)
template <int D, bool QSPLIT, bool KSPLIT, bool WIDE, typename TIdx, bool DENSE, typename TOut, bool SEEDS, bool E8,
          bool TQ>
__device__ __forceinline__ void gather_task(const AttnArgs &a, int eb, uint32_t tbase)
{
    static_assert(!E8 || (D == 128 && QSPLIT && KSPLIT && WIDE), "the fp8 operands: head dim 128, 32-byte loads");
    static_assert(!TQ || E8, "query fragments and accumulators in TMEM: the fp8 form");
    constexpr int KSTEPS = D / 16;  // k-steps of the score product
    constexpr int KW = D / 8;       // 32-bit words of one K row per lane (D/4 elements)
    constexpr int VW = D / 16;      // 32-bit words of one V row per lane (D/8 elements)
    constexpr int MT = D / 16;      // m-tiles of the value product (head dim)
    constexpr bool VWIDE = WIDE && D == 128;

    const int lane = threadIdx.x & 31;
    const int64_t tid = (int64_t)blockIdx.x * kAttnWarps + (threadIdx.x >> 5);
    if (tid >= a.n_tasks) return;
    const int p = lane >> 2, q = lane & 3;
    Task t;
    if (SEEDS) {
        t.g = (int)(tid % a.Hkv);
        t.i = a.row1 - 1 - tid / a.Hkv;
        t.s = 0;
        t.mask_id = a.heads_keyed > 1 ? t.g : 0;
    } else {
        t = decode_task(a, tid);
    }
    int64_t beg, n;
    key_range<DENSE>(a, t, beg, n);
    // dense-suffix split: the row's dense suffix (its Structural block and / or local window,
    // i - lo + 1 keys up to the row) ends the ascending list and was attended by the tile
    // kernel's suffix pass
    const bool split = a.part_o != nullptr;
    if (split) {
        n -= t.i - dense_suffix_start(a, t.i) + 1;
        if (n < 0) n = 0;
    }
    const TIdx *cols = DENSE ? nullptr : reinterpret_cast<const TIdx *>(a.col) + beg;
    int64_t set_n = n;  // keys of the current set (SEEDS: reloaded per set)

    // ---- query fragments (B operand of the score product), head p of this KV group
    uint32_t qh[KSTEPS][2], ql[KSTEPS][2];
    uint32_t q8[E8 ? 8 : 1];  // E8: e4m3(q_h 2^-ea), elements 32q .. 32q + 31 (natural order)
    {
        const bool hv = p < a.G;
        const int64_t qrow = (t.i * a.Hq + (int64_t)t.g * a.G + (hv ? p : 0)) * D;
        if constexpr (E8) {
            const unsigned char *rec = reinterpret_cast<const unsigned char *>(a.q_lo) + 2 * qrow;
            const uint4 x0 = hv ? *reinterpret_cast<const uint4 *>(rec + 32 * q) : make_uint4(0u, 0u, 0u, 0u);
            const uint4 x1 = hv ? *reinterpret_cast<const uint4 *>(rec + 32 * q + 16) : make_uint4(0u, 0u, 0u, 0u);
            const uint32_t w[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
            for (int e = 0; e < 8; ++e) q8[e] = w[e];
        }
        const float ql_scale = E8 ? pow2i(-12 - eb) : 1.f;
#pragma unroll
        for (int ks = 0; ks < KSTEPS; ++ks) {
            const int d0 = kelem<D, WIDE>(ks, q);
            if constexpr (E8) {  // fp16 hi part; lo part from its e4m3 operand
                const uint2 wh = hv ? *reinterpret_cast<const uint2 *>(reinterpret_cast<const __half *>(a.q) + qrow + d0)
                                    : make_uint2(0u, 0u);
                const uint32_t w8 = hv ? *reinterpret_cast<const uint32_t *>(
                                             reinterpret_cast<const unsigned char *>(a.q_lo) + 2 * qrow + D + d0)
                                       : 0u;
                qh[ks][0] = wh.x;
                qh[ks][1] = wh.y;
                ql[ks][0] = e4m3x2_to_f16x2(w8, ql_scale);
                ql[ks][1] = e4m3x2_to_f16x2(w8 >> 16, ql_scale);
            } else if (QSPLIT && a.q_lo != nullptr) {  // the split given as a bf16 pair
                const uint2 wh = hv ? *reinterpret_cast<const uint2 *>(reinterpret_cast<const __nv_bfloat16 *>(a.q) + qrow + d0)
                                    : make_uint2(0u, 0u);
                const uint2 wl = hv ? *reinterpret_cast<const uint2 *>(reinterpret_cast<const __nv_bfloat16 *>(a.q_lo) + qrow + d0)
                                    : make_uint2(0u, 0u);
                qh[ks][0] = wh.x;
                qh[ks][1] = wh.y;
                ql[ks][0] = wl.x;
                ql[ks][1] = wl.y;
            } else if (QSPLIT) {
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

    // TQ: this thread's TMEM lane; the query fragments in columns 0-39 (k-step ks: hi, hi, lo,
    // lo at 4 ks .. 4 ks + 3; the e4m3 words at 32-39), the output accumulators in 64-95
    const uint32_t tl = tbase + ((uint32_t)(32 * ((threadIdx.x >> 5) & 3)) << 16);
    if constexpr (TQ) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            uint32_t w[16];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                w[4 * k] = qh[4 * h + k][0];
                w[4 * k + 1] = qh[4 * h + k][1];
                w[4 * k + 2] = ql[4 * h + k][0];
                w[4 * k + 3] = ql[4 * h + k][1];
            }
            tm_st<16>(tl + 16 * h, w);
        }
        tm_st<8>(tl + 32, q8);
        tm_wait_st();
    }
    const size_t row_bytes = (size_t)a.Hkv * D * sizeof(__nv_bfloat16);
    const size_t head_off = (size_t)t.g * D * sizeof(__nv_bfloat16);
    const char *kb = reinterpret_cast<const char *>(a.k) + head_off + 2 * kelem<D, WIDE>(0, q);
    // E8: the e4m3 lo part of a key row, bytes D .. 2D - 1 of its record (the record stride is the
    // hi part's row stride), elements 32q .. 32q + 31 to lane q
    const char *kbl = !KSPLIT ? nullptr
                      : E8    ? reinterpret_cast<const char *>(a.k_lo) + head_off + D + 32 * q
                              : reinterpret_cast<const char *>(a.k_lo) + head_off + 2 * kelem<D, WIDE>(0, q);
    // E8: the values are read as their fp16 copy (scaled into range by 2^-E, E from the largest
    // |v|), and P enters the value product as one fp16 with the row sums adding P as rounded
    const char *vb = reinterpret_cast<const char *>(E8 ? a.v16 : a.v) + head_off + 2 * velem<D, WIDE>(0, p);
    const float vsc = E8 ? pow2i(v_scale_exp(*a.v_absmax)) : 1.f;  // 2^E, undone in the epilogue

    float o[MT][4];
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
    const float sc = a.scale_log2;
    if (split) {
        // start from the suffix pass's softmax: maximum = its log-sum-exp, sum 1 (on one lane
        // of the eight that share heads 2q, 2q+1), O = its normalised output, laid out as the
        // epilogue stores it
        const int hh0 = 2 * q, hh1 = 2 * q + 1;
        const float *po = a.part_o + (t.i * a.Hq + (int64_t)t.g * a.G) * D;
        const float *pl = a.part_lse + t.i * a.Hq + (int64_t)t.g * a.G;
#pragma unroll
        for (int hs = 0; hs < 2; ++hs) {
            const int hh = hs ? hh1 : hh0;
            if (hh >= a.G) continue;
            (hs ? m1 : m0) = pl[hh];
            (hs ? l1 : l0) = p == 0 ? 1.f : 0.f;
#pragma unroll
            for (int r = 0; r < MT / 4; ++r) {
                const float4 *src = reinterpret_cast<const float4 *>(po + (int64_t)hh * D + velem<D, WIDE>(4 * r, p));
                const float4 x0 = src[0], x1 = src[1];
                const float run[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {  // into the values' scale (E8: 2^-E, exact)
                    o[4 * r + j][hs] = run[2 * j] / vsc;
                    o[4 * r + j][2 + hs] = run[2 * j + 1] / vsc;
                }
            }
        }
    }

    if constexpr (TQ) tm_st_o(tl + 64, o);

    // ---- key indices, prefetched 64 keys (4 groups) ahead: lane holds positions
    //      64c + lane and 64c + 32 + lane of chunk c; slots past the row read the row itself
    int cur[2], nxt[2];
    auto load_chunk_at = [&](const TIdx *cl, int nk, int cbase, int (&dst)[2]) {
#pragma unroll
        for (int w = 0; w < 2; ++w) {
            const int pos = cbase + 32 * w + lane;
            dst[w] = pos < nk ? key_at<DENSE, TIdx>(cl, pos) : (int)t.i;
        }
    };
    auto load_chunk = [&](int cbase, int (&dst)[2]) { load_chunk_at(cols, (int)set_n, cbase, dst); };
    load_chunk(0, cur);
    load_chunk(64, nxt);
    // index of slot r (0..15) of group slot gs (0..3) of a chunk held in (c0, c1)
    auto slot = [&](int c0, int c1, int gs, int r) -> int {
        return __shfl_sync(0xFFFFFFFFu, (gs >> 1) ? c1 : c0, (16 * gs + r) & 31);
    };

    // ---- gathered rows of one group: K rows p and p+8, V rows 2q, 2q+1, 2q+8, 2q+9
    uint32_t k0[KW], k1[KW], kl0[KSPLIT ? KW : 1], kl1[KSPLIT ? KW : 1], v0[VW], v1[VW], v2[VW], v3[VW];
    auto load_row = [&](const char *rowp, uint32_t *w, int nwords, int stride, bool wide) {
        if (wide) {
#pragma unroll
            for (int u = 0; u < nwords / 8; ++u) ldg32(rowp + stride * u, w + 8 * u);
        } else {
#pragma unroll
            for (int u = 0; u < nwords / 4; ++u) ldg16w(rowp + stride * u, w + 4 * u);
        }
    };
    auto issue_k = [&](int c0, int c1, int gs) {
        const int ik0 = slot(c0, c1, gs, p), ik1 = slot(c0, c1, gs, p + 8);
        load_row(kb + (size_t)ik0 * row_bytes, k0, KW, WIDE ? 128 : 64, WIDE);
        load_row(kb + (size_t)ik1 * row_bytes, k1, KW, WIDE ? 128 : 64, WIDE);
        if (E8) {
            ldg32(kbl + (size_t)ik0 * row_bytes, kl0);
            ldg32(kbl + (size_t)ik1 * row_bytes, kl1);
        } else if (KSPLIT) {
            load_row(kbl + (size_t)ik0 * row_bytes, kl0, KW, WIDE ? 128 : 64, WIDE);
            load_row(kbl + (size_t)ik1 * row_bytes, kl1, KW, WIDE ? 128 : 64, WIDE);
        }
    };
    auto issue_v = [&](int c0, int c1, int gs) {
        const int iv0 = slot(c0, c1, gs, 2 * q), iv1 = slot(c0, c1, gs, 2 * q + 1);
        const int iv2 = slot(c0, c1, gs, 2 * q + 8), iv3 = slot(c0, c1, gs, 2 * q + 9);
        load_row(vb + (size_t)iv0 * row_bytes, v0, VW, 128, VWIDE);
        load_row(vb + (size_t)iv1 * row_bytes, v1, VW, 128, VWIDE);
        load_row(vb + (size_t)iv2 * row_bytes, v2, VW, 128, VWIDE);
        load_row(vb + (size_t)iv3 * row_bytes, v3, VW, 128, VWIDE);
    };

    // Phase-shifted pipeline: the next group's K rows are requested as soon as this group's
    // scores are formed, its V rows as soon as this group's values are accumulated.
    issue_k(cur[0], cur[1], 0);
    issue_v(cur[0], cur[1], 0);
    const int n_sets = SEEDS ? a.n_sets : 1;
    for (int set = 0; set < n_sets; ++set) {
    // SEEDS: the next set's key range and first 64 keys, requested now
    const TIdx *ncols = cols;
    int64_t nn = 0;
    int ncur[2] = {0, 0};
    if (SEEDS && set + 1 < n_sets) {
        Task tn = t;
        tn.s = set + 1;
        tn.mask_id = tn.s * a.heads_keyed + (a.heads_keyed > 1 ? t.g : 0);
        int64_t nbeg;
        key_range<DENSE>(a, tn, nbeg, nn);
        ncols = DENSE ? nullptr : reinterpret_cast<const TIdx *>(a.col) + nbeg;
        load_chunk_at(ncols, (int)nn, 0, ncur);
    }
    n = set_n;
    // key positions and group indices in 32 bits (N < 2^31, so a row holds fewer keys): the
    // same loop with 64-bit positions ran 10% slower
    const int nk = (int)n;
    const int ngroups = (nk + 15) / 16;
    for (int g = 0; g < ngroups; ++g) {
        const int base = 16 * g;
        const int gs = (int)(g & 3), gs1 = (gs + 1) & 3;
        const bool more = g + 1 < ngroups;
        const bool cross = SEEDS && !more && set + 1 < n_sets;  // the next set's first group
        const int n0 = gs1 == 0 ? nxt[0] : cur[0], n1 = gs1 == 0 ? nxt[1] : cur[1];
        const bool val0 = base + p < nk, val1 = base + p + 8 < nk;

        // ---- S^T = K~ Q~^T: independent accumulator chains (hi*hi, hi*lo, lo*hi, and even/odd
        //      k-steps) so the tensor-core latencies overlap instead of forming one serial chain
        float sa[2][4], sb[2][4], sl[2][4];
#pragma unroll
        for (int c = 0; c < 2; ++c)
#pragma unroll
            for (int e = 0; e < 4; ++e) sa[c][e] = sb[c][e] = sl[c][e] = 0.f;
        if constexpr (TQ) {
            uint32_t wq[2][16], w8[8];
            tm_issue<16>(tl, wq[0]);
            tm_issue<16>(tl + 16, wq[1]);
            tm_issue<8>(tl + 32, w8);
            tm_wait_ld();
            tm_pin<16>(wq[0]);
            tm_pin<16>(wq[1]);
            tm_pin<8>(w8);
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const uint32_t *w = wq[h];
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const int ks = 4 * h + k;
                    mma16816_f16(sa[ks & 1], k0[2 * ks], k1[2 * ks], k0[2 * ks + 1], k1[2 * ks + 1], w[4 * k], w[4 * k + 1]);
                    mma16816_f16(sb[ks & 1], k0[2 * ks], k1[2 * ks], k0[2 * ks + 1], k1[2 * ks + 1], w[4 * k + 2],
                                 w[4 * k + 3]);
                }
            }
#pragma unroll
            for (int ks = 0; ks < D / 32; ++ks)
                mma16832_e4m3(sl[ks & 1], kl0[2 * ks], kl1[2 * ks], kl0[2 * ks + 1], kl1[2 * ks + 1], w8[2 * ks],
                              w8[2 * ks + 1]);
        } else if constexpr (E8) {
#pragma unroll
            for (int ks = 0; ks < KSTEPS; ++ks) {
                mma16816_f16(sa[ks & 1], k0[2 * ks], k1[2 * ks], k0[2 * ks + 1], k1[2 * ks + 1], qh[ks][0], qh[ks][1]);
                mma16816_f16(sb[ks & 1], k0[2 * ks], k1[2 * ks], k0[2 * ks + 1], k1[2 * ks + 1], ql[ks][0], ql[ks][1]);
            }
#pragma unroll
            for (int ks = 0; ks < D / 32; ++ks)
                mma16832_e4m3(sl[ks & 1], kl0[2 * ks], kl1[2 * ks], kl0[2 * ks + 1], kl1[2 * ks + 1], q8[2 * ks],
                              q8[2 * ks + 1]);
        } else {
#pragma unroll
        for (int ks = 0; ks < KSTEPS; ++ks) {
            mma16816(sa[ks & 1], k0[2 * ks], k1[2 * ks], k0[2 * ks + 1], k1[2 * ks + 1], qh[ks][0], qh[ks][1]);
            if (QSPLIT)
                mma16816(sb[ks & 1], k0[2 * ks], k1[2 * ks], k0[2 * ks + 1], k1[2 * ks + 1], ql[ks][0], ql[ks][1]);
            if (KSPLIT) {
                constexpr int LW = KSPLIT ? KW : 1;
                mma16816(sl[ks & 1], kl0[(2 * ks) % LW], kl1[(2 * ks) % LW], kl0[(2 * ks + 1) % LW],
                         kl1[(2 * ks + 1) % LW], qh[ks][0], qh[ks][1]);
            }
        }
        }
        float s[4];
        constexpr float kLoScale = E8 ? 0x1p-12f : 1.f;  // E8: the e4m3 product carries 2^12
#pragma unroll
        for (int e = 0; e < 4; ++e)
            s[e] = ((sa[0][e] + sa[1][e]) + (sb[0][e] + sb[1][e])) + kLoScale * (sl[0][e] + sl[1][e]);
        if (more)
            issue_k(n0, n1, gs1);
        else if (cross)
            issue_k(ncur[0], ncur[1], 0);

        // ---- online softmax; lane holds keys p, p+8 x heads 2q, 2q+1
        float s0 = val0 ? s[0] * sc : -INFINITY, s1 = val0 ? s[1] * sc : -INFINITY;
        float s2 = val1 ? s[2] * sc : -INFINITY, s3 = val1 ? s[3] * sc : -INFINITY;
        float mx0 = fmaxf(s0, s2), mx1 = fmaxf(s1, s3);
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
            mx0 = fmaxf(mx0, __shfl_xor_sync(0xFFFFFFFFu, mx0, off));
            mx1 = fmaxf(mx1, __shfl_xor_sync(0xFFFFFFFFu, mx1, off));
        }
        // Lazy rescaling: the reference maximum only moves when a score exceeds it by more
        // than 2^kLazyLog2 (probabilities then stay below 2^kLazyLog2 and the fp32 sums stay
        // exact enough), so most groups skip the rescale of O; the branch is warp-uniform.
        const bool need0 = mx0 > m0 + kLazyLog2, need1 = mx1 > m1 + kLazyLog2;
        if (__any_sync(0xFFFFFFFFu, need0 || need1)) {
            const float mn0 = need0 ? mx0 : m0, mn1 = need1 ? mx1 : m1;
            const float al0 = need0 ? exp2f(m0 - mn0) : 1.f, al1 = need1 ? exp2f(m1 - mn1) : 1.f;
            m0 = mn0;
            m1 = mn1;
            l0 *= al0;
            l1 *= al1;
            if constexpr (TQ) tm_ld_o(tl + 64, o);
#pragma unroll
            for (int mt = 0; mt < MT; ++mt) {
                o[mt][0] *= al0;
                o[mt][1] *= al1;
                o[mt][2] *= al0;
                o[mt][3] *= al1;
            }
            if constexpr (TQ) tm_st_o(tl + 64, o);
        }
        const float mu0 = (m0 == -INFINITY) ? 0.f : m0, mu1 = (m1 == -INFINITY) ? 0.f : m1;
        const float p0 = exp2f(s0 - mu0), p1 = exp2f(s1 - mu1);
        const float p2 = exp2f(s2 - mu0), p3 = exp2f(s3 - mu1);
        // P transposed into the B operand P[head p][keys 2q.., 2q+8..]: E8 one fp16 (the row sums
        // add it as rounded, so each weight's rounding moves the output by at most 2^-11 of that
        // weight times |v_j - o|), else P_hi + P_lo in bf16
        uint32_t pb0, pb1, pl0 = 0u, pl1 = 0u;
        if constexpr (E8) {
            const __half2 f01 = __floats2half2_rn(p0, p1), f23 = __floats2half2_rn(p2, p3);
            const float2 r01 = __half22float2(f01), r23 = __half22float2(f23);
            l0 += r01.x + r23.x;
            l1 += r01.y + r23.y;
            pb0 = transpose8x8(*reinterpret_cast<const uint32_t *>(&f01));
            pb1 = transpose8x8(*reinterpret_cast<const uint32_t *>(&f23));
        } else {
            l0 += p0 + p2;
            l1 += p1 + p3;
            const float h0 = __bfloat162float(__float2bfloat16_rn(p0)), h1 = __bfloat162float(__float2bfloat16_rn(p1));
            const float h2 = __bfloat162float(__float2bfloat16_rn(p2)), h3 = __bfloat162float(__float2bfloat16_rn(p3));
            pb0 = transpose8x8(pack_bf16(h0, h1));
            pb1 = transpose8x8(pack_bf16(h2, h3));
            pl0 = transpose8x8(pack_bf16(p0 - h0, p1 - h1));
            pl1 = transpose8x8(pack_bf16(p2 - h2, p3 - h3));
        }

        // ---- O^T += V^T P^T
        if constexpr (TQ) tm_ld_o(tl + 64, o);
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
            const uint32_t a0 = __byte_perm(v0[mt], v1[mt], 0x5410);
            const uint32_t a1 = __byte_perm(v0[mt], v1[mt], 0x7632);
            const uint32_t a2 = __byte_perm(v2[mt], v3[mt], 0x5410);
            const uint32_t a3 = __byte_perm(v2[mt], v3[mt], 0x7632);
            if constexpr (E8) {
                mma16816_f16(o[mt], a0, a1, a2, a3, pb0, pb1);
            } else {
                mma16816(o[mt], a0, a1, a2, a3, pb0, pb1);
                mma16816(o[mt], a0, a1, a2, a3, pl0, pl1);
            }
        }
        if constexpr (TQ) tm_st_o(tl + 64, o);
        if (more)
            issue_v(n0, n1, gs1);
        else if (cross)
            issue_v(ncur[0], ncur[1], 0);
        if (gs == 3) {  // the next group starts the prefetched chunk; fetch the one after it
            cur[0] = nxt[0];
            cur[1] = nxt[1];
            load_chunk(base + 16 + 64, nxt);
        }
    }

    // ---- epilogue: full row sums, normalise, undo the head-dim permutation
    if constexpr (TQ) tm_ld_o(tl + 64, o);
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
        l0 += __shfl_xor_sync(0xFFFFFFFFu, l0, off);
        l1 += __shfl_xor_sync(0xFFFFFFFFu, l1, off);
    }
    const float inv0 = vsc / l0, inv1 = vsc / l1;
    const int h0 = 2 * q, h1 = 2 * q + 1;
    TOut *out = reinterpret_cast<TOut *>(a.out) + (((int64_t)t.s * a.N + t.i) * a.Hq + (int64_t)t.g * a.G) * D;
    // runs of 8 consecutive head-dim elements: words 4r .. 4r+3 of the lane's V layout
    constexpr int RUNS = MT / 4;
#pragma unroll
    for (int r = 0; r < RUNS; ++r) {
        float run[8];
        const int d = velem<D, WIDE>(4 * r, p);
        if (h0 < a.G) {
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                run[2 * j] = o[4 * r + j][0] * inv0;
                run[2 * j + 1] = o[4 * r + j][2] * inv0;
            }
            store_run<TOut>(out + (int64_t)h0 * D + d, run, 8);
        }
        if (h1 < a.G) {
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                run[2 * j] = o[4 * r + j][1] * inv1;
                run[2 * j + 1] = o[4 * r + j][3] * inv1;
            }
            store_run<TOut>(out + (int64_t)h1 * D + d, run, 8);
        }
    }
    if (a.lse != nullptr && p == 0) {
        float *lse = a.lse + ((int64_t)t.s * a.Hq + (int64_t)t.g * a.G) * a.lse_ld + t.i;
        if (h0 < a.G) lse[(int64_t)h0 * a.lse_ld] = (m0 + __log2f(l0)) * kLn2;
        if (h1 < a.G) lse[(int64_t)h1 * a.lse_ld] = (m1 + __log2f(l1)) * kLn2;
    }
    if (SEEDS && set + 1 < n_sets) {
        // on to the next set: its first group's rows are in flight
        t.s = set + 1;
        t.mask_id = t.s * a.heads_keyed + (a.heads_keyed > 1 ? t.g : 0);
        cols = ncols;
        set_n = nn;
        cur[0] = ncur[0];
        cur[1] = ncur[1];
        load_chunk(64, nxt);
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
        if constexpr (TQ) tm_st_o(tl + 64, o);
        m0 = m1 = -INFINITY;
        l0 = l1 = 0.f;
    }
    }  // sets
}

// F8: the queries and keys came from launch_fp8_prep; which of its two schemes it wrote
// follows from the bounds at a.qk_bound, read here on the device as it did.
// F8: the query fragments and output accumulators live in tensor memory
// (each thread's own TMEM lane, 128 columns per CTA), which leaves room for three CTAs of four
// warps per SM instead of two, and so more gathered rows in flight.
constexpr int kGatherTmemCols = 128;
template <int D, bool QSPLIT, bool KSPLIT, bool WIDE, typename TIdx, bool DENSE, typename TOut, bool SEEDS, bool F8>
__global__ void __launch_bounds__(kAttnWarps * 32, F8 ? 3 : RIS_ATTN_MIN_BLOCKS) k_attn_bf16(const AttnArgs a)
{
    if constexpr (F8) {
        __shared__ uint32_t tbase_sh;
        const int warp = threadIdx.x >> 5;
        if (warp == 0) {
            asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                         ::"r"((uint32_t)__cvta_generic_to_shared(&tbase_sh)), "r"(kGatherTmemCols) : "memory");
            asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
        }
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncthreads();
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t tb = tbase_sh;
        int ea = 0, eb = 0;
        if (fp8_score_scales(a.qk_bound[0], a.qk_bound[1], ea, eb))
            gather_task<D, QSPLIT, KSPLIT, WIDE, TIdx, DENSE, TOut, SEEDS, true, true>(a, eb, tb);
        else
            gather_task<D, QSPLIT, KSPLIT, WIDE, TIdx, DENSE, TOut, SEEDS, false, false>(a, 0, 0u);
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        __syncthreads();
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        if (warp == 0)
            asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tb), "r"(kGatherTmemCols)
                         : "memory");
    } else {
        gather_task<D, QSPLIT, KSPLIT, WIDE, TIdx, DENSE, TOut, SEEDS, false, false>(a, 0, 0u);
    }
}

template <int D, bool QSPLIT, bool WIDE, typename TOut, bool F8>
cudaError_t launch_f(const AttnArgs &a, int col_bytes, bool dense, cudaStream_t s)
{
    // rotated inputs: fp32 queries and hi + lo keys; as given: bf16 queries and keys
    constexpr bool KSPLIT = QSPLIT;
    const dim3 block(kAttnWarps * 32);
    if (!dense && a.n_sets > 1) {  // per-seed sets: one warp per (row, KV head) walks them all
        AttnArgs b = a;
        b.n_tasks = (a.row1 - a.row0) * a.Hkv;
        const unsigned grid = (unsigned)((b.n_tasks + kAttnWarps - 1) / kAttnWarps);
        if (col_bytes == 2)
            k_attn_bf16<D, QSPLIT, KSPLIT, WIDE, uint16_t, false, TOut, true, F8><<<grid, block, 0, s>>>(b);
        else
            k_attn_bf16<D, QSPLIT, KSPLIT, WIDE, uint32_t, false, TOut, true, F8><<<grid, block, 0, s>>>(b);
        note_launch();
        return cudaGetLastError();
    }
    const unsigned grid = (unsigned)((a.n_tasks + kAttnWarps - 1) / kAttnWarps);
    if (dense)
        k_attn_bf16<D, QSPLIT, KSPLIT, WIDE, uint32_t, true, TOut, false, F8><<<grid, block, 0, s>>>(a);
    else if (col_bytes == 2)
        k_attn_bf16<D, QSPLIT, KSPLIT, WIDE, uint16_t, false, TOut, false, F8><<<grid, block, 0, s>>>(a);
    else
        k_attn_bf16<D, QSPLIT, KSPLIT, WIDE, uint32_t, false, TOut, false, F8><<<grid, block, 0, s>>>(a);
    note_launch();
    return cudaGetLastError();
}

template <int D, bool QSPLIT, bool WIDE, typename TOut>
cudaError_t launch_w(const AttnArgs &a, int col_bytes, bool dense, cudaStream_t s)
{
    // operands in launch_fp8_prep's form (a.qk_bound set) are read only by the F8 kernel, which
    // needs head dim 128 and 32-byte aligned inputs (the caller checks both)
    if constexpr (D == 128 && QSPLIT && WIDE) {
        if (a.qk_bound != nullptr) return launch_f<D, QSPLIT, WIDE, TOut, true>(a, col_bytes, dense, s);
    } else {
        if (a.qk_bound != nullptr) return cudaErrorInvalidValue;
    }
    return launch_f<D, QSPLIT, WIDE, TOut, false>(a, col_bytes, dense, s);
}

bool aligned32(const void *p) { return p == nullptr || (reinterpret_cast<uintptr_t>(p) & 31u) == 0; }

template <int D, bool QSPLIT, typename TOut>
cudaError_t launch_d(const AttnArgs &a, int col_bytes, bool dense, cudaStream_t s)
{
    // 32-byte loads need 32-byte aligned K, K lo and V (the ABI promises 16)
    if (aligned32(a.k) && aligned32(a.k_lo) && aligned32(a.v))
        return launch_w<D, QSPLIT, true, TOut>(a, col_bytes, dense, s);
    return launch_w<D, QSPLIT, false, TOut>(a, col_bytes, dense, s);
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
