// RIS sparse attention, masked dense-tile design on the 5th-generation tensor cores
// (paper, Methods, "Hybrid Anchor and Pre-Fusion Unified Softmax (PFUS)"; the dense causal
// upper bound of Table tab:results_32k is the same kernel with every causal pair kept).
//
// Where the master mask keeps a large share of the causal pairs (union densities of tens of
// percent, and the dense mode) a dense 128 x 64 score tile with the mask applied as -inf
// beats gathering rows pair by pair. One CTA owns one (128-query tile, query head, set):
//
//   warp 4 (TMA)   loads the query tile once (bf16 hi and lo) and streams 64-key stages of
//                  K~ hi, K~ lo and V (128-byte swizzled boxes) into a two-stage ring;
//   warp 5 (MMA)   one elected lane issues tcgen05.mma: S = Q_hi K_hi^T + Q_lo K_hi^T +
//                  Q_hi K_lo^T into a double-buffered TMEM score tile, and O += P_hi V + P_lo V
//                  into the TMEM output tile, committing each step to an mbarrier;
//   warps 0-3      one thread per query row: tcgen05.ld its 64 scores, apply the bitmap
//                  (or the causal cut), fp32 online softmax with lazy rescaling of O in TMEM
//                  (only when the row max grows by more than 2^8), write P hi / lo to shared
//                  memory in the canonical K-major 128-byte-swizzled layout, and at the end
//                  normalise O and store the row.
//
// Every mbarrier wait is bounded; a wait that gives up sets bit 1 of the device error word,
// every role falls through to the end, TMEM is released and the CTA returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>

#include <cstdint>
#include <mutex>

#include "attn_common.cuh"

namespace ris {

// Device error word of this kernel (bit 1: a bounded wait gave up); read by read_tile_error.
__device__ unsigned int g_ris_tile_error;

namespace {

constexpr int BM = 128;          // query rows per tile (TMEM lanes)
constexpr int BN = 64;           // keys per stage
constexpr int DT = 128;          // head dim handled by this kernel
constexpr int kThreads = 192;    // warps 0-3 softmax, 4 TMA, 5 MMA
constexpr uint32_t kTmemCols = 256;  // S[2] (2 x 64) + O (128)

// shared-memory map (bytes, from a 1024-aligned base)
constexpr int Q_ARR = BM * DT * 2;          // 32 KB: one of Q hi / Q lo (two 64-column blocks)
constexpr int Q_BLK = BM * 128;             // 16 KB: one 64-column block of the query tile
constexpr int KV_ARR = BN * DT * 2;         // 16 KB: one of K hi / K lo / V
constexpr int KV_BLK = BN * 128;            // 8 KB: one 64-column block
constexpr int STAGE = 3 * KV_ARR;           // 48 KB
constexpr int P_ARR = BM * BN * 2;          // 16 KB: P hi or P lo
constexpr int OFF_Q = 0;
constexpr int OFF_KV = 2 * Q_ARR;           // 64 KB
constexpr int OFF_P = OFF_KV + 2 * STAGE;   // 160 KB
constexpr int SMEM_BYTES = OFF_P + 2 * P_ARR + 1024;  // + alignment slack = 197632

enum Bar { B_Q = 0, B_KV_FULL = 1, B_KV_EMPTY = 3, B_S_FULL = 5, B_S_EMPTY = 7, B_P_FULL = 9, B_PV_DONE = 10, NBAR = 11 };

__device__ __forceinline__ uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
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
// Bounded wait (about 2^31 cycles); false if the phase did not complete in time.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity)
{
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity)) {
        if (clock64() - t0 > (1LL << 31)) return false;
        if (*reinterpret_cast<volatile unsigned int *>(&g_ris_tile_error) != 0u) return false;
    }
    return true;
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map, int c0, int c1, int c2, uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cta.global.tile.mbarrier::complete_tx::bytes "
        "[%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(bar)
        : "memory");
}

// ---- tcgen05 helpers
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }

// Shared-memory matrix descriptor: K-major or MN-major, 128-byte swizzle, version 1.
__device__ __forceinline__ uint64_t sdesc(uint32_t addr, uint32_t lbo, uint32_t sbo)
{
    uint64_t d = 0;
    d |= (uint64_t)((addr >> 4) & 0x3FFF);
    d |= (uint64_t)((lbo >> 4) & 0x3FFF) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFF) << 32;
    d |= (uint64_t)1 << 46;  // descriptor version
    d |= (uint64_t)2 << 61;  // 128-byte swizzle
    return d;
}

// Instruction descriptor, kind::f16: bf16 x bf16 -> f32, dense.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, bool b_mn_major)
{
    return (1u << 4)                      // D format f32
           | (1u << 7)                    // A bf16
           | (1u << 10)                   // B bf16
           | ((b_mn_major ? 1u : 0u) << 16)
           | ((uint32_t)(N >> 3) << 17)
           | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}

__device__ __forceinline__ void tc_commit(uint32_t bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

// 32 lanes x 32 consecutive 32-bit columns: thread t of the warp gets lane (base + t).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float *v)
{
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const float *v)
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
        "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])), "r"(__float_as_uint(v[3])),
        "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])), "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])),
        "r"(__float_as_uint(v[8])), "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
        "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])), "r"(__float_as_uint(v[15])),
        "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])), "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])),
        "r"(__float_as_uint(v[20])), "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
        "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])), "r"(__float_as_uint(v[27])),
        "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])), "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
        : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t *>(&v);
}

__device__ __forceinline__ int64_t row_word_offset(int64_t i)
{
    const int64_t a = i >> 5, b = i & 31;
    return i + 16 * a * (a - 1) + a * b;
}

template <typename TOut>
__device__ __forceinline__ void store8(TOut *dst, const float *x);
template <>
__device__ __forceinline__ void store8<float>(float *dst, const float *x)
{
    reinterpret_cast<float4 *>(dst)[0] = make_float4(x[0], x[1], x[2], x[3]);
    reinterpret_cast<float4 *>(dst)[1] = make_float4(x[4], x[5], x[6], x[7]);
}
template <>
__device__ __forceinline__ void store8<__nv_bfloat16>(__nv_bfloat16 *dst, const float *x)
{
    uint4 w;
    w.x = pack_bf16(x[0], x[1]);
    w.y = pack_bf16(x[2], x[3]);
    w.z = pack_bf16(x[4], x[5]);
    w.w = pack_bf16(x[6], x[7]);
    *reinterpret_cast<uint4 *>(dst) = w;
}

struct TileMaps {
    CUtensorMap qh, ql, kh, kl, v;
};

template <bool SPLIT, bool DENSE, typename TOut>
__global__ void __launch_bounds__(kThreads, 1) k_attn_tile(const AttnArgs a, const __grid_constant__ TileMaps maps)
{
    extern __shared__ unsigned char smem_raw[];
    __shared__ __align__(8) uint64_t bars[NBAR];
    __shared__ uint32_t tmem_base_sh;
    unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                            ~uintptr_t(1023));
    const uint32_t sbase = smem_u32(smem);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // ---- tile of this CTA: heavier (later) query tiles first
    const int n_qt = (int)((a.N + BM - 1) / BM);
    const int64_t b = blockIdx.x;
    const int h = (int)(b % a.Hq);
    const int64_t r2 = b / a.Hq;
    const int s = (int)(r2 % a.n_sets);
    const int qt = n_qt - 1 - (int)(r2 / a.n_sets);
    const int64_t q0 = (int64_t)qt * BM;
    const int g = h / a.G;
    const int mask_id = s * a.heads_keyed + (a.heads_keyed > 1 ? g : 0);
    const int64_t last_row = (q0 + BM - 1 < a.N - 1) ? q0 + BM - 1 : a.N - 1;
    const int n_kt = (int)(last_row / BN) + 1;  // causal: key tiles 0 .. last_row / BN

    if (threadIdx.x == 0) {
        for (int i = 0; i < NBAR; ++i) {
            uint32_t cnt = 1;
            if (i == B_S_EMPTY || i == B_S_EMPTY + 1 || i == B_P_FULL) cnt = 128;
            mbar_init(smem_u32(&bars[i]), cnt);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 5) {  // TMEM allocation by one full warp
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_base_sh)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base_sh;
    const uint32_t t_s0 = tmem, t_s1 = tmem + BN, t_o = tmem + 2 * BN;
    bool ok = true;

    if (warp == 4) {
        // =============================== TMA producer
        if (lane == 0) {
            const uint32_t bq = smem_u32(&bars[B_Q]);
            mbar_arrive_expect_tx(bq, (SPLIT ? 2 : 1) * Q_ARR);
            for (int blk = 0; blk < 2; ++blk) {
                tma_load_3d(sbase + OFF_Q + blk * Q_BLK, &maps.qh, 64 * blk, h, (int)q0, bq);
                if (SPLIT) tma_load_3d(sbase + OFF_Q + Q_ARR + blk * Q_BLK, &maps.ql, 64 * blk, h, (int)q0, bq);
            }
            for (int j = 0; j < n_kt && ok; ++j) {
                const int st = j & 1;
                if (j >= 2) ok = mbar_wait(smem_u32(&bars[B_KV_EMPTY + st]), ((j >> 1) - 1) & 1);
                if (!ok) break;
                const uint32_t bf = smem_u32(&bars[B_KV_FULL + st]);
                const uint32_t dst = sbase + OFF_KV + st * STAGE;
                mbar_arrive_expect_tx(bf, (SPLIT ? 3 : 2) * KV_ARR);
                for (int blk = 0; blk < 2; ++blk) {
                    tma_load_3d(dst + 0 * KV_ARR + blk * KV_BLK, &maps.kh, 64 * blk, g, j * BN, bf);
                    if (SPLIT) tma_load_3d(dst + 1 * KV_ARR + blk * KV_BLK, &maps.kl, 64 * blk, g, j * BN, bf);
                    tma_load_3d(dst + 2 * KV_ARR + blk * KV_BLK, &maps.v, 64 * blk, g, j * BN, bf);
                }
            }
            // let the last stages land before the CTA can leave
            for (int j = n_kt - 2; j < n_kt; ++j)
                if (j >= 0) mbar_wait(smem_u32(&bars[B_KV_FULL + (j & 1)]), (j >> 1) & 1);
        }
    } else if (warp == 5) {
        // =============================== MMA issuer
        if (lane == 0) {
            constexpr uint32_t ID_S = idesc_bf16(BM, BN, false);  // S[128 x 64] = Q K^T, both K-major
            constexpr uint32_t ID_O = idesc_bf16(BM, DT, true);   // O[128 x 128] += P V, V MN-major
            ok = mbar_wait(smem_u32(&bars[B_Q]), 0);
            tc_fence_after();
            auto issue_s = [&](int j) {
                const int st = j & 1;
                const uint32_t kv = sbase + OFF_KV + st * STAGE;
                const uint32_t dt = (j & 1) ? t_s1 : t_s0;
                uint32_t acc = 0;
                // (A, B) pairs: (Q hi, K hi), (Q lo, K hi), (Q hi, K lo); 8 k-steps of 16 over D
                for (int prod = 0; prod < (SPLIT ? 3 : 1); ++prod) {
                    const uint32_t qa = sbase + OFF_Q + (prod == 1 ? Q_ARR : 0);
                    const uint32_t kb = kv + (prod == 2 ? KV_ARR : 0);
                    for (int ks = 0; ks < DT / 16; ++ks) {
                        const uint32_t koff = (uint32_t)((ks & 3) * 32);  // 16 columns = 32 B inside a 128 B row
                        const uint64_t ad = sdesc(qa + (ks >> 2) * Q_BLK + koff, 16, 1024);
                        const uint64_t bd = sdesc(kb + (ks >> 2) * KV_BLK + koff, 16, 1024);
                        tc_mma(dt, ad, bd, ID_S, acc);
                        acc = 1;
                    }
                }
                tc_commit(smem_u32(&bars[B_S_FULL + st]));
            };
            auto issue_o = [&](int j) {
                const int st = j & 1;
                const uint32_t vb = sbase + OFF_KV + st * STAGE + 2 * KV_ARR;
                for (int prod = 0; prod < 2; ++prod) {
                    const uint32_t pa = sbase + OFF_P + prod * P_ARR;
                    for (int ks = 0; ks < BN / 16; ++ks) {
                        const uint64_t ad = sdesc(pa + ks * 32, 16, 1024);
                        // V block: 64 keys x 128 B rows; 16 keys = two 8-row atoms (SBO 1024);
                        // the second 64-column block of head dim is LBO = 8 KB away
                        const uint64_t bd = sdesc(vb + ks * 2048, KV_BLK, 1024);
                        tc_mma(t_o, ad, bd, ID_O, (j > 0 || prod > 0 || ks > 0) ? 1u : 0u);
                    }
                }
                tc_commit(smem_u32(&bars[B_PV_DONE]));
                tc_commit(smem_u32(&bars[B_KV_EMPTY + st]));
            };
            for (int j = 0; j < n_kt && ok; ++j) {
                const int st = j & 1;
                ok = mbar_wait(smem_u32(&bars[B_KV_FULL + st]), (j >> 1) & 1);
                if (ok && j >= 2) ok = mbar_wait(smem_u32(&bars[B_S_EMPTY + st]), ((j >> 1) - 1) & 1);
                if (!ok) break;
                tc_fence_after();
                issue_s(j);
                if (j >= 1) {
                    ok = mbar_wait(smem_u32(&bars[B_P_FULL]), (j - 1) & 1);
                    if (!ok) break;
                    tc_fence_after();
                    issue_o(j - 1);
                }
            }
            if (ok) {
                ok = mbar_wait(smem_u32(&bars[B_P_FULL]), (n_kt - 1) & 1);
                if (ok) {
                    tc_fence_after();
                    issue_o(n_kt - 1);
                }
            }
            // the last commit has to land before TMEM is released
            mbar_wait(smem_u32(&bars[B_PV_DONE]), (n_kt - 1) & 1);
        }
    } else {
        // =============================== softmax: thread r owns query row q0 + r
        const int r = threadIdx.x;  // 0..127 == TMEM lane
        const int64_t i = q0 + r;
        const bool row_ok = i < a.N;
        const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
        const uint32_t *bm = DENSE ? nullptr
                                   : a.bitmap + (int64_t)mask_id * a.words_per_mask + (row_ok ? row_word_offset(i) : 0);
        const int64_t last_word = i >> 5;
        const float sc = a.scale_log2;
        float m_used = -INFINITY, l = 0.f;
        unsigned char *prow_hi = smem + OFF_P + r * 128;
        unsigned char *prow_lo = smem + OFF_P + P_ARR + r * 128;
        for (int j = 0; j < n_kt; ++j) {
            const int st = j & 1;
            ok = __all_sync(0xFFFFFFFFu, mbar_wait(smem_u32(&bars[B_S_FULL + st]), (j >> 1) & 1));
            if (!ok) break;
            tc_fence_after();
            float sv[BN];
            tmem_ld32(((j & 1) ? t_s1 : t_s0) + lane_off, sv);
            tmem_ld32(((j & 1) ? t_s1 : t_s0) + lane_off + 32, sv + 32);
            tc_fence_before();
            mbar_arrive(smem_u32(&bars[B_S_EMPTY + st]));

            // mask bits of keys 64j .. 64j + 63 for this row
            const int64_t k0 = (int64_t)j * BN;
            uint32_t w0 = 0, w1 = 0;
            if (row_ok) {
                if (DENSE) {
                    const int64_t lim = i - k0;  // keys k0 .. i are kept
                    w0 = lim >= 31 ? 0xFFFFFFFFu : (lim < 0 ? 0u : ((2u << lim) - 1u));
                    const int64_t lim1 = lim - 32;
                    w1 = lim1 >= 31 ? 0xFFFFFFFFu : (lim1 < 0 ? 0u : ((2u << lim1) - 1u));
                } else {
                    const int64_t wd = k0 >> 5;
                    if (wd <= last_word) w0 = bm[wd];
                    if (wd + 1 <= last_word) w1 = bm[wd + 1];
                }
            }
            float mx = -INFINITY;
#pragma unroll
            for (int c = 0; c < BN; ++c) {
                const uint32_t bit = (c < 32 ? (w0 >> c) : (w1 >> (c - 32))) & 1u;
                sv[c] = bit ? sv[c] * sc : -INFINITY;
                mx = fmaxf(mx, sv[c]);
            }
            // P of the previous tile has been consumed and O is settled
            if (j >= 1) {
                ok = __all_sync(0xFFFFFFFFu, mbar_wait(smem_u32(&bars[B_PV_DONE]), (j - 1) & 1));
                if (!ok) break;
                tc_fence_after();
            }
            // Lazy rescale: a row rescales O only when its max grows by more than 2^8. The
            // TMEM loads / stores are warp-collective (.sync.aligned), so the whole warp runs
            // them when any of its rows needs it; the other rows multiply by 1.
            const bool upd = mx > m_used + 8.f;
            const float al = upd ? (m_used == -INFINITY ? 0.f : exp2f(m_used - mx)) : 1.f;
            if (upd) {
                l *= al;
                m_used = mx;
            }
            if (__any_sync(0xFFFFFFFFu, upd)) {
                float ov[32];
#pragma unroll
                for (int c4 = 0; c4 < DT / 32; ++c4) {
                    tmem_ld32(t_o + lane_off + 32 * c4, ov);
#pragma unroll
                    for (int c = 0; c < 32; ++c) ov[c] *= al;
                    tmem_st32(t_o + lane_off + 32 * c4, ov);
                }
            }
            const float mu = (m_used == -INFINITY) ? 0.f : m_used;
            // P = exp2(s - m_used) in hi + lo, stored as the K-major 128-byte-swizzled A operand
#pragma unroll
            for (int c8 = 0; c8 < BN / 8; ++c8) {
                uint32_t hw[4], lw[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float p0 = exp2f(sv[8 * c8 + 2 * e] - mu), p1 = exp2f(sv[8 * c8 + 2 * e + 1] - mu);
                    l += p0 + p1;
                    const float h0 = __bfloat162float(__float2bfloat16_rn(p0));
                    const float h1 = __bfloat162float(__float2bfloat16_rn(p1));
                    hw[e] = pack_bf16(h0, h1);
                    lw[e] = pack_bf16(p0 - h0, p1 - h1);
                }
                const int chunk = (c8 ^ (r & 7)) << 4;
                *reinterpret_cast<uint4 *>(prow_hi + chunk) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
                *reinterpret_cast<uint4 *>(prow_lo + chunk) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
            }
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            tc_fence_before();
            mbar_arrive(smem_u32(&bars[B_P_FULL]));
        }
        if (ok) ok = __all_sync(0xFFFFFFFFu, mbar_wait(smem_u32(&bars[B_PV_DONE]), (n_kt - 1) & 1));
        if (ok) {
            tc_fence_after();
            const float inv = l > 0.f ? 1.f / l : 0.f;
            TOut *out = reinterpret_cast<TOut *>(a.out) + (((int64_t)s * a.N + (row_ok ? i : 0)) * a.Hq + h) * DT;
            float ov[32];
#pragma unroll
            for (int c4 = 0; c4 < DT / 32; ++c4) {
                tmem_ld32(t_o + lane_off + 32 * c4, ov);
                if (row_ok) {
#pragma unroll
                    for (int c = 0; c < 32; ++c) ov[c] *= inv;
#pragma unroll
                    for (int e = 0; e < 4; ++e) store8<TOut>(out + 32 * c4 + 8 * e, ov + 8 * e);
                }
            }
            if (row_ok && a.lse != nullptr)
                a.lse[((int64_t)s * a.Hq + h) * a.N + i] = (m_used + __log2f(l)) * kLn2;
        }
    }

    if (!ok) atomicOr(&g_ris_tile_error, 2u);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 5)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
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

// [N][H][128] bf16 viewed as 3D (d, head, token); box = 64 d x 1 head x `rows` tokens.
bool make_map3(CUtensorMap *m, const void *base, int64_t N, int H, int rows)
{
    auto fn = encode_fn();
    if (fn == nullptr) return false;
    cuuint64_t dims[3] = {(cuuint64_t)DT, (cuuint64_t)H, (cuuint64_t)N};
    cuuint64_t strides[2] = {(cuuint64_t)DT * 2, (cuuint64_t)H * DT * 2};
    cuuint32_t box[3] = {64, 1, (cuuint32_t)rows};
    cuuint32_t estr[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <bool SPLIT, bool DENSE, typename TOut>
cudaError_t launch_t(const AttnArgs &a, const TileMaps &maps, cudaStream_t s)
{
    auto kern = k_attn_tile<SPLIT, DENSE, TOut>;
    static bool attr = false;
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    const int64_t n_qt = (a.N + BM - 1) / BM;
    const unsigned grid = (unsigned)(n_qt * a.Hq * a.n_sets);
    kern<<<grid, kThreads, SMEM_BYTES, s>>>(a, maps);
    note_launch();
    return cudaGetLastError();
}

}  // namespace

bool tile_design_available() { return encode_fn() != nullptr; }

// Read and clear this kernel's device error word (the caller has synchronised).
cudaError_t read_tile_error(unsigned int *out)
{
    cudaError_t e = cudaMemcpyFromSymbol(out, g_ris_tile_error, sizeof(unsigned int));
    if (e != cudaSuccess || *out == 0u) return e;
    const unsigned int zero = 0u;
    return cudaMemcpyToSymbol(g_ris_tile_error, &zero, sizeof(unsigned int));
}

// q_hi / q_lo: queries as a bf16 pair [N][Hq][128] (q_lo null: exact bf16 queries and keys,
// one score product); a.k / a.k_lo: keys as a pair; a.v: values. Head dim 128 only.
cudaError_t launch_attention_tile(const AttnArgs &a, const void *q_hi, const void *q_lo, int out_dtype, bool dense,
                                  cudaStream_t s)
{
    static std::mutex mu;
    std::lock_guard<std::mutex> lk(mu);
    const bool split = q_lo != nullptr;
    alignas(64) TileMaps maps;
    if (!make_map3(&maps.qh, q_hi, a.N, a.Hq, BM) || !make_map3(&maps.kh, a.k, a.N, a.Hkv, BN) ||
        !make_map3(&maps.v, a.v, a.N, a.Hkv, BN))
        return cudaErrorInvalidValue;
    if (split) {
        if (!make_map3(&maps.ql, q_lo, a.N, a.Hq, BM) || !make_map3(&maps.kl, a.k_lo, a.N, a.Hkv, BN))
            return cudaErrorInvalidValue;
    } else {
        maps.ql = maps.qh;
        maps.kl = maps.kh;
    }
    if (out_dtype == RIS_F32) {
        if (split) return dense ? launch_t<true, true, float>(a, maps, s) : launch_t<true, false, float>(a, maps, s);
        return dense ? launch_t<false, true, float>(a, maps, s) : launch_t<false, false, float>(a, maps, s);
    }
    if (split)
        return dense ? launch_t<true, true, __nv_bfloat16>(a, maps, s) : launch_t<true, false, __nv_bfloat16>(a, maps, s);
    return dense ? launch_t<false, true, __nv_bfloat16>(a, maps, s) : launch_t<false, false, __nv_bfloat16>(a, maps, s);
}

}  // namespace ris
