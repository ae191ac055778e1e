// RIS sparse attention, masked dense-tile design on the 5th-generation tensor cores
// (paper, Methods, "Hybrid Anchor and Pre-Fusion Unified Softmax (PFUS)"; the dense causal
// upper bound of Table tab:results_32k is the same kernel with every causal pair kept).
//
// Where the master mask keeps a large share of the causal pairs (union densities of tens of
// percent, and the dense mode) a dense 128 x 128 score tile with the mask applied as -inf
// beats gathering rows pair by pair. One CTA owns one (128-query tile, query head, set):
//
//   warp 8 (TMA)   streams 128-key tiles of the keys (64 KB: hi parts and corrections) and of
//                  the values (fp16, 32 KB) in 128-byte swizzled boxes into two two-stage
//                  shared-memory rings: a key stage is refilled as soon as its score products
//                  are done, a value stage once its value product is; it also waits for each
//                  tile's values to land and then arrives on that tile's P_FULL barrier, so
//                  that the MMA warp waits once per value product;
//   warp 9 (MMA)   one elected lane issues tcgen05.mma: the score tile S (A = the query tile,
//                  kept in TMEM) into a double-buffered TMEM score tile, and O += P V (A = P
//                  as fp16, written into TMEM over the consumed scores) into the TMEM output
//                  tile, committing each step to an mbarrier; TMEM holds S/P twice (2 x 128
//                  columns), O (128) and the query operands (128), all 512 columns;
//   warps 0-7      two threads per query row (score and output columns 0-63 / 64-127): write
//                  the row's query part into TMEM, then per tile tcgen05.ld the scores, apply
//                  the bitmap (words fetched three tiles ahead) or the causal cut, exchange the
//                  partial row max with the partner thread, fp32 online softmax with lazy
//                  rescaling of O in TMEM (only when the row max grows by more than 2^8),
//                  write P into TMEM, and at the end normalise O (and undo the values'
//                  power-of-two scale) and store the row.
//
// Precision. With activation outlier channels the scores reach tens of units while the
// output moves by p (v_j - o) per unit of score error, so the scores need about 17
// significant bits. At head dim 128 with rotated inputs (the operands written by
// launch_fp8_prep) S = q_h k_h + 2^-12 (e4m3(q_h) e4m3(k_l) + e4m3(q_l) e4m3(k_h)) with fp16
// hi parts and power-of-two scales taken from bounds of |q~| and |k~| (fp8_score_scales): the
// two e4m3 products (kind::f8f6f4, twice the rate) go first and the fp16 product folds them in
// with scale-input-d; max-abs about 7e-3 in CPU emulation. Where the bounds rule that out, at
// head dim 64, and for inputs not rotated here, S = Q_hi K_hi^T + Q_lo K_hi^T + Q_hi K_lo^T
// with bf16 hi + lo pairs. One fp16 key product alone moves outputs by up to 0.1. P enters the
// value product as one fp16 (11 significant bits; max-abs 6.5e-3 in the same emulation
// against 1.7e-3 for a bf16 hi + lo pair), and the row sum adds P as rounded, so that each
// weight's rounding moves the output by at most 2^-11 of that weight times |v_j - o|. The
// values are exact in fp16 after a power-of-two scale (none unless some |v| reaches 2^14),
// undone in the epilogue.
//
// Measured: a tile pair takes 24 slots of 16-bit product time (8 fp16 score products, 2 x 4
// e4m3 corrections at twice the rate, 8 fp16 value products); C5's Stochastic layer at 64k
// runs in 13.3-13.5 ms per launch (16.4 ms with three bf16 score products, 19.6 with a bf16 P
// pair as well). What holds the pipe below its rate is the MMA warp's own time between issues
// (each mbarrier wait costs its thread about 100 cycles even on a completed phase, and the
// issue blocks until the pipe takes each product) and, with a bitmap, the softmax's wait for
// the bitmap words: so the MMA warp waits on one barrier before a tile's score products (the
// keys; the score buffer's reuse is implied by the P_FULL it waited on two tiles before) and
// one before its value product, and the bitmap words come three tiles ahead. Four threads per
// row (16 softmax warps) measured the same as two. 128-key tiles with the query in TMEM beat
// 64-key tiles with the query in shared memory.
//
// The suffix pass of the dense-suffix split (SUFFIX) runs the same pipeline over the key
// tiles of each row's dense suffix only (its Structural block and / or local window: every key
// kept, no bitmap), and writes the normalised partial output and its log-sum-exp for the
// register gather to continue from.
//
// Every mbarrier wait is bounded; a wait that gives up sets bit 1 of the device error word,
// every role falls through to the end, TMEM is released and the CTA returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cstdint>
#include <mutex>

#include "attn_common.cuh"

namespace ris {

// Device error word of this kernel (bit 1: a bounded wait gave up); read by read_tile_error.
__device__ unsigned int g_ris_tile_error;

namespace {

constexpr int BM = 128;          // query rows per tile (TMEM lanes)
constexpr int BN = 128;          // keys per stage
// Softmax: kRowThreads threads per query row, each owning BN / kRowThreads score columns of
// every tile and DT / kRowThreads output columns; 4 warps cover the 128 TMEM lanes, so there
// are 4 * kRowThreads softmax warps (four per SM sub-partition, to hide the latency of each
// warp's dependent TMEM load -> max exchange -> exp -> TMEM store chain), then the TMA and MMA warps.
constexpr int kRowThreads = 2;
// P as one fp16 (11 significant bits, one value product against fp16 values) instead of a
// bf16 hi + lo pair (two value products against bf16 values)
constexpr bool kP16 = true;
constexpr int kSoftmaxWarps = 4 * kRowThreads;
constexpr int kSoftmaxThreads = 32 * kSoftmaxWarps;
constexpr int kTmaWarp = kSoftmaxWarps, kMmaWarp = kSoftmaxWarps + 1;
constexpr int kThreads = 32 * (kSoftmaxWarps + 2);
constexpr uint32_t kTmemCols = 512;  // S/P[2] (2 x 128) + O (128) + Q hi / lo (2 x 64)

// shared-memory map (bytes, from a 1024-aligned base) for head dim DT (128 or 64)
template <int DT>
struct Smem {
    static constexpr int KV_ARR = BN * DT * 2;  // 32 KB at DT = 128: one of K hi / K lo / V
    static constexpr int K_STAGE = 2 * KV_ARR;  // K hi, K lo
    static constexpr int V_STAGE = KV_ARR;
};
constexpr int KV_BLK = BN * 128;            // 16 KB: one 64-column block
constexpr int kStages = 2;                  // stages of each ring
constexpr int OFF_K = 0;
// the head-dim-128 layout (197632 bytes with the alignment slack) is requested at either
// head dim: it keeps one CTA per SM, as the CTA holds all 512 TMEM columns
constexpr int SMEM_BYTES = OFF_K + kStages * (Smem<128>::K_STAGE + Smem<128>::V_STAGE) + 1024;

// P_FULL and PV_DONE have one barrier per P buffer (tile parity), so that no waiter can fall
// two phases behind a barrier it polls by parity.
// B_X: per group of kRowThreads softmax warps sharing rows (one per column quarter) and tile
// parity, the exchange of their partial row maxima (and at the end their partial sums).
enum Bar {
    B_Q = 0, B_K_FULL = 1, B_V_FULL = 3, B_S_FULL = 5, B_P_FULL = 7, B_PV_DONE = 9, B_X = 11, B_END = 19, NBAR = 20
};

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
// Bounded wait for this CTA's own asynchronous work (copies or products already issued):
// about 2^31 cycles at most, whatever other CTAs reported.
__device__ __forceinline__ bool mbar_wait_own(uint32_t bar, uint32_t parity)
{
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity))
        if (clock64() - t0 > (1LL << 31)) return false;
    return true;
}

// Bounded wait (`limit` cycles, about 2^31 unless a test lowers it); false if the phase did
// not complete in time or another CTA already gave up.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, long long limit)
{
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity)) {
        if (clock64() - t0 > limit) return false;
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

// Instruction descriptor, kind::f16: fp16 x fp16 -> f32, dense.
__host__ __device__ constexpr uint32_t idesc_f16(int M, int N, bool b_mn_major)
{
    return (1u << 4)                      // D format f32 (A and B format 0: fp16)
           | ((b_mn_major ? 1u : 0u) << 16)
           | ((uint32_t)(N >> 3) << 17)
           | ((uint32_t)(M >> 4) << 24);
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

// A operand from TMEM (rows in lanes, 16-bit values packed two per column), B from shared memory.
__device__ __forceinline__ void tc_mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t idesc, uint32_t acc)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}

// kind::f8f6f4 (e4m3 x e4m3 with the instruction descriptor's format fields 0), A from TMEM
// (four 8-bit values per column), B from shared memory.
__device__ __forceinline__ void tc_mma_ts_f8(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t idesc, uint32_t acc)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}

// kind::f16 accumulating onto D scaled by 2^-12 on entry: D = A B + 2^-12 D.
__device__ __forceinline__ void tc_mma_ts_scaled12(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t idesc)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, 1, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p, 12;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(idesc)
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

// 32 lanes x 64 consecutive 32-bit columns, loaded and waited for in one statement (the
// registers are defined only once the wait has passed).
__device__ __forceinline__ void tmem_ld64(uint32_t taddr, float *v)
{
    uint32_t r[64];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x64.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [%64];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]), "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]), "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 64; ++i) v[i] = __uint_as_float(r[i]);
}

// 32 lanes x 16 consecutive 32-bit columns, loaded and waited for in one statement.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float *v)
{
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n\t"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Two 16-column stores (32 lanes each) and one wait for both.
__device__ __forceinline__ void tmem_st16x2(uint32_t ta, const uint32_t *a, uint32_t tb, const uint32_t *b)
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17};\n\t"
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%1], {%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32,%33};\n\t"
        "tcgen05.wait::st.sync.aligned;" ::"r"(ta), "r"(tb),
        "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(a[4]), "r"(a[5]), "r"(a[6]), "r"(a[7]), "r"(a[8]), "r"(a[9]),
        "r"(a[10]), "r"(a[11]), "r"(a[12]), "r"(a[13]), "r"(a[14]), "r"(a[15]),
        "r"(b[0]), "r"(b[1]), "r"(b[2]), "r"(b[3]), "r"(b[4]), "r"(b[5]), "r"(b[6]), "r"(b[7]), "r"(b[8]), "r"(b[9]),
        "r"(b[10]), "r"(b[11]), "r"(b[12]), "r"(b[13]), "r"(b[14]), "r"(b[15])
        : "memory");
}

__device__ __forceinline__ void tmem_st8(uint32_t taddr, const uint32_t *v)
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr), "r"(v[0]), "r"(v[1]),
        "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7])
        : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t *v)
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
        "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
        : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_st32u(uint32_t taddr, const uint32_t *v)
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
        "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]), "r"(v[16]), "r"(v[17]), "r"(v[18]),
        "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]), "r"(v[25]), "r"(v[26]), "r"(v[27]),
        "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])
        : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// NC consecutive 32-bit columns (64, 32 or 16) of 32 lanes, loaded and waited for.
template <int NC>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, float *v)
{
    if constexpr (NC == 64)
        tmem_ld64(taddr, v);
    else if constexpr (NC == 32)
        tmem_ld32(taddr, v);
    else {
        static_assert(NC == 16, "64, 32 or 16 columns");
        tmem_ld16(taddr, v);
    }
}

// NC consecutive 32-bit columns (32, 16 or 8) of 32 lanes, stored and waited for.
template <int NC>
__device__ __forceinline__ void tmem_st_words(uint32_t taddr, const uint32_t *w)
{
    if constexpr (NC == 32)
        tmem_st32u(taddr, w);
    else if constexpr (NC == 16)
        tmem_st16(taddr, w);
    else {
        static_assert(NC == 8, "32, 16 or 8 columns");
        tmem_st8(taddr, w);
    }
}

// max of three floats in one instruction
__device__ __forceinline__ float fmax3(float x, float y, float z)
{
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(x), "f"(y), "f"(z));
    return d;
}

// 2^x by the SFU (ex2.approx, relative error about 2^-22, subnormal results flushed to 0);
// 2^-inf = 0.
__device__ __forceinline__ float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
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
    CUtensorMap kh, kl, v;
};

template <int DT, bool SPLIT, bool DENSE, bool SUFFIX, typename TOut>
__global__ void __launch_bounds__(kThreads, 1)
    k_attn_tile(const AttnArgs a, const __grid_constant__ TileMaps maps, const void *q_hi, const void *q_lo)
{
    static_assert(DT == 128 || DT == 64, "head dim 64 or 128");
    constexpr int KV_ARR = Smem<DT>::KV_ARR, K_STAGE = Smem<DT>::K_STAGE, V_STAGE = Smem<DT>::V_STAGE;
    constexpr int OFF_V = OFF_K + kStages * K_STAGE;
    constexpr int NB = DT / 64;  // 64-column blocks of a row
    extern __shared__ unsigned char smem_raw[];
    __shared__ __align__(8) uint64_t bars[NBAR];
    __shared__ uint32_t tmem_base_sh;
    __shared__ float xch[2][kRowThreads][BM];  // [tile parity][column quarter][row]
    unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                            ~uintptr_t(1023));
    const uint32_t sbase = smem_u32(smem);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // ---- tile of this CTA (tiles covering rows row0 .. row1-1): heavier (later) tiles first
    const int qt_end = (int)((a.row1 + BM - 1) / BM);
    const int64_t b = blockIdx.x;
    const int h = (int)(b % a.Hq);
    const int64_t r2 = b / a.Hq;
    const int s = (int)(r2 % a.n_sets);
    const int qt = qt_end - 1 - (int)(r2 / a.n_sets);
    const int64_t q0 = (int64_t)qt * BM;
    const int g = h / a.G;
    const int mask_id = s * a.heads_keyed + (a.heads_keyed > 1 ? g : 0);
    const int64_t last_row = (q0 + BM - 1 < a.row1 - 1) ? q0 + BM - 1 : a.row1 - 1;
    // causal: key tiles kt0 .. last_row / BN (kt0 = 0, or the tile of the first row's dense
    // suffix start, the earliest of the tile's rows)
    const int kt0 = SUFFIX ? (int)(dense_suffix_start(a, q0) / BN) : 0;
    const int n_kt = (int)(last_row / BN) + 1 - kt0;

    if (threadIdx.x == 0) {
        for (int i = 0; i < NBAR; ++i) {
            uint32_t cnt = 1;
            if (i == B_Q) cnt = kSoftmaxThreads;
            if (i == B_P_FULL || i == B_P_FULL + 1) cnt = kSoftmaxThreads + 1;  // + the loader's relay
            if (i >= B_X && i < B_END) cnt = 32 * kRowThreads;
            mbar_init(smem_u32(&bars[i]), cnt);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == kMmaWarp) {  // TMEM allocation by one full warp
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&tmem_base_sh)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base_sh;
    const uint32_t t_s0 = tmem, t_s1 = tmem + BN, t_o = tmem + 2 * BN, t_q = tmem + 2 * BN + DT;
    const long long wl = a.wait_limit > 0 ? (long long)a.wait_limit : (1LL << 31);
    bool ok = true;

    if (warp == kTmaWarp) {
        // =============================== TMA producer
        if (lane == 0 && a.debug_no_loads == 0) {
            // tile j: keys once the score products of tile j - 2 are done, then values once the
            // value product of tile j - 2 is (it was issued after the score products of tile
            // j - 1, whose keys are already in flight: no wait here depends on a later load).
            // The ring stages and the score / P buffers are both indexed by tile parity, so a
            // stage is free exactly when the barrier that announces those products completes
            // (S_FULL, PV_DONE): the loader waits on them instead of on barriers of its own,
            // which saves the tensor pipe two commits per tile.
            // The loader also waits for each tile's values to land and then arrives on that tile's
            // P_FULL (which counts the softmax threads and this one), so that the MMA warp waits
            // once before a value product instead of twice: each wait costs its issuing thread
            // about 100 cycles even on a completed phase, and the tensor pipe idles meanwhile.
            static_assert(kStages == 2, "ring stages share the parity of the score buffers");
            int nk = 0, nv = 0, nr = 0;  // tiles whose keys / values were requested; values relayed
            auto relay = [&](int jv) -> bool {
                if (!mbar_wait(smem_u32(&bars[B_V_FULL + jv % kStages]), (jv / kStages) & 1, wl)) return false;
                mbar_arrive(smem_u32(&bars[B_P_FULL + (jv & 1)]));
                nr = jv + 1;
                return true;
            };
            for (int j = 0; j < n_kt && ok; ++j) {
                const int st = j % kStages;
                const uint32_t par = ((j / kStages) - 1) & 1;
                if (j >= kStages) ok = mbar_wait(smem_u32(&bars[B_S_FULL + st]), par, wl);
                if (!ok) break;
                const uint32_t bk = smem_u32(&bars[B_K_FULL + st]);
                const uint32_t dk = sbase + OFF_K + st * K_STAGE;
                mbar_arrive_expect_tx(bk, (SPLIT ? 2 : 1) * KV_ARR);
                for (int blk = 0; blk < NB; ++blk) {
                    tma_load_3d(dk + blk * KV_BLK, &maps.kh, 64 * blk, g, (kt0 + j) * BN, bk);
                    if (SPLIT) tma_load_3d(dk + KV_ARR + blk * KV_BLK, &maps.kl, 64 * blk, g, (kt0 + j) * BN, bk);
                }
                nk = j + 1;
                if (j >= 1) ok = relay(j - 1);
                if (!ok) break;
                if (j >= kStages) ok = mbar_wait(smem_u32(&bars[B_PV_DONE + st]), par, wl);
                if (!ok) break;
                const uint32_t bv = smem_u32(&bars[B_V_FULL + st]);
                const uint32_t dv = sbase + OFF_V + st * V_STAGE;
                mbar_arrive_expect_tx(bv, KV_ARR);
                for (int blk = 0; blk < NB; ++blk) tma_load_3d(dv + blk * KV_BLK, &maps.v, 64 * blk, g, (kt0 + j) * BN, bv);
                nv = j + 1;
            }
            if (ok && nv == n_kt && nr < nv) ok = relay(nv - 1);
            // let the copies requested last into each stage land before the CTA can leave
            // (earlier ones were consumed before their stage was refilled)
            for (int j = nk - kStages; j < nk; ++j)
                if (j >= 0) mbar_wait_own(smem_u32(&bars[B_K_FULL + j % kStages]), (j / kStages) & 1);
            for (int j = nv - kStages; j < nv; ++j)
                if (j >= 0) mbar_wait_own(smem_u32(&bars[B_V_FULL + j % kStages]), (j / kStages) & 1);
        }
    } else if (warp == kMmaWarp) {
        // =============================== MMA issuer
        if (lane == 0) {
            constexpr uint32_t ID_S = idesc_bf16(BM, BN, false);  // S[128 x 128] = Q K^T, both K-major
            // O[128 x DT] += P V, V MN-major (fp16 P against fp16 values, or bf16 P hi / lo
            // against bf16 values)
            constexpr uint32_t ID_O = kP16 ? idesc_f16(BM, DT, true) : idesc_bf16(BM, DT, true);
            // fp8-correction scores (rotated q / k at head dim 128, operands written by
            // launch_fp8_prep when the bounds allow): the same bytes in the same places as the
            // bf16 pair, read as fp16 hi parts (query columns 0-63, key bytes 0-255 of a row) and
            // e4m3 corrections (query columns 64-95 / 96-127, key boxes at KV_ARR / KV_ARR + KV_BLK)
            int ea = 0, eb = 0;
            const bool use8 = DT == 128 && SPLIT && a.qk_bound != nullptr &&
                              fp8_score_scales(a.qk_bound[0], a.qk_bound[1], ea, eb);
            constexpr uint32_t ID_SH = idesc_f16(BM, BN, false);  // fp16 x fp16 (and e4m3 x e4m3 for kind::f8f6f4)
            ok = mbar_wait(smem_u32(&bars[B_Q]), 0, wl);
            tc_fence_after();
            auto issue_s = [&](int j) {
                const int st = j & 1;
                const uint32_t kv = sbase + OFF_K + (j % kStages) * K_STAGE;
                const uint32_t dt = (j & 1) ? t_s1 : t_s0;
                uint32_t acc = 0;
                if (use8) {
                    // 2^12 (q_h8 k_l8 + q_l8 k_h8): two e4m3 products of 4 k-steps of 32
                    for (int prod = 0; prod < 2; ++prod) {
                        const uint32_t qa = t_q + DT / 2 + (prod == 0 ? 0 : DT / 4);
                        const uint32_t kb = kv + KV_ARR + (prod == 0 ? KV_BLK : 0);
                        for (int ks = 0; ks < DT / 32; ++ks) {
                            tc_mma_ts_f8(dt, qa + 8 * ks, sdesc(kb + ks * 32, 16, 1024), ID_SH, acc);
                            acc = 1;
                        }
                    }
                    // + q_h k_h in fp16, the corrections brought back by 2^-12 on the first k-step
                    for (int ks = 0; ks < DT / 16; ++ks) {
                        const uint64_t bd = sdesc(kv + (ks >> 2) * KV_BLK + (uint32_t)((ks & 3) * 32), 16, 1024);
                        if (ks == 0)
                            tc_mma_ts_scaled12(dt, t_q, bd, ID_SH);
                        else
                            tc_mma_ts(dt, t_q + 8 * ks, bd, ID_SH, 1u);
                    }
                    tc_commit(smem_u32(&bars[B_S_FULL + st]));
                    return;
                }
                // (A, B) pairs: (Q hi, K hi), (Q lo, K hi), (Q hi, K lo); 8 k-steps of 16 over D
                // the query tile lives in TMEM (16-bit values packed two per column): A from TMEM
                for (int prod = 0; prod < (SPLIT ? 3 : 1); ++prod) {
                    const uint32_t qa = t_q + (prod == 1 ? DT / 2 : 0);
                    const uint32_t kb = kv + (prod == 2 ? KV_ARR : 0);
                    for (int ks = 0; ks < DT / 16; ++ks) {
                        const uint32_t koff = (uint32_t)((ks & 3) * 32);  // 16 columns = 32 B inside a 128 B row
                        const uint64_t bd = sdesc(kb + (ks >> 2) * KV_BLK + koff, 16, 1024);
                        tc_mma_ts(dt, qa + 8 * ks, bd, ID_S, acc);
                        acc = 1;
                    }
                }
                tc_commit(smem_u32(&bars[B_S_FULL + st]));
            };
            auto issue_o = [&](int j) {
                const int st = j % kStages;
                const uint32_t vb = sbase + OFF_V + st * V_STAGE;
                // P of this tile sits in TMEM over its score columns: 128 keys of 16-bit values
                // packed two per column, in columns 0-63 (fp16 P, or the bf16 hi part) and 64-127
                // (the bf16 lo part)
                const uint32_t pt = (j & 1) ? t_s1 : t_s0;
                for (int prod = 0; prod < (kP16 ? 1 : 2); ++prod) {
                    for (int ks = 0; ks < BN / 16; ++ks) {
                        // V block: 64 keys x 128 B rows; 16 keys = two 8-row atoms (SBO 1024);
                        // the second 64-column block of head dim is LBO = 8 KB away
                        const uint64_t bd = sdesc(vb + ks * 2048, KV_BLK, 1024);
                        tc_mma_ts(t_o, pt + (BN / 2) * prod + 8 * ks, bd, ID_O, (j > 0 || prod > 0 || ks > 0) ? 1u : 0u);
                    }
                }
                tc_commit(smem_u32(&bars[B_PV_DONE + (j & 1)]));
            };
            for (int j = 0; j < n_kt && ok; ++j) {
                // the score buffer j & 1 held P of tile j - 2, and P_FULL of that tile (waited for
                // before its value product) came after the softmax threads had read its scores:
                // so only the keys are waited for here
                ok = mbar_wait(smem_u32(&bars[B_K_FULL + j % kStages]), (j / kStages) & 1, wl);
                if (!ok) break;
                tc_fence_after();
                issue_s(j);
                if (j >= 1) {
                    // P of tile j - 1 written and its values landed (relayed by the loader)
                    ok = mbar_wait(smem_u32(&bars[B_P_FULL + ((j - 1) & 1)]), ((j - 1) >> 1) & 1, wl);
                    if (!ok) break;
                    tc_fence_after();
                    issue_o(j - 1);
                }
            }
            if (ok) {
                ok = mbar_wait(smem_u32(&bars[B_P_FULL + ((n_kt - 1) & 1)]), ((n_kt - 1) >> 1) & 1, wl);
                if (ok) {
                    tc_fence_after();
                    issue_o(n_kt - 1);
                }
            }
            // every product issued has to finish before TMEM is released
            tc_commit(smem_u32(&bars[B_END]));
            mbar_wait_own(smem_u32(&bars[B_END]), 0);
        }
    } else {
        // =============================== softmax: kRowThreads threads per query row q0 + r,
        // thread cq owning score columns SC cq .. SC cq + SC - 1 of every tile and output
        // columns OC cq .. OC cq + OC - 1
        constexpr int SC = BN / kRowThreads;   // scores of a tile per thread (64 or 32)
        constexpr int OC = DT / kRowThreads;   // output columns per thread (64, 32 or 16)
        constexpr int OCH = OC < 32 ? OC : 32; // output columns per TMEM access
        const int wq = warp & 3, cq = warp >> 2;
        const int r = wq * 32 + lane;  // TMEM lane
        const int64_t i = q0 + r;
        const bool row_ok = i >= a.row0 && i < a.row1;
        const uint32_t lane_off = (uint32_t)(wq * 32) << 16;
        const uint32_t *bm = (DENSE || SUFFIX) ? nullptr
                                               : a.bitmap + (int64_t)mask_id * a.words_per_mask + (row_ok ? row_word_offset(i) : 0);
        const int64_t last_word = i >> 5;
        const float sc = a.scale_log2;
        float m_used = -INFINITY, l = 0.f;
        // bitmap word e of keys 128 (kt0 + j) + SC cq + 32 e .. +31 of this row, fetched one
        // tile ahead
        auto mask_word = [&](int j, int e) -> uint32_t {
            if (!row_ok) return 0u;
            const int64_t k0 = (int64_t)(kt0 + j) * BN + SC * cq + 32 * e;
            if (SUFFIX) {  // the row's dense suffix: offsets lo .. hi of the word
                const int64_t lo = dense_suffix_start(a, i) - k0, hi = i - k0;
                if (hi < 0 || lo > 31) return 0u;
                uint32_t w = hi >= 31 ? 0xFFFFFFFFu : ((2u << hi) - 1u);
                if (lo > 0) w &= ~((1u << lo) - 1u);
                return w;
            }
            if (DENSE) {
                const int64_t lim = i - k0;  // keys k0 .. i are kept
                return lim >= 31 ? 0xFFFFFFFFu : (lim < 0 ? 0u : ((2u << lim) - 1u));
            }
            const int64_t wd = k0 >> 5;
            return wd <= last_word ? bm[wd] : 0u;
        };
        // exchange a value with the other threads of the row (bounded wait); v[q] = the value of
        // column part q, in the same order for every thread of the row
        auto exchange = [&](int tag, float mine, float *v) -> bool {
            const int pb = tag & 1;
            xch[pb][cq][r] = mine;
            const uint32_t bar = smem_u32(&bars[B_X + 2 * wq + pb]);
            mbar_arrive(bar);
            const bool got = __all_sync(0xFFFFFFFFu, mbar_wait(bar, (tag >> 1) & 1, wl));
#pragma unroll
            for (int qq = 0; qq < kRowThreads; ++qq) v[qq] = xch[pb][qq][r];
            return got;
        };
        // this thread's part of the query row (head-dim OC cq .. OC cq + OC - 1, OC / 2 packed
        // columns of each of hi and lo) into TMEM
        {
            uint32_t qw[OC / 2];
            const int64_t qrow = ((row_ok ? i : 0) * a.Hq + h) * DT + OC * cq;
            for (int part = 0; part < (SPLIT ? 2 : 1); ++part) {
                const uint4 *src = reinterpret_cast<const uint4 *>(
                    reinterpret_cast<const __nv_bfloat16 *>(part == 0 ? q_hi : q_lo) + qrow);
#pragma unroll
                for (int u = 0; u < OC / 8; ++u) {
                    const uint4 x = row_ok ? src[u] : make_uint4(0u, 0u, 0u, 0u);
                    qw[4 * u] = x.x;
                    qw[4 * u + 1] = x.y;
                    qw[4 * u + 2] = x.z;
                    qw[4 * u + 3] = x.w;
                }
                const uint32_t tq = t_q + lane_off + (DT / 2) * part + (OC / 2) * cq;
#pragma unroll
                for (int c = 0; c < OC / 2; c += (OC / 2 < 16 ? OC / 2 : 16))
                    tmem_st_words<(OC / 2 < 16 ? OC / 2 : 16)>(tq + c, qw + c);
            }
            tc_fence_before();
            mbar_arrive(smem_u32(&bars[B_Q]));
        }
        // bitmap words fetched three tiles ahead (one tile ahead left part of a DRAM miss exposed:
        // two ahead gained 3.5% at 64k, three 1-2% more)
        uint32_t cw[SC / 32], nw[SC / 32], n2w[SC / 32];
#pragma unroll
        for (int e = 0; e < SC / 32; ++e) {
            cw[e] = mask_word(0, e);
            nw[e] = (1 < n_kt) ? mask_word(1, e) : 0u;
            n2w[e] = (2 < n_kt) ? mask_word(2, e) : 0u;
        }
        for (int j = 0; j < n_kt; ++j) {
            const int st = j & 1;
            uint32_t nnw[SC / 32];
#pragma unroll
            for (int e = 0; e < SC / 32; ++e) nnw[e] = (j + 3 < n_kt) ? mask_word(j + 3, e) : 0u;
            ok = __all_sync(0xFFFFFFFFu, mbar_wait(smem_u32(&bars[B_S_FULL + st]), (j >> 1) & 1, wl));
            if (!ok) break;
            tc_fence_after();
            float sv[SC];
            const uint32_t sb = ((j & 1) ? t_s1 : t_s0) + lane_off + SC * cq;
            tmem_ld_cols<SC>(sb, sv);
            tc_fence_before();

            // mask, partial row max as a tree (the scale is positive: it is applied to the max
            // and folded into the exponent of P), then the full row max from the other threads
#pragma unroll
            for (int e = 0; e < SC / 32; ++e) {
#pragma unroll
                for (int c = 0; c < 32; ++c) sv[32 * e + c] = ((cw[e] >> c) & 1u) ? sv[32 * e + c] : -INFINITY;
                cw[e] = nw[e];
                nw[e] = n2w[e];
                n2w[e] = nnw[e];
            }
            float mx9[9];
#pragma unroll
            for (int e = 0; e < 9; ++e) {
                mx9[e] = sv[e];
#pragma unroll
                for (int c = e + 9; c < SC; c += 18)
                    mx9[e] = c + 9 < SC ? fmax3(mx9[e], sv[c], sv[c + 9]) : fmaxf(mx9[e], sv[c]);
            }
            const float pm = fmax3(fmax3(mx9[0], mx9[1], mx9[2]), fmax3(mx9[3], mx9[4], mx9[5]),
                                   fmax3(mx9[6], mx9[7], mx9[8])) * sc;
            float pms[kRowThreads];
            ok = exchange(j, pm, pms);
            if (!ok) break;
            float mx = pms[0];
#pragma unroll
            for (int qq = 1; qq < kRowThreads; ++qq) mx = fmaxf(mx, pms[qq]);
            // Lazy rescale: a row rescales O only when its max grows by more than 2^8 (all
            // threads of the row see the same max and decide alike). The TMEM loads / stores
            // are warp-collective (.sync.aligned), so the whole warp runs them when any of its
            // rows needs it; the other rows multiply by 1.
            const bool upd = mx > m_used + 8.f;
            const float al = upd ? (m_used == -INFINITY ? 0.f : exp2f(m_used - mx)) : 1.f;
            if (upd) {
                l *= al;
                m_used = mx;
            }
            if (__any_sync(0xFFFFFFFFu, upd && al != 0.f)) {
                // O must have settled: the value product of tile j - 1 has to be done
                if (j >= 1) {
                    ok = __all_sync(0xFFFFFFFFu,
                                    mbar_wait(smem_u32(&bars[B_PV_DONE + ((j - 1) & 1)]), ((j - 1) >> 1) & 1, wl));
                    if (!ok) break;
                }
                tc_fence_after();
#pragma unroll
                for (int c0 = 0; c0 < OC; c0 += OCH) {
                    float ov[OCH];
                    uint32_t ow[OCH];
                    tmem_ld_cols<OCH>(t_o + lane_off + OC * cq + c0, ov);
#pragma unroll
                    for (int c = 0; c < OCH; ++c) ow[c] = __float_as_uint(ov[c] * al);
                    tmem_st_words<OCH>(t_o + lane_off + OC * cq + c0, ow);
                }
            }
            const float mu = (m_used == -INFINITY) ? 0.f : m_used;
            // P = exp2(s - m_used), written into TMEM over this tile's score columns (every
            // thread of the row has read its scores: the max exchange came first) as the A
            // operand of the value product, keys SC cq .. SC cq + SC - 1 in packed columns
            // (SC / 2) cq .. (SC / 2) cq + SC / 2 - 1 (and the bf16 lo part 64 columns on).
            // fp16 P: the row sum adds P as rounded, so that the rounding of each weight moves
            // the output by at most 2^-11 of the weight times |v_j - o| (a normalised average
            // of the values with slightly perturbed weights). bf16 pair: hi = p with its low 16
            // bits cleared (exactly a bf16), lo = p - hi rounded to bf16 (~16 significant bits).
            float lsum[4] = {0.f, 0.f, 0.f, 0.f};
            uint32_t hw[SC / 2];
            const uint32_t pt = ((j & 1) ? t_s1 : t_s0) + lane_off;
            if constexpr (kP16) {
#pragma unroll
                for (int w = 0; w < SC / 2; ++w) {
                    const float p0 = ex2(fmaf(sv[2 * w], sc, -mu)), p1 = ex2(fmaf(sv[2 * w + 1], sc, -mu));
                    const __half2 hp = __floats2half2_rn(p0, p1);
                    const float2 pr = __half22float2(hp);
                    lsum[w & 3] += pr.x + pr.y;
                    hw[w] = *reinterpret_cast<const uint32_t *>(&hp);
                }
#pragma unroll
                for (int c = 0; c < SC / 2; c += 16) tmem_st16(pt + (SC / 2) * cq + c, hw + c);
            } else {
                uint32_t lw[SC / 2];
#pragma unroll
                for (int w = 0; w < SC / 2; ++w) {
                    const float p0 = ex2(fmaf(sv[2 * w], sc, -mu)), p1 = ex2(fmaf(sv[2 * w + 1], sc, -mu));
                    lsum[w & 3] += p0 + p1;
                    const uint32_t b0 = __float_as_uint(p0), b1 = __float_as_uint(p1);
                    hw[w] = __byte_perm(b0, b1, 0x7632);
                    lw[w] = pack_bf16(p0 - __uint_as_float(b0 & 0xFFFF0000u), p1 - __uint_as_float(b1 & 0xFFFF0000u));
                }
#pragma unroll
                for (int c = 0; c < SC / 2; c += 16)
                    tmem_st16x2(pt + (SC / 2) * cq + c, hw + c, pt + BN / 2 + (SC / 2) * cq + c, lw + c);
            }
            l += (lsum[0] + lsum[1]) + (lsum[2] + lsum[3]);
            tc_fence_before();
            mbar_arrive(smem_u32(&bars[B_P_FULL + st]));
        }
        float ls[kRowThreads];
        if (ok) ok = exchange(n_kt, l, ls);
        if (ok)
            ok = __all_sync(0xFFFFFFFFu,
                            mbar_wait(smem_u32(&bars[B_PV_DONE + ((n_kt - 1) & 1)]), ((n_kt - 1) >> 1) & 1, wl));
        if (ok) {
            tc_fence_after();
            float lt = 0.f;
#pragma unroll
            for (int qq = 0; qq < kRowThreads; ++qq) lt += ls[qq];
            // fp16 values were scaled by 2^-E for the value product
            const float vs = kP16 ? __uint_as_float((uint32_t)(127 + v_scale_exp(*a.v_absmax)) << 23) : 1.f;
            const float inv = lt > 0.f ? vs / lt : 0.f;
            TOut *out = SUFFIX ? reinterpret_cast<TOut *>(a.part_o + ((row_ok ? i : 0) * a.Hq + h) * DT + OC * cq)
                               : reinterpret_cast<TOut *>(a.out) + (((int64_t)s * a.N + (row_ok ? i : 0)) * a.Hq + h) * DT +
                                     OC * cq;
#pragma unroll
            for (int c0 = 0; c0 < OC; c0 += OCH) {
                float ov[OCH];
                tmem_ld_cols<OCH>(t_o + lane_off + OC * cq + c0, ov);
                if (row_ok) {
#pragma unroll
                    for (int c = 0; c < OCH; ++c) ov[c] *= inv;
#pragma unroll
                    for (int e = 0; e < OCH / 8; ++e) store8<TOut>(out + c0 + 8 * e, ov + 8 * e);
                }
            }
            if (SUFFIX) {
                if (row_ok && cq == 0) a.part_lse[i * a.Hq + h] = m_used + __log2f(lt);
            } else if (row_ok && cq == 0 && a.lse != nullptr) {
                a.lse[((int64_t)s * a.Hq + h) * a.lse_ld + i] = (m_used + __log2f(lt)) * kLn2;
            }
        }
    }

    if (!ok) atomicOr(&g_ris_tile_error, 2u);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == kMmaWarp)
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

// [N][H][DT] 16-bit values (bf16, or fp16 with f16 set) viewed as 3D (d, head, token); box =
// 64 d x 1 head x `rows` tokens.
bool make_map3(CUtensorMap *m, const void *base, int64_t N, int H, int rows, int DT, bool f16 = false)
{
    auto fn = encode_fn();
    if (fn == nullptr) return false;
    cuuint64_t dims[3] = {(cuuint64_t)DT, (cuuint64_t)H, (cuuint64_t)N};
    cuuint64_t strides[2] = {(cuuint64_t)DT * 2, (cuuint64_t)H * DT * 2};
    cuuint32_t box[3] = {64, 1, (cuuint32_t)rows};
    cuuint32_t estr[3] = {1, 1, 1};
    return fn(m, f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base),
              dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int DT, bool SPLIT, bool DENSE, typename TOut, bool SUFFIX = false>
cudaError_t launch_t(const AttnArgs &a, const TileMaps &maps, const void *q_hi, const void *q_lo, cudaStream_t s)
{
    auto kern = k_attn_tile<DT, SPLIT, DENSE, SUFFIX, TOut>;
    static bool attr = false;
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    const int64_t n_qt = (a.row1 + BM - 1) / BM - a.row0 / BM;  // tiles covering rows row0 .. row1-1
    const unsigned grid = (unsigned)(n_qt * a.Hq * a.n_sets);
    kern<<<grid, kThreads, SMEM_BYTES, s>>>(a, maps, q_hi, q_lo);
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

// K / V tensor maps of a call (the key low part only with split queries and keys; the values
// as fp16 when P is fp16).
bool make_maps(TileMaps &maps, const AttnArgs &a, bool split, int D)
{
    if (kP16 && (a.v16 == nullptr || a.v_absmax == nullptr)) return false;
    if (!make_map3(&maps.kh, a.k, a.N, a.Hkv, BN, D) ||
        !make_map3(&maps.v, kP16 ? a.v16 : a.v, a.N, a.Hkv, BN, D, kP16))
        return false;
    if (split) return make_map3(&maps.kl, a.k_lo, a.N, a.Hkv, BN, D);
    maps.kl = maps.kh;
    return true;
}

template <int DT>
cudaError_t launch_tile_d(const AttnArgs &a, const TileMaps &maps, const void *q_hi, const void *q_lo, int out_dtype,
                          bool dense, cudaStream_t s)
{
    const bool split = q_lo != nullptr;
    if (out_dtype == RIS_F32) {
        if (split) return dense ? launch_t<DT, true, true, float>(a, maps, q_hi, q_lo, s) : launch_t<DT, true, false, float>(a, maps, q_hi, q_lo, s);
        return dense ? launch_t<DT, false, true, float>(a, maps, q_hi, q_lo, s) : launch_t<DT, false, false, float>(a, maps, q_hi, q_lo, s);
    }
    if (split)
        return dense ? launch_t<DT, true, true, __nv_bfloat16>(a, maps, q_hi, q_lo, s)
                     : launch_t<DT, true, false, __nv_bfloat16>(a, maps, q_hi, q_lo, s);
    return dense ? launch_t<DT, false, true, __nv_bfloat16>(a, maps, q_hi, q_lo, s)
                 : launch_t<DT, false, false, __nv_bfloat16>(a, maps, q_hi, q_lo, s);
}

// q_hi / q_lo: queries as a bf16 pair [N][Hq][D] (q_lo null: exact bf16 queries and keys,
// one score product); a.k / a.k_lo: keys as a pair; a.v: values. Head dim 128 or 64.
cudaError_t launch_attention_tile(const AttnArgs &a, int D, const void *q_hi, const void *q_lo, int out_dtype,
                                  bool dense, cudaStream_t s)
{
    static std::mutex mu;
    std::lock_guard<std::mutex> lk(mu);
    if (D != 128 && D != 64) return cudaErrorInvalidValue;
    alignas(64) TileMaps maps;
    if (!make_maps(maps, a, q_lo != nullptr, D)) return cudaErrorInvalidValue;
    return D == 128 ? launch_tile_d<128>(a, maps, q_hi, q_lo, out_dtype, dense, s)
                    : launch_tile_d<64>(a, maps, q_hi, q_lo, out_dtype, dense, s);
}

cudaError_t launch_attention_tile_suffix(const AttnArgs &a, int D, const void *q_hi, const void *q_lo, cudaStream_t s)
{
    static std::mutex mu;
    std::lock_guard<std::mutex> lk(mu);
    if (a.part_o == nullptr || a.part_lse == nullptr || a.n_sets != 1 || (D != 128 && D != 64))
        return cudaErrorInvalidValue;
    const bool split = q_lo != nullptr;
    alignas(64) TileMaps maps;
    if (!make_maps(maps, a, split, D)) return cudaErrorInvalidValue;
    if (D == 128)
        return split ? launch_t<128, true, false, float, true>(a, maps, q_hi, q_lo, s)
                     : launch_t<128, false, false, float, true>(a, maps, q_hi, q_lo, s);
    return split ? launch_t<64, true, false, float, true>(a, maps, q_hi, q_lo, s)
                 : launch_t<64, false, false, float, true>(a, maps, q_hi, q_lo, s);
}

}  // namespace ris
