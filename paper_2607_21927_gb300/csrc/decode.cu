// Hybrid Anchor decode step (paper, Methods, "Hybrid Anchor and Pre-Fusion Unified Softmax
// (PFUS)"): the token generated at position t attends to the frozen Stochastic Anchor (the key
// set of the first generated token, kept as an ascending list) merged with the Dynamic Local
// Window t - W < j <= t, with one softmax over the merged set.
//
// The merge needs no sort and no search: the anchor keys at or after the window's first key
// win_lo = max(0, t - W + 1) are exactly the duplicates (every anchor key is below t0 <= t).
// So the CTAs are split into anchor chunks (32 consecutive entries of the anchor list, a key
// kept iff it is below win_lo) and window chunks (32 consecutive positions from win_lo, kept
// iff at most t). A CTA needs only its slice of the list and the position, loaded side by
// side, before it can request its rows; and nothing in the launch depends on t, so the
// position may live in device memory and a captured CUDA graph of a whole token can be
// replayed token after token.
//
//   k_decode_partial : one CTA per (chunk of 32 keys, KV head): issues all of the chunk's
//                      16-byte K~ (high + low parts) and V row loads at once, rotates the G
//                      query heads of the KV head at position t (fp64 angle, as the prefill
//                      RoPE) while they are in flight, takes the scores of all heads from the
//                      key pieces in registers (bf16 caches: mma.sync with the pieces as B
//                      fragments), and writes each head's partial (max, sum, unnormalised
//                      output) to global memory, head-major.
//   k_decode_combine : one CTA per (query head, 32 channels): rescales the chunk partials to
//                      the global maximum, sums and normalises; optional natural-log LSE.
//
// A decode step is one query row: a GEMV-shaped step that reads each selected K/V row once and
// is bound by the latency of the loads that find and fetch them. For bf16 caches the scores
// (8 heads x 32 keys) and the value product (8 heads x D channels over 32 keys) are small
// tensor-core products with fp32 accumulation; the softmax is fp32.
#include <utility>
#include <cuda_bf16.h>

#include <cmath>
#include <cstdint>

#include "ris_internal.h"


namespace ris {
namespace {

__device__ unsigned int g_ris_decode_error;

constexpr int kDecodeThreads = 256;  // eight warps (the softmax: one per query head of the KV head)
constexpr int kMaxG = 8;

template <typename T>
__device__ __forceinline__ float ldf(const T *p);
template <>
__device__ __forceinline__ float ldf<float>(const float *p) { return *p; }
template <>
__device__ __forceinline__ float ldf<__nv_bfloat16>(const __nv_bfloat16 *p) { return __bfloat162float(*p); }

// sin and cos of the angle a (fp64), reduced by the nearest multiple of 2 pi in fp64
__device__ __forceinline__ void sincos_reduced(double a, float *sn, float *cs)
{
    const double n = rint(a * 0.15915494309189533577);
    double red = fma(-n, 6.28318530717958623200, a);
    red = fma(-n, 2.4492935982947064e-16, red);
    sincosf((float)red, sn, cs);
}

// Asynchronous prefetch of `bytes` (a multiple of 16, 16-byte aligned address) into L2; no
// result comes back to the thread.
__device__ __forceinline__ void prefetch_l2(const void *p, int bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(__cvta_generic_to_global(p)), "r"(bytes)
                 : "memory");
}

// d += A B on the tensor cores (m16n8k16, bf16 in, fp32 accumulate) with rows 8..15 of A zero:
// a0 / a2 hold row lane/4 of A at columns 2(lane%4) + {0, 1} / + {8, 9}, b0 / b1 rows
// 2(lane%4) + {0, 1} / + {8, 9} of B at column lane/4; d0 / d1 are row lane/4 of the product at
// columns 2(lane%4) + {0, 1}.
__device__ __forceinline__ void mma_bf16(float &d0, float &d1, float &d2, float &d3, uint32_t a0, uint32_t a2,
                                         uint32_t b0, uint32_t b1)
{
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
                 "{%0, %1, %2, %3};"
                 : "+f"(d0), "+f"(d1), "+f"(d2), "+f"(d3)
                 : "r"(a0), "r"(0u), "r"(a2), "r"(0u), "r"(b0), "r"(b1));
}

// B operand of mma m16n8k16 from a row-major [k][n] bf16 tile in shared memory: lanes 0..7
// give the addresses of rows k = 0..7, lanes 8..15 of rows 8..15 (8 columns from n0 each).
__device__ __forceinline__ void ldmatrix_x2_trans(uint32_t &b0, uint32_t &b1, const void *row)
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0, %1}, [%2];"
                 : "=r"(b0), "=r"(b1)
                 : "r"((uint32_t)__cvta_generic_to_shared(row))
                 : "memory");
}

// 16-byte row pieces of the staged K/V rows: bf16 holds 8 values per piece, fp32 holds 4.
template <typename T>
struct Piece {
    static constexpr int kVals = 16 / sizeof(T);
};

__device__ __forceinline__ void unpack(const uint4 &u, float *o, const __nv_bfloat16 *)
{
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        o[2 * i] = __uint_as_float(w[i] << 16);
        o[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
}

__device__ __forceinline__ void unpack(const uint4 &u, float *o, const float *)
{
    o[0] = __uint_as_float(u.x);
    o[1] = __uint_as_float(u.y);
    o[2] = __uint_as_float(u.z);
    o[3] = __uint_as_float(u.w);
}

// One CTA per (chunk of kDecodeChunk keys, KV head), each writing its own partial. Chunks below
// n_anchor_chunks take anchor entries, the others window positions. On the way to the K/V
// rows there is one round of dependent global loads: the position and this chunk's slice of
// the anchor list, side by side. (Merging the partials of 2, 4 or 8 CTAs on chip through
// thread-block clusters and distributed shared memory measured slower: the cluster barriers
// and the remote reads cost more than the combine kernel's extra partials.)
template <typename T, bool LO, int D>
__global__ void __launch_bounds__(kDecodeThreads, 4) k_decode_partial(const DecodeArgs a)
{
    constexpr int kPiecesRow = D * (int)sizeof(T) / 16;                   // 16-byte pieces per row
    constexpr int kPieces = kDecodeChunk * kPiecesRow / kDecodeThreads;  // per thread and plane
    constexpr int kHalf = D / 2;
    constexpr int kVals = Piece<T>::kVals;                               // values per piece
    constexpr int kRowStep = kDecodeThreads / kPiecesRow;                // rows between a thread's pieces
    constexpr int kLog = kPiecesRow == 8 ? 3 : kPiecesRow == 16 ? 4 : 5;  // log2(kPiecesRow)
    // bf16 caches: score and value products on the tensor cores (mma m16n8k16); 4 warps load
    // the keys, 4 the value rows
    constexpr bool kTc = sizeof(T) == 2;
    constexpr int kKSteps = D / 16;                 // k-steps of 16 head-dim columns
    constexpr int kKQ = kKSteps / 2;                // key pieces per lane and plane
    constexpr int kVRowStep = 128 / kPiecesRow;     // value rows between a value thread's pieces
    constexpr int kVPieces = kDecodeChunk / kVRowStep;
    static_assert(!kTc || (kDecodeChunk == 32 && kDecodeThreads == 256), "4 key warps of 8 keys, 4 value warps");
    constexpr int kQItems = kMaxG * kHalf / kDecodeThreads;  // query rotation items per thread
    static_assert(kMaxG * kHalf % kDecodeThreads == 0, "rotation items per thread");
    static_assert(kDecodeChunk * kPiecesRow % kDecodeThreads == 0, "pieces per thread");
    static_assert(kDecodeThreads % kPiecesRow == 0 && (1 << kLog) == kPiecesRow, "a row's pieces in one warp");
    static_assert(kMaxG == 8, "the score butterfly splits 8 heads");
    static_assert(D <= kDecodeThreads, "one thread per channel in the value product");
    __shared__ __align__(16) float qs[kMaxG][D];  // rotated query heads (rows G .. kMaxG-1 zero)
    __shared__ __align__(16) __nv_bfloat16 qb[2][kMaxG][D + 8];  // the same as a bf16 high / low pair
    __shared__ __align__(16) float vs[kDecodeChunk][D];               // fp32 caches: value rows
    __shared__ __align__(16) __nv_bfloat16 vb[kDecodeChunk][D + 8];   // bf16 caches: value rows
    __shared__ __align__(16) __nv_bfloat16 pb[2][kMaxG][kDecodeChunk + 8];  // bf16 caches: P high / low
    __shared__ float sc[kMaxG][kDecodeChunk];     // scores
    __shared__ __align__(16) float ps[kMaxG][kDecodeChunk];
    __shared__ float2 rot[kHalf];                 // (cos, sin) of t * f_c
    __shared__ int32_t keys[kDecodeChunk];

    __shared__ uint32_t kept;  // bit r: key r of the chunk is in the merged set

    const int g = blockIdx.y, chunk = blockIdx.x, tid = threadIdx.x;
    const int warp = tid >> 5, lane = tid & 31;
    const int pc = tid % kPiecesRow, r0 = tid / kPiecesRow;  // this thread's 16-byte column piece and first row
    const int pcv = (tid & 127) % kPiecesRow, rv0 = (tid & 127) / kPiecesRow;  // the same for a value warp
    const int G = a.G;
    const int m = a.heads_keyed > 1 ? g : 0;
    const bool from_anchor = chunk < a.n_anchor_chunks;
    const int64_t k0 = (int64_t)(from_anchor ? chunk : chunk - a.n_anchor_chunks) * kDecodeChunk;
    // Launched as a programmatic dependent of the kernel before it (in a token chain, the
    // previous layer step's combine), this CTA may start while that kernel still runs. Until
    // the wait below it only warms L2: warp 0 reads the position and the chunk's anchor slice
    // through L2 (no L1 copy) and prefetches the K/V rows they name, so that the row loads
    // after the wait hit L2 instead of HBM. What is read here may be stale; it only steers
    // prefetches of rows inside the cache, and everything is read again after the wait.
    if (warp == 0) {
        const int64_t tg = a.t_dev != nullptr ? (int64_t)__ldcg(reinterpret_cast<const long long *>(a.t_dev)) : a.t;
        int64_t key = -1;
        if (from_anchor) {
            if (k0 + lane < a.anchor_len[m]) key = __ldcg(a.anchor + a.anchor_base[m] + k0 + lane);
        } else if (tg >= 0 && tg < a.cache_len) {
            key = (tg - a.window + 1 > 0 ? tg - a.window + 1 : 0) + k0 + lane;
            if (key > tg) key = -1;
        }
        if (key >= 0 && key < a.cache_len) {
            const int64_t row = (key * a.Hkv + g) * D;
            prefetch_l2(reinterpret_cast<const T *>(a.k) + row, D * (int)sizeof(T));
            if (LO) prefetch_l2(reinterpret_cast<const __nv_bfloat16 *>(a.k_lo) + row, D * 2);
            prefetch_l2(reinterpret_cast<const T *>(a.v) + row, D * (int)sizeof(T));
        }
    }
    // The rotation table of the query at the position as read now (each thread its own entry
    // and its own read of the position; an entry is computed again after the wait if the
    // position turns out to differ), so that its fp64 angles stay off the path after the wait.
    int64_t t_rot = 0;
    if (tid < kHalf) {
        t_rot = a.t_dev != nullptr ? (int64_t)__ldcg(reinterpret_cast<const long long *>(a.t_dev)) : a.t;
        float sn, cs;
        sincos_reduced((double)t_rot * a.f[tid], &sn, &cs);
        rot[tid] = make_float2(cs, sn);
    }
    // Wait for the kernel before (the position, q, the anchor list of a fresh build and the
    // partials' buffer come after it), then let the next kernel be scheduled while this one runs.
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    // this lane's anchor entry, loaded alongside the position
    int32_t spec = -1;
    if (from_anchor && tid < kDecodeChunk && k0 + tid < a.anchor_len[m])
        spec = __ldcg(a.anchor + a.anchor_base[m] + k0 + tid);
    const int64_t t = a.t_dev != nullptr ? *a.t_dev : a.t;
    // this thread's query values (rotation items tid + i * kDecodeThreads), in the same round
    float qx0[kQItems], qx1[kQItems];
#pragma unroll
    for (int i = 0; i < kQItems; ++i) {
        const int idx = tid + i * kDecodeThreads, h = idx / kHalf, c = idx - h * kHalf;
        qx0[i] = 0.f;
        qx1[i] = 0.f;
        if (h < G) {
            const T *qp = reinterpret_cast<const T *>(a.q) + (int64_t)(g * G + h) * D;
            qx0[i] = ldf(qp + c);
            qx1[i] = ldf(qp + c + kHalf);
        }
    }
    const bool valid = t >= a.t0 && t < a.cache_len;  // only a device-side t can be outside
    if (!valid && tid == 0 && chunk == 0 && g == 0) atomicOr(&g_ris_decode_error, 2u);
    const int64_t win_lo = t - a.window + 1 > 0 ? t - a.window + 1 : 0;
    if (warp == 0) {
        // an anchor key stays unless the window holds it; a window position stays up to t
        const int64_t key = from_anchor ? (int64_t)spec : win_lo + k0 + lane;
        const bool in = valid && (from_anchor ? (spec >= 0 && key < win_lo) : key <= t);
        const uint32_t bits = __ballot_sync(0xFFFFFFFFu, in);
        keys[lane] = in ? (int32_t)key : 0;  // rows of dropped keys read key 0 and are masked out
        if (lane == 0) kept = bits;
    }
    __syncthreads();
    const uint32_t kbits = kept;
    const bool active = kbits != 0u;  // block-uniform
    // partials are head-major: those of query head (g, h) are slots (g * G + h) * n_chunks + i
    const int64_t slot0 = (int64_t)g * G * a.n_chunks + chunk;  // this CTA's slot for h = 0
    const int64_t hstride = a.n_chunks;

    if (active) {
      if constexpr (kTc) {
        // bf16 cache: warps 0..3 load the chunk's key pieces in the mma B-fragment layout (warp
        // w takes keys 8w .. 8w+7; lane l the key 8w + l/4 and its pieces 4q + l%4, which hold
        // the stored head-dim columns of k-steps 2q and 2q+1 as the fragment wants them), warps
        // 4..7 load the value rows; every load is issued before any is used
        uint4 kb[kKQ], kbl[kKQ], vv[kVPieces];
        if (warp < 4) {
            const int64_t row = ((int64_t)keys[warp * 8 + (lane >> 2)] * a.Hkv + g) * D;
            const uint4 *kp = reinterpret_cast<const uint4 *>(reinterpret_cast<const T *>(a.k) + row);
            const uint4 *klp = reinterpret_cast<const uint4 *>(reinterpret_cast<const __nv_bfloat16 *>(a.k_lo) + row);
#pragma unroll
            for (int q = 0; q < kKQ; ++q) {
                kb[q] = __ldg(kp + 4 * q + (lane & 3));
                if (LO) kbl[q] = __ldg(klp + 4 * q + (lane & 3));
            }
        } else {
#pragma unroll
            for (int j = 0; j < kVPieces; ++j) {
                const int64_t row = ((int64_t)keys[rv0 + j * kVRowStep] * a.Hkv + g) * D;
                vv[j] = __ldg(reinterpret_cast<const uint4 *>(reinterpret_cast<const T *>(a.v) + row) + pcv);
            }
        }
        // rotate the G query heads at position t while the rows are in flight, as a bf16 high
        // + low pair (heads G .. kMaxG-1 zero)
        if (tid < kHalf && t_rot != t) {
            float sn, cs;
            sincos_reduced((double)t * a.f[tid], &sn, &cs);
            rot[tid] = make_float2(cs, sn);
        }
        __syncthreads();
#pragma unroll
        for (int i = 0; i < kQItems; ++i) {
            const int idx = tid + i * kDecodeThreads, h = idx / kHalf, c = idx - h * kHalf;
            const float2 cs = rot[c];
            const float y0 = fmaf(qx0[i], cs.x, -qx1[i] * cs.y) * a.mscale;  // heads >= G: zero
            const float y1 = fmaf(qx1[i], cs.x, qx0[i] * cs.y) * a.mscale;
            const __nv_bfloat16 h0 = __float2bfloat16_rn(y0), h1 = __float2bfloat16_rn(y1);
            qb[0][h][c] = h0;
            qb[1][h][c] = __float2bfloat16_rn(y0 - __bfloat162float(h0));
            qb[0][h][c + kHalf] = h1;
            qb[1][h][c + kHalf] = __float2bfloat16_rn(y1 - __bfloat162float(h1));
        }
        if (warp >= 4) {  // the value rows go to shared memory as they are (bf16)
#pragma unroll
            for (int j = 0; j < kVPieces; ++j)
                *reinterpret_cast<uint4 *>(&vb[rv0 + j * kVRowStep][pcv * 8]) = vv[j];
        }
        __syncthreads();
        if (warp < 4) {
            // scores of the 8 heads x 8 keys of this warp on the tensor cores: A = query (rows =
            // heads, rows 8..15 zero), B = keys; q hi.k hi + q lo.k hi + q hi.k lo in fp32
            const int hq = lane >> 2, c = lane & 3;
            float d0 = 0.f, d1 = 0.f, d2 = 0.f, d3 = 0.f;
#pragma unroll
            for (int s = 0; s < kKSteps; ++s) {
                const int off = 8 * (4 * (s >> 1) + c) + 4 * (s & 1);
                const uint2 ah = *reinterpret_cast<const uint2 *>(&qb[0][hq][off]);
                const uint2 al = *reinterpret_cast<const uint2 *>(&qb[1][hq][off]);
                const uint32_t b0 = (s & 1) ? kb[s >> 1].z : kb[s >> 1].x;
                const uint32_t b1 = (s & 1) ? kb[s >> 1].w : kb[s >> 1].y;
                mma_bf16(d0, d1, d2, d3, ah.x, ah.y, b0, b1);
                mma_bf16(d0, d1, d2, d3, al.x, al.y, b0, b1);
                if (LO) {
                    const uint32_t l0 = (s & 1) ? kbl[s >> 1].z : kbl[s >> 1].x;
                    const uint32_t l1 = (s & 1) ? kbl[s >> 1].w : kbl[s >> 1].y;
                    mma_bf16(d0, d1, d2, d3, ah.x, ah.y, l0, l1);
                }
            }
            if (hq < G) {  // d0, d1: head hq, keys 8w + 2c and 8w + 2c + 1
                sc[hq][warp * 8 + 2 * c] = d0;
                sc[hq][warp * 8 + 2 * c + 1] = d1;
            }
        }
      } else {
        // fp32 caches: every row load of the chunk is issued before any is used; a thread's
        // pieces are all at the same column offset (pc), in rows r0, r0 + kRowStep, ...
        uint4 kh[kPieces], kl[kPieces], vv[kPieces];
#pragma unroll
        for (int j = 0; j < kPieces; ++j) {
            const int64_t row = ((int64_t)keys[r0 + j * kRowStep] * a.Hkv + g) * D;
            kh[j] = __ldg(reinterpret_cast<const uint4 *>(reinterpret_cast<const T *>(a.k) + row) + pc);
            if (LO) kl[j] = __ldg(reinterpret_cast<const uint4 *>(reinterpret_cast<const __nv_bfloat16 *>(a.k_lo) + row) + pc);
            vv[j] = __ldg(reinterpret_cast<const uint4 *>(reinterpret_cast<const T *>(a.v) + row) + pc);
        }
        // rotate the G query heads at position t while the rows are in flight (heads G .. kMaxG-1
        // are zero, so that the score loop below runs over kMaxG heads without guards)
        if (tid < kHalf && t_rot != t) {
            float sn, cs;
            sincos_reduced((double)t * a.f[tid], &sn, &cs);
            rot[tid] = make_float2(cs, sn);
        }
        __syncthreads();
#pragma unroll
        for (int i = 0; i < kQItems; ++i) {
            const int idx = tid + i * kDecodeThreads, h = idx / kHalf, c = idx - h * kHalf;
            const float2 cs = rot[c];
            const float y0 = fmaf(qx0[i], cs.x, -qx1[i] * cs.y) * a.mscale;  // heads >= G: zero
            const float y1 = fmaf(qx1[i], cs.x, qx0[i] * cs.y) * a.mscale;
            qs[h][c] = y0;
            qs[h][c + kHalf] = y1;
        }
        // the value rows go to shared memory for the value product
#pragma unroll
        for (int j = 0; j < kPieces; ++j) {
            float y[kVals];
            unpack(vv[j], y, (const T *)nullptr);
#pragma unroll
            for (int e = 0; e < kVals; e += 4)
                *reinterpret_cast<float4 *>(&vs[r0 + j * kRowStep][pc * kVals + e]) =
                    make_float4(y[e], y[e + 1], y[e + 2], y[e + 3]);
        }
        __syncthreads();
        // scores straight from the key pieces in registers: each thread forms the partial dot
        // products of its kVals channels with all kMaxG heads, and the kPiecesRow lanes of a row
        // add them up with a splitting butterfly (each exchange halves the heads a lane keeps:
        // 4 + 2 + 1 shuffles, then plain sums over the remaining lane bits), after which lane
        // pair ((lane >> (kLog - 3)) & 7) holds the full score of that head
#pragma unroll
        for (int j = 0; j < kPieces; ++j) {
            float x[kVals];
            unpack(kh[j], x, (const T *)nullptr);
            if (LO) {
                float lo8[8];
                unpack(kl[j], lo8, (const __nv_bfloat16 *)nullptr);
#pragma unroll
                for (int e = 0; e < kVals; ++e) x[e] += lo8[e];
            }
            float sh[kMaxG];
#pragma unroll
            for (int h = 0; h < kMaxG; ++h) {
                float acc = 0.f;
#pragma unroll
                for (int e = 0; e < kVals; e += 4) {
                    const float4 q4 = *reinterpret_cast<const float4 *>(&qs[h][pc * kVals + e]);
                    acc = fmaf(q4.x, x[e], fmaf(q4.y, x[e + 1], fmaf(q4.z, x[e + 2], fmaf(q4.w, x[e + 3], acc))));
                }
                sh[h] = acc;
            }
            {
                const bool b = (lane >> (kLog - 1)) & 1;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float send = b ? sh[i] : sh[i + 4], keep = b ? sh[i + 4] : sh[i];
                    sh[i] = keep + __shfl_xor_sync(0xFFFFFFFFu, send, 1 << (kLog - 1));
                }
            }
            {
                const bool b = (lane >> (kLog - 2)) & 1;
#pragma unroll
                for (int i = 0; i < 2; ++i) {
                    const float send = b ? sh[i] : sh[i + 2], keep = b ? sh[i + 2] : sh[i];
                    sh[i] = keep + __shfl_xor_sync(0xFFFFFFFFu, send, 1 << (kLog - 2));
                }
            }
            {
                const bool b = (lane >> (kLog - 3)) & 1;
                const float send = b ? sh[0] : sh[1], keep = b ? sh[1] : sh[0];
                sh[0] = keep + __shfl_xor_sync(0xFFFFFFFFu, send, 1 << (kLog - 3));
            }
#pragma unroll
            for (int o = 0; o < kLog - 3; ++o) sh[0] += __shfl_xor_sync(0xFFFFFFFFu, sh[0], 1 << o);
            const int lr = lane & (kPiecesRow - 1);
            const int h = ((lr >> (kLog - 1)) & 1) * 4 + ((lr >> (kLog - 2)) & 1) * 2 + ((lr >> (kLog - 3)) & 1);
            if ((lr & ((1 << (kLog - 3)) - 1)) == 0 && h < G) sc[h][r0 + j * kRowStep] = sh[0];
        }
      }
        __syncthreads();
        // the chunk's softmax: warp h takes query head h, lane r takes key r
        if (warp < G) {
            const int h = warp, r = lane;
            const float x = ((kbits >> r) & 1u) ? sc[h][r] * a.scale_log2 : -INFINITY;
            float mx = x;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, o));
            const float p = exp2f(x - mx);  // an active chunk keeps at least one key: mx is finite
            float l = p;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xFFFFFFFFu, l, o);
            if constexpr (kTc) {  // P as a bf16 high + low pair, the A operand of the value product
                const __nv_bfloat16 ph = __float2bfloat16_rn(p);
                pb[0][h][r] = ph;
                pb[1][h][r] = __float2bfloat16_rn(p - __bfloat162float(ph));
            } else {
                ps[h][r] = p;
            }
            if (lane == 0) a.part_ml[slot0 + h * hstride] = make_float2(mx, l);
        }
        __syncthreads();
        if constexpr (kTc) {
            // value product on the tensor cores: A = P (heads x keys, hi + lo), B = V (keys x
            // channels, read transposed by ldmatrix); warp w takes the channel tiles of 8
            // columns w * kNT .. w * kNT + kNT - 1 and stores its rows of the partial
            constexpr int kNT = D / 64;
            const int hq = lane >> 2, c = lane & 3;
#pragma unroll
            for (int nt = 0; nt < kNT; ++nt) {
                const int n0 = (warp * kNT + nt) * 8;
                float d0 = 0.f, d1 = 0.f, d2 = 0.f, d3 = 0.f;
#pragma unroll
                for (int ks = 0; ks < kDecodeChunk / 16; ++ks) {
                    uint32_t b0, b1;
                    ldmatrix_x2_trans(b0, b1, &vb[ks * 16 + (lane & 15)][n0]);
                    const int k = ks * 16 + 2 * c;
                    mma_bf16(d0, d1, d2, d3, *reinterpret_cast<const uint32_t *>(&pb[0][hq][k]),
                             *reinterpret_cast<const uint32_t *>(&pb[0][hq][k + 8]), b0, b1);
                    mma_bf16(d0, d1, d2, d3, *reinterpret_cast<const uint32_t *>(&pb[1][hq][k]),
                             *reinterpret_cast<const uint32_t *>(&pb[1][hq][k + 8]), b0, b1);
                }
                if (hq < G)
                    *reinterpret_cast<float2 *>(&a.part_o[(slot0 + hq * hstride) * D + n0 + 2 * c]) = make_float2(d0, d1);
            }
        } else {
        // value product: thread (channel c, head set hs) over heads hs, hs + step, ...
            constexpr int kStep = kDecodeThreads / D;
            constexpr int kPer = (kMaxG + kStep - 1) / kStep;
            const int c = tid % D, hs = tid / D;
            float acc[kPer];
#pragma unroll
            for (int e = 0; e < kPer; ++e) acc[e] = 0.f;
            for (int r = 0; r < kDecodeChunk; r += 4) {  // dropped keys: p = 0, rows finite
                const float v0 = vs[r][c], v1 = vs[r + 1][c], v2 = vs[r + 2][c], v3 = vs[r + 3][c];
#pragma unroll
                for (int e = 0; e < kPer; ++e) {
                    const int h = hs + e * kStep;
                    if (h < G) {
                        const float4 p4 = *reinterpret_cast<const float4 *>(&ps[h][r]);
                        acc[e] = fmaf(p4.x, v0, fmaf(p4.y, v1, fmaf(p4.z, v2, fmaf(p4.w, v3, acc[e]))));
                    }
                }
            }
#pragma unroll
            for (int e = 0; e < kPer; ++e) {
                const int h = hs + e * kStep;
                if (h < G) a.part_o[(slot0 + h * hstride) * D + c] = acc[e];
            }
        }
    } else {
        // a chunk with no key: an empty partial (weight 0 in the combine, finite outputs)
        for (int idx = tid; idx < G * D; idx += kDecodeThreads)
            a.part_o[(slot0 + (idx / D) * hstride) * D + idx % D] = 0.f;
        if (tid < G) a.part_ml[slot0 + tid * hstride] = make_float2(-INFINITY, 0.f);
    }
}

// One CTA per (query head, 32-channel slice). Warp w takes the ranges of 32 consecutive
// partials w, w + kCombineWarps, ...: lane j loads the (max, sum) of partial j of the range
// while every lane loads the outputs of all 32 partials at its channel (head-major partials
// are D floats apart, so the 32 loads are immediate offsets from one address), all in one
// round; then the range's maximum, the lane's weight (broadcast by shuffle) and the fold.
// The warps are merged in shared memory.
constexpr int kCombineWarps = 8;

template <typename TO, int D>
__global__ void __launch_bounds__(kCombineWarps * 32) k_decode_combine(const DecodeArgs a)
{
    // a programmatic dependent of the partial kernel: wait for its partials
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    __shared__ float wm[kCombineWarps], wl[kCombineWarps], wacc[kCombineWarps][32];
    const int h = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int c = blockIdx.y * 32 + lane;
    const int n = a.n_chunks;
    const float2 *ml = a.part_ml + (int64_t)h * n;  // query head h = g * G + hl: slots h * n + i
    const float *po = a.part_o + (int64_t)h * n * D + c;
    float M = -INFINITY, L = 0.f, acc = 0.f;  // the same M and L in every lane of the warp
    for (int r0 = warp * 32; r0 < n; r0 += kCombineWarps * 32) {
        const int cnt = n - r0 < 32 ? n - r0 : 32;
        const float2 mv = lane < cnt ? ml[r0 + lane] : make_float2(-INFINITY, 0.f);
        const float *pb = po + (int64_t)r0 * D;
        float oi[32];
#pragma unroll
        for (int u = 0; u < 32; ++u) {
            oi[u] = 0.f;
            if (u < cnt) oi[u] = pb[u * D];
        }
        float bm = mv.x;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) bm = fmaxf(bm, __shfl_xor_sync(0xFFFFFFFFu, bm, o));
        const float nm = fmaxf(M, bm);
        if (nm == -INFINITY) continue;  // warp-uniform: nothing kept so far
        const float so = exp2f(M - nm);  // M = -inf gives 0
        M = nm;
        const float w = exp2f(mv.x - M);  // this lane's partial; an empty one (-inf) weighs 0
        float lw = w * mv.y;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) lw += __shfl_xor_sync(0xFFFFFFFFu, lw, o);
        L = fmaf(L, so, lw);
        acc *= so;
#pragma unroll
        for (int u = 0; u < 32; ++u) acc = fmaf(oi[u], __shfl_sync(0xFFFFFFFFu, w, u), acc);
    }
    if (lane == 0) {
        wm[warp] = M;
        wl[warp] = L;
    }
    wacc[warp][lane] = acc;
    __syncthreads();
    if (warp == 0) {
        float Mt = -INFINITY;
#pragma unroll
        for (int w = 0; w < kCombineWarps; ++w) Mt = fmaxf(Mt, wm[w]);
        float Lt = 0.f, o = 0.f;
#pragma unroll
        for (int w = 0; w < kCombineWarps; ++w) {
            if (wm[w] == -INFINITY) continue;
            const float sw = exp2f(wm[w] - Mt);
            Lt = fmaf(wl[w], sw, Lt);
            o = fmaf(wacc[w][lane], sw, o);
        }
        o /= Lt;
        if constexpr (sizeof(TO) == 4)
            reinterpret_cast<float *>(a.out)[(int64_t)h * D + c] = o;
        else
            reinterpret_cast<__nv_bfloat16 *>(a.out)[(int64_t)h * D + c] = __float2bfloat16_rn(o);
        if (lane == 0 && blockIdx.y == 0 && a.lse != nullptr) a.lse[h] = (Mt + log2f(Lt)) * 0.69314718055994530942f;
        // the partial kernel, the only reader of t, has finished: move to the next position
        if (a.advance && a.t_dev != nullptr && h == 0 && blockIdx.y == 0 && lane == 0) *a.t_dev += 1;
    }
}

}  // namespace

unsigned int read_decode_error()
{
    unsigned int v = 0, zero = 0;
    if (cudaMemcpyFromSymbol(&v, g_ris_decode_error, sizeof(v)) != cudaSuccess) return 0;
    if (v != 0) cudaMemcpyToSymbol(g_ris_decode_error, &zero, sizeof(zero));
    return v;
}

// Launch as a programmatic dependent of the previous kernel in the stream: it may be scheduled
// while that kernel runs and waits for it (griddepcontrol.wait) before touching its results.
template <typename... P, typename... A>
cudaError_t launch_pdl(void (*kern)(P...), dim3 grid, dim3 block, cudaStream_t s, A &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, std::forward<A>(args)...);
}

template <int D>
cudaError_t launch_partial(const DecodeArgs &a, int dtype, dim3 grid, cudaStream_t s)
{
    if (dtype == RIS_F32) return launch_pdl(k_decode_partial<float, false, D>, grid, dim3(kDecodeThreads), s, a);
    if (a.k_lo != nullptr)
        return launch_pdl(k_decode_partial<__nv_bfloat16, true, D>, grid, dim3(kDecodeThreads), s, a);
    return launch_pdl(k_decode_partial<__nv_bfloat16, false, D>, grid, dim3(kDecodeThreads), s, a);
}

cudaError_t launch_decode(const DecodeArgs &a, int dtype, int out_dtype, cudaStream_t s)
{
    const dim3 grid_p((unsigned)a.n_chunks, (unsigned)a.Hkv);
    cudaError_t e = a.D == 128 ? launch_partial<128>(a, dtype, grid_p, s) : launch_partial<64>(a, dtype, grid_p, s);
    if (e != cudaSuccess) return e;
    const dim3 grid_c((unsigned)a.Hq, (unsigned)(a.D / 32));
    if (a.D == 128)
        e = out_dtype == RIS_F32 ? launch_pdl(k_decode_combine<float, 128>, grid_c, dim3(kCombineWarps * 32), s, a)
                                 : launch_pdl(k_decode_combine<__nv_bfloat16, 128>, grid_c, dim3(kCombineWarps * 32), s, a);
    else
        e = out_dtype == RIS_F32 ? launch_pdl(k_decode_combine<float, 64>, grid_c, dim3(kCombineWarps * 32), s, a)
                                 : launch_pdl(k_decode_combine<__nv_bfloat16, 64>, grid_c, dim3(kCombineWarps * 32), s, a);
    note_launch(2);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace ris
