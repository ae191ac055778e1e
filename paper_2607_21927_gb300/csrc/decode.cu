// Hybrid Anchor decode step (paper, Methods, "Hybrid Anchor and Pre-Fusion Unified Softmax
// (PFUS)"): the token generated at position t attends to the frozen Stochastic Anchor (the key
// set of the first generated token, kept as an ascending list) merged with the Dynamic Local
// Window t - W < j <= t, with one softmax over the merged set.
//
// The merge needs no sort: the anchor keys at or above the window's first key are exactly the
// duplicates, so the merged set is the anchor list cut at win_lo followed by the contiguous
// window. The cut is one load from a rank table built with the anchor (rank[j] = anchor keys
// below j). Key number k of KV head g is anchor[k] for k < nA, else win_lo + (k - nA).
// Nothing in the launch depends on t, so the position may live in device memory and a
// captured CUDA graph of a whole token can be replayed token after token.
//
//   k_decode_partial : one CTA per (chunk of 32 keys, KV head): rotates the G query heads of
//                      the KV head at position t (fp64 angle, as the prefill RoPE), stages the
//                      chunk's K~ (high + low parts, fp32) and V rows in shared memory, and
//                      writes each head's partial (max, sum) and unnormalised output.
//   k_decode_combine : one CTA per query head: rescales the partials to the global maximum,
//                      sums and normalises; optional natural-log LSE.
//
// A decode step is one query row: a GEMV-shaped product that reads each selected K/V row once,
// so it runs on the FP32 pipes (no tensor-core tile to fill) and is bound by the K/V row
// reads; fp32 scores and probabilities keep it well inside the bf16 tolerance.
#include <cuda_bf16.h>

#include <cmath>
#include <cstdint>

#include "ris_internal.h"

namespace ris {
namespace {

__device__ unsigned int g_ris_decode_error;

constexpr int kDecodeThreads = 128;
constexpr int kMaxG = 8;
constexpr int kMaxD = 128;

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

template <typename T, bool LO>
__global__ void __launch_bounds__(kDecodeThreads) k_decode_partial(const DecodeArgs a)
{
    __shared__ float qs[kMaxG][kMaxD];
    __shared__ float ks[kDecodeChunk][kMaxD + 1];  // +1: rows fall in distinct banks
    __shared__ float vs[kDecodeChunk][kMaxD];
    __shared__ float ps[kMaxG][kDecodeChunk];
    __shared__ int32_t keys[kDecodeChunk];

    const int g = blockIdx.y, chunk = blockIdx.x, tid = threadIdx.x;
    const int D = a.D, G = a.G, half = D >> 1;
    const int64_t slot = (int64_t)g * a.n_chunks + chunk;
    const int64_t t = a.t_dev != nullptr ? *a.t_dev : a.t;
    if (t < a.t0 || t >= a.cache_len) {  // only reachable through t_dev: flag it, attend to nothing
        if (tid == 0 && chunk == 0 && g == 0) atomicOr(&g_ris_decode_error, 2u);
        for (int h = tid; h < G; h += kDecodeThreads) a.part_ml[slot * G + h] = make_float2(-INFINITY, 0.f);
        return;
    }
    const int64_t win_lo = t - a.window + 1 > 0 ? t - a.window + 1 : 0;
    const int m = a.heads_keyed > 1 ? g : 0;
    const int64_t nA = a.rank[(int64_t)m * (a.t0 + 1) + (win_lo < a.t0 ? win_lo : a.t0)];
    const int64_t n = nA + (t - win_lo + 1);
    const int64_t k0 = (int64_t)chunk * kDecodeChunk;
    if (k0 >= n) {  // fewer keys than the grid covers: an empty partial
        for (int h = tid; h < G; h += kDecodeThreads) a.part_ml[slot * G + h] = make_float2(-INFINITY, 0.f);
        return;
    }
    const int nk = (int)((n - k0) < kDecodeChunk ? (n - k0) : kDecodeChunk);
    const int32_t *anchor = a.anchor + a.anchor_off[m];
    if (tid < kDecodeChunk) {
        const int64_t kk = k0 + tid;
        int64_t key = 0;  // rows past the set read key 0 and are masked out below
        if (kk < n) key = kk < nA ? (int64_t)anchor[kk] : win_lo + (kk - nA);
        keys[tid] = (int32_t)key;
    }
    for (int idx = tid; idx < G * half; idx += kDecodeThreads) {
        const int h = idx / half, c = idx - h * half;
        float sn, cs;
        sincos_reduced((double)t * a.f[c], &sn, &cs);
        const T *qp = reinterpret_cast<const T *>(a.q) + (int64_t)(g * G + h) * D;
        const float x0 = ldf(qp + c), x1 = ldf(qp + c + half);
        qs[h][c] = fmaf(x0, cs, -x1 * sn) * a.mscale;
        qs[h][c + half] = fmaf(x1, cs, x0 * sn) * a.mscale;
    }
    __syncthreads();
    for (int idx = tid; idx < kDecodeChunk * D; idx += kDecodeThreads) {
        const int r = idx / D, c = idx - r * D;
        const int64_t off = ((int64_t)keys[r] * a.Hkv + g) * D + c;
        float kv = ldf(reinterpret_cast<const T *>(a.k) + off);
        if (LO) kv += ldf(reinterpret_cast<const __nv_bfloat16 *>(a.k_lo) + off);
        ks[r][c] = kv;
        vs[r][c] = ldf(reinterpret_cast<const T *>(a.v) + off);
    }
    __syncthreads();
    for (int idx = tid; idx < G * kDecodeChunk; idx += kDecodeThreads) {
        const int h = idx / kDecodeChunk, r = idx - h * kDecodeChunk;
        float s = 0.f;
        for (int c = 0; c < D; ++c) s = fmaf(qs[h][c], ks[r][c], s);
        ps[h][r] = r < nk ? s * a.scale_log2 : -INFINITY;
    }
    __syncthreads();
    const int warp = tid >> 5, lane = tid & 31;
    for (int h = warp; h < G; h += kDecodeThreads / 32) {  // kDecodeChunk == 32: one key per lane
        const float x = ps[h][lane];
        float mx = x;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, o));
        const float p = exp2f(x - mx);  // the chunk holds at least one key, so mx is finite
        float l = p;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xFFFFFFFFu, l, o);
        ps[h][lane] = p;
        if (lane == 0) a.part_ml[slot * G + h] = make_float2(mx, l);
    }
    __syncthreads();
    for (int idx = tid; idx < G * D; idx += kDecodeThreads) {
        const int h = idx / D, c = idx - h * D;
        float acc = 0.f;
        for (int r = 0; r < nk; ++r) acc = fmaf(ps[h][r], vs[r][c], acc);
        a.part_o[(slot * G + h) * D + c] = acc;
    }
}

template <typename TO>
__global__ void k_decode_combine(const DecodeArgs a)
{
    const int h = blockIdx.x, c = threadIdx.x;
    const int g = h / a.G, hl = h - g * a.G;
    const int64_t base = (int64_t)g * a.n_chunks;
    float M = -INFINITY;
    for (int ch = 0; ch < a.n_chunks; ++ch) M = fmaxf(M, a.part_ml[(base + ch) * a.G + hl].x);
    float L = 0.f, acc = 0.f;
    for (int ch = 0; ch < a.n_chunks; ++ch) {
        const float2 ml = a.part_ml[(base + ch) * a.G + hl];
        if (ml.x == -INFINITY) continue;  // empty chunk: no output was written
        const float w = exp2f(ml.x - M);
        L = fmaf(ml.y, w, L);
        acc = fmaf(a.part_o[((base + ch) * a.G + hl) * a.D + c], w, acc);
    }
    const float o = acc / L;
    if constexpr (sizeof(TO) == 4)
        reinterpret_cast<float *>(a.out)[(int64_t)h * a.D + c] = o;
    else
        reinterpret_cast<__nv_bfloat16 *>(a.out)[(int64_t)h * a.D + c] = __float2bfloat16_rn(o);
    if (c == 0 && a.lse != nullptr) a.lse[h] = (M + log2f(L)) * 0.69314718055994530942f;
    // the partial kernel, the only reader of t, has finished: move to the next position
    if (a.advance && a.t_dev != nullptr && h == 0 && c == 0) *a.t_dev += 1;
}

// rank[m][j] = lower_bound(keys of list m, j) - start, for j = 0 .. t0
__global__ void k_anchor_rank(const int32_t *keys, const int64_t *off, int32_t n_masks, int64_t t0, int32_t *rank)
{
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (int64_t)n_masks * (t0 + 1)) return;
    const int32_t m = (int32_t)(idx / (t0 + 1));
    const int64_t j = idx - (int64_t)m * (t0 + 1);
    int64_t lo = off[m], hi = off[m + 1];
    const int64_t b = lo;
    while (lo < hi) {
        const int64_t mid = (lo + hi) >> 1;
        if ((int64_t)keys[mid] < j)
            lo = mid + 1;
        else
            hi = mid;
    }
    rank[idx] = (int32_t)(lo - b);
}

}  // namespace

cudaError_t launch_anchor_rank(const int32_t *keys, const int64_t *off, int32_t n_masks, int64_t t0, int32_t *rank,
                               cudaStream_t s)
{
    const int64_t n = (int64_t)n_masks * (t0 + 1);
    k_anchor_rank<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(keys, off, n_masks, t0, rank);
    note_launch();
    return cudaGetLastError();
}

unsigned int read_decode_error()
{
    unsigned int v = 0, zero = 0;
    if (cudaMemcpyFromSymbol(&v, g_ris_decode_error, sizeof(v)) != cudaSuccess) return 0;
    if (v != 0) cudaMemcpyToSymbol(g_ris_decode_error, &zero, sizeof(zero));
    return v;
}

cudaError_t launch_decode(const DecodeArgs &a, int dtype, int out_dtype, cudaStream_t s)
{
    const dim3 grid_p((unsigned)a.n_chunks, (unsigned)a.Hkv);
    if (dtype == RIS_F32)
        k_decode_partial<float, false><<<grid_p, kDecodeThreads, 0, s>>>(a);
    else if (a.k_lo != nullptr)
        k_decode_partial<__nv_bfloat16, true><<<grid_p, kDecodeThreads, 0, s>>>(a);
    else
        k_decode_partial<__nv_bfloat16, false><<<grid_p, kDecodeThreads, 0, s>>>(a);
    if (out_dtype == RIS_F32)
        k_decode_combine<float><<<a.Hq, a.D, 0, s>>>(a);
    else
        k_decode_combine<__nv_bfloat16><<<a.Hq, a.D, 0, s>>>(a);
    note_launch(2);
    return cudaGetLastError();
}

}  // namespace ris
