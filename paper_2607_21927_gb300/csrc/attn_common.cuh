// Device helpers shared by the attention kernels of libris.
#pragma once

#include <cuda_bf16.h>

#include <cstdint>

#include "ris_internal.h"

namespace ris {

constexpr int kAttnWarps = 4;  // tasks (one per warp) per CTA
constexpr float kLn2 = 0.69314718055994530942f;

// A task is (output set s, row i, KV head g), row0 <= i < row1. Rows are handed out from the
// last (longest key list) to the first so the short rows fill the tail of the grid.
struct Task {
    int64_t i;
    int g;
    int s;
    int mask_id;
};

__device__ __forceinline__ Task decode_task(const AttnArgs &a, int64_t t)
{
    Task k;
    k.g = (int)(t % a.Hkv);
    const int64_t r = t / a.Hkv;
    k.s = (int)(r % a.n_sets);
    k.i = a.row1 - 1 - r / a.n_sets;
    k.mask_id = k.s * a.heads_keyed + (a.heads_keyed > 1 ? k.g : 0);
    return k;
}

// Key range of a task: [beg, beg + n) of the CSR, or keys 0..i when dense.
template <bool DENSE>
__device__ __forceinline__ void key_range(const AttnArgs &a, const Task &t, int64_t &beg, int64_t &n)
{
    if (DENSE) {
        beg = 0;
        n = t.i + 1;
    } else {
        const int64_t rr = (int64_t)t.mask_id * a.N + t.i;
        beg = a.row_ptr[rr];
        n = a.row_ptr[rr + 1] - beg;
    }
}

// First key of row i's dense suffix (AttnArgs::part_o): the earlier of its Structural block
// start and its local window start.
__device__ __forceinline__ int64_t dense_suffix_start(const AttnArgs &a, int64_t i)
{
    int64_t lo = i;
    if (a.clique_B > 0) lo = min(lo, (i / a.clique_B) * a.clique_B);
    if (a.window > 1) lo = min(lo, max((int64_t)0, i - (int64_t)a.window + 1));
    return lo;
}

template <bool DENSE, typename TIdx>
__device__ __forceinline__ int key_at(const TIdx *cols, int64_t pos)
{
    if (DENSE) return (int)pos;
    return (int)cols[pos];
}

// Power-of-two exponent E that brings the values into fp16's range for the value product
// (v / 2^E with |v| / 2^E < 2^14): 0 unless the largest |v| is 2^14 or more. The conversion
// kernel and the tile kernel's epilogue take E from the same max, so they agree exactly.
__device__ __forceinline__ int v_scale_exp(float vmax)
{
    const int e = (int)((__float_as_uint(vmax) >> 23) & 0xFF) - 127;  // floor(log2 vmax) for normal vmax
    return e >= 14 ? e - 13 : 0;
}

// 2^e as a float, for -126 <= e <= 127
__device__ __forceinline__ float pow2i(int e) { return __uint_as_float((uint32_t)(127 + e) << 23); }

// Scores of the tile kernel with fp8 corrections (rotated queries and keys, head dim 128):
// q = q_h + q_l and k = k_h + k_l with fp16 q_h, k_h, and
//   q.k ~ q_h.k_h + 2^-12 (e4m3(q_h 2^-ea) . e4m3(k_l 2^(12+ea)) + e4m3(q_l 2^(12+eb)) . e4m3(k_h 2^-eb)),
// the dropped q_l.k_l being below 2^-22 of q.k. The exponents keep every e4m3 operand within
// its range of 448 given bounds mq >= |q~| and mk >= |k~| (|k_l| <= 2^-11 |k|, so
// |k_l 2^(12+ea)| <= 2^(1+ea) mk), and the fp16 hi parts finite (bounds below 2^15); false
// when no pair exists (very large q and k together, or either beyond fp16), and the call then
// keeps the bf16 hi / lo scheme. The RoPE kernel that writes the operands and the
// tile kernel that reads them take the exponents from the same bounds, so they agree.
__device__ __forceinline__ int ceil_log2_ratio(float x, float y)  // ceil(log2(x / y)) for x, y > 0
{
    int e;
    const float m = frexpf(x / y, &e);  // x / y = m 2^e, m in [0.5, 1)
    return m == 0.5f ? e - 1 : e;
}
__device__ __forceinline__ bool fp8_score_scales(float mq, float mk, int &ea, int &eb)
{
    if (!(mq > 0.f) || !(mk > 0.f) || !(mq < 32768.f) || !(mk < 32768.f)) return false;
    ea = ceil_log2_ratio(mq, 448.f);
    eb = ceil_log2_ratio(mk, 448.f);
    if (ea < -40 || ea > 40 || eb < -40 || eb > 40) return false;
    return ldexpf(mk, 1 + ea) <= 448.f && ldexpf(mq, 1 + eb) <= 448.f;
}

__device__ __forceinline__ float warp_max(float x)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xFFFFFFFFu, x, o));
    return x;
}

__device__ __forceinline__ float warp_sum(float x)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
    return x;
}

}  // namespace ris
