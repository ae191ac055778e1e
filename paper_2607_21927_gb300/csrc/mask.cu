// RIS mask sampler (paper, Methods, "Memory-Bounded Geometry Generation" and "Sampling
// Modes: Stochastic and Structural").
//
// Instead of one N x N boolean tensor per seed, every (mask, row) is expanded once into a
// causal bitmap row with all seeds OR-merged in registers (the paper's streaming merge,
// without ever holding a seed's mask), then compacted into ascending per-row key lists.
//
//   k_mask_bits : per (mask, row) CTA, per 32-key word: Philox4x32-10 draws of every seed
//                 (8 calls = 32 keys per seed), OR, forced window/anchors, Structural
//                 block clique, causal cut; writes the word and the row's key count.
//   k_mask_draws: index-draw sampler only: per (mask, row) CTA, the row's index draws of
//                 every seed (one Philox call = 4 draws), j = floor(u N / 2^32), kept when
//                 j < i by an atomic OR into the zeroed bitmap row; k_mask_bits then ORs the
//                 forced and clique keys into those words and counts the row.
//   k_scan_*    : exclusive scan of the counts into row_ptr (int64).
//   k_mask_fill : per (mask, row) CTA, expands the bitmap row into ascending key indices.
//
// Integer-only; every decision is an exact comparison of a 32-bit word with a host-resolved
// 64-bit threshold, so the result is bit-exact across devices and hosts.
#include <cstdint>

#include "ris_internal.h"

namespace ris {
namespace {

// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds of two 32x32 -> 64-bit
// products (multipliers 0xD2511F53 on word 0, 0xCD9E8D57 on word 2) whose high halves are
// xored with the other counter words and the round key; the key advances by the Weyl
// constants (0x9E3779B9, 0xBB67AE85) after each round.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1)
{
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint64_t p0 = (uint64_t)0xD2511F53u * c.x;
        const uint64_t p1 = (uint64_t)0xCD9E8D57u * c.z;
        c = make_uint4((uint32_t)(p1 >> 32) ^ c.y ^ k0, (uint32_t)p1, (uint32_t)(p0 >> 32) ^ c.w ^ k1, (uint32_t)p0);
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    return c;
}

__device__ __forceinline__ uint32_t bits_below(int64_t n)  // bits [0, n) set, n in [0, 32]
{
    return n >= 32 ? 0xFFFFFFFFu : (n <= 0 ? 0u : ((1u << n) - 1u));
}

// Set bits for keys [lo, hi] (inclusive) inside the word holding keys [j0, j0 + 32).
__device__ __forceinline__ uint32_t range_bits(int64_t j0, int64_t lo, int64_t hi)
{
    if (hi < lo) return 0u;
    const int64_t a = lo - j0, b = hi - j0 + 1;  // [a, b) relative to j0
    return bits_below(b) & ~bits_below(a);
}

__device__ __forceinline__ int64_t row_word_offset(int64_t i)
{
    const int64_t a = i >> 5, b = i & 31;
    return i + 16 * a * (a - 1) + a * b;
}

constexpr int kBitsThreads = 128;

__global__ void __launch_bounds__(kBitsThreads) k_mask_bits(const MaskBitsArgs a)
{
    // rows are visited from the last (longest) to the first
    const int64_t r = (int64_t)blockIdx.x;
    const int32_t m = (int32_t)(r % a.n_masks);
    const bool one = a.single_row >= 0;
    const int64_t i = one ? a.single_row : a.N - 1 - r / a.n_masks;
    const uint32_t head_key = (a.heads_keyed > 1) ? (uint32_t)(m % a.heads_keyed) : 0u;
    const int32_t s0 = a.per_seed ? m / a.heads_keyed : 0;
    const int32_t s1 = a.per_seed ? s0 + 1 : a.n_seeds;
    const int64_t nw = (i >> 5) + 1;
    uint32_t *row = a.bitmap + (int64_t)m * a.words_per_mask + (one ? 0 : row_word_offset(i));
    const int64_t blk0 = (a.mode == RIS_MODE_STRUCTURAL) ? (i / a.B) * a.B : i + 1;

    int64_t count = 0;
    for (int64_t w = threadIdx.x; w < nw; w += kBitsThreads) {
        const int64_t j0 = w << 5;
        // forced keys: local window (i-W, i], anchors [0, A), Structural clique [blk0, i]
        uint32_t bits = a.or_existing ? row[w] : 0u;
        bits |= range_bits(j0, i - a.W + 1, i);
        bits |= range_bits(j0, 0, (int64_t)a.A - 1);
        bits |= range_bits(j0, blk0, i);
        const uint32_t causal = range_bits(j0, 0, i - 1);  // drawn pairs are j < i
        if (a.thr > 0) {
            // u < thr for thr in [1, 2^32] is u <= thr - 1 in 32 bits
            const uint32_t tm1 = a.thr > 0xFFFFFFFFull ? 0xFFFFFFFFu : (uint32_t)(a.thr - 1);
#pragma unroll 1
            for (int32_t s = s0; s < s1; ++s) {
                const uint32_t seed = a.seeds.v[s];
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    const uint32_t need = (causal >> (4 * c)) & ~(bits >> (4 * c)) & 0xFu;
                    if (need == 0) continue;
                    const uint4 u = philox4x32_10(
                        make_uint4((uint32_t)((j0 >> 2) + c), (uint32_t)i, a.stream, a.layer_key),
                        seed, head_key);
                    uint32_t keep = 0;
                    keep |= (u.x <= tm1) ? 1u : 0u;
                    keep |= (u.y <= tm1) ? 2u : 0u;
                    keep |= (u.z <= tm1) ? 4u : 0u;
                    keep |= (u.w <= tm1) ? 8u : 0u;
                    bits |= (keep & need) << (4 * c);
                }
            }
        }
        bits &= range_bits(j0, 0, one ? i - 1 : i);  // a single row keeps keys j < i only
        row[w] = bits;
        count += __popc(bits);
    }
    // block reduction of the row count
    __shared__ int64_t red[kBitsThreads / 32];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) count += __shfl_xor_sync(0xFFFFFFFFu, count, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = count;
    __syncthreads();
    if (threadIdx.x == 0) {
        int64_t t = 0;
#pragma unroll
        for (int k = 0; k < kBitsThreads / 32; ++k) t += red[k];
        a.counts[one ? (int64_t)m : (int64_t)m * a.N + i] = t;
    }
}

constexpr int kDrawThreads = 128;

__global__ void __launch_bounds__(kDrawThreads) k_mask_draws(const MaskBitsArgs a)
{
    const int64_t r = (int64_t)blockIdx.x;
    const int32_t m = (int32_t)(r % a.n_masks);
    const bool one = a.single_row >= 0;
    const int64_t i = one ? a.single_row : a.N - 1 - r / a.n_masks;
    if (i == 0) return;  // no j < 0
    const uint32_t head_key = (a.heads_keyed > 1) ? (uint32_t)(m % a.heads_keyed) : 0u;
    const int32_t s0 = a.per_seed ? m / a.heads_keyed : 0;
    const int32_t s1 = a.per_seed ? s0 + 1 : a.n_seeds;
    uint32_t *row = a.bitmap + (int64_t)m * a.words_per_mask + (one ? 0 : row_word_offset(i));
    const int64_t groups = (a.draws + 3) >> 2;
    const uint64_t n = (uint64_t)a.N;
    for (int32_t s = s0; s < s1; ++s) {
        const uint32_t seed = a.seeds.v[s];
        for (int64_t g = threadIdx.x; g < groups; g += kDrawThreads) {
            const uint4 u = philox4x32_10(make_uint4((uint32_t)g, (uint32_t)i, a.stream + 2u, a.layer_key), seed,
                                          head_key);
            const uint32_t w4[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                if (4 * g + c >= a.draws) break;
                const int64_t j = (int64_t)(((uint64_t)w4[c] * n) >> 32);
                if (j < i) atomicOr(row + (j >> 5), 1u << (j & 31));
            }
        }
    }
}

// ---------------------------------------------------------------- exclusive scan (int64)
constexpr int kScanThreads = 1024;
constexpr int kScanPer = 4;
constexpr int64_t kScanTile = (int64_t)kScanThreads * kScanPer;

// Block-level inclusive scan of a tile of kScanTile elements held kScanPer per thread.
__device__ __forceinline__ int64_t block_inclusive(int64_t v, int64_t *smem)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int64_t t = __shfl_up_sync(0xFFFFFFFFu, v, o);
        if (lane >= o) v += t;
    }
    if (lane == 31) smem[warp] = v;
    __syncthreads();
    if (warp == 0) {
        int64_t w = smem[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int64_t t = __shfl_up_sync(0xFFFFFFFFu, w, o);
            if (lane >= o) w += t;
        }
        smem[lane] = w;
    }
    __syncthreads();
    if (warp > 0) v += smem[warp - 1];
    return v;
}

// In-place inclusive scan of each tile of x[0, n); tile totals to partials[tile].
__global__ void __launch_bounds__(kScanThreads) k_scan_tiles(int64_t *x, int64_t n, int64_t *partials)
{
    __shared__ int64_t smem[32];
    const int64_t base = (int64_t)blockIdx.x * kScanTile + (int64_t)threadIdx.x * kScanPer;
    int64_t vals[kScanPer];
    int64_t sum = 0;
#pragma unroll
    for (int e = 0; e < kScanPer; ++e) {
        vals[e] = (base + e < n) ? x[base + e] : 0;
        sum += vals[e];
    }
    const int64_t incl = block_inclusive(sum, smem);
    int64_t run = incl - sum;
#pragma unroll
    for (int e = 0; e < kScanPer; ++e) {
        run += vals[e];
        if (base + e < n) x[base + e] = run;
    }
    if (threadIdx.x == kScanThreads - 1) partials[blockIdx.x] = incl;
}

// Single-CTA exclusive scan of the tile totals (any count, in chunks with a carry).
__global__ void __launch_bounds__(kScanThreads) k_scan_partials(int64_t *p, int64_t n)
{
    __shared__ int64_t smem[32];
    __shared__ int64_t carry;
    if (threadIdx.x == 0) carry = 0;
    __syncthreads();
    for (int64_t b = 0; b < n; b += kScanThreads) {
        const int64_t idx = b + threadIdx.x;
        const int64_t v = idx < n ? p[idx] : 0;
        const int64_t incl = block_inclusive(v, smem);
        const int64_t c = carry;
        if (idx < n) p[idx] = c + incl - v;
        __syncthreads();
        if (threadIdx.x == kScanThreads - 1) carry = c + incl;
        __syncthreads();
    }
}

__global__ void __launch_bounds__(kScanThreads) k_scan_add(int64_t *x, int64_t n, const int64_t *partials)
{
    const int64_t add = partials[blockIdx.x];
    const int64_t base = (int64_t)blockIdx.x * kScanTile;
    for (int e = threadIdx.x; e < kScanTile; e += kScanThreads)
        if (base + e < n) x[base + e] += add;
}

// ---------------------------------------------------------------- CSR fill
constexpr int kFillThreads = 128;

template <typename TIdx>
__global__ void __launch_bounds__(kFillThreads) k_mask_fill(const MaskFillArgs a)
{
    __shared__ int64_t warp_tot[kFillThreads / 32];
    const int64_t r = (int64_t)blockIdx.x;
    const int32_t m = (int32_t)(r % a.n_masks);
    const bool one = a.single_row >= 0;
    const int64_t i = one ? a.single_row : a.N - 1 - r / a.n_masks;
    const int64_t nw = (i >> 5) + 1;
    const uint32_t *row = a.bitmap + (int64_t)m * a.words_per_mask + (one ? 0 : row_word_offset(i));
    TIdx *col = reinterpret_cast<TIdx *>(a.col) + a.row_ptr[one ? (int64_t)m : (int64_t)m * a.N + i];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int64_t carry = 0;
    for (int64_t w0 = 0; w0 < nw; w0 += kFillThreads) {
        const int64_t w = w0 + threadIdx.x;
        uint32_t bits = w < nw ? row[w] : 0u;
        const int c = __popc(bits);
        int incl = c;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
            if (lane >= o) incl += t;
        }
        if (lane == 31) warp_tot[warp] = incl;
        __syncthreads();
        int64_t before = carry;
        int64_t chunk = 0;
#pragma unroll
        for (int k = 0; k < kFillThreads / 32; ++k) {
            if (k < warp) before += warp_tot[k];
            chunk += warp_tot[k];
        }
        int64_t pos = before + incl - c;
        const int64_t j0 = w << 5;
        while (bits) {
            const int b = __ffs(bits) - 1;
            col[pos++] = (TIdx)(j0 + b);
            bits &= bits - 1;
        }
        carry += chunk;
        __syncthreads();
    }
}

}  // namespace

cudaError_t launch_mask_bits(const MaskBitsArgs &a, cudaStream_t s)
{
    const int64_t blocks = (int64_t)a.n_masks * (a.single_row >= 0 ? 1 : a.N);
    k_mask_bits<<<(unsigned)blocks, kBitsThreads, 0, s>>>(a);
    note_launch();
    return cudaGetLastError();
}

cudaError_t launch_mask_draws(const MaskBitsArgs &a, cudaStream_t s)
{
    const int64_t blocks = (int64_t)a.n_masks * (a.single_row >= 0 ? 1 : a.N);
    k_mask_draws<<<(unsigned)blocks, kDrawThreads, 0, s>>>(a);
    note_launch();
    return cudaGetLastError();
}

int64_t scan_partials_count(int64_t n) { return (n + kScanTile - 1) / kScanTile; }

cudaError_t launch_scan_inplace(int64_t *x, int64_t n, int64_t *partials, cudaStream_t s)
{
    const int64_t tiles = scan_partials_count(n);
    k_scan_tiles<<<(unsigned)tiles, kScanThreads, 0, s>>>(x, n, partials);
    k_scan_partials<<<1, kScanThreads, 0, s>>>(partials, tiles);
    k_scan_add<<<(unsigned)tiles, kScanThreads, 0, s>>>(x, n, partials);
    note_launch(3);
    return cudaGetLastError();
}

cudaError_t launch_mask_fill(const MaskFillArgs &a, cudaStream_t s)
{
    const int64_t blocks = (int64_t)a.n_masks * (a.single_row >= 0 ? 1 : a.N);
    if (a.col_bytes == 2)
        k_mask_fill<uint16_t><<<(unsigned)blocks, kFillThreads, 0, s>>>(a);
    else
        k_mask_fill<uint32_t><<<(unsigned)blocks, kFillThreads, 0, s>>>(a);
    note_launch();
    return cudaGetLastError();
}

}  // namespace ris
