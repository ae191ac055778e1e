// Internal declarations shared by the translation units of libris (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <cstdint>

#include "../../include/ris.h"

namespace ris {

constexpr int kMaxSeeds = 256;
constexpr int kMaxHeadDimHalf = 64;  // head_dim <= 128

// Seeds travel by value in the kernel parameter block (1 KB), so concurrent calls on
// different streams never share a device-side seed table.
struct SeedList {
    uint32_t v[kMaxSeeds];
};

// Arguments of the mask bitmap kernel (one CTA per (mask, row)).
struct MaskBitsArgs {
    int64_t N;
    int32_t n_seeds;      // seeds drawn per mask (all of them for the union, 1 per seed)
    int32_t per_seed;     // 1: mask m draws only seed m / heads_keyed
    int32_t heads_keyed;  // 1 or kv_heads
    int32_t n_masks;
    int32_t mode;         // RIS_MODE_STOCHASTIC or RIS_MODE_STRUCTURAL
    int32_t W;            // local window
    int32_t A;            // anchors
    uint32_t layer_key;
    uint32_t stream;      // Philox counter word 2
    uint64_t thr;         // keep iff word < thr
    int64_t B;            // Structural block size
    int64_t draws;        // index-draw sampler: draws per row and seed
    int32_t or_existing;  // 1: OR into the words already in the bitmap (index draws were set)
    int64_t single_row;   // -1: rows 0..N-1; >= 0: only this row, one CTA per mask, its words at
                          // bitmap + m * words_per_mask and its count at counts[m]
    int64_t words_per_mask;
    uint32_t *bitmap;     // [n_masks][words_per_mask]
    int64_t *counts;      // counts[m * N + i] (row_ptr + 1)
    SeedList seeds;
};

// Arguments of the CSR fill kernel.
struct MaskFillArgs {
    int64_t N;
    int32_t n_masks;
    int32_t col_bytes;
    int64_t words_per_mask;
    const uint32_t *bitmap;
    const int64_t *row_ptr;
    void *col;
    int64_t single_row;   // as MaskBitsArgs::single_row (keys of mask m from col + row_ptr[m])
};

// Arguments of the RoPE kernels: x_out[p][h][c], x_out[p][h][c + D/2] from x_in.
struct RopeArgs {
    const void *x_in;
    void *x_out;
    void *x_out_lo;  // bf16 output only: if set, x_out gets bf16(y) and x_out_lo bf16(y - bf16(y))
    int64_t N;
    int32_t H;
    int32_t D;
    double f[kMaxHeadDimHalf];  // rotation frequencies (fp64)
    float mscale;
    int64_t pos0;    // position of token 0 of x_in
};

// Arguments of the attention kernels. One warp handles one task = (set s, row i, KV head g).
struct AttnArgs {
    const void *q;         // [N][Hq][D]: fp32 rotated queries (split path) or dtype as given;
                           // with q_lo set, the bf16 high part of the rotated queries
    const void *q_lo;      // split path: bf16 low part of the rotated queries (q~ = q + q_lo), or null
    const void *k;         // [N][Hkv][D]
    const void *k_lo;      // bf16 path: low part of the rotated keys (k~ = k + k_lo), or null
    const void *v;         // [N][Hkv][D]
    void *out;             // [n_sets][N][Hq][D]
    float *lse;            // [n_sets][Hq][lse_ld]: row i at lse[(s Hq + h) lse_ld + i], or null
    int64_t lse_ld;        // N, or the row count of a call on local rows (lse then offset by -row0)
    const int64_t *row_ptr;  // [n_masks * N + 1] (null when dense)
    const void *col;       // keys (null when dense)
    const uint32_t *bitmap;  // causal bitmap rows (null when dense)
    int64_t words_per_mask;
    int64_t N;
    int32_t Hq;
    int32_t Hkv;
    int32_t G;             // Hq / Hkv
    int32_t heads_keyed;   // masks keyed per KV head (1 or Hkv)
    int32_t n_sets;        // output sets: n_seeds for per-seed masks, else 1
    int64_t row0;          // query rows row0 .. row1-1 are computed (0 and N for a whole layer)
    int64_t row1;
    // Dense-suffix split (part_o set): every key in [lo(i), i] of row i is kept, lo(i) being
    // the start of the row's Structural block of clique_B tokens (0: no blocks) and / or of its
    // forced local window of `window` keys, whichever reaches further back. The tile kernel's
    // suffix pass attends each row to those keys only and writes part_o / part_lse; the
    // register gather then starts from that partial softmax and skips the same keys, which
    // are the tail of the row's ascending key list.
    int64_t clique_B;
    float *part_o;         // [N][Hq][D] normalised partial outputs, or null
    float *part_lse;       // [N][Hq] their log2-domain log-sum-exp
    int32_t window;
    float scale_log2;      // log2(e) / sqrt(D)
    int64_t n_tasks;       // n_sets * (row1 - row0) * Hkv
    const void *v16;       // tile kernel: the values as fp16, scaled by 2^-E (launch_values_f16)
    const float *v_absmax; // tile kernel: max |v| over the values (device), from which E follows
    const float *qk_bound; // head dim 128 with rotated q / k in launch_fp8_prep's form: bounds of |q~| and |k~|
                           // (device, two floats) when the RoPE kernels wrote the fp8-correction
                           // operands (launch_fp8_prep), else null
    int64_t wait_limit;    // tile kernel: cycles a device-side wait may take (0: about 2^31)
    int32_t debug_no_loads;  // tile kernel, tests only: the loader issues no copies, so the
                             // first wait on them gives up (ris_debug_tile_stall)
};

// Arguments of the Hybrid Anchor decode kernels (one generated token at position t). The
// key set of KV head g is its anchor keys below win_lo = max(0, t - W + 1) plus the window
// win_lo .. t: chunks of kDecodeChunk anchor entries, then chunks of kDecodeChunk window
// positions, one CTA per (chunk, g). The grid does not depend on t, so t may be read from
// device memory.
constexpr int kDecodeChunk = 32;
constexpr int kMaxDecodeKvHeads = 64;

struct DecodeArgs {
    const void *q;             // [Hq][D] query of the token, not rotated (dtype)
    const void *k;             // [T][Hkv][D] rotated keys: bf16 high parts, or fp32
    const void *k_lo;          // bf16 low parts (k~ = k + k_lo), or null
    const void *v;             // [T][Hkv][D]
    const int32_t *anchor;     // anchor keys, ascending; mask m: anchor[anchor_base[m] ..] (anchor_len[m] keys)
    int64_t anchor_base[kMaxDecodeKvHeads];
    int32_t anchor_len[kMaxDecodeKvHeads];
    int64_t t0;                // first generated position (the prefill length)
    int64_t cache_len;
    int32_t heads_keyed;       // 1, or Hkv for per-head anchors
    int32_t Hq;
    int32_t Hkv;
    int32_t G;
    int32_t D;
    int32_t n_chunks;          // chunks per KV head (grid.x): partials per KV head
    int32_t n_anchor_chunks;   // the first n_anchor_chunks chunks take anchor entries
    int32_t window;            // W >= 1
    int32_t advance;           // with t_dev: the combine kernel adds 1 to *t_dev when done
    int64_t t;                 // position of the token (when t_dev is null)
    int64_t *t_dev;            // device position of the token, or null
    unsigned int *error;       // device error word: bit 1 = t outside [t0, cache_len)
    double f[kMaxHeadDimHalf]; // rotation frequencies of q (fp64)
    float mscale;
    float scale_log2;          // log2(e) / sqrt(D)
    float *part_o;             // [Hq][n_chunks][D] partial outputs (query head g * G + h)
    float2 *part_ml;           // [Hq][n_chunks] partial (max, sum) in the log2 domain
    void *out;                 // [Hq][D]
    float *lse;                // [Hq] or null
};

// Forget the allocation-free entry point's cached scratch addresses (ris_shutdown).
void noalloc_forget_addresses();

// Library-wide kernel launch counter (ris_launch_count).
void note_launch(int n = 1);

// Set the calling thread's error text (returned by ris_last_error).
void set_error_text(const char *msg);

// Launchers: each returns the launch error (cudaGetLastError) of its kernels.
cudaError_t launch_mask_bits(const MaskBitsArgs &a, cudaStream_t s);
cudaError_t launch_mask_draws(const MaskBitsArgs &a, cudaStream_t s);
cudaError_t launch_scan_inplace(int64_t *x, int64_t n, int64_t *partials, cudaStream_t s);
int64_t scan_partials_count(int64_t n);
cudaError_t launch_mask_fill(const MaskFillArgs &a, cudaStream_t s);

// Decode step: partial softmax per (chunk, KV head), then one combine per query head.
cudaError_t launch_decode(const DecodeArgs &a, int dtype, int out_dtype, cudaStream_t s);
// Reads and clears the decode error word (bit 1: a step's device-side t was out of range).
unsigned int read_decode_error();

// dtype_in / dtype_out are ris_dtype values.
cudaError_t launch_rope(const RopeArgs &a, int dtype_in, int dtype_out, cudaStream_t s);

// The pre-passes of a layer call whose scores take the fp8-correction operands (see
// fp8_score_scales in attn_common.cuh), bf16 inputs, head dim a multiple of 16, every pointer
// 16-byte aligned. Two launches: bounds of |q~|, |k~| (and max |v| when v16 is set) into
// bounds[0..2] (zeroed by this call), then RoPE of q (positions q_first .. q_first + q_rows - 1)
// and k (positions 0 .. N-1) into q_hi / q_lo and k_hi / k_lo: fp16 hi parts, and per (token,
// head) D bytes of e4m3 corrections of the hi part then D bytes of e4m3 corrections of the lo
// part; or, when the bounds rule the scheme out, the bf16 hi / lo pair. With v16 set, the values
// as fp16 scaled by 2^-E, E = v_scale_exp(bounds[2]), as launch_values_f16 writes them.
struct Fp8PrepArgs {
    const void *q, *k, *v;  // bf16 [q_rows][Hq][D], [N][Hkv][D], [N][Hkv][D]
    void *q_hi, *q_lo, *k_hi, *k_lo;
    void *v16;              // or null
    float *bounds;          // [3]
    int64_t N, q_rows, q_first;
    int32_t Hq, Hkv, D;
    double f[kMaxHeadDimHalf];  // rotation frequencies (fp64)
    float mscale;
};
cudaError_t launch_fp8_prep(const Fp8PrepArgs &a, cudaStream_t s);

// bf16 values v[n] (n a multiple of 8, 16-byte aligned) -> *vmax = max |v| (vmax zeroed by
// this call) and v16[i] = fp16(v[i] / 2^E), E = v_scale_exp(max |v|): the fp16 operand of the
// tile kernel's value product, exact for every bf16 value in fp16's normal range.
cudaError_t launch_values_f16(const void *v, int64_t n, void *v16, float *vmax, cudaStream_t s);

// q_split: q is fp32 and is split into bf16 hi + lo on the tensor-core path; a.k_lo set:
// the keys arrive as a bf16 hi + lo pair.
cudaError_t launch_attention_bf16(const AttnArgs &a, int D, int out_dtype, bool q_split, int col_bytes,
                                  bool dense, cudaStream_t s);
cudaError_t launch_attention_f32(const AttnArgs &a, int D, int out_dtype, int col_bytes, bool dense,
                                 cudaStream_t s);


// Masked dense-tile design (tcgen05, head dim 128 or 64): q_hi / q_lo bf16 query pair (q_lo
// null for exact bf16 inputs).
bool tile_design_available();
cudaError_t launch_attention_tile(const AttnArgs &a, int D, const void *q_hi, const void *q_lo, int out_dtype,
                                  bool dense, cudaStream_t s);
// The suffix pass of the dense-suffix split (a.part_o set): writes a.part_o / a.part_lse.
cudaError_t launch_attention_tile_suffix(const AttnArgs &a, int D, const void *q_hi, const void *q_lo, cudaStream_t s);
cudaError_t read_tile_error(unsigned int *out);

}  // namespace ris
