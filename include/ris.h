/*
 * ris.h -- C ABI of libris, the GB300 (sm_103a) implementation of RIS (Reduced
 * Interaction Sampling) prefill sparse self-attention, arxiv 2607.21927.
 *
 * Conventions shared by every call
 *   - Tensors are caller-owned, contiguous, token-major DEVICE pointers unless a comment
 *     says "host". q is [N][heads][head_dim], k and v are [N][kv_heads][head_dim], out is
 *     [N][heads][head_dim] (per-seed calls: [n_seeds][N][heads][head_dim]).
 *     Every device pointer must be 16-byte aligned.
 *   - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream). Calls
 *     are stream-ordered and asynchronous unless their comment says "blocks".
 *   - Each call returns a ris_status. Arguments are validated before anything is launched;
 *     an invalid call launches nothing and returns RIS_ERR_INVALID. The text of the last
 *     error of the calling thread is returned by ris_last_error(). A device fault of an
 *     earlier launch surfaces as RIS_ERR_CUDA from a later call or at the caller's sync.
 *   - There is no CPU fallback: without a CUDA device every compute call returns
 *     RIS_ERR_CUDA.
 *   - Temporary device memory is taken from the device's stream-ordered pool
 *     (cudaMallocAsync on `stream`) and released on the same stream.
 */
#ifndef RIS_H
#define RIS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    RIS_OK = 0,
    RIS_ERR_INVALID = 1,        /* bad argument; nothing was launched */
    RIS_ERR_OOM = 2,            /* device allocation failed */
    RIS_ERR_CUDA = 3,           /* a CUDA runtime call failed (or no device) */
    RIS_ERR_UNSUPPORTED = 4,    /* valid but not built (e.g. head_dim outside {64,128}) */
    RIS_ERR_DEVICE_TIMEOUT = 5  /* a bounded device-side wait gave up */
} ris_status;

/* Sampling modes (paper, Methods, "Sampling Modes: Stochastic and Structural"). */
typedef enum {
    RIS_MODE_STOCHASTIC = 0, /* the whole density budget drawn uniformly per pivot row */
    RIS_MODE_STRUCTURAL = 1, /* block cliques of B = min(0.1 N, round(d N)) + global draws */
    RIS_MODE_DENSE = 2       /* every causal pair (the dense upper bound, Table tab:results_32k) */
} ris_mode;

typedef enum { RIS_F32 = 0, RIS_BF16 = 1 } ris_dtype;

/* RoPE position extension (Methods, "Dynamic RoPE Scaling"). */
typedef enum { RIS_ROPE_NONE = 0, RIS_ROPE_PLAIN = 1, RIS_ROPE_LINEAR = 2, RIS_ROPE_YARN = 3 } ris_rope_kind;

typedef struct {
    int32_t kind;       /* ris_rope_kind */
    int32_t reserved;   /* must be 0 */
    double theta;       /* base, e.g. 1e6 (Qwen2) or 1e4 (TinyLlama) */
    int64_t native_len; /* trained positional limit, e.g. 32768 or 2048 */
    double factor;      /* extension factor s; <= 0 resolves to max(1, N / native_len) */
    double yarn_alpha;  /* YaRN ramp start in rotations per native window (default 1) */
    double yarn_beta;   /* YaRN ramp end (default 32) */
} ris_rope_cfg;

/* Forced set and keying of a mask; NULL means all defaults. */
typedef struct {
    int32_t local_window; /* W >= 1: keys i-W < j <= i always kept (1 = diagonal only, default) */
    int32_t n_anchor;     /* A >= 0: keys j < A always kept (global anchors, default 0) */
    int32_t per_head;     /* 0: one mask shared by all heads (default); 1: one mask per KV head */
    uint32_t layer_key;   /* mixed into every draw; 0 = shared across layers (default) */
    int32_t sampler;      /* random part: 0 = Bernoulli keep test per causal pair (default);
                             1 = index draws: per row and seed, `draws` indices j drawn with
                             replacement uniformly over [0, N), kept when j < i, repeats merged
                             (the torch.randint wording of Methods, "Memory-Bounded Geometry
                             Generation") */
} ris_mask_opts;

/* The paper's three-part geometry (Results, "Ensemble Stochastic Projection and Retrieval
 * Coverage"): a dense local window of 1024 tokens, a global anchor over the initial tokens
 * and the stochastic ensemble. The paper does not give the anchor count; 4 initial tokens
 * (the attention-sink count of streaming attention) is this library's reading. Use as
 * ris_mask_opts{RIS_PRESET_LOCAL_WINDOW, RIS_PRESET_ANCHORS, 0, 0, 0}. */
#define RIS_PRESET_LOCAL_WINDOW 1024
#define RIS_PRESET_ANCHORS 4

/* Derived scalars of one call, resolved on the host. */
typedef struct {
    int64_t bmax;            /* K = floor(d N + 0.5), the paper's B_max */
    int64_t block;           /* Structural block size B = max(1, min(floor(N/10), K)) */
    int64_t clique_pairs;    /* C, causal clique pairs of all blocks */
    double d_clique;         /* C / N^2 */
    double d_global;         /* max(0, d - d_clique): Structural global draw density */
    uint64_t thr;            /* keep iff Philox word < thr; 2^32 = always */
    uint32_t stream;         /* Philox counter word 2: 0 Stochastic draws, 1 Structural global */
    int32_t dense;           /* 1 when every causal pair is kept (dense mode or density 1) */
    double rope_factor;      /* resolved s */
    double rope_mscale;      /* 0.1 ln s + 1 for YaRN, else 1 */
    int64_t draws;           /* index-draw sampler: draws per row and seed, floor(d N + 0.5) for
                                Stochastic, floor(d_global N + 0.5) for Structural */
} ris_params;

/* Opaque handle to a mask held in device memory. */
typedef struct ris_mask_s *ris_mask_t;

/* Device-side layout of a mask, read by ris_mask_info. All pointers are owned by the mask.
 *   n_masks = (per_seed ? n_seeds : 1) * (per_head ? kv_heads : 1); mask m = s * heads_keyed + h.
 *   CSR: keys of row i of mask m are col[row_ptr[m*N + i] .. row_ptr[m*N + i + 1]),
 *        ascending, int64 row_ptr of n_masks*N + 1 entries, col of col_bytes (2 if N <= 65536,
 *        else 4) each.
 *   Bitmap: row i of mask m holds words floor(i/32)+1 words at
 *        bitmap + m * words_per_mask + row_word_offset(i), with
 *        row_word_offset(32a + b) = 32a + b + 16 a (a - 1) + a b; bit (j mod 32) of word j/32
 *        is pair (i, j); bits above the diagonal are zero.
 *   Dense masks (mode DENSE or density 1) store nothing: row_ptr, col and bitmap are NULL
 *   and row i holds keys 0..i. */
typedef struct {
    int64_t N;
    int32_t n_masks;
    int32_t heads_keyed;   /* 1, or kv_heads when per_head */
    int32_t n_seeds;
    int32_t per_seed;
    int32_t col_bytes;
    int32_t dense;
    int64_t n_pairs;       /* total stored pairs over all masks */
    int64_t words_per_mask;
    const int64_t *row_ptr;
    const void *col;
    const uint32_t *bitmap;
    ris_params params;
    int64_t suffix_pairs;  /* pairs per mask in the rows' dense suffixes: keys lo(i) .. i of row i,
                              all kept, lo(i) the earlier of the row's Structural block start
                              (blocks of >= 256 tokens) and its local window start (0 when the
                              mask is dense, per seed, or has neither span of >= 256); the
                              dense-suffix split attends these on the tiles */
} ris_mask_desc;

/* Resolve the scalars of a call on the host (no device work, usable without a GPU).
 * Structural geometry follows Methods, "Sampling Modes"; B_max = round(d N) matches the
 * B_max column of the sub-1% sweet-spot table. rope may be NULL (factor 1, mscale 1).
 * Returns RIS_ERR_INVALID for N < 1, density outside (0, 1], an unknown mode or rope kind. */
ris_status ris_resolve_params(int64_t N, int32_t mode, double density, const ris_rope_cfg *rope,
                              ris_params *out);

/* RoPE rotation frequencies f[head_dim/2] (host array, fp64) and the vector scale for a
 * sequence of N tokens: plain theta^(-2k/D); linear f/s; YaRN ramp between the two
 * (Methods, "Dynamic RoPE Scaling"; YaRN per Peng et al. 2023). No device work. */
ris_status ris_rope_freqs(const ris_rope_cfg *rope, int64_t N, int32_t head_dim, double *f_out,
                          double *mscale_out);

/* Build the RIS mask of N tokens (Methods, "Memory-Bounded Geometry Generation" and
 * "Sampling Modes"): for every seed, keep causal pair (i, j<i) iff Philox4x32-10 word
 * (j mod 4) of key (seed, head_key) and counter (j/4, i, stream, layer_key) is below thr
 * (opts->sampler 0), or (sampler 1) iff j < i is one of the row's `draws` indices
 * j_t = floor(u_t N / 2^32), u_t word (t mod 4) of key (seed, head_key) and counter
 * (t/4, i, stream + 2, layer_key);
 * Structural adds the block cliques; the forced local window and anchors are added; with
 * per_seed = 0 all seeds are OR-merged into one master mask, with per_seed = 1 each seed
 * keeps its own mask. Output: bitmap + CSR in device memory owned by *out_mask.
 * seeds: HOST array of n_seeds values, 1 <= n_seeds <= 256. kv_heads is used only when
 * opts->per_head = 1. Blocks: the CSR size is read back before the key lists are written.
 * The wait covers `stream` only: a mask built on a stream of its own (ordered before the
 * attention calls that read it, and freed after them) leaves work queued on other streams
 * running while the host waits.
 * Errors: RIS_ERR_INVALID (N < 1 or > 2^31, density outside (0,1], bad opts or seeds),
 * RIS_ERR_OOM, RIS_ERR_CUDA. On error *out_mask is NULL. */
ris_status ris_mask_generate(int64_t N, int32_t kv_heads, int32_t mode, double density,
                             const uint32_t *seeds, int32_t n_seeds, const ris_mask_opts *opts,
                             int32_t per_seed, ris_mask_t *out_mask, void *stream);

/* Describe a mask (host struct filled from host-side metadata; no device work). */
ris_status ris_mask_info(ris_mask_t mask, ris_mask_desc *out);

/* Release a mask's device memory, ordered on the stream it was built on. NULL is a no-op. */
ris_status ris_mask_free(ris_mask_t mask);

/* Rotate x[N][heads][head_dim] in place with RoPE (rotate-half pairs (c, c + D/2)) at
 * positions 0..N-1, then scale by mscale (Methods, "Dynamic RoPE Scaling"). Angles are
 * formed and reduced in fp64; the rotation runs in fp32; bf16 results are rounded to
 * nearest even. head_dim must be even. Errors: RIS_ERR_INVALID. */
ris_status ris_rope_apply(void *x, int32_t dtype, int64_t N, int32_t heads, int32_t head_dim,
                          const ris_rope_cfg *rope, void *stream);

/* RIS sparse attention of one layer (Methods, "Hybrid Anchor and Pre-Fusion Unified Softmax"):
 *   out[i][h] = sum_{j in M_i} softmax_j(<q~_i,h , k~_j,g> / sqrt(D)) v_j,g,  g = h / (heads/kv_heads)
 * with one softmax over the whole key set M_i of the master mask (all seeds OR-merged), q~ and
 * k~ rotated by `rope` (NULL or kind NONE: q and k are used as given). Builds the mask, runs
 * the attention and frees the mask, all on `stream`; blocks once while the mask is sized.
 * dtype: q, k, v element type; out_dtype: out element type (F32 or BF16). lse: optional
 * [heads][N] fp32 natural-log sum of exp of the scaled scores (NULL to skip).
 * head_dim in {64, 128}; heads a multiple of kv_heads; heads/kv_heads <= 8, or any group size
 * with bf16 inputs, which then always run on the tile design (the gathers carry at most 8
 * query heads per KV head; otherwise RIS_ERR_UNSUPPORTED; the decode step keeps the limit
 * of 8).
 * Errors: RIS_ERR_INVALID, RIS_ERR_UNSUPPORTED, RIS_ERR_OOM, RIS_ERR_CUDA. */
ris_status ris_sparse_attention_fwd(const void *q, const void *k, const void *v, void *out,
                                    int64_t N, int32_t heads, int32_t kv_heads, int32_t head_dim,
                                    int32_t mode, double density, const uint32_t *seeds,
                                    int32_t n_seeds, int32_t dtype, int32_t out_dtype,
                                    const ris_rope_cfg *rope, const ris_mask_opts *opts, float *lse,
                                    void *stream);

/* The attention step alone on a mask built by ris_mask_generate (the mask is built once per
 * prefill and reused by every layer, Methods, "Memory-Bounded Geometry Generation"). With a
 * per-seed mask, out is [n_seeds][N][heads][head_dim] and lse [n_seeds][heads][N].
 * kv_heads must equal the mask's kv_heads when it is keyed per head. Asynchronous.
 * Errors: as ris_sparse_attention_fwd. */
ris_status ris_attention_masked(ris_mask_t mask, const void *q, const void *k, const void *v,
                                void *out, int32_t heads, int32_t kv_heads, int32_t head_dim,
                                int32_t dtype, int32_t out_dtype, const ris_rope_cfg *rope,
                                float *lse, void *stream);

/* Ensemble of per-seed sparse views in one launch: seed s attends over F + M_s only and
 * writes out[s] (the "independent sparse views" read of Results, "Linear Interpolation";
 * union coverage of Eq. union_coverage is the OR of these views). Same arguments as
 * ris_sparse_attention_fwd; out is [n_seeds][N][heads][head_dim], lse [n_seeds][heads][N]. */
ris_status ris_ensemble_batch(const void *q, const void *k, const void *v, void *out, int64_t N,
                              int32_t heads, int32_t kv_heads, int32_t head_dim, int32_t mode,
                              double density, const uint32_t *seeds, int32_t n_seeds,
                              int32_t dtype, int32_t out_dtype, const ris_rope_cfg *rope,
                              const ris_mask_opts *opts, float *lse, void *stream);

/* Query rows row_begin .. row_end-1 of ris_attention_masked (same arguments otherwise): the
 * other rows of out and lse are left untouched, and each computed row equals the same row of
 * the whole-layer call bit for bit. K and V must still hold every position (any row may
 * attend to any earlier key). This is how one prefill is split across devices or streams:
 * query rows are independent given K, V and the counter-based mask (each device can build the
 * same mask), so each part needs no exchange. Errors: as ris_attention_masked, and
 * RIS_ERR_INVALID for an empty range or one outside [0, N). */
ris_status ris_attention_masked_rows(ris_mask_t mask, int64_t row_begin, int64_t row_end, const void *q,
                                     const void *k, const void *v, void *out, int32_t heads, int32_t kv_heads,
                                     int32_t head_dim, int32_t dtype, int32_t out_dtype, const ris_rope_cfg *rope,
                                     float *lse, void *stream);

/* Query rows row_begin .. row_end-1 of ris_attention_masked with only those rows in memory:
 * q_rows [row_end - row_begin][heads][head_dim] holds query rows row_begin .., out_rows gets
 * the same rows of the output, and lse_rows (optional) is [heads][row_end - row_begin]. K and V
 * must hold every position 0 .. N-1: this is the per-device step of a prefill split by query
 * rows in which each device holds only its own rows of q, k and v and all-gathers the layer's
 * K and V first (the paper's row independence, Methods, "Memory-Bounded Geometry Generation":
 * every device builds the same counter-based mask). Each row equals the same row of the
 * whole-layer call bit for bit. Masks built per seed are refused (RIS_ERR_UNSUPPORTED).
 * Errors: as ris_attention_masked_rows. */
ris_status ris_attention_masked_local(ris_mask_t mask, int64_t row_begin, int64_t row_end, const void *q_rows,
                                      const void *k, const void *v, void *out_rows, int32_t heads, int32_t kv_heads,
                                      int32_t head_dim, int32_t dtype, int32_t out_dtype, const ris_rope_cfg *rope,
                                      float *lse_rows, void *stream);

/* Balanced contiguous row ranges for `parts` workers: bounds[0] = 0 < bounds[1] < ... <
 * bounds[parts] = N, cut where the running sampled-pair count reaches k/parts of the total
 * (every part gets at least one row). ris_row_split takes a HOST row_ptr of N + 1 offsets
 * (no device work); ris_mask_row_split reads the mask's own counts (summed over its per-seed
 * or per-head masks; row i of a dense mask counts i + 1) and blocks. Errors: RIS_ERR_INVALID
 * (NULL, parts outside [1, N]), RIS_ERR_CUDA. */
ris_status ris_row_split(const int64_t *row_ptr, int64_t N, int32_t parts, int64_t *bounds);
ris_status ris_mask_row_split(ris_mask_t mask, int32_t parts, int64_t *bounds);

/* Allocation-free variant of ris_attention_masked: same arguments and the same results
 * within the parity tolerance (not bit for bit), with these differences.
 * The paper has no counterpart: this entry point exists for callers that may not allocate
 * device memory while a layer runs, such as an inference engine's enqueue callback that may
 * only launch work, or a server that plans all device memory at load time. They build the
 * mask once beforehand (ris_mask_generate allocates) and call this per layer.
 *   - Every mask runs on the register gather (fp32: the fp32 gather), whatever design
 *     ris_attention_masked would pick: dense and high-density masks run at gather speed, not
 *     on the tiles, and heads / kv_heads above 8 are refused (RIS_ERR_UNSUPPORTED).
 *   - Instead of the stream-ordered pool, the rotated q (fp32) and k (bf16 hi + lo, or fp32)
 *     live in one library-owned device array of 64 MiB per device. Every GPU on which the
 *     library's device code is loaded holds it until the process exits: with lazy module
 *     loading (the CUDA default) the GPUs on which a kernel of this library ran, with
 *     CUDA_MODULE_LOADING=EAGER every context that loads the library. The call needs
 *       align256(N*heads*head_dim*4) + (bf16 ? 2 : 1) * align256(N*kv_heads*head_dim*(bf16 ? 2 : 4))
 *     bytes when rope is set (none without rope) and returns RIS_ERR_INVALID, launching
 *     nothing, when that exceeds 64 MiB (about N = 9300 tokens at 12 / 2 heads of 128).
 * It calls no allocation routine. The first call in a device's context looks up the array's
 * device address (and may load the library's device code): make that first call before any
 * stream capture; a context created anew (after cudaDeviceReset) is looked up again.
 * Every call on a device shares the array and leaves its contents behind; each call writes
 * all scratch it reads, so nothing needs clearing, but calls whose GPU work overlaps (e.g.
 * on two streams) race on it and must be ordered by the caller. */
ris_status ris_attention_masked_noalloc(ris_mask_t mask, const void *q, const void *k, const void *v,
                                        void *out, int32_t heads, int32_t kv_heads, int32_t head_dim,
                                        int32_t dtype, int32_t out_dtype, const ris_rope_cfg *rope,
                                        float *lse, void *stream);

/* The allocation-free entry point's scratch array in the current device's context: its
 * device address and size in bytes (the paper has no counterpart). Looks the address up like
 * the entry point's first call does. Errors: RIS_ERR_INVALID (NULL outputs), RIS_ERR_CUDA. */
ris_status ris_noalloc_scratch_info(void **device_address, int64_t *bytes);

/* Kernel timer for measurement (off by default). While enabled, every attention kernel launch
 * (the fused QK^T -> softmax -> PV kernel of a layer, or a decode step's two kernels; not
 * RoPE or mask kernels) is bracketed by CUDA events recorded on the stream it is launched on. Enabling or disabling clears the record.
 * ris_kernel_timer_read blocks until the last recorded launch has finished, returns the summed
 * device milliseconds and the number of launches recorded since the last read, and clears
 * them. Intended for one thread at a time. Errors: RIS_ERR_INVALID (NULL outputs), RIS_ERR_CUDA. */
ris_status ris_kernel_timer_enable(int32_t enable);
ris_status ris_kernel_timer_read(double *total_ms, int64_t *launches);
/* As ris_kernel_timer_read, and also the duration of each of the first `capacity` recorded
 * launches, in launch order, into the HOST array ms_each (NULL when capacity is 0). */
ris_status ris_kernel_timer_samples(double *total_ms, int64_t *launches, double *ms_each, int64_t capacity);

/* Attention kernel design a layer call on `mask` uses for this input dtype and head_dim
 * (host-only, no device work): 0 register gather, 2 tcgen05 masked dense tiles,
 * 3 fp32 gather, 4 dense-suffix split; -1 for invalid arguments. bf16 calls use tiles when
 * the mask is dense or keeps at least 6.8% (head_dim 128) or 11.1% (head_dim 64) of the
 * causal pairs in what a gather would fetch (and always when heads/kv_heads > 8, which this
 * call does not see). The dense-suffix split applies to masks (not per seed) with Structural
 * blocks of at least 256 tokens or a local window of at least 256 keys: every key of row i
 * from the earlier of its block start and its window start up to i is kept (Methods,
 * "Sampling Modes": in-block pairs are cliques; the window is forced), so a first launch
 * attends every row to that suffix on the tiles and the register gather continues that
 * softmax over the row's other keys; the result is the same single softmax over the row's
 * whole key set. RIS_FORCE_DESIGN = gather | tile | suffix in the environment
 * overrides (benchmarking). */
int32_t ris_attention_design(ris_mask_t mask, int32_t dtype, int32_t head_dim);

/* Synchronise `stream` and report (then clear) the device error words: RIS_ERR_DEVICE_TIMEOUT
 * if a kernel's bounded wait gave up since the last call, RIS_ERR_INVALID if a decode step
 * read a position outside [t0, cache_len) from device memory, else RIS_OK. A kernel that sets
 * a word skips the rest of its work, so outputs of that launch are undefined. Blocks.
 * Errors: RIS_ERR_CUDA. */
ris_status ris_device_status(void *stream);

/* Release the library's cached per-device state (the paper has no counterpart): the kernel
 * timer's events, and the device memory that the stream-ordered pools of the devices this
 * library used keep cached (each pool is trimmed and its release threshold set back to the
 * CUDA default, 0). The allocation-free entry point's scratch array is a static device
 * array: it stays mapped until the process exits, and its address is looked up again on the
 * next call. Live masks and anchors stay valid and are still released by ris_mask_free /
 * ris_anchor_free. Testing switches (ris_debug_*) are reset. The library may be used again
 * afterwards. Call it with no library work in flight on any stream. Errors: RIS_ERR_CUDA. */
ris_status ris_shutdown(void);

/* ---- Failure injection for tests (the paper has no counterpart) ---------------------------
 * ris_debug_fail_allocation: the n-th stream-ordered device allocation the library makes from
 * now on (0 = the next one) fails as if the pool were exhausted; later ones succeed again.
 * n < 0 disarms. Every entry point must then return RIS_ERR_OOM, leave its output handle NULL
 * and release, on its stream, whatever it had allocated.
 * ris_debug_tile_stall: with no_loads = 1 the tile kernel's loader issues no copies, so its
 * first wait on them gives up after wait_limit_cycles (0 = the default, about 2^31 cycles):
 * the kernel sets its device error word, releases its tensor memory and returns, and
 * ris_device_status reports RIS_ERR_DEVICE_TIMEOUT (outputs of that launch are undefined).
 * no_loads = 0 with a nonzero limit only shortens the waits. (0, 0) restores the defaults.
 * Both switches are process-wide. Errors: RIS_ERR_INVALID. */
ris_status ris_debug_fail_allocation(int64_t n);
ris_status ris_debug_tile_stall(int32_t no_loads, int64_t wait_limit_cycles);

/* ---- Hybrid Anchor decode (Methods, "Hybrid Anchor and Pre-Fusion Unified Softmax (PFUS)") ----
 * After a prefill of n_prefill tokens, the token generated at position t >= t0 = n_prefill
 * attends, with one softmax, to the union of
 *   - the Stochastic Anchor: the key set of the first generated token, computed once and frozen.
 *     It is row t0 of the prefill's RIS mask (same mode, density, seeds, anchors n_anchor,
 *     per_head / layer_key keying and sampler; parameters resolved for n_prefill tokens)
 *     without its local window: every kept key j < t0;
 *   - the Dynamic Local Window: keys t - window < j <= t.
 * Duplicates are merged (each key counts once). The K/V cache holds the rotated keys. */
typedef struct ris_anchor_s *ris_anchor_t;

/* Build the Stochastic Anchor on the device (one mask row per KV head when opts->per_head,
 * else one) and keep a host copy of its keys for the per-step merge. opts->local_window is
 * ignored (the decode step has its own window). Blocks (reads the key count back).
 * Errors: as ris_mask_generate; RIS_ERR_INVALID also for n_prefill >= 2^31 - 1. */
ris_status ris_decode_anchor(int64_t n_prefill, int32_t kv_heads, int32_t mode, double density,
                             const uint32_t *seeds, int32_t n_seeds, const ris_mask_opts *opts,
                             ris_anchor_t *out, void *stream);

/* Layout of an anchor: t0, number of keyed lists (1 or kv_heads), total keys, and DEVICE
 * pointers to the keys (int32, ascending within each list) and the heads_keyed + 1 int64
 * offsets (list m = keys[offsets[m] .. offsets[m+1])). Any output pointer may be NULL. */
ris_status ris_anchor_info(ris_anchor_t anchor, int64_t *t0, int32_t *heads_keyed, int64_t *n_keys,
                           const int32_t **keys, const int64_t **offsets);
ris_status ris_anchor_free(ris_anchor_t anchor);

/* Rotate x [n][heads][head_dim] (dtype) at positions pos0 .. pos0+n-1 into hi (same dtype)
 * and, for bf16 when lo is not NULL, lo = bf16(y - bf16(y)) so that hi + lo carries the fp32
 * rotation to ~16 bits: the format of a rotated K cache. The extension factor is resolved
 * for n_ctx tokens (rope->factor <= 0). rope NULL or RIS_ROPE_NONE copies x (no rotation).
 * x and hi may be the same buffer. Errors: RIS_ERR_INVALID, RIS_ERR_CUDA. */
ris_status ris_rope_split(const void *x, int32_t dtype, int64_t n, int64_t pos0, int32_t heads, int32_t head_dim,
                          int64_t n_ctx, const ris_rope_cfg *rope, void *hi, void *lo, void *stream);

/* One decode step. q: [heads][head_dim] query of the token at position t, NOT rotated (the
 * kernel rotates it at position t with the extension factor of n_ctx tokens). k (+ k_lo for
 * bf16, may be NULL) and v: the cache [cache_len][kv_heads][head_dim] holding positions
 * 0 .. cache_len-1 with rotated keys (ris_rope_split); it must already hold the token t's own
 * key and value. out: [heads][head_dim] (out_dtype); lse: [heads] natural-log sum of
 * exp(score) or NULL. Scores and probabilities are fp32.
 * Position: t (host value) when t_dev is NULL; otherwise the int64 at t_dev (device memory,
 * 8-byte aligned) is read when the step runs and t is ignored, and with advance != 0 the
 * step adds 1 to *t_dev when it has finished. Nothing in the launch then depends on the
 * position, so a captured CUDA graph of a token's steps can be replayed token after token.
 * A device-side position outside [t0, cache_len) makes the step attend to nothing (undefined
 * output) and is reported by ris_device_status as RIS_ERR_INVALID.
 * Partial results live in a buffer owned by the anchor, grown by the first call of a larger
 * shape (stream-ordered pool allocation: make that call before any stream capture); steps on
 * one anchor must therefore be ordered on the GPU (one stream, or events between streams).
 * Errors: RIS_ERR_INVALID (host t outside [t0, cache_len), window < 1, shapes, pointers,
 * anchor keyed for another kv_heads, advance without t_dev), RIS_ERR_UNSUPPORTED
 * (kv_heads > 64), RIS_ERR_CUDA. */
ris_status ris_decode_step(ris_anchor_t anchor, const void *q, const void *k, const void *k_lo, const void *v,
                           int64_t cache_len, int64_t t, int64_t *t_dev, int32_t advance, int32_t window,
                           int32_t heads, int32_t kv_heads, int32_t head_dim, int32_t dtype, int32_t out_dtype,
                           int64_t n_ctx, const ris_rope_cfg *rope, void *out, float *lse, void *stream);

/* ---- Measurement support (the paper has no counterpart) -------------------------------------
 * Small kernels that measure the ceilings the attention kernels are compared against, for the
 * current device. Each allocates its own device buffers, runs on `stream` (NULL: legacy default
 * stream), synchronises it and frees what it allocated; none belongs on a hot path.
 *
 * ris_probe_l2_read: read bandwidth in GB/s (1e9 B/s) over a device buffer of `working_set`
 * bytes (1 MiB .. 4 GiB, rounded down to 256 B) that is read repeatedly, best of five launches
 * after one untimed launch. pattern 0: every thread streams 16-byte loads with a grid-wide
 * stride; pattern 1: groups of 16 threads read whole 256-byte rows at pseudo-random row
 * indices (the access pattern of the row-gathering attention kernels). Both load with .cg
 * (cached in L2 only), so a working set below the L2 size measures L2 and one well above it
 * measures HBM. Errors: RIS_ERR_INVALID (NULL gbs, size or pattern out of range), RIS_ERR_CUDA.
 *
 * ris_probe_ffma: FP32 fused multiply-add throughput in TFLOP/s (2 FLOPs per FFMA), eight
 * independent chains per thread, four 512-thread blocks per SM. Errors: RIS_ERR_INVALID,
 * RIS_ERR_CUDA.
 *
 * ris_probe_l2_bytes: L2 size in bytes as the driver reports it (cudaDevAttrL2CacheSize).
 *
 * ris_memory_stats: bytes in use now and the high-water mark of the current device's default
 * stream-ordered memory pool, from which this library takes its masks and per-call scratch
 * (the allocation-free entry point's fixed scratch is not counted). Other users of that pool
 * in the same process are counted too. reset_high_water != 0 resets the mark to zero after
 * reading it. Errors: RIS_ERR_INVALID (NULL outputs), RIS_ERR_CUDA. */
ris_status ris_probe_l2_read(int64_t working_set, int32_t pattern, double *gbs, void *stream);
ris_status ris_probe_ffma(double *tflops, void *stream);
ris_status ris_probe_l2_bytes(int64_t *bytes);
ris_status ris_memory_stats(int64_t *in_use, int64_t *high_water, int32_t reset_high_water);

/* Text of the calling thread's last error ("" if none). The string is owned by the library. */
const char *ris_last_error(void);

/* Number of kernels this library has launched since it was loaded (all threads). */
int64_t ris_launch_count(void);

/* Library version string. */
const char *ris_version(void);

#ifdef __cplusplus
}
#endif

#endif /* RIS_H */
