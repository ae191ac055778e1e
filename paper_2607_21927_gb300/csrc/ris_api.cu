// libris C ABI: argument validation, host-side parameter resolution, mask objects and the
// launch sequence of each call. Every step of the path runs in this library's kernels; this
// file only decides, allocates (stream-ordered pool) and launches.
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <utility>
#include <vector>

#include "ris_internal.h"

namespace ris {

static std::atomic<int64_t> g_launches{0};
void note_launch(int n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

cudaError_t launch_attention_bf16(const AttnArgs &a, int D, int out_dtype, bool q_split, int col_bytes,
                                  bool dense, cudaStream_t s);
cudaError_t launch_attention_f32(const AttnArgs &a, int D, int out_dtype, int col_bytes, bool dense,
                                 cudaStream_t s);

}  // namespace ris

using namespace ris;

struct ris_mask_s {
    int64_t N = 0;
    int32_t mode = 0;    // ris_mode of the call that built it
    int32_t window = 1;  // forced local window
    int64_t suffix_pairs = 0;  // pairs in the rows' dense suffixes (dense-suffix split), per mask
    int32_t n_masks = 0, heads_keyed = 1, kv_heads = 1, n_seeds = 0, per_seed = 0;
    int32_t col_bytes = 2, dense = 0;
    int64_t n_pairs = 0, words_per_mask = 0;
    int64_t *row_ptr = nullptr;
    void *col = nullptr;
    uint32_t *bitmap = nullptr;
    ris_params params{};
    cudaStream_t stream = nullptr;
};

struct ris_anchor_s {
    int64_t t0 = 0;  // position of the first generated token (the prefill length)
    int32_t heads_keyed = 1, kv_heads = 1;
    int32_t *keys = nullptr;  // device, ascending per mask
    int64_t *off = nullptr;   // device, heads_keyed + 1 offsets
    int64_t max_keys = 0;     // longest list
    std::vector<int64_t> h_off;
    void *scratch = nullptr;  // decode partials, reused by every step on this anchor
    size_t scratch_bytes = 0;
    ris_params params{};
    cudaStream_t stream = nullptr;
};

namespace {

thread_local std::string t_err;

ris_status fail(ris_status st, const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    t_err = buf;
    return st;
}

ris_status cuda_fail(cudaError_t e, const char *what)
{
    cudaGetLastError();  // clear a sticky launch error of this thread
    return fail(e == cudaErrorMemoryAllocation ? RIS_ERR_OOM : RIS_ERR_CUDA, "%s: %s", what,
                cudaGetErrorString(e));
}

#define RIS_CUDA(call)                                        \
    do {                                                      \
        cudaError_t e_ = (call);                              \
        if (e_ != cudaSuccess) return cuda_fail(e_, #call);   \
    } while (0)

// Keep freed pool memory cached in the process (the default pool would hand it back to the
// driver at every synchronisation, and re-mapping gigabytes costs milliseconds).
std::mutex g_pool_mu;
bool g_pool_done[64] = {false};

void prepare_pool_once()
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return;
    std::lock_guard<std::mutex> lk(g_pool_mu);
    bool *done = g_pool_done;
    if (done[dev]) return;
    cudaMemPool_t pool;
    if (cudaDeviceGetDefaultMemPool(&pool, dev) == cudaSuccess) {
        uint64_t thr = UINT64_MAX;
        cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &thr);
    }
    done[dev] = true;
}

// Allocation-failure injection for tests (ris_debug_fail_allocation): the number of
// stream-ordered allocations still to succeed before one fails, or -1 (off).
std::atomic<int64_t> g_fail_alloc_after{-1};

// Every stream-ordered allocation of the library goes through here.
cudaError_t pool_alloc(void **p, size_t bytes, cudaStream_t st)
{
    int64_t n = g_fail_alloc_after.load(std::memory_order_relaxed);
    while (n >= 0) {
        if (g_fail_alloc_after.compare_exchange_weak(n, n - 1, std::memory_order_relaxed)) {
            if (n == 0) {  // this is the allocation chosen to fail (once)
                *p = nullptr;
                return cudaErrorMemoryAllocation;
            }
            break;
        }
    }
    return cudaMallocAsync(p, bytes, st);
}

// Stream-ordered temporary buffer, released on its stream when it leaves scope.
struct Scratch {
    void *p = nullptr;
    cudaStream_t s = nullptr;
    cudaError_t alloc(size_t bytes, cudaStream_t st)
    {
        s = st;
        return pool_alloc(&p, bytes < 16 ? 16 : bytes, st);
    }
    ~Scratch()
    {
        if (p) cudaFreeAsync(p, s);
    }
};

// Opt-in attention-kernel timer (ris_kernel_timer_*): event pairs recorded around launches.
struct KernelTimer {
    std::mutex mu;
    bool on = false;
    std::vector<std::pair<cudaEvent_t, cudaEvent_t>> used, spare;
};
KernelTimer g_timer;

void timer_clear_locked()
{
    for (auto &e : g_timer.used) g_timer.spare.push_back(e);
    g_timer.used.clear();
}

// Returns the event pair to record around one launch, or {nullptr, nullptr} when off.
std::pair<cudaEvent_t, cudaEvent_t> timer_pair()
{
    std::lock_guard<std::mutex> lk(g_timer.mu);
    if (!g_timer.on) return {nullptr, nullptr};
    std::pair<cudaEvent_t, cudaEvent_t> e{nullptr, nullptr};
    if (!g_timer.spare.empty()) {
        e = g_timer.spare.back();
        g_timer.spare.pop_back();
    } else if (cudaEventCreate(&e.first) != cudaSuccess || cudaEventCreate(&e.second) != cudaSuccess) {
        return {nullptr, nullptr};
    }
    g_timer.used.push_back(e);
    return e;
}

// Device-side wait limit of the tile kernel in cycles (0: the default, about 2^31) and the
// test switch that makes its loader issue no copies (ris_debug_tile_stall).
std::atomic<int64_t> g_wait_limit{0};
std::atomic<int32_t> g_tile_no_loads{0};

// Kernel design override for benchmarking the designs against each other:
// RIS_FORCE_DESIGN = gather (register gather), tile (masked dense tiles) or
// suffix (the dense-suffix split, where the mask allows it).
const char *forced_design()
{
    static const std::string d = [] {
        const char *e = std::getenv("RIS_FORCE_DESIGN");
        return std::string(e ? e : "");
    }();
    return d.c_str();
}


// Union density at and above which masked dense tiles beat gathering pair by pair (bf16,
// head dim 128): a tile costs the dense causal products (an fp16 score product, two e4m3 score
// corrections and one value product) whatever the mask, a gathered pair 1.25 KB of K/V rows.
// Measured crossover on Qwen2-shaped layers (head dim 128): 6.8% of the causal pairs at
// N = 65536 and N = 32768 (tiles 13.25 / 3.34 ms per launch; the gather on the fp8 operands
// 11.38 / 2.89 ms at 5.85%, 13.15 / 3.33 ms at 6.8%); on TinyLlama-shaped layers (head dim 64, 32 query and 4 KV
// heads, N = 16384, three bf16 score products) 11.1% (tiles 1.94 ms, the gather 1.69 / 1.99 ms
// at 9.6% / 11.4%), where the tiles are half the products but the same softmax work.
constexpr double kTileDensity = 0.068;
constexpr double kTileDensity64 = 0.111;

// Shortest dense span (Structural block or local window) for which the split pays: two
// 128-key tiles.
constexpr int64_t kSuffixMin = 256;

// Dense suffix of row i: every key in [lo(i), i] is kept, where lo(i) is the start of the
// row's own Structural block (a causal clique; blocks shorter than kSuffixMin are not used)
// and / or of its forced local window, whichever reaches further back. Those keys end the
// row's ascending key list.
int64_t suffix_block(const ris_mask_s *m)
{
    return (m->mode == RIS_MODE_STRUCTURAL && m->params.block >= kSuffixMin) ? m->params.block : 0;
}

bool suffix_split_allowed(const ris_mask_s *m)
{
    return !m->dense && !m->per_seed && (suffix_block(m) > 0 || m->window >= kSuffixMin);
}

// sum of x over a <= x < b
int64_t range_sum(int64_t a, int64_t b) { return b > a ? (a + b - 1) * (b - a) / 2 : 0; }

// Pairs in all rows' dense suffixes: the suffix of row i holds i - lo(i) + 1 keys, which is
// min(i + 1, W) without blocks, and with blocks i + 1 for i < W, else max(W, i - b0 + 1).
int64_t suffix_pairs_of(int64_t N, int64_t block, int64_t W)
{
    if (W < 1) W = 1;
    if (block <= 0) return N <= W ? range_sum(1, N + 1) : range_sum(1, W + 1) + (N - W) * W;
    int64_t total = 0;
    for (int64_t b0 = 0; b0 < N; b0 += block) {
        const int64_t b1 = std::min(N, b0 + block);
        total += range_sum(b0 + 1, std::min(b1, W) + 1);                  // i < W: i + 1 keys
        const int64_t s = std::max(b0, W);                                // i >= W:
        total += std::max<int64_t>(0, std::min(b1, b0 + W) - s) * W;     //   i - b0 < W: W keys
        total += range_sum(W + 1, b1 - b0 + 1);                           //   else i - b0 + 1 keys
    }
    return total;
}

// Design of a layer call: 0 register gather, 2 masked dense tiles, 3 fp32
// gather, 4 dense-suffix split (each row's dense suffix on the tile kernel, its other keys on
// the register gather, one softmax). The gather's cost grows with the pairs it gathers (with
// the split: all but the suffixes), a tile's does not, hence the density threshold.
int design_of(const ris_mask_s *m, int32_t dtype, int32_t head_dim, int32_t group = 1)
{
    if (dtype == RIS_F32) return 3;
    if (group > 8) return 2;  // only the tiles take more than 8 query heads per KV head
    const std::string f = forced_design();
    if (f == "gather") return 0;
    const bool tiles = (head_dim == 128 || head_dim == 64) && tile_design_available();
    if (tiles && (f == "tile" || m->dense)) return 2;
    const bool split = tiles && suffix_split_allowed(m);
    if (split && f == "suffix") return 4;
    if (tiles) {
        const double causal = (double)m->n_masks * ((double)m->N * (double)(m->N + 1) / 2.0);
        const double gathered = (double)m->n_pairs - (split ? (double)m->n_masks * (double)m->suffix_pairs : 0.0);
        if (gathered >= (head_dim == 64 ? kTileDensity64 : kTileDensity) * causal) return 2;
    }
    return split ? 4 : 0;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool aligned32(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 31u) == 0; }

int64_t row_word_offset(int64_t i)
{
    const int64_t a = i >> 5, b = i & 31;
    return i + 16 * a * (a - 1) + a * b;
}

ris_status check_N(int64_t N)
{
    if (N < 1 || N > 2147483647LL) return fail(RIS_ERR_INVALID, "N=%lld outside [1, 2^31-1]", (long long)N);
    return RIS_OK;
}

ris_status check_mode_density(int32_t mode, double density)
{
    if (mode < RIS_MODE_STOCHASTIC || mode > RIS_MODE_DENSE) return fail(RIS_ERR_INVALID, "unknown mode %d", mode);
    if (!(density > 0.0 && density <= 1.0)) return fail(RIS_ERR_INVALID, "density %g outside (0, 1]", density);
    return RIS_OK;
}

ris_status check_rope(const ris_rope_cfg *r)
{
    if (r == nullptr) return RIS_OK;
    if (r->kind < RIS_ROPE_NONE || r->kind > RIS_ROPE_YARN) return fail(RIS_ERR_INVALID, "unknown rope kind %d", r->kind);
    if (r->kind == RIS_ROPE_NONE) return RIS_OK;
    if (r->reserved != 0) return fail(RIS_ERR_INVALID, "rope.reserved must be 0");
    if (!(r->theta > 1.0) || !std::isfinite(r->theta)) return fail(RIS_ERR_INVALID, "rope.theta %g must be > 1", r->theta);
    if (r->native_len < 1) return fail(RIS_ERR_INVALID, "rope.native_len must be >= 1");
    if (!std::isfinite(r->factor) || (r->factor > 0.0 && r->factor < 1.0))
        return fail(RIS_ERR_INVALID, "rope.factor %g must be <= 0 (auto) or >= 1", r->factor);
    if (r->kind == RIS_ROPE_YARN && !(r->yarn_beta > r->yarn_alpha))
        return fail(RIS_ERR_INVALID, "rope.yarn_beta must exceed rope.yarn_alpha");
    return RIS_OK;
}

ris_status check_opts(const ris_mask_opts *o)
{
    if (o == nullptr) return RIS_OK;
    if (o->local_window < 1) return fail(RIS_ERR_INVALID, "local_window %d must be >= 1", o->local_window);
    if (o->n_anchor < 0) return fail(RIS_ERR_INVALID, "n_anchor %d must be >= 0", o->n_anchor);
    if (o->per_head != 0 && o->per_head != 1) return fail(RIS_ERR_INVALID, "per_head must be 0 or 1");
    if (o->sampler != 0 && o->sampler != 1) return fail(RIS_ERR_INVALID, "sampler %d must be 0 or 1", o->sampler);
    return RIS_OK;
}

ris_status check_seeds(const uint32_t *seeds, int32_t n_seeds)
{
    if (n_seeds < 1 || n_seeds > kMaxSeeds) return fail(RIS_ERR_INVALID, "n_seeds %d outside [1, %d]", n_seeds, kMaxSeeds);
    if (seeds == nullptr) return fail(RIS_ERR_INVALID, "seeds is NULL");
    return RIS_OK;
}

// wide_groups: more than 8 query heads per KV head are allowed (the tile design, which runs
// one CTA per query head, takes them; the gathers carry at most 8 heads in a tensor-core tile)
ris_status check_shape(int32_t heads, int32_t kv_heads, int32_t head_dim, bool wide_groups = false)
{
    if (heads < 1 || kv_heads < 1) return fail(RIS_ERR_INVALID, "heads and kv_heads must be >= 1");
    if (heads % kv_heads != 0) return fail(RIS_ERR_INVALID, "heads %d not a multiple of kv_heads %d", heads, kv_heads);
    if (head_dim != 64 && head_dim != 128) return fail(RIS_ERR_INVALID, "head_dim %d not in {64, 128}", head_dim);
    if (heads / kv_heads > 8 && !wide_groups)
        return fail(RIS_ERR_UNSUPPORTED, "heads/kv_heads = %d > 8 needs bf16 inputs (tile design)",
                    heads / kv_heads);
    return RIS_OK;
}

ris_status check_dtype(int32_t dt, const char *what)
{
    if (dt != RIS_F32 && dt != RIS_BF16) return fail(RIS_ERR_INVALID, "%s %d is neither F32 nor BF16", what, dt);
    return RIS_OK;
}

ris_status check_ptr(const void *p, const char *what)
{
    if (p == nullptr) return fail(RIS_ERR_INVALID, "%s is NULL", what);
    if (!aligned16(p)) return fail(RIS_ERR_INVALID, "%s is not 16-byte aligned", what);
    return RIS_OK;
}

#define RIS_TRY(expr)                    \
    do {                                 \
        ris_status st_ = (expr);         \
        if (st_ != RIS_OK) return st_;   \
    } while (0)

uint64_t keep_threshold(double p)
{
    if (!(p > 0.0)) return 0;
    const double t = std::floor(p * 4294967296.0 + 0.5);
    return t >= 4294967296.0 ? (uint64_t(1) << 32) : (uint64_t)t;
}

double resolve_factor(const ris_rope_cfg *r, int64_t N)
{
    if (r == nullptr || r->kind == RIS_ROPE_NONE) return 1.0;
    if (r->factor > 0.0) return r->factor;
    const double s = (double)N / (double)r->native_len;
    return s > 1.0 ? s : 1.0;
}

ris_status validate_attention(const void *q, const void *k, const void *v, void *out, int32_t heads,
                              int32_t kv_heads, int32_t head_dim, int32_t dtype, int32_t out_dtype,
                              const ris_rope_cfg *rope, const float *lse, bool prefill = true)
{
    RIS_TRY(check_ptr(q, "q"));
    RIS_TRY(check_ptr(k, "k"));
    RIS_TRY(check_ptr(v, "v"));
    RIS_TRY(check_ptr(out, "out"));
    if (lse != nullptr && !aligned16(lse)) return fail(RIS_ERR_INVALID, "lse is not 16-byte aligned");
    RIS_TRY(check_shape(heads, kv_heads, head_dim, prefill && dtype == RIS_BF16 && tile_design_available()));
    RIS_TRY(check_dtype(dtype, "dtype"));
    RIS_TRY(check_dtype(out_dtype, "out_dtype"));
    RIS_TRY(check_rope(rope));
    return RIS_OK;
}

}  // namespace

namespace ris {
void set_error_text(const char *msg) { t_err = msg; }
}  // namespace ris

extern "C" {

const char *ris_last_error(void) { return t_err.c_str(); }

int64_t ris_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

const char *ris_version(void) { return "libris 0.1 (sm_103a)"; }

ris_status ris_resolve_params(int64_t N, int32_t mode, double density, const ris_rope_cfg *rope,
                              ris_params *out)
{
    RIS_TRY(check_N(N));
    RIS_TRY(check_mode_density(mode, density));
    RIS_TRY(check_rope(rope));
    if (out == nullptr) return fail(RIS_ERR_INVALID, "out is NULL");
    ris_params p{};
    p.bmax = (int64_t)std::floor(density * (double)N + 0.5);
    int64_t B = std::min<int64_t>(N / 10, p.bmax);
    if (B < 1) B = 1;
    const int64_t nb = N / B, rem = N - nb * B;
    p.block = B;
    p.clique_pairs = nb * (B * (B + 1) / 2) + rem * (rem + 1) / 2;
    p.d_clique = (double)p.clique_pairs / ((double)N * (double)N);
    p.d_global = std::max(0.0, density - p.d_clique);
    p.dense = (mode == RIS_MODE_DENSE || density >= 1.0) ? 1 : 0;
    if (p.dense) {
        p.thr = uint64_t(1) << 32;
        p.stream = 0;
    } else if (mode == RIS_MODE_STRUCTURAL) {
        p.thr = keep_threshold(p.d_global);
        p.stream = 1;
    } else {
        p.thr = keep_threshold(density);
        p.stream = 0;
    }
    p.draws = (int64_t)std::floor((mode == RIS_MODE_STRUCTURAL ? p.d_global : density) * (double)N + 0.5);
    p.rope_factor = resolve_factor(rope, N);
    p.rope_mscale = (rope != nullptr && rope->kind == RIS_ROPE_YARN) ? 0.1 * std::log(p.rope_factor) + 1.0 : 1.0;
    *out = p;
    return RIS_OK;
}

ris_status ris_rope_freqs(const ris_rope_cfg *rope, int64_t N, int32_t head_dim, double *f_out,
                          double *mscale_out)
{
    RIS_TRY(check_N(N));
    RIS_TRY(check_rope(rope));
    if (head_dim < 2 || (head_dim & 1) || head_dim > 2 * kMaxHeadDimHalf)
        return fail(RIS_ERR_INVALID, "head_dim %d must be even and <= %d", head_dim, 2 * kMaxHeadDimHalf);
    if (f_out == nullptr || mscale_out == nullptr) return fail(RIS_ERR_INVALID, "output pointer is NULL");
    const double s = resolve_factor(rope, N);
    const int kind = rope ? rope->kind : RIS_ROPE_NONE;
    const double theta = (rope && kind != RIS_ROPE_NONE) ? rope->theta : 10000.0;
    const double two_pi = 6.283185307179586476925286766559;
    for (int c = 0; c < head_dim / 2; ++c) {
        const double base = std::pow(theta, -2.0 * (double)c / (double)head_dim);
        double f = base;
        if (kind == RIS_ROPE_LINEAR) {
            f = base / s;
        } else if (kind == RIS_ROPE_YARN) {
            // rotations of this frequency inside the native window, ramped between alpha and beta
            const double r = (double)rope->native_len * base / two_pi;
            const double gmm = std::min(1.0, std::max(0.0, (r - rope->yarn_alpha) / (rope->yarn_beta - rope->yarn_alpha)));
            f = (1.0 - gmm) * (base / s) + gmm * base;
        }
        f_out[c] = f;
    }
    *mscale_out = (kind == RIS_ROPE_YARN) ? 0.1 * std::log(s) + 1.0 : 1.0;
    return RIS_OK;
}

ris_status ris_mask_generate(int64_t N, int32_t kv_heads, int32_t mode, double density, const uint32_t *seeds,
                             int32_t n_seeds, const ris_mask_opts *opts, int32_t per_seed, ris_mask_t *out_mask,
                             void *stream)
{
    if (out_mask == nullptr) return fail(RIS_ERR_INVALID, "out_mask is NULL");
    *out_mask = nullptr;
    RIS_TRY(check_N(N));
    RIS_TRY(check_mode_density(mode, density));
    RIS_TRY(check_seeds(seeds, n_seeds));
    RIS_TRY(check_opts(opts));
    if (per_seed != 0 && per_seed != 1) return fail(RIS_ERR_INVALID, "per_seed must be 0 or 1");
    const ris_mask_opts o = opts ? *opts : ris_mask_opts{1, 0, 0, 0u, 0};
    if (o.per_head && kv_heads < 1) return fail(RIS_ERR_INVALID, "kv_heads must be >= 1 with per_head");
    const int32_t heads_keyed = o.per_head ? kv_heads : 1;
    const int64_t n_masks = (int64_t)(per_seed ? n_seeds : 1) * heads_keyed;
    if (n_masks * N > 2147483647LL) return fail(RIS_ERR_INVALID, "n_masks * N exceeds 2^31-1");

    ris_params p{};
    RIS_TRY(ris_resolve_params(N, mode, density, nullptr, &p));
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);

    ris_mask_s *mk = new (std::nothrow) ris_mask_s();
    if (mk == nullptr) return fail(RIS_ERR_OOM, "host allocation failed");
    mk->N = N;
    mk->n_masks = (int32_t)n_masks;
    mk->heads_keyed = heads_keyed;
    mk->kv_heads = kv_heads;
    mk->n_seeds = n_seeds;
    mk->per_seed = per_seed;
    mk->col_bytes = N <= 65536 ? 2 : 4;
    mk->mode = mode;
    mk->window = o.local_window;
    mk->params = p;
    mk->stream = s;
    mk->suffix_pairs = suffix_pairs_of(N, suffix_block(mk), o.local_window);
    if (p.dense) {
        mk->dense = 1;
        mk->n_pairs = n_masks * (N * (N + 1) / 2);
        *out_mask = mk;
        return RIS_OK;
    }
    prepare_pool_once();
    struct Guard {
        ris_mask_s *m;
        ~Guard()
        {
            if (m) ris_mask_free(m);
        }
    } guard{mk};

    mk->words_per_mask = row_word_offset(N);
    const int64_t n_rows = n_masks * N;
    RIS_CUDA(pool_alloc((void **)&mk->bitmap, sizeof(uint32_t) * (size_t)(n_masks * mk->words_per_mask), s));
    RIS_CUDA(pool_alloc((void **)&mk->row_ptr, sizeof(int64_t) * (size_t)(n_rows + 1), s));
    RIS_CUDA(cudaMemsetAsync(mk->row_ptr, 0, sizeof(int64_t), s));

    MaskBitsArgs a{};
    a.single_row = -1;
    a.N = N;
    a.n_seeds = n_seeds;
    a.per_seed = per_seed;
    a.heads_keyed = heads_keyed;
    a.n_masks = (int32_t)n_masks;
    a.mode = mode;
    a.W = o.local_window;
    a.A = o.n_anchor;
    a.layer_key = o.layer_key;
    a.stream = p.stream;
    a.thr = p.thr;
    a.B = p.block;
    a.words_per_mask = mk->words_per_mask;
    a.bitmap = mk->bitmap;
    a.counts = mk->row_ptr + 1;
    a.draws = p.draws;
    for (int k = 0; k < n_seeds; ++k) a.seeds.v[k] = seeds[k];
    if (o.sampler == 1) {
        // index draws first, into a zeroed bitmap; the word pass then adds the forced keys
        RIS_CUDA(cudaMemsetAsync(mk->bitmap, 0, sizeof(uint32_t) * (size_t)(n_masks * mk->words_per_mask), s));
        if (p.draws > 0) RIS_CUDA(launch_mask_draws(a, s));
        a.or_existing = 1;
        a.thr = 0;
    }
    RIS_CUDA(launch_mask_bits(a, s));

    Scratch partials;
    RIS_CUDA(partials.alloc(sizeof(int64_t) * (size_t)scan_partials_count(n_rows), s));
    RIS_CUDA(launch_scan_inplace(mk->row_ptr + 1, n_rows, (int64_t *)partials.p, s));

    int64_t total = 0;
    RIS_CUDA(cudaMemcpyAsync(&total, mk->row_ptr + n_rows, sizeof(int64_t), cudaMemcpyDeviceToHost, s));
    RIS_CUDA(cudaStreamSynchronize(s));
    mk->n_pairs = total;
    RIS_CUDA(pool_alloc(&mk->col, (size_t)(total > 0 ? total : 1) * mk->col_bytes, s));

    MaskFillArgs f{};
    f.single_row = -1;
    f.N = N;
    f.n_masks = (int32_t)n_masks;
    f.col_bytes = mk->col_bytes;
    f.words_per_mask = mk->words_per_mask;
    f.bitmap = mk->bitmap;
    f.row_ptr = mk->row_ptr;
    f.col = mk->col;
    RIS_CUDA(launch_mask_fill(f, s));

    guard.m = nullptr;
    *out_mask = mk;
    return RIS_OK;
}

ris_status ris_mask_info(ris_mask_t m, ris_mask_desc *out)
{
    if (m == nullptr || out == nullptr) return fail(RIS_ERR_INVALID, "mask or out is NULL");
    ris_mask_desc d{};
    d.N = m->N;
    d.n_masks = m->n_masks;
    d.heads_keyed = m->heads_keyed;
    d.n_seeds = m->n_seeds;
    d.per_seed = m->per_seed;
    d.col_bytes = m->col_bytes;
    d.dense = m->dense;
    d.n_pairs = m->n_pairs;
    d.words_per_mask = m->words_per_mask;
    d.row_ptr = m->row_ptr;
    d.col = m->col;
    d.bitmap = m->bitmap;
    d.params = m->params;
    d.suffix_pairs = suffix_split_allowed(m) ? m->suffix_pairs : 0;
    *out = d;
    return RIS_OK;
}

ris_status ris_mask_free(ris_mask_t m)
{
    if (m == nullptr) return RIS_OK;
    cudaError_t e = cudaSuccess;
    if (m->bitmap) e = cudaFreeAsync(m->bitmap, m->stream);
    if (m->row_ptr) {
        cudaError_t e2 = cudaFreeAsync(m->row_ptr, m->stream);
        if (e == cudaSuccess) e = e2;
    }
    if (m->col) {
        cudaError_t e2 = cudaFreeAsync(m->col, m->stream);
        if (e == cudaSuccess) e = e2;
    }
    delete m;
    if (e != cudaSuccess) return cuda_fail(e, "cudaFreeAsync");
    return RIS_OK;
}

ris_status ris_rope_apply(void *x, int32_t dtype, int64_t N, int32_t heads, int32_t head_dim,
                          const ris_rope_cfg *rope, void *stream)
{
    RIS_TRY(check_ptr(x, "x"));
    RIS_TRY(check_dtype(dtype, "dtype"));
    RIS_TRY(check_N(N));
    if (heads < 1) return fail(RIS_ERR_INVALID, "heads must be >= 1");
    if (head_dim < 8 || (head_dim % 8) || head_dim > 2 * kMaxHeadDimHalf)
        return fail(RIS_ERR_INVALID, "head_dim %d must be a multiple of 8 in [8, 128]", head_dim);
    RIS_TRY(check_rope(rope));
    if (rope == nullptr || rope->kind == RIS_ROPE_NONE) return RIS_OK;
    RopeArgs a{};
    double ms = 1.0;
    RIS_TRY(ris_rope_freqs(rope, N, head_dim, a.f, &ms));
    a.x_in = x;
    a.x_out = x;
    a.N = N;
    a.H = heads;
    a.D = head_dim;
    a.mscale = (float)ms;
    RIS_CUDA(launch_rope(a, dtype, dtype, reinterpret_cast<cudaStream_t>(stream)));
    return RIS_OK;
}

namespace {

// Attention of query rows row0 .. row1-1 over an existing mask; arguments already validated.
// local: q, out and lse hold only those rows (q [rows][heads][D], out likewise, lse
// [heads][rows]); otherwise they hold all N rows. K and V always hold all N positions.
ris_status run_attention(const ris_mask_s *m, const void *q, const void *k, const void *v, void *out,
                         int32_t heads, int32_t kv_heads, int32_t head_dim, int32_t dtype, int32_t out_dtype,
                         const ris_rope_cfg *rope, float *lse, cudaStream_t s, int64_t row0 = 0, int64_t row1 = -1,
                         bool local = false)
{
    const int64_t N = m->N;
    if (row1 < 0) row1 = N;
    // Local rows: the kernels index q, out and lse by absolute row, so they are handed base
    // pointers moved back by row0 rows; only rows row0 .. row1-1 are ever addressed.
    const int64_t q_rows = local ? row1 - row0 : N, q_first = local ? row0 : 0;
    auto back = [&](const void *p, size_t row_bytes) -> const void * {
        return p == nullptr ? nullptr : static_cast<const char *>(p) - (size_t)q_first * row_bytes;
    };
    prepare_pool_once();
    const int design = design_of(m, dtype, head_dim, heads / kv_heads);
    const bool tile = design == 2, suffix = design == 4;
    const bool rotated = rope != nullptr && rope->kind != RIS_ROPE_NONE;
    // bf16 inputs rotated here at head dim 128, on the tiles, the dense-suffix split or the bf16
    // gather: fp16 + e4m3 score operands when the bounds allow (else the bf16 pairs), written
    // by launch_fp8_prep and read alike by the tile kernel and the gather (whose fp8 form
    // needs its 32-byte loads: values 32-byte aligned), per-seed sets included
    const bool tile8 = dtype == RIS_BF16 && head_dim == 128 && rotated &&
                       (tile || ((suffix || design == 0) && aligned32(v)));
    const bool q_pair = tile || suffix || tile8;  // queries as a 16-bit pair (else fp32)
    Scratch qt, qtl, kt, ktl, po, pl, v16, vmax, bound;
    const void *qu = q, *ku = k, *kl = nullptr, *q_lo = nullptr;
    bool q_split = false;
    if (rotated) {
        RopeArgs ra{};
        double ms = 1.0;
        RIS_TRY(ris_rope_freqs(rope, N, head_dim, ra.f, &ms));
        ra.N = N;
        ra.D = head_dim;
        ra.mscale = (float)ms;
        const size_t nq = (size_t)q_rows * heads * head_dim, nk = (size_t)N * kv_heads * head_dim;
        // rotated queries: fp32 (split into bf16 hi + lo by the gather kernels) or a 16-bit pair
        // (the fp8 scheme's operands, or a bf16 hi + lo pair); rotated keys in fp32, or for bf16
        // inputs a 16-bit pair
        if (q_pair) {
            RIS_CUDA(qt.alloc(nq * 2, s));
            RIS_CUDA(qtl.alloc(nq * 2, s));
        } else {
            RIS_CUDA(qt.alloc(nq * sizeof(float), s));
        }
        RIS_CUDA(kt.alloc(nk * (dtype == RIS_BF16 ? 2 : 4), s));
        if (dtype == RIS_BF16) RIS_CUDA(ktl.alloc(nk * 2, s));
        if (tile8) {
            // bounds, then the operands and the values as fp16: two launches
            RIS_CUDA(bound.alloc(3 * sizeof(float), s));
            RIS_CUDA(v16.alloc(nk * 2, s));
            Fp8PrepArgs pa{};
            pa.q = q;
            pa.k = k;
            pa.v = v;
            pa.q_hi = qt.p;
            pa.q_lo = qtl.p;
            pa.k_hi = kt.p;
            pa.k_lo = ktl.p;
            pa.v16 = v16.p;
            pa.bounds = (float *)bound.p;
            pa.N = N;
            pa.q_rows = q_rows;
            pa.q_first = q_first;
            pa.Hq = heads;
            pa.Hkv = kv_heads;
            pa.D = head_dim;
            std::memcpy(pa.f, ra.f, sizeof(pa.f));
            pa.mscale = ra.mscale;
            RIS_CUDA(launch_fp8_prep(pa, s));
        } else {
            ra.x_in = q;
            ra.x_out = qt.p;
            ra.x_out_lo = q_pair ? qtl.p : nullptr;
            ra.H = heads;
            ra.N = q_rows;
            ra.pos0 = q_first;
            RIS_CUDA(launch_rope(ra, dtype, q_pair ? RIS_BF16 : RIS_F32, s));
            ra.N = N;
            ra.pos0 = 0;
            ra.x_in = k;
            ra.x_out = kt.p;
            ra.x_out_lo = ktl.p;
            ra.H = kv_heads;
            RIS_CUDA(launch_rope(ra, dtype, dtype, s));
        }
        qu = back(qt.p, (size_t)heads * head_dim * (q_pair ? 2 : 4));
        q_lo = back(qtl.p, (size_t)heads * head_dim * 2);
        ku = kt.p;
        kl = ktl.p;
        q_split = (dtype == RIS_BF16);
    }
    if (qu == q) qu = back(q, (size_t)heads * head_dim * (dtype == RIS_BF16 ? 2 : 4));
    AttnArgs a{};
    a.q = qu;
    a.q_lo = q_pair ? q_lo : nullptr;
    a.k = ku;
    a.k_lo = kl;
    a.v = v;
    a.out = const_cast<void *>(back(out, (size_t)heads * head_dim * (out_dtype == RIS_BF16 ? 2 : 4)));
    a.lse = lse == nullptr ? nullptr : lse - q_first;
    a.lse_ld = q_rows;
    a.row_ptr = m->row_ptr;
    a.col = m->col;
    a.bitmap = m->bitmap;
    a.words_per_mask = m->words_per_mask;
    a.N = N;
    a.Hq = heads;
    a.Hkv = kv_heads;
    a.G = heads / kv_heads;
    a.heads_keyed = m->heads_keyed;
    a.n_sets = m->per_seed ? m->n_seeds : 1;
    a.scale_log2 = (float)(1.4426950408889634074 / std::sqrt((double)head_dim));
    a.wait_limit = g_wait_limit.load(std::memory_order_relaxed);
    a.debug_no_loads = g_tile_no_loads.load(std::memory_order_relaxed);
    a.row0 = row0;
    a.row1 = row1;
    a.n_tasks = (int64_t)a.n_sets * (row1 - row0) * kv_heads;
    a.qk_bound = tile8 ? (const float *)bound.p : nullptr;
    if (tile || suffix || tile8) {
        // the value products of the tile kernel and of the gather's fp8 form take the values as
        // fp16 (scaled into range), written above with the fp8 operands or here
        if (!tile8) {
            const size_t nv = (size_t)N * kv_heads * head_dim;
            RIS_CUDA(v16.alloc(nv * 2, s));
            RIS_CUDA(vmax.alloc(sizeof(float), s));
            RIS_CUDA(launch_values_f16(v, (int64_t)nv, v16.p, (float *)vmax.p, s));
        }
        a.v16 = v16.p;
        a.v_absmax = tile8 ? (const float *)bound.p + 2 : (const float *)vmax.p;
    }
    if (suffix) {
        RIS_CUDA(po.alloc((size_t)N * heads * head_dim * sizeof(float), s));
        RIS_CUDA(pl.alloc((size_t)N * heads * sizeof(float), s));
        a.clique_B = suffix_block(m);
        a.window = m->window;
        a.part_o = (float *)po.p;
        a.part_lse = (float *)pl.p;
    }
    const auto ev = timer_pair();
    if (ev.first) RIS_CUDA(cudaEventRecord(ev.first, s));
    if (tile) {
        RIS_CUDA(launch_attention_tile(a, head_dim, qu, q_lo, out_dtype, m->dense != 0, s));
    } else if (suffix) {  // the dense suffixes on the tiles, then the gather continues their softmax
        RIS_CUDA(launch_attention_tile_suffix(a, head_dim, qu, a.q_lo, s));
        RIS_CUDA(launch_attention_bf16(a, head_dim, out_dtype, q_split, m->col_bytes, false, s));
    } else if (dtype == RIS_BF16)
        RIS_CUDA(launch_attention_bf16(a, head_dim, out_dtype, q_split, m->col_bytes, m->dense != 0, s));
    else
        RIS_CUDA(launch_attention_f32(a, head_dim, out_dtype, m->col_bytes, m->dense != 0, s));
    if (ev.second) RIS_CUDA(cudaEventRecord(ev.second, s));
    return RIS_OK;
}

ris_status fwd_common(const void *q, const void *k, const void *v, void *out, int64_t N, int32_t heads,
                      int32_t kv_heads, int32_t head_dim, int32_t mode, double density, const uint32_t *seeds,
                      int32_t n_seeds, int32_t dtype, int32_t out_dtype, const ris_rope_cfg *rope,
                      const ris_mask_opts *opts, float *lse, void *stream, int32_t per_seed)
{
    RIS_TRY(validate_attention(q, k, v, out, heads, kv_heads, head_dim, dtype, out_dtype, rope, lse));
    RIS_TRY(check_N(N));
    RIS_TRY(check_mode_density(mode, density));
    RIS_TRY(check_seeds(seeds, n_seeds));
    RIS_TRY(check_opts(opts));
    ris_mask_t m = nullptr;
    RIS_TRY(ris_mask_generate(N, kv_heads, mode, density, seeds, n_seeds, opts, per_seed, &m, stream));
    const ris_status st = run_attention(m, q, k, v, out, heads, kv_heads, head_dim, dtype, out_dtype, rope, lse,
                                        reinterpret_cast<cudaStream_t>(stream));
    const std::string keep = t_err;
    const ris_status st2 = ris_mask_free(m);
    if (st != RIS_OK) {
        t_err = keep;
        return st;
    }
    return st2;
}

}  // namespace

ris_status ris_kernel_timer_enable(int32_t enable)
{
    std::lock_guard<std::mutex> lk(g_timer.mu);
    timer_clear_locked();
    g_timer.on = enable != 0;
    return RIS_OK;
}

ris_status ris_kernel_timer_samples(double *total_ms, int64_t *launches, double *ms_each, int64_t capacity)
{
    if (total_ms == nullptr || launches == nullptr) return fail(RIS_ERR_INVALID, "output pointer is NULL");
    if (capacity < 0 || (capacity > 0 && ms_each == nullptr)) return fail(RIS_ERR_INVALID, "ms_each / capacity");
    std::lock_guard<std::mutex> lk(g_timer.mu);
    double tot = 0.0;
    int64_t k = 0;
    for (auto &e : g_timer.used) {
        RIS_CUDA(cudaEventSynchronize(e.second));
        float ms = 0.f;
        RIS_CUDA(cudaEventElapsedTime(&ms, e.first, e.second));
        tot += ms;
        if (k < capacity) ms_each[k] = ms;
        ++k;
    }
    *total_ms = tot;
    *launches = (int64_t)g_timer.used.size();
    timer_clear_locked();
    return RIS_OK;
}

ris_status ris_kernel_timer_read(double *total_ms, int64_t *launches)
{
    return ris_kernel_timer_samples(total_ms, launches, nullptr, 0);
}

int32_t ris_attention_design(ris_mask_t mask, int32_t dtype, int32_t head_dim)
{
    if (mask == nullptr || (dtype != RIS_F32 && dtype != RIS_BF16) || (head_dim != 64 && head_dim != 128)) return -1;
    return design_of(mask, dtype, head_dim);
}

ris_status ris_device_status(void *stream)
{
    unsigned int word = 0, tile_word = 0;
    RIS_CUDA(cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)));
    RIS_CUDA(read_tile_error(&tile_word));
    const unsigned int decode_word = read_decode_error();
    word |= tile_word;
    if (word != 0u) return fail(RIS_ERR_DEVICE_TIMEOUT, "a device-side wait gave up (error word 0x%x)", word);
    if (decode_word != 0u)
        return fail(RIS_ERR_INVALID, "a decode step read a position outside [t0, cache_len) from t_dev");
    return RIS_OK;
}

ris_status ris_shutdown(void)
{
    {
        std::lock_guard<std::mutex> lk(g_timer.mu);
        timer_clear_locked();
        for (auto &e : g_timer.spare) {
            cudaEventDestroy(e.first);
            cudaEventDestroy(e.second);
        }
        g_timer.spare.clear();
        g_timer.on = false;
    }
    cudaError_t first = cudaSuccess;
    {
        std::lock_guard<std::mutex> lk(g_pool_mu);
        for (int dev = 0; dev < 64; ++dev) {
            if (!g_pool_done[dev]) continue;
            cudaMemPool_t pool;
            cudaError_t e = cudaDeviceGetDefaultMemPool(&pool, dev);
            if (e == cudaSuccess) {
                uint64_t thr = 0;  // the CUDA default: cached memory goes back at each synchronisation
                e = cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &thr);
                if (e == cudaSuccess) e = cudaMemPoolTrimTo(pool, 0);
            }
            if (e != cudaSuccess && first == cudaSuccess) first = e;
            g_pool_done[dev] = false;
        }
    }
    noalloc_forget_addresses();
    g_fail_alloc_after.store(-1);
    g_wait_limit.store(0);
    g_tile_no_loads.store(0);
    if (first != cudaSuccess) return cuda_fail(first, "releasing the memory pool cache");
    return RIS_OK;
}

ris_status ris_debug_fail_allocation(int64_t n)
{
    g_fail_alloc_after.store(n < 0 ? -1 : n);
    return RIS_OK;
}

ris_status ris_debug_tile_stall(int32_t no_loads, int64_t wait_limit_cycles)
{
    if (no_loads != 0 && no_loads != 1) return fail(RIS_ERR_INVALID, "no_loads must be 0 or 1");
    if (wait_limit_cycles < 0) return fail(RIS_ERR_INVALID, "wait_limit_cycles must be >= 0");
    g_wait_limit.store(wait_limit_cycles);
    g_tile_no_loads.store(no_loads);
    return RIS_OK;
}

ris_status ris_attention_masked(ris_mask_t mask, const void *q, const void *k, const void *v, void *out,
                                int32_t heads, int32_t kv_heads, int32_t head_dim, int32_t dtype,
                                int32_t out_dtype, const ris_rope_cfg *rope, float *lse, void *stream)
{
    if (mask == nullptr) return fail(RIS_ERR_INVALID, "mask is NULL");
    RIS_TRY(validate_attention(q, k, v, out, heads, kv_heads, head_dim, dtype, out_dtype, rope, lse));
    if (mask->heads_keyed > 1 && mask->heads_keyed != kv_heads)
        return fail(RIS_ERR_INVALID, "mask keyed for %d KV heads, call has %d", mask->heads_keyed, kv_heads);
    return run_attention(mask, q, k, v, out, heads, kv_heads, head_dim, dtype, out_dtype, rope, lse,
                         reinterpret_cast<cudaStream_t>(stream));
}

ris_status ris_attention_masked_rows(ris_mask_t mask, int64_t row_begin, int64_t row_end, const void *q,
                                     const void *k, const void *v, void *out, int32_t heads, int32_t kv_heads,
                                     int32_t head_dim, int32_t dtype, int32_t out_dtype, const ris_rope_cfg *rope,
                                     float *lse, void *stream)
{
    if (mask == nullptr) return fail(RIS_ERR_INVALID, "mask is NULL");
    RIS_TRY(validate_attention(q, k, v, out, heads, kv_heads, head_dim, dtype, out_dtype, rope, lse));
    if (mask->heads_keyed > 1 && mask->heads_keyed != kv_heads)
        return fail(RIS_ERR_INVALID, "mask keyed for %d KV heads, call has %d", mask->heads_keyed, kv_heads);
    if (row_begin < 0 || row_end > mask->N || row_begin >= row_end)
        return fail(RIS_ERR_INVALID, "rows [%lld, %lld) not a non-empty range of [0, %lld)", (long long)row_begin,
                    (long long)row_end, (long long)mask->N);
    return run_attention(mask, q, k, v, out, heads, kv_heads, head_dim, dtype, out_dtype, rope, lse,
                         reinterpret_cast<cudaStream_t>(stream), row_begin, row_end);
}

ris_status ris_attention_masked_local(ris_mask_t mask, int64_t row_begin, int64_t row_end, const void *q_rows,
                                      const void *k, const void *v, void *out_rows, int32_t heads, int32_t kv_heads,
                                      int32_t head_dim, int32_t dtype, int32_t out_dtype, const ris_rope_cfg *rope,
                                      float *lse_rows, void *stream)
{
    if (mask == nullptr) return fail(RIS_ERR_INVALID, "mask is NULL");
    RIS_TRY(validate_attention(q_rows, k, v, out_rows, heads, kv_heads, head_dim, dtype, out_dtype, rope, lse_rows));
    if (mask->heads_keyed > 1 && mask->heads_keyed != kv_heads)
        return fail(RIS_ERR_INVALID, "mask keyed for %d KV heads, call has %d", mask->heads_keyed, kv_heads);
    if (row_begin < 0 || row_end > mask->N || row_begin >= row_end)
        return fail(RIS_ERR_INVALID, "rows [%lld, %lld) not a non-empty range of [0, %lld)", (long long)row_begin,
                    (long long)row_end, (long long)mask->N);
    if (mask->per_seed) return fail(RIS_ERR_UNSUPPORTED, "local rows of a per-seed mask (use ris_attention_masked_rows)");
    return run_attention(mask, q_rows, k, v, out_rows, heads, kv_heads, head_dim, dtype, out_dtype, rope, lse_rows,
                         reinterpret_cast<cudaStream_t>(stream), row_begin, row_end, true);
}

ris_status ris_row_split(const int64_t *row_ptr, int64_t N, int32_t parts, int64_t *bounds)
{
    if (row_ptr == nullptr || bounds == nullptr) return fail(RIS_ERR_INVALID, "row_ptr or bounds is NULL");
    RIS_TRY(check_N(N));
    if (parts < 1 || parts > N) return fail(RIS_ERR_INVALID, "parts %d outside [1, N]", parts);
    // cut k: the first row whose prefix of pairs reaches k / parts of the total (each part
    // gets at least one row)
    const int64_t total = row_ptr[N] - row_ptr[0];
    bounds[0] = 0;
    int64_t r = 0;
    for (int32_t k = 1; k < parts; ++k) {
        const double target = (double)total * k / parts;
        while (r < N && (double)(row_ptr[r] - row_ptr[0]) < target) ++r;
        int64_t c = r;
        if (c < bounds[k - 1] + 1) c = bounds[k - 1] + 1;
        if (c > N - (parts - k)) c = N - (parts - k);
        bounds[k] = c;
    }
    bounds[parts] = N;
    return RIS_OK;
}

ris_status ris_mask_row_split(ris_mask_t mask, int32_t parts, int64_t *bounds)
{
    if (mask == nullptr || bounds == nullptr) return fail(RIS_ERR_INVALID, "mask or bounds is NULL");
    const int64_t N = mask->N;
    if (parts < 1 || parts > N) return fail(RIS_ERR_INVALID, "parts %d outside [1, N]", parts);
    std::vector<int64_t> rp((size_t)N + 1);
    RIS_CUDA(cudaStreamSynchronize(mask->stream));
    if (mask->dense) {
        for (int64_t i = 0; i <= N; ++i) rp[(size_t)i] = i * (i + 1) / 2;  // row i holds keys 0..i
    } else {
        // per-seed or per-head masks: the cost of row i is summed over the masks
        std::vector<int64_t> all((size_t)(mask->n_masks * N + 1));
        RIS_CUDA(cudaMemcpy(all.data(), mask->row_ptr, sizeof(int64_t) * all.size(), cudaMemcpyDeviceToHost));
        rp[0] = 0;
        for (int64_t i = 0; i < N; ++i) {
            int64_t c = 0;
            for (int32_t mm = 0; mm < mask->n_masks; ++mm)
                c += all[(size_t)(mm * N + i + 1)] - all[(size_t)(mm * N + i)];
            rp[(size_t)i + 1] = rp[(size_t)i] + c;
        }
    }
    return ris_row_split(rp.data(), N, parts, bounds);
}

ris_status ris_sparse_attention_fwd(const void *q, const void *k, const void *v, void *out, int64_t N,
                                    int32_t heads, int32_t kv_heads, int32_t head_dim, int32_t mode,
                                    double density, const uint32_t *seeds, int32_t n_seeds, int32_t dtype,
                                    int32_t out_dtype, const ris_rope_cfg *rope, const ris_mask_opts *opts,
                                    float *lse, void *stream)
{
    return fwd_common(q, k, v, out, N, heads, kv_heads, head_dim, mode, density, seeds, n_seeds, dtype,
                      out_dtype, rope, opts, lse, stream, 0);
}

ris_status ris_ensemble_batch(const void *q, const void *k, const void *v, void *out, int64_t N, int32_t heads,
                              int32_t kv_heads, int32_t head_dim, int32_t mode, double density,
                              const uint32_t *seeds, int32_t n_seeds, int32_t dtype, int32_t out_dtype,
                              const ris_rope_cfg *rope, const ris_mask_opts *opts, float *lse, void *stream)
{
    return fwd_common(q, k, v, out, N, heads, kv_heads, head_dim, mode, density, seeds, n_seeds, dtype,
                      out_dtype, rope, opts, lse, stream, 1);
}

// ---------------------------------------------------------------- Hybrid Anchor decode
ris_status ris_decode_anchor(int64_t n_prefill, int32_t kv_heads, int32_t mode, double density,
                             const uint32_t *seeds, int32_t n_seeds, const ris_mask_opts *opts, ris_anchor_t *out,
                             void *stream)
{
    if (out == nullptr) return fail(RIS_ERR_INVALID, "out is NULL");
    *out = nullptr;
    RIS_TRY(check_N(n_prefill));
    if (n_prefill >= 2147483647LL) return fail(RIS_ERR_INVALID, "n_prefill must be < 2^31 - 1");
    RIS_TRY(check_mode_density(mode, density));
    RIS_TRY(check_seeds(seeds, n_seeds));
    RIS_TRY(check_opts(opts));
    const ris_mask_opts o = opts ? *opts : ris_mask_opts{1, 0, 0, 0u, 0};
    if (o.per_head && (kv_heads < 1 || kv_heads > kMaxDecodeKvHeads))
        return fail(RIS_ERR_INVALID, "kv_heads %d outside [1, %d]", kv_heads, kMaxDecodeKvHeads);
    ris_params p{};
    RIS_TRY(ris_resolve_params(n_prefill, mode, density, nullptr, &p));
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const int32_t hk = o.per_head ? kv_heads : 1;
    const int64_t t0 = n_prefill;

    ris_anchor_s *an = new (std::nothrow) ris_anchor_s();
    if (an == nullptr) return fail(RIS_ERR_OOM, "host allocation failed");
    struct Guard {
        ris_anchor_s *a;
        ~Guard()
        {
            if (a) ris_anchor_free(a);
        }
    } guard{an};
    an->t0 = t0;
    an->heads_keyed = hk;
    an->kv_heads = kv_heads;
    an->params = p;
    an->stream = s;
    prepare_pool_once();
    RIS_CUDA(pool_alloc((void **)&an->off, sizeof(int64_t) * (size_t)(hk + 1), s));
    // row t0 of the prefill's mask, without its local window (the decode window replaces it);
    // the dense mode keeps every earlier key
    const int64_t words = (t0 >> 5) + 1;
    Scratch bits, partials;
    RIS_CUDA(bits.alloc(sizeof(uint32_t) * (size_t)(hk * words), s));
    MaskBitsArgs a{};
    a.single_row = t0;
    a.N = n_prefill;
    a.n_seeds = n_seeds;
    a.per_seed = 0;
    a.heads_keyed = hk;
    a.n_masks = hk;
    a.mode = mode;
    a.W = 0;
    a.A = o.n_anchor;
    a.layer_key = o.layer_key;
    a.stream = p.stream;
    a.thr = p.dense ? (uint64_t(1) << 32) : p.thr;
    a.mode = p.dense ? RIS_MODE_STOCHASTIC : mode;
    a.B = p.block;
    a.draws = p.draws;
    a.words_per_mask = words;
    a.bitmap = (uint32_t *)bits.p;
    a.counts = an->off + 1;
    for (int k = 0; k < n_seeds; ++k) a.seeds.v[k] = seeds[k];
    if (o.sampler == 1 && !p.dense) {
        RIS_CUDA(cudaMemsetAsync(bits.p, 0, sizeof(uint32_t) * (size_t)(hk * words), s));
        if (p.draws > 0) RIS_CUDA(launch_mask_draws(a, s));
        a.or_existing = 1;
        a.thr = 0;
    }
    RIS_CUDA(cudaMemsetAsync(an->off, 0, sizeof(int64_t), s));
    RIS_CUDA(launch_mask_bits(a, s));
    RIS_CUDA(partials.alloc(sizeof(int64_t) * (size_t)scan_partials_count(hk), s));
    RIS_CUDA(launch_scan_inplace(an->off + 1, hk, (int64_t *)partials.p, s));
    an->h_off.resize((size_t)hk + 1);
    RIS_CUDA(cudaMemcpyAsync(an->h_off.data(), an->off, sizeof(int64_t) * (size_t)(hk + 1), cudaMemcpyDeviceToHost, s));
    RIS_CUDA(cudaStreamSynchronize(s));
    const int64_t total = an->h_off[hk];
    RIS_CUDA(pool_alloc((void **)&an->keys, sizeof(int32_t) * (size_t)(total > 0 ? total : 1), s));
    MaskFillArgs f{};
    f.single_row = t0;
    f.N = n_prefill;
    f.n_masks = hk;
    f.col_bytes = 4;
    f.words_per_mask = words;
    f.bitmap = (const uint32_t *)bits.p;
    f.row_ptr = an->off;
    f.col = an->keys;
    RIS_CUDA(launch_mask_fill(f, s));
    for (int32_t m = 0; m < hk; ++m) an->max_keys = std::max(an->max_keys, an->h_off[m + 1] - an->h_off[m]);
    RIS_CUDA(cudaStreamSynchronize(s));
    guard.a = nullptr;
    *out = an;
    return RIS_OK;
}

ris_status ris_anchor_info(ris_anchor_t anchor, int64_t *t0, int32_t *heads_keyed, int64_t *n_keys,
                           const int32_t **keys, const int64_t **offsets)
{
    if (anchor == nullptr) return fail(RIS_ERR_INVALID, "anchor is NULL");
    if (t0) *t0 = anchor->t0;
    if (heads_keyed) *heads_keyed = anchor->heads_keyed;
    if (n_keys) *n_keys = anchor->h_off.empty() ? 0 : anchor->h_off.back();
    if (keys) *keys = anchor->keys;
    if (offsets) *offsets = anchor->off;
    return RIS_OK;
}

ris_status ris_anchor_free(ris_anchor_t anchor)
{
    if (anchor == nullptr) return RIS_OK;
    cudaError_t e = cudaSuccess;
    for (void *p : {(void *)anchor->keys, (void *)anchor->off, anchor->scratch}) {
        if (p == nullptr) continue;
        cudaError_t e2 = cudaFreeAsync(p, anchor->stream);
        if (e == cudaSuccess) e = e2;
    }
    delete anchor;
    if (e != cudaSuccess) return cuda_fail(e, "cudaFreeAsync");
    return RIS_OK;
}

ris_status ris_rope_split(const void *x, int32_t dtype, int64_t n, int64_t pos0, int32_t heads, int32_t head_dim,
                          int64_t n_ctx, const ris_rope_cfg *rope, void *hi, void *lo, void *stream)
{
    RIS_TRY(check_ptr(x, "x"));
    RIS_TRY(check_ptr(hi, "hi"));
    RIS_TRY(check_dtype(dtype, "dtype"));
    RIS_TRY(check_N(n));
    RIS_TRY(check_N(n_ctx));
    if (pos0 < 0 || pos0 + n > 2147483647LL) return fail(RIS_ERR_INVALID, "positions outside [0, 2^31-1)");
    if (heads < 1) return fail(RIS_ERR_INVALID, "heads must be >= 1");
    if (head_dim < 8 || (head_dim % 8) || head_dim > 2 * kMaxHeadDimHalf)
        return fail(RIS_ERR_INVALID, "head_dim %d must be a multiple of 8 in [8, 128]", head_dim);
    if (dtype == RIS_F32 && lo != nullptr) return fail(RIS_ERR_INVALID, "lo must be NULL for fp32");
    if (lo != nullptr && !aligned16(lo)) return fail(RIS_ERR_INVALID, "lo is not 16-byte aligned");
    RIS_TRY(check_rope(rope));
    RopeArgs a{};
    double ms = 1.0;
    if (rope != nullptr && rope->kind != RIS_ROPE_NONE) RIS_TRY(ris_rope_freqs(rope, n_ctx, head_dim, a.f, &ms));
    a.x_in = x;
    a.x_out = hi;
    a.x_out_lo = lo;
    a.N = n;
    a.H = heads;
    a.D = head_dim;
    a.mscale = (float)ms;
    a.pos0 = pos0;
    RIS_CUDA(launch_rope(a, dtype, dtype, reinterpret_cast<cudaStream_t>(stream)));
    return RIS_OK;
}

ris_status ris_decode_step(ris_anchor_t anchor, const void *q, const void *k, const void *k_lo, const void *v,
                           int64_t cache_len, int64_t t, int64_t *t_dev, int32_t advance, int32_t window,
                           int32_t heads, int32_t kv_heads, int32_t head_dim, int32_t dtype, int32_t out_dtype,
                           int64_t n_ctx, const ris_rope_cfg *rope, void *out, float *lse, void *stream)
{
    if (anchor == nullptr) return fail(RIS_ERR_INVALID, "anchor is NULL");
    RIS_TRY(validate_attention(q, k, v, out, heads, kv_heads, head_dim, dtype, out_dtype, rope, lse, false));
    if (k_lo != nullptr && (dtype != RIS_BF16 || !aligned16(k_lo)))
        return fail(RIS_ERR_INVALID, "k_lo must be NULL for fp32 and 16-byte aligned for bf16");
    if (kv_heads > kMaxDecodeKvHeads) return fail(RIS_ERR_UNSUPPORTED, "kv_heads %d > %d", kv_heads, kMaxDecodeKvHeads);
    if (anchor->heads_keyed > 1 && anchor->heads_keyed != kv_heads)
        return fail(RIS_ERR_INVALID, "anchor keyed for %d KV heads, call has %d", anchor->heads_keyed, kv_heads);
    if (cache_len <= anchor->t0 || cache_len > 2147483647LL)
        return fail(RIS_ERR_INVALID, "cache_len=%lld must exceed t0=%lld and be < 2^31", (long long)cache_len,
                    (long long)anchor->t0);
    if (t_dev == nullptr && (t < anchor->t0 || t >= cache_len))
        return fail(RIS_ERR_INVALID, "t=%lld outside [t0=%lld, cache_len=%lld)", (long long)t, (long long)anchor->t0,
                    (long long)cache_len);
    if (t_dev != nullptr && (reinterpret_cast<uintptr_t>(t_dev) & 7u))
        return fail(RIS_ERR_INVALID, "t_dev is not 8-byte aligned");
    if (advance != 0 && t_dev == nullptr) return fail(RIS_ERR_INVALID, "advance needs t_dev");
    if (window < 1) return fail(RIS_ERR_INVALID, "window %d must be >= 1", window);
    RIS_TRY(check_N(n_ctx));

    DecodeArgs a{};
    a.q = q;
    a.k = k;
    a.k_lo = k_lo;
    a.v = v;
    a.anchor = anchor->keys;
    for (int32_t m = 0; m < anchor->heads_keyed; ++m) {
        a.anchor_base[m] = anchor->h_off[m];
        a.anchor_len[m] = (int32_t)(anchor->h_off[m + 1] - anchor->h_off[m]);
    }
    a.t0 = anchor->t0;
    a.cache_len = cache_len;
    a.heads_keyed = anchor->heads_keyed;
    a.Hq = heads;
    a.Hkv = kv_heads;
    a.G = heads / kv_heads;
    a.D = head_dim;
    a.window = window;
    a.advance = advance;
    a.t = t;
    a.t_dev = t_dev;
    // anchor chunks cover the longest list, window chunks a full window, whatever t is
    a.n_anchor_chunks = (int32_t)((anchor->max_keys + kDecodeChunk - 1) / kDecodeChunk);
    const int64_t chunks = a.n_anchor_chunks + ((int64_t)window + kDecodeChunk - 1) / kDecodeChunk;
    a.n_chunks = (int32_t)chunks;
    double ms = 1.0;
    if (rope != nullptr && rope->kind != RIS_ROPE_NONE) RIS_TRY(ris_rope_freqs(rope, n_ctx, head_dim, a.f, &ms));
    a.mscale = (float)ms;
    // the keys were rotated with the same scale: scores carry mscale^2
    a.scale_log2 = (float)(1.4426950408889634074 / std::sqrt((double)head_dim));
    a.out = out;
    a.lse = lse;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const size_t slots = (size_t)kv_heads * a.n_chunks * a.G;
    const size_t o_bytes = (sizeof(float) * slots * head_dim + 255) & ~size_t(255);
    const size_t need = o_bytes + sizeof(float2) * slots;
    if (need > anchor->scratch_bytes) {
        // grow the anchor's partials buffer (stream-ordered; the first call of a shape allocates)
        prepare_pool_once();
        if (anchor->scratch) RIS_CUDA(cudaFreeAsync(anchor->scratch, s));
        anchor->scratch = nullptr;
        anchor->scratch_bytes = 0;
        RIS_CUDA(pool_alloc(&anchor->scratch, need, s));
        anchor->scratch_bytes = need;
        anchor->stream = s;
    }
    a.part_o = (float *)anchor->scratch;
    a.part_ml = (float2 *)((char *)anchor->scratch + o_bytes);
    const auto ev = timer_pair();
    if (ev.first) RIS_CUDA(cudaEventRecord(ev.first, s));
    RIS_CUDA(launch_decode(a, dtype, out_dtype, s));
    if (ev.second) RIS_CUDA(cudaEventRecord(ev.second, s));
    return RIS_OK;
}

}  // extern "C"
