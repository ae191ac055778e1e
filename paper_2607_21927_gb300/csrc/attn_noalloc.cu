// ris_attention_masked_noalloc: the attention step on a prebuilt mask without any device
// allocation.
//
// Who needs it: callers that may not allocate device memory while they run a layer, e.g.
// an inference engine's enqueue callback that must only launch work, or a server that
// plans its whole memory budget at load time and forbids cudaMalloc afterwards (allocation
// can block, synchronise or fail under fragmentation in the middle of a request). They
// build the mask once at set-up (ris_mask_generate allocates) and call this per layer.
//
// The rotated queries (fp32) and keys (bf16 hi + lo, or fp32) that ris_attention_masked
// takes from the stream-ordered pool live here in one file-scope device array of
// kNoAllocScratchBytes. Every GPU on which this library's device code is loaded holds it
// until the process exits: with the default lazy module loading only GPUs on which this
// entry point (or another kernel of the library) ran, with CUDA_MODULE_LOADING=EAGER every
// context that loads the library. The array is shared by every call on a device and keeps the
// last call's contents; this entry point writes every byte it later reads within the same
// call, so nothing has to be cleared, but calls whose work overlaps on the GPU (for
// example on two streams) race on it and must be ordered by the caller.
//
// Every layer runs on the register gather (or the fp32 gather), whatever design
// ris_attention_masked would pick: the tile and dense-suffix designs need more scratch
// (the suffix pass's partial outputs) than the array holds at useful sizes. The results
// agree with ris_attention_masked within the parity tolerance, not bit for bit.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <mutex>

#include "ris_internal.h"

namespace ris {

cudaError_t launch_attention_bf16(const AttnArgs &a, int D, int out_dtype, bool q_split, int col_bytes,
                                  bool dense, cudaStream_t s);
cudaError_t launch_attention_f32(const AttnArgs &a, int D, int out_dtype, int col_bytes, bool dense,
                                 cudaStream_t s);

constexpr size_t kNoAllocScratchBytes = size_t(64) << 20;  // 64 MiB per device

// The scratch itself. In host code this name is only a host-side stand-in, never a device
// address: kernels receive the address that scratch_address() looks up.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

namespace {

// Errors go to the same per-thread text that ris_last_error() returns.
ris_status na_fail(ris_status st, const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    set_error_text(buf);
    return st;
}

// Unique ID of the calling thread's current CUDA context (0 if none or unknown). Context
// IDs are never reused within a process, unlike context handles.
unsigned long long current_context_id()
{
    using GetCurrent = CUresult (*)(CUcontext *);
    using GetId = CUresult (*)(CUcontext, unsigned long long *);
    static std::once_flag once;
    static GetCurrent get_current = nullptr;
    static GetId get_id = nullptr;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_current = reinterpret_cast<GetCurrent>(p);
        p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<GetId>(p);
    });
    CUcontext c = nullptr;
    unsigned long long id = 0;
    if (get_current == nullptr || get_id == nullptr || get_current(&c) != CUDA_SUCCESS || c == nullptr) return 0;
    if (get_id(c, &id) != CUDA_SUCCESS) return 0;
    return id;
}

// Device address of the scratch array in the current device's context (host code must not
// use the array's name as an address). The lookup is made once per (device, context): a
// context torn down and created again (cudaDeviceReset, then later use) maps the array at a
// new address, so a cached address is reused only while the same context is current.
std::mutex g_addr_mu;
void *g_addr[64] = {nullptr};
unsigned long long g_ctx_of[64] = {0};

ris_status scratch_address(void **out)
{
    std::mutex &mu = g_addr_mu;
    void **addr = g_addr;
    unsigned long long *ctx_of = g_ctx_of;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return na_fail(RIS_ERR_CUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
    if (dev < 0 || dev >= 64) return na_fail(RIS_ERR_UNSUPPORTED, "device ordinal %d >= 64", dev);
    std::lock_guard<std::mutex> lk(mu);
    const unsigned long long ctx = current_context_id();
    if (addr[dev] == nullptr || ctx == 0 || ctx != ctx_of[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || p == nullptr) {
            cudaGetLastError();
            addr[dev] = nullptr;
            return na_fail(RIS_ERR_CUDA, "cudaGetSymbolAddress(scratch): %s", cudaGetErrorString(e));
        }
        addr[dev] = p;
        ctx_of[dev] = current_context_id();  // the lookup has made the runtime's context current
    }
    *out = addr[dev];
    return RIS_OK;
}

}  // namespace

void noalloc_forget_addresses()
{
    std::lock_guard<std::mutex> lk(g_addr_mu);
    for (int d = 0; d < 64; ++d) {
        g_addr[d] = nullptr;
        g_ctx_of[d] = 0;
    }
}

namespace {

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace ris

using namespace ris;

extern "C" ris_status ris_attention_masked_noalloc(ris_mask_t mask, const void *q, const void *k, const void *v,
                                                   void *out, int32_t heads, int32_t kv_heads, int32_t head_dim,
                                                   int32_t dtype, int32_t out_dtype, const ris_rope_cfg *rope,
                                                   float *lse, void *stream)
{
    if (mask == nullptr) return na_fail(RIS_ERR_INVALID, "mask is NULL");
    const void *ptrs[4] = {q, k, v, out};
    const char *names[4] = {"q", "k", "v", "out"};
    for (int t = 0; t < 4; ++t) {
        if (ptrs[t] == nullptr) return na_fail(RIS_ERR_INVALID, "%s is NULL", names[t]);
        if (!aligned16(ptrs[t])) return na_fail(RIS_ERR_INVALID, "%s is not 16-byte aligned", names[t]);
    }
    if (lse != nullptr && !aligned16(lse)) return na_fail(RIS_ERR_INVALID, "lse is not 16-byte aligned");
    if (heads < 1 || kv_heads < 1 || heads % kv_heads != 0)
        return na_fail(RIS_ERR_INVALID, "heads %d / kv_heads %d", heads, kv_heads);
    if (head_dim != 64 && head_dim != 128) return na_fail(RIS_ERR_INVALID, "head_dim %d not in {64, 128}", head_dim);
    if (heads / kv_heads > 8) return na_fail(RIS_ERR_UNSUPPORTED, "heads/kv_heads = %d > 8", heads / kv_heads);
    if ((dtype != RIS_F32 && dtype != RIS_BF16) || (out_dtype != RIS_F32 && out_dtype != RIS_BF16))
        return na_fail(RIS_ERR_INVALID, "dtype %d / out_dtype %d", dtype, out_dtype);
    ris_mask_desc md{};
    ris_status st = ris_mask_info(mask, &md);
    if (st != RIS_OK) return st;
    if (md.heads_keyed > 1 && md.heads_keyed != kv_heads)
        return na_fail(RIS_ERR_INVALID, "mask keyed for %d KV heads, call has %d", md.heads_keyed, kv_heads);
    const int64_t N = md.N;
    const bool rotate = rope != nullptr && rope->kind != RIS_ROPE_NONE;

    // scratch plan: rotated q~ (fp32), then rotated k~ (bf16 hi, bf16 lo) or (fp32)
    const size_t nq = (size_t)N * heads * head_dim, nk = (size_t)N * kv_heads * head_dim;
    const size_t q_bytes = align256(nq * sizeof(float));
    const size_t k_bytes = align256(nk * (dtype == RIS_BF16 ? 2 : 4));
    const size_t need = rotate ? q_bytes + k_bytes * (dtype == RIS_BF16 ? 2 : 1) : 0;
    if (need > kNoAllocScratchBytes)
        return na_fail(RIS_ERR_INVALID,
                       "N=%lld with %d heads / %d KV heads x %d needs %zu bytes of scratch; the allocation-free "
                       "entry point holds at most %zu bytes (use ris_attention_masked)",
                       (long long)N, heads, kv_heads, head_dim, need, kNoAllocScratchBytes);

    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const void *qu = q, *ku = k, *kl = nullptr;
    bool q_split = false;
    if (rotate) {
        double f[kMaxHeadDimHalf];
        double ms = 1.0;
        st = ris_rope_freqs(rope, N, head_dim, f, &ms);
        if (st != RIS_OK) return st;
        void *base = nullptr;
        st = scratch_address(&base);
        if (st != RIS_OK) return st;
        unsigned char *b = static_cast<unsigned char *>(base);
        RopeArgs ra{};
        for (int c = 0; c < head_dim / 2; ++c) ra.f[c] = f[c];
        ra.N = N;
        ra.D = head_dim;
        ra.mscale = (float)ms;
        ra.x_in = q;
        ra.x_out = b;
        ra.H = heads;
        cudaError_t e = launch_rope(ra, dtype, RIS_F32, s);
        if (e != cudaSuccess) return na_fail(RIS_ERR_CUDA, "rope(q): %s", cudaGetErrorString(e));
        ra.x_in = k;
        ra.x_out = b + q_bytes;
        ra.x_out_lo = dtype == RIS_BF16 ? b + q_bytes + k_bytes : nullptr;
        ra.H = kv_heads;
        e = launch_rope(ra, dtype, dtype, s);
        if (e != cudaSuccess) return na_fail(RIS_ERR_CUDA, "rope(k): %s", cudaGetErrorString(e));
        qu = b;
        ku = b + q_bytes;
        kl = ra.x_out_lo;
        q_split = (dtype == RIS_BF16);
    }
    AttnArgs a{};
    a.q = qu;
    a.k = ku;
    a.k_lo = kl;
    a.v = v;
    a.out = out;
    a.lse = lse;
    a.lse_ld = N;
    a.row_ptr = md.row_ptr;
    a.col = md.col;
    a.N = N;
    a.Hq = heads;
    a.Hkv = kv_heads;
    a.G = heads / kv_heads;
    a.heads_keyed = md.heads_keyed;
    a.n_sets = md.per_seed ? md.n_seeds : 1;
    a.scale_log2 = (float)(1.4426950408889634074 / std::sqrt((double)head_dim));
    a.row0 = 0;
    a.row1 = N;
    a.n_tasks = (int64_t)a.n_sets * N * kv_heads;
    cudaError_t e = dtype == RIS_BF16
                        ? launch_attention_bf16(a, head_dim, out_dtype, q_split, md.col_bytes, md.dense != 0, s)
                        : launch_attention_f32(a, head_dim, out_dtype, md.col_bytes, md.dense != 0, s);
    if (e != cudaSuccess) return na_fail(RIS_ERR_CUDA, "attention: %s", cudaGetErrorString(e));
    return RIS_OK;
}

extern "C" ris_status ris_noalloc_scratch_info(void **device_address, int64_t *bytes)
{
    if (device_address == nullptr || bytes == nullptr) return na_fail(RIS_ERR_INVALID, "output pointer is NULL");
    *device_address = nullptr;
    *bytes = (int64_t)kNoAllocScratchBytes;
    return scratch_address(device_address);
}
