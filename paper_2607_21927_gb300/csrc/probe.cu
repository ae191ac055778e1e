// Measurement support: the hardware ceilings the attention kernels are measured against that
// a plain copy or a library GEMM does not give, each measured by a small kernel of its own.
//
//  - L2 read bandwidth for streaming 16-byte loads over a working set that stays resident in
//    L2 (loads with .cg so that L1 is not involved);
//  - L2 read bandwidth for the access pattern of the gathering attention kernels: whole
//    256-byte rows at pseudo-random row indices (a bf16 key or value row of 128 channels);
//  - FP32 FFMA throughput (independent fused multiply-add chains in registers);
//  - the device's L2 size as the driver reports it.
//
// The paper has no counterpart: it describes what is computed, not the GPU ceilings.
// These calls allocate device memory, synchronise their stream and are not meant for a hot
// path.
#include <cuda_runtime.h>

#include <cstdint>
#include <cstdio>

#include "ris_internal.h"

namespace ris {
namespace {

constexpr int kProbeThreads = 512;

__device__ __forceinline__ uint4 ld_cg_v4(const uint4 *p)
{
    uint4 v;
    asm volatile("ld.global.cg.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// Every thread walks the working set with a grid-wide stride, `reps` times. The xor of all
// words feeds a store that depends on it, so no load can be dropped.
__global__ void __launch_bounds__(kProbeThreads) k_probe_stream(const uint4 *buf, int64_t n_vec, int reps,
                                                                uint32_t *sink)
{
    uint32_t acc = 0;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int r = 0; r < reps; ++r) {
        int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
        for (; i + 3 * stride < n_vec; i += 4 * stride) {
            const uint4 a = ld_cg_v4(buf + i), b = ld_cg_v4(buf + i + stride);
            const uint4 c = ld_cg_v4(buf + i + 2 * stride), d = ld_cg_v4(buf + i + 3 * stride);
            acc ^= a.x ^ a.y ^ a.z ^ a.w ^ b.x ^ b.y ^ b.z ^ b.w ^ c.x ^ c.y ^ c.z ^ c.w ^ d.x ^ d.y ^ d.z ^ d.w;
        }
        for (; i < n_vec; i += stride) {
            const uint4 a = ld_cg_v4(buf + i);
            acc ^= a.x ^ a.y ^ a.z ^ a.w;
        }
    }
    if (acc == 0x9E3779B9u) sink[0] = acc;
}

// Row gather: each group of 16 lanes reads one 256-byte row per step at a row index drawn
// from a 32-bit mixing function of (thread, step); four rows in flight per group.
__device__ __forceinline__ uint32_t mix32(uint32_t x)
{
    x ^= x >> 16;
    x *= 0x7FEB352Du;
    x ^= x >> 15;
    x *= 0x846CA68Bu;
    x ^= x >> 16;
    return x;
}

__global__ void __launch_bounds__(kProbeThreads) k_probe_rows(const uint4 *buf, uint32_t n_rows, int steps,
                                                              uint32_t *sink)
{
    const uint32_t group = (blockIdx.x * blockDim.x + threadIdx.x) >> 4;
    const uint32_t lane16 = threadIdx.x & 15;
    uint32_t acc = 0;
    for (int s = 0; s < steps; s += 4) {
        uint4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const uint32_t row = mix32(group * 0x9E3779B1u + (uint32_t)(s + u)) % n_rows;
            v[u] = ld_cg_v4(buf + (size_t)row * 16 + lane16);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) acc ^= v[u].x ^ v[u].y ^ v[u].z ^ v[u].w;
    }
    if (acc == 0x9E3779B9u) sink[0] = acc;
}

// Eight independent FFMA chains per thread; 2 FLOPs per FFMA.
__global__ void __launch_bounds__(kProbeThreads) k_probe_ffma(float *sink, int iters, float a, float b)
{
    float x[8];
#pragma unroll
    for (int c = 0; c < 8; ++c) x[c] = (float)(threadIdx.x + c) * 1e-3f;
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int u = 0; u < 16; ++u) {
#pragma unroll
            for (int c = 0; c < 8; ++c) x[c] = fmaf(x[c], a, b);
        }
    }
    float s = 0.f;
#pragma unroll
    for (int c = 0; c < 8; ++c) s += x[c];
    if (s == 1234.5f) sink[0] = s;
}

struct DevBuf {
    void *p = nullptr;
    ~DevBuf()
    {
        if (p) cudaFree(p);
    }
};

struct EventPair {
    cudaEvent_t a = nullptr, b = nullptr;
    ~EventPair()
    {
        if (a) cudaEventDestroy(a);
        if (b) cudaEventDestroy(b);
    }
};

int sm_count()
{
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    return n;
}

// Best of `trials` launches of `launch` (each preceded by one untimed launch), in ms.
template <class F>
cudaError_t best_ms(F launch, cudaStream_t s, int trials, float *out)
{
    EventPair ev;
    cudaError_t e = cudaEventCreate(&ev.a);
    if (e == cudaSuccess) e = cudaEventCreate(&ev.b);
    if (e != cudaSuccess) return e;
    launch();
    float best = 1e30f;
    for (int t = 0; t < trials; ++t) {
        cudaEventRecord(ev.a, s);
        launch();
        cudaEventRecord(ev.b, s);
        e = cudaEventSynchronize(ev.b);
        if (e != cudaSuccess) return e;
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        float ms = 0.f;
        cudaEventElapsedTime(&ms, ev.a, ev.b);
        if (ms < best) best = ms;
    }
    *out = best;
    return cudaSuccess;
}

ris_status probe_fail(cudaError_t e, const char *what)
{
    char buf[256];
    snprintf(buf, sizeof(buf), "%s: %s", what, cudaGetErrorString(e));
    set_error_text(buf);
    cudaGetLastError();
    return RIS_ERR_CUDA;
}

}  // namespace
}  // namespace ris

using namespace ris;

extern "C" ris_status ris_probe_l2_bytes(int64_t *bytes)
{
    if (bytes == nullptr) {
        set_error_text("bytes is NULL");
        return RIS_ERR_INVALID;
    }
    int dev = 0, v = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&v, cudaDevAttrL2CacheSize, dev);
    if (e != cudaSuccess) return probe_fail(e, "L2 size");
    *bytes = v;
    return RIS_OK;
}

extern "C" ris_status ris_probe_l2_read(int64_t working_set, int32_t pattern, double *gbs, void *stream)
{
    if (gbs == nullptr || working_set < (1 << 20) || working_set > ((int64_t)1 << 32) || (pattern != 0 && pattern != 1)) {
        set_error_text("ris_probe_l2_read: gbs NULL, working_set outside [1 MiB, 4 GiB] or pattern not 0/1");
        return RIS_ERR_INVALID;
    }
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const int sms = sm_count();
    if (sms <= 0) return probe_fail(cudaErrorUnknown, "SM count");
    const int64_t bytes = working_set & ~(int64_t)255;
    DevBuf buf, sink;
    cudaError_t e = cudaMalloc(&buf.p, (size_t)bytes);
    if (e == cudaSuccess) e = cudaMalloc(&sink.p, 64);
    if (e == cudaSuccess) e = cudaMemsetAsync(buf.p, 0x5A, (size_t)bytes, s);
    if (e != cudaSuccess) return probe_fail(e, "probe buffers");
    float ms = 0.f;
    double moved = 0.0;
    const int grid = sms * (2048 / kProbeThreads);
    if (pattern == 0) {
        const int64_t n_vec = bytes / 16;
        const int reps = (int)((((int64_t)16) << 30) / bytes) + 1;  // about 16 GiB read per launch
        e = best_ms([&] { k_probe_stream<<<grid, kProbeThreads, 0, s>>>((const uint4 *)buf.p, n_vec, reps,
                                                                           (uint32_t *)sink.p); },
                    s, 5, &ms);
        moved = (double)n_vec * 16.0 * reps;
    } else {
        const uint32_t n_rows = (uint32_t)(bytes / 256);
        const int steps = 256;
        e = best_ms([&] { k_probe_rows<<<grid * 4, kProbeThreads, 0, s>>>((const uint4 *)buf.p, n_rows, steps,
                                                                            (uint32_t *)sink.p); },
                    s, 5, &ms);
        moved = (double)grid * 4 * kProbeThreads / 16 * steps * 256.0;
    }
    if (e != cudaSuccess) return probe_fail(e, "probe launch");
    *gbs = moved / (ms * 1e-3) / 1e9;
    return RIS_OK;
}

extern "C" ris_status ris_probe_ffma(double *tflops, void *stream)
{
    if (tflops == nullptr) {
        set_error_text("tflops is NULL");
        return RIS_ERR_INVALID;
    }
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const int sms = sm_count();
    if (sms <= 0) return probe_fail(cudaErrorUnknown, "SM count");
    DevBuf sink;
    cudaError_t e = cudaMalloc(&sink.p, 64);
    if (e != cudaSuccess) return probe_fail(e, "probe buffer");
    const int grid = sms * 4, iters = 4096;
    float ms = 0.f;
    e = best_ms([&] { k_probe_ffma<<<grid, kProbeThreads, 0, s>>>((float *)sink.p, iters, 0.999f, 1e-4f); }, s, 5,
                &ms);
    if (e != cudaSuccess) return probe_fail(e, "probe launch");
    const double flops = 2.0 * grid * kProbeThreads * (double)iters * 16 * 8;
    *tflops = flops / (ms * 1e-3) / 1e12;
    return RIS_OK;
}

extern "C" ris_status ris_memory_stats(int64_t *in_use, int64_t *high_water, int32_t reset_high_water)
{
    if (in_use == nullptr || high_water == nullptr) {
        set_error_text("in_use or high_water is NULL");
        return RIS_ERR_INVALID;
    }
    int dev = 0;
    cudaMemPool_t pool;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetDefaultMemPool(&pool, dev);
    uint64_t cur = 0, high = 0;
    if (e == cudaSuccess) e = cudaMemPoolGetAttribute(pool, cudaMemPoolAttrUsedMemCurrent, &cur);
    if (e == cudaSuccess) e = cudaMemPoolGetAttribute(pool, cudaMemPoolAttrUsedMemHigh, &high);
    if (e == cudaSuccess && reset_high_water) {
        uint64_t zero = 0;
        e = cudaMemPoolSetAttribute(pool, cudaMemPoolAttrUsedMemHigh, &zero);
    }
    if (e != cudaSuccess) return probe_fail(e, "memory pool attributes");
    *in_use = (int64_t)cur;
    *high_water = (int64_t)high;
    return RIS_OK;
}
