// RoPE with position extension (paper, Methods, "Dynamic RoPE Scaling"; linear and YaRN
// per Results, "RoPE Scaling: Linear versus YaRN"; YaRN per Peng et al. 2023).
//
// One thread per (token p, frequency c) rotates the pair (c, c + D/2) of every head of the
// token: the angle p * f_c is formed in fp64 and reduced to [-pi, pi] in fp64 (an fp32
// product loses ~4e-3 rad at p = 65535), then sin/cos of the reduced angle come from the
// CUDA math library in fp32 and the rotation runs in fp32. The work is HBM-bound: one read
// and one write of the tensor.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cstdint>

#include "attn_common.cuh"
#include "ris_internal.h"

namespace ris {
namespace {

template <typename T>
__device__ __forceinline__ float ld_f(const T *p);
template <>
__device__ __forceinline__ float ld_f<float>(const float *p) { return *p; }
template <>
__device__ __forceinline__ float ld_f<__nv_bfloat16>(const __nv_bfloat16 *p) { return __bfloat162float(*p); }

template <typename T>
__device__ __forceinline__ void st_f(T *p, float x);
template <>
__device__ __forceinline__ void st_f<float>(float *p, float x) { *p = x; }
template <>
__device__ __forceinline__ void st_f<__nv_bfloat16>(__nv_bfloat16 *p, float x) { *p = __float2bfloat16_rn(x); }

constexpr int kRopeTokens = 4;  // tokens per CTA (blockDim.y)

template <typename TIn, typename TOut, bool LO>
__global__ void k_rope(const RopeArgs a)
{
    const int half = a.D >> 1;
    const int c = threadIdx.x;  // blockDim.x == D/2
    const int64_t p = (int64_t)blockIdx.x * kRopeTokens + threadIdx.y;
    if (p >= a.N || c >= half) return;
    // angle in fp64, reduced by the nearest multiple of 2 pi (two-term 2 pi)
    const double ang = (double)(p + a.pos0) * a.f[c];
    const double n = rint(ang * 0.15915494309189533577);  // 1 / (2 pi)
    double red = fma(-n, 6.28318530717958623200, ang);  // 2 pi, high part
    red = fma(-n, 2.4492935982947064e-16, red);            // 2 pi, low part
    float sn, cs;
    sincosf((float)red, &sn, &cs);
    const TIn *xi = reinterpret_cast<const TIn *>(a.x_in) + p * (int64_t)a.H * a.D;
    TOut *xo = reinterpret_cast<TOut *>(a.x_out) + p * (int64_t)a.H * a.D;
    for (int h = 0; h < a.H; ++h) {
        const float x0 = ld_f(xi + h * a.D + c);
        const float x1 = ld_f(xi + h * a.D + c + half);
        const float y0 = fmaf(x0, cs, -x1 * sn) * a.mscale;
        const float y1 = fmaf(x1, cs, x0 * sn) * a.mscale;
        st_f(xo + h * a.D + c, y0);
        st_f(xo + h * a.D + c + half, y1);
        if (LO) {
            // residual of the bf16 rounding, so that hi + lo carries ~16 significant bits
            __nv_bfloat16 *lo = reinterpret_cast<__nv_bfloat16 *>(a.x_out_lo) + p * (int64_t)a.H * a.D;
            lo[h * a.D + c] = __float2bfloat16_rn(y0 - __bfloat162float(__float2bfloat16_rn(y0)));
            lo[h * a.D + c + half] = __float2bfloat16_rn(y1 - __bfloat162float(__float2bfloat16_rn(y1)));
        }
    }
}

// max |v| over 8 bf16 values per thread and step (grid-stride), one atomic per warp; |v| >= 0,
// so the order of the float bit patterns is the order of the values
__global__ void k_absmax_bf16(const uint4 *v, int64_t n8, unsigned int *vmax)
{
    float m = 0.f;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < n8; t += (int64_t)gridDim.x * blockDim.x) {
        const uint4 x = v[t];
        const uint32_t w[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            m = fmaxf(m, fabsf(__uint_as_float(w[k] << 16)));
            m = fmaxf(m, fabsf(__uint_as_float(w[k] & 0xFFFF0000u)));
        }
    }
    m = warp_max(m);
    if ((threadIdx.x & 31) == 0) atomicMax(vmax, __float_as_uint(m));
}

__global__ void k_values_f16(const uint4 *v, int64_t n8, const float *vmax, uint4 *v16)
{
    const float scale = __uint_as_float((uint32_t)(127 - v_scale_exp(*vmax)) << 23);  // 2^-E
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < n8; t += (int64_t)gridDim.x * blockDim.x) {
        const uint4 x = v[t];
        const uint32_t w[4] = {x.x, x.y, x.z, x.w};
        uint32_t o[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const __half2 h = __floats2half2_rn(__uint_as_float(w[k] << 16) * scale,
                                                __uint_as_float(w[k] & 0xFFFF0000u) * scale);
            o[k] = *reinterpret_cast<const uint32_t *>(&h);
        }
        v16[t] = make_uint4(o[0], o[1], o[2], o[3]);
    }
}

}  // namespace

cudaError_t launch_values_f16(const void *v, int64_t n, void *v16, float *vmax, cudaStream_t s)
{
    if ((n & 7) != 0) return cudaErrorInvalidValue;
    const int64_t n8 = n / 8;
    cudaError_t e = cudaMemsetAsync(vmax, 0, sizeof(float), s);
    if (e != cudaSuccess) return e;
    const int threads = 256;
    const int64_t need = (n8 + threads - 1) / threads;
    const unsigned grid = (unsigned)(need < 152 * 8 ? (need > 0 ? need : 1) : 152 * 8);
    k_absmax_bf16<<<grid, threads, 0, s>>>(reinterpret_cast<const uint4 *>(v), n8, reinterpret_cast<unsigned int *>(vmax));
    k_values_f16<<<grid, threads, 0, s>>>(reinterpret_cast<const uint4 *>(v), n8, vmax, reinterpret_cast<uint4 *>(v16));
    note_launch(2);
    return cudaGetLastError();
}

cudaError_t launch_rope(const RopeArgs &a, int dtype_in, int dtype_out, cudaStream_t s)
{
    const dim3 block(a.D / 2, kRopeTokens);
    const dim3 grid((unsigned)((a.N + kRopeTokens - 1) / kRopeTokens));
    if (dtype_in == RIS_F32 && dtype_out == RIS_F32)
        k_rope<float, float, false><<<grid, block, 0, s>>>(a);
    else if (dtype_in == RIS_BF16 && dtype_out == RIS_BF16) {
        if (a.x_out_lo != nullptr)
            k_rope<__nv_bfloat16, __nv_bfloat16, true><<<grid, block, 0, s>>>(a);
        else
            k_rope<__nv_bfloat16, __nv_bfloat16, false><<<grid, block, 0, s>>>(a);
    } else if (dtype_in == RIS_BF16 && dtype_out == RIS_F32)
        k_rope<__nv_bfloat16, float, false><<<grid, block, 0, s>>>(a);
    else
        k_rope<float, __nv_bfloat16, false><<<grid, block, 0, s>>>(a);
    note_launch();
    return cudaGetLastError();
}

}  // namespace ris
