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
#include <cuda_fp8.h>

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

// The largest pair norm of x [rows][D] (bf16), times mscale with a margin of 2^-20 for the
// rotation's fp32 rounding: a bound of every rotated value (a rotation keeps the pair norm).
// Each thread takes 8 consecutive pairs (16-byte loads of both halves of a row).
__global__ void k_rotation_bound(const __nv_bfloat16 *x, int64_t rows, int D, float mscale, unsigned int *bound)
{
    const int half = D >> 1, per_row = half / 8;
    float m = 0.f;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < rows * per_row; t += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = t / per_row;
        const int c = 8 * (int)(t - r * per_row);
        const uint4 a = *reinterpret_cast<const uint4 *>(x + r * D + c);
        const uint4 b = *reinterpret_cast<const uint4 *>(x + r * D + c + half);
        const uint32_t wa[4] = {a.x, a.y, a.z, a.w}, wb[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float a0 = __uint_as_float(wa[k] << 16), a1 = __uint_as_float(wa[k] & 0xFFFF0000u);
            const float b0 = __uint_as_float(wb[k] << 16), b1 = __uint_as_float(wb[k] & 0xFFFF0000u);
            m = fmaxf(m, fmaxf(fmaf(a0, a0, b0 * b0), fmaf(a1, a1, b1 * b1)));
        }
    }
    m = sqrtf(warp_max(m)) * mscale * (1.f + 0x1p-20f);
    if ((threadIdx.x & 31) == 0) atomicMax(bound, __float_as_uint(m));
}

__device__ __forceinline__ unsigned char to_e4m3(float x)
{
    return (unsigned char)__nv_cvt_float_to_fp8(x, __NV_SATFINITE, __NV_E4M3);
}

// RoPE for the tile kernel's fp8-correction scores (see fp8_score_scales): the same rotation
// as k_rope, then fp16 hi parts into x_out and the two e4m3 correction operands into x_out_lo,
// or the bf16 hi / lo pair when the bounds rule the scheme out. ROLE 0: queries (hi part
// scaled by 2^-ea, lo part by 2^(12+eb)); ROLE 1: keys (hi part by 2^-eb, lo part by 2^(12+ea)).
template <int ROLE>
__global__ void k_rope_tile8(const RopeArgs a, const float *qk_bound)
{
    const int half = a.D >> 1;
    const int c = threadIdx.x;  // blockDim.x == D/2
    const int64_t p = (int64_t)blockIdx.x * kRopeTokens + threadIdx.y;
    if (p >= a.N || c >= half) return;
    int ea = 0, eb = 0;
    const bool f8 = fp8_score_scales(qk_bound[0], qk_bound[1], ea, eb);
    const float s_hi = f8 ? pow2i(ROLE == 0 ? -ea : -eb) : 1.f;
    const float s_lo = f8 ? pow2i(12 + (ROLE == 0 ? eb : ea)) : 1.f;
    const double ang = (double)(p + a.pos0) * a.f[c];
    const double n = rint(ang * 0.15915494309189533577);
    double red = fma(-n, 6.28318530717958623200, ang);
    red = fma(-n, 2.4492935982947064e-16, red);
    float sn, cs;
    sincosf((float)red, &sn, &cs);
    const __nv_bfloat16 *xi = reinterpret_cast<const __nv_bfloat16 *>(a.x_in) + p * (int64_t)a.H * a.D;
    for (int h = 0; h < a.H; ++h) {
        const float x0 = __bfloat162float(xi[h * a.D + c]);
        const float x1 = __bfloat162float(xi[h * a.D + c + half]);
        const float y[2] = {fmaf(x0, cs, -x1 * sn) * a.mscale, fmaf(x1, cs, x0 * sn) * a.mscale};
        const int64_t e0 = (p * (int64_t)a.H + h) * a.D;
        for (int u = 0; u < 2; ++u) {
            const int cc = c + u * half;
            if (f8) {
                const __half hh = __float2half_rn(y[u]);
                const float hv = __half2float(hh);
                reinterpret_cast<__half *>(a.x_out)[e0 + cc] = hh;
                unsigned char *lo = reinterpret_cast<unsigned char *>(a.x_out_lo) + 2 * e0;
                lo[cc] = to_e4m3(hv * s_hi);
                lo[a.D + cc] = to_e4m3((y[u] - hv) * s_lo);
            } else {
                const __nv_bfloat16 hb = __float2bfloat16_rn(y[u]);
                reinterpret_cast<__nv_bfloat16 *>(a.x_out)[e0 + cc] = hb;
                reinterpret_cast<__nv_bfloat16 *>(a.x_out_lo)[e0 + cc] = __float2bfloat16_rn(y[u] - __bfloat162float(hb));
            }
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

cudaError_t launch_rotation_bound(const void *x, int64_t N, int H, int D, float mscale, float *bound, cudaStream_t s)
{
    if ((D % 16) != 0) return cudaErrorInvalidValue;
    const int64_t work = N * H * (D / 16);
    const int threads = 256;
    const int64_t need = (work + threads - 1) / threads;
    const unsigned grid = (unsigned)(need < 152 * 8 ? (need > 0 ? need : 1) : 152 * 8);
    k_rotation_bound<<<grid, threads, 0, s>>>(reinterpret_cast<const __nv_bfloat16 *>(x), N * H, D, mscale,
                                              reinterpret_cast<unsigned int *>(bound));
    note_launch();
    return cudaGetLastError();
}

cudaError_t launch_rope_tile8(const RopeArgs &a, int role, const float *qk_bound, cudaStream_t s)
{
    const dim3 block(a.D / 2, kRopeTokens);
    const dim3 grid((unsigned)((a.N + kRopeTokens - 1) / kRopeTokens));
    if (role == 0)
        k_rope_tile8<0><<<grid, block, 0, s>>>(a, qk_bound);
    else
        k_rope_tile8<1><<<grid, block, 0, s>>>(a, qk_bound);
    note_launch();
    return cudaGetLastError();
}

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
