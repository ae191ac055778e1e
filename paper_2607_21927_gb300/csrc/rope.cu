// RoPE with position extension (paper, Methods, "Dynamic RoPE Scaling"; linear and YaRN
// per Results, "RoPE Scaling: Linear versus YaRN"; YaRN per Peng et al. 2023).
//
// One thread per (token p, frequency c) rotates the pair (c, c + D/2) of every head of the
// token: the angle p * f_c is formed in fp64 and reduced to [-pi, pi] in fp64 (an fp32
// product loses ~4e-3 rad at p = 65535), then sin/cos of the reduced angle come from the
// CUDA math library in fp32 and the rotation runs in fp32. The work is HBM-bound: one read
// and one write of the tensor. For the fp16 + e4m3 score operands (head dim 128, bf16 inputs)
// two launches serve a whole layer call: k_fp8_bounds bounds q, k (and v) in one pass, then
// k_fp8_rotate rotates q and k (one thread per token and 8 frequencies, 16-byte accesses) into
// those operands and writes the fp16 values.
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

constexpr int kRopeTokens = 4;   // tokens per CTA (blockDim.y) of k_rope
constexpr int kPrepTokens = 32;  // tokens per CTA (blockDim.y) of k_fp8_rotate

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

// largest squared pair norm over the 8 pairs (c + e, c + e + D/2), e < 8, of a bf16 row
__device__ __forceinline__ float pair_norm2_max8(const __nv_bfloat16 *row, int c, int half)
{
    const uint4 a = *reinterpret_cast<const uint4 *>(row + c);
    const uint4 b = *reinterpret_cast<const uint4 *>(row + c + half);
    const uint32_t wa[4] = {a.x, a.y, a.z, a.w}, wb[4] = {b.x, b.y, b.z, b.w};
    float m = 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float a0 = __uint_as_float(wa[k] << 16), a1 = __uint_as_float(wa[k] & 0xFFFF0000u);
        const float b0 = __uint_as_float(wb[k] << 16), b1 = __uint_as_float(wb[k] & 0xFFFF0000u);
        m = fmaxf(m, fmaxf(fmaf(a0, a0, b0 * b0), fmaf(a1, a1, b1 * b1)));
    }
    return m;
}

// Pass 1 of the fp8-operand pre-passes: bounds[0] / bounds[1] = mscale times the largest pair
// norm of q / k, with a margin of 2^-20 for the rotation's fp32 rounding (a rotation keeps
// every pair's norm, so these bound every rotated value), bounds[2] = max |v| (when v16 is
// set). One grid-stride pass over the three tensors in 16-byte pieces (8 pairs of a row, or 8
// values), one atomic per warp and bound; the bounds are >= 0, so the order of their bit
// patterns is the order of the values.
__global__ void k_fp8_bounds(const Fp8PrepArgs a)
{
    const int half = a.D >> 1, per_row = half / 8;
    const int64_t nq = a.q_rows * a.Hq * per_row, nk = a.N * a.Hkv * per_row;
    const int64_t nv = a.v16 != nullptr ? a.N * a.Hkv * (a.D / 8) : 0;
    const __nv_bfloat16 *q = reinterpret_cast<const __nv_bfloat16 *>(a.q);
    const __nv_bfloat16 *k = reinterpret_cast<const __nv_bfloat16 *>(a.k);
    float mq = 0.f, mk = 0.f, mv = 0.f;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < nq + nk + nv;
         t += (int64_t)gridDim.x * blockDim.x) {
        if (t < nq) {
            const int64_t r = t / per_row;
            mq = fmaxf(mq, pair_norm2_max8(q + r * a.D, 8 * (int)(t - r * per_row), half));
        } else if (t < nq + nk) {
            const int64_t u = t - nq, r = u / per_row;
            mk = fmaxf(mk, pair_norm2_max8(k + r * a.D, 8 * (int)(u - r * per_row), half));
        } else {
            const uint4 x = reinterpret_cast<const uint4 *>(a.v)[t - nq - nk];
            const uint32_t w[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
            for (int e = 0; e < 4; ++e)
                mv = fmaxf(mv, fmaxf(fabsf(__uint_as_float(w[e] << 16)), fabsf(__uint_as_float(w[e] & 0xFFFF0000u))));
        }
    }
    mq = sqrtf(warp_max(mq)) * a.mscale * (1.f + 0x1p-20f);
    mk = sqrtf(warp_max(mk)) * a.mscale * (1.f + 0x1p-20f);
    mv = warp_max(mv);
    if ((threadIdx.x & 31) == 0) {
        unsigned int *b = reinterpret_cast<unsigned int *>(a.bounds);
        atomicMax(b, __float_as_uint(mq));
        atomicMax(b + 1, __float_as_uint(mk));
        if (a.v16 != nullptr) atomicMax(b + 2, __float_as_uint(mv));
    }
}

// eight e4m3 values, lowest address first, as one 8-byte word
__device__ __forceinline__ uint2 to_e4m3x8(const float *x)
{
    uint32_t w[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const uint32_t lo = __nv_cvt_float2_to_fp8x2(make_float2(x[4 * h], x[4 * h + 1]), __NV_SATFINITE, __NV_E4M3);
        const uint32_t hi = __nv_cvt_float2_to_fp8x2(make_float2(x[4 * h + 2], x[4 * h + 3]), __NV_SATFINITE, __NV_E4M3);
        w[h] = (lo & 0xFFFFu) | (hi << 16);
    }
    return make_uint2(w[0], w[1]);
}

// Rotate the 8 pairs (c + e, c + e + D/2), e < 8, of each of H heads of one token (bf16 in) and
// write them in the tile kernel's form: fp16 hi parts to hi and, in the 2D-byte record of
// each (token, head) in lo, e4m3(hi s_hi) at bytes [0, D) and e4m3((y - hi) s_lo) at [D, 2D);
// or (f8 false) the bf16 hi / lo pair.
__device__ __forceinline__ void rotate_heads8(const __nv_bfloat16 *x, void *hi, void *lo, int H, int D, int c,
                                              const float *cs, const float *sn, float mscale, bool f8, float s_hi,
                                              float s_lo)
{
    const int half = D >> 1;
    for (int h = 0; h < H; ++h) {
        const uint4 a = *reinterpret_cast<const uint4 *>(x + (int64_t)h * D + c);
        const uint4 b = *reinterpret_cast<const uint4 *>(x + (int64_t)h * D + c + half);
        const uint32_t wa[4] = {a.x, a.y, a.z, a.w}, wb[4] = {b.x, b.y, b.z, b.w};
        float y[2][8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const float x0 = __uint_as_float((e & 1) ? (wa[e >> 1] & 0xFFFF0000u) : (wa[e >> 1] << 16));
            const float x1 = __uint_as_float((e & 1) ? (wb[e >> 1] & 0xFFFF0000u) : (wb[e >> 1] << 16));
            y[0][e] = fmaf(x0, cs[e], -x1 * sn[e]) * mscale;
            y[1][e] = fmaf(x1, cs[e], x0 * sn[e]) * mscale;
        }
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int64_t e0 = (int64_t)h * D + c + u * half;
            uint32_t wh[4], wl[4];
            if (f8) {
                float h8[8], l8[8];
#pragma unroll
                for (int e = 0; e < 8; e += 2) {
                    const __half2 hh = __floats2half2_rn(y[u][e], y[u][e + 1]);
                    const float2 hv = __half22float2(hh);
                    wh[e >> 1] = *reinterpret_cast<const uint32_t *>(&hh);
                    h8[e] = hv.x * s_hi;
                    h8[e + 1] = hv.y * s_hi;
                    l8[e] = (y[u][e] - hv.x) * s_lo;
                    l8[e + 1] = (y[u][e + 1] - hv.y) * s_lo;
                }
                *reinterpret_cast<uint4 *>(reinterpret_cast<__half *>(hi) + e0) = make_uint4(wh[0], wh[1], wh[2], wh[3]);
                unsigned char *rec = reinterpret_cast<unsigned char *>(lo) + 2 * ((int64_t)h * D) + c + u * half;
                *reinterpret_cast<uint2 *>(rec) = to_e4m3x8(h8);
                *reinterpret_cast<uint2 *>(rec + D) = to_e4m3x8(l8);
            } else {
#pragma unroll
                for (int e = 0; e < 8; e += 2) {
                    const __nv_bfloat162 hb = __floats2bfloat162_rn(y[u][e], y[u][e + 1]);
                    const float2 hv = __bfloat1622float2(hb);
                    const __nv_bfloat162 lb = __floats2bfloat162_rn(y[u][e] - hv.x, y[u][e + 1] - hv.y);
                    wh[e >> 1] = *reinterpret_cast<const uint32_t *>(&hb);
                    wl[e >> 1] = *reinterpret_cast<const uint32_t *>(&lb);
                }
                *reinterpret_cast<uint4 *>(reinterpret_cast<__nv_bfloat16 *>(hi) + e0) = make_uint4(wh[0], wh[1], wh[2], wh[3]);
                *reinterpret_cast<uint4 *>(reinterpret_cast<__nv_bfloat16 *>(lo) + e0) = make_uint4(wl[0], wl[1], wl[2], wl[3]);
            }
        }
    }
}

// Pass 2: one thread per (token p, frequencies 8j .. 8j+7): the eight rotation angles (fp64,
// reduced as in k_rope), then the keys of the token, its query row if it has one (rows q_first
// .. q_first + q_rows - 1), and, when v16 is set, elements 16j .. 16j+15 of each of its value
// heads as fp16 scaled by 2^-E (E = v_scale_exp(max |v|)). Queries: hi parts scaled by 2^-ea, lo
// parts by 2^(12+eb); keys: 2^-eb and 2^(12+ea) (fp8_score_scales).
__global__ void k_fp8_rotate(const Fp8PrepArgs a)
{
    const int j = threadIdx.x, c = 8 * j;  // blockDim.x == D / 16
    const int64_t p = (int64_t)blockIdx.x * blockDim.y + threadIdx.y;
    if (p >= a.N) return;
    int ea = 0, eb = 0;
    const bool f8 = fp8_score_scales(a.bounds[0], a.bounds[1], ea, eb);
    float cs[8], sn[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const double ang = (double)p * a.f[c + e];
        const double n = rint(ang * 0.15915494309189533577);
        double red = fma(-n, 6.28318530717958623200, ang);
        red = fma(-n, 2.4492935982947064e-16, red);
        sincosf((float)red, &sn[e], &cs[e]);
    }
    const int64_t hk = p * (int64_t)a.Hkv * a.D;
    rotate_heads8(reinterpret_cast<const __nv_bfloat16 *>(a.k) + hk, reinterpret_cast<__half *>(a.k_hi) + hk,
                  reinterpret_cast<unsigned char *>(a.k_lo) + 2 * hk, a.Hkv, a.D, c, cs, sn, a.mscale, f8,
                  f8 ? pow2i(-eb) : 1.f, f8 ? pow2i(12 + ea) : 1.f);
    if (p >= a.q_first && p < a.q_first + a.q_rows) {
        const int64_t hq = (p - a.q_first) * (int64_t)a.Hq * a.D;
        rotate_heads8(reinterpret_cast<const __nv_bfloat16 *>(a.q) + hq, reinterpret_cast<__half *>(a.q_hi) + hq,
                      reinterpret_cast<unsigned char *>(a.q_lo) + 2 * hq, a.Hq, a.D, c, cs, sn, a.mscale, f8,
                      f8 ? pow2i(-ea) : 1.f, f8 ? pow2i(12 + eb) : 1.f);
    }
    if (a.v16 != nullptr) {
        const float scale = pow2i(-v_scale_exp(a.bounds[2]));
        for (int h = 0; h < a.Hkv; ++h) {
            const int64_t e0 = hk + (int64_t)h * a.D + 16 * j;
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const uint4 x = *reinterpret_cast<const uint4 *>(reinterpret_cast<const __nv_bfloat16 *>(a.v) + e0 + 8 * u);
                const uint32_t w[4] = {x.x, x.y, x.z, x.w};
                uint32_t o[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const __half2 hh = __floats2half2_rn(__uint_as_float(w[e] << 16) * scale,
                                                         __uint_as_float(w[e] & 0xFFFF0000u) * scale);
                    o[e] = *reinterpret_cast<const uint32_t *>(&hh);
                }
                *reinterpret_cast<uint4 *>(reinterpret_cast<__half *>(a.v16) + e0 + 8 * u) = make_uint4(o[0], o[1], o[2], o[3]);
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

cudaError_t launch_fp8_prep(const Fp8PrepArgs &a, cudaStream_t s)
{
    if ((a.D % 16) != 0 || a.D / 2 > kMaxHeadDimHalf || a.D / 16 * kPrepTokens > 1024) return cudaErrorInvalidValue;
    cudaError_t e = cudaMemsetAsync(a.bounds, 0, 3 * sizeof(float), s);
    if (e != cudaSuccess) return e;
    const int64_t pieces = (a.q_rows * a.Hq + a.N * a.Hkv) * (a.D / 16) + (a.v16 != nullptr ? a.N * a.Hkv * (a.D / 8) : 0);
    const int threads = 256;
    const int64_t need = (pieces + threads - 1) / threads;
    const unsigned grid = (unsigned)(need < 152 * 8 ? (need > 0 ? need : 1) : 152 * 8);
    k_fp8_bounds<<<grid, threads, 0, s>>>(a);
    const dim3 block(a.D / 16, kPrepTokens);
    k_fp8_rotate<<<(unsigned)((a.N + kPrepTokens - 1) / kPrepTokens), block, 0, s>>>(a);
    note_launch(2);
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
