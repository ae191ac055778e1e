// RIS sparse attention, fp32 inputs (paper, Methods, "Pre-Fusion Unified Softmax"): fp32
// FFMA throughout, no TF32, for the fp32 configuration whose bar is 1e-5 relative L2.
//
// One warp owns one task (row i, KV head g, output set s). Keys are taken 32 at a time, one
// per lane: the lane streams its key's K~ row and forms the scores of the group's query
// heads (held in shared memory, read as broadcasts); the warp then updates the running
// max / sum and, key by key, every lane adds p * v to its own slice of the head dimension
// (coalesced V row loads).
#include <cuda_bf16.h>

#include <cstdint>

#include "attn_common.cuh"

namespace ris {
namespace {

template <typename TOut>
__device__ __forceinline__ void st_out(TOut *p, float x);
template <>
__device__ __forceinline__ void st_out<float>(float *p, float x) { *p = x; }
template <>
__device__ __forceinline__ void st_out<__nv_bfloat16>(__nv_bfloat16 *p, float x) { *p = __float2bfloat16_rn(x); }

// NG: compile-time bound on the query heads per KV head (1 or 8).
template <int D, int NG, typename TIdx, bool DENSE, typename TOut>
__global__ void __launch_bounds__(kAttnWarps * 32) k_attn_f32(const AttnArgs a)
{
    constexpr int DL = D / 32;  // head-dim elements per lane in the value sum
    __shared__ __align__(16) float qs[kAttnWarps][NG][D];

    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t tid = (int64_t)blockIdx.x * kAttnWarps + warp;
    if (tid >= a.n_tasks) return;
    const Task t = decode_task(a, tid);
    int64_t beg, n;
    key_range<DENSE>(a, t, beg, n);
    const TIdx *cols = DENSE ? nullptr : reinterpret_cast<const TIdx *>(a.col) + beg;

    const float *qg = reinterpret_cast<const float *>(a.q) + (t.i * a.Hq + (int64_t)t.g * a.G) * D;
    for (int e = lane; e < NG * D; e += 32) {
        const int h = e / D;
        qs[warp][h][e % D] = h < a.G ? qg[e] : 0.f;
    }
    __syncwarp();

    const float *kbase = reinterpret_cast<const float *>(a.k) + (int64_t)t.g * D;
    const float *vbase = reinterpret_cast<const float *>(a.v) + (int64_t)t.g * D + lane * DL;
    const int64_t rs = (int64_t)a.Hkv * D;
    float o[NG][DL];
    float m[NG], l[NG];
#pragma unroll
    for (int h = 0; h < NG; ++h) {
        m[h] = -INFINITY;
        l[h] = 0.f;
#pragma unroll
        for (int e = 0; e < DL; ++e) o[h][e] = 0.f;
    }

    for (int64_t base = 0; base < n; base += 32) {
        const bool valid = base + lane < n;
        const int idx = valid ? key_at<DENSE, TIdx>(cols, base + lane) : (int)t.i;
        float s[NG];
#pragma unroll
        for (int h = 0; h < NG; ++h) s[h] = 0.f;
        const float4 *kr = reinterpret_cast<const float4 *>(kbase + (int64_t)idx * rs);
#pragma unroll 4
        for (int d4 = 0; d4 < D / 4; ++d4) {
            const float4 kk = __ldg(kr + d4);
#pragma unroll
            for (int h = 0; h < NG; ++h) {
                const float4 qq = *reinterpret_cast<const float4 *>(&qs[warp][h][4 * d4]);
                s[h] = fmaf(qq.x, kk.x, s[h]);
                s[h] = fmaf(qq.y, kk.y, s[h]);
                s[h] = fmaf(qq.z, kk.z, s[h]);
                s[h] = fmaf(qq.w, kk.w, s[h]);
            }
        }
        float pr[NG];
#pragma unroll
        for (int h = 0; h < NG; ++h) {
            const float z = valid ? s[h] * a.scale_log2 : -INFINITY;
            const float mn = fmaxf(m[h], warp_max(z));
            const float mu = (mn == -INFINITY) ? 0.f : mn;
            const float al = exp2f(m[h] - mu);
            m[h] = mn;
            pr[h] = exp2f(z - mu);
            l[h] = l[h] * al + pr[h];
#pragma unroll
            for (int e = 0; e < DL; ++e) o[h][e] *= al;
        }
        const int cnt = (int)((n - base) < 32 ? (n - base) : 32);
        for (int kk = 0; kk < cnt; ++kk) {
            const int j = __shfl_sync(0xFFFFFFFFu, idx, kk);
            const float *vr = vbase + (int64_t)j * rs;
            float vv[DL];
            if (DL == 4) {
                const float4 x = __ldg(reinterpret_cast<const float4 *>(vr));
                vv[0] = x.x;
                vv[1] = x.y;
                vv[2] = x.z;
                vv[3] = x.w;
            } else {
#pragma unroll
                for (int e = 0; e < DL; ++e) vv[e] = __ldg(vr + e);
            }
#pragma unroll
            for (int h = 0; h < NG; ++h) {
                const float ph = __shfl_sync(0xFFFFFFFFu, pr[h], kk);
#pragma unroll
                for (int e = 0; e < DL; ++e) o[h][e] = fmaf(ph, vv[e], o[h][e]);
            }
        }
    }

    TOut *out = reinterpret_cast<TOut *>(a.out) +
                (((int64_t)t.s * a.N + t.i) * a.Hq + (int64_t)t.g * a.G) * D + lane * DL;
#pragma unroll
    for (int h = 0; h < NG; ++h) {
        if (h >= a.G) break;
        const float lt = warp_sum(l[h]);
        const float inv = 1.f / lt;
#pragma unroll
        for (int e = 0; e < DL; ++e) st_out<TOut>(out + (int64_t)h * D + e, o[h][e] * inv);
        if (a.lse != nullptr && lane == 0)
            a.lse[((int64_t)t.s * a.Hq + (int64_t)t.g * a.G + h) * a.lse_ld + t.i] = (m[h] + log2f(lt)) * kLn2;
    }
}

template <int D, int NG, typename TOut>
cudaError_t launch_d(const AttnArgs &a, int col_bytes, bool dense, cudaStream_t s)
{
    const unsigned grid = (unsigned)((a.n_tasks + kAttnWarps - 1) / kAttnWarps);
    const dim3 block(kAttnWarps * 32);
    if (dense)
        k_attn_f32<D, NG, uint32_t, true, TOut><<<grid, block, 0, s>>>(a);
    else if (col_bytes == 2)
        k_attn_f32<D, NG, uint16_t, false, TOut><<<grid, block, 0, s>>>(a);
    else
        k_attn_f32<D, NG, uint32_t, false, TOut><<<grid, block, 0, s>>>(a);
    note_launch();
    return cudaGetLastError();
}

template <typename TOut>
cudaError_t launch_o(const AttnArgs &a, int D, int col_bytes, bool dense, cudaStream_t s)
{
    if (a.G == 1)
        return D == 64 ? launch_d<64, 1, TOut>(a, col_bytes, dense, s)
                       : launch_d<128, 1, TOut>(a, col_bytes, dense, s);
    return D == 64 ? launch_d<64, 8, TOut>(a, col_bytes, dense, s)
                   : launch_d<128, 8, TOut>(a, col_bytes, dense, s);
}

}  // namespace

cudaError_t launch_attention_f32(const AttnArgs &a, int D, int out_dtype, int col_bytes, bool dense,
                                 cudaStream_t s)
{
    return out_dtype == RIS_F32 ? launch_o<float>(a, D, col_bytes, dense, s)
                                : launch_o<__nv_bfloat16>(a, D, col_bytes, dense, s);
}

}  // namespace ris
