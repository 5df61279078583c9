// fav_simt.cu -- generic CUDA-core attention kernel: any I/O dtype, any D <= 256.
//
// One warp per query row, following the streaming softmax of the paper's Algorithm
// "ggml-vec FlashAttention in llama.cpp" (running maximum, rescale of the accumulator by
// exp(M_old - M), running sum), but over chunks of 32 keys so that the warp's 32 lanes
// compute 32 scores at once:
//   lane j of the chunk computes s_j = scale * q . k_j (fp32 FMA chain over D);
//   the chunk maximum updates the running maximum m, the accumulator and the sum are
//   rescaled by exp(m_old - m_new), and O[d] += sum_j exp(s_j - m_new) * V[j][d] with the
//   lanes splitting d.
// For fp32 I/O every operation is an fp32 operation (no TF32, no approximate exp), which is
// this library's exact fp32 path.  For fp16/bf16 the same code upcasts to fp32 and keeps the
// weights in fp32.  Masked keys (causal, bottom-right aligned) get weight exactly 0.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <math.h>

#include "fav_internal.h"

namespace {

__device__ __forceinline__ float ld(const float *p) { return *p; }
__device__ __forceinline__ float ld(const __half *p) { return __half2float(*p); }
__device__ __forceinline__ float ld(const __nv_bfloat16 *p) { return __bfloat162float(*p); }
__device__ __forceinline__ void st(float *p, float x) { *p = x; }
__device__ __forceinline__ void st(__half *p, float x) { *p = __float2half_rn(x); }
__device__ __forceinline__ void st(__nv_bfloat16 *p, float x) { *p = __float2bfloat16_rn(x); }

constexpr int kWarps = 4;
constexpr int kMaxD = 256;

template <typename T>
__global__ void __launch_bounds__(kWarps * 32)
fav_simt_kernel(const T *__restrict__ q, const T *__restrict__ k, const T *__restrict__ v,
                T *__restrict__ o, FavStrides sq, FavStrides sk, FavStrides sv, FavStrides so,
                float *__restrict__ lse, int Hq, int Hkv, int Nq, int Nkv, int D, float scale,
                int causal, long long rows) {
    __shared__ float qs[kWarps][kMaxD];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long row = (long long)blockIdx.x * kWarps + warp;
    if (row >= rows) return;
    const int i = (int)(row % Nq);
    const long long bh = row / Nq;
    const int h = (int)(bh % Hq);
    const long long b = bh / Hq;
    const int g = h / (Hq / Hkv);
    const T *qr = q + b * sq.b + h * sq.h + (long long)i * sq.n;
    const T *Kh = k + b * sk.b + g * sk.h;
    const T *Vh = v + b * sv.b + g * sv.h;
    const int n = causal ? (Nkv - Nq + i + 1) : Nkv;

    for (int d = lane; d < D; d += 32) qs[warp][d] = ld(qr + d);
    __syncwarp();

    float acc[kMaxD / 32];
#pragma unroll
    for (int c = 0; c < kMaxD / 32; ++c) acc[c] = 0.f;
    float m = -INFINITY, l = 0.f;

    for (int j0 = 0; j0 < n; j0 += 32) {
        const int j = j0 + lane;
        float s = -INFINITY;
        if (j < n) {
            const T *kr = Kh + (long long)j * sk.n;
            float dot = 0.f;
            for (int d = 0; d < D; ++d) dot = fmaf(qs[warp][d], ld(kr + d), dot);
            s = dot * scale;
        }
        float cmax = s;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) cmax = fmaxf(cmax, __shfl_xor_sync(~0u, cmax, off));
        const float m_new = fmaxf(m, cmax);        // finite: key j0 is always visible
        const float alpha = expf(m - m_new);        // exp(-inf) = 0 on the first chunk
        const float p = (j < n) ? expf(s - m_new) : 0.f;
        float psum = p;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) psum += __shfl_xor_sync(~0u, psum, off);
        l = l * alpha + psum;
        m = m_new;
#pragma unroll
        for (int c = 0; c < kMaxD / 32; ++c) acc[c] *= alpha;
        const int cnt = min(32, n - j0);
        for (int jj = 0; jj < cnt; ++jj) {
            const float pj = __shfl_sync(~0u, p, jj);
            const T *vr = Vh + (long long)(j0 + jj) * sv.n;
#pragma unroll
            for (int c = 0; c < kMaxD / 32; ++c) {
                const int d = lane + 32 * c;
                if (d < D) acc[c] = fmaf(pj, ld(vr + d), acc[c]);
            }
        }
    }
    const float inv = 1.f / l;
    T *orow = o + b * so.b + h * so.h + (long long)i * so.n;
#pragma unroll
    for (int c = 0; c < kMaxD / 32; ++c) {
        const int d = lane + 32 * c;
        if (d < D) st(orow + d, acc[c] * inv);
    }
    if (lse && lane == 0) lse[row] = m + logf(l);
}

}  // namespace

bool fav_simt_supported(const FavArgs &a) {
    if (a.D > kMaxD) return false;
    return (a.dtype == FAV_F32) ? (a.D % 4 == 0) : (a.D % 8 == 0);
}

fav_status fav_launch_simt(const FavArgs &a, cudaStream_t s) {
    const long long rows = (long long)a.B * a.Hq * a.Nq;
    const long long blocks = (rows + kWarps - 1) / kWarps;
    if (blocks > 0x7fffffffLL) return FAV_ERR_UNSUPPORTED;
    dim3 grid((unsigned)blocks), block(kWarps * 32);
    switch (a.dtype) {
    case FAV_F32:
        fav_simt_kernel<float><<<grid, block, 0, s>>>(
            (const float *)a.q, (const float *)a.k, (const float *)a.v, (float *)a.o, a.qs, a.ks,
            a.vs, a.os, a.lse, a.Hq, a.Hkv, a.Nq, a.Nkv, a.D, a.scale, a.causal, rows);
        break;
    case FAV_F16:
        fav_simt_kernel<__half><<<grid, block, 0, s>>>(
            (const __half *)a.q, (const __half *)a.k, (const __half *)a.v, (__half *)a.o, a.qs,
            a.ks, a.vs, a.os, a.lse, a.Hq, a.Hkv, a.Nq, a.Nkv, a.D, a.scale, a.causal, rows);
        break;
    case FAV_BF16:
        fav_simt_kernel<__nv_bfloat16><<<grid, block, 0, s>>>(
            (const __nv_bfloat16 *)a.q, (const __nv_bfloat16 *)a.k, (const __nv_bfloat16 *)a.v,
            (__nv_bfloat16 *)a.o, a.qs, a.ks, a.vs, a.os, a.lse, a.Hq, a.Hkv, a.Nq, a.Nkv, a.D,
            a.scale, a.causal, rows);
        break;
    }
    if (cudaGetLastError() != cudaSuccess || fav_debug_sync("fav_simt_kernel", s)) return FAV_ERR_CUDA;
    return FAV_OK;
}
