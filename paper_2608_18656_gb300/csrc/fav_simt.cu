// fav_simt.cu -- generic CUDA-core attention kernel: any I/O dtype, any D <= 256.
//
// The streaming softmax of the paper's Algorithm "ggml-vec FlashAttention in llama.cpp"
// (running maximum, rescale of the accumulator by exp(M_old - M), running sum), over chunks of
// 32 keys:
//   a block serves kRows consecutive query rows of one (batch, head), one warp per row; the
//   block stages each chunk's 32 K rows and 32 V rows in shared memory once (coalesced 16-byte
//   loads), for all of its rows (the paper's sharing of a loaded K/V block by every query that
//   reads it);
//   lane j of a warp computes s_j = scale * q . k_j (fp32 FMAs in four interleaved partial
//   sums over D; K rows padded by one word so that the 32 lanes read 32 banks);
//   the chunk maximum updates the running maximum m, the accumulator and the sum are rescaled
//   by exp(m_old - m_new), and O[d] += sum_j exp(s_j - m_new) * V[j][d] with the lanes
//   splitting d.
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

constexpr int kRows = 4;             // query rows (warps) per block
constexpr int kChunk = 32;           // keys per chunk (one per lane)
constexpr int kMaxD = 256;

// 16-byte pieces of a row of D elements of T (D * sizeof(T) is a multiple of 16).
template <typename T> struct Vec;
template <> struct Vec<float> {
    static constexpr int kPer = 4;
    static __device__ __forceinline__ void load(const float *p, float *out) {
        const float4 x = *reinterpret_cast<const float4 *>(p);
        out[0] = x.x; out[1] = x.y; out[2] = x.z; out[3] = x.w;
    }
};
template <typename T> struct Vec16 {          // __half and __nv_bfloat16: 8 per 16 bytes
    static constexpr int kPer = 8;
    static __device__ __forceinline__ void load(const T *p, float *out) {
        const uint4 x = *reinterpret_cast<const uint4 *>(p);
        const T *e = reinterpret_cast<const T *>(&x);
#pragma unroll
        for (int i = 0; i < 8; ++i) out[i] = ld(e + i);
    }
};
template <> struct Vec<__half> : Vec16<__half> {};
template <> struct Vec<__nv_bfloat16> : Vec16<__nv_bfloat16> {};

template <typename T>
__global__ void __launch_bounds__(kRows * 32)
fav_simt_kernel(const T *__restrict__ q, const T *__restrict__ k, const T *__restrict__ v,
                T *__restrict__ o, FavStrides sq, FavStrides sk, FavStrides sv, FavStrides so,
                float *__restrict__ lse, int Hq, int Hkv, int Nq, int Nkv, int D, float scale,
                int causal, int tiles) {
    extern __shared__ float sm[];
    const int ldk = D + 1;                                   // padded K row (bank spread)
    float *Ks = sm;                                          // [kChunk][D + 1]
    float *Vs = Ks + kChunk * ldk;                           // [kChunk][D]
    float *Qs = Vs + kChunk * D;                             // [kRows][D]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long bh = blockIdx.x / tiles;                 // b * Hq + h
    const int h = (int)(bh % Hq);
    const long long b = bh / Hq;
    const int g = h / (Hq / Hkv);
    const int i0 = (int)(blockIdx.x % tiles) * kRows;
    const int i = i0 + warp;                                 // this warp's query row
    const bool has_row = i < Nq;
    const T *Kh = k + b * sk.b + g * sk.h;
    const T *Vh = v + b * sv.b + g * sv.h;
    // keys visible to this warp's row, and to the block's last row (the longest)
    const int n = !has_row ? 0 : (causal ? (Nkv - Nq + i + 1) : Nkv);
    const int i_last = min(Nq - 1, i0 + kRows - 1);
    const int n_blk = causal ? (Nkv - Nq + i_last + 1) : Nkv;

    constexpr int P = Vec<T>::kPer;
    const int pieces = D / P;                                // 16-byte pieces per row
    if (has_row) {
        const T *qr = q + b * sq.b + h * sq.h + (long long)i * sq.n;
        for (int c = lane; c < pieces; c += 32) {
            float x[P];
            Vec<T>::load(qr + c * P, x);
#pragma unroll
            for (int e = 0; e < P; ++e) Qs[warp * D + c * P + e] = x[e];
        }
    }
    const float *qw = Qs + warp * D;

    float acc[kMaxD / 32];
#pragma unroll
    for (int c = 0; c < kMaxD / 32; ++c) acc[c] = 0.f;
    float m = -INFINITY, l = 0.f;

    for (int j0 = 0; j0 < n_blk; j0 += kChunk) {
        const int cnt = min(kChunk, Nkv - j0);
        __syncthreads();                                     // the previous chunk is consumed
        for (int e = threadIdx.x; e < cnt * pieces; e += kRows * 32) {
            const int r = e / pieces, c = e - r * pieces;
            float xk[P], xv[P];
            Vec<T>::load(Kh + (long long)(j0 + r) * sk.n + c * P, xk);
            Vec<T>::load(Vh + (long long)(j0 + r) * sv.n + c * P, xv);
#pragma unroll
            for (int t = 0; t < P; ++t) {
                Ks[r * ldk + c * P + t] = xk[t];
                Vs[r * D + c * P + t] = xv[t];
            }
        }
        __syncthreads();
        if (j0 >= n) continue;                               // past this row's visible keys
        const int j = j0 + lane;
        float s = -INFINITY;
        if (j < n) {
            const float *kr = Ks + lane * ldk;
            float d0 = 0.f, d1 = 0.f, d2 = 0.f, d3 = 0.f;
            for (int d = 0; d < D; d += 4) {               // D % 4 == 0 (fav_simt_supported)
                d0 = fmaf(qw[d], kr[d], d0);
                d1 = fmaf(qw[d + 1], kr[d + 1], d1);
                d2 = fmaf(qw[d + 2], kr[d + 2], d2);
                d3 = fmaf(qw[d + 3], kr[d + 3], d3);
            }
            s = ((d0 + d1) + (d2 + d3)) * scale;
        }
        float cmax = s;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) cmax = fmaxf(cmax, __shfl_xor_sync(~0u, cmax, off));
        const float m_new = fmaxf(m, cmax);        // finite: key j0 is visible to this row
        const float alpha = expf(m - m_new);        // exp(-inf) = 0 on the first chunk
        const float p = (j < n) ? expf(s - m_new) : 0.f;
        float psum = p;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) psum += __shfl_xor_sync(~0u, psum, off);
        l = l * alpha + psum;
        m = m_new;
#pragma unroll
        for (int c = 0; c < kMaxD / 32; ++c) acc[c] *= alpha;
        const int cv = min(kChunk, n - j0);
        for (int jj = 0; jj < cv; ++jj) {
            const float pj = __shfl_sync(~0u, p, jj);
            const float *vr = Vs + jj * D;
#pragma unroll
            for (int c = 0; c < kMaxD / 32; ++c) {
                const int d = lane + 32 * c;
                if (d < D) acc[c] = fmaf(pj, vr[d], acc[c]);
            }
        }
    }
    if (!has_row) return;
    const float inv = 1.f / l;
    T *orow = o + b * so.b + h * so.h + (long long)i * so.n;
#pragma unroll
    for (int c = 0; c < kMaxD / 32; ++c) {
        const int d = lane + 32 * c;
        if (d < D) st(orow + d, acc[c] * inv);
    }
    if (lse && lane == 0) lse[bh * Nq + i] = m + logf(l);
}

}  // namespace

bool fav_simt_supported(const FavArgs &a) {
    if (a.D > kMaxD) return false;
    return (a.dtype == FAV_F32) ? (a.D % 4 == 0) : (a.D % 8 == 0);
}

fav_status fav_launch_simt(const FavArgs &a, cudaStream_t s) {
    const long long bh = (long long)a.B * a.Hq;
    const long long tiles = (a.Nq + kRows - 1) / kRows;       // row blocks per (batch, head)
    if (tiles * bh > 0x7fffffffLL) return FAV_ERR_UNSUPPORTED;
    dim3 grid((unsigned)(tiles * bh)), block(kRows * 32);
    const size_t smem = sizeof(float) * ((size_t)kChunk * (a.D + 1) + (size_t)kChunk * a.D +
                                         (size_t)kRows * a.D);
    auto go = [&](auto kern, auto *qq, auto *kk, auto *vv, auto *oo) {
        if (smem > 48 * 1024 &&
            cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
            return false;
        kern<<<grid, block, smem, s>>>(qq, kk, vv, oo, a.qs, a.ks, a.vs, a.os, a.lse, a.Hq,
                                       a.Hkv, a.Nq, a.Nkv, a.D, a.scale, a.causal, (int)tiles);
        return true;
    };
    bool ok = true;
    switch (a.dtype) {
    case FAV_F32:
        ok = go(fav_simt_kernel<float>, (const float *)a.q, (const float *)a.k, (const float *)a.v,
                (float *)a.o);
        break;
    case FAV_F16:
        ok = go(fav_simt_kernel<__half>, (const __half *)a.q, (const __half *)a.k,
                (const __half *)a.v, (__half *)a.o);
        break;
    case FAV_BF16:
        ok = go(fav_simt_kernel<__nv_bfloat16>, (const __nv_bfloat16 *)a.q,
                (const __nv_bfloat16 *)a.k, (const __nv_bfloat16 *)a.v, (__nv_bfloat16 *)a.o);
        break;
    }
    if (!ok || cudaGetLastError() != cudaSuccess || fav_debug_sync("fav_simt_kernel", s))
        return FAV_ERR_CUDA;
    return FAV_OK;
}
