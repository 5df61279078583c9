// fav_nonflash.cu -- the non-flash self-attention of the paper's Self-attention section, as an
// in-library comparison point: the full score matrix is materialised.
//
//   S = scale * Q K^T      one batched GEMM per KV head (its G query heads stacked as the rows),
//                          fp32 scores in a workspace [B * Hq, Nq, Nkv]
//   P = softmax(S) (mask)  one block per query row, the row in registers (float4 loads; rows up
//                          to 8192 keys, a multiple of 4) or else in shared memory; the weights,
//                          stored as p * 2^11 in fp16, overwrite the first half of their own fp32
//                          row, and LSE = max + log(sum)
//   O = P V                a second batched GEMM per KV head, fp16 x fp16 with alpha = 2^-11
//
// The weights are fp16 for both I/O types, as in the fused kernels: 11 significant bits (a bf16
// weight has 8, and its rounding alone can move O by 2^-9 max|v|), scaled by 2^11 so that weights
// down to 2^-25 stay fp16 normals.  For bf16 I/O, V is first converted to fp16 under a power of
// two per KV head (fav_v16_convert, the fused path's conversion), the P V GEMM writes O * 2^-e in
// fp16 into the output buffer, and fav_nonflash_unscale_kernel turns it into bf16 O in place.
//
// The GEMMs are cuBLAS (cublasGemmStridedBatchedEx, fp32 accumulation), loaded on first use with
// dlopen so that libfav itself does not depend on cuBLAS; without it the entry point returns
// FAV_ERR_UNSUPPORTED.  The paper's point is that the fused (flash) form avoids writing and
// reading the N x N scores; this path exists to measure that difference on this GPU.
#include <cuda_runtime.h>
#include <dlfcn.h>
#include <math.h>

#include <mutex>

#include "fav_device.cuh"
#include "fav_internal.h"

namespace {

// The few cuBLAS declarations used here (cublas_v2.h's types, restated as plain integers so
// that this file builds without the header on the include path).
using cublasHandle_t = void *;
using cublasStatus_t = int;
constexpr int kCublasOpN = 0, kCublasOpT = 1;
constexpr int kCudaR32F = 0, kCudaR16F = 2, kCudaR16BF = 14;     // cudaDataType_t
constexpr int kCublasCompute32F = 68;                           // cublasComputeType_t
constexpr int kCublasGemmDefault = -1;                          // cublasGemmAlgo_t
using CreateFn = cublasStatus_t (*)(cublasHandle_t *);
using SetStreamFn = cublasStatus_t (*)(cublasHandle_t, cudaStream_t);
// cublasGemmStridedBatchedEx(handle, transa, transb, m, n, k, alpha, A, Atype, lda, strideA,
//                            B, Btype, ldb, strideB, beta, C, Ctype, ldc, strideC, batchCount,
//                            computeType, algo)
using GemmFn = cublasStatus_t (*)(cublasHandle_t, int, int, int, int, int, const void *,
                                  const void *, int, int, long long, const void *, int, int,
                                  long long, const void *, void *, int, int, long long, int, int,
                                  int);

struct Cublas {
    bool ok = false;
    cublasHandle_t handle[64] = {};
    CreateFn create = nullptr;
    SetStreamFn set_stream = nullptr;
    GemmFn gemm = nullptr;
};

Cublas &cublas() {
    static Cublas c;
    static std::once_flag once;
    std::call_once(once, [] {
        // the copy already in the process (loaded by the caller's framework), else the loader's
        void *h = dlopen("libcublas.so.13", RTLD_NOW | RTLD_GLOBAL);
        if (!h) h = dlopen("/usr/local/cuda/lib64/libcublas.so.13", RTLD_NOW | RTLD_GLOBAL);
        if (!h) return;
        c.create = reinterpret_cast<CreateFn>(dlsym(h, "cublasCreate_v2"));
        c.set_stream = reinterpret_cast<SetStreamFn>(dlsym(h, "cublasSetStream_v2"));
        c.gemm = reinterpret_cast<GemmFn>(dlsym(h, "cublasGemmStridedBatchedEx"));
        c.ok = c.create && c.set_stream && c.gemm;
    });
    return c;
}

// One block per query row: the row's Nkv scores (fp32) in shared memory, the causal mask
// (bottom-right: key j visible while j <= Nkv - Nq + i), maximum, sum of exponentials, then the
// weights p_j = exp(s_j - max) / sum rounded to T over the first half of the row's bytes
// (row stride in T elements: 2 * Nkv), and LSE = max + log(sum).
constexpr float kPScale = 2048.f;       // weights stored as p * 2^11 (fp16)
constexpr float kPUnscale = 1.f / 2048.f;

__global__ void __launch_bounds__(256)
fav_nonflash_softmax_kernel(float *__restrict__ s, float *__restrict__ lse, int Nq, int Nkv,
                            int causal) {
    extern __shared__ float row[];
    __shared__ float red[8];
    const long long r = blockIdx.x;
    const int i = (int)(r % Nq);
    const int lim = causal ? min(Nkv, Nkv - Nq + i + 1) : Nkv;      // visible keys [0, lim)
    float *src = s + r * Nkv;
    float mx = -INFINITY;
    for (int j = threadIdx.x; j < Nkv; j += blockDim.x) {
        const float x = j < lim ? src[j] : -INFINITY;
        row[j] = x;
        mx = fmaxf(mx, x);
    }
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(~0u, mx, o));
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
    __syncthreads();
    mx = red[0];
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) mx = fmaxf(mx, red[w]);
    __syncthreads();
    float sum = 0.f;
    for (int j = threadIdx.x; j < Nkv; j += blockDim.x) {
        const float e = (mx == -INFINITY) ? 0.f : expf(row[j] - mx);
        row[j] = e;
        sum += e;
    }
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(~0u, sum, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = sum;
    __syncthreads();
    sum = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) sum += red[w];
    const float inv = sum > 0.f ? kPScale / sum : 0.f;
    __half *p = reinterpret_cast<__half *>(src);          // every score of the row is in shared memory
    for (int j = threadIdx.x; j < Nkv; j += blockDim.x) p[j] = __float2half_rn(row[j] * inv);
    if (lse && threadIdx.x == 0) lse[r] = sum > 0.f ? mx + logf(sum) : -INFINITY;
}

// The same row softmax with the row in registers, for Nkv % 4 == 0 and Nkv <= 1024 * kVec:
// each of the 256 threads holds kVec float4 of the row (16-byte loads; causal rows read only
// their visible prefix), so the row is read once from HBM and the weights written once.
template <int kVec>
__global__ void __launch_bounds__(256)
fav_nonflash_softmax_reg_kernel(float *__restrict__ s, float *__restrict__ lse, int Nq,
                                int Nkv, int causal) {
    __shared__ float red[2][8];
    const long long r = blockIdx.x;
    const int i = (int)(r % Nq);
    const int lim = causal ? min(Nkv, Nkv - Nq + i + 1) : Nkv;      // visible keys [0, lim)
    float *src = s + r * Nkv;
    float4 x[kVec];
    float mx = -INFINITY;
#pragma unroll
    for (int v = 0; v < kVec; ++v) {
        const int j = 4 * (v * 256 + (int)threadIdx.x);
        float4 a = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
        if (j < lim) {
            a = *reinterpret_cast<const float4 *>(src + j);
            if (j + 1 >= lim) a.y = -INFINITY;
            if (j + 2 >= lim) a.z = -INFINITY;
            if (j + 3 >= lim) a.w = -INFINITY;
        }
        x[v] = a;
        mx = fmaxf(mx, fmaxf(fmaxf(a.x, a.y), fmaxf(a.z, a.w)));
    }
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(~0u, mx, o));
    if ((threadIdx.x & 31) == 0) red[0][threadIdx.x >> 5] = mx;
    __syncthreads();          // also: every thread has read its part of the row
    mx = red[0][0];
#pragma unroll
    for (int w = 1; w < 8; ++w) mx = fmaxf(mx, red[0][w]);
    float sum = 0.f;
#pragma unroll
    for (int v = 0; v < kVec; ++v) {
        float4 &a = x[v];
        a.x = expf(a.x - mx);     // masked entries: exp(-inf) = 0 (mx is finite: lim >= 1)
        a.y = expf(a.y - mx);
        a.z = expf(a.z - mx);
        a.w = expf(a.w - mx);
        sum += (a.x + a.y) + (a.z + a.w);
    }
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(~0u, sum, o);
    if ((threadIdx.x & 31) == 0) red[1][threadIdx.x >> 5] = sum;
    __syncthreads();
    sum = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) sum += red[1][w];
    const float inv = kPScale / sum;
    __half *p = reinterpret_cast<__half *>(src);
#pragma unroll
    for (int v = 0; v < kVec; ++v) {
        const int j = 4 * (v * 256 + (int)threadIdx.x);
        if (j < Nkv) {
            const uint2 q = make_uint2(fav::Elem<__half>::pack(x[v].x * inv, x[v].y * inv),
                                       fav::Elem<__half>::pack(x[v].z * inv, x[v].w * inv));
            *reinterpret_cast<uint2 *>(p + j) = q;
        }
    }
    if (lse && threadIdx.x == 0) lse[r] = mx + logf(sum);
}

// O (fp16, holding O * 2^-e of its KV head: the P V GEMM of the bf16 path) -> bf16 O in place.
// One thread per 8 elements (16 bytes); rows of D elements, row r = (b * Hq + h) * Nq + i.
__global__ void __launch_bounds__(256)
fav_nonflash_unscale_kernel(uint4 *__restrict__ o, const float *__restrict__ v_scale,
                            long long n8, int D, int Nq, int Hq, int G, int Hkv) {
    const long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x;
    if (i >= n8) return;
    const long long r = i * 8 / D;
    const long long bh = r / Nq;
    const int h = (int)(bh % Hq);
    const long long b = bh / Hq;
    const float sc = v_scale[b * Hkv + h / G];
    uint4 w = o[i];
    uint32_t *u = reinterpret_cast<uint32_t *>(&w);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const __half2 x = *reinterpret_cast<const __half2 *>(&u[k]);
        const float2 f = __half22float2(x);
        u[k] = fav::Elem<__nv_bfloat16>::pack(f.x * sc, f.y * sc);
    }
    o[i] = w;
}

// The softmax launch: registers when the row fits (and is 16-byte aligned), shared memory
// otherwise.
cudaError_t launch_softmax(float *S, float *lse, long long rows, int Nq, int Nk, int causal,
                           cudaStream_t stream) {
    const unsigned grid = (unsigned)rows;
    if (Nk % 4 == 0 && Nk <= 8192) {
        const int vec = (Nk + 1023) / 1024;
        if (vec <= 1)
            fav_nonflash_softmax_reg_kernel<1><<<grid, 256, 0, stream>>>(S, lse, Nq, Nk, causal);
        else if (vec <= 2)
            fav_nonflash_softmax_reg_kernel<2><<<grid, 256, 0, stream>>>(S, lse, Nq, Nk, causal);
        else if (vec <= 4)
            fav_nonflash_softmax_reg_kernel<4><<<grid, 256, 0, stream>>>(S, lse, Nq, Nk, causal);
        else
            fav_nonflash_softmax_reg_kernel<8><<<grid, 256, 0, stream>>>(S, lse, Nq, Nk, causal);
        return cudaGetLastError();
    }
    const size_t smem = (size_t)Nk * sizeof(float);
    auto kern = fav_nonflash_softmax_kernel;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)(smem > 48 * 1024 ? smem : 48 * 1024));
    if (e != cudaSuccess) return e;
    kern<<<grid, 256, smem, stream>>>(S, lse, Nq, Nk, causal);
    return cudaGetLastError();
}

}  // namespace

size_t fav_nonflash_workspace_bytes(const FavArgs &a) {
    return (size_t)a.B * a.Hq * a.Nq * a.Nkv * sizeof(float);
}

bool fav_nonflash_shape_ok(const FavArgs &a) {
    if (a.dtype != FAV_F16 && a.dtype != FAV_BF16) return false;
    const long long G = a.Hq / a.Hkv;
    return a.Nkv <= 32768 && G * a.Nq * a.Nkv < (1LL << 31) &&
           (long long)a.B * a.Hq * a.Nq <= 0x7fffffffLL;
}

bool fav_nonflash_available() { return cublas().ok; }

fav_status fav_launch_nonflash(const FavArgs &a, void *workspace, void *v_workspace,
                               cudaStream_t stream) {
    Cublas &c = cublas();
    if (!c.ok) return FAV_ERR_UNSUPPORTED;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return FAV_ERR_CUDA;
    // one handle per device; the stream binding and the two GEMMs stay under the lock
    static std::mutex mu;
    std::lock_guard<std::mutex> lk(mu);
    if (!c.handle[dev] && c.create(&c.handle[dev]) != 0) return FAV_ERR_CUDA;
    if (c.set_stream(c.handle[dev], stream) != 0) return FAV_ERR_CUDA;
    const int G = a.Hq / a.Hkv, N = a.Nq, Nk = a.Nkv, D = a.D, M = G * N;
    const int batch = a.B * a.Hkv;
    const bool bf = a.dtype == FAV_BF16;
    const int io = bf ? kCudaR16BF : kCudaR16F;
    float *S = static_cast<float *>(workspace);
    const float alpha_s = a.scale, alpha_o = kPUnscale, zero = 0.f;
    // bf16: V as fp16 under a power of two per KV head (contiguous [B, Hkv, Nkv, D])
    const void *v16 = a.v;
    const float *v_scale = nullptr;
    if (bf) {
        FavStrides vs16;
        const fav_status st = fav_v16_convert(a, v_workspace, stream, &v16, &vs16, &v_scale);
        if (st != FAV_OK) return st;
    }
    // S^T (Nk x M, column-major) = K (Nk x D) . Q^T (D x M): row-major S = Q K^T, per KV head
    if (c.gemm(c.handle[dev], kCublasOpT, kCublasOpN, Nk, M, D, &alpha_s, a.k, io, D,
               (long long)Nk * D, a.q, io, D, (long long)M * D, &zero, S, kCudaR32F, Nk,
               (long long)M * Nk, batch, kCublasCompute32F, kCublasGemmDefault) != 0)
        return FAV_ERR_CUDA;
    const long long rows = (long long)a.B * a.Hq * N;
    const cudaError_t e = launch_softmax(S, a.lse, rows, N, Nk, a.causal, stream);
    if (e != cudaSuccess || fav_debug_sync("fav_nonflash_softmax_kernel", stream))
        return FAV_ERR_CUDA;
    // O^T (D x M) = 2^-11 V^T (D x Nk) . P^T (Nk x M), all fp16; P rows are 2 * Nk elements
    // apart (in place).  fp16 I/O: O itself; bf16 I/O: O * 2^-e, converted in place below.
    if (c.gemm(c.handle[dev], kCublasOpN, kCublasOpN, D, M, Nk, &alpha_o, v16, kCudaR16F, D,
               (long long)Nk * D, S, kCudaR16F, 2 * Nk, (long long)M * Nk * 2, &zero, a.o,
               kCudaR16F, D, (long long)M * D, batch, kCublasCompute32F, kCublasGemmDefault) != 0)
        return FAV_ERR_CUDA;
    if (bf) {
        const long long n8 = rows * D / 8;
        fav_nonflash_unscale_kernel<<<(unsigned)((n8 + 255) / 256), 256, 0, stream>>>(
            static_cast<uint4 *>(a.o), v_scale, n8, D, N, a.Hq, G, a.Hkv);
        if (cudaGetLastError() != cudaSuccess ||
            fav_debug_sync("fav_nonflash_unscale_kernel", stream))
            return FAV_ERR_CUDA;
    }
    return FAV_OK;
}
