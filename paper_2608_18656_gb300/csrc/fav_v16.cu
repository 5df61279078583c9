// fav_v16.cu -- bf16 V converted to fp16 under a power-of-two scale per KV head, for the
// prefill kernels' P.V products (both run P.V with fp16 weights: see fav_prefill.cu).
#include <math.h>

#include <algorithm>

#include "fav_device.cuh"
#include "fav_internal.h"

namespace {

// Pass 1: per KV head and block, the largest finite |v| (as float bits: non-negative floats
// order like their bit patterns), written to vmax_part[head * gridDim.x + blockIdx.x]; every
// slot is written, so the array needs no initialisation and no atomics.  The next pass is
// launched as a programmatic dependent: it may be scheduled once every block here has started.
// V rows are read through its strides (element offsets of head (b, g): b * vs.b + g * vs.h,
// row n: + n * vs.n), D / 8 16-byte chunks per row.  The head's first element is computed once
// per thread; chunk i of the head is 8 i elements further when its rows are contiguous
// (vs.n == D), else row i / d8, chunk i % d8 (32-bit arithmetic: i < 2^31).  (64-bit divisions
// per chunk had left these passes bound by integer arithmetic.)
__device__ __forceinline__ const uint16_t *fav_v_head(const uint16_t *v, FavStrides vs, int Hkv,
                                                      long long head) {
    return v + (head / Hkv) * vs.b + (head % Hkv) * vs.h;
}
__device__ __forceinline__ const uint4 *fav_v_chunk(const uint16_t *vh, long long row_stride,
                                                    bool dense, uint32_t i, uint32_t d8) {
    if (dense) return reinterpret_cast<const uint4 *>(vh) + i;
    return reinterpret_cast<const uint4 *>(vh + (long long)(i / d8) * row_stride + (i % d8) * 8);
}

// Each thread keeps kLoads independent 16-byte loads in flight (chunks i, i + stride, ...):
// one load per iteration left the passes bound by load latency (1.6 TB/s).
constexpr int kLoads = 4;

__global__ void __launch_bounds__(256)
fav_vmax_kernel(const uint16_t *__restrict__ v, FavStrides vs, int Hkv, int d8,
                unsigned *__restrict__ vmax_part, long long per_head) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    __shared__ unsigned wmax[8];
    const long long head = blockIdx.y;
    const long long stride = (long long)gridDim.x * blockDim.x;
    const uint16_t *vh = fav_v_head(v, vs, Hkv, head);
    const bool dense = vs.n == 8LL * d8;
    unsigned mx = 0;
    for (long long i0 = blockIdx.x * (long long)blockDim.x + threadIdx.x; i0 < per_head;
         i0 += kLoads * stride) {
        uint4 w[kLoads];
#pragma unroll
        for (int r = 0; r < kLoads; ++r) {
            const long long i = i0 + r * stride;
            w[r] = i < per_head ? *fav_v_chunk(vh, vs.n, dense, (uint32_t)i, (uint32_t)d8)
                                : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int r = 0; r < kLoads; ++r) {
            const uint32_t u[4] = {w[r].x, w[r].y, w[r].z, w[r].w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                // two bf16 values: |x| bits are the low 15 bits of each half, moved to float bits
                const uint32_t lo = (u[k] & 0x7FFFu) << 16, hi = u[k] & 0x7FFF0000u;
                if (lo < 0x7F800000u) mx = max(mx, lo);      // finite only
                if (hi < 0x7F800000u) mx = max(mx, hi);
            }
        }
    }
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) mx = max(mx, __shfl_xor_sync(~0u, mx, d));
    if ((threadIdx.x & 31) == 0) wmax[threadIdx.x >> 5] = mx;
    __syncthreads();
    if (threadIdx.x == 0) {
#pragma unroll
        for (int w = 1; w < 8; ++w) mx = max(mx, wmax[w]);
        vmax_part[head * gridDim.x + blockIdx.x] = mx;
    }
}

// Scale exponent of a head: e = floor(log2(max|v|)) - 14, so that max|v| * 2^-e < 2^15 (fp16
// max 65504); a head of zeros keeps e = 0.  Clamped to [-126, 127] so that 2^e and 2^-e are
// both finite normal floats (a head whose maximum is below 2^-112 is scaled by 2^126 only).
__device__ __forceinline__ int fav_v16_exponent(unsigned vmax_bits) {
    if (vmax_bits == 0) return 0;
    const int e2 = (int)(vmax_bits >> 23) - 127;        // floor(log2), -127 for subnormals
    return min(127, max(-126, e2 - 14));
}

// Pass 2: v16 = fp16(v * 2^-e).  A bf16 value has 8 significant bits, which fp16 holds exactly
// down to 2^-17 (subnormals included), so every |v| >= 2^(e-17) -- everything within about
// 2^-31 of the head's maximum -- converts exactly; smaller values err by less than 2^(e-25).
// Non-finite values stay non-finite.  Also stores v_scale = 2^e.  A programmatic dependent of
// pass 1 (it waits for that grid's completion before reading the partial maxima); the prefill
// kernel is in turn launched as a dependent of this one.
__global__ void __launch_bounds__(256)
fav_v16_kernel(const uint16_t *__restrict__ v, FavStrides vs, int Hkv, int d8,
               uint4 *__restrict__ v16, const unsigned *__restrict__ vmax_part,
               float *__restrict__ v_scale, long long per_head) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    __shared__ unsigned head_max;
    const long long head = blockIdx.y;
    if (threadIdx.x < 32) {   // the head's maximum from pass 1's gridDim.x (= this grid's) partials
        unsigned m = 0;
        for (unsigned i = threadIdx.x; i < gridDim.x; i += 32) m = max(m, vmax_part[head * gridDim.x + i]);
#pragma unroll
        for (int d = 16; d > 0; d >>= 1) m = max(m, __shfl_xor_sync(~0u, m, d));
        if (threadIdx.x == 0) head_max = m;
    }
    __syncthreads();
    const int e = fav_v16_exponent(head_max);
    if (blockIdx.x == 0 && threadIdx.x == 0) v_scale[head] = ldexpf(1.f, e);
    const float inv = ldexpf(1.f, -e);
    uint4 *dst = v16 + head * per_head;        // contiguous [B, Hkv, Nkv, D]
    const long long stride = (long long)gridDim.x * blockDim.x;
    const uint16_t *vh = fav_v_head(v, vs, Hkv, head);
    const bool dense = vs.n == 8LL * d8;
    for (long long i0 = blockIdx.x * (long long)blockDim.x + threadIdx.x; i0 < per_head;
         i0 += kLoads * stride) {
        uint4 w[kLoads];
#pragma unroll
        for (int r = 0; r < kLoads; ++r) {
            const long long i = i0 + r * stride;
            w[r] = i < per_head ? *fav_v_chunk(vh, vs.n, dense, (uint32_t)i, (uint32_t)d8)
                                : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int r = 0; r < kLoads; ++r) {
            const long long i = i0 + r * stride;
            if (i >= per_head) break;
            const uint32_t u[4] = {w[r].x, w[r].y, w[r].z, w[r].w};
            uint32_t h[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float lo = __uint_as_float(u[k] << 16) * inv;
                const float hi = __uint_as_float(u[k] & 0xFFFF0000u) * inv;
                h[k] = fav::Elem<__half>::pack(lo, hi);
            }
            dst[i] = make_uint4(h[0], h[1], h[2], h[3]);
        }
    }
}

// Blocks per KV head of both passes: about eight 256-thread blocks per SM over all heads, each
// thread with kLoads loads in flight.
unsigned v16_blocks_x(const FavArgs &a) {
    const long long heads = (long long)a.B * a.Hkv;
    const long long per_head = (long long)a.Nkv * a.D / 8;      // uint4 chunks (D % 8 == 0)
    return (unsigned)std::max<long long>(
        1, std::min<long long>((per_head + 256LL * kLoads - 1) / (256LL * kLoads),
                               std::max<long long>(1, 8LL * std::max(1, a.num_sms) / std::max(1LL, heads))));
}

// workspace of the kV16 path: [fp16 V][per-block maxima: heads x blocks][scale per KV head]
struct V16Layout {
    size_t v16, vmax, scale, total;
    explicit V16Layout(const FavArgs &a) {
        const size_t heads = (size_t)a.B * a.Hkv;
        auto up = [](size_t x) { return (x + 255) & ~(size_t)255; };
        v16 = 0;
        vmax = up(heads * a.Nkv * a.D * 2);
        scale = vmax + up(heads * v16_blocks_x(a) * 4);
        total = scale + up(heads * 4);
    }
};

}  // namespace

size_t fav_v16_workspace_bytes(const FavArgs &a) { return V16Layout(a).total; }

fav_status fav_v16_convert(const FavArgs &a, void *workspace, cudaStream_t stream,
                           const void **v16, FavStrides *v16_strides, const float **v_scale) {
    const int D = a.D;
    if (!workspace) return FAV_ERR_NO_MEMORY;
    const V16Layout L(a);
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    unsigned *vmax = reinterpret_cast<unsigned *>(ws + L.vmax);
    float *vsc = reinterpret_cast<float *>(ws + L.scale);
    const long long heads = (long long)a.B * a.Hkv;
    const long long per_head = (long long)a.Nkv * a.D / 8;      // uint4 chunks (D % 8 == 0)
    if (heads > 65535 || per_head >= (1LL << 31)) return FAV_ERR_UNSUPPORTED;
    const uint16_t *vsrc = static_cast<const uint16_t *>(a.v);
    uint4 *v16p = reinterpret_cast<uint4 *>(ws + L.v16);
    const unsigned bx = v16_blocks_x(a);
    fav_vmax_kernel<<<dim3(bx, (unsigned)heads), 256, 0, stream>>>(vsrc, a.vs, a.Hkv, D / 8, vmax,
                                                                   per_head);
    if (cudaGetLastError() != cudaSuccess || fav_debug_sync("fav_vmax_kernel", stream))
        return FAV_ERR_CUDA;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(bx, (unsigned)heads);
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, fav_v16_kernel, vsrc, a.vs, a.Hkv, D / 8, v16p,
                           (const unsigned *)vmax, vsc, per_head) != cudaSuccess ||
        cudaGetLastError() != cudaSuccess || fav_debug_sync("fav_v16_kernel", stream))
        return FAV_ERR_CUDA;
    *v16 = ws + L.v16;
    *v16_strides = fav_contiguous_strides(a.Hkv, a.Nkv, D);
    *v_scale = vsc;
    return FAV_OK;
}
