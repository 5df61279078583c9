// fav_v16.cu -- bf16 V converted to fp16 under a power-of-two scale per KV head, for the
// prefill kernels' P.V products (both run P.V with fp16 weights: see fav_prefill.cu).
#include <math.h>

#include <algorithm>

#include "fav_device.cuh"
#include "fav_internal.h"

namespace {

// Pass 1: per KV head, the largest finite |v| (as float bits: non-negative floats order like
// their bit patterns, so an unsigned atomicMax finds it).
// V rows are read through its strides (element offsets of head (b, g): b * vs.b + g * vs.h,
// row n: + n * vs.n), D / 8 16-byte chunks per row.
__device__ __forceinline__ const uint4 *fav_v_chunk(const uint16_t *v, FavStrides vs, int Hkv,
                                                    long long head, long long i, int d8) {
    const long long b = head / Hkv, g = head % Hkv, n = i / d8, c = i % d8;
    return reinterpret_cast<const uint4 *>(v + b * vs.b + g * vs.h + n * vs.n + c * 8);
}

__global__ void __launch_bounds__(256)
fav_vmax_kernel(const uint16_t *__restrict__ v, FavStrides vs, int Hkv, int d8,
                unsigned *__restrict__ vmax_bits, long long per_head) {
    const long long head = blockIdx.y;
    unsigned mx = 0;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < per_head;
         i += (long long)gridDim.x * blockDim.x) {
        const uint4 w = *fav_v_chunk(v, vs, Hkv, head, i, d8);
        const uint32_t u[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            // two bf16 values: |x| bits are the low 15 bits of each half, moved to float bits
            const uint32_t lo = (u[k] & 0x7FFFu) << 16, hi = u[k] & 0x7FFF0000u;
            if (lo < 0x7F800000u) mx = max(mx, lo);      // finite only
            if (hi < 0x7F800000u) mx = max(mx, hi);
        }
    }
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) mx = max(mx, __shfl_xor_sync(~0u, mx, d));
    if ((threadIdx.x & 31) == 0 && mx) atomicMax(vmax_bits + head, mx);
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
// Non-finite values stay non-finite.  Also stores v_scale = 2^e.
__global__ void __launch_bounds__(256)
fav_v16_kernel(const uint16_t *__restrict__ v, FavStrides vs, int Hkv, int d8,
               uint4 *__restrict__ v16, const unsigned *__restrict__ vmax_bits,
               float *__restrict__ v_scale, long long per_head) {
    const long long head = blockIdx.y;
    const int e = fav_v16_exponent(vmax_bits[head]);
    if (blockIdx.x == 0 && threadIdx.x == 0) v_scale[head] = ldexpf(1.f, e);
    const float inv = ldexpf(1.f, -e);
    uint4 *dst = v16 + head * per_head;        // contiguous [B, Hkv, Nkv, D]
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < per_head;
         i += (long long)gridDim.x * blockDim.x) {
        const uint4 w = *fav_v_chunk(v, vs, Hkv, head, i, d8);
        const uint32_t u[4] = {w.x, w.y, w.z, w.w};
        uint32_t r[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float lo = __uint_as_float(u[k] << 16) * inv;
            const float hi = __uint_as_float(u[k] & 0xFFFF0000u) * inv;
            r[k] = fav::Elem<__half>::pack(lo, hi);
        }
        dst[i] = make_uint4(r[0], r[1], r[2], r[3]);
    }
}

// workspace of the kV16 path: [fp16 V][vmax bits per KV head][scale per KV head]
struct V16Layout {
    size_t v16, vmax, scale, total;
    explicit V16Layout(const FavArgs &a) {
        const size_t heads = (size_t)a.B * a.Hkv;
        auto up = [](size_t x) { return (x + 255) & ~(size_t)255; };
        v16 = 0;
        vmax = up(heads * a.Nkv * a.D * 2);
        scale = vmax + up(heads * 4);
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
    if (heads > 65535) return FAV_ERR_UNSUPPORTED;
    const unsigned bx = (unsigned)std::max<long long>(
        1, std::min<long long>((per_head + 255) / 256, std::max<long long>(1, 4LL * a.num_sms / heads)));
    if (cudaMemsetAsync(vmax, 0, heads * sizeof(unsigned), stream) != cudaSuccess)
        return FAV_ERR_CUDA;
    fav_vmax_kernel<<<dim3(bx, (unsigned)heads), 256, 0, stream>>>(
        static_cast<const uint16_t *>(a.v), a.vs, a.Hkv, D / 8, vmax, per_head);
    fav_v16_kernel<<<dim3(bx, (unsigned)heads), 256, 0, stream>>>(
        static_cast<const uint16_t *>(a.v), a.vs, a.Hkv, D / 8,
        reinterpret_cast<uint4 *>(ws + L.v16), vmax, vsc, per_head);
    if (cudaGetLastError() != cudaSuccess || fav_debug_sync("fav_v16_kernel", stream))
        return FAV_ERR_CUDA;
    *v16 = ws + L.v16;
    *v16_strides = fav_contiguous_strides(a.Hkv, a.Nkv, D);
    *v_scale = vsc;
    return FAV_OK;
}
