// fav_noalloc.cu -- fav_decode_noalloc: the split-KV decode path without any device allocation.
//
// fav_forward keeps its split-KV partials in a workspace it allocates on first use with
// cudaMallocAsync.  Some callers cannot let a library allocate device memory: an inference
// server that reserves all device memory for its own pool at start-up (a library allocation
// then fails, or fragments and competes with that pool), or a latency-critical decode loop that
// forbids allocator calls after initialisation because they can take driver locks and stall.
// This entry point runs the same decode and combine kernels with the partials in a fixed
// file-scope device array instead, so it never calls cudaMalloc, cudaMallocAsync, cudaFree or
// any allocating library routine.
//
// Set-up: the first call on each device (with that device current) looks up the array's
// device address with cudaGetSymbolAddress -- in host code the array's name is only a host-side
// stand-in, not a device address -- and caches it per device.  That first call should come
// before any stream capture on the device.  The array is shared by every call and keeps the
// last call's contents; nothing in it needs to start at zero, because every partial that the
// combine kernel reads is written by the decode kernel of the same call.  Calls that overlap on
// the GPU (e.g. on two streams at once) race on the array and must be serialised by the caller.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <algorithm>
#include <mutex>

#include "fav_internal.h"

namespace {

constexpr int kMaxDevices = 64;

// Every GPU that loads the library holds this array until the process exits.
static __device__ __align__(256) unsigned char g_noalloc_scratch[FAV_NOALLOC_SCRATCH_BYTES];

struct NoallocDevice {
    bool ready = false;
    void *scratch = nullptr;   // device address of g_noalloc_scratch on this device
};
std::mutex g_noalloc_mu;
NoallocDevice g_noalloc_dev[kMaxDevices];

// Once per device, with that device current: the array's device address.
fav_status noalloc_scratch(void **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return FAV_ERR_CUDA;
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    NoallocDevice &d = g_noalloc_dev[dev];
    if (!d.ready) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) {
            cudaGetLastError();
            return FAV_ERR_CUDA;
        }
        d.scratch = p;
        d.ready = true;
    }
    *out = d.scratch;
    return FAV_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" FAV_API fav_status fav_decode_noalloc(const void *q, const void *k, const void *v,
                                                 void *o, float *lse, int B, int Hq, int Hkv,
                                                 int Nq, int Nkv, int D, float scale, int causal,
                                                 fav_dtype dtype, void *stream) {
    if (!q || !k || !v || !o) return FAV_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o)) return FAV_ERR_INVALID_ARG;
    if (lse && (reinterpret_cast<uintptr_t>(lse) & 3u)) return FAV_ERR_INVALID_ARG;
    fav_status st = fav_internal_validate(B, Hq, Hkv, Nq, Nkv, D, scale, causal, dtype);
    if (st != FAV_OK) return st;
    FavArgs a;
    a.q = q; a.k = k; a.v = v; a.o = o; a.lse = lse;
    a.qs = a.os = fav_contiguous_strides(Hq, Nq, D);
    a.ks = a.vs = fav_contiguous_strides(Hkv, Nkv, D);
    a.B = B; a.Hq = Hq; a.Hkv = Hkv; a.Nq = Nq; a.Nkv = Nkv; a.D = D;
    a.scale = scale; a.causal = causal; a.dtype = dtype;
    if (!fav_decode_supported(a)) return FAV_ERR_UNSUPPORTED;
    st = fav_internal_device_info(&a.dev_status, &a.num_sms);
    if (st != FAV_OK) return st;
    void *scratch = nullptr;
    st = noalloc_scratch(&scratch);
    if (st != FAV_OK) return st;
    // Same split count as fav_forward (automatic, or the process-wide override).
    const int n_tiles = fav_decode_num_tiles(a);
    int splits = fav_internal_decode_splits_override();
    if (splits <= 0) splits = fav_decode_auto_splits(a);
    splits = std::max(1, std::min(splits, n_tiles));
    const int tps = (n_tiles + splits - 1) / splits;
    splits = (n_tiles + tps - 1) / tps;
    if (fav_decode_workspace_bytes(a, splits) > (size_t)FAV_NOALLOC_SCRATCH_BYTES)
        return FAV_ERR_UNSUPPORTED;   // partials beyond the fixed array: see fav.h
    cudaGetLastError();
    return fav_launch_decode(a, splits, splits > 1 ? scratch : nullptr,
                             static_cast<cudaStream_t>(stream));
}
