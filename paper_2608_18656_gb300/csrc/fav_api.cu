// fav_api.cu -- the C ABI of libfav (declared in include/fav.h): argument validation,
// kernel-family dispatch, the internal split-KV workspace, host-buffer calls, tensor maps.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>

#include <algorithm>
#include <vector>
#include <atomic>
#include <mutex>

#include "fav_device.cuh"
#include "fav_internal.h"

// Status word written by kernels whose bounded waits gave up (FAV_ERR_DEVICE_TIMEOUT).
__device__ int g_fav_device_status;

// Self-test of the bounded waits: one warp initialises a shared-memory mbarrier that nothing
// arrives on and waits for its first phase with the kernels' own wait (fav::mbar_wait_il),
// given up after limit_ns instead of FAV_WAIT_NS.  No copy and no tensor-core operation is in
// flight; the kernel records the give-up in *status and returns.
__global__ void __launch_bounds__(32) fav_wait_probe_kernel(int *status, unsigned long long limit_ns) {
    __shared__ unsigned long long bar_word;
    const uint32_t bar = fav::smem_u32(&bar_word);
    if (threadIdx.x == 0) {
        fav::mbar_init(bar, 1);
        fav::mbar_fence_init();
    }
    __syncwarp();
    (void)__all_sync(~0u, fav::mbar_wait_il(bar, 0, status, limit_ns));
}

namespace {

constexpr int kMaxDevices = 64;

struct DeviceState {
    std::atomic<bool> init{false};   // set once, under g_mu, after the fields below
    int *status = nullptr;     // device address of g_fav_device_status
    int num_sms = 0;
    void *ws = nullptr;        // split-KV partials
    size_t ws_bytes = 0;
    void *ws_pre = nullptr;    // prefill workspace (bf16: fp16 copy of V and its scales)
    size_t ws_pre_bytes = 0;
    void *ws_units = nullptr;  // unit table of a packed variable-length prefill
    size_t ws_units_bytes = 0;
    void *hbuf = nullptr;      // device copies for fav_forward_host
    size_t hbuf_bytes = 0;
    bool pipe_init = false;    // fav_forward_host pipeline: copy-in, compute, copy-out streams
    cudaStream_t s_in = nullptr, s_comp = nullptr, s_out = nullptr;
    cudaEvent_t ev_start = nullptr, ev_in[4] = {}, ev_comp[4] = {};
};

constexpr int kHostChunks = 4;

std::mutex g_mu;
DeviceState g_dev[kMaxDevices];
std::atomic<int> g_path{FAV_PATH_AUTO};
std::atomic<int> g_last_path{FAV_PATH_AUTO};
std::atomic<int> g_splits{0};
std::atomic<int> g_last_splits{0};
std::atomic<int> g_prefill_grid{0};

// The calling thread's current device's state, set up on first use (under g_mu, so that two
// threads' first calls on one device do not race).  Callers must not hold g_mu.
fav_status device_state(DeviceState **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return FAV_ERR_CUDA;
    DeviceState &d = g_dev[dev];
    if (!d.init.load(std::memory_order_acquire)) {
        std::lock_guard<std::mutex> lk(g_mu);
        if (!d.init.load(std::memory_order_relaxed)) {
            void *p = nullptr;
            if (cudaGetSymbolAddress(&p, g_fav_device_status) != cudaSuccess) return FAV_ERR_CUDA;
            int sms = 0;
            if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
                return FAV_ERR_CUDA;
            d.status = static_cast<int *>(p);
            d.num_sms = sms;
            d.init.store(true, std::memory_order_release);
        }
    }
    *out = &d;
    return FAV_OK;
}

bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

fav_status validate_shape(int B, int Hq, int Hkv, int Nq, int Nkv, int D, float scale,
                          int causal, fav_dtype dtype) {
    if (B <= 0 || Hq <= 0 || Hkv <= 0 || Nq <= 0 || Nkv <= 0 || D <= 0) return FAV_ERR_INVALID_ARG;
    if (Hq % Hkv != 0) return FAV_ERR_INVALID_ARG;
    if (causal != 0 && causal != 1) return FAV_ERR_INVALID_ARG;
    if (causal && Nq > Nkv) return FAV_ERR_INVALID_ARG;
    if (!(scale > 0.f) || !isfinite(scale)) return FAV_ERR_INVALID_ARG;
    if (dtype != FAV_F32 && dtype != FAV_F16 && dtype != FAV_BF16) return FAV_ERR_INVALID_ARG;
    const int es = dtype == FAV_F32 ? 4 : 2;
    if ((D * es) % 16 != 0) return FAV_ERR_UNSUPPORTED;        // rows must stay 16-byte aligned
    // Element counts must fit the kernels' 32-bit grid and 64-bit index arithmetic.
    const long long rows = (long long)B * Hq * Nq;
    if (rows > (1LL << 40) || (long long)B * Hkv * Nkv > (1LL << 40)) return FAV_ERR_UNSUPPORTED;
    return FAV_OK;
}

FavArgs make_args(const void *q, const void *k, const void *v, void *o, float *lse, int B, int Hq,
                  int Hkv, int Nq, int Nkv, int D, float scale, int causal, fav_dtype dtype) {
    FavArgs a;
    a.q = q; a.k = k; a.v = v; a.o = o; a.lse = lse;
    a.qs = a.os = fav_contiguous_strides(Hq, Nq, D);
    a.ks = a.vs = fav_contiguous_strides(Hkv, Nkv, D);
    a.B = B; a.Hq = Hq; a.Hkv = Hkv; a.Nq = Nq; a.Nkv = Nkv; a.D = D;
    a.scale = scale; a.causal = causal; a.dtype = dtype;
    a.dev_status = nullptr;
    a.num_sms = 0;
    return a;
}

bool decode_shaped(const FavArgs &a) {
    return (long long)a.Nq * (a.Hq / a.Hkv) <= 16;
}

// Chooses the kernel family for a validated call; FAV_PATH_AUTO if none can run it.
fav_path choose_path(const FavArgs &a) {
    const int forced = g_path.load();
    switch (forced) {
    case FAV_PATH_SIMT: return fav_simt_supported(a) ? FAV_PATH_SIMT : FAV_PATH_AUTO;
    case FAV_PATH_DECODE: return fav_decode_supported(a) ? FAV_PATH_DECODE : FAV_PATH_AUTO;
    case FAV_PATH_PREFILL: return fav_prefill_supported(a) ? FAV_PATH_PREFILL : FAV_PATH_AUTO;
    default: break;
    }
    if (a.dtype != FAV_F32) {
        if (decode_shaped(a) && fav_decode_supported(a)) return FAV_PATH_DECODE;
        if (fav_prefill_supported(a)) return FAV_PATH_PREFILL;
        if (fav_decode_supported(a)) return FAV_PATH_DECODE;
    }
    if (fav_simt_supported(a)) return FAV_PATH_SIMT;
    return FAV_PATH_AUTO;
}

fav_status ensure_buffer(void **ptr, size_t *have, size_t need, cudaStream_t s) {
    if (need <= *have) return FAV_OK;
    if (*ptr) {
        cudaFreeAsync(*ptr, s);
        *ptr = nullptr;
        *have = 0;
    }
    void *p = nullptr;
    if (cudaMallocAsync(&p, need, s) != cudaSuccess) {
        cudaGetLastError();
        return FAV_ERR_NO_MEMORY;
    }
    *ptr = p;
    *have = need;
    return FAV_OK;
}

fav_status forward_impl(const FavArgs &in, cudaStream_t stream) {
    DeviceState *ds = nullptr;
    fav_status st = device_state(&ds);
    if (st != FAV_OK) return st;
    FavArgs a = in;
    a.dev_status = ds->status;
    a.num_sms = ds->num_sms;
    a.prefill_grid = g_prefill_grid.load();
    const fav_path path = choose_path(a);
    if (path == FAV_PATH_AUTO) return FAV_ERR_UNSUPPORTED;
    cudaGetLastError();   // a stale error from elsewhere must not be reported as ours
    switch (path) {
    case FAV_PATH_SIMT:
        st = fav_launch_simt(a, stream);
        break;
    case FAV_PATH_PREFILL: {
        void *ws = nullptr;
        const size_t need = fav_prefill_workspace_bytes(a);
        if (need) {
            std::lock_guard<std::mutex> lk(g_mu);
            st = ensure_buffer(&ds->ws_pre, &ds->ws_pre_bytes, need, stream);
            ws = ds->ws_pre;
        }
        if (st == FAV_OK) st = fav_launch_prefill(a, ws, stream);
        break;
    }
    case FAV_PATH_DECODE: {
        const int n_tiles = fav_decode_num_tiles(a);
        int splits = g_splits.load();
        if (splits <= 0) splits = fav_decode_auto_splits(a);
        splits = std::max(1, std::min(splits, n_tiles));
        const int tps = (n_tiles + splits - 1) / splits;
        splits = (n_tiles + tps - 1) / tps;
        void *ws = nullptr;
        const size_t need = fav_decode_workspace_bytes(a, splits);
        if (need) {
            std::lock_guard<std::mutex> lk(g_mu);
            st = ensure_buffer(&ds->ws, &ds->ws_bytes, need, stream);
            ws = ds->ws;
        }
        if (st == FAV_OK) st = fav_launch_decode(a, splits, ws, stream);
        if (st == FAV_OK) g_last_splits.store(splits);
        break;
    }
    default:
        st = FAV_ERR_UNSUPPORTED;
    }
    if (st == FAV_OK) g_last_path.store(path);
    return st;
}

}  // namespace

fav_status fav_internal_validate(int B, int Hq, int Hkv, int Nq, int Nkv, int D, float scale,
                                 int causal, fav_dtype dtype) {
    return validate_shape(B, Hq, Hkv, Nq, Nkv, D, scale, causal, dtype);
}

fav_status fav_internal_device_info(int **dev_status, int *num_sms) {
    DeviceState *ds = nullptr;
    const fav_status st = device_state(&ds);
    if (st != FAV_OK) return st;
    *dev_status = ds->status;
    *num_sms = ds->num_sms;
    return FAV_OK;
}

int fav_internal_decode_splits_override() { return g_splits.load(); }

bool fav_debug_sync(const char *what, cudaStream_t s) {
    static const bool on = [] {
        const char *e = getenv("FAV_DEBUG_SYNC");
        return e && e[0] == '1';
    }();
    if (!on) return false;
    const cudaError_t e = cudaStreamSynchronize(s);
    fprintf(stderr, "[fav debug] %s: %s\n", what, cudaGetErrorString(e));
    return e != cudaSuccess;
}

static PFN_cuTensorMapEncodeTiled_v12000 tmap_encoder() {
    static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    });
    return encode;
}

fav_status fav_make_tmap_4d(void *tmap, const void *base, int D, int rows, int heads, int batch,
                            FavStrides st, int box_rows) {
    const PFN_cuTensorMapEncodeTiled_v12000 encode = tmap_encoder();
    if (!encode) return FAV_ERR_CUDA;
    const cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)rows, (cuuint64_t)heads,
                                (cuuint64_t)batch};
    // A stride of 0 is only accepted on an axis of size 1 (validation), where only coordinate 0
    // is ever read: it gets a nominal nonzero stride for the encoder.
    auto bstride = [](long long e, long long fallback) {
        return (cuuint64_t)((e > 0 ? e : fallback) * 2);
    };
    const cuuint64_t strides[3] = {bstride(st.n, D), bstride(st.h, (long long)rows * D),
                                   bstride(st.b, (long long)heads * rows * D)};
    const cuuint32_t box[4] = {64, (cuuint32_t)box_rows, 1, 1};
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = encode(reinterpret_cast<CUtensorMap *>(tmap), CU_TENSOR_MAP_DATA_TYPE_UINT16, 4,
                        const_cast<void *>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? FAV_OK : FAV_ERR_CUDA;
}

// 5-D view (64 elements, rows, D / 64 column blocks, heads, batch) of a [B, H, N, D] tensor: a
// box of box_rows rows spans all D columns in ONE copy instruction and lands in shared memory
// as D / 64 consecutive 64-column blocks of box_rows x 128 bytes (128-byte swizzle) -- the same
// layout as D / 64 separate 64-column boxes.  (A TMA engine's throughput per issuing thread is
// bounded per instruction, so one copy per tile instead of two matters for D = 128.)
fav_status fav_make_tmap_tiles(void *tmap, const void *base, int D, int rows, int heads,
                               int batch, FavStrides st, int box_rows) {
    const PFN_cuTensorMapEncodeTiled_v12000 encode = tmap_encoder();
    if (!encode) return FAV_ERR_CUDA;
    const int blocks = D / 64;
    const cuuint64_t dims[5] = {64, (cuuint64_t)rows, (cuuint64_t)blocks, (cuuint64_t)heads,
                                (cuuint64_t)batch};
    auto bstride = [](long long e, long long fallback) {
        return (cuuint64_t)((e > 0 ? e : fallback) * 2);
    };
    const cuuint64_t strides[4] = {bstride(st.n, D), 128, bstride(st.h, (long long)rows * D),
                                   bstride(st.b, (long long)heads * rows * D)};
    const cuuint32_t box[5] = {64, (cuuint32_t)box_rows, (cuuint32_t)blocks, 1, 1};
    const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    CUresult r = encode(reinterpret_cast<CUtensorMap *>(tmap), CU_TENSOR_MAP_DATA_TYPE_UINT16, 5,
                        const_cast<void *>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? FAV_OK : FAV_ERR_CUDA;
}

extern "C" {

fav_status fav_forward(const void *q, const void *k, const void *v, void *o, float *lse, int B,
                       int Hq, int Hkv, int Nq, int Nkv, int D, float scale, int causal,
                       fav_dtype dtype, void *stream) {
    if (!q || !k || !v || !o) return FAV_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(o, 16))
        return FAV_ERR_INVALID_ARG;
    if (lse && !aligned(lse, 4)) return FAV_ERR_INVALID_ARG;
    fav_status st = validate_shape(B, Hq, Hkv, Nq, Nkv, D, scale, causal, dtype);
    if (st != FAV_OK) return st;
    const FavArgs a = make_args(q, k, v, o, lse, B, Hq, Hkv, Nq, Nkv, D, scale, causal, dtype);
    return forward_impl(a, static_cast<cudaStream_t>(stream));
}

fav_status fav_prefill_varlen(const void *q, const void *k, const void *v, void *o, float *lse,
                              const int *cu_seqlens_q, const int *cu_seqlens_k, int B, int Hq,
                              int Hkv, int D, float scale, int causal, fav_dtype dtype,
                              void *stream) {
    if (!q || !k || !v || !o || !cu_seqlens_q || !cu_seqlens_k) return FAV_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(o, 16))
        return FAV_ERR_INVALID_ARG;
    if (lse && !aligned(lse, 4)) return FAV_ERR_INVALID_ARG;
    if (B <= 0 || (causal != 0 && causal != 1)) return FAV_ERR_INVALID_ARG;
    if (cu_seqlens_q[0] != 0 || cu_seqlens_k[0] != 0) return FAV_ERR_INVALID_ARG;
    for (int b = 0; b < B; ++b) {
        const int lq = cu_seqlens_q[b + 1] - cu_seqlens_q[b];
        const int lk = cu_seqlens_k[b + 1] - cu_seqlens_k[b];
        if (cu_seqlens_q[b + 1] < cu_seqlens_q[b] || cu_seqlens_k[b + 1] < cu_seqlens_k[b])
            return FAV_ERR_INVALID_ARG;
        if (lq > 0 && lk == 0) return FAV_ERR_INVALID_ARG;   // queries with no key at all
        if (causal && lq > lk) return FAV_ERR_INVALID_ARG;   // bottom-right alignment
    }
    const int total_q = cu_seqlens_q[B], total_k = cu_seqlens_k[B];
    fav_status st = validate_shape(1, Hq, Hkv, std::max(total_q, 1), std::max(total_k, 1), D,
                                   scale, 0, dtype);
    if (st != FAV_OK) return st;
    if ((dtype != FAV_F16 && dtype != FAV_BF16) || (D != 128 && D != 64)) return FAV_ERR_UNSUPPORTED;
    if (total_q == 0) return FAV_OK;                       // nothing to compute
    auto key_tiles = [&](int t, int lq, int lk) {          // key tiles of query tile t
        const int kv_end = causal ? std::min(lk, t * 128 + 128 + lk - lq) : lk;
        return (kv_end + 127) / 128;
    };
    // units: one 128-row query tile of one head of one sequence, heaviest causal work first
    // (then sequence, tile, head: the heads of a GQA group side by side), as in the dense kernel
    // D = 64 (two-tile kernel): a unit is a pair of query tiles of one sequence -- tile t of
    // heads (h, h+1) of one GQA group when the group size is even, else tiles (2p, 2p+1) of
    // one head (a missing second tile has no key tiles).
    struct U { int s, h0, h1, t0, t1, n0, n1, q0, k0, lq, lk; };
    std::vector<U> units;
    const bool pair_heads = (Hq / Hkv) % 2 == 0;
    for (int b = 0; b < B; ++b) {
        const int lq = cu_seqlens_q[b + 1] - cu_seqlens_q[b];
        const int lk = cu_seqlens_k[b + 1] - cu_seqlens_k[b];
        const int ntq = (lq + 127) / 128;
        const int q0 = cu_seqlens_q[b], k0 = cu_seqlens_k[b];
        if (D == 128) {
            for (int t = 0; t < ntq; ++t)
                for (int h = 0; h < Hq; ++h)
                    units.push_back(U{b, h, h, t, t, key_tiles(t, lq, lk), 0, q0, k0, lq, lk});
        } else if (pair_heads) {
            for (int t = 0; t < ntq; ++t)
                for (int h = 0; h < Hq; h += 2) {
                    const int n = key_tiles(t, lq, lk);
                    units.push_back(U{b, h, h + 1, t, t, n, n, q0, k0, lq, lk});
                }
        } else {
            for (int t = 0; t < ntq; t += 2)
                for (int h = 0; h < Hq; ++h)
                    units.push_back(U{b, h, h, t, t + 1, key_tiles(t, lq, lk),
                                      t + 1 < ntq ? key_tiles(t + 1, lq, lk) : 0, q0, k0, lq, lk});
        }
    }
    if (units.size() + 4096 > 0x7fffffffu) return FAV_ERR_UNSUPPORTED;
    std::stable_sort(units.begin(), units.end(), [](const U &x, const U &y) {
        const int wx = std::max(x.n0, x.n1), wy = std::max(y.n0, y.n1);
        if (wx != wy) return wx > wy;
        if (x.s != y.s) return x.s < y.s;
        if (x.t0 != y.t0) return x.t0 < y.t0;
        return x.h0 < y.h0;
    });
    const int per = D == 128 ? 8 : 12;                     // ints per unit in the table
    std::vector<int> table(units.size() * per);
    for (size_t i = 0; i < units.size(); ++i) {
        const U &u = units[i];
        if (D == 128) {
            const int e[8] = {u.s, u.h0, u.t0, u.n0, u.q0, u.k0, u.lq, u.lk};
            std::copy(e, e + 8, table.begin() + 8 * i);
        } else {
            const int e[12] = {u.s, u.h0, u.h1, u.t0, u.t1, u.n0, u.n1, u.q0, u.k0, u.lq, u.lk, 0};
            std::copy(e, e + 12, table.begin() + 12 * i);
        }
    }
    FavArgs a = make_args(q, k, v, o, lse, 1, Hq, Hkv, total_q, total_k, D, scale, causal, dtype);
    a.qs = a.os = FavStrides{(long long)total_q * Hq * D, (long long)D, (long long)Hq * D};
    a.ks = a.vs = FavStrides{(long long)total_k * Hkv * D, (long long)D, (long long)Hkv * D};
    DeviceState *ds = nullptr;
    st = device_state(&ds);
    if (st != FAV_OK) return st;
    a.dev_status = ds->status;
    a.num_sms = ds->num_sms;
    a.prefill_grid = g_prefill_grid.load();
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaGetLastError();
    void *ws = nullptr;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        const size_t tb = table.size() * sizeof(int);
        st = ensure_buffer(&ds->ws_units, &ds->ws_units_bytes, tb, s);
        // (pageable source: the call returns once the table has been staged for the copy)
        if (st == FAV_OK && cudaMemcpyAsync(ds->ws_units, table.data(), tb,
                                            cudaMemcpyHostToDevice, s) != cudaSuccess)
            st = FAV_ERR_CUDA;
        const size_t need = fav_prefill_workspace_bytes(a);
        if (st == FAV_OK && need) st = ensure_buffer(&ds->ws_pre, &ds->ws_pre_bytes, need, s);
        ws = ds->ws_pre;
    }
    if (st == FAV_OK)
        st = D == 128 ? fav_launch_prefill_varlen(a, static_cast<const int4 *>(ds->ws_units),
                                                  (int)units.size(), ws, s)
                      : fav_launch_prefill_pair_varlen(a, static_cast<const int4 *>(ds->ws_units),
                                                       (int)units.size(), ws, s);
    if (st == FAV_OK) g_last_path.store(FAV_PATH_PREFILL);
    return st;
}

fav_status fav_decode_paged(const void *q, const void *k_cache, const void *v_cache, void *o,
                            float *lse, const int *block_table, const int *seq_lens, int B,
                            int Hq, int Hkv, int Nq, int max_pages, int page_size, int num_pages,
                            int D, float scale, int causal, fav_dtype dtype, void *stream) {
    if (!q || !k_cache || !v_cache || !o || !block_table || !seq_lens) return FAV_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(o, 16))
        return FAV_ERR_INVALID_ARG;
    if ((lse && !aligned(lse, 4)) || !aligned(block_table, 4) || !aligned(seq_lens, 4))
        return FAV_ERR_INVALID_ARG;
    if (max_pages <= 0 || num_pages <= 0 || page_size <= 0) return FAV_ERR_INVALID_ARG;
    // pages of 16 .. 65536 rows, a power of two: a key tile then lies in one page, or a page
    // holds whole 1024-byte swizzle atoms of a tile
    if (page_size < 16 || page_size > 65536 || (page_size & (page_size - 1)) != 0)
        return FAV_ERR_UNSUPPORTED;
    const long long max_len = (long long)max_pages * page_size;
    if (max_len > 0x7fffffffLL / 2) return FAV_ERR_UNSUPPORTED;
    fav_status st = validate_shape(B, Hq, Hkv, Nq, (int)max_len, D, scale, causal, dtype);
    if (st != FAV_OK) return st;
    FavArgs a = make_args(q, k_cache, v_cache, o, lse, B, Hq, Hkv, Nq, (int)max_len, D, scale,
                          causal, dtype);
    if (!fav_decode_supported(a)) return FAV_ERR_UNSUPPORTED;
    if ((long long)page_size * Hkv * D * 2 >= (1LL << 40)) return FAV_ERR_UNSUPPORTED;
    DeviceState *ds = nullptr;
    st = device_state(&ds);
    if (st != FAV_OK) return st;
    a.dev_status = ds->status;
    a.num_sms = ds->num_sms;
    const FavPaged pg{block_table, seq_lens, max_pages, page_size, num_pages};
    // splits sized for the longest possible sequence; each block's boxes must fit its page list
    const int tk = fav_decode_tile_keys(D);
    const int n_tiles = fav_decode_num_tiles(a);
    const int bpt = page_size >= tk ? 1 : tk / page_size;
    int splits = g_splits.load();
    if (splits <= 0) splits = fav_decode_auto_splits(a);
    const long long min_splits =
        ((long long)n_tiles * bpt + fav_decode_page_slots() - 1) / fav_decode_page_slots();
    splits = (int)std::max<long long>(splits, min_splits);
    splits = std::max(1, std::min(splits, n_tiles));
    const int tps = (n_tiles + splits - 1) / splits;
    splits = (n_tiles + tps - 1) / tps;
    if ((long long)tps * bpt > fav_decode_page_slots()) return FAV_ERR_UNSUPPORTED;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaGetLastError();
    void *ws = nullptr;
    const size_t need = fav_decode_workspace_bytes(a, splits);
    if (need) {
        std::lock_guard<std::mutex> lk(g_mu);
        st = ensure_buffer(&ds->ws, &ds->ws_bytes, need, s);
        ws = ds->ws;
    }
    if (st == FAV_OK) st = fav_launch_decode_paged(a, pg, splits, ws, s);
    if (st == FAV_OK) {
        g_last_splits.store(splits);
        g_last_path.store(FAV_PATH_DECODE);
    }
    return st;
}

fav_status fav_forward_strided(const void *q, const void *k, const void *v, void *o, float *lse,
                               fav_strides q_strides, fav_strides k_strides,
                               fav_strides v_strides, fav_strides o_strides, int B, int Hq,
                               int Hkv, int Nq, int Nkv, int D, float scale, int causal,
                               fav_dtype dtype, void *stream) {
    if (!q || !k || !v || !o) return FAV_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(o, 16))
        return FAV_ERR_INVALID_ARG;
    if (lse && !aligned(lse, 4)) return FAV_ERR_INVALID_ARG;
    fav_status st = validate_shape(B, Hq, Hkv, Nq, Nkv, D, scale, causal, dtype);
    if (st != FAV_OK) return st;
    const long long es = dtype == FAV_F32 ? 4 : 2;
    const fav_strides all[4] = {q_strides, k_strides, v_strides, o_strides};
    for (const fav_strides &x : all) {
        if (x.batch < 0 || x.head < 0 || x.token < 0) return FAV_ERR_INVALID_ARG;
        // every row starts on a 16-byte boundary (vector loads, TMA), and TMA strides < 2^40 B
        for (long long e : {x.batch, x.head, x.token})
            if ((e * es) % 16 != 0 || e * es >= (1LL << 40)) return FAV_ERR_UNSUPPORTED;
    }
    // The output is written: its rows must not coincide (no zero stride on an axis longer than
    // 1).  Inputs: broadcasting (zero stride on a longer axis) is not supported.
    if ((o_strides.batch == 0 && B > 1) || (o_strides.head == 0 && Hq > 1) ||
        (o_strides.token == 0 && Nq > 1))
        return FAV_ERR_INVALID_ARG;
    auto broadcast = [&](const fav_strides &x, int H, int N) {
        return (x.batch == 0 && B > 1) || (x.head == 0 && H > 1) || (x.token == 0 && N > 1);
    };
    if (broadcast(q_strides, Hq, Nq) || broadcast(k_strides, Hkv, Nkv) || broadcast(v_strides, Hkv, Nkv))
        return FAV_ERR_UNSUPPORTED;
    FavArgs a = make_args(q, k, v, o, lse, B, Hq, Hkv, Nq, Nkv, D, scale, causal, dtype);
    auto conv = [](const fav_strides &x) { return FavStrides{x.batch, x.head, x.token}; };
    a.qs = conv(q_strides);
    a.ks = conv(k_strides);
    a.vs = conv(v_strides);
    a.os = conv(o_strides);
    return forward_impl(a, static_cast<cudaStream_t>(stream));
}

size_t fav_nonflash_workspace_size(int B, int Hq, int Nq, int Nkv) {
    if (B <= 0 || Hq <= 0 || Nq <= 0 || Nkv <= 0) return 0;
    FavArgs a{};
    a.B = B; a.Hq = Hq; a.Nq = Nq; a.Nkv = Nkv;
    return fav_nonflash_workspace_bytes(a);
}

fav_status fav_forward_nonflash(const void *q, const void *k, const void *v, void *o, float *lse,
                                int B, int Hq, int Hkv, int Nq, int Nkv, int D, float scale,
                                int causal, fav_dtype dtype, void *workspace,
                                size_t workspace_bytes, void *stream) {
    if (!q || !k || !v || !o || !workspace) return FAV_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(o, 16) ||
        !aligned(workspace, 16))
        return FAV_ERR_INVALID_ARG;
    if (lse && !aligned(lse, 4)) return FAV_ERR_INVALID_ARG;
    fav_status st = validate_shape(B, Hq, Hkv, Nq, Nkv, D, scale, causal, dtype);
    if (st != FAV_OK) return st;
    FavArgs a = make_args(q, k, v, o, lse, B, Hq, Hkv, Nq, Nkv, D, scale, causal, dtype);
    if (!fav_nonflash_shape_ok(a)) return FAV_ERR_UNSUPPORTED;
    if (workspace_bytes < fav_nonflash_workspace_bytes(a)) return FAV_ERR_INVALID_ARG;
    if (!fav_nonflash_available()) return FAV_ERR_UNSUPPORTED;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    void *vws = nullptr;
    if (dtype == FAV_BF16) {   // the fp16 copy of V (internal, as for fav_forward's bf16 prefill)
        DeviceState *ds = nullptr;
        st = device_state(&ds);
        if (st != FAV_OK) return st;
        a.num_sms = ds->num_sms;
        std::lock_guard<std::mutex> lk(g_mu);
        st = ensure_buffer(&ds->ws_pre, &ds->ws_pre_bytes, fav_v16_workspace_bytes(a), s);
        if (st != FAV_OK) return st;
        vws = ds->ws_pre;
    }
    cudaGetLastError();
    return fav_launch_nonflash(a, workspace, vws, s);
}

fav_status fav_forward_host(const void *q, const void *k, const void *v, void *o, float *lse,
                            int B, int Hq, int Hkv, int Nq, int Nkv, int D, float scale,
                            int causal, fav_dtype dtype, void *stream) {
    if (!q || !k || !v || !o) return FAV_ERR_INVALID_ARG;
    fav_status st = validate_shape(B, Hq, Hkv, Nq, Nkv, D, scale, causal, dtype);
    if (st != FAV_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DeviceState *ds = nullptr;
    st = device_state(&ds);
    if (st != FAV_OK) return st;
    const size_t es = dtype == FAV_F32 ? 4 : 2;
    auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
    const size_t qb = (size_t)B * Hq * Nq * D * es;
    const size_t kb = (size_t)B * Hkv * Nkv * D * es;
    const size_t lb = (size_t)B * Hq * Nq * sizeof(float);
    const size_t need = up(qb) * 2 + up(kb) * 2 + up(lb);
    uint8_t *base = nullptr;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        if (!ds->pipe_init) {
            bool okp = cudaStreamCreateWithFlags(&ds->s_in, cudaStreamNonBlocking) == cudaSuccess &&
                       cudaStreamCreateWithFlags(&ds->s_comp, cudaStreamNonBlocking) == cudaSuccess &&
                       cudaStreamCreateWithFlags(&ds->s_out, cudaStreamNonBlocking) == cudaSuccess &&
                       cudaEventCreateWithFlags(&ds->ev_start, cudaEventDisableTiming) == cudaSuccess;
            for (int c = 0; okp && c < kHostChunks; ++c)
                okp = cudaEventCreateWithFlags(&ds->ev_in[c], cudaEventDisableTiming) == cudaSuccess &&
                      cudaEventCreateWithFlags(&ds->ev_comp[c], cudaEventDisableTiming) == cudaSuccess;
            if (!okp) return FAV_ERR_CUDA;
            ds->pipe_init = true;
        }
        st = ensure_buffer(&ds->hbuf, &ds->hbuf_bytes, need, ds->s_comp);
        base = static_cast<uint8_t *>(ds->hbuf);
    }
    if (st != FAV_OK) return st;
    uint8_t *dq = base, *dk = dq + up(qb), *dv = dk + up(kb), *dout = dv + up(kb);
    float *dl = reinterpret_cast<float *>(dout + up(qb));
    // Pipeline over chunks of KV heads (batch and heads flattened: query head b*Hq + h reads KV
    // head (b*Hq + h) / G = b*Hkv + h/G, so a chunk of KV heads owns a contiguous block of q, k,
    // v, o and lse).  Chunk c is copied in on s_in, computed on s_comp, copied out on s_out;
    // the three streams overlap across chunks.
    const int G = Hq / Hkv;
    const long long heads_kv = (long long)B * Hkv;
    const int nch = (int)std::min<long long>(kHostChunks, heads_kv);
    const size_t q_head = (size_t)Nq * D * es, kv_head = (size_t)Nkv * D * es, l_head = (size_t)Nq * 4;
    const uint8_t *hq = static_cast<const uint8_t *>(q), *hk = static_cast<const uint8_t *>(k);
    const uint8_t *hv = static_cast<const uint8_t *>(v);
    uint8_t *ho = static_cast<uint8_t *>(o);
    uint8_t *hl = reinterpret_cast<uint8_t *>(lse);
    if (cudaEventRecord(ds->ev_start, s) != cudaSuccess ||
        cudaStreamWaitEvent(ds->s_in, ds->ev_start, 0) != cudaSuccess ||
        cudaStreamWaitEvent(ds->s_comp, ds->ev_start, 0) != cudaSuccess ||
        cudaStreamWaitEvent(ds->s_out, ds->ev_start, 0) != cudaSuccess)
        return FAV_ERR_CUDA;
    for (int c = 0; c < nch; ++c) {
        const long long k0 = heads_kv * c / nch, k1 = heads_kv * (c + 1) / nch;
        const size_t qo = (size_t)k0 * G * q_head, qn = (size_t)(k1 - k0) * G * q_head;
        const size_t ko = (size_t)k0 * kv_head, kn = (size_t)(k1 - k0) * kv_head;
        const size_t lo = (size_t)k0 * G * l_head, ln = (size_t)(k1 - k0) * G * l_head;
        if (cudaMemcpyAsync(dq + qo, hq + qo, qn, cudaMemcpyHostToDevice, ds->s_in) != cudaSuccess ||
            cudaMemcpyAsync(dk + ko, hk + ko, kn, cudaMemcpyHostToDevice, ds->s_in) != cudaSuccess ||
            cudaMemcpyAsync(dv + ko, hv + ko, kn, cudaMemcpyHostToDevice, ds->s_in) != cudaSuccess ||
            cudaEventRecord(ds->ev_in[c], ds->s_in) != cudaSuccess ||
            cudaStreamWaitEvent(ds->s_comp, ds->ev_in[c], 0) != cudaSuccess)
            return FAV_ERR_CUDA;
        const FavArgs a = make_args(dq + qo, dk + ko, dv + ko, dout + qo,
                                    lse ? dl + (size_t)k0 * G * Nq : nullptr, 1,
                                    (int)((k1 - k0) * G), (int)(k1 - k0), Nq, Nkv, D, scale,
                                    causal, dtype);
        st = forward_impl(a, ds->s_comp);
        if (st != FAV_OK) return st;
        if (cudaEventRecord(ds->ev_comp[c], ds->s_comp) != cudaSuccess ||
            cudaStreamWaitEvent(ds->s_out, ds->ev_comp[c], 0) != cudaSuccess ||
            cudaMemcpyAsync(ho + qo, dout + qo, qn, cudaMemcpyDeviceToHost, ds->s_out) != cudaSuccess)
            return FAV_ERR_CUDA;
        if (lse && cudaMemcpyAsync(hl + lo, reinterpret_cast<uint8_t *>(dl) + lo, ln,
                                   cudaMemcpyDeviceToHost, ds->s_out) != cudaSuccess)
            return FAV_ERR_CUDA;
    }
    if (cudaStreamSynchronize(ds->s_out) != cudaSuccess) return FAV_ERR_CUDA;
    if (cudaStreamSynchronize(ds->s_comp) != cudaSuccess) return FAV_ERR_CUDA;
    return FAV_OK;
}

const char *fav_status_string(fav_status s) {
    switch (s) {
    case FAV_OK: return "ok";
    case FAV_ERR_INVALID_ARG: return "invalid argument";
    case FAV_ERR_UNSUPPORTED: return "unsupported problem for the available kernels";
    case FAV_ERR_CUDA: return "CUDA runtime error";
    case FAV_ERR_NO_MEMORY: return "workspace allocation failed";
    case FAV_ERR_DEVICE_TIMEOUT: return "a bounded device wait timed out";
    case FAV_ERR_DEVICE_CHECK: return "a device-side check of the self-checking build failed";
    case FAV_ERR_BAD_PAGE: return "a block-table entry lies outside the page pool";
    }
    return "unknown status";
}

fav_status fav_get_last_device_status(void) {
    DeviceState *ds = nullptr;
    if (device_state(&ds) != FAV_OK) return FAV_ERR_CUDA;
    if (cudaDeviceSynchronize() != cudaSuccess) return FAV_ERR_CUDA;
    int v = 0;
    const int zero = 0;
    if (cudaMemcpyFromSymbol(&v, g_fav_device_status, sizeof(int)) != cudaSuccess) return FAV_ERR_CUDA;
    if (cudaMemcpyToSymbol(g_fav_device_status, &zero, sizeof(int)) != cudaSuccess) return FAV_ERR_CUDA;
    return v == 0 ? FAV_OK : static_cast<fav_status>(v);
}

void fav_release_workspace(void) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return;
    std::lock_guard<std::mutex> lk(g_mu);
    DeviceState &d = g_dev[dev];
    cudaDeviceSynchronize();
    if (d.ws) cudaFree(d.ws);
    if (d.ws_pre) cudaFree(d.ws_pre);
    if (d.hbuf) cudaFree(d.hbuf);
    if (d.ws_units) cudaFree(d.ws_units);
    d.ws = d.ws_pre = d.hbuf = d.ws_units = nullptr;
    d.ws_bytes = d.ws_pre_bytes = d.hbuf_bytes = d.ws_units_bytes = 0;
}

fav_status fav_set_path(fav_path p) {
    if (p < FAV_PATH_AUTO || p > FAV_PATH_PREFILL) return FAV_ERR_INVALID_ARG;
    g_path.store(p);
    return FAV_OK;
}

fav_path fav_last_path(void) { return static_cast<fav_path>(g_last_path.load()); }

fav_status fav_set_decode_splits(int n) {
    if (n < 0 || n > 4096) return FAV_ERR_INVALID_ARG;
    g_splits.store(n);
    return FAV_OK;
}

int fav_last_decode_splits(void) { return g_last_splits.load(); }

fav_status fav_check_wait_timeout(int limit_us, void *stream) {
    if (limit_us < 1 || limit_us > 1000000) return FAV_ERR_INVALID_ARG;
    DeviceState *ds = nullptr;
    const fav_status st = device_state(&ds);
    if (st != FAV_OK) return st;
    cudaGetLastError();
    fav_wait_probe_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(
        ds->status, 1000ull * (unsigned long long)limit_us);
    return cudaGetLastError() == cudaSuccess ? FAV_OK : FAV_ERR_CUDA;
}

fav_status fav_set_prefill_grid(int n) {
    if (n < 0) return FAV_ERR_INVALID_ARG;
    g_prefill_grid.store(n);
    return FAV_OK;
}

}  // extern "C"
