// fav_internal.h -- host-side interface between the C ABI (fav_api.cu) and the kernel files.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/fav.h"

// Element strides of a [B, H, N, D] tensor whose D axis is contiguous (batch, head, token).
struct FavStrides {
    long long b, h, n;
};

struct FavArgs {
    const void *q, *k, *v;
    void *o;
    float *lse;                          // [B, Hq, Nq] contiguous
    FavStrides qs, ks, vs, os;           // strides of q, k, v, o
    int B, Hq, Hkv, Nq, Nkv, D;
    float scale;
    int causal;
    fav_dtype dtype;
    int *dev_status;   // device word set by bounded waits that gave up
    int num_sms;
    int prefill_grid = 0;   // cap on the persistent prefill grid (0 = one CTA per SM)
};

// Generic CUDA-core kernel (fav_simt.cu).
bool fav_simt_supported(const FavArgs &a);
fav_status fav_launch_simt(const FavArgs &a, cudaStream_t s);

// Split-KV decode kernel + combine (fav_decode.cu).
bool fav_decode_supported(const FavArgs &a);
int fav_decode_num_tiles(const FavArgs &a);
int fav_decode_auto_splits(const FavArgs &a);
size_t fav_decode_workspace_bytes(const FavArgs &a, int splits);
fav_status fav_launch_decode(const FavArgs &a, int splits, void *workspace, cudaStream_t s);
// Paged KV cache for the decode kernel: K and V are pools of num_pages pages of
// [page_size, Hkv, D]; sequence b's key n lives in page block_table[b * max_pages +
// n / page_size], row n % page_size; sequence b has seq_lens[b] keys (device arrays).
struct FavPaged {
    const int *block_table;
    const int *seq_lens;
    int max_pages, page_size, num_pages;
};
// Keys per tile of the decode kernel at head dimension D, and the capacity (page references
// per thread block) of its page list: a split must cover at most that many boxes.
int fav_decode_tile_keys(int D);
int fav_decode_page_slots();
fav_status fav_launch_decode_paged(const FavArgs &a, const FavPaged &pg, int splits,
                                   void *workspace, cudaStream_t s);

// tcgen05 prefill kernel (fav_prefill.cu).
bool fav_prefill_supported(const FavArgs &a);
// Device workspace the prefill launch needs (0 for fp16; bf16: the fp16 copy of V and its
// per-head scales), and the launch itself with that workspace.
size_t fav_prefill_workspace_bytes(const FavArgs &a);
// bf16 V -> fp16 V with a power-of-two scale per KV head (fav_v16.cu), for the prefill
// kernels: workspace size, and the conversion (two kernels on `stream`), which returns the
// fp16 copy (contiguous [B, Hkv, Nkv, D], its strides) and the per-head scales 2^e.
size_t fav_v16_workspace_bytes(const FavArgs &a);
fav_status fav_v16_convert(const FavArgs &a, void *workspace, cudaStream_t stream,
                           const void **v16, FavStrides *v16_strides, const float **v_scale);
// The two prefill kernel designs (fav_prefill.cu: D = 128; fav_prefill_pair.cu: D = 64).
fav_status fav_launch_prefill_split(const FavArgs &a, void *workspace, cudaStream_t s);
fav_status fav_launch_prefill_pair(const FavArgs &a, void *workspace, cudaStream_t s);
// Packed variable-length batch (D = 128): a is the [1, H, total, D] view of the packed tensors
// (Nq = total_q, Nkv = total_k, token strides H * D); units is the device table built by
// fav_prefill_varlen, two int4 per unit: {sequence, head, query tile, key tiles},
// {first query row, first key row, query length, key length}, heaviest causal work first.
fav_status fav_launch_prefill_varlen(const FavArgs &a, const int4 *units, int n_units,
                                     void *workspace, cudaStream_t s);
// The same for D = 64 (fav_prefill_pair.cu): three int4 per unit, a pair of query tiles of one
// sequence: {sequence, head 0, head 1, tile 0}, {tile 1, key tiles 0, key tiles 1, first query
// row}, {first key row, query length, key length, -}.
fav_status fav_launch_prefill_pair_varlen(const FavArgs &a, const int4 *units, int n_units,
                                          void *workspace, cudaStream_t s);
fav_status fav_launch_prefill(const FavArgs &a, void *workspace, cudaStream_t s);

// Non-fused attention (fav_nonflash.cu): cuBLAS S = scale Q K^T (fp32), masked row softmax
// (fp16 weights * 2^11 in place over S, LSE), cuBLAS O = P V.  workspace:
// fav_nonflash_workspace_bytes; v_workspace (bf16 only): fav_v16_workspace_bytes, for the fp16
// copy of V and its per-head scales (a.num_sms sizes the conversion grid).
size_t fav_nonflash_workspace_bytes(const FavArgs &a);
// Shape limits of this path (fp16/bf16, a score row in shared memory, int GEMM sizes).
bool fav_nonflash_shape_ok(const FavArgs &a);
// Whether cuBLAS could be loaded.
bool fav_nonflash_available();
fav_status fav_launch_nonflash(const FavArgs &a, void *workspace, void *v_workspace,
                               cudaStream_t s);

// With FAV_DEBUG_SYNC=1 in the environment: synchronise `s` after a launch and report a
// failure of kernel `what` on stderr.  Returns true if the kernel failed.  No-op otherwise.
bool fav_debug_sync(const char *what, cudaStream_t s);

// Shared with the allocation-free decode entry point (fav_noalloc.cu), defined in fav_api.cu:
// the same shape/argument rules as fav_forward, the device's status word and SM count, and
// the process-wide decode split override (0 = automatic).
fav_status fav_internal_validate(int B, int Hq, int Hkv, int Nq, int Nkv, int D, float scale,
                                 int causal, fav_dtype dtype);
fav_status fav_internal_device_info(int **dev_status, int *num_sms);
int fav_internal_decode_splits_override();

// Contiguous strides of a [B, H, N, D] tensor.
inline FavStrides fav_contiguous_strides(int H, int N, int D) {
    return FavStrides{(long long)H * N * D, (long long)N * D, (long long)D};
}

// Tensor-map encoding through the driver entry point (fav_api.cu).
// 4-D map over a [batch, heads, rows, D] tensor of 16-bit elements with element strides `st`
// (D contiguous; the strides must be multiples of 8 elements), box {64, box_rows, 1, 1},
// 128-byte swizzle, zero fill out of bounds.  Coordinates (x, row, head, batch).
fav_status fav_make_tmap_4d(void *tmap /* CUtensorMap* */, const void *base, int D, int rows,
                            int heads, int batch, FavStrides st, int box_rows);
// The same tensor as a 5-D view whose box of box_rows rows covers all D columns in one TMA
// copy (D / 64 blocks of 64 columns, each box_rows x 128 bytes, 128-byte swizzle).
fav_status fav_make_tmap_tiles(void *tmap /* CUtensorMap* */, const void *base, int D, int rows,
                               int heads, int batch, FavStrides st, int box_rows);
