// fav_decode.cu -- bandwidth-bound decode attention: split-KV over thread blocks, the query
// heads of one GQA/MQA group packed as MMA rows, and a log-sum-exp combine of the splits.
//
// Method (paper, Method section): the decode stage is attention of a 1 x D query per head
// against the whole N x D key/value cache; heads that share a KV head read it once
// (GQA support: "K and V are loaded once and reused across shared attention heads").  On this
// GPU the roles of the paper's vector register packing are taken by tensor-core MMA rows:
// the Nq * G query rows that read KV head g form the M = 16 rows of an m16n8k16 MMA, so one
// pass over a K/V tile serves the whole group.
//
// Work decomposition: grid = (split, b * Hkv + g, 16-row chunk).  Each block streams its
// range of key tiles (32 keys at D = 128, 64 at D = 64) through a ring of shared-memory stages
// filled by TMA (a K producer warp and a V producer warp, 128-byte swizzle); six consumer
// warps own two ring stages each and take the tiles in turn:
//   S = Q K^T (mma.sync, fp32 accumulate)  ->  mask (key >= Nkv; causal, bottom-right)
//   -> online softmax in the exp2 domain (running max, rescale of O and l)
//   -> O += P V with P rounded to the I/O type.
// The consumer warp states are merged through shared memory; with one split the block writes
// O and LSE directly, otherwise it writes the fp32 partial (O_s, lse_s) of its key range and
// fav_combine_kernel (a programmatic dependent launch) merges them:
// L = logsumexp_s lse_s, O = sum_s exp(lse_s - L) O_s (associativity of the online softmax of
// the paper's Algorithm "ggml-vec FlashAttention").
#include <cuda.h>
#include <math.h>

#include "fav_device.cuh"
#include "fav_internal.h"

namespace {

constexpr int kConsumers = 6;     // consumer warps
constexpr int kThreads = (kConsumers + 2) * 32;   // + the K producer and the V producer
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kLog2e = 1.4426950408889634f;

// Ring of kStages stages; tile lt goes to stage lt % kStages and to consumer warp
// lt % kConsumers.  kStages is a multiple of the number of consumer warps, so each stage (and
// its pair of barriers) belongs to exactly one warp, which waits on its phases strictly in
// order: a warp can never be two phases behind a barrier it polls (parity would alias).  Two
// stages per warp let a warp compute on one tile while its next tile is loading; 12 stages of
// 16 KB keep ~192 KB of K/V reads in flight per SM (one block per SM).
template <int D> struct DecodeCfg {
    static constexpr int TK = (D == 128) ? 32 : 64;           // keys per tile
    static constexpr int kStagesPerWarp = 2;
    static constexpr int kStages = kConsumers * kStagesPerWarp;
    static constexpr int kBoxes = D / 64;                     // 64-element (128 B) boxes per row
    static constexpr int kTileBytes = TK * D * 2;             // one K (or V) tile
    static constexpr int kStageBytes = 2 * kTileBytes;
    static constexpr int kRingBytes = kStages * kStageBytes;
    static constexpr int kSmemBytes = kRingBytes + 1024 /*align*/ + 2 * kStages * 8;
    // paged cache: the page id of every box this block loads, gathered once at the start
    static constexpr int kPageSlots = 4096;
    static constexpr int kSmemBytesPaged = kSmemBytes + 4 * kPageSlots;
    static_assert(kStages % kConsumers == 0, "stages must be owned by single warps");
    static_assert(kRingBytes >= kConsumers * 16 * D * 4 + 2 * kConsumers * 16 * 4,
                  "reduction buffer must fit in the ring");
};

// Byte offset of 16-byte chunk `c` (of D/8) in key row `j` of a tile written by TMA with
// 128-byte swizzle: boxes of 64 elements, each TK rows of 128 B; chunk index XOR (row % 8).
template <int TK>
__device__ __forceinline__ uint32_t swz(int j, int c) {
    return (uint32_t)((c >> 3) * (TK * 128) + j * 128 + (((c & 7) ^ (j & 7)) << 4));
}

// kPaged: K and V are page pools ([num_pages, page_size, Hkv, D], tmK / tmV boxes of box_rows
// rows); sequence b has min(seq_lens[b], max_pages * page_size) keys, and the producer warp
// first gathers the page id of every box of the block's key range into shared memory.
template <typename T, int D, bool kPaged>
__global__ void __launch_bounds__(kThreads, 1)
fav_decode_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                  const T *__restrict__ q, FavStrides qs, T *__restrict__ o, FavStrides os,
                  float *__restrict__ lse,
                  float *__restrict__ part_o, float *__restrict__ part_lse, int Hq, int Hkv,
                  int Nq, int Nkv, int n_tiles, int tiles_per_split, int splits,
                  float scale_log2, int causal, int *status, FavPaged pg, int box_rows) {
    using Cfg = DecodeCfg<D>;
    constexpr int S = Cfg::kStages;
    constexpr int TK = Cfg::TK;
    extern __shared__ uint8_t smem_raw[];
    // 1024-byte alignment of the ring in the shared window (the 128-byte swizzle atom)
    const uint32_t raw_u32 = fav::smem_u32(smem_raw);
    uint8_t *ring = smem_raw + ((1024u - (raw_u32 & 1023u)) & 1023u);
    uint64_t *bars = reinterpret_cast<uint64_t *>(ring + Cfg::kRingBytes);
    const uint32_t ring_u32 = fav::smem_u32(ring);
    const uint32_t full0 = fav::smem_u32(bars), empty0 = full0 + 8 * S;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int split = blockIdx.x;
    const int bkv = blockIdx.y;                  // b * Hkv + g
    const int b = bkv / Hkv, g = bkv % Hkv;
    const int G = Hq / Hkv;
    const int M = Nq * G;                        // query rows that read this KV head
    const int m0 = blockIdx.z * 16;
    if constexpr (kPaged) {
        // this sequence's length (clamped to its block-table row); tiles beyond it are empty
        Nkv = min(max(pg.seq_lens[b], 0), pg.max_pages * pg.page_size);
        n_tiles = (Nkv + TK - 1) / TK;
    }
    const int tile0 = split * tiles_per_split;
    const int my_tiles = max(0, min(tiles_per_split, n_tiles - tile0));
    int *page_list = reinterpret_cast<int *>(ring + Cfg::kRingBytes + 16 * S);
    const int bpt = kPaged ? TK / box_rows : 1;               // boxes per tile and 64-column block

    // Let a dependent combine grid be scheduled once every block of this grid has started; it
    // still waits for this grid's completion before reading anything.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (threadIdx.x == 0) {
        (void)FAV_CHECK((ring_u32 & 1023u) == 0, status);
        (void)FAV_CHECK((ring_u32 - raw_u32) + Cfg::kRingBytes + 16 * S +
                            (kPaged ? 4 * Cfg::kPageSlots : 0) <= fav::dynamic_smem_bytes(), status);
        for (int s = 0; s < S; ++s) {
            fav::mbar_init(full0 + 8 * s, 2);          // the K and the V producer
            fav::mbar_init(empty0 + 8 * s, 1);
        }
        fav::mbar_fence_init();
    }
    __syncthreads();

    if (warp >= kConsumers) {
        // ---------------- producers: lane 0 of warp kConsumers streams K, of the next warp V
        // (two issuing threads double the copy instructions a block can issue per unit time) --
        const bool is_v = warp == kConsumers + 1;
        const CUtensorMap *tm = is_v ? &tmV : &tmK;
        if constexpr (kPaged) {
            // page id of box e (tile e / bpt, rows (e % bpt) * box_rows .. + box_rows); boxes
            // past the sequence read page 0 (their keys are masked).  A block-table entry outside
            // [0, num_pages) sets the device status word (FAV_ERR_BAD_PAGE) and is stored as -1:
            // the copy reads the zero fill and the consumers mask that box's keys, so they take
            // no part in the softmax.  Filled by the K warp; both producer warps then meet at a
            // named barrier (neither leaves before it).
            if (!is_v) {
                const int n_box = my_tiles * bpt;
                for (int e = lane; e < n_box && e < Cfg::kPageSlots; e += 32) {
                    const int key = (tile0 + e / bpt) * TK + (e % bpt) * box_rows;
                    int pid = 0;
                    if (key < Nkv) {
                        pid = pg.block_table[(long long)b * pg.max_pages + key / pg.page_size];
                        if (pid < 0 || pid >= pg.num_pages) {
                            atomicExch(status, (int)FAV_ERR_BAD_PAGE);
                            pid = -1;
                        }
                    }
                    page_list[e] = pid;
                }
            }
            fav::named_bar_sync(2, 64);
        }
        if (lane == 0) {
            fav::tma_prefetch_desc(tm);
            for (int lt = 0; lt < my_tiles; ++lt) {
                const int st = lt % S;
                if (lt >= S && !fav::mbar_wait(empty0 + 8 * st, ((lt / S) - 1) & 1, status)) break;
                const uint32_t full = full0 + 8 * st;
                fav::mbar_arrive_expect_tx(full, Cfg::kTileBytes);
                const int key0 = (tile0 + lt) * TK;
                const uint32_t dst = ring_u32 + st * Cfg::kStageBytes + (is_v ? Cfg::kTileBytes : 0);
                if (!FAV_CHECK(dst + Cfg::kBoxes * TK * 128 <= ring_u32 + Cfg::kRingBytes &&
                                   (dst & 1023u) == 0 && key0 < n_tiles * TK &&
                                   bkv < (int)gridDim.y, status))
                    continue;
                // One copy instruction per box: the tensor maps are 5-D views whose box covers
                // all D / 64 column blocks (each TK x 128 bytes in shared memory; a copy
                // instruction costs the producer the same time whatever its size).
                if constexpr (kPaged) {
                    // bpt boxes of box_rows rows, each inside one page (row offsets keep the
                    // 1024-byte swizzle atoms aligned: box_rows >= 16); page sizes are powers
                    // of two, so the row in the page is a mask.  A box shorter than the tile
                    // (bpt > 1) with several column blocks is copied block by block (4-D maps):
                    // a 5-D box would pack its blocks box_rows (not TK) rows apart.
                    for (int i = 0; i < bpt; ++i) {
                        const int e = lt * bpt + i;
                        if (!FAV_CHECK(e < Cfg::kPageSlots, status)) continue;
                        const int pid = page_list[e];
                        const int row = (key0 + i * box_rows) & (pg.page_size - 1);
                        if (Cfg::kBoxes == 1 || bpt == 1) {
                            fav::tma_load_5d(dst + i * box_rows * 128, tm, full, 0, row, 0, g, pid);
                        } else {
#pragma unroll
                            for (int bx = 0; bx < Cfg::kBoxes; ++bx)
                                fav::tma_load_4d(dst + bx * TK * 128 + i * box_rows * 128, tm, full,
                                                 bx * 64, row, g, pid);
                        }
                    }
                } else {
                    fav::tma_load_5d(dst, tm, full, 0, key0, 0, g, b);
                }
            }
        }
        return;
    }

    // ---------------- consumers ----------------
    const int r = lane >> 2, t = lane & 3;
    // The two MMA rows this thread holds: r and r + 8 of the block's 16-row chunk.
    int lim[2];        // keys visible to the row: [0, lim)
    const T *qrow[2];
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
        const int m = m0 + r + 8 * h2;
        if (m < M) {
            const int i = m / G, hh = m % G;
            qrow[h2] = q + b * qs.b + (long long)(g * G + hh) * qs.h + (long long)i * qs.n;
            lim[h2] = causal ? (Nkv - Nq + i + 1) : Nkv;
        } else {
            qrow[h2] = nullptr;
            lim[h2] = Nkv;
        }
    }
    int lim_min = min(lim[0], lim[1]);
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) lim_min = min(lim_min, __shfl_xor_sync(~0u, lim_min, off));

    uint32_t qa[D / 16][4];
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
        const int c = 16 * kk + 2 * t;
        const uint32_t *q0 = reinterpret_cast<const uint32_t *>(qrow[0]);
        const uint32_t *q1 = reinterpret_cast<const uint32_t *>(qrow[1]);
        qa[kk][0] = q0 ? __ldg(q0 + c / 2) : 0u;
        qa[kk][1] = q1 ? __ldg(q1 + c / 2) : 0u;
        qa[kk][2] = q0 ? __ldg(q0 + c / 2 + 4) : 0u;
        qa[kk][3] = q1 ? __ldg(q1 + c / 2 + 4) : 0u;
    }

    float acc[D / 8][4];
#pragma unroll
    for (int nd = 0; nd < D / 8; ++nd) acc[nd][0] = acc[nd][1] = acc[nd][2] = acc[nd][3] = 0.f;
    float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
    bool ok = true;

    for (int lt = warp; lt < my_tiles; lt += kConsumers) {
        const int st = lt % S;
        if (!fav::mbar_wait(full0 + 8 * st, (lt / S) & 1, status)) { ok = false; break; }
        const uint32_t kbase = ring_u32 + st * Cfg::kStageBytes;
        const uint32_t vbase = kbase + Cfg::kTileBytes;
        const int key0 = (tile0 + lt) * TK;

        // S = Q K^T over the tile: 8 n-tiles of 8 keys, fp32 accumulate.
        float s[TK / 8][4];
#pragma unroll
        for (int nt = 0; nt < TK / 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
        for (int kp = 0; kp < D / 32; ++kp) {
#pragma unroll
            for (int nt = 0; nt < TK / 8; ++nt) {
                uint32_t bfr[4] = {0u, 0u, 0u, 0u};
                const uint32_t la = kbase + swz<TK>(8 * nt + (lane & 7), 4 * kp + (lane >> 3));
                if (FAV_CHECK(la >= ring_u32 && la + 16 <= vbase && (la & 15u) == 0, status))
                    fav::ldmatrix_x4(bfr, la);
                fav::mma16816<T>(s[nt], qa[2 * kp], bfr[0], bfr[1]);
                fav::mma16816<T>(s[nt], qa[2 * kp + 1], bfr[2], bfr[3]);
            }
        }

        // Mask, scale into the log2 domain, online softmax.  (Paged: boxes whose block-table
        // entry was out of range, bad_boxes bit i for rows i * box_rows .. of the tile, are
        // masked as well.)
        uint32_t bad_boxes = 0;
        if constexpr (kPaged) {
            for (int i = 0; i < bpt; ++i)
                if (page_list[lt * bpt + i] < 0) bad_boxes |= 1u << i;
        }
        const bool need_mask = key0 + TK > lim_min || bad_boxes != 0;
        float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
        for (int nt = 0; nt < TK / 8; ++nt) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                float x = s[nt][e] * scale_log2;
                if (need_mask) {
                    const int j = key0 + 8 * nt + 2 * t + (e & 1);
                    if (j >= lim[e >> 1]) x = -INFINITY;
                    if (kPaged && ((bad_boxes >> ((j - key0) / box_rows)) & 1u)) x = -INFINITY;
                }
                s[nt][e] = x;
                mx[e >> 1] = fmaxf(mx[e >> 1], x);
            }
        }
        float alpha[2], mu[2];
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
            mx[h2] = fmaxf(mx[h2], __shfl_xor_sync(~0u, mx[h2], 1));
            mx[h2] = fmaxf(mx[h2], __shfl_xor_sync(~0u, mx[h2], 2));
            const float mn = fmaxf(mrow[h2], mx[h2]);
            mu[h2] = (mn == -INFINITY) ? 0.f : mn;
            alpha[h2] = fav::fast_exp2(mrow[h2] - mu[h2]);
            mrow[h2] = mn;
            lrow[h2] *= alpha[h2];
        }
#pragma unroll
        for (int nt = 0; nt < TK / 8; ++nt) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float p = fav::fast_exp2(s[nt][e] - mu[e >> 1]);
                s[nt][e] = p;
                lrow[e >> 1] += p;
            }
        }
#pragma unroll
        for (int nd = 0; nd < D / 8; ++nd) {
            acc[nd][0] *= alpha[0]; acc[nd][1] *= alpha[0];
            acc[nd][2] *= alpha[1]; acc[nd][3] *= alpha[1];
        }

        // O += P V: P (rounded to T) is the A operand straight from the S accumulators.
#pragma unroll
        for (int ks = 0; ks < TK / 16; ++ks) {
            uint32_t pa[4];
            pa[0] = fav::Elem<T>::pack(s[2 * ks][0], s[2 * ks][1]);
            pa[1] = fav::Elem<T>::pack(s[2 * ks][2], s[2 * ks][3]);
            pa[2] = fav::Elem<T>::pack(s[2 * ks + 1][0], s[2 * ks + 1][1]);
            pa[3] = fav::Elem<T>::pack(s[2 * ks + 1][2], s[2 * ks + 1][3]);
            const int i4 = lane >> 3;
            const int krow = 16 * ks + ((i4 & 1) << 3) + (lane & 7);
#pragma unroll
            for (int np = 0; np < D / 16; ++np) {
                uint32_t bfr[4] = {0u, 0u, 0u, 0u};
                const uint32_t la = vbase + swz<TK>(krow, 2 * np + (i4 >> 1));
                if (FAV_CHECK(la >= vbase && la + 16 <= ring_u32 + Cfg::kRingBytes && (la & 15u) == 0, status))
                    fav::ldmatrix_x4_trans(bfr, la);
                fav::mma16816<T>(acc[2 * np], pa, bfr[0], bfr[1]);
                fav::mma16816<T>(acc[2 * np + 1], pa, bfr[2], bfr[3]);
            }
        }
        __syncwarp();
        if (lane == 0) fav::mbar_arrive(empty0 + 8 * st);
    }

    // ---------------- merge the four warp states through shared memory ----------------
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
        lrow[h2] += __shfl_xor_sync(~0u, lrow[h2], 1);
        lrow[h2] += __shfl_xor_sync(~0u, lrow[h2], 2);
    }
    fav::named_bar_sync(1, kConsumers * 32);   // every consumer is done with the ring
    float *red = reinterpret_cast<float *>(ring);          // [warp][16][D]
    float *redm = red + kConsumers * 16 * D;                // [warp][16]
    float *redl = redm + kConsumers * 16;                   // [warp][16]
    float *mine = red + warp * 16 * D;
#pragma unroll
    for (int nd = 0; nd < D / 8; ++nd) {
        const int c = 8 * nd + 2 * t;
        *reinterpret_cast<float2 *>(mine + r * D + c) = make_float2(acc[nd][0], acc[nd][1]);
        *reinterpret_cast<float2 *>(mine + (r + 8) * D + c) = make_float2(acc[nd][2], acc[nd][3]);
    }
    if (t == 0) {
        redm[warp * 16 + r] = mrow[0];
        redm[warp * 16 + r + 8] = mrow[1];
        redl[warp * 16 + r] = lrow[0];
        redl[warp * 16 + r + 8] = lrow[1];
    }
    fav::named_bar_sync(1, kConsumers * 32);
    if (!ok) return;

    constexpr int kCols = D / 8;                 // columns per thread (8 threads per row)
    if (threadIdx.x >= 128) return;              // 16 rows x 8 threads merge the warps
    const int rr = threadIdx.x >> 3;             // 0..15
    const int c0 = (threadIdx.x & 7) * kCols;
    const int m = m0 + rr;
    if (m >= M) return;
    float mw[kConsumers], Mx = -INFINITY;
#pragma unroll
    for (int w = 0; w < kConsumers; ++w) {
        mw[w] = redm[w * 16 + rr];
        Mx = fmaxf(Mx, mw[w]);
    }
    float ew[kConsumers], L = 0.f;
#pragma unroll
    for (int w = 0; w < kConsumers; ++w) {
        ew[w] = (Mx == -INFINITY) ? 0.f : exp2f(mw[w] - Mx);
        L += ew[w] * redl[w * 16 + rr];
    }
    const float invL = (L > 0.f) ? 1.f / L : 0.f;
    float out[kCols];
#pragma unroll
    for (int c = 0; c < kCols; ++c) {
        float x = 0.f;
#pragma unroll
        for (int w = 0; w < kConsumers; ++w) x += ew[w] * red[(w * 16 + rr) * D + c0 + c];
        out[c] = x * invL;
    }
    const int i = m / G, hh = m % G;
    const long long flat = (long long)(b * Hq + g * G + hh) * Nq + i;
    const long long rows_total = (long long)gridDim.y * G * Nq;
    (void)rows_total;
    if (!FAV_CHECK(flat >= 0 && flat < rows_total && c0 + kCols <= D, status)) return;
    const float lse_val = (L > 0.f) ? (Mx + log2f(L)) * kLn2 : -INFINITY;
    if (splits == 1) {
        T *orow = o + b * os.b + (long long)(g * G + hh) * os.h + (long long)i * os.n + c0;
#pragma unroll
        for (int c = 0; c < kCols; c += 8) {
            uint4 pk;
            pk.x = fav::Elem<T>::pack(out[c + 0], out[c + 1]);
            pk.y = fav::Elem<T>::pack(out[c + 2], out[c + 3]);
            pk.z = fav::Elem<T>::pack(out[c + 4], out[c + 5]);
            pk.w = fav::Elem<T>::pack(out[c + 6], out[c + 7]);
            *reinterpret_cast<uint4 *>(orow + c) = pk;
        }
        if (lse && (threadIdx.x & 7) == 0) lse[flat] = lse_val;
    } else {
        float *prow = part_o + (flat * splits + split) * D + c0;
#pragma unroll
        for (int c = 0; c < kCols; c += 4)
            *reinterpret_cast<float4 *>(prow + c) = make_float4(out[c], out[c + 1], out[c + 2], out[c + 3]);
        if ((threadIdx.x & 7) == 0) part_lse[flat * splits + split] = lse_val;
    }
}

// One block per query row: L = logsumexp_s lse_s, O = sum_s exp(lse_s - L) O_s.  The four
// warps take every fourth split, each lane a group of D/32 consecutive columns (vector
// loads); the warp sums are added in shared memory.  Launched as a programmatic dependent of
// the decode kernel: it may be scheduled while the decode grid drains, and waits for that
// grid's completion (and memory) before reading the partials.
template <typename T, int D>
__global__ void __launch_bounds__(128)
fav_combine_kernel(const float *__restrict__ part_o, const float *__restrict__ part_lse,
                   T *__restrict__ o, FavStrides os, int Hq, int Nq, float *__restrict__ lse,
                   long long rows, int splits) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    __shared__ float red[4][D];
    __shared__ float wred[4];
    const long long row = blockIdx.x;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (row >= rows) return;
    const float *pl = part_lse + row * splits;
    // Each warp's first two splits of O are requested together with the LSE partials (one round
    // trip to L2 instead of two on the call's critical path).
    constexpr int kPer = D / 32;                  // consecutive columns per lane
    const float *po = part_o + row * splits * D + lane * kPer;
    float pre[2][kPer];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        const int sp = warp + 4 * r;
        if (sp < splits) {
            const float *src = po + (long long)sp * D;
            if constexpr (kPer == 4) {
                const float4 x = *reinterpret_cast<const float4 *>(src);
                pre[r][0] = x.x; pre[r][1] = x.y; pre[r][2] = x.z; pre[r][3] = x.w;
            } else {
                const float2 x = *reinterpret_cast<const float2 *>(src);
                pre[r][0] = x.x; pre[r][1] = x.y;
            }
        } else {
#pragma unroll
            for (int c = 0; c < kPer; ++c) pre[r][c] = 0.f;
        }
    }
    float mx = -INFINITY;
    for (int s = threadIdx.x; s < splits; s += 128) mx = fmaxf(mx, pl[s]);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(~0u, mx, off));
    if (lane == 0) wred[warp] = mx;
    __syncthreads();
    mx = fmaxf(fmaxf(wred[0], wred[1]), fmaxf(wred[2], wred[3]));
    __syncthreads();
    float sum = 0.f;
    for (int s = threadIdx.x; s < splits; s += 128)
        sum += (pl[s] == -INFINITY) ? 0.f : expf(pl[s] - mx);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(~0u, sum, off);
    if (lane == 0) wred[warp] = sum;
    __syncthreads();
    const float L = mx + logf(wred[0] + wred[1] + wred[2] + wred[3]);
    float acc[kPer];
#pragma unroll
    for (int c = 0; c < kPer; ++c) acc[c] = 0.f;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        const int sp = warp + 4 * r;
        if (sp < splits) {
            const float ls = pl[sp];
            const float w = (ls == -INFINITY) ? 0.f : expf(ls - L);
#pragma unroll
            for (int c = 0; c < kPer; ++c) acc[c] = fmaf(w, pre[r][c], acc[c]);
        }
    }
#pragma unroll 4
    for (int s = warp + 8; s < splits; s += 4) {
        const float ls = pl[s];
        const float w = (ls == -INFINITY) ? 0.f : expf(ls - L);
        const float *src = po + (long long)s * D;
        if constexpr (kPer == 4) {
            const float4 x = *reinterpret_cast<const float4 *>(src);
            acc[0] = fmaf(w, x.x, acc[0]);
            acc[1] = fmaf(w, x.y, acc[1]);
            acc[2] = fmaf(w, x.z, acc[2]);
            acc[3] = fmaf(w, x.w, acc[3]);
        } else {
            const float2 x = *reinterpret_cast<const float2 *>(src);
            acc[0] = fmaf(w, x.x, acc[0]);
            acc[1] = fmaf(w, x.y, acc[1]);
        }
    }
#pragma unroll
    for (int c = 0; c < kPer; ++c) red[warp][lane * kPer + c] = acc[c];
    __syncthreads();
    if (threadIdx.x < D / 2) {
        const int c = threadIdx.x * 2;
        const float x0 = red[0][c] + red[1][c] + red[2][c] + red[3][c];
        const float x1 = red[0][c + 1] + red[1][c + 1] + red[2][c + 1] + red[3][c + 1];
        const long long b = row / ((long long)Hq * Nq), h = (row / Nq) % Hq, i = row % Nq;
        *reinterpret_cast<uint32_t *>(o + b * os.b + h * os.h + i * os.n + c) =
            fav::Elem<T>::pack(x0, x1);
    }
    if (lse && threadIdx.x == 0) lse[row] = L;
}

// Shared by the dense and paged launches: the decode grid (splits, B * Hkv, 16-row chunks)
// and, with several splits, the combine kernel as a programmatic dependent launch.
template <typename T, int D, bool kPaged>
fav_status launch_grids(const FavArgs &a, const CUtensorMap &tmK, const CUtensorMap &tmV,
                        int n_tiles, int splits, void *workspace, cudaStream_t stream,
                        const FavPaged &pg, int box_rows) {
    using Cfg = DecodeCfg<D>;
    const int tps = (n_tiles + splits - 1) / splits;
    splits = (n_tiles + tps - 1) / tps;
    const int outer = a.B * a.Hkv;
    const int M = a.Nq * (a.Hq / a.Hkv);
    const int chunks = (M + 15) / 16;
    auto kern = fav_decode_kernel<T, D, kPaged>;
    constexpr int smem = kPaged ? Cfg::kSmemBytesPaged : Cfg::kSmemBytes;
    static bool attr_set = false;   // per-process; the attribute is per function, not per device
    if (!attr_set) {
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
            cudaSuccess)
            return FAV_ERR_CUDA;
        attr_set = true;
    }
    const long long rows = (long long)a.B * a.Hq * a.Nq;
    float *part_o = reinterpret_cast<float *>(workspace);
    float *part_lse = part_o ? part_o + rows * splits * D : nullptr;
    const float scale_log2 = a.scale * kLog2e;
    dim3 grid(splits, outer, chunks);
    kern<<<grid, kThreads, smem, stream>>>(
        tmK, tmV, (const T *)a.q, a.qs, (T *)a.o, a.os, a.lse, part_o, part_lse, a.Hq, a.Hkv,
        a.Nq, a.Nkv, n_tiles, tps, splits, scale_log2, a.causal, a.dev_status, pg, box_rows);
    if (cudaGetLastError() != cudaSuccess || fav_debug_sync("fav_decode_kernel", stream))
        return FAV_ERR_CUDA;
    if (splits > 1) {
        if (rows > 0x7fffffffLL) return FAV_ERR_UNSUPPORTED;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)rows);
        cfg.blockDim = dim3(128);
        cfg.dynamicSmemBytes = 0;
        cfg.stream = stream;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        T *out = (T *)a.o;
        float *lse_out = a.lse;
        cudaLaunchKernelEx(&cfg, fav_combine_kernel<T, D>, (const float *)part_o,
                           (const float *)part_lse, out, a.os, a.Hq, a.Nq, lse_out, rows, splits);
        if (cudaGetLastError() != cudaSuccess || fav_debug_sync("fav_combine_kernel", stream))
            return FAV_ERR_CUDA;
    }
    return FAV_OK;
}

template <typename T, int D>
fav_status launch(const FavArgs &a, int splits, void *workspace, cudaStream_t stream) {
    constexpr int TK = DecodeCfg<D>::TK;
    alignas(64) CUtensorMap tmK, tmV;
    fav_status st = fav_make_tmap_tiles(&tmK, a.k, D, a.Nkv, a.Hkv, a.B, a.ks, TK);
    if (st != FAV_OK) return st;
    st = fav_make_tmap_tiles(&tmV, a.v, D, a.Nkv, a.Hkv, a.B, a.vs, TK);
    if (st != FAV_OK) return st;
    const FavPaged none{nullptr, nullptr, 0, 0, 0};
    return launch_grids<T, D, false>(a, tmK, tmV, fav_decode_num_tiles(a), splits, workspace,
                                     stream, none, TK);
}

// Paged cache: the pools viewed as [num_pages][page_size][Hkv][D] -- a 4-D tensor (D,
// page_size, Hkv, num_pages) with boxes of min(page_size, TK) rows of one head of one page.
template <typename T, int D>
fav_status launch_paged(const FavArgs &a, const FavPaged &pg, int splits, void *workspace,
                        cudaStream_t stream) {
    constexpr int TK = DecodeCfg<D>::TK;
    const int box_rows = std::min(pg.page_size, TK);
    const FavStrides ps{(long long)pg.page_size * a.Hkv * D, (long long)D, (long long)a.Hkv * D};
    alignas(64) CUtensorMap tmK, tmV;
    // one 5-D box per page piece when it spans the whole tile or D has one column block; 4-D
    // per-block boxes otherwise (the kernel makes the same choice)
    const bool tiles5 = (D == 64) || (box_rows == TK);
    auto make = [&](CUtensorMap *m, const void *base) {
        return tiles5 ? fav_make_tmap_tiles(m, base, D, pg.page_size, a.Hkv, pg.num_pages, ps, box_rows)
                      : fav_make_tmap_4d(m, base, D, pg.page_size, a.Hkv, pg.num_pages, ps, box_rows);
    };
    fav_status st = make(&tmK, a.k);
    if (st != FAV_OK) return st;
    st = make(&tmV, a.v);
    if (st != FAV_OK) return st;
    return launch_grids<T, D, true>(a, tmK, tmV, fav_decode_num_tiles(a), splits, workspace,
                                    stream, pg, box_rows);
}

}  // namespace

bool fav_decode_supported(const FavArgs &a) {
    if (a.dtype != FAV_F16 && a.dtype != FAV_BF16) return false;
    if (a.D != 64 && a.D != 128) return false;
    const long long M = (long long)a.Nq * (a.Hq / a.Hkv);
    return M <= 64 && (long long)a.B * a.Hkv <= 65535;
}

int fav_decode_num_tiles(const FavArgs &a) {
    const int tk = (a.D == 128) ? DecodeCfg<128>::TK : DecodeCfg<64>::TK;
    return (a.Nkv + tk - 1) / tk;
}

// Split count: a single wave of blocks covering ~90% of the SMs.  A block streams its whole
// key range through the ring, and ~0.9 x SMs streaming blocks already saturate HBM, while
// every extra block (a second wave, or a partly filled one) adds a ring fill and a final merge
// to the critical path; measured on the decode workloads, one wave of ~128-144 blocks beat
// three waves by 10-15%.  Each block keeps at least two tiles per ring stage.
int fav_decode_auto_splits(const FavArgs &a) {
    const int n_tiles = fav_decode_num_tiles(a);
    const long long M = (long long)a.Nq * (a.Hq / a.Hkv);
    const long long groups = (long long)a.B * a.Hkv * ((M + 15) / 16);
    const long long sms = a.num_sms > 0 ? a.num_sms : 148;
    long long splits = (9 * sms) / (10 * groups);
    const int min_tiles = 2 * DecodeCfg<128>::kStages;
    splits = std::min<long long>(splits, std::max(1, n_tiles / min_tiles));
    splits = std::max<long long>(1, std::min<long long>(splits, 4096));
    return (int)splits;
}

size_t fav_decode_workspace_bytes(const FavArgs &a, int splits) {
    if (splits <= 1) return 0;
    const size_t rows = (size_t)a.B * a.Hq * a.Nq;
    return rows * splits * ((size_t)a.D + 1) * sizeof(float);
}

int fav_decode_tile_keys(int D) { return D == 128 ? DecodeCfg<128>::TK : DecodeCfg<64>::TK; }
int fav_decode_page_slots() { return DecodeCfg<128>::kPageSlots; }

fav_status fav_launch_decode_paged(const FavArgs &a, const FavPaged &pg, int splits,
                                   void *workspace, cudaStream_t s) {
    if (a.dtype == FAV_F16)
        return a.D == 128 ? launch_paged<__half, 128>(a, pg, splits, workspace, s)
                          : launch_paged<__half, 64>(a, pg, splits, workspace, s);
    return a.D == 128 ? launch_paged<__nv_bfloat16, 128>(a, pg, splits, workspace, s)
                      : launch_paged<__nv_bfloat16, 64>(a, pg, splits, workspace, s);
}

fav_status fav_launch_decode(const FavArgs &a, int splits, void *workspace, cudaStream_t s) {
    if (a.dtype == FAV_F16)
        return a.D == 128 ? launch<__half, 128>(a, splits, workspace, s)
                          : launch<__half, 64>(a, splits, workspace, s);
    return a.D == 128 ? launch<__nv_bfloat16, 128>(a, splits, workspace, s)
                      : launch<__nv_bfloat16, 64>(a, splits, workspace, s);
}
