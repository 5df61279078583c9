// fav_prefill.cu -- prefill attention for D = 128 on the 5th-generation tensor cores
// (tcgen05 + TMEM + TMA): one query tile per unit of work, the softmax split over the keys.
//
// Method (paper, Algorithm "FlashAttention-V for VL > D" and its description): the query
// rows of a block stay on chip for the whole sweep over key/value blocks; for every key block
// the scores are computed, the running maximum / sum / output accumulator of the online
// softmax are updated (rescale by exp(M_old - M), weights exp(S - M)), and after the last
// block the accumulator is normalised.  Heads sharing a K/V head read the same K/V tiles
// (GQA reuse: neighbouring CTAs work on the heads of one group at the same time, so the tiles
// come from L2).  On this GPU that becomes:
//   * a unit is one 128-row query tile; the kernel is persistent (one CTA per SM at most) and
//     CTA c works through units c, 2P-1-c, 2P+c, ... of the units sorted by decreasing causal
//     work within blocks of heads whose K/V fit in L2, with the next unit's Q tile loaded
//     (TMA, 128-byte swizzle) into a second buffer;
//   * 128-key K and V tiles are streamed by TMA (one copy instruction per tile) through rings
//     of shared-memory stages;
//   * S = Q K^T (M = 128, N = 128, K = 128) goes to one of two TMEM score buffers, so the
//     tensor core computes the scores of key tile j+1 while the softmax works on tile j;
//   * the softmax of a tile is split over the keys: split s (of two) owns keys
//     [64 s, 64 s + 64) of every tile and keeps its own running maximum, sum and output
//     accumulator O_s (128 TMEM columns) -- the online softmax applied to each key subset
//     separately, as in the split-KV decode.  O_s += P_s V_s is a burst of tcgen05.mma with
//     the weights P_s read from TMEM.  The splits are merged once per unit:
//     O = sum_s 2^(m_s - M) O_s / sum_s 2^(m_s - M) l_s, M = max_s m_s.
//     The point of the split: a tile's softmax runs on eight warps (two per scheduler) with no
//     exchange between them, and takes about as long as the tile's MMAs.
//   * an epilogue warpgroup merges the splits once the unit's last P.V has completed, writes
//     the O tile into the unit's (by then free) Q buffer, and one TMA tensor store writes it
//     out; the softmax warps go on with the next unit meanwhile, and the next unit's first P.V
//     (which overwrites O_0 and O_1) waits only until the epilogue has read them.
// TMEM (512 columns): score buffers 0 | 1 (128 columns each; the fp16 weights of split s
// overwrite the first half of its own score columns), then O_0 | O_1.
// The running maximum is updated lazily: O_s and l_s are rescaled only when the maximum grows
// by more than 2^4 (log2 domain); the weights are stored as p * 2^11 (below 2^15, inside
// fp16's range).  O_s / l_s keeps the same maximum as its weights, so the result is unchanged.
//
// Warp roles (512 threads, four warpgroups with their own register budgets, setmaxnreg):
// warps 0-7 softmax (TMEM lane quarter = warp % 4, key split = warp / 4; one thread per query
// row and split; 176 registers); warp 8 = TMEM owner + MMA issuer (the whole warp, one elected
// lane issuing each burst and committing the barrier arrivals inside the same asm block);
// warp 9 = Q/K producer, warp 10 = V producer (two issuing warps keep more TMA copies in
// flight than one); warp 11 = O stores (warps 8-11: 56 registers); warps 12-15 = epilogue (one
// thread per query row; 96 registers).
//
// Issue order of the tensor core, per CTA over the global sequence G of key tiles (all units):
//   S(0), S(1), P(0).V, S(2), P(1).V, S(3), ...    S(G) into score buffer G % 2
// S(G + 2) overwrites the weights of tile G, so it follows P(G).V in the same (in-order) pipe.
// (For D = 64 the two-tile kernel of fav_prefill_pair.cu is faster: its products are short
// and two query tiles sharing each K/V tile keep the softmax warps busier.)
#include <cuda.h>
#include <math.h>

#include <algorithm>
#include <type_traits>

#include "fav_device.cuh"
#include "fav_internal.h"
#include "fav_tc.cuh"

namespace {

constexpr int BM = 128;          // query rows per tile (= TMEM lanes)
constexpr int BN = 128;          // keys per tile
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kRescaleThreshold = 4.0f;   // log2 units: rescale when max grows by > 2^4
// The weights are stored as p * 2^kPShift (exponent reference m - kPShift): with the lazy
// threshold they stay below 2^(4 + kPShift) = 2^15, inside fp16's range, and weights down to
// 2^-25 of the reference stay fp16 normals.  O / l is unchanged (l carries the same factor);
// the LSE subtracts kPShift.
constexpr float kPShift = 11.0f;

// Calls f(std::integral_constant-like index) for kI = 0 .. kN-1, each a compile-time constant.
template <int kI, int kN, typename F>
__device__ __forceinline__ void static_for(F &&f) {
    if constexpr (kI < kN) {
        f(std::integral_constant<int, kI>{});
        static_for<kI + 1, kN>(f);
    }
}

template <typename T> struct IsBF16 { static constexpr bool value = false; };
template <> struct IsBF16<__nv_bfloat16> { static constexpr bool value = true; };

// Precision of the weights P in the P.V MMA.  A single bf16 P (8 significant bits) can move O
// by up to 2^-9 of |v| when a few weights dominate (any reference maximum, lazy or not, leaves
// most of them inexact), which with the bf16 rounding of O itself does not fit a 3e-3 error
// budget.  So P is fp16 (11 bits, one MMA per k-step) for both I/O types: for bf16 I/O, V is
// converted to fp16 first (fav_v16_kernel).  With the weights stored as p * 2^kPShift, fp16
// weights down to 2^-25 of the reference are normal numbers; smaller ones err by at most
// 2^-36 of it, which stays below the tolerance even next to a value of V 2^25 times larger
// than the others.

template <int D> struct PrefillCfg {
    static_assert(D == 128, "the key-split kernel serves D = 128");
    static constexpr int kSplits = 2;                        // key splits per tile
    static constexpr int kSplitKeys = BN / kSplits;          // keys per split and tile
    static constexpr int kSoftWarps = 4 * kSplits;
    static constexpr int kMmaWarp = kSoftWarps;
    static constexpr int kLoadKWarp = kSoftWarps + 1;        // Q and K
    static constexpr int kLoadVWarp = kSoftWarps + 2;
    static constexpr int kStoreWarp = kSoftWarps + 3;        // O tiles (TMA store)
    static constexpr int kEpiWarp0 = kSoftWarps + 4;         // epilogue warpgroup (4 warps)
    static constexpr int kThreads = 32 * (kSoftWarps + 8);
    // Register budgets per warpgroup (setmaxnreg; launched with 65536 / kThreads = 128 each):
    // softmax 176, MMA / producers / store 56, epilogue 96.  Sum 2*128*176 + 128*56 + 128*96 =
    // 64512 <= 65536, and per scheduler (one warp of each warpgroup) 32 * 504 <= 16384.
    static constexpr int kRegSoftmax = 176, kRegIssue = 56, kRegEpi = 96;
    static constexpr int kRegLaunch = 65536 / kThreads;       // every warpgroup at the join
    static_assert(2 * 128 * kRegSoftmax + 128 * kRegIssue + 128 * kRegEpi <= 65536, "registers");
    static constexpr int kKStages = 2;                       // K ring depth
    static constexpr int kVStages = 2;                       // V ring depth
    static constexpr int kQBytes = BM * D * 2;               // one Q tile (or one O tile)
    static constexpr int kKVBytes = BN * D * 2;              // one K or V tile
    static constexpr int kUnitTab = 256;                     // units precomputed per CTA
    // L2 prefetch distance in key tiles: dense calls 2, packed batches 4 (measured: the
    // headline 36.4 -> 35.4 us with 2, dense batches and long sequences equal or faster; packed
    // batches of short prompts 2 % slower with 2)
    static constexpr int kPrefetchDense = 2, kPrefetchVarlen = 4;
    // shared-memory map (offsets from the 1024-aligned base)
    static constexpr int kOffQ = 0;                          // Q buffers 0, 1 (O staging)
    static constexpr int kOffK = kOffQ + 2 * kQBytes;
    static constexpr int kOffV = kOffK + kKStages * kKVBytes;
    static constexpr int kOffXch = kOffV + kVStages * kKVBytes;   // (m, l) [2][4][splits][32]
    static constexpr int kXchBytes = 2 * 4 * kSplits * 32 * 8;
    static constexpr int kOffUnits = kOffXch + kXchBytes;         // int[kUnitTab][12]
    static constexpr int kOffBar = kOffUnits + kUnitTab * 48;
    static constexpr int kNumBars = 2 + 2 + 2 * kKStages + 2 * kVStages + 2 + 2 + 2 + 2 + 2 + 1 + 2;
    static constexpr int kOffTmemSlot = kOffBar + kNumBars * 8;
    static constexpr int kOffDbg = kOffTmemSlot + 16;             // debug builds: per-role totals
    static constexpr int kSmemBytes = kOffDbg + 32 + 1024;
    static constexpr uint32_t kTmemCols = 512;
    static __host__ __device__ constexpr uint32_t colS(int buf) { return buf ? 128u : 0u; }
    static constexpr uint32_t kColO = 256;                   // O_s at kColO + s * D
    static_assert(256 + kSplits * D == 512, "TMEM budget");
    static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
};

// bf16 I/O (kV16): Q, K and O are bf16; V has been converted to fp16 (tmV, scaled per KV head
// by v_scale^-1, a power of two) so that P.V runs with fp16 weights, and the epilogue multiplies
// O back by v_scale.  fp16 I/O: tmV is V itself.
// kVarlen: the units come from the packed variable-length table `vunits` (the dense kernel
// compiles without any of the per-sequence offsets, lengths and partial-tile stores).
template <typename T, int D, bool kV16, bool kVarlen>
__global__ void __launch_bounds__(PrefillCfg<D>::kThreads, 1)
fav_prefill_split_kernel(const __grid_constant__ CUtensorMap tmQ,
                         const __grid_constant__ CUtensorMap tmK,
                         const __grid_constant__ CUtensorMap tmV,
                         const __grid_constant__ CUtensorMap tmO, T *__restrict__ o,
                         FavStrides os, float *__restrict__ lse,
                         const float *__restrict__ v_scale, int B, int Hq, int Hkv, int Nq,
                         int Nkv, int n_qtiles, int head_block, float scale_log2, int causal,
                         int *status, const int4 *__restrict__ vunits, int n_vunits) {
    using C = PrefillCfg<D>;
    using TP = __half;    // type of the weights P and of V in shared memory (P.V MMA)
    constexpr int KS = C::kKStages, VS = C::kVStages, NS = C::kSplits, SK = C::kSplitKeys;
    extern __shared__ uint8_t smem_raw[];
    // 1024-byte alignment in the shared window (the 128-byte swizzle atom of TMA and MMA)
    const uint32_t raw_u32 = fav::smem_u32(smem_raw);
    uint8_t *smem = smem_raw + ((1024u - (raw_u32 & 1023u)) & 1023u);
    const uint32_t sbase = fav::smem_u32(smem);
    const uint32_t sQ = sbase + C::kOffQ, sK = sbase + C::kOffK, sV = sbase + C::kOffV;
    const uint32_t bar0 = sbase + C::kOffBar;
    const uint32_t q_full = bar0;                 // [2] per Q buffer
    const uint32_t q_empty = q_full + 16;         // [2] the buffer's last S read (and O stored)
    const uint32_t k_full = q_empty + 16, k_empty = k_full + 8 * KS;
    const uint32_t v_full = k_empty + 8 * KS, v_empty = v_full + 8 * VS;
    const uint32_t s_full = v_empty + 8 * VS;     // [2] per score buffer
    const uint32_t p_full = s_full + 16;          // [2] per score buffer (weights stored)
    const uint32_t pv_done = p_full + 16;         // P(G).V completed, once per key tile
    const uint32_t o_done = pv_done + 8;          // a unit's last P.V completed, once per unit
    const uint32_t xch_bar = o_done + 8;          // [2] (m, l) of every row and split written
    const uint32_t o_staged = xch_bar + 16;       // [2] O tile written into Q buffer k % 2
    const uint32_t o_free = o_staged + 16;        // the epilogue has read the unit's O
    const uint32_t xch_free = o_free + 8;         // [2] the epilogue has read (m, l) slot k % 2
    float2 *xch = reinterpret_cast<float2 *>(smem + C::kOffXch);
    int *utab = reinterpret_cast<int *>(smem + C::kOffUnits);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + C::kOffTmemSlot);
#ifdef FAV_DEBUG_CHECKS
    // per role, what it processed: softmax key tiles, K tiles loaded, V tiles loaded, P.V
    // products, S products, epilogue units, stored units
    int *dbg_tot = reinterpret_cast<int *>(smem + C::kOffDbg);
#endif

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int G = Hq / Hkv;
    const int off = Nkv - Nq;                                   // bottom-right causal offset
    const int BH = B * Hq;

    // ---- work units: one query tile each, heaviest causal first ----
    // The B * Hq heads are taken in blocks of head_block heads (a multiple of the GQA group,
    // chosen on the host so that a block's K and V fit in about half the L2); within a block,
    // unit u is query tile t = n_qtiles - 1 - u / hb of head (b, h) = block start + u % hb
    // (hb = the block's head count), so the heads of one GQA group (consecutive h) run side by
    // side and a block's K/V tiles stay in L2 while all of its query tiles pass.  The CTA
    // takes units c, 2P-1-c, 2P+c, 4P-1-c, ... (P CTAs, "snake" order), which evens out the
    // work per CTA.
    // Variable-length batches (kVarlen): the units come from a table built on the host
    // (sorted the same way), Q/O are [1, Hq, total_q, D] and K/V [1, Hkv, total_k, D] views of
    // the packed tensors, and a unit's rows start at its sequence's offsets q_y0 / k_y0.
    // Unit: TMA batch coordinate b, head h, query tile t of its sequence, key tiles n_kv, KV head
    // kvh, sequence offsets and lengths.
    struct Unit {
        int b, h, t, n_kv, kvh, q_y0, k_y0, len_q, len_k;
    };
    constexpr bool varlen = kVarlen;
    constexpr int kPrefetch = kVarlen ? C::kPrefetchVarlen : C::kPrefetchDense;
    constexpr int kUnitInts = kVarlen ? 12 : 8;                 // ints per unit-table entry
    const int n_units = varlen ? n_vunits : n_qtiles * BH;
    auto unit_at = [&](int k) {   // the k-th unit of this CTA, or -1
        const int P = gridDim.x, c = blockIdx.x;
        const int u = k * P + ((k & 1) ? (P - 1 - c) : c);
        return u < n_units ? u : -1;
    };
    auto make_unit = [&](int u) {
        Unit U;
        if constexpr (varlen) {
            const int4 a = vunits[2 * u], c = vunits[2 * u + 1];
            U.b = 0;
            U.h = a.y;
            U.t = a.z;
            U.n_kv = a.w;
            U.q_y0 = c.x;
            U.k_y0 = c.y;
            U.len_q = c.z;
            U.len_k = c.w;
        } else {
            const int bh = u % BH;
            U.t = n_qtiles - 1 - u / BH;
            U.b = bh / Hq;
            U.h = bh % Hq;
            U.q_y0 = U.k_y0 = 0;
            U.len_q = Nq;
            U.len_k = Nkv;
            const int kv_end = causal ? min(Nkv, U.t * BM + BM + off) : Nkv;
            U.n_kv = (kv_end + BN - 1) / BN;
        }
        U.kvh = U.h / G;
        return U;
    };
    // With several head blocks (head_block < B * Hq; the host allows that only when every unit
    // of a CTA fits the table below) unit u maps to the blocked order instead.
    auto make_unit_blocked = [&](int u) {
        if (varlen || head_block >= BH) return make_unit(u);
        const int blk_units = n_qtiles * head_block;
        const int blk = u / blk_units;
        const int ul = u - blk * blk_units;
        const int hb = min(head_block, BH - blk * head_block);
        // the unit that the one-block order numbers (ul / hb) * BH + (head of this unit)
        return make_unit((ul / hb) * BH + blk * head_block + ul % hb);
    };
    // The CTA's first kUnitTab units are computed once, in parallel, into shared memory (the
    // integer divisions would otherwise sit on the critical path at every unit switch); every
    // entry is written (a unit past the CTA's last one has no key tiles).  Units beyond the
    // table are computed where they are needed: the host chooses the blocked order only when
    // every unit of every CTA fits the table, so past it the plain order (make_unit) is the
    // order the table would have held.
    auto unit = [&](int k) {
        if (k < C::kUnitTab) {
            const int *e = utab + kUnitInts * k;
            Unit U;
            U.b = e[0]; U.h = e[1]; U.t = e[2]; U.n_kv = e[3]; U.kvh = e[4];
            if constexpr (varlen) {
                U.q_y0 = e[5]; U.k_y0 = e[6]; U.len_q = e[7]; U.len_k = e[8];
            } else {
                U.q_y0 = U.k_y0 = 0;
                U.len_q = Nq;
                U.len_k = Nkv;
            }
            return U;
        }
        return make_unit(unit_at(k));
    };
    // Key tiles of the CTA's unit k (k must be one of its units).
    auto unit_nkv = [&](int k) -> int {
        return k < C::kUnitTab ? utab[kUnitInts * k + 3] : make_unit(unit_at(k)).n_kv;
    };
    // Position in the CTA's sequence of key tiles, for the L2 prefetches that run ahead of the
    // loads (it steers prefetches only; the loads follow the unit table): unit index k (-1 past
    // the end), key tile j of that unit.
    struct TileIt {
        int k, j;
        Unit U;
    };
    auto tile_next = [&](TileIt &it) {
        if (it.k < 0) return;
        if (++it.j == it.U.n_kv) {
            it.j = 0;
            ++it.k;
            if (unit_at(it.k) >= 0) it.U = unit(it.k);
            else it.k = -1;
        }
    };
    // L2 prefetch of the key tile at `it` (K or V, by the tensor map), then step `it` on
    auto prefetch_next = [&](const CUtensorMap *tm, TileIt &it) {
        if (it.k >= 0) fav::tma_prefetch_l2_5d(tm, 0, it.U.k_y0 + it.j * BN, 0, it.U.kvh, it.U.b);
        tile_next(it);
    };
    if (warp == C::kLoadKWarp && lane == 0) {
        (void)FAV_CHECK((sbase & 1023u) == 0, status);
        (void)FAV_CHECK((sbase - raw_u32) + C::kOffTmemSlot + 4 <= fav::dynamic_smem_bytes(), status);
        for (int i = 0; i < 2; ++i) {
            fav::mbar_init(q_full + 8 * i, 1);
            // last S commit, + the O store's read of the buffer when O is staged there
            fav::mbar_init(q_empty + 8 * i, varlen ? 1 : 2);
            fav::mbar_init(xch_free + 8 * i, 128);          // epilogue threads
            fav::mbar_init(o_staged + 8 * i, 128);          // epilogue threads
            fav::mbar_init(xch_bar + 8 * i, C::kSoftWarps * 32);
            fav::mbar_init(s_full + 8 * i, 1);
            fav::mbar_init(p_full + 8 * i, C::kSoftWarps);
        }
        for (int s = 0; s < KS; ++s) {
            fav::mbar_init(k_full + 8 * s, 1);
            fav::mbar_init(k_empty + 8 * s, 1);
        }
        for (int s = 0; s < VS; ++s) {
            fav::mbar_init(v_full + 8 * s, 1);
            fav::mbar_init(v_empty + 8 * s, 1);
        }
        fav::mbar_init(pv_done, 1);
        fav::mbar_init(o_done, 1);
        fav::mbar_init(o_free, 128);
        fav::mbar_fence_init();
        // The first Q and K tiles are requested before the rest of the set-up (unit table,
        // TMEM allocation): they come from HBM and bound the time to the first scores.
        fav::tma_prefetch_desc(&tmQ);
        fav::tma_prefetch_desc(&tmK);
        const Unit U0 = make_unit_blocked(unit_at(0));
        fav::mbar_arrive_expect_tx(q_full, C::kQBytes);
        fav::tma_load_5d(sQ, &tmQ, q_full, 0, U0.q_y0 + U0.t * BM, 0, U0.h, U0.b);
        for (int g = 0; g < KS && g < U0.n_kv; ++g) {
            fav::mbar_arrive_expect_tx(k_full + 8 * g, C::kKVBytes);
            fav::tma_load_5d(sK + g * C::kKVBytes, &tmK, k_full + 8 * g, 0, U0.k_y0 + g * BN, 0, U0.kvh, U0.b);
        }
    }
    for (int k = threadIdx.x; k < C::kUnitTab; k += blockDim.x) {
        const int u = unit_at(k);
        int *e = utab + kUnitInts * k;
        if (u < 0) {
#pragma unroll
            for (int i = 0; i < kUnitInts; ++i) e[i] = 0;
            continue;
        }
        const Unit U = make_unit_blocked(u);
        e[0] = U.b; e[1] = U.h; e[2] = U.t; e[3] = U.n_kv; e[4] = U.kvh;
        if constexpr (varlen) {
            e[5] = U.q_y0; e[6] = U.k_y0; e[7] = U.len_q; e[8] = U.len_k;
        }
    }

    if (warp == C::kMmaWarp) {
        fav::tc::tmem_alloc(fav::smem_u32(tmem_slot), C::kTmemCols);
        fav::tc::tmem_relinquish();
    }
    fav::tc::fence_before();
    __syncthreads();
    fav::tc::fence_after();
    const uint32_t tmem = *tmem_slot;
    (void)FAV_CHECK((tmem & 0xFFFFu) + C::kTmemCols <= 512u && (tmem >> 16) == 0u, status);

    // Barrier phases run on across units: key tile G of the CTA's sequence uses K stage G % KS
    // (parity (G / KS) & 1), V stage G % VS, score buffer G % 2 (s_full / p_full parity
    // (G / 2) & 1) and completes pv_done phase G; unit k uses Q buffer k % 2 (parity
    // (k / 2) & 1) and exchange slot k % 2, and completes o_done phase k.
    // Roles by warpgroup; each branch opens with its register budget (setmaxnreg).
    if (warp < C::kSoftWarps) {
        fav::setmaxnreg_inc<C::kRegSoftmax>();
        // ---------------- softmax / correction: one thread per query row and split ----------------
        const int quarter = warp & 3, split = warp >> 2;
        const int row = quarter * 32 + lane;
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
        const uint32_t colO = C::kColO + split * D;
        int Gt = 0;                // key tiles consumed so far (the CTA's sequence)
        bool ok = true;
        for (int k = 0, u; ok && (u = unit_at(k)) >= 0; ++k) {
            const Unit U = unit(k);
            const int q0 = U.t * BM;
            const int qi = q0 + row;                          // query index of this row
            const int uoff = U.len_k - U.len_q;               // bottom-right causal offset
            const int lim = causal ? min(U.len_k, qi + uoff + 1) : U.len_k;      // visible keys: [0, lim)
            const int lim_tile = causal ? min(U.len_k, q0 + uoff + 1) : U.len_k; // smallest lim in the tile
            float m = -INFINITY, l = 0.f;
            for (int j = 0; j < U.n_kv; ++j, ++Gt) {
                if (!__all_sync(~0u, fav::mbar_wait_il(s_full + 8 * (Gt & 1), (Gt >> 1) & 1, status))) {
                    ok = false;
                    break;
                }
                fav::tc::fence_after();
                const uint32_t colS = C::colS(Gt & 1) + split * SK;
                const int key0 = j * BN + split * SK;
                const bool crosses = key0 + SK > lim_tile;   // the split crosses the diagonal or the end
                float s[SK];
                // scores of this split from TMEM (and the mask: keys at or beyond lim get -inf)
                {
                    static_assert(SK == 64, "one 64-column load per split");
                    uint32_t r[SK];
                    fav::tc::ld_32x32b_x64(trow + colS, r);
                    fav::tc::wait_ld_dep(r);
#pragma unroll
                    for (int c = 0; c < SK; ++c) s[c] = __uint_as_float(r[c]);
                    if (crosses) {
                        const int nvis = lim - key0;              // keys [0, nvis) of the split visible
#pragma unroll
                        for (int c = 0; c < SK; ++c)
                            if (c >= nvis) s[c] = -INFINITY;
                    }
                }
                // raw maximum of the split: 8 independent chains of 3-input max, then a tree
                float mx;
                {
                    float m8[8];
#pragma unroll
                    for (int c = 0; c < 8; ++c) m8[c] = s[c];
#pragma unroll
                    for (int c = 8; c < SK; c += 16) {
#pragma unroll
                        for (int q = 0; q < 8; ++q)
                            m8[q] = (c + 8 < SK) ? fav::fmax3(m8[q], s[c + q], s[c + 8 + q])
                                                 : fmaxf(m8[q], s[c + q]);
                    }
                    mx = fav::fmax3(fav::fmax3(m8[0], m8[1], m8[2]), fav::fmax3(m8[3], m8[4], m8[5]),
                                    fmaxf(m8[6], m8[7])) * scale_log2;
                }
                // lazy rescale: move the reference maximum only when it grows by > 2^4
                float alpha = 1.f;
                bool rescale = false;
                if (mx > m + kRescaleThreshold) {
                    alpha = fav::fast_exp2(m - mx);   // 0 while m = -inf
                    rescale = (j > 0);
                    m = mx;
                    l *= alpha;
                }
                // weights p = exp2(s * scale_log2 - mref) on pairs (one packed FMA, two ex2, one
                // packed add), stored as fp16 over the split's first SK / 2 score columns (read
                // above); a split with no visible key so far (m = -inf) stores zeros.
                {
                    const float mref = (m == -INFINITY) ? 0.f : m - kPShift;
                    const float2 sc2 = make_float2(scale_log2, scale_log2);
                    const float2 nm2 = make_float2(-mref, -mref);
                    float2 l4[4] = {{0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}};
                    uint32_t pk[SK / 2];
                    static_for<0, SK / 2>([&](auto pc) {
                        constexpr int e = decltype(pc)::value;
                        const float2 x = fav::ffma2(make_float2(s[2 * e], s[2 * e + 1]), sc2, nm2);
                        const float2 p = make_float2(fav::fast_exp2(x.x), fav::fast_exp2(x.y));
                        l4[e & 3] = fav::fadd2(l4[e & 3], p);
                        pk[e] = fav::Elem<TP>::pack(p.x, p.y);
                    });
                    fav::tc::st_32x32b_x32(trow + colS, pk);
                    const float2 a = fav::fadd2(fav::fadd2(l4[0], l4[1]), fav::fadd2(l4[2], l4[3]));
                    l += a.x + a.y;
                }
                // O_s *= alpha, once P(G-1).V (the last product into O_s) has completed.  S(G)
                // was issued after P(G-2).V and has completed, so pv_done has completed phase
                // G-2 and cannot have completed G (that needs these weights): the parity of phase
                // G-1 is unambiguous.
                if (__any_sync(~0u, rescale)) {
                    if (!__all_sync(~0u, fav::mbar_wait_il(pv_done, (Gt - 1) & 1, status))) {
                        ok = false;
                        break;
                    }
                    fav::tc::fence_after();
#pragma unroll
                    for (int c = 0; c < D / 32; ++c) {
                        const uint32_t col = colO + c * 32;
                        uint32_t v[32];
                        fav::tc::ld_32x32b_x32(trow + col, v);
                        fav::tc::wait_ld_dep(v);
#pragma unroll
                        for (int e = 0; e < 32; e += 2) {
                            const float2 y = fav::fmul2(make_float2(__uint_as_float(v[e]), __uint_as_float(v[e + 1])),
                                                        make_float2(alpha, alpha));
                            v[e] = __float_as_uint(y.x);
                            v[e + 1] = __float_as_uint(y.y);
                        }
                        fav::tc::st_32x32b_x32(trow + col, v);
                    }
                }
                fav::tc::wait_st();
                fav::tc::fence_before();
                __syncwarp();
                if (lane == 0) fav::mbar_arrive(p_full + 8 * (Gt & 1));
            }
            if (!ok) break;
            // (m, l) of this row and split for the epilogue warpgroup (slot k % 2).  Packed
            // batches release a Q buffer with its unit's last S (O is not staged there), so unit
            // k + 2 can reach this point before the epilogue has read unit k's slot: wait for it.
            if constexpr (varlen) {
                if (k >= 2 && !__all_sync(~0u, fav::mbar_wait_il(xch_free + 8 * (k & 1),
                                                                ((k >> 1) - 1) & 1, status)))
                    break;
            }
            xch[((((k & 1) * 4 + quarter) * NS) + split) * 32 + lane] = make_float2(m, l);
            fav::mbar_arrive(xch_bar + 8 * (k & 1));
        }
#ifdef FAV_DEBUG_CHECKS
        if (threadIdx.x == 0) dbg_tot[0] = Gt;
#endif
        fav::setmaxnreg_dec<C::kRegLaunch>();      // back to the launch budget for the join
    } else if (warp >= C::kEpiWarp0) {
        fav::setmaxnreg_dec<C::kRegEpi>();
        // ---------------- epilogue: merge the splits, O / L, LSE; one thread per query row ----------------
        // O = (2^(m_0 - M) O_0 + 2^(m_1 - M) O_1) / L, L = 2^(m_0 - M) l_0 + 2^(m_1 - M) l_1,
        // M = max(m_0, m_1).  The O tile goes, rounded to the I/O type, into the unit's Q buffer
        // (free: the unit's S products have completed) in the TMA box layout (rows of 128 bytes,
        // 16-byte chunks XOR-swizzled by row % 8); the store warp writes it out with one TMA
        // store (rows beyond Nq are not written).  As soon as O has been read, the next unit's
        // first P.V (which overwrites O_0 and O_1) may run.
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
        for (int k = 0, u; (u = unit_at(k)) >= 0; ++k) {
            const Unit U = unit(k);
            if (!__all_sync(~0u, fav::mbar_wait_il(o_done, k & 1, status))) break;
            if (!__all_sync(~0u, fav::mbar_wait_il(xch_bar + 8 * (k & 1), (k >> 1) & 1, status))) break;
            fav::tc::fence_after();
            const float2 ml0 = xch[((((k & 1) * 4 + quarter) * NS) + 0) * 32 + lane];
            const float2 ml1 = xch[((((k & 1) * 4 + quarter) * NS) + 1) * 32 + lane];
            if constexpr (varlen) fav::mbar_arrive(xch_free + 8 * (k & 1));
            const float Mx = fmaxf(ml0.x, ml1.x);
            const float w0 = (ml0.x == -INFINITY) ? 0.f : fav::fast_exp2(ml0.x - Mx);
            const float w1 = (ml1.x == -INFINITY) ? 0.f : fav::fast_exp2(ml1.x - Mx);
            const float L = w0 * ml0.y + w1 * ml1.y;
            const int qi = U.t * BM + row;
            if constexpr (kV16) asm volatile("griddepcontrol.wait;" ::: "memory");   // v_scale
            const float vsc = kV16 ? v_scale[U.b * Hkv + U.kvh] : 1.f;   // V = v_scale * (fp16 copy)
            const float inv_l = vsc / L;
            const float a0 = w0 * inv_l, a1 = w1 * inv_l;
            const uint32_t stage = sQ + (k & 1) * C::kQBytes + row * 128;
            // Dense calls: the tile goes through the Q buffer and one TMA store.  Packed batches:
            // every row is written straight to the output (a sequence's last tile has rows of the
            // next sequence past its end, and the Q buffer is released with the unit's last S, so
            // short units do not wait on the O store to load the next-but-one Q tile).
            const bool direct = varlen;
            const bool valid = qi < U.len_q;
            T *orow = o + U.b * os.b + U.h * os.h + (long long)(U.q_y0 + qi) * os.n;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {   // 32 columns at a time, both splits in flight
                uint32_t v0[32], v1[32];
                fav::tc::ld_32x32b_x32(trow + C::kColO + c * 32, v0);
                fav::tc::ld_32x32b_x32(trow + C::kColO + D + c * 32, v1);
                fav::tc::wait_ld_dep(v0);
                fav::tc::wait_ld_dep(v1);
                if (c + 1 == D / 32) {
                    // O has been read: release it to the next unit's first P.V
                    fav::tc::fence_before();
                    fav::mbar_arrive(o_free);
                }
#pragma unroll
                for (int h = 0; h < 4; ++h) {
                    // 8 columns = one 16-byte chunk: column block c / 2, chunk 4 (c % 2) + h
                    uint32_t x[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int i = 8 * h + 2 * e;
                        x[e] = fav::Elem<T>::pack(
                            fmaf(a0, __uint_as_float(v0[i]), a1 * __uint_as_float(v1[i])),
                            fmaf(a0, __uint_as_float(v0[i + 1]), a1 * __uint_as_float(v1[i + 1])));
                    }
                    if (!direct) {
                        const uint32_t chunk = (uint32_t)(4 * (c & 1) + h) ^ (uint32_t)(row & 7);
                        const uint32_t addr = stage + (c >> 1) * (BM * 128) + (chunk << 4);
                        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};"
                                     ::"r"(addr), "r"(x[0]), "r"(x[1]), "r"(x[2]), "r"(x[3])
                                     : "memory");
                    } else if (valid) {
                        *reinterpret_cast<uint4 *>(orow + c * 32 + 8 * h) = make_uint4(x[0], x[1], x[2], x[3]);
                    }
                }
            }
            if constexpr (!varlen) {
                fav::tc::fence_proxy_async_smem();   // visible to the TMA store (async proxy)
                fav::mbar_arrive(o_staged + 8 * (k & 1));
            }
            if (valid && lse) {
                // [B, Hq, Nq] (dense) or [Hq, total_q] (packed: Nq = total_q)
                const long long li = varlen ? (long long)U.h * Nq + U.q_y0 + qi
                                            : (long long)(U.b * Hq + U.h) * Nq + qi;
                lse[li] = (Mx - kPShift + log2f(L)) * kLn2;
            }
#ifdef FAV_DEBUG_CHECKS
            if (threadIdx.x == 32 * C::kEpiWarp0) dbg_tot[5] = k + 1;
#endif
        }
        fav::setmaxnreg_inc<C::kRegLaunch>();
    } else {
        fav::setmaxnreg_dec<C::kRegIssue>();
        if (warp == C::kLoadKWarp) {
            // ---------------- TMA producer: Q tiles and K tiles ----------------
            // (The stage waits poll with short suspensions: a thread suspended in a plain wait
            // resumed several hundred cycles after the stage was released, and a K tile is needed
            // by S about one key-tile period after its stage frees.)
            if (lane == 0) {
                int g = 0;
                bool ok = true;
                // L2 prefetches run kPrefetch key tiles ahead of the loads (the ring only covers
                // the L2 latency; a tile that misses L2 would stall S otherwise), and Q tiles a unit
                // ahead.
                TileIt pf{0, 0, unit(0)};
                for (int i = 0; i < kPrefetch; ++i) prefetch_next(&tmK, pf);
                const int early = min(KS, unit(0).n_kv);      // K tiles requested at the start
                for (int k = 0, u; ok && (u = unit_at(k)) >= 0; ++k) {
                    const Unit U = unit(k);
                    const int qb = k & 1;
                    if (unit_at(k + 1) >= 0) {
                        const Unit Un = unit(k + 1);
                        fav::tma_prefetch_l2_5d(&tmQ, 0, Un.q_y0 + Un.t * BM, 0, Un.h, Un.b);
                    }
                    // Q buffer qb was last read by unit k - 2's S MMAs (unit 0's Q: requested at the start)
                    if (k >= 2 && !fav::mbar_wait_il(q_empty + 8 * qb, ((k >> 1) - 1) & 1, status)) break;
                    if (k > 0) {
                        fav::mbar_arrive_expect_tx(q_full + 8 * qb, C::kQBytes);
                        fav::tma_load_5d(sQ + qb * C::kQBytes, &tmQ, q_full + 8 * qb, 0, U.q_y0 + U.t * BM, 0, U.h, U.b);
                    }
                    for (int j = 0; j < U.n_kv; ++j, ++g) {
                        const int st = g % KS;
                        if (g < early) {                // requested at the start
                            prefetch_next(&tmK, pf);
                            continue;
                        }
                        if (g >= KS && !fav::mbar_wait_fast_il(k_empty + 8 * st, ((g / KS) - 1) & 1, status)) {
                            ok = false;
                            break;
                        }
                        fav::mbar_arrive_expect_tx(k_full + 8 * st, C::kKVBytes);
                        fav::tma_load_5d(sK + st * C::kKVBytes, &tmK, k_full + 8 * st, 0, U.k_y0 + j * BN, 0, U.kvh, U.b);
                        prefetch_next(&tmK, pf);
                    }
                }
#ifdef FAV_DEBUG_CHECKS
                dbg_tot[1] = g;
#endif
            }
        } else if (warp == C::kLoadVWarp) {
            // ---------------- TMA producer: V tiles ----------------
            if (lane == 0) {
                // bf16 I/O: this kernel is a programmatic dependent of the V conversion, whose
                // output the V copies read (the set-up, Q and K copies go ahead of it)
                if constexpr (kV16) asm volatile("griddepcontrol.wait;" ::: "memory");
                fav::tma_prefetch_desc(&tmV);
                int g = 0;
                bool ok = true;
                TileIt pf{0, 0, unit(0)};
                for (int i = 0; i < kPrefetch; ++i) prefetch_next(&tmV, pf);
                for (int k = 0, u; ok && (u = unit_at(k)) >= 0; ++k) {
                    const Unit U = unit(k);
                    for (int j = 0; j < U.n_kv; ++j, ++g) {
                        const int st = g % VS;
                        prefetch_next(&tmV, pf);
                        if (g >= VS && !fav::mbar_wait_fast_il(v_empty + 8 * st, ((g / VS) - 1) & 1, status)) {
                            ok = false;
                            break;
                        }
                        fav::mbar_arrive_expect_tx(v_full + 8 * st, C::kKVBytes);
                        fav::tma_load_5d(sV + st * C::kKVBytes, &tmV, v_full + 8 * st, 0, U.k_y0 + j * BN, 0, U.kvh, U.b);
                    }
                }
#ifdef FAV_DEBUG_CHECKS
                dbg_tot[2] = g;
#endif
            }
        } else if (warp == C::kStoreWarp) {
            // ---------------- O tiles (dense calls): one TMA store per unit from its (free) Q buffer ----------------
            // (packed batches: the epilogue writes O itself)
            if (!varlen && lane == 0) {
                fav::tma_prefetch_desc(&tmO);
                for (int k = 0, u; (u = unit_at(k)) >= 0; ++k) {
                    const Unit U = unit(k);
                    const int qb = k & 1;
                    if (!fav::mbar_wait_il(o_staged + 8 * qb, (k >> 1) & 1, status)) break;
                    fav::tma_store_5d(&tmO, sQ + qb * C::kQBytes, 0, U.q_y0 + U.t * BM, 0, U.h, U.b);
                    fav::bulk_commit_group();
                    fav::bulk_wait_read_all();     // the buffer may take the next Q tile
                    fav::mbar_arrive(q_empty + 8 * qb);
#ifdef FAV_DEBUG_CHECKS
                    dbg_tot[6] = k + 1;
#endif
                }
                fav::bulk_wait_all();
            }
        } else {
            // ---------------- MMA issuer: the whole warp, converged; one elected lane issues ----------------
            constexpr bool bf = IsBF16<T>::value;
            constexpr uint32_t idesc_qk = fav::tc::idesc_f16(BM, BN, bf, false);
            constexpr uint32_t idesc_pv = fav::tc::idesc_f16(BM, D, false, true);      // fp16 P, V
            // Base descriptors are built once; a tile only adds its byte offset (>> 4) to the
            // start-address field, which cannot carry out of its 14 bits (addresses < 256 KB).
            const uint64_t dq0 = fav::tc::sdesc_sw128(sQ, 16, 1024);
            const uint64_t dk0 = fav::tc::sdesc_sw128(sK, 16, 1024);
            const uint64_t dv0 = fav::tc::sdesc_sw128(sV, BN * 128, 1024);
            // Every lane waits; the outcome is made warp-uniform so that a bounded wait that gives
            // up takes the whole warp out of the loop together (the bursts' elect.sync needs all
            // 32 lanes).
            // (A non-blocking test first: most of these phases have completed long before.)
            auto wait_all = [&](uint32_t bar, uint32_t parity) -> bool {
                if (__all_sync(0xffffffffu, fav::mbar_test(bar, parity))) return true;
                return __all_sync(0xffffffffu, fav::mbar_wait_il(bar, parity, status)) != 0;
            };
            // One flat loop: step t issues P(t-2).V (from t = 2 on) and then S(t), so the scores
            // run two key tiles ahead of the P.V products.  Each side walks the CTA's units with
            // its own indices (P.V: unit kp, key tile jp, count np; S: unit ks, key tile js,
            // count ns, us = unit_at(ks) or -1 past the end), and reads a unit's key-tile count
            // from the unit table when it moves on to that unit.  (One copy of each side's
            // bookkeeping: an earlier form issued the first two S products in a separate
            // prologue, and a unit count assigned there was seen as 0 in the main loop when the
            // CTA's first unit ended within the prologue.)
            int ks = 0, js = 0, Gs = 0;
            int us = unit_at(0);
            int ns = us >= 0 ? unit_nkv(0) : 0;
            int kp = 0, jp = 0, Gp = 0;
            int np = ns;
            bool ok = true;
            for (int t = 0; ok; ++t) {
                if (t >= 2) {
                    if (unit_at(kp) < 0) break;          // every P.V has been issued
                    const int vs = Gp % VS;
                    // lane 0: P(G); lane 1: V(G)
                    uint32_t tb = p_full + 8 * (Gp & 1), tp = (Gp >> 1) & 1;
                    if (lane == 1) { tb = v_full + 8 * vs; tp = (Gp / VS) & 1; }
                    const bool ready_pv = fav::mbar_test(tb, tp);
                    if (!__all_sync(0xffffffffu, ready_pv)) {
                        if (!(ok = wait_all(p_full + 8 * (Gp & 1), (Gp >> 1) & 1))) break;
                        if (!(ok = wait_all(v_full + 8 * vs, (Gp / VS) & 1))) break;
                    }
                    // a unit's first P.V overwrites O: the previous unit's O must have been read
                    if (jp == 0 && kp > 0 && !(ok = wait_all(o_free, (kp - 1) & 1))) break;
                    fav::tc::fence_after();
                    fav::tc::mma_pv_split<NS>(tmem + C::kColO, tmem + C::colS(Gp & 1),
                                              dv0 + (uint64_t)((vs * C::kKVBytes) >> 4), idesc_pv,
                                              jp > 0 ? 1u : 0u, v_empty + 8 * vs, pv_done);
                    if (jp + 1 == np) fav::tc::commit_elect(o_done);   // the unit's O is final
                    ++Gp;
                    if (++jp == np) {
                        jp = 0;
                        ++kp;
                        np = unit_at(kp) >= 0 ? unit_nkv(kp) : 0;
                    }
                }
                if (us < 0) continue;                    // no further S
                // operands of S(Gs): its unit's Q tile (first key tile only) and K(Gs) -- tested
                // at once (lane 0: K, lane 1: Q) behind the queued P.V MMAs
                {
                    uint32_t kb = k_full + 8 * (Gs % KS), kp_ = (Gs / KS) & 1;
                    if (js == 0 && lane == 1) { kb = q_full + 8 * (ks & 1); kp_ = (ks >> 1) & 1; }
                    const bool ready_s = fav::mbar_test(kb, kp_);
                    if (!__all_sync(0xffffffffu, ready_s)) {
                        if (js == 0 && !(ok = wait_all(q_full + 8 * (ks & 1), (ks >> 1) & 1))) break;
                        if (!(ok = wait_all(k_full + 8 * (Gs % KS), (Gs / KS) & 1))) break;
                    }
                }
                fav::tc::fence_after();
                {
                    const int qb = ks & 1, st = Gs % KS;
                    fav::tc::mma_ss_burst_k128<D / 16>(
                        tmem + C::colS(Gs & 1), dq0 + (uint64_t)((qb * C::kQBytes) >> 4),
                        dk0 + (uint64_t)((st * C::kKVBytes) >> 4), idesc_qk, 0u,
                        s_full + 8 * (Gs & 1), k_empty + 8 * st);
                }
                // the Q buffer is released with the unit's last S
                if (js + 1 == ns) fav::tc::commit_elect(q_empty + 8 * (ks & 1));
                ++Gs;
                if (++js == ns) {
                    js = 0;
                    us = unit_at(++ks);
                    ns = us >= 0 ? unit_nkv(ks) : 0;
                }
            }
#ifdef FAV_DEBUG_CHECKS
            if (lane == 0) { dbg_tot[3] = Gp; dbg_tot[4] = Gs; }
#endif
        }
        // (warps 9-11 ran their roles on lane 0 alone: the register budget below is changed by
        // each warp as a whole, so the warp is reconverged first)
        __syncwarp();
        fav::setmaxnreg_inc<C::kRegLaunch>();
    }

    fav::tc::fence_before();
    __syncthreads();
    fav::tc::fence_after();
    if (warp == C::kMmaWarp) fav::tc::tmem_dealloc(tmem, C::kTmemCols);
#ifdef FAV_DEBUG_CHECKS
    // every role processed the CTA's units and key tiles exactly (status 6 otherwise; a role
    // whose bounded wait gave up has already set status 5)
    if (threadIdx.x == 0 && *(volatile int *)status == 0) {
        int units = 0, tiles = 0;
        for (int k = 0; unit_at(k) >= 0; ++k) {
            ++units;
            tiles += unit_nkv(k);
        }
        (void)FAV_CHECK(dbg_tot[0] == tiles && dbg_tot[1] == tiles && dbg_tot[2] == tiles &&
                            dbg_tot[3] == tiles && dbg_tot[4] == tiles && dbg_tot[5] == units &&
                            (varlen || dbg_tot[6] == units),
                        status);
    }
#endif
}

// vunits: the unit table of a packed variable-length batch (device, 2 int4 per unit), or null
// (then kVarlen is false).
template <typename T, int D, bool kV16, bool kVarlen = false>
fav_status launch(const FavArgs &a, void *workspace, cudaStream_t stream,
                  const int4 *vunits = nullptr, int n_vunits = 0) {
    using C = PrefillCfg<D>;
    const void *vsrc = a.v;
    FavStrides vstr = a.vs;
    const float *v_scale = nullptr;
    if constexpr (kV16) {
        const fav_status st = fav_v16_convert(a, workspace, stream, &vsrc, &vstr, &v_scale);
        if (st != FAV_OK) return st;
    }
    alignas(64) CUtensorMap tmQ, tmK, tmV, tmO;
    fav_status st = fav_make_tmap_tiles(&tmQ, a.q, D, a.Nq, a.Hq, a.B, a.qs, BM);
    if (st == FAV_OK) st = fav_make_tmap_tiles(&tmK, a.k, D, a.Nkv, a.Hkv, a.B, a.ks, BN);
    if (st == FAV_OK) st = fav_make_tmap_tiles(&tmV, vsrc, D, a.Nkv, a.Hkv, a.B, vstr, BN);
    if (st == FAV_OK) st = fav_make_tmap_tiles(&tmO, a.o, D, a.Nq, a.Hq, a.B, a.os, BM);
    if (st != FAV_OK) return st;
    auto kern = fav_prefill_split_kernel<T, D, kV16, kVarlen>;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes) !=
        cudaSuccess)
        return FAV_ERR_CUDA;
    const int n_qtiles = (a.Nq + BM - 1) / BM;
    const long long units = vunits ? n_vunits : (long long)n_qtiles * a.B * a.Hq;
    if (units <= 0) return FAV_OK;
    // (unit indices up to units + grid size are formed in int)
    if (units + a.num_sms > 0x7fffffffLL) return FAV_ERR_UNSUPPORTED;
    // persistent: one CTA per SM at most, each working through its share of the units
    long long blocks = std::min<long long>(units, std::max(1, a.num_sms));
    if (a.prefill_grid > 0) blocks = std::min<long long>(blocks, a.prefill_grid);
    // Heads per L2 block: K and V of head_block query heads (shared by the G heads of a group)
    // within ~64 MB, a whole number of groups, at least one group and at most every head.  The
    // blocked order is applied where the unit table is filled, so it needs every unit of a
    // CTA in the table; otherwise one block.
    const int G = a.Hq / a.Hkv;
    const long long kv_bytes_group = 4LL * a.Nkv * D;             // K + V of one KV head
    long long groups_per_block = std::max(1LL, (64LL << 20) / std::max(1LL, kv_bytes_group));
    groups_per_block = std::min<long long>(groups_per_block, (long long)a.B * a.Hkv);
    int head_block = (int)(groups_per_block * G);
    if ((units + blocks - 1) / blocks > C::kUnitTab) head_block = a.B * a.Hq;
    // bf16 I/O: a programmatic dependent of the V conversion (set-up, Q and K copies overlap its
    // tail; V and its scales are read after griddepcontrol.wait)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)blocks);
    cfg.blockDim = dim3(C::kThreads);
    cfg.dynamicSmemBytes = C::kSmemBytes;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = kV16 ? 1 : 0;
    if (cudaLaunchKernelEx(&cfg, kern, tmQ, tmK, tmV, tmO, (T *)a.o, a.os, a.lse, v_scale, a.B,
                           a.Hq, a.Hkv, a.Nq, a.Nkv, n_qtiles, head_block, a.scale * kLog2e,
                           a.causal, a.dev_status, vunits, n_vunits) != cudaSuccess ||
        cudaGetLastError() != cudaSuccess || fav_debug_sync("fav_prefill_split_kernel", stream))
        return FAV_ERR_CUDA;
    return FAV_OK;
}

}  // namespace

fav_status fav_launch_prefill_split(const FavArgs &a, void *workspace, cudaStream_t s) {
    if (a.D != 128) return FAV_ERR_UNSUPPORTED;
    return a.dtype == FAV_F16 ? launch<__half, 128, false>(a, workspace, s)
                              : launch<__nv_bfloat16, 128, true>(a, workspace, s);
}

fav_status fav_launch_prefill_varlen(const FavArgs &a, const int4 *units, int n_units,
                                     void *workspace, cudaStream_t s) {
    if (a.D != 128) return FAV_ERR_UNSUPPORTED;
    return a.dtype == FAV_F16
               ? launch<__half, 128, false, true>(a, workspace, s, units, n_units)
               : launch<__nv_bfloat16, 128, true, true>(a, workspace, s, units, n_units);
}

bool fav_prefill_supported(const FavArgs &a) {
    if (a.dtype != FAV_F16 && a.dtype != FAV_BF16) return false;
    if (a.D != 64 && a.D != 128) return false;
    return (long long)a.B * a.Hq <= 0x7fffffffLL && (long long)a.B * a.Hkv <= 0x7fffffffLL;
}

size_t fav_prefill_workspace_bytes(const FavArgs &a) {
    return a.dtype == FAV_BF16 ? fav_v16_workspace_bytes(a) : 0;
}

// D = 128: the key-split kernel above; D = 64: the two-tile kernel (fav_prefill_pair.cu).  Each
// design is the faster one at its head dimension (measured on the prefill workloads).
fav_status fav_launch_prefill(const FavArgs &a, void *workspace, cudaStream_t s) {
    return a.D == 128 ? fav_launch_prefill_split(a, workspace, s)
                      : fav_launch_prefill_pair(a, workspace, s);
}
