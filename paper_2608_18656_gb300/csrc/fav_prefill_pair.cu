// fav_prefill_pair.cu -- prefill attention for D = 64 on the 5th-generation tensor cores
// (tcgen05 + TMEM + TMA): two query tiles per unit of work.
//
// Method (paper, Algorithm "FlashAttention-V for VL > D" and its description): the query
// rows of a block stay on chip for the whole sweep over key/value blocks; for every key block
// the scores are computed, the running maximum / sum / output accumulator of the online
// softmax are updated (rescale by exp(M_old - M), weights exp(S - M)), and after the last
// block the accumulator is normalised.  Heads sharing a K/V head read the same K/V tiles
// (GQA reuse), and several heads are processed by one unit of work (the paper's inter-head
// parallelism).  On this GPU that becomes:
//   * a unit is two 128-row query tiles that read the same K/V head: the same query tile of
//     two heads of one GQA group (even group sizes), or two consecutive query tiles of one
//     head.  The kernel is persistent (one CTA per SM at most); CTA c works through units
//     c, 2P-1-c, 2P+c, ... of the units sorted by decreasing causal work, loading the next
//     unit's Q tiles (TMA, 128-byte swizzle) during the current unit's tail;
//   * 128-key K and V tiles are streamed by TMA through a ring of shared-memory stages and
//     serve both query tiles;
//   * S_i = Q_i K^T (M = 128, N = 128, K = 64) and O_i += P_i V (M = 128, N = 64, K = 128) are
//     bursts of tcgen05.mma issued by one elected lane of a converged warp, accumulating in
//     tensor memory (TMEM), with P_i read from TMEM;
//   * one softmax warpgroup per query tile, one thread per query row (= TMEM lane): tcgen05.ld
//     of its scores, mask, row maximum, exp2 in the log2 domain, row sum, fp16 weights stored
//     with tcgen05.st.
// TMEM holds S0 | S1 | P0 | P1 | O0 | O1: the weights have columns of their own, S_i(j+1) is
// issued as soon as the softmax has read S_i(j), and the two tiles' softmaxes run back to
// back, half a period apart.  (With D = 64 the products are short and the softmax bounds the
// tile rate: two query tiles share each K/V tile and their softmaxes interleave.  D = 128 uses
// the key-split kernel of fav_prefill.cu.)
// The running maximum is updated lazily: O and l are rescaled only when the maximum grows by
// more than 2^4 (log2 domain); the weights are stored as p * 2^11 (below 2^15, inside fp16's
// range).  The final O / l uses the same maximum as every weight, so the result is unchanged.
//
// Warp roles (320 threads): warps 0-3 softmax of tile 0, warps 4-7 softmax of tile 1
// (TMEM lane quarter = warp % 4); warp 8 = TMEM owner + MMA issuer (the whole warp, one
// elected lane issuing each burst and committing the barrier arrivals inside the same asm
// block); warp 9 = TMA producer.  The issuing lane blocks while the tensor pipe is busy, and a
// wait on an mbarrier costs ~80 cycles of latency even when the phase is already complete; so
// the warp tests the barriers it will need next *before* a burst of MMAs where it can, and
// only waits for real on the ones that were not complete.
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
constexpr int kThreads = 320;
constexpr int kMmaWarp = 8, kLoadWarp = 9;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kRescaleThreshold = 4.0f;   // log2 units: rescale when max grows by > 2^4
// The weights are stored as p * 2^kPShift (exponent reference m - kPShift): with the lazy
// threshold they stay below 2^(4 + kPShift) = 2^15, inside fp16's range, and weights down to
// 2^-25 of the reference stay fp16 normals.  O / l is unchanged (l carries the same factor);
// the LSE subtracts kPShift.
constexpr float kPShift = 11.0f;

// 2^x for a pair of weights with ex2 on the special-function unit.  (Computing a share of them
// with a polynomial on the FMA pipe was measured slower on this GPU: the softmax is bound by
// issue slots and latency, not by the ex2 rate.)
template <int kPair>
__device__ __forceinline__ float2 exp2_pair(float2 x) {
    return make_float2(fav::fast_exp2(x.x), fav::fast_exp2(x.y));
}

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
    static_assert(D == 64, "the two-tile kernel serves D = 64");
    static constexpr int kStages = 3;                        // K/V ring depth
    static constexpr int kBoxes = D / 64;
    static constexpr int kQBytes = BM * D * 2;               // one Q tile
    static constexpr int kKVBytes = BN * D * 2;              // one K or V tile
    // shared-memory map (offsets from the 1024-aligned base)
    static constexpr int kOffQ = 0;                          // Q tile 0, Q tile 1
    static constexpr int kOffK = kOffQ + 2 * kQBytes;
    static constexpr int kOffV = kOffK + kStages * kKVBytes;
    static constexpr int kOffBar = kOffV + kStages * kKVBytes;
    static constexpr int kNumBars = 2 + 1 + 4 * kStages + 2 + 2 + 2 + 2 + 2;
    static constexpr int kOffTmemSlot = kOffBar + kNumBars * 8;
    static constexpr int kSmemBytes = kOffTmemSlot + 16 + 1024;
    // TMEM columns: S0 | S1 | P0 | P1 | O0 | O1; the weights have columns of their own, so the
    // next scores of a tile can be computed while its softmax still works on the current ones.
    static constexpr uint32_t kTmemCols = 512;
    static __host__ __device__ constexpr uint32_t colS(int i) { return i ? 128u : 0u; }
    static __host__ __device__ constexpr uint32_t colP(int i) { return 256u + 64u * i; }
    static __host__ __device__ constexpr uint32_t colO(int i) { return 384u + 64u * i; }
    static_assert(384 + 2 * D <= 512, "TMEM budget");
};

// bf16 I/O (kV16): Q, K and O are bf16; V has been converted to fp16 (tmV, scaled per KV head
// by v_scale^-1, a power of two) so that P.V runs with fp16 weights, and the epilogue multiplies
// O back by v_scale.  fp16 I/O: tmV is V itself.
template <typename T, int D, bool kV16>
__global__ void __launch_bounds__(kThreads, 1)
fav_prefill_pair_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV, T *__restrict__ o, FavStrides os,
                   float *__restrict__ lse, const float *__restrict__ v_scale, int B, int Hq,
                   int Hkv, int Nq, int Nkv, int n_qtiles, int pair_heads, float scale_log2,
                   int causal, int *status, const int4 *__restrict__ vunits, int n_vunits) {
    using C = PrefillCfg<D>;
    using TP = __half;    // type of the weights P and of V in shared memory (P.V MMA)
    constexpr int S = C::kStages;
    extern __shared__ uint8_t smem_raw[];
    // 1024-byte alignment in the shared window (the 128-byte swizzle atom of TMA and MMA)
    const uint32_t raw_u32 = fav::smem_u32(smem_raw);
    uint8_t *smem = smem_raw + ((1024u - (raw_u32 & 1023u)) & 1023u);
    const uint32_t sbase = fav::smem_u32(smem);
    const uint32_t sK = sbase + C::kOffK, sV = sbase + C::kOffV;
    const uint32_t bar0 = sbase + C::kOffBar;
    const uint32_t q_full = bar0;                 // [2], one per query tile
    const uint32_t q_empty = q_full + 16;         // Q buffers free (last S MMA of a unit done)
    const uint32_t k_full = q_empty + 8, k_empty = k_full + 8 * S;
    const uint32_t v_full = k_empty + 8 * S, v_empty = v_full + 8 * S;
    const uint32_t s_full = v_empty + 8 * S;      // [2], one per query tile
    const uint32_t p_full = s_full + 16;          // [2]
    const uint32_t o_done = p_full + 16;          // [2]
    const uint32_t s_free = o_done + 16;          // [2] (kSepP) the softmax has read S_i
    const uint32_t p_free = s_free + 16;          // [2] (kSepP) P_i.V has completed
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + C::kOffTmemSlot);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int G = Hq / Hkv;
    const int off = Nkv - Nq;                                   // bottom-right causal offset

    // ---- work units: two query tiles that read the same K/V head, heaviest causal first ----
    // Unit u: the same query tile of two heads of one GQA group (even group sizes), or two
    // consecutive query tiles of one head.  The CTA takes units c, 2P-1-c, 2P+c, 4P-1-c, ...
    // (P CTAs, "snake" order): with the units sorted by decreasing work, this evens out the
    // sums per CTA.
    // Variable-length batches (vunits != null): units from a table built on the host (three
    // int4 each: {sequence, h0, h1, t0}, {t1, key tiles 0, key tiles 1, first query row},
    // {first key row, query length, key length, -}), Q/O and K/V viewed as [1, H, total, D].
    struct Unit {
        int b, h[2], t[2], n_kv_tiles[2], n_kv, kvh, bkv, q_y0, k_y0, len_q, len_k;
    };
    const bool varlen = vunits != nullptr;
    const int n_units = varlen ? n_vunits
                               : pair_heads ? n_qtiles * B * (Hq / 2) : ((n_qtiles + 1) / 2) * B * Hq;
    auto unit_at = [&](int k) {   // the k-th unit of this CTA, or -1
        const int P = gridDim.x, c = blockIdx.x;
        const int u = k * P + ((k & 1) ? (P - 1 - c) : c);
        return u < n_units ? u : -1;
    };
    auto make_unit = [&](int u) {
        Unit U;
        if (varlen) {
            const int4 a = vunits[3 * u], c = vunits[3 * u + 1], e = vunits[3 * u + 2];
            U.b = 0;
            U.h[0] = a.y;
            U.h[1] = a.z;
            U.t[0] = a.w;
            U.t[1] = c.x;
            U.n_kv_tiles[0] = c.y;
            U.n_kv_tiles[1] = c.z;
            U.q_y0 = c.w;
            U.k_y0 = e.x;
            U.len_q = e.y;
            U.len_k = e.z;
            U.kvh = U.h[0] / G;
            U.bkv = U.kvh;
            U.n_kv = max(U.n_kv_tiles[0], U.n_kv_tiles[1]);
            return U;
        }
        U.q_y0 = U.k_y0 = 0;
        U.len_q = Nq;
        U.len_k = Nkv;
        if (pair_heads) {
            const int units = B * (Hq / 2);
            const int r = u % units;
            U.t[0] = U.t[1] = n_qtiles - 1 - u / units;
            U.b = r / (Hq / 2);
            U.h[0] = 2 * (r % (Hq / 2));
            U.h[1] = U.h[0] + 1;
        } else {
            const int BH = B * Hq;
            const int n_pairs = (n_qtiles + 1) / 2;
            const int bh = u % BH;
            const int pr = n_pairs - 1 - u / BH;
            U.b = bh / Hq;
            U.h[0] = U.h[1] = bh % Hq;
            U.t[0] = 2 * pr;
            U.t[1] = 2 * pr + 1;
        }
        U.kvh = U.h[0] / G;
        U.bkv = U.b * Hkv + U.kvh;
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            if (U.t[i] >= n_qtiles) {
                U.n_kv_tiles[i] = 0;
            } else {
                const int kv_end = causal ? min(Nkv, U.t[i] * BM + BM + off) : Nkv;
                U.n_kv_tiles[i] = (kv_end + BN - 1) / BN;
            }
        }
        U.n_kv = max(U.n_kv_tiles[0], U.n_kv_tiles[1]);
        return U;
    };

    if (warp == kLoadWarp && lane == 0) {
        (void)FAV_CHECK((sbase & 1023u) == 0, status);
        (void)FAV_CHECK((sbase - raw_u32) + C::kOffTmemSlot + 4 <= fav::dynamic_smem_bytes(), status);
        fav::mbar_init(q_full, 1);
        fav::mbar_init(q_full + 8, 1);
        fav::mbar_init(q_empty, 1);
        for (int s = 0; s < S; ++s) {
            fav::mbar_init(k_full + 8 * s, 1);
            fav::mbar_init(k_empty + 8 * s, 1);
            fav::mbar_init(v_full + 8 * s, 1);
            fav::mbar_init(v_empty + 8 * s, 1);
        }
        for (int i = 0; i < 2; ++i) {
            fav::mbar_init(s_full + 8 * i, 1);
            fav::mbar_init(p_full + 8 * i, 4);
            fav::mbar_init(o_done + 8 * i, 1);
            fav::mbar_init(s_free + 8 * i, 4);
            fav::mbar_init(p_free + 8 * i, 1);
        }
        fav::mbar_fence_init();
    }
    if (warp == kMmaWarp) {
        fav::tc::tmem_alloc(fav::smem_u32(tmem_slot), C::kTmemCols);
        fav::tc::tmem_relinquish();
    }
    fav::tc::fence_before();
    __syncthreads();
    fav::tc::fence_after();
    const uint32_t tmem = *tmem_slot;
    (void)FAV_CHECK((tmem & 0xFFFFu) + C::kTmemCols <= 512u && (tmem >> 16) == 0u, status);

    // Barrier phases run on across units: K/V stages follow one sequence g of key tiles
    // (stage g % S, parity (g / S) & 1) on both sides; s_full / p_full of tile i complete once
    // per key tile of i, o_done once per unit in which tile i has work, q_full once per unit.
    if (warp == kLoadWarp) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            fav::tma_prefetch_desc(&tmQ);
            fav::tma_prefetch_desc(&tmK);
            fav::tma_prefetch_desc(&tmV);
            int g = 0;
            bool ok = true;
            // bf16 I/O: this kernel is a programmatic dependent of the V conversion, whose output
            // the V copies read: wait for that grid before the first one (Q and K copies go ahead)
            bool v_ready = !kV16;
            for (int k = 0, u; ok && (u = unit_at(k)) >= 0; ++k) {
                const Unit U = make_unit(u);
                // the Q buffers are free once the previous unit's last S MMA has completed; both
                // tiles are loaded (a tile beyond the sequence reads the zero fill)
                if (k > 0 && !fav::mbar_wait(q_empty, (k - 1) & 1, status)) break;
#pragma unroll
                for (int i = 0; i < 2; ++i) {
                    fav::mbar_arrive_expect_tx(q_full + 8 * i, C::kQBytes);
#pragma unroll
                    for (int bx = 0; bx < C::kBoxes; ++bx)
                        fav::tma_load_4d(sbase + C::kOffQ + i * C::kQBytes + bx * BM * 128, &tmQ,
                                         q_full + 8 * i, bx * 64, U.q_y0 + U.t[i] * BM, U.h[i], U.b);
                }
                // Each stage has its own empty barriers (one commit per use, waited in order).
                for (int j = 0; j < U.n_kv; ++j, ++g) {
                    const int st = g % S;
                    const uint32_t ph = ((g / S) + 1) & 1;   // parity of the previous use's phase
                    if (g >= S && !fav::mbar_wait(k_empty + 8 * st, ph, status)) { ok = false; break; }
                    fav::mbar_arrive_expect_tx(k_full + 8 * st, C::kKVBytes);
#pragma unroll
                    for (int bx = 0; bx < C::kBoxes; ++bx)
                        fav::tma_load_4d(sK + st * C::kKVBytes + bx * BN * 128, &tmK, k_full + 8 * st,
                                         bx * 64, U.k_y0 + j * BN, U.kvh, U.b);
                    if (g >= S && !fav::mbar_wait(v_empty + 8 * st, ph, status)) { ok = false; break; }
                    if (!v_ready) {
                        asm volatile("griddepcontrol.wait;" ::: "memory");
                        v_ready = true;
                    }
                    fav::mbar_arrive_expect_tx(v_full + 8 * st, C::kKVBytes);
#pragma unroll
                    for (int bx = 0; bx < C::kBoxes; ++bx)
                        fav::tma_load_4d(sV + st * C::kKVBytes + bx * BN * 128, &tmV, v_full + 8 * st,
                                         bx * 64, U.k_y0 + j * BN, U.kvh, U.b);
                }
            }
        }
    } else if (warp == kMmaWarp) {
        // ---------------- MMA issuer: the whole warp, converged; one elected lane issues ----------------
        constexpr bool bf = IsBF16<T>::value;
        constexpr uint32_t idesc_qk = fav::tc::idesc_f16(BM, BN, bf, false);
        constexpr uint32_t idesc_pv = fav::tc::idesc_f16(BM, D, false, true);      // fp16 P, V
        // Base descriptors are built once; a tile only adds its byte offset (>> 4) to the
        // start-address field, which cannot carry out of its 14 bits (addresses < 256 KB).
        const uint64_t dq0 = fav::tc::sdesc_sw128(sbase + C::kOffQ, 16, 1024);
        const uint64_t dk0 = fav::tc::sdesc_sw128(sK, 16, 1024);
        const uint64_t dv0 = fav::tc::sdesc_sw128(sV, BN * 128, 1024);
        // S_i = Q_i K^T (K in ring stage st): D/16 k-steps over the 64-column boxes of Q_i and
        // K; the burst ends with commits to bar_a and bar_b (0 = none).
        auto issue_s = [&](int i, int st, uint32_t bar_a, uint32_t bar_b) {
            fav::tc::mma_ss_burst_k128<D / 16>(
                tmem + C::colS(i), dq0 + (uint64_t)((i * C::kQBytes) >> 4),
                dk0 + (uint64_t)((st * C::kKVBytes) >> 4), idesc_qk, 0u, bar_a, bar_b);
        };
        // O_i (+)= P_i V, with P_i read from TMEM (8 columns = 16 keys per k-step) and V MN-major
        // in shared memory (8-key groups 1024 B apart, 64-column blocks one box apart).
        auto issue_pv = [&](int i, int st, uint32_t acc, uint32_t bar_a, uint32_t bar_b) {
            fav::tc::mma_ts_burst_k128(tmem + C::colO(i), tmem + C::colP(i),
                                       dv0 + (uint64_t)((st * C::kKVBytes) >> 4), idesc_pv, acc,
                                       bar_a, bar_b);
        };
        // Every lane waits; the outcome is made warp-uniform so that a bounded wait that gives
        // up takes the whole warp out of the loop together (the bursts' elect.sync needs all
        // 32 lanes).
        auto wait_all = [&](uint32_t bar, uint32_t parity) {
            return __all_sync(0xffffffffu, fav::mbar_wait(bar, parity, status));
        };
        // Two barriers tested with one instruction (lane 0: a, if need_a; lane 1: b), then waited
        // for one by one only if one of them was not complete.  Each test instruction of this warp
        // costs it about as much as a short burst of MMAs takes to issue (it waits for the warp's
        // queued MMAs and commits), and the K / V stages are almost always complete by the time
        // the softmax has released its scores / stored its weights: testing them with those
        // barriers instead of separately took C3 from 315.5 to 307.2 us.
        auto wait_two = [&](uint32_t bar_a, uint32_t par_a, bool need_a, uint32_t bar_b,
                            uint32_t par_b) -> bool {
            uint32_t tb = bar_b, tp = par_b;
            bool need = lane == 1;
            if (lane == 0) { tb = bar_a; tp = par_a; need = need_a; }
            if (__all_sync(0xffffffffu, !need || fav::mbar_test(tb, tp))) return true;
            if (need_a && !wait_all(bar_a, par_a)) return false;
            return wait_all(bar_b, par_b) != 0;
        };
        auto try_all = [&](uint32_t bar, uint32_t parity) {
            return __all_sync(0xffffffffu, fav::mbar_try(bar, parity));
        };
        int g = 0;                 // key tiles streamed so far (ring sequence)
        int np[2] = {0, 0};        // P_i(.) consumed so far, per tile (p_full parity)
        int nsi[2] = {0, 0};       // S_i(.) issued so far, per tile (s_free parity, kSepP)
        bool ok = true;
        for (int k = 0, u; ok && (u = unit_at(k)) >= 0; ++k) {
            const Unit U = make_unit(u);
            const int g0 = g;
            {
                // Weights in their own columns: S_i(j+1) is issued as soon as the softmax has
                // read S_i(j) (s_free), before P_i(j).V, which is issued when P_i(j) is ready;
                // the softmax waits for P_i(j).V (p_free) before it stores P_i(j+1) or rescales
                // O_i.  Each tile's softmax can then run from one key tile to the next without
                // waiting for the tensor core.
                const int last0 = U.n_kv_tiles[1] > 0 ? 1 : 0;      // last tile with work
                if (!(ok = wait_all(k_full + 8 * (g0 % S), (g0 / S) & 1))) break;
                // S_1(0) waits until tile 0's softmax has reached its exponentials: the two
                // softmaxes then run half a period apart, so that one's exponentials (MUFU) overlap
                // the other's loads and maxima instead of competing for the MUFU in lockstep;
                // the offset carries over to the following key tiles.
#pragma unroll
                for (int i = 0; i < 2; ++i) {
                    // Both Q copies are waited for, an unused tile's too: q_empty lets the
                    // producer re-arm q_full for the next unit, which must not happen while this
                    // unit's copy is still in flight (a second arrival in one phase).
                    if (!(ok = wait_all(q_full + 8 * i, k & 1))) break;
                    if (U.n_kv_tiles[i] == 0) continue;
                    if (i == 1 && !(ok = wait_all(s_free, (nsi[0] - 1) & 1))) break;
                    if (nsi[i] > 0 && !(ok = wait_all(s_free + 8 * i, (nsi[i] - 1) & 1))) break;
                    fav::tc::fence_after();
                    issue_s(i, g0 % S, s_full + 8 * i, i == last0 ? k_empty + 8 * (g0 % S) : 0u);
                    ++nsi[i];
                }
                if (!ok) break;
                if (U.n_kv == 1) fav::tc::commit_elect(q_empty);    // no further S in this unit
                // Per key tile j, tile by tile: S_i(j+1) (once the softmax has read S_i(j)), then
                // P_i(j).V_j (once P_i(j) is stored).  Tile 1's softmax runs half a period behind
                // tile 0's, so this order never holds one tile's MMAs behind the other's events.
                // K_{j+1} and V_j are released by the last tile's bursts.
                for (int j = 0; ok && j < U.n_kv; ++j) {
                    const int gj = g0 + j;
                    const int st = gj % S, st1 = (gj + 1) % S;
                    const int last1 = j + 1 < U.n_kv_tiles[1] ? 1 : 0;   // last tile with S(j+1)
                    const int last = j < U.n_kv_tiles[1] ? 1 : 0;        // last tile with P(j)
                    bool k_ok = false, v_ok = false;
#pragma unroll
                    for (int i = 0; i < 2; ++i) {
                        if (j + 1 < U.n_kv_tiles[i]) {
                            if (!(ok = wait_two(k_full + 8 * st1, ((gj + 1) / S) & 1, !k_ok,
                                                s_free + 8 * i, (nsi[i] - 1) & 1))) break;
                            k_ok = true;
                            fav::tc::fence_after();
                            issue_s(i, st1, s_full + 8 * i, i == last1 ? k_empty + 8 * st1 : 0u);
                            ++nsi[i];
                        }
                        if (j < U.n_kv_tiles[i]) {
                            if (!(ok = wait_two(v_full + 8 * st, (gj / S) & 1, !v_ok,
                                                p_full + 8 * i, np[i] & 1))) break;
                            v_ok = true;
                            ++np[i];
                            fav::tc::fence_after();
                            issue_pv(i, st, j > 0 ? 1u : 0u, p_free + 8 * i, i == last ? v_empty + 8 * st : 0u);
                            if (j + 1 == U.n_kv_tiles[i]) fav::tc::commit_elect(o_done + 8 * i);
                        }
                    }
                    if (!ok) break;
                    // after the unit's last scores (issued in this key tile), its Q buffers can be
                    // refilled: the commit covers every MMA issued so far
                    if (j + 2 == U.n_kv) fav::tc::commit_elect(q_empty);
                }
                g += U.n_kv;
            }
        }
    } else {
        // ---------------- softmax / correction / epilogue: one thread per query row ----------------
        const int i = warp >> 2;                          // query tile of this warpgroup
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
        const uint32_t colS = i ? C::colS(1) : C::colS(0);
        const uint32_t colO = i ? C::colO(1) : C::colO(0);
        int ns = 0, no = 0;        // S_i(.) and O_i completions consumed so far (parities)
        int npst = 0;              // P_i(.) stored so far (kSepP: p_free parity)
        const uint32_t colP = i ? C::colP(1) : C::colP(0);
        bool ok = true;
        for (int k = 0, u; ok && (u = unit_at(k)) >= 0; ++k) {
            const Unit U = make_unit(u);
            const int n_mine = U.n_kv_tiles[i];
            if (n_mine == 0) continue;
            const int ti = U.t[i], hi = U.h[i];
            const int q0 = ti * BM;
            const int qi = q0 + row;                          // query index of this row
            const int uoff = U.len_k - U.len_q;               // bottom-right causal offset
            const int lim = causal ? min(U.len_k, qi + uoff + 1) : U.len_k;      // visible keys: [0, lim)
            const int lim_tile = causal ? min(U.len_k, q0 + uoff + 1) : U.len_k; // smallest lim in the tile
            float m = -INFINITY, l = 0.f;
            for (int j = 0; j < n_mine; ++j) {
                if (!__all_sync(~0u, fav::mbar_wait(s_full + 8 * i, ns & 1, status))) { ok = false; break; }
                ++ns;
                fav::tc::fence_after();
                const int key0 = j * BN;
                const bool crosses = key0 + BN > lim_tile;   // tile crosses the diagonal or the end
                float s[BN];
                // S row from TMEM (and the mask: keys at or beyond lim get -inf)
                auto load_s = [&]() {
                    uint32_t r[BN / 64][64];
#pragma unroll
                    for (int c = 0; c < BN / 64; ++c) fav::tc::ld_32x32b_x64(trow + colS + c * 64, r[c]);
#pragma unroll
                    for (int c = 0; c < BN / 64; ++c) fav::tc::wait_ld_dep(r[c]);
#pragma unroll
                    for (int c = 0; c < BN; ++c) s[c] = __uint_as_float(r[c >> 6][c & 63]);
                    if (crosses) {
#pragma unroll
                        for (int c = 0; c < BN; ++c)
                            if (key0 + c >= lim) s[c] = -INFINITY;
                    }
                };
                // raw row maximum: 8 independent chains of 3-input max, then a tree
                auto row_max = [&]() {
                    float m8[8];
#pragma unroll
                    for (int c = 0; c < 8; ++c) m8[c] = s[c];
#pragma unroll
                    for (int c = 8; c < BN; c += 16) {
#pragma unroll
                        for (int q = 0; q < 8; ++q) m8[q] = fav::fmax3(m8[q], s[c + q], s[c + 8 + q]);
                    }
                    return fav::fmax3(fav::fmax3(m8[0], m8[1], m8[2]), fav::fmax3(m8[3], m8[4], m8[5]),
                                      fmaxf(m8[6], m8[7]));
                };
                // p = exp2(s * scale_log2 - mref) on pairs (one packed FMA, two ex2, one packed
                // add), fp16 weights stored to TMEM half a row at a time (keys [64h, 64h + 64)
                // over S columns [32h, 32h + 32), whose scores are already in registers); the
                // fp32 sum goes to psum.
                float psum = 0.f;
                auto exp_store = [&](float mref) {
                    const float2 sc2 = make_float2(scale_log2, scale_log2);
                    const float2 nm2 = make_float2(-mref, -mref);
                    float2 l4[4] = {{0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}, {0.f, 0.f}};
                    static_for<0, 2>([&](auto hc) {
                        constexpr int h = decltype(hc)::value;
                        uint32_t pk[32];
                        static_for<0, 32>([&](auto pc) {
                            constexpr int e = 2 * decltype(pc)::value;
                            constexpr int c = 64 * h + e;
                            const float2 x = fav::ffma2(make_float2(s[c], s[c + 1]), sc2, nm2);
                            const float2 p = exp2_pair<c / 2>(x);
                            l4[(e >> 1) & 3] = fav::fadd2(l4[(e >> 1) & 3], p);
                            pk[e >> 1] = fav::Elem<TP>::pack(p.x, p.y);
                        });
                        fav::tc::st_32x32b_x32(trow + colP + 32 * h, pk);
                    });
                    const float2 a = fav::fadd2(fav::fadd2(l4[0], l4[1]), fav::fadd2(l4[2], l4[3]));
                    psum = a.x + a.y;
                };
                float alpha = 1.f;
                bool rescale = false;
                // lazy rescale: move the reference maximum only when it grows by > 2^4
                auto move_max = [&](float mx) {
                    if (mx > m + kRescaleThreshold) {
                        alpha = fav::fast_exp2(m - mx);   // 0 on the first tile (m = -inf)
                        rescale = (j > 0);
                        m = mx;
                        l *= alpha;
                    }
                };
                // two passes: the row maximum, then the weights against the (lazy) reference
                load_s();
                move_max(row_max() * scale_log2);
                {
                    // S_i has been read (long ago; the signal waits for the start of the
                    // exponentials, which also paces the other tile: see the MMA warp)
                    fav::tc::fence_before();
                    __syncwarp();
                    if (lane == 0) fav::mbar_arrive(s_free + 8 * i);
                }
                // P_i over the first 64 columns of S_i (two 16-bit weights per column)
                {
                    // P_i's columns and O_i are free and stable once the previous P_i.V is done
                    if (npst > 0 && !__all_sync(~0u, fav::mbar_wait(p_free + 8 * i, (npst - 1) & 1, status))) {
                        ok = false;
                        break;
                    }
                    fav::tc::fence_after();
                }
                ++npst;
                exp_store(m - kPShift);
                l += psum;
                // O_i is stable here: P_i(j-1).V has completed (D = 128: it was issued before
                // S_i(j) and MMAs complete in issue order; D = 64: the p_free wait above).
                if (__any_sync(~0u, rescale)) {
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
                if (lane == 0) fav::mbar_arrive(p_full + 8 * i);
            }
            if (!ok) break;
            // ---------------- epilogue: O / l, LSE ----------------
            // (the next unit's first P.V, which overwrites O_i, waits for this warpgroup's next
            // P_i: it cannot run before these loads)
            if (!__all_sync(~0u, fav::mbar_wait(o_done + 8 * i, no & 1, status))) { ok = false; break; }
            ++no;
            fav::tc::fence_after();
            if constexpr (kV16) asm volatile("griddepcontrol.wait;" ::: "memory");   // v_scale
            const float vsc = kV16 ? v_scale[U.bkv] : 1.f;     // V = v_scale * (fp16 copy)
            const float inv_l = vsc / l;
            const bool valid = qi < U.len_q;
            T *orow = o + U.b * os.b + hi * os.h + (long long)(U.q_y0 + qi) * os.n;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                uint32_t v[32];
                fav::tc::ld_32x32b_x32(trow + colO + c * 32, v);
                fav::tc::wait_ld_dep(v);
                if (valid) {
#pragma unroll
                    for (int e = 0; e < 32; e += 8) {
                        uint4 v4;
                        v4.x = fav::Elem<T>::pack(__uint_as_float(v[e]) * inv_l, __uint_as_float(v[e + 1]) * inv_l);
                        v4.y = fav::Elem<T>::pack(__uint_as_float(v[e + 2]) * inv_l, __uint_as_float(v[e + 3]) * inv_l);
                        v4.z = fav::Elem<T>::pack(__uint_as_float(v[e + 4]) * inv_l, __uint_as_float(v[e + 5]) * inv_l);
                        v4.w = fav::Elem<T>::pack(__uint_as_float(v[e + 6]) * inv_l, __uint_as_float(v[e + 7]) * inv_l);
                        *reinterpret_cast<uint4 *>(orow + c * 32 + e) = v4;
                    }
                }
            }
            if (valid && lse) {
                // [B, Hq, Nq] (dense) or [Hq, total_q] (packed: Nq = total_q)
                const long long li = varlen ? (long long)hi * Nq + U.q_y0 + qi
                                            : (long long)(U.b * Hq + hi) * Nq + qi;
                lse[li] = (m - kPShift + log2f(l)) * kLn2;
            }
            fav::tc::fence_before();
        }
    }

    fav::tc::fence_before();
    __syncthreads();
    fav::tc::fence_after();
    if (warp == kMmaWarp) fav::tc::tmem_dealloc(tmem, C::kTmemCols);
}

// vunits: the unit table of a packed variable-length batch (device, 3 int4 per unit), or null.
template <typename T, int D, bool kV16>
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
    alignas(64) CUtensorMap tmQ, tmK, tmV;
    fav_status st = fav_make_tmap_4d(&tmQ, a.q, D, a.Nq, a.Hq, a.B, a.qs, BM);
    if (st == FAV_OK) st = fav_make_tmap_4d(&tmK, a.k, D, a.Nkv, a.Hkv, a.B, a.ks, BN);
    if (st == FAV_OK) st = fav_make_tmap_4d(&tmV, vsrc, D, a.Nkv, a.Hkv, a.B, vstr, BN);
    if (st != FAV_OK) return st;
    auto kern = fav_prefill_pair_kernel<T, D, kV16>;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes) !=
        cudaSuccess)
        return FAV_ERR_CUDA;
    const int n_qtiles = (a.Nq + BM - 1) / BM;
    const int G = a.Hq / a.Hkv;
    const int pair_heads = (G % 2 == 0) ? 1 : 0;
    const long long units = vunits ? n_vunits
                          : pair_heads ? (long long)n_qtiles * a.B * (a.Hq / 2)
                                       : (long long)((n_qtiles + 1) / 2) * a.B * a.Hq;
    if (units <= 0) return FAV_OK;
    if (units + a.num_sms > 0x7fffffffLL) return FAV_ERR_UNSUPPORTED;
    // persistent: one CTA per SM at most, each working through its share of the units
    long long blocks = std::min<long long>(units, std::max(1, a.num_sms));
    if (a.prefill_grid > 0) blocks = std::min<long long>(blocks, a.prefill_grid);
    // bf16 I/O: a programmatic dependent of the V conversion (set-up, Q and K copies overlap its
    // tail; V and its scales are read after griddepcontrol.wait)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)blocks);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = C::kSmemBytes;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = kV16 ? 1 : 0;
    if (cudaLaunchKernelEx(&cfg, kern, tmQ, tmK, tmV, (T *)a.o, a.os, a.lse, v_scale, a.B, a.Hq,
                           a.Hkv, a.Nq, a.Nkv, n_qtiles, pair_heads, a.scale * kLog2e, a.causal,
                           a.dev_status, vunits, n_vunits) != cudaSuccess ||
        cudaGetLastError() != cudaSuccess || fav_debug_sync("fav_prefill_pair_kernel", stream))
        return FAV_ERR_CUDA;
    return FAV_OK;
}

}  // namespace

fav_status fav_launch_prefill_pair(const FavArgs &a, void *workspace, cudaStream_t s) {
    if (a.D != 64) return FAV_ERR_UNSUPPORTED;
    return a.dtype == FAV_F16 ? launch<__half, 64, false>(a, workspace, s)
                              : launch<__nv_bfloat16, 64, true>(a, workspace, s);
}

fav_status fav_launch_prefill_pair_varlen(const FavArgs &a, const int4 *units, int n_units,
                                          void *workspace, cudaStream_t s) {
    if (a.D != 64) return FAV_ERR_UNSUPPORTED;
    return a.dtype == FAV_F16 ? launch<__half, 64, false>(a, workspace, s, units, n_units)
                              : launch<__nv_bfloat16, 64, true>(a, workspace, s, units, n_units);
}
