// fav_prefill.cu -- prefill attention on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
// Method (paper, Algorithm "FlashAttention-V for VL > D" and its description): the query
// rows of a block stay on chip for the whole sweep over key/value blocks; for every key block
// the scores are computed, the running maximum / sum / output accumulator of the online
// softmax are updated (rescale by exp(M_old - M), weights exp(S - M)), and after the last
// block the accumulator is normalised.  Heads sharing a K/V head read the same K/V tiles
// (GQA reuse).  On this GPU the paper's register blocking becomes:
//   * a 128 x D query tile in shared memory (TMA, 128-byte swizzle), loaded once;
//   * 128-key K and V tiles streamed by TMA through a ring of shared-memory stages;
//   * S = Q K^T (M = 128, N = 128, K = D) and O += P V (M = 128, N = D, K = 128) as
//     tcgen05.mma issued by one thread, accumulating in tensor memory (TMEM):
//     two S buffers (so S_{j+1} is computed while the softmax works on S_j) and one O;
//   * a softmax warpgroup, one thread per query row (= TMEM lane): tcgen05.ld of its S row,
//     mask, row max, exp2 in the log2 domain, row sum, P rounded to the I/O type and written
//     to shared memory in the K-major 128-byte-swizzled layout the MMA reads.
// The running maximum is updated lazily: O and l are rescaled only when the maximum grows by
// more than 2^8 (log2 domain); otherwise the stale maximum is kept and the weights may reach
// 256.  The final O / l uses the same maximum as every weight, so the result is unchanged.
//
// Warp roles (192 threads): warp 0 = TMA producer, warp 1 = TMEM owner + MMA issuer,
// warps 2..5 = softmax / correction / epilogue (TMEM lane quarter = warp % 4).
#include <cuda.h>
#include <math.h>

#include "fav_device.cuh"
#include "fav_internal.h"
#include "fav_tc.cuh"

namespace {

constexpr int BM = 128;          // query rows per tile (= TMEM lanes)
constexpr int BN = 128;          // keys per tile
constexpr int kThreads = 192;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kRescaleThreshold = 8.0f;   // log2 units: rescale when max grows by > 2^8

template <int D> struct PrefillCfg {
    static constexpr int kStages = (D == 128) ? 2 : 3;      // K/V ring depth
    static constexpr int kBoxes = D / 64;
    static constexpr int kQBytes = BM * D * 2;
    static constexpr int kKVBytes = BN * D * 2;              // one K or V tile
    static constexpr int kPBytes = BM * BN * 2;
    // shared-memory map (offsets from the 1024-aligned base)
    static constexpr int kOffQ = 0;
    static constexpr int kOffK = kOffQ + kQBytes;
    static constexpr int kOffV = kOffK + kStages * kKVBytes;
    static constexpr int kOffP = kOffV + kStages * kKVBytes;
    static constexpr int kOnesBytes = 16 * 128;              // 16 rows x 64 ones (bf16)
    static constexpr int kOffOnes = kOffP + kPBytes;
    static constexpr int kOffBar = kOffOnes + 1024 * ((kOnesBytes + 1023) / 1024);
    static constexpr int kNumBars = 1 + 4 * kStages + 2 + 2 + 2;
    static constexpr int kOffTmemSlot = kOffBar + kNumBars * 8;
    static constexpr int kSmemBytes = kOffTmemSlot + 16 + 1024;
    static constexpr uint32_t kTmemCols = 512;               // S0 | S1 | O
    static constexpr uint32_t kColS0 = 0, kColS1 = 128, kColO = 256;
    static constexpr uint32_t kColL = kColO + D;             // 16 columns of sum_k P~[row][k]
};

template <typename T> struct IsBF16 { static constexpr bool value = false; };
template <> struct IsBF16<__nv_bfloat16> { static constexpr bool value = true; };

// With bf16 I/O the weights P are rounded to 8 significant bits before the P.V product.  With
// the lazy maximum a dominant weight can be any value up to 2^8, so normalising the rounded
// numerator by the unrounded fp32 sum would leave the dominant term off by up to 2^-9 of |v|.
// The bf16 kernel therefore divides by l~ = sum_k P~[row][k], accumulated by the tensor core
// (P~ times a column of ones) next to O, so numerator and denominator use the same weights;
// the fp32 sum of the unrounded weights still gives the LSE.  fp16 keeps 11 bits and divides
// by the fp32 sum.
template <typename T> struct RoundedNorm { static constexpr bool value = IsBF16<T>::value; };

template <typename T, int D>
__global__ void __launch_bounds__(kThreads, 1)
fav_prefill_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV, T *__restrict__ o,
                   float *__restrict__ lse, int Hq, int Hkv, int Nq, int Nkv, int n_qtiles,
                   float scale_log2, int causal, int *status) {
    using C = PrefillCfg<D>;
    constexpr int S = C::kStages;
    extern __shared__ uint8_t smem_raw[];
    // 1024-byte alignment in the shared window (the 128-byte swizzle atom of TMA and MMA)
    const uint32_t raw_u32 = fav::smem_u32(smem_raw);
    uint8_t *smem = smem_raw + ((1024u - (raw_u32 & 1023u)) & 1023u);
    const uint32_t sbase = fav::smem_u32(smem);
    const uint32_t sQ = sbase + C::kOffQ, sK = sbase + C::kOffK, sV = sbase + C::kOffV;
    const uint32_t sP = sbase + C::kOffP;
    // barriers
    const uint32_t bar0 = sbase + C::kOffBar;
    const uint32_t q_full = bar0;
    const uint32_t k_full = bar0 + 8, k_empty = k_full + 8 * S;
    const uint32_t v_full = k_empty + 8 * S, v_empty = v_full + 8 * S;
    const uint32_t s_full = v_empty + 8 * S;      // [2]
    const uint32_t s_free = s_full + 16;          // [2]
    const uint32_t p_full = s_free + 16;
    const uint32_t p_empty = p_full + 8;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + C::kOffTmemSlot);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int BH = gridDim.x / n_qtiles;
    const int qtile = n_qtiles - 1 - (int)(blockIdx.x / BH);   // heaviest (causal) tiles first
    const int bh = blockIdx.x % BH;                            // b * Hq + h
    const int b = bh / Hq, h = bh % Hq;
    const int G = Hq / Hkv;
    const int bkv = b * Hkv + h / G;
    const int q0 = qtile * BM;
    const int off = Nkv - Nq;                                  // bottom-right causal offset
    const int kv_end = causal ? min(Nkv, q0 + BM + off) : Nkv; // keys any row of the tile sees
    const int n_kv = (kv_end + BN - 1) / BN;

    if (warp == 0 && lane == 0) {
        (void)FAV_CHECK((sbase & 1023u) == 0, status);
        (void)FAV_CHECK((sbase - raw_u32) + C::kOffTmemSlot + 4 <= fav::dynamic_smem_bytes(), status);
        fav::mbar_init(q_full, 1);
        for (int s = 0; s < S; ++s) {
            fav::mbar_init(k_full + 8 * s, 1);
            fav::mbar_init(k_empty + 8 * s, 1);
            fav::mbar_init(v_full + 8 * s, 1);
            fav::mbar_init(v_empty + 8 * s, 1);
        }
        for (int s = 0; s < 2; ++s) {
            fav::mbar_init(s_full + 8 * s, 1);
            fav::mbar_init(s_free + 8 * s, 4);
        }
        fav::mbar_init(p_full, 4);
        fav::mbar_init(p_empty, 1);
        fav::mbar_fence_init();
    }
    if (RoundedNorm<T>::value && warp >= 2) {
        // bf16 1.0 = 0x3F80; every element of the tile is one, so its layout is irrelevant.
        uint32_t *ones = reinterpret_cast<uint32_t *>(smem + C::kOffOnes);
        for (int i = threadIdx.x - 64; i < C::kOnesBytes / 4; i += kThreads - 64) ones[i] = 0x3F803F80u;
        fav::tc::fence_proxy_async_smem();
    }
    if (warp == 1) {
        fav::tc::tmem_alloc(fav::smem_u32(tmem_slot), C::kTmemCols);
        fav::tc::tmem_relinquish();
    }
    fav::tc::fence_before();
    __syncthreads();
    fav::tc::fence_after();
    const uint32_t tmem = *tmem_slot;
    (void)FAV_CHECK((tmem & 0xFFFFu) + C::kTmemCols <= 512u && (tmem >> 16) == 0u, status);

    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            fav::tma_prefetch_desc(&tmQ);
            fav::tma_prefetch_desc(&tmK);
            fav::tma_prefetch_desc(&tmV);
            fav::mbar_arrive_expect_tx(q_full, C::kQBytes);
#pragma unroll
            for (int bx = 0; bx < C::kBoxes; ++bx)
                fav::tma_load_3d(sQ + bx * BM * 128, &tmQ, q_full, bx * 64, q0, bh);
            for (int j = 0; j < n_kv; ++j) {
                const int st = j % S;
                const uint32_t ph = ((j / S) + 1) & 1;   // parity of the previous use's phase
                if (j >= S && !fav::mbar_wait(k_empty + 8 * st, ph, status)) break;
                fav::mbar_arrive_expect_tx(k_full + 8 * st, C::kKVBytes);
#pragma unroll
                for (int bx = 0; bx < C::kBoxes; ++bx)
                    fav::tma_load_3d(sK + st * C::kKVBytes + bx * BN * 128, &tmK, k_full + 8 * st,
                                     bx * 64, j * BN, bkv);
                if (j >= S && !fav::mbar_wait(v_empty + 8 * st, ph, status)) break;
                fav::mbar_arrive_expect_tx(v_full + 8 * st, C::kKVBytes);
#pragma unroll
                for (int bx = 0; bx < C::kBoxes; ++bx)
                    fav::tma_load_3d(sV + st * C::kKVBytes + bx * BN * 128, &tmV, v_full + 8 * st,
                                     bx * 64, j * BN, bkv);
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            constexpr bool bf = IsBF16<T>::value;
            constexpr uint32_t idesc_qk = fav::tc::idesc_f16(BM, BN, bf, false);
            constexpr uint32_t idesc_pv = fav::tc::idesc_f16(BM, D, bf, true);
            constexpr uint32_t idesc_l = fav::tc::idesc_f16(BM, 16, bf, false);
            const uint64_t ones_desc = fav::tc::sdesc_sw128(sbase + C::kOffOnes, 16, 1024);
            bool ok = fav::mbar_wait(q_full, 0, status);
            // S_j = Q K_j^T into S buffer j % 2
            auto issue_s = [&](int j) -> bool {
                const int st = j % S;
                if (!fav::mbar_wait(k_full + 8 * st, (j / S) & 1, status)) return false;
                if (j >= 2 && !fav::mbar_wait(s_free + 8 * (j & 1), ((j >> 1) + 1) & 1, status))
                    return false;
                fav::tc::fence_after();
                const uint32_t d_tmem = tmem + ((j & 1) ? C::kColS1 : C::kColS0);
                const uint32_t kst = sK + st * C::kKVBytes;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t koff = (kk >> 2) * (BM * 128) + (kk & 3) * 32;
                    const uint64_t ad = fav::tc::sdesc_sw128(sQ + koff, 16, 1024);
                    const uint64_t bd = fav::tc::sdesc_sw128(kst + (kk >> 2) * (BN * 128) + (kk & 3) * 32,
                                                             16, 1024);
                    fav::tc::mma_ss(d_tmem, ad, bd, idesc_qk, kk > 0);
                }
                fav::tc::commit(s_full + 8 * (j & 1));
                fav::tc::commit(k_empty + 8 * st);
                return true;
            };
            if (ok && n_kv > 0) ok = issue_s(0);
            for (int j = 0; ok && j < n_kv; ++j) {
                if (j + 1 < n_kv && !issue_s(j + 1)) { ok = false; break; }
                const int st = j % S;
                if (!fav::mbar_wait(p_full, j & 1, status)) { ok = false; break; }
                if (!fav::mbar_wait(v_full + 8 * st, (j / S) & 1, status)) { ok = false; break; }
                fav::tc::fence_after();
                const uint32_t vst = sV + st * C::kKVBytes;
#pragma unroll
                for (int kk = 0; kk < BN / 16; ++kk) {
                    // A = P (128 rows x 16 keys, K-major); B = V (16 keys x D, MN-major:
                    // 8-key groups 1024 B apart, 64-column blocks one TMA box apart).
                    const uint64_t ad = fav::tc::sdesc_sw128(
                        sP + (kk >> 2) * (BM * 128) + (kk & 3) * 32, 16, 1024);
                    const uint64_t bd = fav::tc::sdesc_sw128(vst + kk * 16 * 128, BN * 128, 1024);
                    fav::tc::mma_ss(tmem + C::kColO, ad, bd, idesc_pv, (j > 0 || kk > 0));
                    if (RoundedNorm<T>::value)
                        fav::tc::mma_ss(tmem + C::kColL, ad, ones_desc, idesc_l, (j > 0 || kk > 0));
                }
                fav::tc::commit(v_empty + 8 * st);
                fav::tc::commit(p_empty);
            }
        }
    } else {
        // ---------------- softmax / correction / epilogue (one thread per row) ----------------
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;
        const int qi = q0 + row;                          // query index of this row
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
        const int lim = causal ? min(Nkv, qi + off + 1) : Nkv;   // visible keys: [0, lim)
        const int lim_tile = causal ? min(Nkv, q0 + off + 1) : Nkv;  // smallest lim in tile
        float m = -INFINITY, l = 0.f;
        bool ok = true;
        for (int j = 0; j < n_kv; ++j) {
            const uint32_t sb = j & 1;
            if (!fav::mbar_wait(s_full + 8 * sb, (j >> 1) & 1, status)) { ok = false; break; }
            fav::tc::fence_after();
            float s[BN];
            {
                const uint32_t scol = trow + (sb ? C::kColS1 : C::kColS0);
#pragma unroll
                for (int c = 0; c < BN / 32; ++c) {
                    uint32_t r[32];
                    fav::tc::ld_32x32b_x32(scol + c * 32, r);
                    fav::tc::wait_ld();
#pragma unroll
                    for (int e = 0; e < 32; ++e) s[c * 32 + e] = __uint_as_float(r[e]);
                }
            }
            fav::tc::fence_before();
            __syncwarp();
            if (lane == 0) fav::mbar_arrive(s_free + 8 * sb);

            const int key0 = j * BN;
            if (key0 + BN > lim_tile) {     // tile crosses the causal diagonal or the end
#pragma unroll
                for (int c = 0; c < BN; ++c)
                    if (key0 + c >= lim) s[c] = -INFINITY;
            }
            float mx = s[0];
#pragma unroll
            for (int c = 1; c < BN; ++c) mx = fmaxf(mx, s[c]);
            mx *= scale_log2;
            // lazy rescale: move the reference maximum only when it grows by > 2^8
            float alpha = 1.f;
            bool rescale = false;
            if (mx > m + kRescaleThreshold) {
                alpha = fav::fast_exp2(m - mx);       // 0 on the first tile (m = -inf)
                rescale = (j > 0);
                m = mx;
                l *= alpha;
            }
            uint32_t pk[BN / 2];
            const float neg_m = -m;
#pragma unroll
            for (int c = 0; c < BN; c += 2) {
                const float p0 = fav::fast_exp2(fmaf(s[c], scale_log2, neg_m));
                const float p1 = fav::fast_exp2(fmaf(s[c + 1], scale_log2, neg_m));
                l += p0 + p1;
                pk[c / 2] = fav::Elem<T>::pack(p0, p1);
            }
            // PV_{j-1} must be done: it reads the P buffer and accumulates into O.
            if (j > 0 && !fav::mbar_wait(p_empty, (j - 1) & 1, status)) { ok = false; break; }
            fav::tc::fence_after();
            if (__any_sync(~0u, rescale)) {
                constexpr int kChunks = D / 32 + (RoundedNorm<T>::value ? 1 : 0);   // O (+ l~)
#pragma unroll
                for (int c = 0; c < kChunks; ++c) {
                    uint32_t r[32];
                    fav::tc::ld_32x32b_x32(trow + C::kColO + c * 32, r);
                    fav::tc::wait_ld();
#pragma unroll
                    for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * alpha);
                    fav::tc::st_32x32b_x32(trow + C::kColO + c * 32, r);
                }
                fav::tc::wait_st();
            }
            // P row -> shared memory, K-major, 128-byte swizzle (two 64-key blocks).
#pragma unroll
            for (int cc = 0; cc < BN / 8; ++cc) {
                const uint32_t addr = sP + (cc >> 3) * (BM * 128) + row * 128 +
                                      ((((uint32_t)cc & 7u) ^ ((uint32_t)row & 7u)) << 4);
                if (!FAV_CHECK(addr >= sP && addr + 16 <= sP + C::kPBytes, status)) continue;
                asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};"
                             ::"r"(addr), "r"(pk[4 * cc]), "r"(pk[4 * cc + 1]), "r"(pk[4 * cc + 2]),
                               "r"(pk[4 * cc + 3]) : "memory");
            }
            fav::tc::fence_proxy_async_smem();
            fav::tc::fence_before();
            __syncwarp();
            if (lane == 0) fav::mbar_arrive(p_full);
        }
        // ---------------- epilogue: O / l, LSE ----------------
        if (ok && n_kv > 0 && fav::mbar_wait(p_empty, (n_kv - 1) & 1, status)) {
            fav::tc::fence_after();
            float inv_l = 1.f / l;
            if (RoundedNorm<T>::value) {
                uint32_t r[32];
                fav::tc::ld_32x32b_x32(trow + C::kColL, r);
                fav::tc::wait_ld();
                inv_l = 1.f / __uint_as_float(r[0]);
            }
            const bool valid = qi < Nq;
            T *orow = o + ((long long)bh * Nq + qi) * D;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                uint32_t r[32];
                fav::tc::ld_32x32b_x32(trow + C::kColO + c * 32, r);
                fav::tc::wait_ld();
                if (valid) {
#pragma unroll
                    for (int e = 0; e < 32; e += 8) {
                        uint4 v4;
                        v4.x = fav::Elem<T>::pack(__uint_as_float(r[e]) * inv_l, __uint_as_float(r[e + 1]) * inv_l);
                        v4.y = fav::Elem<T>::pack(__uint_as_float(r[e + 2]) * inv_l, __uint_as_float(r[e + 3]) * inv_l);
                        v4.z = fav::Elem<T>::pack(__uint_as_float(r[e + 4]) * inv_l, __uint_as_float(r[e + 5]) * inv_l);
                        v4.w = fav::Elem<T>::pack(__uint_as_float(r[e + 6]) * inv_l, __uint_as_float(r[e + 7]) * inv_l);
                        *reinterpret_cast<uint4 *>(orow + c * 32 + e) = v4;
                    }
                }
            }
            if (valid && lse) lse[(long long)bh * Nq + qi] = (m + log2f(l)) * kLn2;
        }
    }

    fav::tc::fence_before();
    __syncthreads();
    fav::tc::fence_after();
    if (warp == 1) fav::tc::tmem_dealloc(tmem, C::kTmemCols);
}

template <typename T, int D>
fav_status launch(const FavArgs &a, cudaStream_t stream) {
    using C = PrefillCfg<D>;
    alignas(64) CUtensorMap tmQ, tmK, tmV;
    fav_status st = fav_make_tmap_3d(&tmQ, a.q, D, a.Nq, a.B * a.Hq, BM);
    if (st == FAV_OK) st = fav_make_tmap_3d(&tmK, a.k, D, a.Nkv, a.B * a.Hkv, BN);
    if (st == FAV_OK) st = fav_make_tmap_3d(&tmV, a.v, D, a.Nkv, a.B * a.Hkv, BN);
    if (st != FAV_OK) return st;
    auto kern = fav_prefill_kernel<T, D>;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes) !=
        cudaSuccess)
        return FAV_ERR_CUDA;
    const int n_qtiles = (a.Nq + BM - 1) / BM;
    const long long blocks = (long long)n_qtiles * a.B * a.Hq;
    if (blocks > 0x7fffffffLL) return FAV_ERR_UNSUPPORTED;
    kern<<<(unsigned)blocks, kThreads, C::kSmemBytes, stream>>>(
        tmQ, tmK, tmV, (T *)a.o, a.lse, a.Hq, a.Hkv, a.Nq, a.Nkv, n_qtiles, a.scale * kLog2e,
        a.causal, a.dev_status);
    if (cudaGetLastError() != cudaSuccess || fav_debug_sync("fav_prefill_kernel", stream))
        return FAV_ERR_CUDA;
    return FAV_OK;
}

}  // namespace

bool fav_prefill_supported(const FavArgs &a) {
    if (a.dtype != FAV_F16 && a.dtype != FAV_BF16) return false;
    if (a.D != 64 && a.D != 128) return false;
    return (long long)a.B * a.Hq <= 0x7fffffffLL && (long long)a.B * a.Hkv <= 0x7fffffffLL;
}

fav_status fav_launch_prefill(const FavArgs &a, cudaStream_t s) {
    if (a.dtype == FAV_F16)
        return a.D == 128 ? launch<__half, 128>(a, s) : launch<__half, 64>(a, s);
    return a.D == 128 ? launch<__nv_bfloat16, 128>(a, s) : launch<__nv_bfloat16, 64>(a, s);
}
