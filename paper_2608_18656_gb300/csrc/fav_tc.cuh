// fav_tc.cuh -- tcgen05 (5th-generation tensor core) building blocks in inline PTX:
// tensor-memory allocation, shared-memory matrix descriptors, instruction descriptors,
// MMA issue / commit, and tensor-memory loads and stores.
#pragma once
#include <stdint.h>

namespace fav {
namespace tc {

// ---- tensor memory allocation (one full warp) ----
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 ::"r"(dst_smem), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;"
                 ::"r"(taddr), "r"(ncols) : "memory");
}

// ---- ordering of tcgen05 operations around thread synchronisation ----
__device__ __forceinline__ void fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// Generic-proxy shared-memory writes become visible to the async proxy (MMA operand reads).
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ---- descriptors ----
// Shared-memory matrix descriptor: start address, leading / stride byte offsets (16-byte
// units), descriptor version 1, 128-byte swizzle.  The swizzle atom is 8 rows of 128 bytes
// (1024 bytes); operand tiles start on 1024-byte boundaries.
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// Instruction descriptor for kind::f16: fp32 accumulator, A/B both fp16 or both bf16,
// A K-major, B K-major (b_mn_major = false) or MN-major, shape M x N.
__host__ __device__ constexpr uint32_t idesc_f16(int M, int N, bool bf16, bool b_mn_major) {
    return (1u << 4) | ((bf16 ? 1u : 0u) << 7) | ((bf16 ? 1u : 0u) << 10) |
           ((b_mn_major ? 1u : 0u) << 16) | ((uint32_t)(N >> 3) << 17) |
           ((uint32_t)(M >> 4) << 24);
}

// D[tmem] (+)= A[smem] * B[smem]; issued by one thread.
__device__ __forceinline__ void mma_ss(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                       uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
        ::"r"(d_tmem), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// D[tmem] (+)= A[tmem] * B[smem]; A (M x 16 of 16-bit elements) is read from tensor memory,
// one row per lane, two elements per 32-bit column.  Issued by one thread.
__device__ __forceinline__ void mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc,
                                       uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}"
        ::"r"(d_tmem), "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive once on `bar` when every tcgen05 operation issued so far by this thread completes.
__device__ __forceinline__ void commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];"
                 ::"r"(bar) : "memory");
}

// ---- warp-converged MMA bursts ----
// The whole (converged) warp executes these.  elect.sync inside the asm block picks one lane,
// which issues every MMA of the burst back to back; the k-step offsets are immediates.
// Measured on GB300 with two FMA-bound warps on the issuing warp's scheduler: 64-65 cycles per
// M128 N128 K16 MMA in this form, against 96-154 cycles when one lane, branched off from its
// warp, issued the same MMAs one asm statement at a time (the issuing thread waits for each
// MMA to be accepted, so every slot the other warps take from it between two MMAs idles the
// tensor pipe).

// After a burst, the issuing lane commits to barrier %5 and then %6 (shared-memory addresses;
// 0 = no commit): each arrives once when every MMA this lane issued so far has completed.
#define FAV_MMA_COMMITS                                                          \
    "setp.ne.and.b32 ca, %5, 0, e;\n\tsetp.ne.and.b32 cb, %6, 0, e;\n\t"       \
    "@ca tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%5];\n\t" \
    "@cb tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%6];\n\t"

#define FAV_MMA_SS_STEP(OFF)                                                     \
    "add.s64 a1, %1, " #OFF ";\n\tadd.s64 b1, %2, " #OFF ";\n\t"                 \
    "@e tcgen05.mma.cta_group::1.kind::f16 [%0], a1, b1, %3, t;\n\t"

// D (+)= A B^T over NK k-steps of 16, A and B both K-major 128-row tiles with 128-byte swizzle
// stored as 64-element-wide boxes of 128 rows (16 KB apart): k-step kk starts (kk % 4) * 32
// bytes into box kk / 4.  `acc` = 0 overwrites D with the first k-step.
template <int NK>
__device__ __forceinline__ void mma_ss_burst_k128(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                                  uint32_t idesc, uint32_t acc,
                                                  uint32_t bar_a = 0, uint32_t bar_b = 0) {
    static_assert(NK == 4 || NK == 8, "k-steps per burst");
    if constexpr (NK == 4) {
        asm volatile(
            "{\n\t.reg .pred e, p, t, ca, cb;\n\t.reg .b64 a1, b1;\n\t"
            "elect.sync _|e, 0xffffffff;\n\tsetp.ne.b32 p, %4, 0;\n\tsetp.eq.b32 t, %4, %4;\n\t"
            "@e tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t"
            FAV_MMA_SS_STEP(2) FAV_MMA_SS_STEP(4) FAV_MMA_SS_STEP(6)
            FAV_MMA_COMMITS
            "}"
            ::"r"(d_tmem), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(acc), "r"(bar_a), "r"(bar_b)
            : "memory");
    } else {
        asm volatile(
            "{\n\t.reg .pred e, p, t, ca, cb;\n\t.reg .b64 a1, b1;\n\t"
            "elect.sync _|e, 0xffffffff;\n\tsetp.ne.b32 p, %4, 0;\n\tsetp.eq.b32 t, %4, %4;\n\t"
            "@e tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t"
            FAV_MMA_SS_STEP(2) FAV_MMA_SS_STEP(4) FAV_MMA_SS_STEP(6)
            FAV_MMA_SS_STEP(1024) FAV_MMA_SS_STEP(1026) FAV_MMA_SS_STEP(1028) FAV_MMA_SS_STEP(1030)
            FAV_MMA_COMMITS
            "}"
            ::"r"(d_tmem), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(acc), "r"(bar_a), "r"(bar_b)
            : "memory");
    }
}
#undef FAV_MMA_SS_STEP

#define FAV_MMA_TS_STEP(AOFF, BOFF)                                              \
    "add.u32 ta, %1, " #AOFF ";\n\tadd.s64 b1, %2, " #BOFF ";\n\t"               \
    "@e tcgen05.mma.cta_group::1.kind::f16 [%0], [ta], b1, %3, t;\n\t"

// D (+)= A B over 8 k-steps of 16 (K = 128): A (M x 128 of 16-bit elements) read from TMEM,
// 8 columns per k-step; B MN-major in shared memory, 16 rows of 128 bytes (2048 B) per k-step.
// `acc` = 0 overwrites D with the first MMA.
__device__ __forceinline__ void mma_ts_burst_k128(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc,
                                                  uint32_t idesc, uint32_t acc,
                                                  uint32_t bar_a = 0, uint32_t bar_b = 0) {
    asm volatile(
        "{\n\t.reg .pred e, p, t, ca, cb;\n\t.reg .b32 ta;\n\t.reg .b64 b1;\n\t"
        "elect.sync _|e, 0xffffffff;\n\tsetp.ne.b32 p, %4, 0;\n\tsetp.eq.b32 t, %4, %4;\n\t"
        "@e tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t"
        FAV_MMA_TS_STEP(8, 128) FAV_MMA_TS_STEP(16, 256) FAV_MMA_TS_STEP(24, 384)
        FAV_MMA_TS_STEP(32, 512) FAV_MMA_TS_STEP(40, 640) FAV_MMA_TS_STEP(48, 768)
        FAV_MMA_TS_STEP(56, 896)
        FAV_MMA_COMMITS
        "}"
        ::"r"(d_tmem), "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(acc), "r"(bar_a), "r"(bar_b)
        : "memory");
}
#undef FAV_MMA_TS_STEP

// One step of a split P.V burst: D at %0 + DOFF columns, A (weights) at %1 + AOFF columns, B
// at descriptor %2 + BOFF (16-byte units), accumulate predicate PRED.
#define FAV_MMA_PV_STEP(DOFF, AOFF, BOFF, PRED)                                  \
    "add.u32 td, %0, " #DOFF ";\n\tadd.u32 ta, %1, " #AOFF ";\n\t"           \
    "add.s64 b1, %2, " #BOFF ";\n\t"                                          \
    "@e tcgen05.mma.cta_group::1.kind::f16 [td], [ta], b1, %3, " #PRED ";\n\t"

// O_s (+)= P_s V_s for the NSPLIT (= 2) key splits of a 128-key tile, in one burst: split s has its
// own accumulator of D columns at d_tmem + s * D, its weights (128 / NSPLIT keys, two per
// column) at a_tmem + s * (128 / NSPLIT) and its V rows (MN-major, 128 bytes per key row) at
// s * (128 / NSPLIT) * 128 bytes past bdesc.  k-steps of 16 keys: A +8 columns, B +2048 bytes.
// `acc` = 0 overwrites each accumulator with its first MMA.
template <int NSPLIT>
__device__ __forceinline__ void mma_pv_split(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc,
                                             uint32_t idesc, uint32_t acc, uint32_t bar_a = 0,
                                             uint32_t bar_b = 0) {
    static_assert(NSPLIT == 2, "key splits (D = 128)");
    if constexpr (NSPLIT == 2) {   // D = 128: 64 keys per split, 4 k-steps
        asm volatile(
            "{\n\t.reg .pred e, p, t, ca, cb;\n\t.reg .b32 td, ta;\n\t.reg .b64 b1;\n\t"
            "elect.sync _|e, 0xffffffff;\n\tsetp.ne.b32 p, %4, 0;\n\tsetp.eq.b32 t, %4, %4;\n\t"
            FAV_MMA_PV_STEP(0, 0, 0, p) FAV_MMA_PV_STEP(0, 8, 128, t)
            FAV_MMA_PV_STEP(0, 16, 256, t) FAV_MMA_PV_STEP(0, 24, 384, t)
            FAV_MMA_PV_STEP(128, 64, 512, p) FAV_MMA_PV_STEP(128, 72, 640, t)
            FAV_MMA_PV_STEP(128, 80, 768, t) FAV_MMA_PV_STEP(128, 88, 896, t)
            FAV_MMA_COMMITS
            "}"
            ::"r"(d_tmem), "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(acc), "r"(bar_a), "r"(bar_b)
            : "memory");
    }
}

#undef FAV_MMA_PV_STEP
#undef FAV_MMA_COMMITS

// commit() from a converged warp: one elected lane commits.
__device__ __forceinline__ void commit_elect(uint32_t bar) {
    asm volatile(
        "{\n\t.reg .pred e;\n\telect.sync _|e, 0xffffffff;\n\t"
        "@e tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n\t}"
        ::"r"(bar) : "memory");
}

// ---- tensor memory <-> registers: 32 lanes x 32 consecutive 32-bit columns ----
__device__ __forceinline__ void ld_32x32b_x32(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
          "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
          "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
          "=r"(r[31])
        : "r"(taddr));
}

// 32 lanes x 64 consecutive 32-bit columns in one load (one instruction in the scheduler's
// memory-instruction queue instead of two; that queue also holds the MMA warp's pending MMAs).
__device__ __forceinline__ void ld_32x32b_x64(uint32_t taddr, uint32_t (&r)[64]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x64.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31,"
        "%32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63}, [%64];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
          "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]),
          "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]),
          "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
          "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
        : "r"(taddr));
}

__device__ __forceinline__ void wait_ld_dep(uint32_t (&r)[64]) {
    asm volatile(
        "tcgen05.wait::ld.sync.aligned;"
        : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
          "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15]),
          "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]),
          "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]), "+r"(r[30]), "+r"(r[31]),
          "+r"(r[32]), "+r"(r[33]), "+r"(r[34]), "+r"(r[35]), "+r"(r[36]), "+r"(r[37]), "+r"(r[38]), "+r"(r[39]),
          "+r"(r[40]), "+r"(r[41]), "+r"(r[42]), "+r"(r[43]), "+r"(r[44]), "+r"(r[45]), "+r"(r[46]), "+r"(r[47]),
          "+r"(r[48]), "+r"(r[49]), "+r"(r[50]), "+r"(r[51]), "+r"(r[52]), "+r"(r[53]), "+r"(r[54]), "+r"(r[55]),
          "+r"(r[56]), "+r"(r[57]), "+r"(r[58]), "+r"(r[59]), "+r"(r[60]), "+r"(r[61]), "+r"(r[62]), "+r"(r[63])
        :
        : "memory");
}

__device__ __forceinline__ void st_32x32b_x32(uint32_t taddr, const uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};"
        ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]),
          "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]),
          "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]),
          "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]),
          "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}

// 32 lanes x 16 consecutive 32-bit columns.
__device__ __forceinline__ void ld_32x32b_x16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}

__device__ __forceinline__ void st_32x32b_x16(uint32_t taddr, const uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};"
        ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]),
          "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]),
          "r"(r[13]), "r"(r[14]), "r"(r[15])
        : "memory");
}

__device__ __forceinline__ void wait_ld_dep(uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.wait::ld.sync.aligned;"
        : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]),
          "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]),
          "+r"(r[13]), "+r"(r[14]), "+r"(r[15])
        :
        : "memory");
}

__device__ __forceinline__ void wait_ld() {
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
// Waits like wait_ld and ties the 32 registers of one tcgen05.ld to the wait, so that no use
// of them can be scheduled before it.
__device__ __forceinline__ void wait_ld_dep(uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.wait::ld.sync.aligned;"
        : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]),
          "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]),
          "+r"(r[13]), "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]),
          "+r"(r[19]), "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]), "+r"(r[24]),
          "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]), "+r"(r[30]),
          "+r"(r[31])
        :
        : "memory");
}
__device__ __forceinline__ void wait_st() {
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

}  // namespace tc
}  // namespace fav
