/*
 * fav.h -- libfav: exact fused attention forward on one NVIDIA GB300 (sm_103a).
 *
 * The operation is scaled dot-product attention as defined in the FlashAttention-V paper
 * (Background section: Attention(Q,K,V) = softmax(Q K^T / sqrt(D)) V), evaluated with the
 * tiled online softmax of its Method section (Algorithm "ggml-vec FlashAttention in
 * llama.cpp" and Algorithm "FlashAttention-V for VL > D"), for multi-head, grouped-query and
 * multi-query attention (Method section on GQA), prefill (Nq = Nkv) and decode (Nq = 1).
 *
 * Conventions shared by every entry point below
 * ---------------------------------------------
 *  Layouts   q, o : [B, Hq,  Nq,  D]  contiguous row-major, element type `dtype`
 *            k, v : [B, Hkv, Nkv, D]  contiguous row-major, element type `dtype`
 *            lse  : [B, Hq,  Nq]      contiguous fp32, natural-log log-sum-exp of the scaled
 *                                      scores of each query row (may be NULL: not written)
 *  Heads     query head h reads K/V head h / (Hq / Hkv): consecutive query heads share.
 *  Causal    bottom-right aligned: query i sees keys j <= Nkv - Nq + i (needs Nq <= Nkv).
 *  Scale     applied to Q.K before the softmax; callers pass 1/sqrt(D).  Must be finite, > 0.
 *  Precision fp32 I/O: exact fp32 arithmetic.  fp16 / bf16 I/O: fp32 accumulation; on the
 *            tensor-core paths the softmax weights P are rounded (to nearest even) to the
 *            I/O type before the P.V product (the CUDA-core path keeps them in fp32);
 *            O is rounded to the I/O type once, at the end.
 *  Ownership every pointer is caller-owned; the library never frees or retains it.
 *  Errors    arguments are validated before anything is launched, so an error status
 *            leaves o and lse untouched.  There is no CPU fallback.
 */
#ifndef FAV_H
#define FAV_H

#include <stddef.h>

#if defined(__GNUC__)
#define FAV_API __attribute__((visibility("default")))
#else
#define FAV_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum { FAV_F32 = 0, FAV_F16 = 1, FAV_BF16 = 2 } fav_dtype;

typedef enum {
    FAV_OK = 0,
    FAV_ERR_INVALID_ARG = 1,    /* null or misaligned pointer, bad size, Hq % Hkv != 0, ...   */
    FAV_ERR_UNSUPPORTED = 2,    /* valid attention problem that no kernel here implements     */
    FAV_ERR_CUDA = 3,           /* a CUDA runtime call or kernel launch failed                */
    FAV_ERR_NO_MEMORY = 4,      /* the internal workspace could not be allocated              */
    FAV_ERR_DEVICE_TIMEOUT = 5, /* a bounded wait inside a kernel ran out (see below)         */
    FAV_ERR_DEVICE_CHECK = 6,   /* a check of the self-checking -DFAV_DEBUG_CHECKS build failed
                                   (an access it would have made was skipped)                 */
    FAV_ERR_BAD_PAGE = 7        /* fav_decode_paged met a block-table entry outside
                                   [0, num_pages): that page's keys were left out             */
} fav_status;

/* Kernel families (for fav_set_path / fav_last_path). */
typedef enum {
    FAV_PATH_AUTO = 0,    /* choose by dtype and shape (default)                               */
    FAV_PATH_SIMT = 1,    /* generic CUDA-core kernel, any dtype, D % 8 == 0 (D % 4 for fp32),
                             D <= 256; exact fp32 arithmetic for fp32 I/O                     */
    FAV_PATH_DECODE = 2,  /* split-KV decode kernel + log-sum-exp combine; fp16/bf16,
                             D in {64, 128}, Nq * (Hq / Hkv) <= 64 query rows per KV head
                             (taken in blocks of 16 MMA rows; auto-chosen when <= 16)         */
    FAV_PATH_PREFILL = 3  /* tcgen05 / TMEM / TMA prefill kernel; fp16/bf16, D in {64, 128}   */
} fav_path;

/*
 * fav_forward -- O = softmax(scale * Q K^T [masked]) V and LSE, asynchronously on `stream`.
 *
 *  q, k, v   device pointers (layouts above), 16-byte aligned
 *  o         device pointer, [B, Hq, Nq, D] of `dtype`, 16-byte aligned
 *  lse       device pointer [B, Hq, Nq] fp32 (4-byte aligned), or NULL
 *  B..D      sizes, all > 0; Hq % Hkv == 0; causal requires Nq <= Nkv
 *  scale     finite and > 0
 *  causal    0 or 1
 *  dtype     FAV_F32, FAV_F16 or FAV_BF16 (the type of q, k, v and o)
 *  stream    a cudaStream_t (NULL = the legacy default stream)
 *
 * Decode-shaped calls (small Nq * Hq / Hkv) split the key range over thread blocks and merge
 * the partial results with a log-sum-exp combine (associativity of the online softmax); the
 * partials live in an internal device workspace.  bf16 prefill computes P.V with fp16 weights:
 * V is first converted to fp16 in an internal workspace under a power-of-two scale per KV head
 * (exact for every element within 2^-31 of its head's largest |v|; smaller ones err by less
 * than 2^-39 of it) and O is scaled back.  Both workspaces grow on demand (cudaMallocAsync on
 * `stream`) and are kept until fav_release_workspace(); FAV_ERR_NO_MEMORY if that fails.
 * Calls on different streams of one device share them: serialise such calls.
 * Returns FAV_OK once the kernels are enqueued; it does not synchronise.
 */
FAV_API fav_status fav_forward(const void *q, const void *k, const void *v, void *o, float *lse,
                       int B, int Hq, int Hkv, int Nq, int Nkv, int D,
                       float scale, int causal, fav_dtype dtype, void *stream);

/*
 * Element strides of a [B, H, N, D] tensor whose D axis is contiguous: the distance, in
 * elements, between consecutive batches, heads and tokens.  The contiguous layout is
 * {H * N * D, N * D, D}; the heads-interleaved layout [B, N, H, D] (one token's heads stored
 * together) is {N * H * D, D, H * D}; a padded or sliced cache has larger token strides.
 */
typedef struct {
    long long batch, head, token;
} fav_strides;

/*
 * fav_forward_strided -- fav_forward on tensors given by their strides.  (Method section,
 * optimizations for VL > D: in the ggml memory layout the paper works on, the heads of one
 * token lie next to each other, [B, N, H, D], and its kernel reorders the loop over heads to
 * read that layout directly.  This entry point takes that layout, and any other with a
 * contiguous D axis, without copies.)
 *
 *  q, k, v, o   device pointers to element (0, 0, 0, 0), 16-byte aligned
 *  *_strides    element strides; each stride times the element size must be a multiple of 16
 *               bytes and below 2^40, else FAV_ERR_UNSUPPORTED.  Negative strides:
 *               FAV_ERR_INVALID_ARG.  A stride of 0 is accepted only on an axis of size 1
 *               (o: FAV_ERR_INVALID_ARG otherwise; q, k, v: FAV_ERR_UNSUPPORTED).  Distinct
 *               rows of o must not overlap (not checked otherwise).
 *  lse          [B, Hq, Nq] fp32, contiguous, or NULL
 *  other arguments and statuses as fav_forward; the call is asynchronous on `stream`.
 */
FAV_API fav_status fav_forward_strided(const void *q, const void *k, const void *v, void *o,
                                       float *lse, fav_strides q_strides, fav_strides k_strides,
                                       fav_strides v_strides, fav_strides o_strides, int B,
                                       int Hq, int Hkv, int Nq, int Nkv, int D, float scale,
                                       int causal, fav_dtype dtype, void *stream);

/*
 * fav_prefill_varlen -- prefill attention over a batch of sequences of different lengths packed
 * one after another (the cu_seqlens layout), in one launch of the persistent prefill kernel.
 * (Method / experiments: prompts of different lengths; each sequence attends only to itself.)
 *
 *  q, o           device, [total_q, Hq, D] contiguous (token-major, the heads of a token side by
 *                 side), `dtype`, 16-byte aligned; total_q = cu_seqlens_q[B]
 *  k, v           device, [total_k, Hkv, D] contiguous, `dtype`, 16-byte aligned
 *  lse            device [Hq, total_q] fp32, or NULL
 *  cu_seqlens_q,  HOST int32 [B + 1], non-decreasing from 0: sequence b's queries are rows
 *  cu_seqlens_k   cu_seqlens_q[b] .. cu_seqlens_q[b+1]-1 of q (keys likewise of k and v).  A
 *                 sequence with queries needs at least one key; causal (bottom-right aligned per
 *                 sequence) needs no more queries than keys; else FAV_ERR_INVALID_ARG.
 *  dtype, D       fp16 or bf16 with D = 64 or 128 (else FAV_ERR_UNSUPPORTED)
 *  other arguments as fav_forward.  The library builds the kernel's work list from the host
 *  arrays and copies it to a device buffer on `stream` (returning once the copy is staged);
 *  the call is otherwise asynchronous on `stream`.  total_q = 0 computes nothing.
 */
FAV_API fav_status fav_prefill_varlen(const void *q, const void *k, const void *v, void *o,
                                      float *lse, const int *cu_seqlens_q,
                                      const int *cu_seqlens_k, int B, int Hq, int Hkv, int D,
                                      float scale, int causal, fav_dtype dtype, void *stream);

/*
 * fav_decode_paged -- decode (and small-Nq) attention over a PAGED key/value cache, per sequence
 * of its own length.  (Method section: the decode stage attends one query row per head to the
 * whole cached sequence; a serving system keeps that cache in fixed-size pages shared by many
 * sequences, so the keys of one sequence are not contiguous.)
 *
 *  q, o         device, [B, Hq, Nq, D] contiguous, `dtype`, 16-byte aligned
 *  k_cache,     device page pools, [num_pages, page_size, Hkv, D] contiguous (the heads of a
 *  v_cache      token side by side), `dtype`, 16-byte aligned
 *  block_table  device int32 [B, max_pages]: key n of sequence b is row n % page_size of page
 *               block_table[b * max_pages + n / page_size].  Pages may be shared between
 *               sequences.  Entries past a sequence's length are not read.  An entry inside
 *               a sequence's length that lies outside [0, num_pages) is not dereferenced:
 *               that page's keys take no part in the softmax (a row with no other key gets
 *               O = 0, LSE = -inf) and the kernel sets FAV_ERR_BAD_PAGE in the device status
 *               word, which fav_get_last_device_status() reports.
 *  seq_lens     device int32 [B]: keys of each sequence, clamped to [0, max_pages * page_size]
 *  lse          device [B, Hq, Nq] fp32, or NULL
 *  page_size    a power of two in [16, 65536] (else FAV_ERR_UNSUPPORTED)
 *  causal       bottom-right aligned per sequence: query i of sequence b sees keys
 *               j <= seq_lens[b] - Nq + i.  A query row that sees no key (seq_lens[b] = 0, or a
 *               causal row before the start) gets O = 0 and LSE = -inf.
 *  other arguments as fav_forward, for decode-shaped calls: fp16/bf16, D in {64, 128},
 *  Nq * Hq / Hkv <= 64 (else FAV_ERR_UNSUPPORTED).  Arguments are validated before anything is
 *  launched (the device arrays' contents are not); the call is asynchronous on `stream` and
 *  uses the split-KV workspace of fav_forward (sized for max_pages * page_size keys).
 */
FAV_API fav_status fav_decode_paged(const void *q, const void *k_cache, const void *v_cache,
                                    void *o, float *lse, const int *block_table,
                                    const int *seq_lens, int B, int Hq, int Hkv, int Nq,
                                    int max_pages, int page_size, int num_pages, int D,
                                    float scale, int causal, fav_dtype dtype, void *stream);

/*
 * fav_forward_nonflash -- the same attention computed the non-fused way, as a comparison point
 * for the fused kernels (Background section, self-attention: the scores S = scale * Q K^T are
 * materialised, the masked row softmax gives P, and O = P V).  Two cuBLAS GEMMs per call
 * (batched over the KV heads of all batches; the G = Hq / Hkv query heads sharing a KV head are
 * stacked as the rows of one GEMM) and one softmax kernel of this library, which also writes
 * LSE.  The weights are fp16 (p * 2^11) for both I/O types, as on the fused tensor-core paths;
 * for bf16 I/O, V is first converted to fp16 under a power-of-two scale per KV head in an
 * internal workspace (allocated on `stream` like fav_forward's, kept until
 * fav_release_workspace) and O is scaled back and rounded to bf16 by one more kernel.
 *
 *  q, k, v, o, lse, B..dtype   as fav_forward; dtype fp16 or bf16 (else FAV_ERR_UNSUPPORTED)
 *  workspace        device buffer of at least fav_nonflash_workspace_size(B, Hq, Nq, Nkv)
 *                   bytes (the fp32 scores, then the weights in place), 16-byte aligned,
 *                   caller-owned; else FAV_ERR_INVALID_ARG
 *  workspace_bytes  its size in bytes
 *  Nkv <= 32768 (a score row lives in shared memory) and (Hq / Hkv) * Nq * Nkv < 2^31, else
 *  FAV_ERR_UNSUPPORTED.  cuBLAS (libcublas.so.13) is loaded on the first call; if it cannot
 *  be loaded the call returns FAV_ERR_UNSUPPORTED.  Asynchronous on `stream`.
 */
FAV_API size_t fav_nonflash_workspace_size(int B, int Hq, int Nq, int Nkv);
FAV_API fav_status fav_forward_nonflash(const void *q, const void *k, const void *v, void *o,
                                        float *lse, int B, int Hq, int Hkv, int Nq, int Nkv,
                                        int D, float scale, int causal, fav_dtype dtype,
                                        void *workspace, size_t workspace_bytes, void *stream);

/*
 * fav_forward_host -- the same operation on HOST buffers (end-to-end call).
 *
 * Copies q, k, v (host, ideally pinned) to internal device buffers, computes, copies o and lse
 * (lse may be NULL) back to the host, and returns when the results are on the host.  The work
 * is pipelined over up to four chunks of KV heads (batch and heads flattened), each chunk
 * copied in, computed and copied out on three internal streams, so that copies in both
 * directions overlap each other and the kernels.  It starts after the work already queued on
 * `stream` (a cudaStream_t, NULL = legacy default stream).  The device buffers grow on demand
 * and are kept until fav_release_workspace().  Host pointers need no alignment.  Same argument
 * rules and statuses as fav_forward.
 */
FAV_API fav_status fav_forward_host(const void *q, const void *k, const void *v, void *o, float *lse,
                            int B, int Hq, int Hkv, int Nq, int Nkv, int D,
                            float scale, int causal, fav_dtype dtype, void *stream);

/* A short English description of a status code (static storage, never NULL). */
FAV_API const char *fav_status_string(fav_status s);

/*
 * fav_get_last_device_status -- synchronises the device, then reports and clears the status
 * word that kernels set: FAV_ERR_DEVICE_TIMEOUT when one of their bounded waits (on an
 * mbarrier) gave up, FAV_ERR_BAD_PAGE when fav_decode_paged met an out-of-range block-table
 * entry, FAV_ERR_DEVICE_CHECK when a check of the self-checking build failed; FAV_OK if none
 * did since the last call (the last one set wins).  FAV_ERR_CUDA if the device could not be
 * queried.
 */
FAV_API fav_status fav_get_last_device_status(void);

/* Frees the internal workspace and host-call buffers of the current device (synchronises). */
FAV_API void fav_release_workspace(void);

/*
 * fav_set_path -- process-wide override of the kernel family (FAV_PATH_AUTO restores the
 * default choice).  A forced path that cannot run a given call makes fav_forward return
 * FAV_ERR_UNSUPPORTED.  Intended for tests and measurements.
 */
FAV_API fav_status fav_set_path(fav_path p);

/* The kernel family used by the last successful fav_forward call of this process. */
FAV_API fav_path fav_last_path(void);

/*
 * fav_set_decode_splits -- process-wide number of key-range splits for the decode path
 * (0 = automatic, from the problem size and the SM count).  Values are clamped to the number
 * of key tiles.  FAV_ERR_INVALID_ARG for n < 0 or n > 4096.
 */
FAV_API fav_status fav_set_decode_splits(int n);

/* The split count the last decode-path fav_forward call used (0 if none ran yet). */
FAV_API int fav_last_decode_splits(void);

/*
 * fav_set_prefill_grid -- process-wide cap on the number of thread blocks of the persistent
 * prefill kernel (0 = automatic: one per SM, at most one per query tile).  With a small cap
 * each block works through many query tiles in turn, which tests use to exercise that path on
 * small problems.  The results do not depend on the cap.  FAV_ERR_INVALID_ARG for n < 0.
 */
FAV_API fav_status fav_set_prefill_grid(int n);

/*
 * fav_check_wait_timeout -- self-test of the kernels' bounded waits (no counterpart in the
 * paper: it checks this library's failure reporting).  Launches one warp on `stream` that
 * waits on a shared-memory mbarrier that nothing ever arrives on, with the same wait code as
 * the kernels but a give-up limit of limit_us microseconds instead of their 2 s.  The wait gives
 * up, records FAV_ERR_DEVICE_TIMEOUT in the device status word and the kernel returns normally
 * (no copy or tensor-core operation is in flight, the context stays usable); read the outcome
 * with fav_get_last_device_status(), which also clears it.  Asynchronous.
 * FAV_ERR_INVALID_ARG unless 1 <= limit_us <= 1000000; FAV_ERR_CUDA if the launch failed.
 */
FAV_API fav_status fav_check_wait_timeout(int limit_us, void *stream);

/*
 * fav_decode_noalloc -- the decode path (split-KV decode kernel + log-sum-exp combine) with no
 * device allocation at all.  The paper has no counterpart: this entry point exists for callers
 * that cannot let a library allocate device memory -- a server whose own pool reserves all
 * device memory at start-up (a library cudaMalloc would fail or compete with it), or a
 * latency-critical decode loop that forbids allocator calls after initialisation.
 *
 * Same arguments, layouts, ownership and status codes as fav_forward, for decode-shaped calls
 * (fp16/bf16, D in {64, 128}, Nq * Hq / Hkv <= 64); the result equals fav_forward's on the
 * decode path.  The split-KV partials live in a fixed file-scope device array of
 * FAV_NOALLOC_SCRATCH_BYTES (16 MiB), held by every GPU that loads the library until the
 * process exits.  The split count is fav_forward's (automatic, or fav_set_decode_splits);
 * FAV_ERR_UNSUPPORTED if its partials, B*Hq*Nq * splits * (D + 1) * 4 bytes, exceed the array,
 * or if the call is not decode-shaped.  The first call on each device (with that device
 * current) looks up the array's device address; make that first call before any stream
 * capture.  Every call shares the array: calls that overlap on the GPU (several streams at
 * once) race and must be serialised by the caller.  Never calls cudaMalloc, cudaMallocAsync,
 * cudaFree or any allocating library routine.
 */
#define FAV_NOALLOC_SCRATCH_BYTES (16u * 1024u * 1024u)
FAV_API fav_status fav_decode_noalloc(const void *q, const void *k, const void *v, void *o,
                                      float *lse, int B, int Hq, int Hkv, int Nq, int Nkv,
                                      int D, float scale, int causal, fav_dtype dtype,
                                      void *stream);

#ifdef __cplusplus
}
#endif

#endif /* FAV_H */
