/*
 * sq.h — C ABI of libsq, the GB300 (sm_103a) hot path behind SideQuest's
 * model-driven KV-cache management (Kariyappa & Suh, "SideQuest: Model-Driven
 * KV Cache Management for Long-Horizon Agentic Reasoning").
 *
 * The library keeps a paged bf16 KV pool on one GPU.  A main reasoning
 * sequence and the auxiliary sequences forked from it share their prefix
 * pages (reference-counted, copy-on-write); decode attention reads the pages
 * through per-sequence page tables; span eviction removes cursor-identified
 * message spans and compacts the surviving rows in place.
 *
 * Conventions for every call:
 *   - Return value: SQ_OK (0) or one of the negative SQ_ERR_* codes below.
 *   - On any error the host-side state (sequences, page tables, reference
 *     counts, free pages) is left exactly as it was before the call.
 *   - Device work is enqueued asynchronously on the `stream` argument
 *     (a cudaStream_t passed as void*; NULL = the legacy default stream).
 *     Nothing is copied back to the host; device-side faults detected by
 *     the kernels' own checks are reported by sq_sync_status().
 *   - Pointers named "device" must point to GPU memory of the cache's device;
 *     pointers named "host" to CPU memory.  The caller keeps ownership of all
 *     buffers it passes; the library never frees them.  Device input buffers
 *     must stay valid until the enqueued work has run.
 *   - A cache is not thread-safe: one host thread issues its calls.  Calls
 *     may use different streams; the caller orders work on one sequence
 *     (e.g. evicting a sequence after its own decode on another stream,
 *     Sec. 3.1 step 4: eviction waits for the main thread's current turn).
 *
 * KV pool layout (bf16, 16-bit elements), for layer l, page p, plane kv
 * (0 = K, 1 = V), KV head h, slot s, dimension e:
 *     pool[((((l * num_pages + p) * 2 + kv) * num_kv_heads + h) * page_size
 *           + s) * head_dim + e]
 * Logical token j of a sequence lives in slot j % page_size of page
 * page_table[j / page_size].
 */
#ifndef SQ_H_
#define SQ_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SQ_API __attribute__((visibility("default")))
#else
#define SQ_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Opaque cache object, owned by the library. */
typedef struct sq_cache sq_cache;

/* Sequence handle: slot | generation << 20; always > 0.  A released
 * handle is rejected with SQ_ERR_BAD_HANDLE. */
typedef int32_t sq_seq;

/* A half-open span [start, end) of CURRENT logical token positions of one
 * sequence — the tokens of a tool call and its response (Sec. 3, Goal and
 * its footnote; Algorithm 1, C.clear_kv(Delta_ids)).  The caller maps the
 * auxiliary thread's cursor ids to spans. */
typedef struct {
    int32_t start;
    int32_t end;
} sq_span;

typedef struct {
    int32_t num_layers;        /* L   >= 1 */
    int32_t num_q_heads;       /* Hq  >= 1, multiple of num_kv_heads */
    int32_t num_kv_heads;      /* Hkv >= 1; Hq / Hkv <= 16 */
    int32_t head_dim;          /* d: 64 or 128 */
    int32_t page_size;         /* P: power of two, 8 .. 256 */
    int32_t num_pages;         /* pages in the pool (each holds P tokens of every layer) */
    int32_t max_seqs;          /* live sequences at most (<= 2^20 - 1) */
    int32_t max_pages_per_seq; /* page-table capacity of one sequence */
    void *kv_pool;             /* device; NULL = the library allocates (and zeroes) the
                                  pool; else caller memory of sq_pool_bytes() bytes,
                                  256-byte aligned, owned by the caller */
    int32_t decode_ctas;       /* 0 = automatic (SMs x resident CTAs per SM); else the
                                  number of persistent CTAs decode attention uses
                                  (a decode call that would split one sequence's KV
                                  head over more than 65,535 of them returns
                                  SQ_ERR_CAPACITY) */
} sq_config;

enum {
    SQ_OK = 0,
    SQ_ERR_INVALID_ARG = -1,     /* a bad pointer, size, span, dtype or layer */
    SQ_ERR_BAD_HANDLE = -2,      /* unknown or released sequence / cache */
    SQ_ERR_NO_PAGES = -3,        /* the pool has too few free pages */
    SQ_ERR_CAPACITY = -4,        /* a sequence would exceed max_pages_per_seq,
                                    or max_seqs sequences are live */
    SQ_ERR_CUDA = -5,            /* a CUDA runtime call failed */
    SQ_ERR_DEVICE = -6,          /* a kernel's own bounds check fired */
    SQ_ERR_DEVICE_TIMEOUT = -7,  /* a kernel's bounded wait ran out */
    SQ_ERR_UNSUPPORTED = -8,     /* a geometry this build does not handle */
    SQ_ERR_NO_MEMORY = -9        /* host or device allocation failed */
};

enum { SQ_OUT_BF16 = 0, SQ_OUT_F32 = 1 };

/* Bytes of the KV pool for a configuration (0 if it is invalid). */
SQ_API size_t sq_pool_bytes(const sq_config *cfg);

/* Create a cache on the current CUDA device.  *out receives the handle.
 * Paper: Sec. 3.4 (Storage Costs) — one pool shared by the main and
 * auxiliary threads.  Errors: INVALID_ARG, UNSUPPORTED, NO_MEMORY, CUDA. */
SQ_API int sq_cache_create(const sq_config *cfg, sq_cache **out);

/* Destroy a cache (synchronises the device first; frees library memory). */
SQ_API int sq_cache_destroy(sq_cache *cache);

/* A new, empty main sequence (Algorithm 1: C <- [Q] starts empty here and
 * the query tokens are appended).  Errors: CAPACITY. */
SQ_API int sq_seq_new(sq_cache *cache, sq_seq *out);

/* Append n_tokens K/V rows to the end of `seq` (Algorithm 1: C <- C + R,
 * C <- C + O; the aux thread's C_aux <- C + p).
 *   k, v: device, bf16, contiguous [num_layers][n_tokens][num_kv_heads][head_dim]
 *         (keys already rotated: the library never applies positional
 *         encodings).
 * If the sequence's last page is partial and shared with another sequence it
 * is first copied (copy-on-write); then fresh pages are taken, lowest free id
 * first, in increasing logical order.  n_tokens == 0 is a no-op.
 * Cached decode plans holding `seq`, last used on `stream`, stay valid when
 * the rows fit in the last page and its 64-token stage (pages of >= 64
 * tokens): the launch rewrites the plan's row limit for the sequence, so the
 * next sq_decode_attention on `stream` reuses the plan without an upload.
 * Errors: BAD_HANDLE, INVALID_ARG, NO_PAGES, CAPACITY, CUDA. */
SQ_API int sq_append_kv(sq_cache *cache, sq_seq seq, int32_t n_tokens, const void *k,
                 const void *v, void *stream);

/* Append one token to each of n_seqs sequences in one launch (a decode step
 * of a batch; Algorithm 1: C <- C + R one generated token at a time).
 *   seqs: host, n_seqs distinct live handles
 *   k, v: device, bf16, contiguous [num_layers][n_seqs][num_kv_heads][head_dim]:
 *         row i belongs to seqs[i]
 * Same page rules (and the same reuse of cached decode plans) as
 * sq_append_kv, sequence by sequence in the order given; all or nothing: on
 * any error no sequence changes.
 * Errors: BAD_HANDLE, INVALID_ARG, NO_PAGES, CAPACITY, CUDA. */
SQ_API int sq_append_kv_batch(sq_cache *cache, const sq_seq *seqs, int32_t n_seqs,
                              const void *k, const void *v, void *stream);

/* Fork an auxiliary sequence that shares the whole context of `parent`
 * (Sec. 3.1 step 1; Algorithm 1 phase 2, C_aux <- C + p; Sec. 3.4: the
 * auxiliary thread does not duplicate the KV cache).  The child gets the same
 * page ids and token count; every page's reference count grows by one; no
 * K/V byte is copied and no device work is enqueued.
 * Errors: BAD_HANDLE, CAPACITY. */
SQ_API int sq_fork_aux(sq_cache *cache, sq_seq parent, sq_seq *child_out);

/* Decode attention for one new query token of each of n_seqs sequences at
 * layer `layer` (Sec. 1 and Sec. 3.4: attention reads the whole KV cache of
 * the context for every generated token; Sec. 2.1: grouped-query attention).
 * For sequence i, query head h and KV head g = h / (Hq / Hkv):
 *     out[i][h] = sum_t softmax_t(sm_scale * q[i][h] . K_g[t]) V_g[t]
 * over all n_i tokens of the sequence in logical order.
 *   seqs: host, n_seqs distinct live handles, each with >= 1 token
 *   q:    device, bf16 [n_seqs][num_q_heads][head_dim]
 *   out:  device, [n_seqs][num_q_heads][head_dim], bf16 (SQ_OUT_BF16, round
 *         to nearest even) or fp32 (SQ_OUT_F32); must not overlap q (rows are
 *         written while other rows' queries are still being read): an
 *         overlap is INVALID_ARG
 * Sequences that share pages (a main thread and its forks) in one call read
 * each shared page once for all of them (Sec. 3.4, shared-context kernels).
 * Errors: BAD_HANDLE, INVALID_ARG, CAPACITY, NO_MEMORY, CUDA. */
SQ_API int sq_decode_attention(sq_cache *cache, const sq_seq *seqs, int32_t n_seqs,
                        int32_t layer, const void *q, void *out,
                        int32_t out_dtype, float sm_scale, void *stream);

/* Evict spans from `seq` (Algorithm 1 phase 1, C.clear_kv(Delta_ids);
 * Sec. 3.1 step 3).  The kept tokens keep their order and their K/V bytes
 * (keys are never re-rotated); row j of the result is the j-th kept row.
 *   spans: host, n_spans half-open spans of current positions, any order;
 *          empty, overlapping or out-of-range spans are INVALID_ARG;
 *          n_spans == 0 is a no-op.
 * The kept rows are packed into full pages (every page full but the last;
 * a sequence that had partial pages from sq_evict_spans_ragged is packed
 * too).  Pages whose contents change and that are shared with another
 * sequence are replaced by fresh pages (copy-on-write, increasing logical
 * page order); others are compacted in place; pages past the new end are
 * released.
 * Errors: BAD_HANDLE, INVALID_ARG, NO_PAGES, NO_MEMORY, CUDA. */
SQ_API int sq_evict_spans(sq_cache *cache, sq_seq seq, const sq_span *spans,
                   int32_t n_spans, void *stream);

/* The same eviction (Algorithm 1 phase 1, C.clear_kv; same arguments, same
 * logical result) with work proportional to the spans instead of the
 * sequence: pages the spans do not touch keep their rows; each maximal run
 * of touched pages (a window) has its kept rows packed from slot 0 of its
 * first page, and its pages that are no longer needed leave the sequence by
 * remapping alone, without a copy.  About P rows per span are copied.  The
 * last page of each window may stay partial: every page then carries its own
 * fill (sq_get_page_fill), which decode and prefill attention honour, and
 * appends still go to the sequence's last page.  When a window's last page
 * is written, its slots past the fill are set to zero.  Copy-on-write, page
 * release and error behaviour as for sq_evict_spans.
 * Errors: BAD_HANDLE, INVALID_ARG, NO_PAGES, NO_MEMORY, CUDA. */
SQ_API int sq_evict_spans_ragged(sq_cache *cache, sq_seq seq, const sq_span *spans,
                                 int32_t n_spans, void *stream);

/* Masked prefill attention (Algorithm 2, BuildMask; Sec. 3.3): the
 * training-time counterpart of span eviction.  The last n_q tokens of `seq`
 * (already appended) are the queries; query i sits at logical position
 * p = n - n_q + i and attends causally to the sequence's tokens 0 .. p,
 * except the tokens inside `spans`, which no query sees (a closed cursor's
 * tokens masked out for the whole trace).  With GQA, query head h reads KV
 * head floor(h / G):
 *     o[i][h] = sum_j softmax_j(sm_scale * q[i][h] . K[j]) V[j]   over visible j
 *   q:   device bf16 [n_q][Hq][head_dim], 16-byte aligned, caller-owned;
 *        row i is the query of position n - n_q + i (post-RoPE, like K);
 *   out: device [n_q][Hq][head_dim], SQ_OUT_BF16 (round to nearest even) or
 *        SQ_OUT_F32, 16-byte aligned;
 *   lse: NULL, or device float [n_q][Hq], 4-byte aligned: the natural log of
 *        sum_j exp(sm_scale * q . K[j]) over the visible keys (for a backward
 *        pass or for merging with other key ranges);
 *   q, out and lse must not overlap one another (INVALID_ARG);
 *   sm_scale: finite, >= 0;
 *   spans: host, n_spans half-open spans of current positions, any order;
 *          empty, overlapping or out-of-range spans are INVALID_ARG;
 *          n_spans == 0 is plain causal attention.
 * A query that sees no token (every key up to it masked) gets a zero output
 * and lse = -infinity.  On a sequence with partial pages (sq_evict_spans_ragged)
 * the n_q queries must lie in consecutive page slots, that is no partial page
 * may hold one of them but the last (true for rows appended after the last
 * ragged eviction); otherwise UNSUPPORTED.  The sequence and the cache are
 * not modified.  The
 * kernel runs on the tensor cores (bf16 products, fp32 accumulation; the
 * softmax weights are rounded to bf16 before the value product, and the
 * normaliser sums the same rounded weights).
 * Errors: BAD_HANDLE, INVALID_ARG, UNSUPPORTED, NO_MEMORY, CUDA. */
SQ_API int sq_prefill_attention(sq_cache *cache, sq_seq seq, int32_t layer, int32_t n_q,
                                const void *q, void *out, int32_t out_dtype, float *lse,
                                float sm_scale, const sq_span *spans, int32_t n_spans,
                                void *stream);

/* Release a sequence (Algorithm 1: S_thread <- None; Sec. 3.4: the
 * auxiliary thread's own tokens are discarded).  Every page loses one
 * reference; pages that reach zero become free once all work enqueued on
 * `stream` (and on the stream that last used the sequence) before this call
 * has completed — later work on other streams that takes them waits for it.
 * Errors: BAD_HANDLE, CUDA. */
SQ_API int sq_release(sq_cache *cache, sq_seq seq, void *stream);

/* ---- inspection helpers (host-side, no device work) ---- */

/* Token count and page count of a sequence. */
SQ_API int sq_seq_info(sq_cache *cache, sq_seq seq, int32_t *n_tokens,
                int32_t *n_pages);

/* Position of the sequence's next token: the number of tokens ever appended
 * to it, counting from its parent's at fork time.  Span eviction (Algorithm 1,
 * clear_kv) lowers the token count but not this: the library stores keys after
 * the rotary embedding and never re-rotates them, so kept keys keep the phase
 * of their original positions and a new token continues after the last
 * position handed out (a reading: the paper does not discuss positions after
 * eviction).  Errors: BAD_HANDLE, INVALID_ARG (out is NULL). */
SQ_API int sq_seq_next_pos(sq_cache *cache, sq_seq seq, int64_t *out);

/* Copy the page table of `seq` into host_out[0 .. cap); *n_out = its length.
 * Errors: BAD_HANDLE, INVALID_ARG (cap too small). */
SQ_API int sq_get_page_table(sq_cache *cache, sq_seq seq, int32_t *host_out,
                      int32_t cap, int32_t *n_out);

/* Copy the fill of every page of `seq` (rows it holds, 1 .. page_size, in
 * its first slots; the sequence's rows are the pages' filled slots in page
 * order) into host_out[0 .. cap); *n_out = the page count.  Every page is
 * full but the last unless sq_evict_spans_ragged left partial pages.
 * Errors: BAD_HANDLE, INVALID_ARG (cap too small). */
SQ_API int sq_get_page_fill(sq_cache *cache, sq_seq seq, int32_t *host_out,
                            int32_t cap, int32_t *n_out);

/* Reference count of a page (0 = free). */
SQ_API int sq_page_refcount(sq_cache *cache, int32_t page, int32_t *out);

/* Number of free pages. */
SQ_API int sq_free_pages(sq_cache *cache, int32_t *out);

/* Device pointer of the KV pool (layout above). */
SQ_API int sq_pool_ptr(sq_cache *cache, void **out);

typedef struct {
    int64_t live_pages;          /* pages with a nonzero reference count now */
    int64_t peak_live_pages;     /* Sec. 4.5, Peak Token Utilization (in pages) */
    int64_t decode_calls;
    int64_t decode_logical_bytes;/* Sec. 4.5, KV Cache Memory Reads: sum over calls
                                    and sequences of tokens x 2 x Hkv x d x 2 B */
    int64_t decode_unique_bytes; /* the same with pages shared inside one call
                                    counted once */
    int64_t evict_calls;
    int64_t evicted_tokens;
    int64_t evict_moved_rows;    /* token rows rewritten (all layers/planes count once) */
    int64_t evict_bytes;         /* algorithmic bytes read + written by compaction */
    int64_t appended_tokens;
    int64_t cow_pages;           /* pages copied on write (append + evict) */
    int64_t prefill_calls;
    int64_t prefill_pairs;       /* visible (query, key) pairs per query head,
                                    summed over prefill calls */
    int64_t decode_early_calls;  /* decode calls that loaded their first stages before
                                    waiting for the preceding kernel */
    int64_t decode_early_held;   /* pages those calls left for after the wait (a write
                                    to them not yet known complete) */
    int64_t decode_plans_built;  /* sq_decode_attention calls that planned and uploaded a
                                    plan (the others reused a cached one, also after
                                    appends that stayed inside a sequence's last page and
                                    stage); sq_decode_attention_noalloc plans every call
                                    and is not counted here */
} sq_stats_t;

SQ_API int sq_stats(sq_cache *cache, sq_stats_t *out);

/* ---- allocation-free decode (the paper has no counterpart) ---- */

/* Bytes of the fixed device scratch behind sq_decode_attention_noalloc. */
#define SQ_NOALLOC_SCRATCH_BYTES (32u << 20)

/* The same decode attention as sq_decode_attention (same arguments, same
 * kernels, same result), for callers that may not allocate GPU memory while
 * decoding: runtimes that reserve the device for their KV pool up front and
 * forbid allocations on the hot path, or hosts whose device allocator cannot
 * be reached from C.  This call allocates no device memory — no cudaMalloc,
 * no cudaFree, no library allocator.  The call's split-K plan and partial
 * results go to a fixed scratch array of SQ_NOALLOC_SCRATCH_BYTES that is
 * part of the library's device image.
 *   - sq_cache_create makes that array resident on the cache's device (its
 *     device address is looked up there, which loads it; it then stays until
 *     the process exits) and allocates two pinned host buffers of 2 MiB for
 *     this call's plan uploads.  The call itself loads and allocates nothing
 *     on the device.  If that set-up failed, the call returns its error.
 *   - The plan is copied asynchronously from one of those pinned buffers; a
 *     plan larger than 2 MiB is copied from pageable host memory instead.
 *   - The current device must be the cache's device (else INVALID_ARG).
 *   - A call whose plan and partials need more than SQ_NOALLOC_SCRATCH_BYTES
 *     (very many sequences, or a very large decode_ctas) returns
 *     SQ_ERR_CAPACITY and enqueues nothing.
 *   - Every call, on every cache of the device, shares the one scratch array
 *     and leaves its contents behind; nothing in it has to start at zero
 *     (every value read is written first by the same call).  Calls whose GPU
 *     work overlaps — on different streams without ordering between them —
 *     race on the scratch: order them (one stream, or events).
 *   - After a reset of the device (cudaDeviceReset) every cache of it is
 *     gone with its context: destroy them and create new ones.
 * Errors: BAD_HANDLE, INVALID_ARG, CAPACITY, CUDA. */
SQ_API int sq_decode_attention_noalloc(sq_cache *cache, const sq_seq *seqs, int32_t n_seqs,
                                       int32_t layer, const void *q, void *out,
                                       int32_t out_dtype, float sm_scale, void *stream);

/* Measurement helper: streams `bytes` (a multiple of 16, 16-byte aligned)
 * of device memory at `buf` once with plain loads and no writes, so that the
 * caller can time the read-only HBM bandwidth of this GPU next to the
 * library's kernels.  Not part of the method.  Errors: INVALID_ARG, CUDA. */
SQ_API int sq_probe_read(sq_cache *cache, const void *buf, size_t bytes, void *stream);

/* Test hook for failure detection (no counterpart in the paper).
 * SQ_DEBUG_DROP_DECODE_STAGE: in the next decode call, the first persistent
 * CTA leaves its first pipeline stage unsignalled, so that CTA's consumer
 * warps wait on a barrier nothing completes.  Their wait is bounded: after
 * about 2 s they give up, the CTA winds down without faulting, the output of
 * that call is undefined, and sq_sync_status returns SQ_ERR_DEVICE_TIMEOUT;
 * the cache and the CUDA context stay usable.  The flag clears itself after
 * one call.  0 clears it.  Errors: BAD_HANDLE, INVALID_ARG. */
enum { SQ_DEBUG_DROP_DECODE_STAGE = 1 };
SQ_API int sq_debug_set(sq_cache *cache, int32_t flags);

/* Synchronise `stream`, then read and clear the device error word.
 * Returns SQ_OK, SQ_ERR_DEVICE, SQ_ERR_DEVICE_TIMEOUT or SQ_ERR_CUDA. */
SQ_API int sq_sync_status(sq_cache *cache, void *stream);

/* Human-readable name of a return code. */
SQ_API const char *sq_strerror(int code);

#ifdef __cplusplus
}
#endif

#endif /* SQ_H_ */
