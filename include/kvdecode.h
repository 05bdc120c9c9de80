/*
 * kvdecode.h -- C ABI of libkvdecode.so: paged bf16 KV cache and batched
 * single-token decode attention for multimodal LLM serving on GB300 (sm_103a).
 *
 * The operation.  Language decoding is the memory-bandwidth-bound phase of
 * multimodal inference: every step streams the KV cache from HBM
 * (HeteroServe, Sec. 2 "Language decoding"; Sec. 5.1 datacenter pool running
 * decode with MHA and GQA backends).  The cache of one request holds
 * s_ctx = N_v + s_text tokens for each of L layers and n_kv KV heads of
 * dimension d_h, 2 * L * n_kv * d_h * s_ctx * b bytes (Sec. 4.1, Eq. 1), and
 * its first N_v positions are the KV of the vision embedding handed over at
 * the modality boundary (Sec. 5.1, the [1, N_v, d] embedding).  Blocks of the
 * cache are taken lazily, only when a request needs them (Sec. 5.4 "Lazy KV
 * Cache Allocation").  One decode step of one layer computes, for sequence b,
 * query head h and KV head g = h / G (G = H_q / H_kv):
 *
 *     o[b][h] = sum_t softmax_t(scale * q[b][h] . k[b][g][t]) * v[b][g][t]
 *
 * over all cached tokens t of b in logical order, including the token that
 * kv_append wrote for this step.
 *
 * Conventions for every function below.
 *  - Return KVC_OK (0) or a negative KVC_ERR_* code; kv_last_error() then
 *    returns a message for the calling thread.  On error nothing has been
 *    changed and nothing has been enqueued, unless the description says so.
 *  - bf16 tensors are IEEE bfloat16 bit patterns, row-major, densely packed.
 *  - "device" pointers must be CUDA device (or managed) memory of the device
 *    that was current at kv_cache_create; "host" pointers are ordinary host
 *    memory that the call reads before returning.  The caller owns every
 *    pointer it passes; the cache owns its pools, page table and scratch.
 *  - `stream` is a cudaStream_t (NULL = legacy default stream).  Device work
 *    is enqueued on it asynchronously; no hot-path call synchronises.  All
 *    calls on one cache must be ordered on one stream (or externally
 *    synchronised): the cache's scratch is shared between calls.
 *  - A handle must not be used from two host threads at once.
 */
#ifndef KVDECODE_H
#define KVDECODE_H

#include <stdint.h>

#if defined(__GNUC__)
#define KVC_API __attribute__((visibility("default")))
#else
#define KVC_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

#define KVC_OK 0
#define KVC_ERR_INVALID (-1)      /* bad argument, shape or sequence id      */
#define KVC_ERR_OOM (-2)          /* page pool or device memory exhausted     */
#define KVC_ERR_CUDA (-3)         /* a CUDA runtime call failed               */
#define KVC_ERR_PAGE_TABLE (-4)   /* device found a page id outside the pool  */
#define KVC_ERR_UNSUPPORTED (-5)  /* valid but unsupported shape              */
#define KVC_ERR_DEVICE (-6)       /* device-side wait gave up (see stats)     */

/* kvc_config.flags */
#define KVC_FLAG_HOST_ONLY 1  /* bookkeeping only: no device memory, no kernels.
                                 Allocation, page tables and sequence calls work;
                                 data and attention calls return KVC_ERR_INVALID. */

/* kvc_stats.device_error bits (sticky until the cache is destroyed) */
#define KVC_DEVERR_PAGE_RANGE 1   /* a page-table entry outside [0, num_pages) */
#define KVC_DEVERR_WAIT_TIMEOUT 2 /* a shared-memory pipeline wait gave up      */
#define KVC_DEVERR_SEQ_RANGE 4    /* a sequence length outside its page row     */
#define KVC_DEVERR_OOM 8          /* a device-side step found the pool exhausted */

typedef struct kvc_config {
    int32_t num_layers;        /* L: layer pools held (>= 1)                              */
    int32_t num_q_heads;       /* H_q (multiple of num_kv_heads)                          */
    int32_t num_kv_heads;      /* H_kv; G = H_q / H_kv must be <= 8                       */
    int32_t head_dim;          /* d_h: 64 or 128                                          */
    int32_t page_size;         /* P: tokens per page; 16                                  */
    int32_t max_seqs;          /* sequence slots (ids 0 .. max_seqs-1), <= 65535          */
    int32_t max_pages_per_seq; /* page-table row length                                   */
    int32_t flags;             /* KVC_FLAG_*                                              */
    int64_t num_pages;         /* pages in the pool; one page id addresses the same slot
                                  in every layer pool, for K and for V                    */
} kvc_config;

typedef struct kvc_stats {
    int64_t kv_bytes_allocated; /* bytes of the pages in use: Eq. 1 with s_ctx rounded up
                                   to whole pages, 2 * L * H_kv * d_h * 2 * P * pages_in_use */
    int64_t pool_bytes;         /* bytes of the K and V pools on the device              */
    int64_t pages_in_use;
    int64_t free_pages;
    int32_t live_seqs;
    int32_t device_error;       /* KVC_DEVERR_* bits found by kernels so far             */
    int64_t kernel_launches;    /* kernels this cache has launched since creation         */
} kvc_stats;

typedef struct kv_cache kv_cache; /* opaque */

/* ---------------------------------------------------------------- cache -- */

/* Create a cache on the current CUDA device.  Allocates the K and V pools,
 * each laid out [L][num_pages][H_kv][P][d_h] bf16 (one (page, head) tile is
 * P * d_h * 2 bytes of consecutive tokens), the page table
 * [max_seqs][max_pages_per_seq] int32 (unused entries -1), the lengths, and
 * step scratch; zero-fills the pools on `stream`.  Initial page pop order is
 * 0, 1, 2, ...  KVC_ERR_UNSUPPORTED for head_dim not in {64, 128},
 * page_size != 16 or G > 8; KVC_ERR_OOM if device memory runs out. */
KVC_API int kv_cache_create(const kvc_config *cfg, void *stream, kv_cache **out);

/* Synchronise the device, then free everything the cache owns.  NULL is
 * accepted. */
KVC_API int kv_cache_destroy(kv_cache *cache);

/* Install the order in which free pages are handed out: order[0] first.
 * `order` (host, n = num_pages entries) must be a permutation of
 * 0 .. num_pages-1, and no page may be in use. */
KVC_API int kv_cache_set_page_order(kv_cache *cache, const int32_t *order, int64_t n);

/* Wait for the cache's stream (the stream of its latest call, which must
 * still exist; should waiting on it fail, the whole device) and report usage
 * and device error bits, read back on a stream the cache owns.  Returns
 * KVC_ERR_PAGE_TABLE (page or length range), KVC_ERR_OOM (a device-side step
 * ran out of pages) or KVC_ERR_DEVICE (a pipeline wait gave up) if
 * device_error is non-zero; the stats are filled in either way. */
KVC_API int kv_cache_query(kv_cache *cache, kvc_stats *stats);

/* Device pointers of one layer's K and V pools ([num_pages][H_kv][P][d_h]
 * bf16), for inspection; owned by the cache. */
KVC_API int kv_cache_pool(kv_cache *cache, int32_t layer, void **k_pool, void **v_pool);

/* Override the target split size (pages per work item of decode_attention)
 * used by later kv_begin_step calls; 0 restores the automatic choice.
 * Range 0 .. 1024.  A row of n pages is cut into ceil(n / T') items of
 * near-equal size, T' = max(T, ceil(n / 32)): never more than 32 items per
 * (sequence, KV head). */
KVC_API int kv_cache_set_split_pages(kv_cache *cache, int32_t pages);

/* -------------------------------------------------------- sequences ------ */

/* Open a sequence of length 0; *seq_id = the lowest free id.  No page is
 * taken until tokens are reserved (lazy allocation, Sec. 5.4). */
KVC_API int kv_seq_create(kv_cache *cache, int32_t *seq_id);

/* Reserve n_tokens more positions at the end of a sequence.  Walking the new
 * positions in order, a page is taken from the pop order exactly when a
 * position is the first slot of a page.  All or nothing: KVC_ERR_OOM if the
 * pool lacks pages, KVC_ERR_INVALID if the row would exceed
 * max_pages_per_seq.  The page-table and length update is enqueued on
 * `stream`.  While device-side steps are enabled (kv_cache_device_steps) the
 * device holds the free pages and lengths: the reservation is then one
 * kernel on `stream`, with no host synchronisation, that takes the same pages
 * in the same order; a full page row sets KVC_DEVERR_SEQ_RANGE and an
 * exhausted pool KVC_DEVERR_OOM (read by kv_cache_query) and that
 * reservation changes nothing; the return code then only covers the
 * arguments (a live sequence, 0 <= n_tokens <= max_pages_per_seq * 16). */
KVC_API int kv_seq_reserve(kv_cache *cache, int32_t seq_id, int32_t n_tokens, void *stream);

/* Close a sequence: its pages go back to the front of the pop order in its
 * logical page order.  The device row is reset on `stream`.  With device-side
 * steps enabled this is one kernel on `stream` and no host synchronisation;
 * the sequence id is free again at once. */
KVC_API int kv_seq_free(kv_cache *cache, int32_t seq_id, void *stream);

/* Host view of one sequence: *len = reserved positions; page_ids (host,
 * capacity entries, may be NULL) receives its pages in logical order;
 * *n_pages = ceil(len / P). */
KVC_API int kv_seq_info(kv_cache *cache, int32_t seq_id, int32_t *len, int32_t *page_ids,
                int32_t capacity, int32_t *n_pages);

/* Write n tokens of one layer into reserved positions [first_pos,
 * first_pos + n) of a sequence: the prefix (the N_v vision tokens handed over
 * at the modality boundary, then the prompt) or any later rewrite.
 * k, v: device, [n][H_kv][d_h] bf16.  Requires first_pos + n <= length:
 * checked on the host, or, while device-side steps are enabled (the length
 * is the device's), by the kernel, which then writes nothing and sets
 * KVC_DEVERR_SEQ_RANGE. */
KVC_API int kv_write_tokens(kv_cache *cache, int32_t layer, int32_t seq_id, int32_t first_pos,
                    int32_t n, const void *k, const void *v, void *stream);

/* Bulk write of a packed variable-length batch of token blocks, in one launch
 * (one per 512 non-empty blocks): the vision-prefix K/V handed over at the
 * modality boundary plus the prompt, for many sequences and layers at once
 * (Sec. 5.1 handoff; Sec. 5.4 "Flash Attention Varlen for Packed Prefill":
 * one packed tensor with cumulative lengths, one launch instead of one per
 * sequence).  Block i holds the rows cu_seqlens[i] ..
 * cu_seqlens[i+1]-1 of k and v and goes to positions first_pos[i] ..
 * first_pos[i] + n_i - 1 of sequence seq_ids[i], in layers layer_first ..
 * layer_first + n_layers - 1.
 *   seq_ids, first_pos, cu_seqlens: host arrays of n_blocks, n_blocks and
 *     n_blocks + 1 entries; cu_seqlens[0] == 0 and non-decreasing; first_pos
 *     NULL means 0 for every block.  Blocks may name the same sequence but
 *     not the same position (KVC_ERR_INVALID); empty blocks are skipped.
 *   k, v: device, [n_layers][cu_seqlens[n_blocks]][H_kv][d_h] bf16, 16-byte
 *     aligned, read when the kernel runs.
 * The positions must already be reserved (kv_seq_reserve on this stream or
 * before it).  A page id outside the pool found by the kernel sets
 * KVC_DEVERR_PAGE_RANGE and that page is not written. */
KVC_API int kv_write_varlen(kv_cache *cache, int32_t layer_first, int32_t n_layers, int32_t n_blocks,
                    const int32_t *seq_ids, const int32_t *first_pos, const int32_t *cu_seqlens,
                    const void *k, const void *v, void *stream);

/* Copy positions [first_pos, first_pos + n) of one layer back into logical
 * order: k_out, v_out device [n][H_kv][d_h] bf16. */
KVC_API int kv_read_tokens(kv_cache *cache, int32_t layer, int32_t seq_id, int32_t first_pos,
                   int32_t n, void *k_out, void *v_out, void *stream);

/* -------------------------------------------------------- decode step ---- */

/* Start one decode step for `batch` distinct live sequences (seq_ids: host,
 * batch entries; batch order is the row order of q, out, k_new, v_new in the
 * calls below).  Reserves one position s_b (the old length) per sequence,
 * taking a page when s_b % P == 0, all or nothing (KVC_ERR_OOM leaves
 * everything unchanged), and enqueues one kernel that updates the device page
 * table and lengths and builds the split plan the layers of this step share.
 * batch <= max_seqs. */
KVC_API int kv_begin_step(kv_cache *cache, int32_t batch, const int32_t *seq_ids, void *stream);

/* Fused K+V append for one layer of the current step: writes k_new[b] and
 * v_new[b] (device, [batch][H_kv][d_h] bf16) into position s_b of each
 * sequence of the step.  `batch` must equal the step's batch.  Each decode
 * step adds one token to every request's cache, which holds the K and V of
 * all its tokens per layer and KV head (Sec. 2 "Language decoding"; what the
 * cache holds and its size: Sec. 4.1, Eq. 1).  Pools are written in place;
 * the caller keeps ownership of k_new / v_new, which must be 16-byte aligned.
 * Errors (no active step, batch mismatch, bad layer or pointer) are reported
 * before anything is enqueued. */
KVC_API int kv_append(kv_cache *cache, int32_t layer, int32_t batch, const void *k_new,
              const void *v_new, void *stream);

/* Decode attention for one layer of the current step: the memory-bound
 * decode phase that streams each request's KV cache from HBM once per layer
 * (Sec. 2 "Language decoding"), over a cache laid out as Eq. 1 counts it
 * (Sec. 4.1), MHA or GQA (Sec. 5.1).  q: device
 * [batch][H_q][d_h] bf16; out: device [batch][H_q][d_h] bf16 (written).
 * Attends over positions 0 .. s_b of each sequence, so call kv_append for the
 * same layer first, on the same stream.  softmax_scale <= 0 selects
 * 1/sqrt(d_h).  Split-KV: the step's plan cuts each (sequence, KV head) into
 * work items of consecutive pages; each item runs an online softmax in fp32
 * over its pages for all G query heads of the KV head, and a second kernel
 * merges the partial results of every (sequence, KV head) cut into several
 * items by log-sum-exp. */
KVC_API int decode_attention(kv_cache *cache, int32_t layer, int32_t batch, const void *q, void *out,
                     float softmax_scale, void *stream);

/* kv_append and decode_attention of one layer in a single kernel: the new
 * token's K and V (k_new, v_new: device [batch][H_kv][d_h] bf16) are written
 * into position s_b of each sequence and used in place of that slot's old
 * contents while the layer's pages stream through shared memory.  Same
 * result and cache contents as kv_append followed by decode_attention.
 * When the library's previous launch on `stream` was an attention launch
 * (decode_attention or decode_attention_append of this cache), the kernel is
 * launched with programmatic dependent launch: it may start, and stream this
 * layer's cached pages (positions < s_b), while that launch is finishing; it
 * reads q, k_new and v_new and writes anything only after the kernel before
 * it has completed.  After any other call of this library it is an ordinary
 * launch.  So a kernel the caller enqueues between two layers must not write
 * the cache's pages (a foreign kernel could only race with the early reads
 * if it signalled its dependents early). */
KVC_API int decode_attention_append(kv_cache *cache, int32_t layer, int32_t batch, const void *q,
                                    const void *k_new, const void *v_new, void *out,
                                    float softmax_scale, void *stream);

/* ------------------------------------------- graph-replayable decode step -- */

/* Enable (enable = 1) or disable device-side steps.  While enabled, the free
 * page stack also lives on the device and kv_begin_step_device performs the
 * step's lazy allocation and split plan there, so a whole decode step
 * (kv_begin_step_device, then per layer decode_attention_append or
 * kv_append + decode_attention) can be captured once into a CUDA graph and
 * replayed every step with no host work (the role CUDA graphs play in the
 * paper's engine, Sec. 5.4).  Enabling reserves plan, page-list and partial
 * buffers for up to max_batch sequences at the longest page-table row, and
 * fixes the work-item size from the pages currently held.  While enabled,
 * admitting and closing sequences needs no host synchronisation:
 * kv_seq_create is host bookkeeping, kv_seq_reserve and kv_seq_free are
 * kernels on their stream, and kv_write_tokens, kv_write_varlen and
 * kv_read_tokens check positions against the device's lengths in their
 * kernels.  The host allocator's view is refreshed from the device lazily,
 * by the next call that reads it (kv_seq_info, kv_begin_step,
 * kv_cache_query, kv_cache_set_page_order, kv_cache_device_steps or
 * kv_cache_sync), which waits for the cache's stream (the stream of the
 * cache's latest call, so replay the graphs on that stream; it must still
 * exist, and should waiting on it fail, the whole device) and reads the
 * state back on a stream the cache owns.  Graphs captured while device
 * steps are enabled stay valid until they are disabled, enabled again (which
 * may resize the buffers) or the cache is destroyed: meanwhile a host-planned
 * step that would need larger buffers fails with KVC_ERR_INVALID instead of
 * moving them. */
KVC_API int kv_cache_device_steps(kv_cache *cache, int32_t max_batch, int32_t enable, void *stream);

/* kv_begin_step with everything on the device: seq_ids is DEVICE memory
 * ([batch] distinct live sequence ids, read when the kernel runs, so a
 * replayed graph may change them between replays); pages come off the
 * device free stack in batch order, exactly as kv_begin_step takes them.
 * A pool that runs out sets KVC_DEVERR_OOM, a sequence id outside the cache
 * or a full page row KVC_DEVERR_SEQ_RANGE; such a row keeps its length, and
 * the layer calls of the step (kv_append, decode_attention,
 * decode_attention_append) leave its cache and its output row untouched.  No
 * host synchronisation; graph-capturable. */
KVC_API int kv_begin_step_device(kv_cache *cache, int32_t batch, const int32_t *seq_ids, void *stream);

/* Wait for the cache's stream (the stream of its latest call, which must
 * still exist) and refresh the host allocator's view after device-side steps
 * and allocator calls. */
KVC_API int kv_cache_sync(kv_cache *cache);

/* ------------------------------------------------ allocation-free decode -- */

/* decode_attention for callers that may not allocate device memory while they
 * serve: an engine plugin held to a memory budget fixed when the engine was
 * built, a runtime whose device memory all belongs to another framework's
 * allocator, a decode thread that must not take the allocator's locks.  Such a
 * caller owns the K/V pools and the page table and passes them in; this call
 * allocates nothing (no cudaMalloc, cudaMallocAsync, cudaFree or allocating
 * library routine).  The paper has no counterpart: it is a convenience of this
 * library, computing the same attention as decode_attention.
 *   k_pool, v_pool  device, [num_pages][num_kv_heads][16][head_dim] bf16 (the
 *                   layout kv_cache_pool exposes), 16-byte aligned
 *   page_table      device, [batch][max_pages] int32: row b lists the pages of
 *                   sequence b in logical order
 *   lens            host, [batch]: tokens attended by row b, 1 .. max_pages*16
 *   q, out          device, [batch][num_q_heads][head_dim] bf16
 *   device_error    device int32 that receives KVC_DEVERR_* bits (OR-ed, never
 *                   cleared by this call), or NULL to discard them
 * Work space is a 16 MiB array in this library's device code, held by every
 * GPU that loads the library until the process exits.  batch <= 1024.
 * Work items are enlarged (doubled, up to 1024 pages each) until the split
 * plan and partial results fit the 16 MiB (one item per row needs no
 * partials at all); KVC_ERR_UNSUPPORTED, with nothing enqueued, if they
 * still do not fit at 1024 pages.  The first call on
 * each device looks up the array's device address (cudaGetSymbolAddress);
 * make that first call before any stream capture.  Every call uses the same
 * array and clears the counters it needs at its start, so calls that overlap
 * on the GPU race: order them on one stream.  Same shape limits as
 * kv_cache_create (head_dim 64 or 128, G <= 8, 16-token pages). */
KVC_API int decode_attention_noalloc(const void *k_pool, const void *v_pool, int64_t num_pages,
                                     int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                                     int32_t batch, const int32_t *page_table, int32_t max_pages,
                                     const int32_t *lens, const void *q, void *out,
                                     float softmax_scale, int32_t *device_error, void *stream);

/* Diagnostics: one warp runs the bounded shared-memory wait that every
 * pipeline wait of the decode kernels uses, on a barrier that nothing ever
 * completes, and writes 1 to *status (device int32) when the wait gave up
 * after limit_ns nanoseconds (0 < limit_ns <= 2e9), 0 if it completed.  The
 * GPU context stays usable afterwards.  Asynchronous on `stream`. */
KVC_API int kv_selftest_wait_timeout(int64_t limit_ns, int32_t *status, void *stream);

/* Message of the last failed call on this thread ("" if none). */
KVC_API const char *kv_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* KVDECODE_H */
