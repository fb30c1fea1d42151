/*
 * dms.h -- C ABI of libdms: Dynamic Memory Sparsification (DMS) decode on one
 * NVIDIA GB300 (sm_103a).  arXiv 2506.05345, "Inference-Time Hyper-Scaling with
 * KV Cache Compression".
 *
 * What the library does.  Every (layer, sequence, KV head) keeps its own KV
 * cache.  Each appended token carries a binary eviction decision alpha, taken
 * from a bf16 logit as round(sigmoid(logit)) == [logit > 0] (Sec. 3.2; the tie
 * logit = 0 keeps, NaN keeps).  The eviction is delayed (Sec. 3.1, "Delayed
 * Eviction via Sliding Window"): a flagged token stays visible while it is within
 * the window and is dropped when it leaves it.  Precisely, after the token at
 * position j has been appended, the retained set of a head is
 *     R_j = { i <= j : alpha_i == 0  or  j - i <= window },
 * which reproduces the mask of Fig. 1b with window = 3.  The slot of a dropped
 * token is overwritten by the incoming one (Sec. 3.2: evicted tokens are simply
 * overwritten; pages belong to individual heads), so each head's retained tokens
 * occupy slots [0, n_h) of its own page list.  Decode attention is plain softmax
 * attention of the query heads of a GQA group (Sec. 4) over R_j of their KV head.
 *
 * Conventions for every entry point:
 *   - Data pointers (k, v, decision_logit, q, out) are DEVICE pointers to
 *     caller-owned, contiguous memory, 16-byte aligned.  bf16 means IEEE
 *     bfloat16 (the upper half of a binary32).  The caller keeps them alive
 *     until the work queued on `stream` has completed.
 *   - `stream` is a cudaStream_t (NULL = the legacy default stream).  Calls
 *     are asynchronous unless stated; only dms_cache_stats and
 *     dms_cache_export_positions wait for the stream.
 *   - One cache is driven from one stream at a time (calls are not
 *     thread-safe on the same cache).  All sequences of the batch advance in
 *     lockstep: every call appends the same number of tokens to every sequence,
 *     and each layer keeps its own length.
 *   - Argument errors are detected on the host and return
 *     DMS_ERR_INVALID_ARGUMENT without queuing any work.  Errors found on the
 *     device (page pool exhausted, a bounded wait that ran out) set a sticky
 *     flag in the cache; the call that queued the work still returns DMS_OK and
 *     dms_cache_stats reports the flag.  No entry point traps or throws.
 */
#ifndef DMS_H_
#define DMS_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct dms_cache dms_cache; /* opaque; the library owns all cache memory */

typedef enum dms_status {
  DMS_OK = 0,
  DMS_ERR_INVALID_ARGUMENT = 1, /* bad pointer, shape, layer or option        */
  DMS_ERR_OUT_OF_MEMORY = 2,    /* device allocation failed                   */
  DMS_ERR_CAPACITY = 3,         /* sequence longer than `capacity`, or the
                                   page pool ran out (sticky device flag)      */
  DMS_ERR_CUDA = 4,             /* a CUDA runtime call failed                 */
  DMS_ERR_TIMEOUT = 5,          /* a bounded in-kernel wait gave up (sticky)  */
  DMS_ERR_STATE = 6             /* call not valid in the cache's current state */
} dms_status;

/* Eviction policies selectable through dms_options.eviction_policy. */
enum {
  DMS_EVICT_DELAYED = 0,   /* default, the method (Sec. 3.1): the token leaving the window
                              at step j is evicted iff its own decision alpha_{j-w-1} = 1 */
  DMS_EVICT_IMMEDIATE = 1  /* the ablation of Sec. 5: it is evicted iff the decision of
                              token j - 1 (= (j - w - 1) + w) is 1; the same as delayed
                              when window = 0                                            */
};

/* Decode kernels selectable through dms_options.decode_kernel. */
enum {
  DMS_DECODE_TILED = 0,   /* default: TMA-staged tensor-core kernels; as
                             DMS_DECODE_CLUSTER when clusters of the largest size
                             in [1, 16] that fits for every head would cover at
                             least half of the SMs, else as DMS_DECODE_SPLIT       */
  DMS_DECODE_SIMPLE = 1,  /* one CTA per KV head, CUDA cores; a cross-check path     */
  DMS_DECODE_SPLIT = 2,   /* the tiled kernel with the flat, page-balanced split-K of
                             all heads' pages over all SMs, for every batch          */
  DMS_DECODE_CLUSTER = 3  /* per-head thread-block clusters: when bf16 pages, G <= 8,
                             the default ctas_per_sm / min_pages_per_cta, and a
                             resident cluster for every (sequence, KV head) at once
                             (up to one head per SM), each head's pages are split
                             over its own cluster of C CTAs and merged in
                             distributed shared memory, C = 6 for layers of up to
                             8192 tokens, else 10, or the largest size in [1, 16]
                             that fits if smaller (1: one CTA takes the whole head);
                             otherwise as DMS_DECODE_SPLIT                           */
};

/*
 * Page formats selectable through dms_options.kv_format.  The paper treats KV
 * quantisation as orthogonal to DMS and combinable with it (related-work section:
 * quantisation, e.g. per-channel keys and per-token values, is a separate axis of
 * KV-cache reduction).
 */
enum {
  DMS_KV_BF16 = 0,     /* default: K and V rows of 128 bf16; pages of 32 KiB          */
  DMS_KV_FP8_E4M3 = 1  /* K and V rows of 128 fp8 E4M3 codes (OCP E4M3FN: bias 7,
                          no infinities, largest finite 448) with one fp32 scale per
                          row and tensor: scale = amax(|row|) / 448 (fp32 division),
                          code = E4M3(row / scale) rounded to nearest even and
                          saturated; a row of zeros has scale 0.  Pages of 16.5
                          KiB: K codes, V^T codes, then the 128 row scales (one
                          bulk copy each).  Rows must be finite.  Read by
                          the tiled kernels (the flat split and the per-head
                          clusters), not by DMS_DECODE_SIMPLE; the single-token
                          append + decode runs in one launch.                        */
};

typedef struct dms_options {
  int32_t batch;         /* sequences per layer (required, >= 1)                    */
  int32_t page_tokens;   /* tokens per page; 0 = 64 (only 64 is accepted)           */
  int64_t pool_tokens;   /* page pool size in tokens (rounded up to whole pages),
                            shared by all layers and heads; 0 = the dense worst
                            case, layers * batch * kv_heads * ceil(capacity / 64)
                            pages                                                  */
  int32_t decode_kernel; /* DMS_DECODE_TILED (0), _SIMPLE (1), _SPLIT (2), _CLUSTER (3) */
  int32_t ctas_per_sm;   /* split-K CTAs per SM for the tiled kernel; 0 = 1         */
  int32_t min_pages_per_cta; /* lower bound on pages per split-K CTA; 0 = 2         */
  int32_t eviction_policy;   /* DMS_EVICT_DELAYED (0) or DMS_EVICT_IMMEDIATE (1)    */
  int32_t kv_format;     /* DMS_KV_BF16 (0) or DMS_KV_FP8_E4M3 (1); fp8 requires a
                            tiled decode kernel (not SIMPLE)                        */
  int32_t reserved[3];   /* must be zero                                            */
} dms_options;

typedef struct dms_stats {
  int64_t total_retained; /* sum over layers, sequences, KV heads of n_h            */
  int64_t total_appended; /* tokens appended, summed the same way                  */
  int64_t total_evicted;  /* total_appended - total_retained                       */
  int64_t pages_in_use;   /* pages handed out from the pool                        */
  int64_t pool_pages;     /* pages in the pool                                     */
  int64_t peak_pages;     /* largest pages_in_use seen since creation              */
  int32_t max_retained;   /* largest n_h over all heads                            */
  int32_t min_retained;   /* smallest n_h over all heads                           */
  int32_t device_error;   /* sticky device-side dms_status (DMS_OK if none)        */
  int32_t reserved;
} dms_stats;

/*
 * Create a cache for `layers` layers of `kv_heads` KV heads (head_dim must be
 * 128), sliding window `window` >= 0 (Sec. 3.1; the paper's default is 256), and
 * at most `capacity` >= 1 appended tokens per sequence.  `opt` must be non-NULL
 * with opt->batch >= 1; zeroed fields take their defaults.  Allocates the page
 * pool, page tables, per-head counts, decision rings and decode scratch, and
 * zeroes the counts.  On success *out receives the cache; on failure *out is
 * NULL and nothing stays allocated.  Limits: batch * kv_heads <= 4096,
 * capacity < 2^30.
 */
dms_status dms_cache_create(int32_t layers, int32_t kv_heads, int32_t head_dim,
                            int32_t window, int64_t capacity, const dms_options* opt,
                            dms_cache** out);

/* Free everything the cache owns (synchronises the device first).  NULL is a no-op. */
dms_status dms_cache_destroy(dms_cache* cache);

/*
 * Empty every head of every layer (all n_h = 0, all layer lengths 0, pool
 * returned, sticky device error cleared).  Queued on `stream`.
 */
dms_status dms_cache_reset(dms_cache* cache, void* stream);

/*
 * Append n_tokens >= 1 tokens to every sequence of `layer` and apply delayed
 * eviction (Sec. 3.1-3.2).  Positions t0 .. t0 + n_tokens - 1 are appended,
 * t0 being the layer's current length.
 *   k, v            [batch, n_tokens, kv_heads, 128] bf16 (keys already carry
 *                   their positional encoding, Sec. 3.2)
 *   decision_logit  [batch, n_tokens, kv_heads] bf16; alpha = [logit > 0]
 * After the call each head holds exactly R_{t0+n_tokens-1}.  A bulk call
 * (prefill) gives the same retained sets as n_tokens single-token calls.
 * Returns DMS_ERR_CAPACITY (nothing queued) if the layer would exceed
 * `capacity`.  Page-pool exhaustion is reported through the sticky flag.
 */
dms_status dms_append_and_evict(dms_cache* cache, int32_t layer, const void* k,
                                const void* v, const void* decision_logit,
                                int32_t n_tokens, void* stream);

/*
 * Decode attention for `layer` over the current retained sets (GQA, Sec. 4):
 *   q    [batch, kv_heads * gqa_group, 128] bf16; query head hq reads KV head
 *        hq / gqa_group
 *   out  [batch, kv_heads * gqa_group, 128] bf16 (round to nearest even)
 * out[b][hq] = sum_{i in R} softmax_i(sm_scale * <q, k_i>) v_i, with fp32
 * accumulation.  sm_scale <= 0 means 1/sqrt(128).  1 <= gqa_group <= 16.  A
 * head with no tokens yet (nothing appended) yields zeros.
 */
dms_status dms_decode_attention(dms_cache* cache, int32_t layer, const void* q, void* out,
                                int32_t gqa_group, float sm_scale, void* stream);

/*
 * One decode step of one layer in a single launch: exactly
 * dms_append_and_evict(cache, layer, k, v, decision_logit, 1, stream) followed by
 * dms_decode_attention(cache, layer, q, out, gqa_group, sm_scale, stream), with
 * the same arguments, layouts and results (n_tokens = 1: k, v are
 * [batch, 1, kv_heads, 128] bf16, decision_logit [batch, 1, kv_heads] bf16).
 * The single-token append is fused into the tiled decode kernel; when the fused
 * kernel does not apply (decode_kernel = DMS_DECODE_SIMPLE, ctas_per_sm >= 2, or
 * batch * kv_heads > 4000) the two separate kernels run instead.
 */
dms_status dms_append_and_decode(dms_cache* cache, int32_t layer, const void* k, const void* v,
                                 const void* decision_logit, const void* q, void* out,
                                 int32_t gqa_group, float sm_scale, void* stream);

/*
 * Shared prompt: append n_tokens tokens that are IDENTICAL in every sequence (the same
 * k, v and decision logits, given once: [1, n_tokens, kv_heads, 128] and
 * [1, n_tokens, kv_heads]) to an EMPTY layer.  The result is the cache that
 * dms_append_and_evict would leave with those inputs repeated for every sequence, but
 * the pages that can no longer change -- those entirely below slot n_h - min(window + 1,
 * n_tokens), whose tokens have already left the window and are kept for good -- are
 * stored once and mapped into every sequence's page table, read-only; the rest are
 * copied per sequence.  Later appends and decodes are unchanged (they never write those
 * pages), and decode reads of the shared pages by the other sequences are served from L2
 * when they are close in time.  Errors: DMS_ERR_STATE if the layer is not empty, else as
 * dms_append_and_evict (pool exhaustion is the sticky device error).
 */
dms_status dms_append_shared_prefix(dms_cache* cache, int32_t layer, const void* k, const void* v,
                                    const void* decision_logit, int32_t n_tokens, void* stream);

/*
 * Decisions from a borrowed query neuron (App. B).  Instead of a separate logit
 * tensor, the decision logit of (sequence b, KV head h) at each token is element 0
 * of that group's FIRST query head, q[b, t, h * gqa_group, 0]; the decision rule
 * is the same (alpha = 1 iff that bf16 value is > 0, Sec. 3.2).  The attention
 * then takes that element as 0 for the first query head of every group, leaving
 * the group's other query heads unchanged.  The caller's q is not modified.
 *
 * dms_append_and_evict_borrowed: as dms_append_and_evict (any n_tokens >= 1), with
 *   q [batch, n_tokens, kv_heads * gqa_group, 128] bf16 supplying the decisions
 *   (only element 0 of each group's first head is read).
 * dms_decode_attention_borrowed: as dms_decode_attention, attending with element 0
 *   of each group's first query head taken as 0.
 * dms_append_and_decode_borrowed: one decode step, as dms_append_and_decode, with
 *   the decisions taken from q [batch, kv_heads * gqa_group, 128] and the
 *   attention as in dms_decode_attention_borrowed.
 * Arguments, alignment, errors and stream semantics are those of the plain forms.
 */
dms_status dms_append_and_evict_borrowed(dms_cache* cache, int32_t layer, const void* k,
                                         const void* v, const void* q, int32_t n_tokens,
                                         int32_t gqa_group, void* stream);
dms_status dms_decode_attention_borrowed(dms_cache* cache, int32_t layer, const void* q, void* out,
                                         int32_t gqa_group, float sm_scale, void* stream);
dms_status dms_append_and_decode_borrowed(dms_cache* cache, int32_t layer, const void* k,
                                          const void* v, const void* q, void* out,
                                          int32_t gqa_group, float sm_scale, void* stream);

/*
 * Sparse prefill attention (Sec. 3.1 mask, Fig. 1b; Sec. 3.2: the eviction sparsity is
 * used in prefill as well).  For a prompt of n_tokens tokens, query j of every query
 * head attends, with plain softmax, to the keys i <= j of its KV head with
 * alpha_i = 0 or j - i <= window, alpha_i = [bf16 decision logit of token i > 0]; the
 * result is what a decode at position j would return after appending tokens 0..j.
 * It is stateless: no cache is read or written (dms_append_and_evict fills a cache
 * from the same k, v and logits).
 *
 * Inputs (device pointers, bf16 unless stated, contiguous, 16-byte aligned):
 *   q, out          [batch, n_tokens, kv_heads * gqa_group, 128]; query head hq uses
 *                   KV head hq / gqa_group.
 *   k, v            [batch, n_tokens, kv_heads, 128]
 *   decision_logit  [batch, n_tokens, kv_heads] (2-byte aligned)
 *   workspace       caller-owned device memory of at least
 *                   dms_prefill_workspace_bytes(batch, n_tokens, kv_heads) bytes (about
 *                   1 KiB per token and KV head), 16-byte aligned; it must not be used by
 *                   other work until the call's stream work completes.
 * sm_scale <= 0 selects 1/sqrt(128).  Limits: batch * kv_heads <= 65535,
 * 1 <= gqa_group <= 16, ceil(n_tokens / 128) * batch * kv_heads * gqa_group < 2^31.
 * Errors: invalid arguments -> DMS_ERR_INVALID_ARGUMENT, a workspace that is too small ->
 * DMS_ERR_CAPACITY, both before any launch.  A bounded in-kernel wait that gives up
 * records DMS_ERR_TIMEOUT in the workspace; dms_prefill_device_error reads it.
 *
 * dms_prefill_attention_borrowed takes the decision logit of (b, t, h) from element 0
 * of query head h * gqa_group (App. B) and attends with that element taken as 0.
 */
dms_status dms_prefill_workspace_bytes(int32_t batch, int32_t n_tokens, int32_t kv_heads,
                                       size_t* out_bytes);
dms_status dms_prefill_attention(const void* q, const void* k, const void* v,
                                 const void* decision_logit, int32_t batch, int32_t n_tokens,
                                 int32_t kv_heads, int32_t gqa_group, int32_t window,
                                 float sm_scale, void* workspace, size_t workspace_bytes,
                                 void* out, void* stream);
dms_status dms_prefill_attention_borrowed(const void* q, const void* k, const void* v,
                                          int32_t batch, int32_t n_tokens, int32_t kv_heads,
                                          int32_t gqa_group, int32_t window, float sm_scale,
                                          void* workspace, size_t workspace_bytes, void* out,
                                          void* stream);
/* Prefill attention kernels (dms_prefill_attention_ex `kernel`). */
enum {
  DMS_PREFILL_TCGEN05 = 0,  /* default: 5th-generation tensor cores, accumulators in TMEM */
  DMS_PREFILL_MMA_SYNC = 1  /* warp-level mma.sync tiles; a cross-check path              */
};
/* The general form: decision_logit == NULL takes the decisions from the queries as in
 * the borrowed form; eviction_policy DMS_EVICT_DELAYED or DMS_EVICT_IMMEDIATE (the Sec. 5
 * ablation: key i is visible outside the window iff the decision of token i + window is 0);
 * kernel DMS_PREFILL_TCGEN05 or DMS_PREFILL_MMA_SYNC. */
dms_status dms_prefill_attention_ex(const void* q, const void* k, const void* v,
                                    const void* decision_logit, int32_t batch, int32_t n_tokens,
                                    int32_t kv_heads, int32_t gqa_group, int32_t window,
                                    int32_t eviction_policy, int32_t kernel, float sm_scale,
                                    void* workspace, size_t workspace_bytes, void* out,
                                    void* stream);
/* Synchronise `stream` and report the sticky device error of the last prefill that used
 * `workspace` into *out (DMS_OK when none). */
dms_status dms_prefill_device_error(const void* workspace, void* stream, dms_status* out);

/*
 * Synchronise `stream`, then report totals into *out (non-NULL) and, if
 * `counts` is non-NULL, copy the per-head retained counts n_h into the HOST
 * array counts[layers * batch * kv_heads] (layer-major, then sequence, then KV
 * head).  Returns the sticky device error, if any, as its own status as well.
 */
dms_status dms_cache_stats(dms_cache* cache, dms_stats* out, int32_t* counts, void* stream);

/*
 * Test/inspection helper.  Synchronise `stream` and write, for every
 * (sequence b, KV head h) of `layer`, the positions held in slots [0, n_h) into
 * the HOST array host_pos[(b * kv_heads + h) * capacity + slot], in slot order
 * (not sorted); unused entries are set to -1.
 */
dms_status dms_cache_export_positions(dms_cache* cache, int32_t layer, int32_t* host_pos,
                                      void* stream);

/*
 * Test/inspection helper.  Synchronise `stream` and write, for every
 * (sequence b, KV head h) of `layer` and every slot s < n_h, the stored key and
 * value rows in head_dim order into the HOST arrays
 *   host_k[((b * kv_heads + h) * capacity + s) * 128 + d]   (and host_v likewise),
 * elements of the cache's format: bf16 bit patterns (uint16) for DMS_KV_BF16,
 * E4M3 codes (uint8) for DMS_KV_FP8_E4M3; and, for fp8 caches, the row scales
 * into host_scales[((b * kv_heads + h) * capacity + s) * 2 + {0: key, 1: value}]
 * (host_scales is ignored, and may be NULL, for bf16 caches).  Entries of slots
 * >= n_h are zero.  Copies page by page (a few calls per page); meant for tests.
 */
dms_status dms_cache_export_kv(dms_cache* cache, int32_t layer, void* host_k, void* host_v,
                               float* host_scales, void* stream);

/* Current length (tokens appended per sequence) of `layer`, into *out. */
dms_status dms_cache_layer_length(const dms_cache* cache, int32_t layer, int64_t* out);

/*
 * How the next dms_append_and_decode of `layer` (its length + 1 tokens) runs with groups
 * of gqa_group query heads (host only, no device work): *kernel = DMS_DECODE_SIMPLE,
 * DMS_DECODE_SPLIT or DMS_DECODE_CLUSTER, the kernel that runs (DMS_DECODE_TILED resolves
 * to one of the last two); *ctas = CTAs per launch; *cluster_size = CTAs per thread-block
 * cluster (0 unless DMS_DECODE_CLUSTER).  The cluster size depends on the layer's length
 * (see DMS_DECODE_TILED).  Errors: DMS_ERR_INVALID_ARGUMENT (NULL pointer, layer out of
 * range, gqa_group outside [1, 16]).
 */
dms_status dms_decode_plan(const dms_cache* cache, int32_t layer, int32_t gqa_group,
                           int32_t* kernel, int32_t* ctas, int32_t* cluster_size);

/*
 * Decode attention over CALLER-OWNED pages, allocating nothing.
 *
 * The paper has no counterpart to this entry point: it exists for callers that
 * cannot call cudaMalloc at all -- for example code running inside a host
 * application whose device memory is wholly owned by that application's own
 * allocator (a framework caching allocator or an arena reserved at start-up),
 * where a direct device allocation would bypass its budget or fail.  Such a
 * caller owns every input and output; the library neither creates a cache nor
 * allocates scratch.  The split-K scratch of the tiled decode kernel lives in a
 * file-scope device array of about 8.5 MB that every GPU loading the library
 * holds until the process exits.
 *
 * Inputs (device pointers, 16-byte aligned where they hold bf16 rows; bf16 pages only):
 *   pool        pages of 32 KiB: page p holds 64 K rows then 64 V rows, each row
 *               128 bf16 (256 bytes) whose sixteen 16-byte chunks are stored
 *               permuted -- logical chunk c of row r at physical chunk
 *               c ^ (r & 7) -- the layout dms_append_and_evict writes.
 *   page_table  [batch * kv_heads][max_pages] int32: slot s of head (b, h) is
 *               row s % 64 of page page_table[(b * kv_heads + h) * max_pages + s / 64].
 *   counts      [batch * kv_heads] int32: head (b, h) attends to its slots
 *               [0, counts[.]); the caller guarantees counts <= 64 * max_pages
 *               and valid page ids for every slot below the count.
 *   q, out      as for dms_decode_attention.
 * Limits: batch * kv_heads + (number of SMs) <= 1024 (872 heads on a 152-SM
 * GB300), else DMS_ERR_CAPACITY; 1 <= gqa_group <= 16.
 *
 * The first call on each device does a one-time set-up on the calling thread
 * with that device current (looks up the scratch array's device address and sets
 * the kernel's shared-memory limit); make that first call before any stream
 * capture.  Every call clears the scratch counters it needs with an asynchronous
 * memset on `stream` and then launches; all calls share the one array, so calls
 * whose work overlaps on the GPU (other streams, other host threads) race and
 * must be serialised by the caller.  A bounded in-kernel wait that gives up
 * (DMS_ERR_TIMEOUT) does not change the return code, which reports only what the
 * host saw; it is kept in the scratch array's error word until the next call
 * clears it, and dms_decode_noalloc_device_error reads it.
 * page_table and counts must be 4-byte aligned.
 */
dms_status dms_decode_attention_paged_noalloc(const void* pool, const int32_t* page_table,
                                              const int32_t* counts, int32_t batch,
                                              int32_t kv_heads, int32_t max_pages,
                                              const void* q, void* out, int32_t gqa_group,
                                              float sm_scale, void* stream);

/*
 * Device-side status of the last dms_decode_attention_paged_noalloc call on the
 * current device (no counterpart in the paper: failure detection of the
 * implementation).  Synchronises `stream`, then writes into *out the error word
 * that call's kernel left in the static scratch array: DMS_OK, or DMS_ERR_TIMEOUT
 * when one of its bounded shared-memory barrier waits gave up (its outputs are
 * then not valid).  Allocates nothing: the word is copied into host stack memory.
 * Returns DMS_ERR_CUDA if the copy or the synchronisation fails.
 */
dms_status dms_decode_noalloc_device_error(void* stream, dms_status* out);

/*
 * Self-test of that report (no counterpart in the paper).  Clears the static
 * scratch array's error word, then runs on `stream` a small kernel whose bounded
 * barrier wait can never complete, with the limit `limit_ns` (1 us .. 10 s): the
 * wait gives up, records DMS_ERR_TIMEOUT in the error word exactly as a decode
 * kernel would, and the kernel exits normally, so the CUDA context stays usable.
 * dms_decode_noalloc_device_error then reports DMS_ERR_TIMEOUT until the next
 * allocation-free decode clears the word.  Synchronises `stream`; allocates nothing.
 */
dms_status dms_selftest_noalloc_timeout(int64_t limit_ns, void* stream);

/*
 * Self-test of the per-head completion flags of the cluster decode kernel (no counterpart
 * in the paper).  Makes the next cluster launch of `layer` wait, with the limit `limit_ns`
 * (1 us .. 10 s), for a flag value no launch ever published: each head's wait gives up,
 * records DMS_ERR_TIMEOUT (sticky, read with dms_cache_stats; cleared by dms_cache_reset)
 * and falls back to the dependency wait, so that launch still reads the completed state and
 * computes the right result.  Host only (nothing is launched here).  Errors:
 * DMS_ERR_INVALID_ARGUMENT (NULL cache, layer out of range, limit out of range).
 */
dms_status dms_selftest_stale_flag(dms_cache* cache, int32_t layer, int64_t limit_ns);

/*
 * Self-test of the bounded wait every kernel of this library uses on its
 * shared-memory barriers (the paper has no counterpart: this is failure
 * detection of the implementation).  Launches one small kernel in which a thread
 * waits on a barrier that a second thread completes only if `arrive` is non-zero.
 * Returns DMS_OK when the wait completed, DMS_ERR_TIMEOUT when it gave up after
 * `limit_ns` nanoseconds (1 us .. 10 s; the kernels use 2 s) -- in both cases the
 * kernel exits normally and the CUDA context stays usable.  Synchronises `stream`;
 * allocates and frees a few bytes of device memory.
 */
dms_status dms_selftest_bounded_wait(int32_t arrive, int64_t limit_ns, void* stream);

/* Static description of a status code. */
const char* dms_status_string(dms_status status);

#ifdef __cplusplus
}
#endif

#endif /* DMS_H_ */
