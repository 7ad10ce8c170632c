/*
 * swan.h -- C ABI of libswan, the SWAN decode hot path on one GB300 (sm_103a).
 *
 * SWAN ("Sparse Winnowed Attention", arXiv 2511.18936) keeps each attention
 * head's key/value history as rotated, pruned sparse vectors plus a small
 * dense buffer of recent vectors, and attends to that cache directly, with no
 * reconstruction.  This library owns the cache in GPU memory and provides:
 *
 *   swan_init          allocate a cache for L layers (Section 4.3's hybrid
 *                      cache; Section 5.1's sparse format)
 *   swan_append        rotate new keys/values by R and insert them
 *                      (Algorithm 1: projection, buffer insert, eviction of
 *                      the oldest vectors with magnitude top-k pruning)
 *   swan_flush_buffer  prune every buffered vector into the sparse history
 *   swan_decode        one decode step of attention over the hybrid cache
 *                      (Algorithm 1: rotated query, sparse-dense and
 *                      dense-dense score products, softmax, value product),
 *                      followed by the rotate-back o = o_hat R_vo^T
 *                      (Appendix A.1, Lemma 2)
 *   swan_append_decode a decode step's append and decode in one call (the
 *                      query rotation runs inside the append's launch)
 *   swan_set_k         runtime keep count (Section 1 contributions, Section
 *                      4.3: the pruning threshold is tunable at inference)
 *
 * Conventions (all entry points):
 *   - Row vectors, as in Section 4.2: x_hat[j] = sum_i x[i] * R[i][j].
 *   - head_dim d must be 128 (uint8 indices, Section 5.1).
 *   - Every pointer named "device" is a CUDA device pointer on the device
 *     that was current at swan_init; the caller keeps ownership of it.
 *   - Work is enqueued asynchronously on cfg.stream; nothing synchronises
 *     except swan_debug_export, swan_check and swan_timing_read.
 *   - Argument and capacity checks happen on the host before any launch; a
 *     failed check returns an error and leaves the cache unchanged.
 *   - A CUDA error during a launch returns SWAN_ERR_CUDA; the context is then
 *     poisoned and every later call returns SWAN_ERR_STATE.
 *   - No call allocates device memory after swan_init.
 *   - One context per stream; a context is not thread-safe.
 *   - Rows (sequences) of a batch may differ in length (swan_append_varlen,
 *     swan_reset_sequence); equal-length batches take the uniform fast path
 *     of every kernel.
 *   - Nothing throws across the ABI and nothing calls abort().
 */
#ifndef SWAN_H
#define SWAN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum swan_status {
  SWAN_OK = 0,
  SWAN_ERR_INVALID_ARG = 1,    /* bad pointer, size, layer, k, ... */
  SWAN_ERR_UNSUPPORTED = 2,    /* valid but not built (e.g. head_dim != 128) */
  SWAN_ERR_CAPACITY = 3,       /* would exceed max_seq; nothing was changed */
  SWAN_ERR_CUDA = 4,           /* a CUDA runtime call failed */
  SWAN_ERR_STATE = 5,          /* context poisoned by an earlier CUDA error */
  SWAN_ERR_DEVICE_TIMEOUT = 6, /* a bounded device wait ran out */
  SWAN_ERR_NOMEM = 7,          /* device or host allocation failed in init */
  SWAN_ERR_DEVICE_CHECK = 8    /* a device-side consistency check failed */
} swan_status;

typedef struct swan_ctx swan_ctx; /* opaque; owned by the library */

typedef struct swan_config {
  int num_layers;  /* >= 1 */
  int batch;       /* B >= 1 */
  int n_q_heads;   /* H_q, a multiple of n_kv_heads */
  int n_kv_heads;  /* H_kv; G = H_q / H_kv query heads share a kv head
                      (Section 4.1.1); G must be 1, 2, 4 or 8 */
  int head_dim;    /* d, must be 128 */
  int k_store;     /* kept entries stored per vector, 1..d; the runtime keep
                      count k_active may be any value 1..k_store */
  int buffer_cap;  /* b, dense buffer capacity in tokens, 0..4096 */
  int max_seq;     /* tokens per sequence the cache can hold (sparse + buffer) */
  int page_tokens; /* tokens per cache page, a power of two in [32, 4096];
                      0 = 128 */
  void* stream;    /* cudaStream_t the context enqueues on; NULL = default */
  int value_format; /* SWAN_VALUES_FP16 (0, default) or SWAN_VALUES_FP8_E4M3:
                       kept sparse values stored as 8-bit floats (Section 4.3,
                       Section 5.1: 2k bytes per vector instead of 3k),
                       E4M3, round to nearest even, saturating to +-448; the
                       entries are still chosen on the fp16 vector and the
                       dense buffer stays fp16 */
  int k_store_v;   /* value entries kept per vector, 1..d; 0 = k_store.  Keys
                      and values may keep different counts (Appendix,
                      ablation on key and value pruning ratios) */
  int pool_pages;  /* 0: every (layer, row, kv head) owns the pages for
                      max_seq tokens.  > 0: one pool of this many pages for
                      all layers and rows; a row takes pages as its sparse
                      history grows and returns them at swan_reset_sequence,
                      so rows of different lengths share the memory
                      (PagedAttention-style paging, Section 2's serving
                      context).  An append or flush that needs more pages
                      than are free returns SWAN_ERR_CAPACITY and changes
                      nothing. */
} swan_config;

enum { SWAN_VALUES_FP16 = 0, SWAN_VALUES_FP8_E4M3 = 1 };

/*
 * Create a context.  R_qk, R_vo: device fp32 [num_layers][n_kv_heads][d][d],
 * row-major, orthogonal (P_QK and P_VO of Section 4.1.2).  R_vo == NULL uses
 * R_qk for the values too.  Both are copied; the caller may free them after
 * the call returns.  All cache memory is allocated here, once.
 * On success *out receives the context and k_active = k_store.
 * Errors: INVALID_ARG, UNSUPPORTED, NOMEM, CUDA.  *out is NULL on error.
 */
swan_status swan_init(swan_ctx** out, const swan_config* cfg,
                      const float* R_qk, const float* R_vo);

/* Release every resource of the context (synchronises its stream).
 * NULL is accepted and ignored. */
swan_status swan_destroy(swan_ctx* ctx);

/*
 * Set the runtime keep count (Section 4.3; Section 1 lists runtime
 * tunability as a contribution).  Entries are stored in decreasing magnitude
 * order, so decoding with k_active < k_store uses exactly the top-k_active
 * entries of every cached vector: the same result as a cache built with
 * k_store = k_active.  Applies to decodes enqueued after the call.
 * Errors: INVALID_ARG unless 1 <= k_active <= k_store.
 */
swan_status swan_set_k(swan_ctx* ctx, int k_active);

/*
 * Separate runtime keep counts for keys (1..k_store) and values
 * (1..k_store_v) (Appendix, ablation on key and value pruning ratios).
 * swan_set_k(ctx, k) is swan_set_kv(ctx, k, min(k, k_store_v)).
 * Errors: INVALID_ARG when a count is out of range.
 */
swan_status swan_set_kv(swan_ctx* ctx, int k_active, int k_active_v);

/*
 * Append T tokens to every sequence of one layer (Algorithm 1, generalised
 * to T tokens at once).
 *   k_new, v_new: device fp16 [batch][n_kv_heads][T][d], 16-byte aligned,
 *   post-RoPE keys and unrotated values.  The library rotates them:
 *   k_hat = k R_qk, v_hat = v R_vo, to fp32 accuracy (decode-step appends on
 *   the CUDA cores; bulk appends on the tensor cores with R split into fp16
 *   hi + 2^-12 lo parts), rounded to fp16 round-to-nearest-even.
 * If buffer_count + T > buffer_cap, the oldest (buffer_count + T - buffer_cap)
 * vectors of (buffer, then new tokens) are pruned to their k_store
 * largest-magnitude coordinates (ties to the lower index; keys and values
 * separately) and appended to the sparse history, in order; the rest stay
 * dense in the buffer.  T == 0 is a no-op.
 * Errors: INVALID_ARG (layer, T < 0, NULL, misaligned), CAPACITY (sparse +
 * buffer would exceed max_seq, or the page pool is exhausted), STATE, CUDA.
 */
swan_status swan_append(swan_ctx* ctx, int layer, const void* k_new,
                        const void* v_new, int T);

/*
 * Prune every buffered vector of a layer into the sparse history (oldest
 * first); the buffer becomes empty.  layer == -1 flushes all layers.
 * Errors: INVALID_ARG, STATE, CUDA.
 */
swan_status swan_flush_buffer(swan_ctx* ctx, int layer);

/*
 * Append a different number of tokens to each row (sequence) of the batch:
 * row b takes the first n_new[b] (0..T) of the T tokens given for it; the
 * rest of k_new / v_new ([batch][n_kv_heads][T][d] fp16, device) is ignored.
 * Each row then follows Algorithm 1 on its own: its buffer evicts its oldest
 * tokens beyond b_cap into its sparse history.  Rows may thus differ in
 * length; every call works per row from then on (swan_decode attends each
 * row over its own tokens; a row with no token outputs zeros).
 * n_new: HOST int32 [batch].  Errors: INVALID_ARG (n_new out of range),
 * CAPACITY (a row beyond max_seq, or the page pool exhausted); nothing
 * changes on error.
 */
swan_status swan_append_varlen(swan_ctx* ctx, int layer, const void* k_new, const void* v_new, int T,
                               const int32_t* n_new);

/*
 * Forget row b in every layer (a finished request): its tokens are dropped
 * and, with a page pool, its pages return to the pool.  Host-side only; the
 * next call on the row starts from an empty cache.  Errors: INVALID_ARG.
 */
swan_status swan_reset_sequence(swan_ctx* ctx, int b);

/*
 * Make row dst a copy of row src in every layer (parallel sampling, beam
 * search: several continuations of one prompt).  Afterwards dst attends over
 * the same history and dense buffer as src, and the two rows go on
 * independently.  Requires a page pool (pool_pages > 0).  dst's own tokens
 * are dropped first, as by swan_reset_sequence.  The sparse pages are
 * shared, not copied: appends only ever write into a row's last, partly
 * filled page, so a row that is about to write into a page other rows still
 * hold gets its own copy first (copy on write, counted against the pool);
 * a page returns to the pool when no row holds it.  The dense buffer is
 * per row and is copied (device to device, on the context's stream).
 * Errors: INVALID_ARG (rows out of range or equal), UNSUPPORTED (no page
 * pool), CUDA.
 */
swan_status swan_fork_sequence(swan_ctx* ctx, int src, int dst);

/*
 * One decode step of attention for one layer (Algorithm 1, attention part):
 *   q:   device fp16 [batch][n_q_heads][d], post-RoPE, unrotated.
 *   out: device fp16 [batch][n_q_heads][d], written as
 *        out = softmax((q R_qk) K_cache^T / sqrt(d)) V_cache R_vo^T
 *        where K_cache / V_cache are the rotated sparse history (first
 *        k_active stored entries of each vector) followed by the dense
 *        buffer.  Query head h attends to kv head h / G.
 * Attends over every token appended so far.  With an empty cache out is 0.
 * q and out must not overlap.  Errors: INVALID_ARG, STATE, CUDA.
 */
swan_status swan_decode(swan_ctx* ctx, int layer, const void* q, void* out);

/*
 * One serving step of a layer (Algorithm 1 in full: compress the step's new
 * tokens, then attend): exactly swan_append_varlen(ctx, layer, k_new, v_new,
 * T, n_new) followed by swan_decode(ctx, layer, q, out), with the same
 * arguments, results and errors (n_new may be NULL: every row takes T
 * tokens).  A decode-step append (few vectors) computes the query rotation
 * q' = q R_qk in its own launch, so the step takes two launches instead of
 * three; q' has the same bits as swan_decode's.  With timing enabled, that
 * launch counts as SWAN_KERNEL_APPEND.  q and out are checked before
 * anything runs: on any error nothing is appended and nothing is decoded.
 */
swan_status swan_append_decode(swan_ctx* ctx, int layer, const void* k_new, const void* v_new, int T,
                               const int32_t* n_new, const void* q, void* out);

/* Host-side view of a layer's cache (no synchronisation). */
typedef struct swan_layer_info {
  int64_t sparse_len;   /* tokens per sequence in the sparse history */
  int64_t buffer_len;   /* tokens per sequence in the dense buffer */
  int k_active;
  int k_store;
  int k_slots;          /* k_store rounded up to a multiple of 8 */
  int page_tokens;
  int64_t page_bytes;   /* bytes of one page (keys and values) */
  int64_t device_bytes; /* device memory owned by the whole context */
  int value_format;     /* SWAN_VALUES_FP16 or SWAN_VALUES_FP8_E4M3 */
  int k_active_v;       /* value entries used per vector */
  int k_store_v;        /* value entries stored per vector */
  int k_slots_v;        /* k_store_v rounded up to a multiple of 8 */
  int uniform;          /* 1 if every row has the same lengths; sparse_len and
                           buffer_len above are the largest over the rows */
  int64_t pool_pages;   /* pages in the pool (all layers) */
  int64_t free_pages;   /* free pages of a shared pool (pool_pages > 0) */
} swan_layer_info;

/* Per-row lengths of a layer: sparse_len, buffer_len HOST arrays [batch]. */
swan_status swan_query_lengths(const swan_ctx* ctx, int layer, int64_t* sparse_len, int32_t* buffer_len);

swan_status swan_query(const swan_ctx* ctx, int layer, swan_layer_info* info);

/*
 * Copy part of a layer's cache to host memory, in a canonical layout
 * (synchronises the stream).  For tests and debugging.
 *   SWAN_EXPORT_BUFFER_K / _V: fp16 [batch][n_kv_heads][buffer_len][d],
 *     oldest first.
 *   SWAN_EXPORT_SPARSE_K / _V: uint8 indices [batch][n_kv_heads]
 *     [sparse_len][k_store] (k_store_v for _V), then fp16 values of the same
 *     shape, each vector's
 *     entries in stored (decreasing magnitude) order (8-bit values are
 *     widened to fp16, exactly).
 * bytes must equal the exact size of the requested view.  Every row must
 * have the same lengths (else INVALID_ARG: export the rows one at a time).
 * Errors: INVALID_ARG (what, layer, size), STATE, CUDA.
 */
enum {
  SWAN_EXPORT_BUFFER_K = 1,
  SWAN_EXPORT_BUFFER_V = 2,
  SWAN_EXPORT_SPARSE_K = 3,
  SWAN_EXPORT_SPARSE_V = 4
};
swan_status swan_debug_export(swan_ctx* ctx, int layer, int what,
                              void* host_dst, size_t bytes);

/* The same for row b alone: shapes [n_kv_heads][len_b][...]. */
swan_status swan_debug_export_seq(swan_ctx* ctx, int layer, int b, int what, void* host_dst, size_t bytes);

/*
 * Synchronise the stream and read the device status word that kernels set
 * when a device-side consistency check fails (for instance a page-table
 * entry out of range, or too little shared memory for a kernel's aligned
 * layout; such a kernel skips the access or the launch instead of faulting) or
 * a bounded wait of a tensor-core pipeline gave up (2 s; the launch's
 * results are then invalid).  Returns OK, DEVICE_TIMEOUT or DEVICE_CHECK
 * (and clears the word), STATE or CUDA.
 */
swan_status swan_check(swan_ctx* ctx);

/*
 * Per-kernel timing with CUDA events on the context's stream.  While enabled,
 * every launch is bracketed by an event pair; swan_timing_read synchronises,
 * sums the elapsed times per kernel kind and resets the sums.
 */
enum {
  SWAN_KERNEL_ROTATE_Q = 0, /* q' = q R_qk */
  SWAN_KERNEL_DECODE = 1,   /* split decode over the packed cache */
  SWAN_KERNEL_COMBINE = 2,  /* split combine + rotate-back */
  SWAN_KERNEL_APPEND = 3,   /* rotate new tokens; buffer insert or prune */
  SWAN_KERNEL_PRUNE = 4,    /* prune buffered vectors (eviction, flush) */
  SWAN_KERNEL_KINDS = 8
};
typedef struct swan_timing {
  double ms[SWAN_KERNEL_KINDS];
  int64_t launches[SWAN_KERNEL_KINDS];
} swan_timing;
swan_status swan_timing_enable(swan_ctx* ctx, int enable);
swan_status swan_timing_read(swan_ctx* ctx, swan_timing* out);

/*
 * Decode without allocating: the paper has no counterpart; this is a
 * deployment interface for callers that cannot call cudaMalloc, such as an
 * engine that hands out all device memory from its own reserved pool and
 * must not see a hidden allocation, or that reserves its memory budget up
 * front.  swan_init allocates the cache and per-call scratch with cudaMalloc;
 * this entry point instead decodes over a cache held in the caller's own
 * device memory and keeps its scratch (rotated queries and split partials)
 * in a fixed static device array inside the library.  It calls no cudaMalloc,
 * cudaFree or other allocating routine.
 *
 * view: the caller's cache, all pointers device pointers on the current
 *   device, caller-owned:
 *   pages       page pool; page p holds P = page_tokens tokens as P/32
 *               blocks of 32 tokens; keys keep ks = k_slots and values
 *               vs = k_slots_v entries.  With fp16 values a block is
 *               96 * (ks + vs) bytes: K values [ks/8][32][8] fp16 at 0,
 *               K indices [ks/8][32][8] uint8 at 64 * ks, V values
 *               [vs/8][32][8] at 96 * ks, V indices at 96 * ks + 64 * vs.
 *               With E4M3 values a block is 64 * (ks + vs) bytes: K records
 *               [ks/8][32][16 bytes] at 0 (8 E4M3 values, then 8 indices),
 *               V records [vs/8][32][16 bytes] at 64 * ks.  Page p starts at
 *               pages + p * (P / 32) * block bytes.  Chunk c of token t holds
 *               entries 8c..8c+7 of the token's kept coordinates in
 *               decreasing magnitude order; indices must be < 128.  This is
 *               the layout swan_init's own pool uses.
 *   page_table  int32 [batch * n_kv_heads][pages_per_unit]: page of the
 *               unit's sparse tokens p*P .. p*P+P-1; entries index `pages`
 *               and must be < num_pages.
 *   buf_k/v     fp16 [batch * n_kv_heads][buffer_cap][d] rotated dense ring;
 *               buffered token i (oldest first) is at slot
 *               (buf_start + i) % buffer_cap.
 *   R_qk        fp32 [n_kv_heads][d][d]; R_vo_t fp32 [n_kv_heads][d][d]
 *               holding R_vo transposed (R_vo_t[h][j][i] = R_vo[h][i][j]).
 * q, out: device fp16 [batch][n_q_heads][d]; out as for swan_decode.
 * stream: cudaStream_t (NULL = default stream).
 *
 * Limits of the static scratch (about 1.6 MB per device, held from the
 * library's first use on that device until the process exits):
 * batch * n_q_heads <= 1024 and (decode CTAs + batch * n_kv_heads) * G <=
 * 2048, where decode CTAs is at most (SM count x resident CTAs per SM; 152 on
 * a GB300).  Larger sizes return SWAN_ERR_INVALID_ARG with a message.
 * Alignment: pages, buf_k, buf_v, R_qk and R_vo_t 16 bytes, q 8 bytes,
 * page_table 4 bytes, out 2 bytes (the kernels' widest accesses); a
 * misaligned pointer returns SWAN_ERR_INVALID_ARG before anything is enqueued.
 * The first call on a device resolves the scratch address and the grid limits
 * (cudaGetSymbolAddress, occupancy queries); make that first call before any
 * stream capture.  The address is resolved again if the device's context is
 * re-created (cudaDeviceReset).  Every call on a device shares the one scratch
 * array, which keeps the last call's contents: calls that overlap on the GPU
 * (different streams, or different host threads) race and give wrong
 * results; serialise them.  Device-side consistency checks (a page-table
 * entry out of range, a kernel skipped for too little shared memory) are
 * recorded in a status word of the scratch that each call clears first;
 * swan_noalloc_check reads it.  Errors: INVALID_ARG, UNSUPPORTED, CUDA.
 */
typedef struct swan_cache_view {
  const void* pages;
  const int32_t* page_table;
  int64_t num_pages;
  int pages_per_unit;
  int page_tokens;       /* P, a power of two in [32, 4096] */
  int k_slots;           /* entries stored per vector, multiple of 8, <= 128 */
  int k_active;          /* entries used, 1..k_slots */
  const void* buf_k;
  const void* buf_v;
  int buffer_cap;
  int buf_start;
  int buf_len;
  int64_t sparse_len;    /* sparse tokens per sequence */
  int batch;
  int n_q_heads;
  int n_kv_heads;
  int head_dim;          /* must be 128 */
  const float* R_qk;
  const float* R_vo_t;
  int value_format;      /* SWAN_VALUES_FP16 or SWAN_VALUES_FP8_E4M3 */
  int k_slots_v;         /* value entries stored per vector; 0 = k_slots */
  int k_active_v;        /* value entries used; 0 = k_active */
} swan_cache_view;
swan_status swan_decode_noalloc(const swan_cache_view* view, const void* q, void* out,
                                void* stream);

/*
 * Status of the last swan_decode_noalloc on the current device: synchronises
 * `stream` (the one that call used), reads the scratch's status word and
 * clears it.  Allocates nothing.  Returns OK, DEVICE_CHECK (the last call's
 * output is not valid: a page-table entry out of range or a kernel skipped),
 * DEVICE_TIMEOUT, or CUDA.
 */
swan_status swan_noalloc_check(void* stream);

/* Number of kernels this context has launched since swan_init. */
int64_t swan_launch_count(const swan_ctx* ctx);

/*
 * Test hooks.  Every device buffer of a context sits between guard regions
 * (64 KB before, 256 bytes after) filled with 0xA5 at swan_init;
 * swan_debug_check_guards
 * synchronises the stream and returns SWAN_ERR_DEVICE_CHECK (naming the
 * buffer) if a kernel wrote into one, else SWAN_OK (STATE, CUDA as usual).
 *
 * swan_debug_fail_after makes the library fail on the host, without calling
 * CUDA, at the (n+1)-th next device allocation (SWAN_FAULT_ALLOC: the call
 * returns SWAN_ERR_NOMEM, and swan_init frees what it had allocated) or
 * kernel launch (SWAN_FAULT_LAUNCH: nothing is launched, the call returns
 * SWAN_ERR_CUDA and the context is poisoned), counted over all contexts of
 * the process; it fires once.  n = -1 turns it off.  Not for concurrent
 * use.  Errors: INVALID_ARG (kind, n < -1).
 */
enum { SWAN_FAULT_ALLOC = 1, SWAN_FAULT_LAUNCH = 2 };
swan_status swan_debug_fail_after(int kind, int64_t n);
swan_status swan_debug_check_guards(swan_ctx* ctx);

/*
 * Test hook for the bounded device waits of the tensor-core kernels (the
 * bulk append of swan_append, and swan_gram of swan_basis.h): the next such
 * launch in the process issues none of its TMA copies, so the barrier its
 * MMA thread waits on is never completed; that wait, and every other barrier
 * wait of the launch, gives up after limit_ns nanoseconds (instead of 2 s),
 * sets the timeout bit of the status word and the kernel returns, with no
 * copy or MMA left in flight and its tensor memory freed.  swan_check (or
 * swan_basis_check) then returns SWAN_ERR_DEVICE_TIMEOUT.  The starved
 * launch's results are invalid: for an append, the context's cache no longer
 * matches its host-side lengths and the context should be destroyed.  Fires
 * once; limit_ns = 0 disarms it.  Not for concurrent use.
 * Errors: INVALID_ARG unless limit_ns == 0 or 1e3 <= limit_ns <= 2e9.
 */
swan_status swan_debug_starve_tc(int64_t limit_ns);

/* Static string for a status code. */
const char* swan_status_string(swan_status s);

/* Detail of the last error returned on this thread ("" if none). */
const char* swan_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* SWAN_H */
