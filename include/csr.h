/*
 * csr.h -- C ABI of the CSR incremental-prefill attention library (libcsr.so).
 *
 * The library keeps one transformer layer's key/value cache for the Cached
 * State Representation of section III-D of the paper:
 *
 *     T_t = (X_static, X_dyn),  X_static = (X_pre, X_chunks),  X_dyn = (X_suff, X_task)
 *
 * X_pre is cached once (csr_init_static), state chunks are appended
 * (csr_append_chunk, Theorem 2 / Eq. incremental_extensibility), the dynamic
 * suffix is attended and dropped again every task (csr_attend_suffix,
 * csr_truncate_suffix; Eq. x_dynamic), and old chunks are evicted
 * (Eq. eviction_operation) with the asynchronous state reconciliation of
 * Algorithm 1 (csr_evict_and_reconcile, csr_poll_swap).  Every call that adds
 * tokens rotates them with RoPE at their absolute positions, appends their
 * keys/values to a paged cache and returns the causal attention of their
 * queries over the whole cached context (Eq. causal_attention_1..3).
 *
 * Conventions shared by every entry point
 *   - Tensors are bfloat16 in row-major, token-major layout:
 *       q, out   [n][num_q_heads][head_dim]
 *       k, v     [n][num_kv_heads][head_dim]
 *       lse      [num_q_heads][n] float32, natural log of the softmax
 *                normaliser sum_tau exp(scale * q.k_tau)
 *     All tensor pointers are DEVICE pointers of the current CUDA device,
 *     16-byte aligned, owned by the caller, borrowed for the call only (the
 *     pools and the workspace are borrowed for the context's lifetime).
 *   - Compute calls are asynchronous: they enqueue kernels on the given
 *     stream and return.  Inputs must stay valid until that work has run.
 *   - Foreground calls share one workspace; issue them on one stream, or
 *     order them yourself.
 *   - Errors are returned as csr_status; nothing is thrown across the ABI.
 *     A call that fails with CSR_EINVAL, CSR_ESTATE or CSR_ENOMEM changes
 *     nothing.  csr_last_error() describes the last failure.
 *   - Query head h reads key/value head h / (num_q_heads / num_kv_heads).
 *   - RoPE pairs element i with element i + head_dim/2 (rotate-half) and
 *     turns the pair by pos * rope_base^(-2i/head_dim).
 *   - A context is not thread-safe: call it from one host thread at a time.
 */
#ifndef CSR_H_
#define CSR_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same object as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st *csr_stream_t;

typedef struct csr_ctx csr_ctx;

typedef enum csr_status {
  CSR_OK = 0,
  CSR_EINVAL = 1,   /* bad argument or configuration */
  CSR_ENOMEM = 2,   /* the page pool or a version's page table is full */
  CSR_ESTATE = 3,   /* call not allowed in the current state */
  CSR_EBUSY = 4,    /* a reconciliation is already running */
  CSR_ECUDA = 5,    /* a CUDA runtime or driver call failed */
  CSR_ETIMEOUT = 6, /* a bounded host-side wait ran out */
  CSR_EDEVICE = 7   /* a kernel reported an error word (see csr_device_status) */
} csr_status;

/* Bits of the device error word. */
#define CSR_DEVERR_WAIT_TIMEOUT 0x1u /* a pipeline wait inside a kernel gave up */
#define CSR_DEVERR_BAD_PAGE 0x2u     /* a page id outside the pool was met */
#define CSR_DEVERR_ALLOC 0x4u        /* the compaction kernel found too few free pages */

/* csr_config.flags */
#define CSR_FLAG_PLAN_ONLY 0x1   /* layout planning only: no device memory is touched
                                    and no kernel runs; compute calls update the page
                                    tables and lengths but produce no outputs */
#define CSR_FLAG_FUSED_ALWAYS 0x2 /* every foreground call is one cooperative launch of the
                                     fused kernel (RoPE + append, attention, merge) */
#define CSR_FLAG_FUSED_NEVER 0x4  /* every foreground call is three chained launches (RoPE +
                                     append, attention items, merge of split items); by
                                     default a call takes the fused launch when its attention
                                     work is at least 600 key tiles per CTA and it has at
                                     most two units (kv head x pair of 128-row query tiles)
                                     per CTA */
#define CSR_FLAG_SCHEDULE_LOCAL 0x10 /* the fused launch takes least-advanced-first steps of 128
                                       key tiles where they keep the load within 1 % of the
                                       default idle-interval schedule's and cut at most twice as
                                       many units: the keys in use stay within ~128 tiles of each
                                       other (120K step: 456 instead of 647 MB of DRAM traffic
                                       per launch) at ~1.5 % more time */
#define CSR_FLAG_UNPACED_REBUILD 0x8 /* the reconciliation thread enqueues each rebuild task
                                        as soon as it is due; by default it keeps one task
                                        (one chunk's recomputation, or the compaction) in
                                        flight on the low-priority stream and starts it only
                                        once the foreground work enqueued before it has
                                        finished, so that a foreground call finds at most
                                        one short task's CTAs on the SMs */

typedef struct csr_config {
  int32_t num_q_heads;    /* H_q */
  int32_t num_kv_heads;   /* H_kv; H_q / H_kv must be a power of two <= 128 */
  int32_t head_dim;       /* 64 or 128 */
  int32_t page_size;      /* tokens per cache page: 16, 32, 64 or 128 */
  double rope_base;       /* RoPE base (e.g. 1e4, 1e6) */
  float softmax_scale;    /* 0 selects 1/sqrt(head_dim) (Eq. causal_attention_1) */
  int32_t max_new_tokens; /* largest n of one call, and of one chunk */
  int32_t pool_pages;     /* physical pages in each of the K and V pools (<= 65536) */
  int32_t max_seq_tokens; /* largest length of one cache version */
  int32_t cap_tokens;     /* tau_mem of Algorithm 1; 0 disables automatic eviction */
  int32_t evict_tokens;   /* tokens of the oldest chunks dropped by an automatic eviction */
  int32_t n_catchup;      /* N_catchup of Algorithm 1 */
  int32_t num_ctas;       /* CTAs of a foreground attention launch (at most one per SM);
                             0 = one per SM */
  int32_t rebuild_tiles_per_cta; /* key tiles (128 keys) per CTA in rebuild launches; 0 = 16 */
  int32_t flags;          /* CSR_FLAG_* */
  int32_t fg_chunk_tiles; /* > 0: a foreground launch cuts every unit's key range into
                             pieces of at most this many 128-key tiles (the three-launch
                             path: chunks of exactly this many, more if the split partials
                             would not fit); 0 = the fused launch cuts only as balance
                             needs, the three-launch path picks the chunk length from a
                             cost estimate (the default) */
  float rebuild_duty;     /* share of wall time the paced reconciliation thread lets the
                             rebuild occupy the GPU (after a task it waits task time *
                             (1 / duty - 1) before the next): a lower share keeps the
                             chip's power, and with it the foreground's clock, down while
                             a rebuild runs; 0 or >= 1 = no wait (the default) */
} csr_config;

/*
 * Sizes of the caller-allocated device buffers for a configuration.
 * csr_pool_bytes: bytes of EACH of the K and V pools, laid out
 *   [pool_pages][num_kv_heads][page_size][head_dim] bfloat16.
 * csr_workspace_bytes: bytes of the workspace (staging, split partials, page
 *   tables, error word).  Both return 0 for an invalid configuration.
 */
size_t csr_pool_bytes(const csr_config *cfg);
size_t csr_workspace_bytes(const csr_config *cfg);

/*
 * Create a context on the current CUDA device.  k_pool, v_pool (csr_pool_bytes
 * each, 256-byte aligned) and workspace (csr_workspace_bytes, 256-byte aligned)
 * are borrowed until csr_destroy; create zero-fills them on `stream`.
 * With CSR_FLAG_PLAN_ONLY the three pointers may be NULL and no CUDA call is
 * made.  On success *out receives the context.
 */
csr_status csr_create(const csr_config *cfg, void *k_pool, void *v_pool,
                      void *workspace, csr_stream_t stream, csr_ctx **out);

/* Release the context (synchronises its streams first).  NULL is a no-op. */
void csr_destroy(csr_ctx *ctx);

/*
 * X_pre (Eq. x_static): cache the static prefix at positions 0..n-1 and write
 * its causal self-attention to out (and lse when not NULL).  Once per context,
 * before any other compute call; 1 <= n <= max_new_tokens.  Prefixes longer
 * than max_new_tokens are built by csr_init_static followed by chunks.
 */
csr_status csr_init_static(csr_ctx *ctx, const void *q, const void *k,
                           const void *v, int32_t n, void *out, float *lse,
                           csr_stream_t stream);

/*
 * Increment of Algorithm 1: append the state chunk x_t at positions
 * len..len+n-1 of the active version, attend its queries over the whole cache,
 * and return its id in *chunk_id (may be NULL).  While a reconciliation runs
 * the chunk is also reserved in the version being rebuilt and buffered for its
 * catch-up; with n_catchup = 0 its catch-up is enqueued on the low-priority
 * stream at once (the provider is called for it inside this call).  If a reconciler is set, cap_tokens > 0 and the length reaches
 * cap_tokens, an eviction of evict_tokens starts (Algorithm 1, Increment); if
 * it cannot start, the chunk stays appended and its error code is returned.
 * CSR_ESTATE while a suffix is live.
 */
csr_status csr_append_chunk(csr_ctx *ctx, const void *q, const void *k,
                            const void *v, int32_t n, void *out, float *lse,
                            csr_stream_t stream, int64_t *chunk_id);

/*
 * X_dyn = (X_suff, X_task) (Eq. x_dynamic, i* = |X_static| + 1 of
 * Eq. csr_i_star): append the transient suffix at positions len..len+n-1 and
 * attend it causally over the cache.  At most one suffix is live: CSR_ESTATE
 * otherwise.
 */
csr_status csr_attend_suffix(csr_ctx *ctx, const void *q, const void *k,
                             const void *v, int32_t n, void *out, float *lse,
                             csr_stream_t stream);

/*
 * One task step in one pass: csr_append_chunk of the first n_chunk tokens
 * followed by csr_attend_suffix of the next n_suffix, computed as a single
 * causal block of n_chunk + n_suffix tokens (the chunk's tokens see the cache
 * and the chunk, the suffix's see the cache, the chunk and the suffix: the
 * same results as the two calls, with one RoPE/append launch, one pass of the
 * attention over the cache and at most one merge).  q, k, v, out and lse hold
 * the n_chunk + n_suffix tokens, chunk first.  The chunk joins X_static
 * (*chunk_id as for csr_append_chunk) and the suffix stays live until
 * csr_truncate_suffix.  When the chunk brings the static length to cap_tokens,
 * the eviction of Algorithm 1 starts at that truncation (ordered after the
 * work enqueued on `stream`).  CSR_EINVAL if either count is < 1 or their sum
 * exceeds max_new_tokens; CSR_ESTATE as for csr_append_chunk.
 */
csr_status csr_append_chunk_attend_suffix(csr_ctx *ctx, const void *q, const void *k,
                                          const void *v, int32_t n_chunk, int32_t n_suffix,
                                          void *out, float *lse, csr_stream_t stream,
                                          int64_t *chunk_id);

/*
 * Drop the live suffix: the length returns to |X_static| and the pages that
 * hold only suffix slots go back to the pool.  Host-only (no kernel), unless a
 * fused csr_append_chunk_attend_suffix reached cap_tokens: then the eviction
 * starts here (as csr_evict_and_reconcile would) and its status is returned.
 * CSR_ESTATE when no suffix is live.
 */
csr_status csr_truncate_suffix(csr_ctx *ctx);

/*
 * Invalidate the cache after its first `length` tokens (section III-B: a
 * cache stays valid up to the first differing token i*, Eq.
 * first_differing_token, so a task that differs from position length+1 on
 * reuses exactly this much).  `length` must be the end of the static prefix or
 * of a chunk of the active version; the later chunks are dropped and their
 * pages return to the pool.  Host-only (no kernel).  CSR_ESTATE while a suffix
 * is live or a reconciliation runs, CSR_EINVAL if length is not a boundary.
 */
csr_status csr_rewind(csr_ctx *ctx, int64_t length);

/*
 * Source of a chunk's layer inputs for the rebuild (the "LLM(X_eps)" of
 * Algorithm 1 recomputes a retained chunk in its new context).  The callback
 * is called on the context's reconciliation thread (a library thread started
 * by csr_set_reconciler; one call at a time, in rebuild order), with the
 * chunk's id and length, and must set *q, *k, *v to device pointers holding
 * that chunk's pre-RoPE queries/keys/values in the layouts above, valid until
 * the reconciliation that asked for them has swapped or failed.  Their
 * contents must be complete when the callback returns or ordered before the
 * fg_stream position of the call that started the reconciliation (or, for a
 * chunk appended during it, of that append).  It may set *out to a device
 * buffer [n][num_q_heads][head_dim] that receives the chunk's rebuilt
 * attention output, or leave it NULL.  Returns 0 on success; any other value
 * aborts the reconciliation (the active version stays as it is), reported by
 * the next csr_poll_swap / csr_wait_reconcile as CSR_ESTATE.
 */
typedef int (*csr_qkv_provider)(void *user, int64_t chunk_id, int32_t n_tokens,
                                const void **q, const void **k, const void **v,
                                void **out);

/*
 * Register the rebuild source and the low-priority stream on which the
 * rebuild runs (the secondary resource R_2 of Algorithm 1 becomes a stream of
 * the same GPU, fed by a library thread that calls the provider and enqueues
 * the rebuild's launches, so the foreground caller never waits for them).
 * Create lo_stream with a lower priority than the foreground stream.  The
 * thread starts at the first registration and ends in csr_destroy.
 * CSR_EBUSY while a reconciliation runs.
 */
csr_status csr_set_reconciler(csr_ctx *ctx, csr_qkv_provider provider,
                              void *user, csr_stream_t lo_stream);

/*
 * Eviction + asynchronous reconciliation (Eq. eviction_operation, Algorithm 1
 * Reconcile, App. D steps 1-3): drop the oldest whole chunks until at least
 * evict_tokens tokens are gone, reserve a second cache version that shares the
 * prefix's full pages, and enqueue on the low-priority stream the compaction
 * kernel (new page table, copy of a partly filled prefix page) and a fresh
 * causal prefill of every retained chunk at its renumbered position.  Work
 * already enqueued on fg_stream is ordered before the rebuild.  Returns at
 * once, before the provider is called: the reconciliation thread enqueues the
 * rebuild while the active version keeps serving foreground calls.
 * CSR_EBUSY if a reconciliation runs, CSR_ESTATE without a reconciler, with a
 * live suffix or with no chunk to evict, CSR_ENOMEM if the pool cannot hold
 * the second version.  A failure during the rebuild (the provider, a launch)
 * is reported by the next csr_poll_swap / csr_wait_reconcile.
 */
csr_status csr_evict_and_reconcile(csr_ctx *ctx, int32_t evict_tokens,
                                   csr_stream_t fg_stream);

/* Values of *state from csr_poll_swap / csr_wait_reconcile. */
#define CSR_RECON_IDLE 0    /* no reconciliation */
#define CSR_RECON_RUNNING 1 /* rebuild or catch-up still running (or swap deferred) */
#define CSR_RECON_SWAPPED 2 /* this call swapped the versions */

/*
 * Non-blocking step of Algorithm 1's catch-up loop.  Call it between tasks,
 * before the task's first compute call: right after an append that enqueued a
 * catch-up it would see that work unfinished.  When the rebuild's last launch
 * has finished: while more than n_catchup chunks are buffered, enqueue
 * their catch-up on the low-priority stream; otherwise compute the remaining
 * buffered chunks on fg_stream ("computed at next task inference") and swap
 * the active version atomically (App. D step 5).  The old version's own pages
 * return to the pool.  The swap waits while a suffix is live.  If the rebuild
 * failed, the reconciliation is aborted (the pending version's pages return
 * to the pool, the active version stays) and its error is returned.
 */
csr_status csr_poll_swap(csr_ctx *ctx, csr_stream_t fg_stream, int *state);

/*
 * Blocking form of csr_poll_swap: polls until the swap happens or timeout_us
 * microseconds pass (CSR_ETIMEOUT; the reconciliation keeps running).
 */
csr_status csr_wait_reconcile(csr_ctx *ctx, csr_stream_t fg_stream,
                              int64_t timeout_us, int *state);

/*
 * Sequence versions of Algorithm 2: *k is the active version (0 at creation,
 * +1 at every swap); *k_ready is k + 1 once the running reconciliation's
 * rebuild and catch-up are complete up to at most n_catchup buffered chunks
 * (as of the last csr_poll_swap / csr_route), else k.  Host-only.
 */
csr_status csr_get_versions(csr_ctx *ctx, int64_t *k, int64_t *k_ready);

/* Values of *route from csr_route. */
#define CSR_ROUTE_CONTINUE 0  /* k_t = k: serve on the active version (case 1) */
#define CSR_ROUTE_BRIDGE 1    /* k_t = k + 1 before k_ready: serve on the active version;
                                 chunks appended now are forked into the rebuild (case 2) */
#define CSR_ROUTE_SWAPPED 2   /* k_t = k + 1 = k_ready: this call swapped the versions;
                                 serve on the new active version (case 2) */
#define CSR_ROUTE_STRAGGLER 3 /* k_t < k: served on the active version; the paper's
                                 secondary copy of the old sequence is not retained (case 3) */

/*
 * Per-query routing of Algorithm 2 (concurrent request routing): classify a
 * query built on sequence version k_t against the context's versions, and
 * perform the resource swap when the query is the first of the rebuilt
 * version and the rebuild is ready (as csr_poll_swap would; never while a
 * suffix is live).  Progresses the reconciliation like csr_poll_swap.
 * CSR_EINVAL if k_t > k + 1, or k_t = k + 1 without a running reconciliation.
 */
csr_status csr_route(csr_ctx *ctx, int64_t k_t, csr_stream_t fg_stream, int *route);

/*
 * Abandon the running reconciliation (App. D: the swap never happens on a
 * rebuild that did not finish): rebuild work not yet enqueued is dropped, work
 * already on the low-priority stream runs to completion (this call waits for
 * it), and the rebuilt version's pages return to the pool.  The active
 * version is untouched.  CSR_ESTATE when no reconciliation runs.
 */
csr_status csr_cancel_reconcile(csr_ctx *ctx);

/* Result of csr_check_viability (times in seconds, sizes in tokens). */
typedef struct csr_viability {
  double t_warm_s;        /* Delta t_warm: warm-up of the evicted state */
  double delta_n_tokens;  /* Delta N = append rate * Delta t_warm */
  double t_recon_s;       /* Delta t_recon: extension of the rebuilt state by Delta N */
  double t_mem_s;         /* Delta t_mem = N_buffer / append rate */
  double n_buffer_tokens; /* N_buffer: tokens that fit before the page pool runs out */
  double rebuilt_tokens;  /* |T^E|: length of the evicted state (prefix + retained chunks) */
  double pair_seconds;    /* time of one query-key pair of the rebuild that was used */
  int32_t viable;         /* 1 when Delta t_warm + Delta t_recon <= Delta t_mem */
  int32_t measured;       /* 1 when pair_seconds was observed on this context */
} csr_viability;

/*
 * Viability of the asynchronous reconciliation (App. D, Eq. recon_time_inequlity
 * Delta t_warm + Delta t_recon <= Delta t_mem, with Eqs. warm-up_time, recon_time
 * and oom_time): would an eviction of evict_tokens started now (the same
 * chunks csr_evict_and_reconcile would drop) finish its rebuild and catch-up
 * before the page pool is exhausted, at append_tokens_per_s new tokens per
 * second?  With c the time of one query-key pair of the rebuild and
 * |T^E| = prefix + retained chunk tokens:
 *   Delta t_warm  = c * sum_{i = |X_pre|+1}^{|T^E|} i   (Eq. TTFT_derivation_2: the
 *                   retained chunks are prefilled over the prefix and themselves;
 *                   the prefix is not recomputed)
 *   Delta N       = append_tokens_per_s * Delta t_warm
 *   Delta t_recon = c * Delta N (2 |T^E| + Delta N + 1) / 2        (Eq. recon_time)
 *   Delta t_mem   = N_buffer / append_tokens_per_s                 (Eq. oom_time)
 * N_buffer is the largest number of tokens x such that the pages both
 * versions need for x more tokens fit in the pool's free pages once the
 * rebuilt version is reserved (while a reconciliation runs an appended chunk
 * takes pages in both), capped by max_seq_tokens.  The paper's two resources
 * give N_max - |T_t|; here one pool holds both versions.
 * c = pair_seconds when > 0; otherwise the value observed on this context's
 * last completed reconciliation (device time from the eviction to the end of
 * its last catch-up on the low-priority stream, the foreground running
 * alongside, divided by the query-key pairs it computed).  Host-only; nothing
 * changes.  CSR_EINVAL for evict_tokens < 1, append_tokens_per_s <= 0 or a
 * NULL out; CSR_ESTATE with a live suffix, while a reconciliation runs, with
 * no chunk to evict, or with pair_seconds <= 0 before any reconciliation has
 * completed.
 */
csr_status csr_check_viability(csr_ctx *ctx, int32_t evict_tokens, double append_tokens_per_s,
                               double pair_seconds, csr_viability *out);

/* Which version an inspection call reads. */
#define CSR_VERSION_ACTIVE 0
#define CSR_VERSION_PENDING 1

/*
 * Host view of a version's layout: its page table (logical page i holds
 * positions i*page_size .. i*page_size+page_size-1 in physical page
 * page_table[i]; the slot of position p is page_table[p/P]*P + p%P), its page
 * count and length.  page_table may be NULL to query the count; capacity is
 * its length in entries.  CSR_ESTATE for PENDING without a reconciliation.
 */
csr_status csr_get_layout(csr_ctx *ctx, int which, int32_t *page_table,
                          int32_t capacity, int32_t *n_pages, int64_t *length);

/* Ascending ids of the free physical pages (ids may be NULL to count). */
csr_status csr_get_free_pages(csr_ctx *ctx, int32_t *ids, int32_t capacity,
                              int32_t *count);

/*
 * Chunk ids and lengths of a version in order (X_chunks), and its prefix
 * length.  Arrays may be NULL to count.
 */
csr_status csr_get_chunks(csr_ctx *ctx, int which, int64_t *ids, int32_t *lens,
                          int32_t capacity, int32_t *count, int64_t *prefix_len);

/* Device pointer of a version's page table (int32, n_pages entries). */
csr_status csr_device_page_table(csr_ctx *ctx, int which, const int32_t **ptr);

/*
 * Gather the cached (rotated) keys and the values of positions pos0..pos0+n-1
 * of a version into k_out, v_out [n][num_kv_heads][head_dim] (device), on
 * stream.  For inspection and tests.
 */
csr_status csr_gather_kv(csr_ctx *ctx, int which, int64_t pos0, int32_t n,
                         void *k_out, void *v_out, csr_stream_t stream);

/*
 * Wait for all of the context's device work (device-wide synchronise), then
 * return and clear the device error word (CSR_DEVERR_* bits) in *flags.
 * Returns CSR_EDEVICE when a bit was set.
 */
csr_status csr_device_status(csr_ctx *ctx, uint32_t *flags);

/* Number of kernels the context has launched since creation. */
int64_t csr_kernel_launches(const csr_ctx *ctx);

/* One piece of a foreground launch's schedule (csr_foreground_schedule). */
typedef struct csr_piece {
  int32_t cta;    /* CTA that runs it */
  int32_t order;  /* its position in that CTA's sequence */
  int32_t unit;   /* pair * num_kv_heads + kv head; a pair is query tiles 2p, 2p+1 of
                     128 packed rows (tokens x group heads) */
  int32_t j0, j1; /* key tiles [j0, j1) of 128 keys */
  int32_t slot;   /* merges == 0: the partial slot the piece writes, or -1 when the piece
                     is the whole unit (written directly); merges > 0 and group == 1: the
                     first of the slots it merges; group > 1: the slot it writes */
  int32_t merges; /* > 0: the piece is in the last group of a cut unit (the pieces that end
                     last); the unit has this many partial slots */
  int32_t group;  /* size g of that group (0 for other pieces).  g == 1: the piece waits for
                     the partials of slots slot .. slot + merges - 1, combines them with
                     its own rows and writes the unit's output.  g > 1: every piece of the
                     unit writes a partial (the group's are the last g of the unit's
                     consecutive slots); member k merges rows [k*256/g, (k+1)*256/g) */
  int32_t member; /* k, the piece's index in its group */
} csr_piece;

/*
 * Inspection: the pieces a fused foreground call of n new tokens over L
 * cached tokens runs, for a configuration and a CTA count (0 = one per SM of
 * the current device; a plan-only configuration needs grid > 0).  Host-only.
 * pieces may be NULL to count; *n_slots receives the partial slots written
 * (0: no unit is cut).  CSR_EINVAL for a bad configuration or sizes, or a
 * block one fused launch cannot run; CSR_ENOMEM if capacity is too small.
 */
csr_status csr_foreground_schedule(const csr_config *cfg, int64_t L, int32_t n, int32_t grid,
                                   csr_piece *pieces, int32_t capacity, int32_t *count,
                                   int32_t *n_slots);

/* Kernel kinds of csr_timing. */
#define CSR_KERNEL_ROPE_APPEND 0
#define CSR_KERNEL_ATTENTION 1
#define CSR_KERNEL_MERGE 2
#define CSR_KERNEL_EVICT 3
#define CSR_KERNEL_KINDS 4

typedef struct csr_timing {
  double ms[CSR_KERNEL_KINDS];        /* summed device time per kernel kind */
  int64_t launches[CSR_KERNEL_KINDS]; /* timed launches per kernel kind */
} csr_timing;

/*
 * Per-kernel timing of the foreground path: while enabled, every kernel a
 * foreground call launches is bracketed by two CUDA events on the call's
 * stream.  csr_get_timing waits for those events, sums their elapsed times
 * per kernel kind into *out and forgets them.  Disabling drops pending events.
 */
csr_status csr_set_timing(csr_ctx *ctx, int enable);
csr_status csr_get_timing(csr_ctx *ctx, csr_timing *out);

/* Text of the last failure on this context (never NULL). */
const char *csr_last_error(const csr_ctx *ctx);

/*
 * Arguments of csr_attend_block_noalloc.  All pointers are device pointers
 * of the current device, owned by the caller; q, k, v, out 16-byte aligned.
 */
typedef struct csr_block_args {
  const void *q, *k, *v;      /* the n new tokens, before RoPE: [n][H][head_dim] bf16 */
  void *k_pool, *v_pool;      /* [pool_pages][num_kv_heads][page_size][head_dim] bf16 */
  const int32_t *page_table;  /* logical page -> physical page; must cover positions
                                 0 .. L+n-1 (the new tokens' slots included) */
  void *out;                  /* [n][num_q_heads][head_dim] bf16 */
  float *lse;                 /* [num_q_heads][n] or NULL */
  int64_t L;                  /* cached tokens before the block (positions of the block: L..L+n-1) */
  int32_t n;
  int32_t num_q_heads, num_kv_heads, head_dim, page_size, pool_pages;
  double rope_base;
  float softmax_scale;        /* 0 selects 1/sqrt(head_dim) */
} csr_block_args;

/*
 * The block path of csr_append_chunk / csr_attend_suffix (RoPE and append of
 * the new keys/values through the caller's page table, causal attention of
 * the new queries over positions 0..L+n-1, merge of split partials) for
 * callers that cannot allocate device memory: code that may not call
 * cudaMalloc at all, e.g. a real-time control loop that must not take the
 * allocator's locks or wait on it, or a process whose device memory belongs
 * to another allocator (a framework's caching allocator) so that it cannot
 * size and hand over the workspace csr_create needs.  The paper has no
 * counterpart: it is a property of this library, not of the method.
 *
 * Allocates nothing (no cudaMalloc, cudaFree or allocating library call).  Its
 * scratch is one static device array of 32.5 MiB that every GPU loading the
 * library holds until the process exits: 8 MiB of packed rotated queries
 * (so n * num_q_heads * head_dim * 2 bytes, rounded up to whole pairs of
 * 128-row tiles, must not exceed 8 MiB: n <= 512 for 64 query heads of 128
 * dims; larger n returns CSR_EINVAL), 24.5 MiB of split-KV partials (the key
 * range is split only as far as they fit) and the device error word.  Every
 * call looks the array's address up (cudaGetSymbolAddress); the first call in
 * a context of the device -- the runtime's primary context, and again after
 * cudaDeviceReset has replaced it -- also sets the kernels' shared-memory
 * limit (cudaFuncSetAttribute): make that call before any stream capture.
 * Every call shares the array and it keeps the last call's contents.  The
 * error word is cleared at the start of each call and not reported: a page
 * id out of range in page_table (which the workspace entry points report
 * through csr_device_status) goes unnoticed here, and the output rows that
 * needed that page are unspecified; check the table before the call.  Calls
 * that overlap on the same GPU (issued on different streams and not ordered)
 * race on the array: order them.  Each GPU has its own copy of the array.
 * Asynchronous on `stream`.
 * CSR_EINVAL for bad arguments or sizes beyond the limit, CSR_ECUDA if a CUDA
 * call fails.
 */
csr_status csr_attend_block_noalloc(const csr_block_args *args, csr_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* CSR_H_ */
