/*
 * vp.h -- C ABI of libvp, a GB300 (sm_103a) implementation of one decode step
 * of VisionPulse step-wise visual-pruned attention (arxiv 2605.31457).
 *
 * One call of vp_decode_step() runs, for every sequence of a batch and one
 * attention layer acting as the anchor layer l_a (Sec. 4.2):
 *   1. logits of the current query against every cached key      (Eq. 6's Z)
 *   2. the temperature-scaled visual attention mass per head and
 *      its head-max                                               (Eq. 5, Eq. 6, Sec. 4.3)
 *   3. the step's retention budget K_t = M_vis,max * N_v, clamped  (Eq. 7, Sec. 5.2)
 *   4. the top-K_t visual tokens by the head-averaged score S_i    (Eq. 2, Eq. 3)
 *   5. attention over the kept visual tokens plus every text token (Sec. 4.2, Sec. 5.7)
 *
 * Conventions shared by every entry point:
 *   - Tensors are caller-owned DEVICE memory unless stated otherwise; the
 *     library never frees or retains them beyond the call.  The context owns
 *     only its own workspace, allocated once in vp_init().
 *   - vp_decode_step() allocates nothing, never synchronises the host and only
 *     enqueues work on the caller's stream; its results are visible to later
 *     work on that stream.
 *   - Errors are returned as vp_status; nothing crosses the ABI as an
 *     exception.  Invalid host-visible arguments are rejected before any work
 *     is enqueued.  Per-sequence values that live on the device (spans, text
 *     lengths, page ids) are checked by the kernels: an out-of-range value is
 *     clamped or skipped, never dereferenced, and recorded in a device error
 *     word that vp_check_errors() reports.
 *   - A context serves one stream at a time; it is not thread-safe.
 */
#ifndef VP_H_
#define VP_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  VP_OK = 0,
  VP_ERR_INVALID_ARG = 1,     /* a host-visible argument is malformed          */
  VP_ERR_UNSUPPORTED = 2,     /* valid, but a shape or mode this build lacks   */
  VP_ERR_CAPACITY = 3,        /* batch or kept_cap exceeds what was configured */
  VP_ERR_NOT_INITIALIZED = 4, /* NULL context                                  */
  VP_ERR_CUDA = 5,            /* a CUDA runtime call failed (text in last_error)*/
  VP_ERR_DEVICE_PRECOND = 6   /* vp_check_errors: a device-side check fired    */
} vp_status;

typedef enum { VP_BF16 = 0, VP_FP32 = 1 } vp_dtype;

/* Budget modes (vp_budget.mode). */
typedef enum {
  VP_ADAPTIVE = 0,    /* K_t = ceil(M_vis,max(tau) * N_v) clamped to [K_lo, K_hi] (Eq. 7, Sec. 5.2) */
  VP_FIXED_RATIO = 1, /* K_t = max(1, ceil(ratio * N_v))   (FastV-VP "Fix Ratio", Table 2)        */
  VP_FIXED_K = 2,     /* K_t = min(fixed_k, N_v)           (Top-k budgeting, App. A.2)             */
  VP_DENSE = 3,       /* K_t = N_v: keep every visual token (full budget)                          */
  VP_TOP_P = 4        /* K_t = the fewest top-ranked tokens whose S_i sum to >= ratio * sum of all
                         visual S_i (Top-p budgeting, App. A.2); granularity 0 only; may keep up
                         to N_v tokens, so kept_cap must be >= max_visual                         */
} vp_budget_mode;

/* Static shapes, fixed for the life of a context (vp_init). */
typedef struct {
  int32_t max_batch;    /* largest batch a call may pass                          */
  int32_t num_q_heads;  /* H, query heads of the layer                            */
  int32_t num_kv_heads; /* Hkv, key/value heads; H % Hkv == 0, G = H / Hkv <= 16  */
  int32_t head_dim;     /* D: 64 or 128                                           */
  int32_t max_visual;   /* largest visual span N_v of any sequence (<= 32768)     */
  int32_t max_seq;      /* largest live cache length N_v + text_len               */
  vp_dtype dtype;       /* q, caches and out share this dtype                     */
  int32_t paged;        /* 0: contiguous caches, 1: paged caches                  */
  int32_t page_size;    /* tokens per page when paged (power of two, <= 256)      */
} vp_config;

/*
 * One key or value cache.  Element (b, kv-head g, token t, dim d) lives at
 *   contiguous: data + b*stride_b + g*stride_h + t*stride_t + d
 *   paged:      data + page*stride_b + g*stride_h + (t % page_size)*stride_t + d,
 *               page = block_table[b*max_pages + t / page_size]
 * (strides in elements; the d axis is contiguous).  Every row (D elements)
 * must start on a 16-byte boundary: data 16-byte aligned and every stride a
 * multiple of 16 bytes.  A page id outside [0, num_pages) is skipped and
 * flagged.  The kernels read whole 32-token tiles: in a contiguous cache,
 * rows t < max_seq of every (sequence, kv-head) must be readable memory, and
 * in a paged cache every row of a mapped page; rows past the live length are
 * read but never used.
 */
typedef struct {
  const void* data;
  int64_t stride_b;            /* contiguous: sequence stride; paged: page stride  */
  int64_t stride_h;            /* kv-head stride                                   */
  int64_t stride_t;            /* token stride                                     */
  const int32_t* block_table;  /* paged only: device [batch][max_pages]; else NULL */
  int32_t max_pages;           /* paged only: row length of block_table            */
  int32_t num_pages;           /* paged only: pages in the pool (bounds check)     */
} vp_kv;

/* Visual span of each sequence: tokens [vis_start[b], vis_start[b] + vis_len[b])
 * of the live cache are visual (X_v of Sec. 4.2); all other live tokens are
 * text (prompt, generated reasoning and the current token).  Device int32 [batch]. */
typedef struct {
  const int32_t* vis_start;
  const int32_t* vis_len;
} vp_span;

typedef struct {
  int32_t mode;        /* vp_budget_mode                                                 */
  float tau;           /* Eq. 6 temperature for the mass, (0, 1]; 0.1 (5%) or 0.4 (10%)  */
  float scale;         /* logit scale; 0 means 1/sqrt(D)                                 */
  int32_t r_lo_ppm;    /* ADAPTIVE clamp, parts per million: K_lo = ceil(r_lo*N_v)       */
  int32_t r_hi_ppm;    /*   K_hi = max(K_lo, floor(r_hi*N_v)); e.g. 10000 / 50000 (Sec. 5.2) */
  int32_t ratio_ppm;   /* FIXED_RATIO ratio, or TOP_P share p, parts per million         */
  int32_t fixed_k;     /* FIXED_K budget                                                 */
  int32_t granularity; /* 0: one kept set per sequence, S averaged over all H heads (Eq. 2);
                          1: one kept set per kv-head, S averaged over its G query heads  */
} vp_budget;

typedef struct vp_ctx vp_ctx;

/* Creates a context for the given static shapes on the current CUDA device and
 * allocates its workspace (logit scratch, split partials, counters) once.
 * Returns VP_ERR_INVALID_ARG / VP_ERR_UNSUPPORTED for bad shapes, VP_ERR_CUDA
 * when allocation fails.  *out_ctx is NULL on failure. */
vp_status vp_init(const vp_config* cfg, vp_ctx** out_ctx);

/*
 * One VisionPulse decode step (Sec. 4.2-4.3) for `batch` sequences.
 *   q            [batch][H][D] cfg.dtype, query of the current token (post-RoPE).
 *   k_cache,
 *   v_cache      caches holding N_v + text_len[b] live tokens of sequence b,
 *                the current token already appended (it counts in text_len).
 *   visual_span  device spans; 0 <= vis_start <= text_len, vis_len <= max_visual.
 *   text_len     device int32 [batch], >= 1; N_v + text_len <= max_seq.
 *   budget       host struct, see vp_budget.
 *   out          [batch][H][D] cfg.dtype: softmax attention of q over the kept
 *                visual tokens plus all text tokens (dropped tokens are
 *                excluded from the normaliser).
 *   kept_idx     int32 [batch][kept_cap] (granularity 1: [batch][Hkv][kept_cap]):
 *                kept visual indices, relative to vis_start, ascending; the
 *                K_t largest S_i, ties to the lower index; unused slots = -1.
 *   kept_cap     must be >= the largest K_t the budget can produce for
 *                max_visual tokens, else VP_ERR_CAPACITY (nothing enqueued).
 *   kept_count   int32 [batch] (granularity 1: [batch][Hkv]): K_t.
 *   mass         float [batch][H]: m_{t,h} of Eq. 5 under the Eq. 6 temperature.
 *   mass_stats   float [batch][4] or NULL: { M_vis(tau), M_vis,max(tau),
 *                M_vis(tau = 1), (float)K_t }.
 *   cuda_stream  cudaStream_t to enqueue on (NULL = legacy default stream).
 * Calls on one stream overlap: a call's kernels start while those of the
 * previous call of this library on the same stream finish (programmatic
 * dependent launch), and vp_decode_step reads q, the caches, spans, lengths
 * and page table before it waits for that call (it waits before its first
 * workspace write).  So no input of vp_decode_step may be written by the
 * immediately preceding call of this library on the stream; any other kernel
 * or copy in between removes the overlap.  vp_compact_kv's output caches are
 * exempt (its kernel completes before the next call starts), and
 * vp_decode_gather waits for the previous call before reading its kept set.
 */
vp_status vp_decode_step(vp_ctx* ctx, int32_t batch, const void* q,
                         const vp_kv* k_cache, const vp_kv* v_cache,
                         const vp_span* visual_span, const int32_t* text_len,
                         const vp_budget* budget, void* out,
                         int32_t* kept_idx, int32_t kept_cap, int32_t* kept_count,
                         float* mass, float* mass_stats, void* cuda_stream);

/*
 * Decode attention of a layer after the anchor layer (Sec. 4.2: importance is
 * computed at the anchor layer l_a and pruning starts from l_a; Sec. 5.1
 * prunes at l_a = 17).  The query attends to every text token of the cache
 * and to the visual tokens of a kept set produced by vp_decode_step at the
 * anchor layer of the same decode step; no budget or selection is computed,
 * and the visual K and V rows outside the kept set are never read.
 *   q, k_cache, v_cache, visual_span, text_len   as for vp_decode_step (this
 *                layer's query and caches; the same spans and lengths).
 *   kept_idx     int32 [batch][kept_cap], or [batch][Hkv][kept_cap] when
 *                granularity = 1: the anchor's kept visual indices (relative
 *                to vis_start, ascending as vp_decode_step writes them).
 *   kept_count   int32 [batch] (granularity 1: [batch][Hkv]): how many of the
 *                slots are used; 0 <= kept_count <= min(kept_cap, vis_len).
 *   granularity  0: one kept set per sequence; 1: one per kv-head.
 *   scale        logit scale; 0 means 1/sqrt(D).
 *   out          [batch][H][D] cfg.dtype.
 * Requires bf16 caches whose layout a tensor map describes (any order of the
 * sequence, kv-head and token axes; pages of at least 8 tokens), else
 * VP_ERR_UNSUPPORTED.  Kept indices outside [0, vis_len) are skipped and
 * flagged (vp_check_errors).  Uses the context's workspace: calls on one
 * context must not overlap with each other or with vp_decode_step.
 */
vp_status vp_decode_gather(vp_ctx* ctx, int32_t batch, const void* q,
                           const vp_kv* k_cache, const vp_kv* v_cache,
                           const vp_span* visual_span, const int32_t* text_len,
                           const int32_t* kept_idx, int32_t kept_cap, const int32_t* kept_count,
                           int32_t granularity, float scale, void* out, void* cuda_stream);

/*
 * Diagnostics of the step-wise analysis (Sec. 4.3, App. B); off by default.
 * Once set on a context, every later vp_decode_step on it also
 *   - writes n_act (int32 [batch]; granularity 1: [batch][Hkv]) = N_act(delta),
 *     the number of visual tokens whose head-averaged attention probability
 *     (the S_i of Eq. 2, compared in float32) exceeds delta;
 *   - sets, in active_bits (uint32 [batch][words]; granularity 1:
 *     [batch][Hkv][words]; words = (max_visual + 31) / 32), bit i % 32 of
 *     word i / 32 for every visual token i with S_i > delta.  Bits are only
 *     ever set: zero the array when a sequence starts; a token whose bit is
 *     still 0 when its decode ends was never active (persistently inactive,
 *     App. B).
 * Either pointer may be NULL; both NULL turns the diagnostics off.  delta
 * must be finite and > 0 (else VP_ERR_INVALID_ARG).  The arrays are
 * caller-owned device memory, 4-byte aligned, valid while set; the setting is
 * read when a call is enqueued (a captured graph keeps the pointers it saw).
 */
vp_status vp_set_diagnostics(vp_ctx* ctx, float delta, int32_t* n_act, uint32_t* active_bits);

/*
 * Prefill-stage compaction for FastV + VisionPulse (the paper's appendix
 * "Complementarity with Prefill Pruning": FastV prunes the visual tokens at
 * the prefill stage with compression ratio 0.5, then VisionPulse prunes step
 * by step over the remaining ones).  FastV ranks the visual tokens by the
 * head-averaged attention of the last prompt token at the pruning layer
 * (Sec. 5.1, l_a = 17) -- Eq. 2 with that token as the query -- so the
 * selection is a vp_decode_step call with VP_FIXED_RATIO (ratio_ppm =
 * 500000) and granularity 0 on that token; this call then writes, for one
 * layer, a cache holding only the surviving visual tokens:
 *   dst row t  =  src row t                      for t <  vis_start
 *              =  src row vis_start + kept[t - vis_start]
 *                                                 for vis_start <= t < vis_start + K
 *              =  src row t - K + vis_len        for t >= vis_start + K, t < K + text_len
 * with K = kept_count[b].  The compacted sequence has visual span
 * (vis_start, K) -- kept_count itself can serve as the new vis_len array --
 * and the same text_len.
 *   src          a cache as for vp_decode_step (contiguous or paged, cfg.dtype).
 *   dst          contiguous cache of cfg.dtype, caller-owned, rows for at
 *                least max(K + text_len) tokens per (sequence, kv-head);
 *                must not overlap src.
 *   kept_idx     int32 [batch][kept_cap]: surviving visual indices (relative to
 *                vis_start), ascending as vp_decode_step writes them.
 *   kept_count   int32 [batch]; 0 <= kept_count <= min(kept_cap, vis_len).
 * Asynchronous on cuda_stream; uses no workspace.  Out-of-range kept indices
 * and unmapped pages are skipped (the row is zeroed) and flagged in the
 * device error word (vp_check_errors).  Host-visible argument errors return
 * VP_ERR_INVALID_ARG before anything is enqueued.
 */
vp_status vp_compact_kv(vp_ctx* ctx, int32_t batch, const vp_kv* src, const vp_kv* dst,
                        const vp_span* visual_span, const int32_t* text_len,
                        const int32_t* kept_idx, int32_t kept_cap, const int32_t* kept_count,
                        void* cuda_stream);

/* Score kernel of later vp_decode_step calls on this context (an
 * implementation choice with no counterpart in the paper; results agree
 * within the documented tolerances either way):
 *   VP_SCORE_AUTO (default)  the library chooses per call;
 *   VP_SCORE_MMA             the mma.sync kernels (32-row tiles);
 *   VP_SCORE_TC              the tcgen05 kernel (128-row tiles, TMEM
 *                            accumulators): bf16, head_dim 128, G <= 16,
 *                            pages of at least 8 tokens, a cache layout a
 *                            tensor descriptor can describe -- a call it
 *                            cannot serve returns VP_ERR_UNSUPPORTED.
 * Returns VP_ERR_INVALID_ARG for another value. */
typedef enum { VP_SCORE_AUTO = 0, VP_SCORE_MMA = 1, VP_SCORE_TC = 2 } vp_score_path;
vp_status vp_set_score_path(vp_ctx* ctx, int32_t path);

/* Launch record of the last successful vp_decode_step or vp_decode_gather
 * call on this context, for profiling (an implementation detail with no
 * counterpart in the paper): *score_path = VP_SCORE_TC when the tcgen05 score
 * kernel ran, else VP_SCORE_MMA (the mma.sync, fallback or fp32 kernels);
 * *kernels = the number of kernels the call enqueued.  Both are 0 before the
 * first call.  Either pointer may be NULL.  Host only, no CUDA call. */
vp_status vp_last_launch(const vp_ctx* ctx, int32_t* score_path, int32_t* kernels);

/* Largest K_t the budget can produce for n_visual tokens (the kept_cap a
 * caller must provide); -1 for an invalid budget.  Host only, no CUDA. */
int32_t vp_max_kept(const vp_budget* budget, int32_t n_visual);

/* Text of the last error on this context ("" if none).  Valid until the next
 * call on the context.  Accepts NULL: then returns the text of the last
 * failure in this thread of a call that takes no context (vp_init or
 * vp_decode_step_noalloc), "" if that call succeeded. */
const char* vp_last_error(const vp_ctx* ctx);

/* Synchronises `cuda_stream`, then reads and clears the device error word.
 * Returns VP_OK, VP_ERR_DEVICE_PRECOND (with the failed checks in
 * vp_last_error) or VP_ERR_CUDA. */
vp_status vp_check_errors(vp_ctx* ctx, void* cuda_stream);

/* Stage timing, for profiling.  vp_timing_enable(ctx, slots) creates
 * 4 * slots CUDA events owned by the context; from then on the n-th call of
 * vp_decode_step on the context records, on its own stream, the events of
 * slot n % slots: before the score kernel and after the score, select and
 * gather kernels.  Inside stream capture the records become event nodes of
 * the graph and fire at every replay.  slots = 0 disables timing and releases
 * the events.  Returns VP_ERR_INVALID_ARG for slots < 0, VP_ERR_CUDA when
 * event creation fails. */
vp_status vp_timing_enable(vp_ctx* ctx, int32_t slots);

/* Synchronises the device, then writes for slot s < *n_slots the device time
 * in milliseconds of stage k (0 score, 1 select, 2 gather) to ms[3 * s + k];
 * *n_slots = min(max_slots, slots, calls recorded so far).  A slot whose
 * events have not fired yet reads as a negative value. */
vp_status vp_timing_read(vp_ctx* ctx, float* ms, int32_t max_slots, int32_t* n_slots);

/* Bytes of the fixed device scratch behind vp_decode_step_noalloc. */
#define VP_NOALLOC_SCRATCH_BYTES (16u << 20)

/* The decode step without a context and without allocating anything.  The
 * paper has no counterpart: this entry point exists for callers that cannot
 * allocate device memory on their inference path -- a plugin or custom-op
 * host whose framework owns all device memory through its own pool, or a
 * latency-critical loop that must not pay for an allocation.  Arguments mean
 * what they mean for vp_decode_step, with the static shapes passed as `cfg`.
 * The intermediate scratch lives in one fixed VP_NOALLOC_SCRATCH_BYTES device
 * array that every GPU loading the library holds until the process exits:
 *   - a (cfg, batch) whose scratch would not fit returns VP_ERR_CAPACITY and
 *     enqueues nothing; malformed arguments return VP_ERR_INVALID_ARG;
 *   - the first call on each device resolves the array's device address and
 *     must therefore come before any stream capture on that device;
 *   - every call shares the array (its counters are cleared at the start of
 *     each call on `cuda_stream`), so calls whose work overlaps on the GPU --
 *     on different streams, or from several threads -- race and corrupt each
 *     other's results; serialise them;
 *   - device-side range checks still clamp bad spans and skip bad page ids,
 *     but their flags are not reported (there is no context to read them);
 *   - on failure the reason (for VP_ERR_CAPACITY, the scratch bytes the call
 *     would need) is readable through vp_last_error(NULL) in the calling
 *     thread.
 * No cudaMalloc, cudaFree or other allocating call is made. */
vp_status vp_decode_step_noalloc(const vp_config* cfg, int32_t batch, const void* q,
                                 const vp_kv* k_cache, const vp_kv* v_cache,
                                 const vp_span* visual_span, const int32_t* text_len,
                                 const vp_budget* budget, void* out,
                                 int32_t* kept_idx, int32_t kept_cap, int32_t* kept_count,
                                 float* mass, float* mass_stats, void* cuda_stream);

/* Releases the workspace and the context; NULL is a no-op.  Waits for the
 * device to finish work that may still use the workspace. */
void vp_free(vp_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* VP_H_ */
