/*
 * mzc.h -- C ABI of libmzc: prefill over a partially evicted LLM memory state
 * on one GB300 (sm_103a).
 *
 * The paper (mzCache) splits LLM memory into per-layer weight units and
 * fixed-size KV chunks per layer (Sec. 4.2), evicts them under memory
 * pressure with a backward-out order (Sec. 4.4), and on the next request
 * restores them while prefill already runs on the resident units ("zero-wait",
 * Sec. 1 and Sec. 4.4, Fig. 8b).  Its interface is evict(size) and
 * restore_generate(input_tokens) (Sec. 5).  This library keeps that model
 * with the restore paths a GB300 has: a copy of swapped blocks from pinned
 * host memory to HBM on a side stream, and recompute of a dropped token tail
 * against the resident prefix (the paper's balance principle of Sec. 4.3
 * applied to these two paths).
 *
 * Conventions for every call:
 *   - Status codes only; nothing throws or aborts across the ABI.
 *     mzc_last_error() returns a text for the last failing call on a ctx.
 *   - The ctx owns every device buffer, the pinned swap store and its CUDA
 *     streams (unless the caller passes its own compute and copy streams in
 *     mzc_options).  Pointers passed in are borrowed for the call only
 *     (mzc_create copies the weights).  Host pointers are plain host memory
 *     unless a parameter says "device".
 *   - One ctx per host thread; calls on one ctx must not overlap.  Different
 *     ctxs share nothing.
 *   - Token ranges are in absolute positions of the context; KV blocks are
 *     block_tokens (16) consecutive positions of one layer.
 *   - KV storage: K/V values are rounded to the shape's kv_dtype (bf16 or
 *     fp16) and held in fp16 encoding in either case, so attention reads one
 *     format.  For a bf16 KV type the encoding is exact only inside fp16's
 *     range: zero and magnitudes in [2^-14, 65504].  A bf16 K/V value below
 *     2^-14 keeps only fp16-subnormal precision, and one of 65520 or more
 *     does not fit at all: the prefill then fails with MZC_ERR_OVERFLOW.
 *     The activations the projections read (RMSNorm outputs, or x * g where
 *     the norm is folded into the projections: see separate_norm; SwiGLU
 *     outputs) and the q/k/v projection outputs are fp16 too, with the same
 *     check.
 */
#ifndef MZC_H
#define MZC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  MZC_OK = 0,
  MZC_ERR_INVALID = 1, /* bad argument: null pointer, unsupported shape, illegal eviction shape */
  MZC_ERR_RANGE = 2,   /* layer / token / block index outside the context or a capacity */
  MZC_ERR_STATE = 3,   /* not legal in the current residency state (e.g. double evict) */
  MZC_ERR_OOM = 4,     /* KV pool, row capacity or pinned store exhausted */
  MZC_ERR_CUDA = 5,    /* a CUDA runtime call failed; the text names it */
  MZC_ERR_TIMEOUT = 6, /* a bounded device wait gave up (kernel status word) */
  MZC_ERR_DEVICE = 7,  /* a device-side bounds check failed (kernel status word) */
  MZC_ERR_OVERFLOW = 8 /* a device-side range check: an fp16 activation (RMSNorm output or
                          folded x * g, q/k/v projection, SwiGLU output) or fp16-encoded K/V value reached
                          65520 in magnitude and was stored as infinity (kernel status word);
                          the results of that call are not to be used */
} mzc_status;

enum { MZC_KV_BF16 = 0, MZC_KV_FP16 = 1 };
enum { MZC_CODEC_NONE = 0, MZC_CODEC_Q8 = 1 };
/* eviction modes: COPY = swap to pinned host (restored by copy); DROP =
 * discard (restored by recompute); AUTO = split by the ctx's policy. */
enum { MZC_COPY = 0, MZC_DROP = 1, MZC_AUTO = 2 };
enum { MZC_POLICY_COPY = 0, MZC_POLICY_RECOMPUTE = 1, MZC_POLICY_HYBRID = 2 };
/* residency of one (layer, logical block) */
enum { MZC_RESIDENT = 0, MZC_SWAPPED = 1, MZC_DROPPED = 2, MZC_INFLIGHT = 3, MZC_EMPTY = 4 };

/* Decoder shape (Llama-style: RMSNorm, rotary q/k with half-split pairs,
 * grouped-query attention, SwiGLU MLP, untied LM head, no biases). */
typedef struct {
  int32_t n_layers, d_model, n_q_heads, n_kv_heads, head_dim, ffn_dim, vocab;
  float rope_theta; /* rotary base; angle(pos, i) = pos * theta^(-2i/head_dim) */
  float rms_eps;
  int32_t kv_dtype;     /* MZC_KV_BF16 or MZC_KV_FP16 (storage type of K/V) */
  int32_t block_tokens; /* positions per KV block; must be 16 */
  int64_t max_ctx;      /* positions the context may hold */
} mzc_model_shape;

/* How a layer's attention waits for the KV blocks a restore copies back
 * (the zero-wait overlap, Sec. 4.4: prefill consumes each unit as soon as it
 * is restored):
 *   MZC_WAIT_LAYER_EVENT: on the copy stream's per-layer event, recorded after
 *     the last copy of that layer (norms, projections and rotary/KV writes of
 *     the layer run before the wait);
 *   MZC_WAIT_BLOCK_FLAG: per physical block.  The copy engine writes a block's
 *     residency flag right after the block's data, and the attention kernels
 *     wait (bounded) for the flag of each block they are about to read, so a
 *     layer's attention starts before its last copy lands and runs behind the
 *     copies.  Not with MZC_CODEC_Q8 (its decode kernels, not the copy
 *     engine, write the restored blocks). */
enum { MZC_WAIT_LAYER_EVENT = 0, MZC_WAIT_BLOCK_FLAG = 1 };

typedef struct {
  int64_t pool_blocks;      /* physical KV blocks; 0 = 2 * n_layers * ceil(max_ctx/16) */
  int64_t max_rows;         /* rows per prefill call (recompute + prompt); 0 = max_ctx */
  int64_t host_store_bytes; /* pinned swap store; 0 = the whole context's KV bytes */
  int32_t overlap;          /* 1 = zero-wait overlap of restore and prefill; 0 = restore
                               completes before prefill starts (ablation) */
  int32_t device;           /* CUDA device ordinal */
  int32_t swap_codec;       /* MZC_CODEC_NONE: COPY swaps blocks as stored; MZC_CODEC_Q8:
                               8-bit quantized (mzc_k_q8_encode; about 0.56 of the bytes),
                               decoded into the pool on restore */
  int32_t wait_mode;        /* MZC_WAIT_LAYER_EVENT (default) or MZC_WAIT_BLOCK_FLAG */
  int32_t debug_checks;     /* 1: before each prefill, check the block tables (every
                               resident or in-flight block maps to its own physical
                               block inside the pool); during it, synchronize after each
                               layer and read the device status word, so an error names
                               the layer where it appeared.  Slower; results unchanged */
  int32_t read_swapped;     /* 1: a prefill may read SWAPPED blocks in place from the pinned
                               store (mapped host memory) when no mzc_restore_async was
                               issued for them: the attention kernels fetch them over the
                               host link with plain loads, and they stay SWAPPED (the
                               paper's shared buffers, Sec. 4.2).  Not with MZC_CODEC_Q8.
                               A block the new rows write into (the context's partial
                               last block) must be resident: MZC_ERR_STATE otherwise */
  void *compute_stream;     /* cudaStream_t the prefill kernels run on, owned by the caller
                               (it must outlive the ctx); NULL = the ctx creates its own.
                               mzc_prefill synchronizes this stream before it returns */
  void *copy_stream;        /* cudaStream_t of the restore copies, owned by the caller;
                               NULL = own.  The same stream as compute_stream is accepted
                               and serializes restore and prefill (no overlap) */
  int32_t separate_norm;    /* 0 (default): for row sets of 5-256 rows, for one-row steps
                               and for the last layer's logits row, each RMSNorm after
                               the first is folded into the projections around it (the
                               residual-add GEMM or GEMV writes x * g and partial sums of
                               squares of x; the next projection scales its rows by
                               1 / RMS); 1: every RMSNorm runs as its own kernel, as for
                               other row sets (ablation).  Results agree within the
                               fp16 rounding of the projection inputs */
  int32_t fused_rope;       /* 1: for row sets of 5-256 rows the rotary embedding and
                               KV-block write run inside the QKV projection (its split-K
                               reduction rotates the fp32 sums and writes q and the K/V
                               blocks), except in a layer whose KV writes wait for a copy;
                               0 (default): as their own kernel after an fp16 QKV output,
                               which measured as fast or faster (the 3B 128-row prompt
                               step: 3.842-3.845 ms against 3.852-3.862 fused) */
} mzc_options;

/* Weights, host memory, bf16 bit patterns, row-major [out_features][in_features]
 * (the layout of torch.nn.Linear.weight).  Norm gains are fp32. */
typedef struct {
  const uint16_t *wq;     /* [n_q_heads*head_dim][d_model] */
  const uint16_t *wk;     /* [n_kv_heads*head_dim][d_model] */
  const uint16_t *wv;     /* [n_kv_heads*head_dim][d_model] */
  const uint16_t *wo;     /* [d_model][n_q_heads*head_dim] */
  const uint16_t *w_gate; /* [ffn_dim][d_model] */
  const uint16_t *w_up;   /* [ffn_dim][d_model] */
  const uint16_t *w_down; /* [d_model][ffn_dim] */
  const float *attn_norm; /* [d_model] */
  const float *ffn_norm;  /* [d_model] */
} mzc_layer_weights;

typedef struct {
  const uint16_t *embed;           /* [vocab][d_model] */
  const uint16_t *lm_head;         /* [vocab][d_model] */
  const float *final_norm;         /* [d_model] */
  const mzc_layer_weights *layers; /* [n_layers] */
} mzc_weights;

/* Per-unit costs of the two restore paths, measured on the device (the
 * paper's offline profiling, Sec. 4.3: each path's time per unit).  Copy:
 * bytes over the host link.  Recompute: the per-layer time of the fused
 * (recomputed + prompt) rows, from measured pieces that the split planner
 * interpolates. */
typedef struct {
  double h2d_gbs;            /* pinned host -> HBM copy rate, GB/s */
  double gemm_us_128;        /* one layer's four projections at 128 rows, us */
  double gemm_us_512;        /* ... at 512 rows, us */
  double gemm_us_2048;       /* ... at 2048 rows, us */
  double attn_tflops;        /* attention of recompute-like rows: marginal rate per key, TFLOP/s */
  double attn_row_ns;        /* ... plus a fixed cost per row and layer, ns */
  double attn_prompt_tflops; /* attention of prompt rows over the whole context, TFLOP/s */
  double row_ns;             /* per row and layer: norms and rotary/KV write, ns */
  double layer_us;           /* per layer fixed cost (launch gaps), us */
} mzc_profile;

typedef struct {
  int64_t context_tokens;   /* positions currently in the context */
  int64_t blocks_resident;  /* (layer, block) pairs by state */
  int64_t blocks_swapped;
  int64_t blocks_dropped;
  int64_t pool_free_blocks;
  int64_t bytes_h2d_last;   /* KV + weight bytes copied by the last restore */
  int64_t copies_last;      /* cudaMemcpyAsync calls of the last restore */
  int64_t rows_last;        /* rows (recompute + prompt) of the last prefill */
  int64_t recompute_rows_last;
  int32_t weights_evicted_layers;
  int32_t reserved;
} mzc_stats_t;

typedef struct mzc_ctx mzc_ctx;

/* Builds a ctx on options->device: uploads the weights (copied; the caller
 * keeps ownership of `weights`), allocates the KV block pool, the per-layer
 * block tables (logical block -> physical block, Sec. 4.2's chunk-pointer
 * array), the residency table and scratch.  The context starts empty.
 * options may be NULL (defaults).  On failure *out is NULL. */
mzc_status mzc_create(const mzc_model_shape *shape, const mzc_options *options,
                      const mzc_weights *weights, mzc_ctx **out);
/* Frees every device buffer, the pinned store and the ctx's own streams (the
 * memory the paper's OS would reclaim, Sec. 3.1). */
mzc_status mzc_destroy(mzc_ctx *ctx);

/* Prefill: appends tokens[0..n) at positions context_tokens.. and runs, in one
 * fused pass, those rows together with any pending recompute rows
 * (mzc_recompute_tail) through every layer.  Each layer's attention waits only
 * for that layer's restore copies (zero-wait, Sec. 4.4).  Writes the fp32
 * logits of the last new token to logits_out[vocab] (host), or nothing when
 * logits_out is NULL or n == 0.  Returns after the logits are on the host.
 * Row sets larger than options->max_rows run in causal chunks of max_rows
 * rows (a chunk goes through all layers before the next).
 * Errors: MZC_ERR_STATE if any block the rows attend to is SWAPPED without a
 * restore in flight (unless the ctx reads swapped blocks in place, option
 * read_swapped), or DROPPED without a pending recompute; MZC_ERR_OOM if
 * the pool is full; MZC_ERR_RANGE past max_ctx. */
mzc_status mzc_prefill(mzc_ctx *ctx, const int32_t *tokens, int64_t n, float *logits_out);

/* Evicts layers [layer_begin, layer_end) x positions [tok_begin, tok_end).
 * The token range is rounded outward to whole blocks (Sec. 6.2 evicts
 * slightly more than asked at chunk granularity).  MZC_COPY swaps the blocks
 * to the pinned store (D2H, packed per layer) and frees their physical
 * blocks; MZC_DROP frees them for later recompute and is legal only across
 * all layers, with the dropped positions forming one contiguous range (it may
 * also take SWAPPED blocks, whose host copies are then discarded);
 * MZC_AUTO splits [tok_begin, context_tokens) into a recomputed front and a
 * copied back by the ctx's policy (mzc_set_policy).  Every block in range
 * must be RESIDENT (for DROP: RESIDENT or SWAPPED; else MZC_ERR_STATE,
 * nothing changes).  With the
 * MZC_CODEC_Q8 option, copied blocks are quantized on the device before the
 * D2H copy, and restored blocks hold the decoded values (lossy; repeated
 * swaps give the same values again).  Synchronous. */
mzc_status mzc_evict(mzc_ctx *ctx, int32_t layer_begin, int32_t layer_end, int64_t tok_begin,
                     int64_t tok_end, int32_t mode);
/* Fine-grained COPY eviction of n scattered (layer[i], logical_block[i]). */
mzc_status mzc_evict_blocks(mzc_ctx *ctx, const int32_t *layer, const int64_t *logical_block,
                            int64_t n, int32_t mode);
/* Evicts the weights of layers [layer_begin, layer_end) (Sec. 4.2: one unit per
 * layer) to a pinned host copy; restored per layer by mzc_restore_async. */
mzc_status mzc_evict_weights(mzc_ctx *ctx, int32_t layer_begin, int32_t layer_end);

/* Enqueues the restore of every swapped unit on the copy stream, forward-in
 * (Sec. 4.4: earliest layer first): per layer, the weight unit, then one
 * host->device copy per packed run of KV blocks into contiguous free physical
 * blocks; then records that layer's event.  Returns without waiting. */
mzc_status mzc_restore_async(mzc_ctx *ctx);

/* Declares the recompute of dropped positions [p, p+n): they are re-prefilled
 * against the resident prefix in the next mzc_prefill (or mzc_sync), fused
 * with its prompt rows.  [p, p+n) must equal the dropped range (MZC_ERR_RANGE
 * otherwise).  (The paper names recomputing the KV cache as the alternative
 * to slow storage reads, Sec. 1; here it is the second restore path that
 * Sec. 4.3's balance weighs against the host-link copy, for a backward-out
 * tail, Sec. 4.4.) */
mzc_status mzc_recompute_tail(mzc_ctx *ctx, int64_t p, int64_t n);

/* Sets the policy MZC_AUTO evictions use and the per-unit profile that sizes
 * the hybrid split (profile may be NULL to keep the current one): Sec. 4.3's
 * offline profile and the choice between its restore paths. */
mzc_status mzc_set_policy(mzc_ctx *ctx, int32_t policy, const mzc_profile *profile);

/* Hybrid split (pure host arithmetic): for an evicted tail [p, n_ctx) and a
 * prompt of n_prompt tokens, the block-aligned s in [p, n_ctx] such that
 * recomputing [p, s) (fused with the prompt) while [s, n_ctx) is copied
 * minimises the predicted TTFT (Sec. 4.3: the two paths balanced by their
 * profiled per-unit times).  The prediction runs the paths layer by layer:
 * a layer's QKV projection, rotary/KV write and attention of recomputed rows
 * never wait; the rest of layer l starts once layer l's copy (copy time / L
 * each, in layer order) has landed.  Attention of recomputed rows runs at a
 * rate reached linearly from the prompt rate (128 rows) to the recompute rate
 * (2048 rows).  Only splits whose per-layer compute stays within 95% of the
 * per-layer copy are taken, and s = p (copy only) is returned unless the best
 * split is predicted to be at least 1% faster. */
mzc_status mzc_plan_split(const mzc_model_shape *shape, const mzc_profile *profile, int64_t p,
                          int64_t n_ctx, int64_t n_prompt, int64_t *s_out);
/* The same split for this ctx's context, with its profile (mzc_set_policy or
 * mzc_profile_measure) and its swap codec: a compressed store moves
 * mzc_q8_block_bytes per block over the link, and (its decode kernels share
 * the SMs with the recompute) splits only for a predicted gain of 5%, with no
 * per-layer compute bound. */
mzc_status mzc_plan_split_ctx(mzc_ctx *ctx, int64_t p, int64_t n_prompt, int64_t *s_out);

/* Measures the per-unit profile on this ctx's device (the paper's one-time
 * offline profiling, Sec. 4.3, which must leave the memory state as it was):
 *   - the host link: timed pinned host -> device copies into device memory
 *     that holds no live KV (the longest run of free pool blocks, poisoned
 *     again afterwards like every freed block, or the ctx's staging buffer);
 *   - the ctx's own GEMM, attention and RMSNorm kernels on its activation
 *     buffers (which hold nothing live between prefills); the attention reads
 *     the resident context's blocks and writes none.
 * Resident KV blocks, block tables and residency are unchanged.  Errors:
 * MZC_ERR_STATE while a restore is in flight or a recompute is pending. */
mzc_status mzc_profile_measure(mzc_ctx *ctx, mzc_profile *out);

/* Eviction policy: the paper's evict(size) (Sec. 5) driving its four-stage
 * placement (Algorithm 1, Sec. 4.3), on this library's two restore paths:
 * the host link (weights, and KV units evicted by COPY) and recompute (KV
 * units evicted by DROP).  Units: a weight layer; a KV unit = one 16-token
 * block of every layer (recompute regenerates all layers of a row at once).
 * With q = floor(t_copy_w / t_rec_kv) and T = w_total * q:
 *   MZC_STAGE_KV_ONLY   while more than T KV units remain: one unit at a
 *                       time, to recompute if that path's total time with it
 *                       stays strictly below the link's total time with it
 *                       (link time counts evicted weights too), else to the
 *                       link: the faster path takes more, in inverse
 *                       proportion to the per-unit times;
 *   MZC_STAGE_KV_AND_W  then, per step, one weight layer to the link and q KV
 *                       units to recompute, so KV and weights run out together;
 *   MZC_STAGE_W_ONLY    then the remaining weight layers;
 *   MZC_STAGE_COMP_KV   nothing left to free on the device (the paper's last
 *                       stage moves compressed KV to storage; no device memory
 *                       is involved): the call stops.
 * A step is never split, so slightly more than asked may be freed (as the
 * paper's chunk granularity does, Sec. 6.2).
 * Placement (backward-out, Sec. 4.4): recomputed units are the context's
 * last kv_rec blocks of every layer, copied units the kv_copy blocks before
 * them, evicted weights the last w_evicted layers.  As later calls add
 * recompute units, the recomputed range grows backward over copied blocks
 * (their host copies are discarded), so the placement stays balanced
 * wherever eviction stops. */
enum { MZC_STAGE_KV_ONLY = 1, MZC_STAGE_KV_AND_W = 2, MZC_STAGE_W_ONLY = 3, MZC_STAGE_COMP_KV = 4 };
typedef struct {
  double t_copy_w;   /* s: one layer's weights over the host link */
  double t_copy_kv;  /* s: one KV unit over the host link */
  double t_rec_kv;   /* s: one KV unit recomputed */
  int64_t kv_total;  /* N_KV^total: KV units of the context, ceil(context / 16) */
  int32_t w_total;   /* N_W^total: weight layers that may be evicted */
  int32_t w_evicted; /* in/out: weight layers on the link path */
  int64_t kv_copy;   /* in/out: KV units on the link path */
  int64_t kv_rec;    /* in/out: KV units on the recompute path */
  int64_t kv_bytes;  /* device bytes one KV unit frees */
  int64_t w_bytes;   /* device bytes one weight layer frees */
} mzc_evict_plan;

/* Pure host arithmetic: advances plan's counts by Algorithm 1 until at least
 * `bytes` are freed or nothing is left; *freed_out = bytes freed, *stage_out
 * = the last stage taken (0 if bytes <= 0).  MZC_ERR_INVALID for negative
 * times or counts, or counts beyond the totals. */
mzc_status mzc_plan_evict_size(mzc_evict_plan *plan, int64_t bytes, int64_t *freed_out,
                               int32_t *stage_out);
/* evict(size) on this ctx: reads the current counts from the residency
 * table (which must have the placement above: MZC_ERR_STATE otherwise, or
 * while a restore or recompute is pending), takes the per-unit times from
 * the ctx's profile (mzc_profile_measure or mzc_set_policy: t_copy_* = bytes
 * / h2d rate; t_rec_kv = 16 rows through every layer at the profile's
 * 2048-row projection rate and recompute attention rate over the whole
 * context), plans, and evicts: COPY of the new copied blocks, DROP of the new
 * recomputed range (over resident or swapped blocks), the new weight layers.
 * After it, mzc_restore_async and mzc_recompute_tail(p, n) over the dropped
 * range [p, context) restore everything.  Synchronous. */
mzc_status mzc_evict_size(mzc_ctx *ctx, int64_t bytes, int64_t *freed_out, int32_t *stage_out);
/* The plan mzc_evict_size starts from on this ctx: the current counts, the
 * totals, the per-unit times and bytes (for a caller that wants to see or
 * replay the policy's decision, e.g. with mzc_plan_evict_size).  Same errors. */
mzc_status mzc_evict_size_plan(mzc_ctx *ctx, mzc_evict_plan *out);

/* Shrinks the context to n_ctx positions (frees the blocks past it; the
 * context-aware request of Sec. 2.2 continues from there). */
mzc_status mzc_truncate(mzc_ctx *ctx, int64_t n_ctx);
/* Runs any pending recompute, waits for both streams, and surfaces device
 * status words (MZC_ERR_TIMEOUT / MZC_ERR_DEVICE): the point where the
 * paper's restore completes (Sec. 4.4, Fig. 8b: restore and prefill
 * overlapped, then joined). */
mzc_status mzc_sync(mzc_ctx *ctx);

/* Residency of (layer, logical_block) and its physical block (-1 if none):
 * the per-chunk state behind Sec. 4.2's chunk-pointer array. */
mzc_status mzc_query(mzc_ctx *ctx, int32_t layer, int64_t logical_block, int32_t *state,
                     int32_t *phys);
/* Reads one resident block's K and V ([n_kv_heads][16][head_dim], fp16 bits
 * of the stored values) into host buffers of block_bytes/2 each. */
mzc_status mzc_read_kv(mzc_ctx *ctx, int32_t layer, int64_t logical_block, void *k_host,
                       void *v_host);
/* Reads K and V of every position [0, n) of every layer, widened to fp32,
 * into host arrays [n_layers][n][n_kv_heads][head_dim].  Every block must be
 * RESIDENT. */
mzc_status mzc_read_kv_all(mzc_ctx *ctx, int64_t n, float *k_host, float *v_host);
/* Counts of the context's units by residency state and of the last restore
 * and prefill (rows, copied bytes): the memory state of Sec. 4.2's units. */
mzc_status mzc_stats(mzc_ctx *ctx, mzc_stats_t *out);
/* Device time in ms of the last mzc_prefill: [0] the call on the compute
 * stream, [1] restore copies on the copy stream, [2] LM head, [3] TTFT on the
 * device (the paper's metric, Sec. 6.2): from the start of the restore copies
 * (or of the prefill when nothing was restored) to the logits' arrival in
 * host memory.  ms must hold 4 floats; -1 marks a phase that did not run. */
mzc_status mzc_last_times(mzc_ctx *ctx, float *ms3);
const char *mzc_last_error(mzc_ctx *ctx);

/* Kernel classes of the prefill path, for launch counts and timing. */
enum {
  MZC_K_GEMM = 0,      /* projections (tcgen05) */
  MZC_K_ATTENTION = 1, /* block-table attention (+ split-KV combine) */
  MZC_K_ROPE_KV = 2,   /* rotary + KV-block write */
  MZC_K_RMSNORM = 3,
  MZC_K_LM_HEAD = 4,
  MZC_K_EMBED = 5,
  MZC_K_NCLASS = 6
};
typedef struct {
  int64_t launches; /* kernels launched (always counted) */
  double ms;        /* summed CUDA-event duration on the compute stream (timing on) */
  double flops;     /* algorithmic FLOPs of those launches */
  double bytes;     /* algorithmic HBM bytes of those launches */
} mzc_kernel_stat;
/* Bit c of class_mask (c = MZC_K_*): bracket every kernel of that class in
 * mzc_prefill with CUDA events on the compute stream (-1: every class; 0:
 * none).  Either way, resets the per-class counters. */
mzc_status mzc_set_kernel_timing(mzc_ctx *ctx, int32_t class_mask);
mzc_status mzc_kernel_stats(mzc_ctx *ctx, int32_t kernel_class, mzc_kernel_stat *out);

/* ---------------------------------------------------------------------------
 * Host bookkeeping without a device (no CUDA call is made): the residency
 * table, block tables, physical-block allocator and restore planner the ctx
 * uses, for planning and for tests.  Same rules and status codes as above.
 */
typedef struct mzc_state mzc_state;

/* One planned host->device copy: n_blocks blocks of `layer` from host store
 * offset host_off to physical blocks [phys_begin, phys_begin + n_blocks). */
typedef struct {
  int32_t layer;
  int32_t n_blocks;
  int64_t host_off;
  int64_t phys_begin;
} mzc_copy_run;

mzc_status mzc_state_create(const mzc_model_shape *shape, int64_t pool_blocks,
                            int64_t host_store_bytes, mzc_state **out);
mzc_status mzc_state_destroy(mzc_state *st);
/* Context grows by n positions (what mzc_prefill does to the state). */
mzc_status mzc_state_append(mzc_state *st, int64_t n);
mzc_status mzc_state_evict(mzc_state *st, int32_t layer_begin, int32_t layer_end,
                           int64_t tok_begin, int64_t tok_end, int32_t mode);
mzc_status mzc_state_evict_blocks(mzc_state *st, const int32_t *layer,
                                  const int64_t *logical_block, int64_t n, int32_t mode);
/* evict(size) on the bookkeeping alone (see mzc_evict_size), with the unit
 * times and byte sizes from *times (its counts are ignored; the state's own
 * are used). */
mzc_status mzc_state_evict_size(mzc_state *st, const mzc_evict_plan *times, int64_t bytes,
                                int64_t *freed_out, int32_t *stage_out);
mzc_status mzc_state_recompute_tail(mzc_state *st, int64_t p, int64_t n);
/* Plans the restore of every swapped block (forward-in); swapped blocks
 * become INFLIGHT.  Writes up to cap runs; *n_runs is the number planned
 * (MZC_ERR_OOM with nothing changed if cap is too small). */
mzc_status mzc_state_plan_restore(mzc_state *st, mzc_copy_run *runs, int64_t cap,
                                  int64_t *n_runs);
/* Completes the restore and any pending recompute: INFLIGHT and recomputed
 * blocks become RESIDENT. */
mzc_status mzc_state_complete(mzc_state *st);
mzc_status mzc_state_truncate(mzc_state *st, int64_t n_ctx);
mzc_status mzc_state_query(mzc_state *st, int32_t layer, int64_t logical_block, int32_t *state,
                           int32_t *phys);
mzc_status mzc_state_counts(mzc_state *st, mzc_stats_t *out);

/* ---------------------------------------------------------------------------
 * Single kernels of the prefill path, for parity tests and profiling.  All
 * pointers are DEVICE pointers; `stream` is a cudaStream_t (NULL = default
 * stream).  Launch errors return MZC_ERR_CUDA; the calls do not synchronize.
 */

/* y[n][d] (fp16) = x / sqrt(mean(x^2) + eps) * g, x fp32 [n][d] (RMSNorm). */
mzc_status mzc_k_rmsnorm(const float *x, const float *g, int64_t n, int32_t d, float eps,
                         uint16_t *y, void *stream);

/* C = A W^T with A fp16 [m][k] and W fp16 [n][k] (IEEE half bits, both
 * row-major, K-major), fp32 accumulation on tcgen05 tensor cores.  (The ctx
 * converts the bf16 model weights to fp16 at creation; fp16 activations keep
 * 3 more mantissa bits than bf16 at the same tensor-core rate.)  epilogue:
 *   0: out fp16 [m][n] = C
 *   1: out fp32 [m][n] += C                       (residual add)
 *   2: out fp16 [m][n/2] = silu(C_gate) * C_up     (SwiGLU; W's rows must be in
 *      the interleaved order mzc_k_swiglu_pack produces)
 * k must be a multiple of 8; n a multiple of 16 (epilogue 2: of 128).
 * Kernel by m: up to 4 rows a GEMV streaming W (K split over two warps for
 * rows of 6 KB and more); up to 256 rows, when n is a multiple of 128, the K
 * range split over a thread-block cluster with the partials summed in a
 * fixed order; above 512 rows the paired-SM kernel (two CTAs of a cluster
 * share 256 x 256 tiles through tcgen05 cta_group::2 MMAs) unless its tiles
 * need more waves than single-CTA ones; otherwise the persistent single-CTA
 * tcgen05 GEMM.  Each path gives the same bits on every run. */
mzc_status mzc_k_gemm(const uint16_t *a, const uint16_t *w, void *out, int64_t m, int64_t n,
                      int64_t k, int32_t epilogue, void *stream);

/* RMSNorm folded into the two projections around it, as mzc_prefill runs row
 * sets of 5-256 rows (the pre-norms of the decoder layer the paper prefills,
 * Sec. 2.1: RMSNorm(x) W^T = diag(1 / RMS(x)) ((x * g) W^T), so the norm needs
 * no launch of its own).
 * m: 5..256 rows (MZC_ERR_INVALID otherwise).  All pointers DEVICE.
 *   mzc_k_gemm_norm_out: the residual add x fp32 [m][n] += A W^T (epilogue 1
 *     of mzc_k_gemm, on the split-K kernel; A fp16 [m][k], W fp16 [n][k]),
 *     writing besides x  h fp16 [m][n] = x * g  (g fp32 [n]) and
 *     ss fp32 [m][n / 128], ss[r][t] = the sum of the new x[r][c]^2 over the
 *     columns c of tile t (128t .. 128t + 127).  n a multiple of 128, k of 8;
 *     MZC_ERR_INVALID when the split-K kernel does not take the shape.
 *   mzc_k_gemm_norm_in: epilogue 0 or 2 of mzc_k_gemm on diag(rstd) (h W^T),
 *     h fp16 [m][k] from mzc_k_gemm_norm_out (d = k), W fp16 [n][k],
 *     rstd_r = 1 / sqrt((ss[r][0] + ... + ss[r][k/128 - 1]) / k + eps), the
 *     tiles summed in order; k a multiple of 128.
 *   status  int32 or NULL: MZC_ERR_OVERFLOW when a value stored as fp16 (h,
 *     or the consumer's output) reaches the fp16 overflow threshold.
 * Each gives the same bits on every run. */
mzc_status mzc_k_gemm_norm_out(const uint16_t *a, const uint16_t *w, float *x, int64_t m, int64_t n,
                               int64_t k, const float *g, uint16_t *h, float *ss, int32_t *status,
                               void *stream);
mzc_status mzc_k_gemm_norm_in(const uint16_t *h, const uint16_t *w, void *out, int64_t m, int64_t n,
                              int64_t k, int32_t epilogue, const float *ss, float eps, int32_t *status,
                              void *stream);

/* The residual-add GEMM (epilogue 1 of mzc_k_gemm: out fp32 [m][n] += A W^T,
 * the O and down projections of every decoder layer) with the persistent
 * kernel's last, partial wave split over k (stream-K), as the prefill runs
 * it.  The last wave's R tiles are shared by up to 2R CTAs (all SMs at most,
 * at least 4 k-blocks of 64 each); each CTA's partial sum is reduce-added into
 * out in a fixed order per tile (highest k first), so the bits are the same
 * on every run, though they differ from mzc_k_gemm's single add per element.
 * The split is taken when the k-blocks it saves, (1 - R / SMs) x k / 64,
 * reach 24 (the ordered adds cost about that much): long-K projections such
 * as down.  Shapes and kernel choice as mzc_k_gemm; only the single-CTA
 * persistent kernel splits (m of 257-512 rows, or m > 4 when n is not a
 * multiple of 128, or above 512 rows when the paired kernel is not taken).
 *   flags   DEVICE, n_flags uint64 entries, caller-owned; any contents.  The
 *           kernel stores (epoch << 32 | k-block) values in the first R.
 *   n_flags at least the device's SM count (else MZC_ERR_INVALID).
 *   epoch   nonzero, and different from the epoch of every earlier launch
 *           that used the same flags (a stale value could then match and the
 *           order of the adds, though not their sum, would be lost).  Launches
 *           sharing flags must run in stream order.
 *   status  DEVICE int32 or NULL: MZC_ERR_TIMEOUT when a CTA waited longer
 *           than about two seconds for the segment above it.
 *   split_ctas  HOST int64 or NULL: the number of CTAs sharing the split
 *           tiles (0: this shape ran unsplit). */
mzc_status mzc_k_gemm_split(const uint16_t *a, const uint16_t *w, float *out, int64_t m,
                            int64_t n, int64_t k, uint64_t *flags, int64_t n_flags,
                            uint32_t epoch, int32_t *status, int64_t *split_ctas, void *stream);
/* Host helper: interleaves gate [f][d] and up [f][d] into the [2f][d] row
 * order epilogue 2 reads (per 64 output features: 64 gate rows then the
 * matching 64 up rows).  f must be a multiple of 64. */
mzc_status mzc_k_swiglu_pack(const uint16_t *gate, const uint16_t *up, int64_t f, int64_t d,
                             uint16_t *out_host);

/* Rotary embedding of q and k and the KV-block write.
 * qkv fp16 [n][(hq + 2*hkv)*hd] (q heads, then k heads, then v heads),
 * pos int32 [n], cos/sin fp32 [max_pos][hd/2] (angle pos*theta^(-2i/hd)),
 * block_table int32 [n_logical] -> physical block, pool: block b holds
 * K [hkv][16][hd] then V [hkv][16][hd], fp16-encoded.
 * Out: q_out [n][hq][hd] rotated, fp16; K/V rounded to kv_dtype precision and
 * stored fp16-encoded at pool[table[pos/16]]
 * slot pos%16.  cos_t/sin_t must cover positions < n_logical*16.  status
 * (device int32, may be NULL) gets MZC_ERR_DEVICE on a bad index or block. */
mzc_status mzc_k_rope_kv_write(const uint16_t *qkv, const int32_t *pos, int64_t n, int32_t hq,
                               int32_t hkv, int32_t hd, const float *cos_t, const float *sin_t,
                               const int32_t *block_table, int64_t n_logical, void *pool,
                               int64_t pool_blocks, int32_t kv_dtype, uint16_t *q_out,
                               int32_t *status, void *stream);

/* Causal grouped-query attention over a block-table KV cache (the paper's
 * attention over non-contiguous KV chunks with online softmax, Sec. 4.2).
 * q fp16 [n][hq][hd] at positions pos int32 [n] over an fp16-encoded pool
 * (kv_dtype is accepted for symmetry and ignored); row i attends to
 * every position <= pos[i] through block_table; out fp16 [n][hq][hd].
 * max_keys: an upper bound of pos[i] + 1 (sizes the split of long key
 * ranges).  scratch: device buffer of mzc_k_attention_scratch_bytes() bytes,
 * 16-byte aligned, for the split-KV partials, or NULL to run without
 * splitting (an unaligned or short buffer also runs without splitting).
 * The pool must be 16-byte aligned (MZC_ERR_INVALID otherwise).  Calls
 * with at most 4 query rows per KV head (n * hq/hkv <= 4: a decode token)
 * take a kernel bound by reading K/V once (bulk copies of each block's K
 * and V rows); larger calls take the tensor-core kernel. */
mzc_status mzc_k_attention(const uint16_t *q, const int32_t *pos, int64_t n, int32_t hq,
                           int32_t hkv, int32_t hd, const int32_t *block_table, int64_t n_logical,
                           const void *pool, int64_t pool_blocks, int32_t kv_dtype,
                           uint16_t *out, int64_t max_keys, void *scratch, int64_t scratch_bytes,
                           int32_t *status, void *stream);
int64_t mzc_k_attention_scratch_bytes(int64_t n, int32_t hq, int32_t hkv, int32_t hd,
                                      int64_t max_keys);
/* mzc_k_attention that first waits for residency flags (the per-block wait
 * of MZC_WAIT_BLOCK_FLAG; Sec. 4.4's zero-wait consumption of restored
 * units): block_flags is a device int32 array [pool_blocks], non-zero once a
 * block's data is in the pool; before fetching a block the kernels wait for
 * its flag, at most flag_wait_cycles SM clocks (0 = the library's default
 * limit of about 2 s).  A flag that stays zero makes the call record
 * MZC_ERR_TIMEOUT in *status and return with that block unread (the output
 * is then undefined); the CUDA context stays usable. */
mzc_status mzc_k_attention_wait(const uint16_t *q, const int32_t *pos, int64_t n, int32_t hq,
                                int32_t hkv, int32_t hd, const int32_t *block_table,
                                int64_t n_logical, const void *pool, int64_t pool_blocks,
                                int32_t kv_dtype, uint16_t *out, int64_t max_keys, void *scratch,
                                int64_t scratch_bytes, const int32_t *block_flags,
                                int64_t flag_wait_cycles, int32_t *status, void *stream);

/* The paper has no counterpart to this entry point: it is a convenience of
 * this library.  Same arguments and result as mzc_k_attention, but the
 * split-KV partials live in a fixed device array inside the library
 * (MZC_ATTENTION_NOALLOC_SCRATCH_BYTES = 8 MiB, held by every GPU that loads
 * the library until the process exits), so the call allocates nothing: no
 * cudaMalloc, no cudaFree, no allocating library routine.  It is for callers
 * that cannot allocate device memory when they call: a process whose device
 * memory is being reclaimed (the memory pressure this library restores
 * from) cannot count on an allocation succeeding at request time, a host
 * framework may own all device memory through its own allocator, and
 * cudaFree synchronizes the device.
 * The first call on a device looks up the array's device address (a CUDA
 * runtime query, no allocation); make that first call before any stream
 * capture.  All calls share the array: calls that overlap on the GPU (for
 * example on two streams) race on it.  Nothing in it has to start at zero.
 * Errors: MZC_ERR_RANGE, with nothing launched, when the call's partials
 * would exceed the array (mzc_k_attention_scratch_bytes() gives the need);
 * MZC_ERR_INVALID for bad arguments; MZC_ERR_CUDA if the address lookup or
 * the launch fails.  mzc_last_error(NULL) holds the text. */
#define MZC_ATTENTION_NOALLOC_SCRATCH_BYTES (8LL << 20)
mzc_status mzc_k_attention_noalloc(const uint16_t *q, const int32_t *pos, int64_t n, int32_t hq,
                                   int32_t hkv, int32_t hd, const int32_t *block_table,
                                   int64_t n_logical, const void *pool, int64_t pool_blocks,
                                   int32_t kv_dtype, uint16_t *out, int64_t max_keys,
                                   int32_t *status, void *stream);

/* 8-bit swap codec (the paper's default KV compression, Sec. 5; idempotent,
 * Sec. 6.5).  Per group of 64 consecutive values of a KV block (64 head_dim
 * entries of one K or V row): fp32 min and step = (max - min) / 255,
 * code = round-half-even((x - min) / step) clamped to [0, 255] (0 for a
 * constant group), decoded value = code * step + min (two fp32 roundings),
 * rounded to kv_dtype and stored fp16-encoded.  A compressed block is the
 * block_elems codes in the block's element order followed by block_elems/64
 * fp32 (min, step) pairs: mzc_q8_block_bytes(hkv, hd) bytes, where
 * block_elems = 2 * hkv * 16 * hd.
 * encode: pool (device, fp16-encoded blocks) blocks phys[i] (device int32
 * [n]) -> out (device) [n][mzc_q8_block_bytes].
 * decode: in (device) [n][...] -> pool blocks phys[i], or phys_begin + i when
 * phys is NULL. */
int64_t mzc_q8_block_bytes(int32_t hkv, int32_t hd);
mzc_status mzc_k_q8_encode(const void *pool, const int32_t *phys, int64_t n, int32_t hkv,
                           int32_t hd, void *out, void *stream);
mzc_status mzc_k_q8_decode(const void *in, int64_t n, int32_t hkv, int32_t hd,
                           const int32_t *phys, int64_t phys_begin, int32_t kv_dtype, void *pool,
                           void *stream);

/* The kernels' pipeline waits are bounded: a wait that runs out records
 * MZC_ERR_TIMEOUT in the kernel's status word and returns, and the CUDA
 * context stays usable.  This entry point runs that wait on an mbarrier
 * nothing arrives on (arrive == 0; or that it arrived on first, arrive != 0)
 * with a limit of limit_cycles SM clocks; *completed (device int32) is 1 if
 * the phase completed, 0 if the wait ran out; status (device int32) is set to
 * MZC_ERR_TIMEOUT when it ran out. */
mzc_status mzc_k_wait_probe(int32_t arrive, int64_t limit_cycles, int32_t *status,
                            int32_t *completed, void *stream);

/* logits fp32 [vocab] = RMSNorm(x_row) * g  W^T, x_row fp32 [d], W bf16 [vocab][d]. */
mzc_status mzc_k_lm_head(const float *x_row, const float *g, int32_t d, float eps,
                         const uint16_t *w, int64_t vocab, float *logits, void *stream);

/* x fp32 [n][d] = embed[tokens[i]] widened (bf16 -> fp32). */
mzc_status mzc_k_embed(const int32_t *tokens, int64_t n, const uint16_t *embed, int32_t d,
                       int64_t vocab, float *x, int32_t *status, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* MZC_H */
