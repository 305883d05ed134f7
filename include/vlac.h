/*
 * vlac — one Gated VLA-Cache step on a single GB300 (sm_103a).
 *
 * The step is Algorithm 1 of the paper: a logit-margin gate on the previous
 * step's Eq. (1) margin either invalidates the cache and runs the full
 * forward pass, or detects static patches (Sec. III-B, Stage 1), applies the
 * per-layer reuse proportion (Stage 3) and recomputes only the remaining
 * tokens; then the D action tokens are decoded and their margins reduced.
 *
 * Conventions for every call:
 *   - Return value: VLAC_OK (0) or a negative VLAC_ERR_* code.  No call
 *     aborts or exits the process.  vlac_strerror() names a code.
 *   - "device" pointers are CUDA device memory of the context's device;
 *     "host" pointers are ordinary host memory read during the call.
 *   - Work is enqueued asynchronously on `stream` (a cudaStream_t, NULL =
 *     the legacy default stream); outputs are valid once the stream has
 *     reached the end of the call's work.
 *   - Errors detected on the device (bad token ids, a bounded wait that gave
 *     up) are latched in a per-context error word; the next call on the
 *     context returns them, and vlac_sync_error() waits for the device and
 *     returns them.
 */
#ifndef VLAC_H
#define VLAC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define VLAC_OK 0
#define VLAC_ERR_INVALID_ARG (-1)  /* a pointer, size or value is out of its documented range */
#define VLAC_ERR_CUDA (-2)         /* a CUDA runtime call or kernel launch failed */
#define VLAC_ERR_OOM (-3)          /* device or host allocation failed */
#define VLAC_ERR_TIMEOUT (-4)      /* a bounded device-side wait gave up */
#define VLAC_ERR_DEVICE_CHECK (-5) /* a device-side bounds check rejected an input value */
#define VLAC_ERR_STATE (-6)        /* cache and context (or batch) do not match */
#define VLAC_ERR_UNSUPPORTED (-7)  /* valid dims this build does not implement */

#define VLAC_F32 0  /* fp32 weights and activations */
#define VLAC_BF16 1 /* bf16 weights and GEMM inputs, fp32 residual stream and accumulation */

#define VLAC_MARGIN_PROB 0  /* gate signal p1 - p2 of the softmax over the action bins (Eq. 1) */
#define VLAC_MARGIN_LOGIT 1 /* gate signal l1 - l2, the top-2 logit gap */
#define VLAC_MARGIN_VOCAB 2 /* gate signal p1 - p2 of the softmax over the whole vocabulary (Sec. IV-A);
                               reads every LM-head row per action token */
#define VLAC_REDUCE_DEFAULT (-1) /* mean for autoregressive decode (Eq. 1), min for a parallel block */
#define VLAC_REDUCE_MEAN 0
#define VLAC_REDUCE_MIN 1

/* Backbone and input geometry (Sec. III-A).  Token layout of a sequence:
 * position 0 = BOS (prompt id 0), 1..n_visual = patches (view-major, row-major),
 * then one proprio token if proprio_dim > 0, then prompt ids 1..n_text-1, then,
 * if parallel, n_action action positions computed in the same pass. */
typedef struct vlac_dims {
  int32_t n_layers, hidden, n_heads, head_dim, ffn, vocab, n_bins;
  int32_t img_h, img_w, patch, n_views;
  int32_t n_text;      /* prompt length including BOS (>= 2 when parallel == 0) */
  int32_t proprio_dim; /* 0 = no proprio token */
  int32_t n_action;    /* D action tokens (autoregressive) or block positions (parallel) */
  int32_t parallel;    /* 0 = autoregressive decode of D tokens, 1 = one parallel block */
  int32_t dtype;       /* VLAC_F32 or VLAC_BF16 */
  float rope_theta, rms_eps;
  int32_t max_batch;   /* largest batch a cache of this context may hold */
} vlac_dims;

/* Weights: device pointers of element type dims.dtype, row-major [out][in].
 * Per-layer members are HOST arrays of n_layers device pointers.  All are read
 * during vlac_create (copied / repacked), so the caller may free them after. */
typedef struct vlac_weights {
  const void* tok_emb;    /* [vocab][hidden] */
  const void* patch_w;    /* [hidden][patch*patch*3], column index (y*patch + x)*3 + c */
  const void* proprio_w;  /* [hidden][proprio_dim], or NULL when proprio_dim == 0 */
  const void* action_emb; /* [n_action][hidden] when parallel, else NULL */
  const void* const* attn_norm; /* [hidden] RMSNorm gains */
  const void* const* wq;        /* [hidden][hidden] */
  const void* const* wk;
  const void* const* wv;
  const void* const* wo;
  const void* const* ffn_norm;
  const void* const* w_gate;    /* [ffn][hidden] */
  const void* const* w_up;      /* [ffn][hidden] */
  const void* const* w_down;    /* [hidden][ffn] */
  const void* final_norm;       /* [hidden] */
  const void* lm_head;          /* [vocab][hidden]; rows vocab-n_bins .. vocab-1 give the action
                                   bins, the others only the whole-vocabulary margin */
} vlac_weights;

/* Stage-1 threshold as an exact fraction: a patch is static iff cos > num/den. */
typedef struct vlac_rational {
  uint32_t num, den; /* den > 0 */
} vlac_rational;

typedef struct vlac_step_opts {
  int32_t margin_kind;         /* VLAC_MARGIN_PROB (default), VLAC_MARGIN_LOGIT or VLAC_MARGIN_VOCAB */
  int32_t reduction;           /* VLAC_REDUCE_* */
  const int8_t* gate_override; /* device [B]: -1 gate decides, 0 force the cached branch,
                                  1 force the full branch; NULL = gate decides.  An empty
                                  cache always runs the full branch. */
  const int32_t* forced_ids;   /* device [B][n_action]: bins fed back during autoregressive
                                  decode instead of the argmax (lock-step replay); NULL = argmax */
  const uint8_t* active;       /* device [B]: 0 = the sequence sits this step out (a running batch
                                  that episodes join and leave): its prefix cache, gate state and
                                  previous frame stay as they are and its outputs are zero (the
                                  batch's decode rows still run, so its decode positions, which
                                  its next step rewrites before reading them, may change);
                                  NULL = all step */
  int32_t s2_top_k;            /* Stage 2 (Sec. III-B task-relevant filtering): the top_k visual
                                  patches by the previous step's relevance are never reused;
                                  0 = Stage 2 off (default) */
  int32_t s2_layer;            /* Stage 2: the layer (0 .. n_layers-1) whose attention gives the
                                  relevance: per visual patch, the softmax probability the text
                                  queries put on its key, summed over text rows and heads */
  const uint8_t* s2_forced;    /* device [B][Nv]: the Stage-2 removal set to apply instead of the
                                  library's own (lock-step replay; `relevant` still reports the
                                  library's own set); NULL = the library's own */
  int32_t s3_adaptive;         /* Stage 3 (Sec. III-B, entropy-adaptive layer-wise reuse): 0 = the
                                  caller's reuse_permille (default); 1 = per sequence, the schedule
                                  the previous step's layer entropies give (the caller's on a
                                  sequence's first step and after a reset).  The paper names the
                                  idea, not a formula; this library's reading: layer l's normalized
                                  attention entropy e_l (the mean over the text rows that see two or
                                  more keys, and the heads, of H / ln(keys)) sets the target
                                  t_l = s3_hi - (s3_hi - s3_lo) * e_l per mille, smoothed over depth
                                  (r_0 = t_0, r_l = r_{l-1} + s3_weight / 1000 * (t_l - r_{l-1}))
                                  and floored */
  int32_t s3_lo, s3_hi;        /* 0 <= s3_lo <= s3_hi <= 1000 */
  int32_t s3_weight;           /* 0 .. 1000 */
  const uint16_t* s3_forced;   /* device [B][L]: the schedule to apply instead of the derived one
                                  (lock-step replay; `schedule` still reports the derived one);
                                  NULL = the derived one */
} vlac_step_opts;

/* Device output buffers of one step (B = the cache's batch, D = n_action,
 * S = positions of the prefix pass, Nv = visual tokens, L = n_layers). */
typedef struct vlac_step_out {
  int32_t* action_ids;  /* [B][D] argmax bin, 0 .. n_bins-1 (token id vocab-n_bins+bin) */
  float* margins;       /* [B][D] p1 - p2 of each action token (Eq. 1 summand) */
  float* logit_gap;     /* [B][D] l1 - l2 */
  uint8_t* recomputed;  /* [B] 1 = the full branch ran this step */
  float* step_margin;   /* [B] m_t: the reduced signal that gates the next step */
  uint8_t* gate_auto;   /* optional [B]: what the gate alone decided */
  float* logits;        /* optional [B][D][n_bins] action-bin logits (fp32) */
  uint8_t* static_mask; /* optional [B][Nv] Stage-1 result (0 without a previous frame) */
  int32_t* idx;         /* optional [B][S] recompute order: rows of layer l are idx[0..M[l]) */
  int32_t* M;           /* optional [B][L] rows recomputed at each layer */
  float* relevance;     /* optional [B][Nv] this step's Stage-2 relevance (0 when Stage 2 is off) */
  uint8_t* relevant;    /* optional [B][Nv] patches Stage 2 kept out of the reusable set this step */
  float* entropy;       /* optional [B][D] entropy (nats) of each action token's bin softmax (Sec. VI) */
  float* vocab_margin;  /* optional [B][D] p1 - p2 of the softmax over the whole vocabulary; asking
                           for it (or for VLAC_MARGIN_VOCAB) reads every LM-head row per token */
  int32_t* action_delta; /* optional [B] sum over d of |a_t^d - a_{t-1}^d| in bins, 0 on a sequence's
                            first step and after a reset (Sec. VI) */
  float* layer_entropy;  /* optional [B][L] normalized attention entropy of each layer measured this
                            step (0 when Stage 3 adaptive is off) */
  uint16_t* schedule;    /* optional [B][L] the per-mille reuse schedule Stage 3 derived for this step */
} vlac_step_out;

typedef struct vlac_ctx vlac_ctx;
typedef struct vlac_cache vlac_cache;

/* Validates dims, copies and repacks the weights into device memory owned by
 * the context, builds RoPE tables and TMA descriptors, and allocates the
 * step workspace for dims.max_batch sequences.  *out is set on success. */
int vlac_create(const vlac_dims* dims, const vlac_weights* w, vlac_ctx** out);
int vlac_destroy(vlac_ctx* ctx);

/* Bytes of device memory a cache for `batch` (1 .. max_batch) sequences needs:
 * per sequence the K/V of every layer and position, the fp32 input of every
 * layer for the prefix positions (tokens that rejoin at a deeper layer start
 * from it), the previous frame, m_{t-1}, a valid flag and the last step's
 * Stage-2 relevance. */
int vlac_cache_bytes(const vlac_ctx* ctx, int batch, size_t* bytes);
/* Formats caller-owned device memory (>= vlac_cache_bytes, 256-byte aligned)
 * as an empty cache; the memory must outlive the cache handle.  Synchronous. */
int vlac_cache_init(vlac_ctx* ctx, void* dev_mem, size_t bytes, int batch, vlac_cache** out);
int vlac_cache_destroy(vlac_cache* cache);

/* One step of Algorithm 1 for every sequence of the cache.
 *   frames:          device [B][n_views][img_h][img_w][3] uint8 (HWC)
 *   prompt_ids:      device [B][n_text] int32 token ids (BOS first)
 *   proprio:         device [B][proprio_dim] fp32, NULL when proprio_dim == 0
 *   tau_sim:         Stage-1 threshold (static iff cos > num/den)
 *   tau_margin:      the gate fires iff m_{t-1} < tau_margin (strict)
 *   reuse_permille:  host [n_layers]: k_l = floor(permille[l] * |reusable| / 1000)
 *                    reusable patches (the most similar) are reused at layer l; each
 *                    <= 1000.  Reusable = static and, with Stage 2, not relevant.
 *   opts:            NULL = defaults; VLAC_ERR_INVALID_ARG if s2_top_k < 0, or if
 *                    s2_top_k > 0 and s2_layer is not a layer
 *   out:             device output buffers (required members non-NULL)
 * Returns VLAC_ERR_STATE if the cache belongs to another context. */
int vlac_step(vlac_ctx* ctx, vlac_cache* cache, const uint8_t* frames, const int32_t* prompt_ids,
              const float* proprio, vlac_rational tau_sim, float tau_margin,
              const uint16_t* reuse_permille, const vlac_step_opts* opts, const vlac_step_out* out,
              void* stream);

/* Invalidates sequence `seq` (-1 = all): its next step runs the full pass as if
 * no cache existed (Algorithm 1, cache invalidation), and Stage 2 and Stage 3
 * adaptive have no previous relevance or entropies to use. */
int vlac_reset(vlac_cache* cache, int seq, void* stream);

/* One decoder layer of the prefix pass on its own: Algorithm 1's partial
 * forward ("recompute the non-cached tokens against the reused cache", Sec.
 * III-B) for one layer, which is the one-layer workload: gather, q/k/v + RoPE
 * + K/V scatter, mixed-cache attention, o-projection, MLP, as vlac_step runs
 * them for each layer.
 *   seq, layer:  the cache sequence (< batch) and layer (< n_layers)
 *   pos:         device int32 [M], distinct positions of the rows, each below
 *                the prefix pass length S (n_text + visual + proprio, plus the
 *                parallel action block); an index outside [0, S) latches
 *                VLAC_ERR_DEVICE_CHECK in the context's error word and is
 *                replaced by 0, so that no access leaves the cache
 *   M:           1 .. S rows
 *   x:           device fp32 [M][hidden]: the rows' layer inputs on entry,
 *                their layer outputs on return
 * The rows' K/V are written into the cache at their positions before any row
 * attends; each row attends causally by position to that layer of the cache
 * (rows of a parallel action block see the whole block).  Asynchronous on
 * `stream`; the context's workspace is used, so calls on one context do not
 * overlap.  VLAC_ERR_INVALID_ARG for NULL pointers or out-of-range seq,
 * layer or M. */
int vlac_layer_bench(vlac_ctx* ctx, vlac_cache* cache, int seq, int layer, const int32_t* pos, int M, float* x,
                     void* stream);

/* K and V of one layer of sequence `seq` as device arrays [T][hidden] in the
 * model's element type (bf16 or fp32), row t the key (value) vector of
 * position t, heads side by side; T = the cache's positions: S + n_action - 1
 * for autoregressive decode, S for a parallel action block.
 * vlac_cache_load copies them into the cache, vlac_cache_store out of it.
 * Asynchronous on `stream`.  VLAC_ERR_INVALID_ARG for NULL or unaligned
 * (4-byte) pointers or out-of-range seq or layer. */
int vlac_cache_load(vlac_cache* cache, int seq, int layer, const void* K, const void* V, void* stream);
int vlac_cache_store(const vlac_cache* cache, int seq, int layer, void* K, void* V, void* stream);

/* Waits for the context's device work and returns (and clears) the latched
 * device error word. */
int vlac_sync_error(vlac_ctx* ctx);

/* Kernels this context has launched so far (every launch of the library's own kernels). */
uint64_t vlac_launch_count(const vlac_ctx* ctx);

/* Self-test of the bounded device wait: one kernel waits on an mbarrier that
 * nothing completes, for at most `spin_limit` polls, then records
 * VLAC_ERR_TIMEOUT in the error word and returns.  Synchronous; returns the
 * recorded status (VLAC_ERR_TIMEOUT when the wait gave up). */
int vlac_selftest_wait(vlac_ctx* ctx, uint32_t spin_limit);

/* Test hook: the number of polls after which the bounded waits of the step's
 * kernels give up (the prefix GEMM's pipeline waits, the decode GEMV's ring
 * waits, the prefix attention's tile waits); 0 makes every such wait give up
 * at once.  A block that gave up latches VLAC_ERR_TIMEOUT, stops, and still
 * lets the copies it issued land (those waits keep their own limit) before it
 * exits, so the context stays usable.  Takes effect for launches made after
 * the call: eager steps and step graphs captured later; a cache's existing
 * step graph keeps the limit it was captured with.  Default 2^24.
 * VLAC_ERR_INVALID_ARG for a NULL context. */
int vlac_set_wait_limit(vlac_ctx* ctx, uint32_t polls);

/* Per-launch timing, for roofline reports and time breakdowns.  While
 * enabled (steps then run without graph replay), each kernel launch of the
 * step is bracketed by CUDA events recorded on the launching stream and
 * filed under one of the kinds below.  vlac_prof_read waits for the events of
 * one kind, returns their summed device time, the number of launches and
 * their algorithmic bytes, and forgets them.  Bytes are counted for kind 0
 * (decode GEMV: weights + inputs + outputs) and kind 1 (prefix GEMM: weights
 * only, the row count being device-resident); other kinds report 0 bytes. */
#define VLAC_PROF_DECODE_GEMV 0
#define VLAC_PROF_PREFIX_GEMM 1
#define VLAC_PROF_PREFIX_ATTN 2 /* attention of the prefix pass */
#define VLAC_PROF_DECODE_ATTN 3 /* attention of the decode passes */
#define VLAC_PROF_ROWS 4        /* prefix row kernels: embedding, norms, epilogues */
#define VLAC_PROF_HEAD 5        /* action head: logits and margins */
#define VLAC_PROF_OTHER 6       /* selection, decode inputs, state update, staging */
#define VLAC_PROF_KINDS 7
int vlac_prof_enable(vlac_ctx* ctx, int on);
int vlac_prof_read(vlac_ctx* ctx, int kind, double* total_ms, uint64_t* launches, double* bytes);

/* Allocation-free selection step.  The paper has no counterpart of this call:
 * it exists for callers that cannot allocate device memory when they run it
 * -- real-time control loops whose memory is fixed up front, host frameworks
 * that own every device allocation and forbid a library its own.  It
 * runs the same kernels as vlac_step's selection (Stage-1 exact patch
 * similarity, the gate on m_prev < tau_margin or gate_override, the Stage-3
 * recompute order) without a context and without allocating: its scratch is
 * one fixed 256 KiB device array inside the library, which every call on a
 * device shares and which keeps the last call's contents.  Calls whose GPU
 * work overlaps (other streams, other host threads) therefore race; order
 * them on one stream.  The first call on each device looks up that array's
 * device address (make it before any stream capture).
 *   d:              host; geometry as for vlac_create (d->max_batch bounds batch)
 *   frames, prev_frames: device [batch][n_views][img_h][img_w][3] uint8
 *   valid:          device [batch] uint8, 0 = no previous frame (full branch)
 *   m_prev:         device [batch] fp32, the previous step's m_{t-1}
 *   reuse_permille: host [n_layers], each <= 1000
 *   gate_override:  device [batch] int8 (-1 gate, 0 cached, 1 full) or NULL
 *   outputs (device): static_mask [batch][Nv], idx [batch][S], M [batch][n_layers],
 *                     recomputed [batch]
 * Returns VLAC_ERR_INVALID_ARG for bad arguments and VLAC_ERR_UNSUPPORTED
 * when valid dims need more than the fixed scratch: batch x visual patches
 * must stay within 20,000.  VLAC_ERR_CUDA when a launch fails (only this
 * call's launches are checked). */
int vlac_select_noalloc(const vlac_dims* d, int batch, const uint8_t* frames, const uint8_t* prev_frames,
                        const uint8_t* valid, const float* m_prev, vlac_rational tau_sim, float tau_margin,
                        const uint16_t* reuse_permille, const int8_t* gate_override, uint8_t* static_mask,
                        int32_t* idx, int32_t* M, uint8_t* recomputed, void* stream);

const char* vlac_strerror(int code);

#ifdef __cplusplus
}
#endif
#endif /* VLAC_H */
