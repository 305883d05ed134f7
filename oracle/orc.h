/*
 * Reference (oracle) implementation of one Gated VLA-Cache step.
 *
 * TEST INFRASTRUCTURE ONLY.  This library is the slow, plain CPU statement
 * of what the method computes; only the tests, the package's smoke check
 * and the benchmark's CPU-baseline leg may load it.  It shares no code,
 * header or table with the CUDA library.
 *
 * What it follows:
 *   - Sec. III-A: image cut into (H/p)(W/p) patches, projected to token
 *     embeddings, concatenated with the language tokens.
 *   - Sec. III-B Stage 1: cosine similarity between corresponding patches
 *     of I_t and I_{t-1}; similarity above tau marks a patch static.
 *   - Sec. III-B Stage 2 (optional): static patches that drew the most
 *     text-to-vision attention are taken out of the reusable set.  The
 *     relevance of a patch is the softmax probability that the text queries
 *     put on its key, summed over text rows and heads, at one caller-chosen
 *     layer of the previous step; the top_k patches by relevance are
 *     removed.
 *   - Sec. III-B Stage 3: a per-layer proportion of the static patches is
 *     reused: a caller-given per-mille schedule, or (optional) one derived
 *     from each layer's normalized attention entropy measured in the
 *     previous step -- lower entropy, more reuse -- smoothed over depth.
 *     The paper names the idea but gives no formula: the mapping and the
 *     smoothing are this library's reading (parity unpinned).
 *   - Sec. IV-A Eq. (1): mean top-1/top-2 probability margin over the D
 *     action tokens, with the softmax over the action bins or (margin kind
 *     2) over the whole vocabulary.
 *   - Sec. VI: the alternative signals the paper evaluated, as outputs: the
 *     entropy of each action token's distribution and the action delta
 *     between consecutive steps.
 *   - Algorithm 1: gate on m_{t-1} < theta_m -> invalidate and run a full
 *     pass; otherwise reuse the cache and recompute only the rest; then
 *     decode the action tokens.
 *
 * Every dot product and reduction accumulates in fp64.  Stored values are
 * rounded at fixed points: the residual stream to fp32; GEMM inputs (norm
 * outputs, attention output, SwiGLU product), Q and the cached K/V to bf16
 * (bf16 workloads) or fp32 (fp32 workloads).
 */
#ifndef ORC_H
#define ORC_H
#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct orc_dims {
  int32_t n_layers, hidden, n_heads, head_dim, ffn, vocab, n_bins;
  int32_t img_h, img_w, patch, n_views;
  int32_t n_text;       /* prompt length including BOS */
  int32_t proprio_dim;  /* 0 = no proprio token */
  int32_t n_action;     /* action tokens (autoregressive) or block positions (parallel) */
  int32_t parallel;     /* 0 = autoregressive decode, 1 = parallel action block */
  int32_t bf16;         /* 1 = weights are bf16 bit patterns and storage rounds to bf16 */
  double rope_theta, rms_eps;
} orc_dims;

/* Host pointers.  Element type: uint16 bf16 bit patterns if dims.bf16, else float.
 * Matrices are row-major [out][in]; per-layer entries are arrays of n_layers pointers. */
typedef struct orc_weights {
  const void* tok_emb;     /* [vocab][hidden] */
  const void* patch_w;     /* [hidden][patch*patch*3], column (y*patch + x)*3 + c */
  const void* proprio_w;   /* [hidden][proprio_dim] or NULL */
  const void* action_emb;  /* [n_action][hidden] (parallel) or NULL */
  const void* const* attn_norm;
  const void* const* wq;
  const void* const* wk;
  const void* const* wv;
  const void* const* wo;
  const void* const* ffn_norm;
  const void* const* w_gate;
  const void* const* w_up;
  const void* const* w_down;
  const void* final_norm;
  const void* lm_head;     /* [vocab][hidden]; rows vocab-n_bins .. vocab-1 are read */
} orc_weights;

typedef struct orc_opts {
  int32_t margin_kind;          /* 0 = probability p1 - p2 over the bins (Eq. 1), 1 = logit gap
                                   l1 - l2, 2 = probability p1 - p2 over the whole vocabulary */
  int32_t reduction;            /* 0 = mean over the action tokens (Eq. 1), 1 = minimum */
  const int8_t* gate_override;  /* [B]: -1 gate, 0 force cached, 1 force full; NULL = gate */
  const int32_t* forced_ids;    /* [B][n_action] bins fed back in decode; NULL = argmax */
  int32_t s2_top_k;             /* Stage 2: patches removed per step; 0 = Stage 2 off */
  int32_t s2_layer;             /* Stage 2: the layer whose attention gives the relevance */
  const uint8_t* active;        /* [B]: 0 = this sequence sits the step out (its cache and state
                                   stay as they are, its outputs are zero); NULL = all step */
  int32_t s3_adaptive;          /* Stage 3 from attention entropy: 0 = the caller's schedule */
  int32_t s3_lo, s3_hi;         /* per-mille reuse of a layer of normalized entropy 1 / 0 */
  int32_t s3_weight;            /* per-mille weight of a layer's own target in the smoothing over depth */
  const uint16_t* s3_forced;    /* [B][n_layers]: lock-step replay, applied instead of the schedule this
                                   step derives (its own is still reported); NULL = none */
} orc_opts;

typedef struct orc_out {
  int32_t* action_ids;  /* [B][n_action] argmax bin (0 .. n_bins-1) */
  double* margins;      /* [B][n_action] p1 - p2 */
  double* logit_gap;    /* [B][n_action] l1 - l2 */
  double* logits;       /* [B][n_action][n_bins] or NULL */
  uint8_t* recomputed;  /* [B] 1 = the full branch ran */
  uint8_t* gate_auto;   /* [B] what the gate alone decided */
  double* step_margin;  /* [B] m_t (reduced per-token signal) */
  uint8_t* static_mask; /* [B][n_visual] or NULL */
  int32_t* idx;         /* [B][S] recompute order or NULL */
  int32_t* M;           /* [B][n_layers] rows recomputed per layer or NULL */
  double* relevance;    /* [B][n_visual] this step's Stage-2 relevance (0 when off) or NULL */
  uint8_t* relevant;    /* [B][n_visual] patches Stage 2 removed this step or NULL */
  double* entropy;      /* [B][n_action] entropy (nats) of the bin softmax or NULL */
  double* vocab_margin; /* [B][n_action] p1 - p2 of the softmax over the whole vocabulary or NULL */
  int32_t* action_delta; /* [B] sum over d of |a_t^d - a_{t-1}^d| in bins (0 without a previous step) or NULL */
  double* layer_entropy; /* [B][n_layers] normalized attention entropy of the text rows measured this
                            step (0 with Stage 3 adaptive off) or NULL */
  uint16_t* schedule;    /* [B][n_layers] the per-mille reuse schedule Stage 3 derived for this step
                            (the caller's when adaptive is off or nothing was measured) or NULL */
} orc_out;

typedef struct orc_ctx orc_ctx;
typedef struct orc_cache orc_cache;

enum { ORC_OK = 0, ORC_ERR_ARG = -1, ORC_ERR_OOM = -3 };

int orc_create(const orc_dims* d, const orc_weights* w, orc_ctx** out);
void orc_destroy(orc_ctx* c);
int orc_cache_new(const orc_ctx* c, int batch, orc_cache** out);
void orc_cache_free(orc_cache* k);
int orc_reset(orc_cache* k, int seq);  /* seq = -1: every sequence */
int orc_step(orc_ctx* c, orc_cache* k, const uint8_t* frames, const int32_t* prompt_ids,
             const float* proprio, uint32_t tau_num, uint32_t tau_den, double tau_margin,
             const uint16_t* reuse_permille, const orc_opts* opts, orc_out* out);
/* Copies one layer of sequence `seq`'s cache: kind 0 = K, 1 = V ([cache_len][hidden]),
 * 2 = H (layer inputs, [S][hidden]).  Values as stored (float). */
int orc_cache_read(const orc_cache* k, int seq, int kind, int layer, float* dst);
/* The reverse of orc_cache_read for K (kind 0) and V (kind 1): the values are
 * stored as given. */
int orc_cache_write(orc_cache* k, int seq, int kind, int layer, const float* src);
/* One decoder layer (the Llama-2 block of Sec. III-A as the prefix pass runs
 * it) for n rows of sequence `seq` at distinct positions pos[i] < the prefix
 * pass length: x [n][hidden] holds the rows' layer inputs and receives their
 * outputs; the rows' K/V are written into the cache at their positions before
 * any row attends; attention is causal by position over the cache. */
int orc_layer(orc_ctx* c, orc_cache* k, int seq, int layer, int n, const int32_t* pos, float* x);
int orc_cache_state(const orc_cache* k, int seq, double* m_prev, int* valid);

/* Pieces exposed for pin tests. */
void orc_patch_stats(const orc_dims* d, const uint8_t* frame, const uint8_t* prev, int v,
                     int64_t* dot, int64_t* na, int64_t* nb);
int orc_is_static(int64_t dot, int64_t na, int64_t nb, uint32_t num, uint32_t den);
int orc_more_similar(int64_t d_i, int64_t na_i, int64_t nb_i, int i,
                     int64_t d_j, int64_t na_j, int64_t nb_j, int j);
int orc_select(const orc_dims* d, const uint8_t* frame, const uint8_t* prev, int have_prev,
               uint32_t num, uint32_t den, const uint16_t* permille, int full,
               uint8_t* mask, int32_t* idx, int32_t* M);
/* orc_select with Stage 2: `relevance` ([n_visual], NULL = none) marks its
 * top_k patches relevant (written to `relevant` if not NULL); a relevant
 * patch is never reused. */
int orc_select2(const orc_dims* d, const uint8_t* frame, const uint8_t* prev, int have_prev,
                uint32_t num, uint32_t den, const uint16_t* permille, int full,
                const double* relevance, int top_k, uint8_t* mask, uint8_t* relevant,
                int32_t* idx, int32_t* M);
/* out[v] = 1 for the top_k entries of rel[0..n): v is in iff fewer than top_k
 * entries rank before it (higher value, or equal value and lower index). */
void orc_top_k(const double* rel, int n, int top_k, uint8_t* out);
void orc_margin(const double* logits, int n, int32_t* argmax, double* pmargin, double* lgap);
/* -sum_j p_j ln p_j of the softmax of logits[0..n), in nats. */
double orc_entropy(const double* logits, int n);
/* Entropy-adaptive Stage 3 (this library's reading): layer l's target
 * t_l = hi - (hi - lo) * ent[l] (per mille; ent in [0, 1]), smoothed over
 * depth r_0 = t_0, r_l = r_{l-1} + (weight / 1000) * (t_l - r_{l-1}), and
 * permille[l] = floor(r_l) clamped to [0, 1000]. */
void orc_entropy_schedule(const double* ent, int n_layers, int lo, int hi, int weight, uint16_t* permille);
double orc_round_bf16(double v);
void orc_rope_table(const orc_dims* d, int n_pos, float* cos_t, float* sin_t);

#ifdef __cplusplus
}
#endif
#endif
