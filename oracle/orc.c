/*
 * Reference (oracle) implementation of one Gated VLA-Cache step.
 * TEST INFRASTRUCTURE ONLY: see orc.h for what may use it and which parts of
 * the paper each function follows.  Plain loops, fp64 accumulation, OpenMP
 * only to spread independent output elements over host cores (results do
 * not depend on the thread count: every output element is computed by one
 * thread in a fixed order).
 */
#include "orc.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

struct orc_ctx {
  orc_dims d;
  orc_weights w;
  const void** layer_ptrs; /* owned copies of the per-layer pointer arrays */
  int P;                   /* prefix length: BOS + visual + proprio + rest of text */
  int S;                   /* positions computed by the prefix pass */
  int T;                   /* cache positions per sequence */
  int Nv;                  /* visual tokens */
  float* cos_t;            /* [T][head_dim/2] */
  float* sin_t;
};

struct orc_cache {
  const orc_ctx* c;
  int B;
  float* K;      /* [B][L][T][hidden] */
  float* V;      /* [B][L][T][hidden] */
  float* H;      /* [B][L][S][hidden]: input of layer l of each prefix position */
  uint8_t* prev; /* [B][frame bytes] */
  double* m_prev;
  uint8_t* valid;
  double* rel;        /* [B][Nv]: Stage-2 relevance from the previous step */
  uint8_t* rel_valid; /* [B]: rel holds the previous step's relevance */
  int32_t* prev_ids;  /* [B][n_action]: the previous step's action bins */
  uint8_t* ids_valid; /* [B]: prev_ids holds them */
  double* ent;        /* [B][L]: per-layer normalized attention entropy from the previous step */
  uint8_t* ent_valid; /* [B]: ent holds it */
};

/* ------------------------------------------------------------------------ */
/* Scalars                                                                  */
/* ------------------------------------------------------------------------ */

/* bf16 round-to-nearest-even of a double, straight from fp64 (8 significant bits). */
double orc_round_bf16(double v) {
  if (!isfinite(v) || v == 0.0) return v;
  int e;
  double f = frexp(v, &e); /* v = f * 2^e, 0.5 <= |f| < 1 */
  double r;
  if (e - 8 < -133) {
    r = ldexp(nearbyint(ldexp(v, 133)), -133); /* bf16 subnormal spacing 2^-133 */
  } else {
    r = ldexp(nearbyint(ldexp(f, 8)), e - 8);
  }
  if (fabs(r) > 3.3895313892515355e38) r = v > 0 ? INFINITY : -INFINITY;
  return r;
}

static double wget(const orc_ctx* c, const void* p, size_t i) {
  if (c->d.bf16) {
    uint32_t bits = (uint32_t)((const uint16_t*)p)[i] << 16;
    float f;
    memcpy(&f, &bits, 4);
    return (double)f;
  }
  return (double)((const float*)p)[i];
}

/* Storage rounding of activations that feed a GEMM, of Q and of cached K/V. */
static double store_act(const orc_ctx* c, double v) {
  return c->d.bf16 ? orc_round_bf16(v) : (double)(float)v;
}

/* fp64 dot product.  Fixed order: lane j (0..7) sums the products of
 * elements j, j+8, j+16, ... in increasing order; lanes are then combined
 * pairwise ((0+1)+(2+3))+((4+5)+(6+7)). */
static double dot(const double* a, const double* b, int n) {
  double s[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  int k = 0;
  for (; k + 8 <= n; k += 8)
    for (int j = 0; j < 8; ++j) s[j] += a[k + j] * b[k + j];
  for (; k < n; ++k) s[k & 7] += a[k] * b[k];
  return ((s[0] + s[1]) + (s[2] + s[3])) + ((s[4] + s[5]) + (s[6] + s[7]));
}

/* y[i][o] = sum_k x[i][k] * W[o][k] for i < n rows (a linear layer, fp64). */
static void linear(const orc_ctx* c, const void* W, int n_out, int n_in, int n,
                   const double* x, double* y) {
#pragma omp parallel
  {
    double* wrow = (double*)malloc(sizeof(double) * (size_t)n_in);
#pragma omp for schedule(static)
    for (int o = 0; o < n_out; ++o) {
      for (int k = 0; k < n_in; ++k) wrow[k] = wget(c, W, (size_t)o * n_in + k);
      for (int i = 0; i < n; ++i) y[(size_t)i * n_out + o] = dot(x + (size_t)i * n_in, wrow, n_in);
    }
    free(wrow);
  }
}

/* RMSNorm of one fp32 row: x / sqrt(mean(x^2) + eps) * g, rounded for storage. */
static void rmsnorm_row(const orc_ctx* c, const float* x, const void* g, double* out) {
  const int n = c->d.hidden;
  double ss = 0.0;
  for (int k = 0; k < n; ++k) ss += (double)x[k] * (double)x[k];
  double r = 1.0 / sqrt(ss / n + c->d.rms_eps);
  for (int k = 0; k < n; ++k) out[k] = store_act(c, ((double)x[k] * r) * wget(c, g, k));
}

/* ------------------------------------------------------------------------ */
/* RoPE (rotate-half convention): pair (i, i + head_dim/2) of each head is    */
/* rotated by pos * theta^(-2i/head_dim); angles in fp64, table in fp32.     */
/* ------------------------------------------------------------------------ */

void orc_rope_table(const orc_dims* d, int n_pos, float* cos_t, float* sin_t) {
  const int half = d->head_dim / 2;
  for (int p = 0; p < n_pos; ++p)
    for (int i = 0; i < half; ++i) {
      double inv = pow(d->rope_theta, -2.0 * i / d->head_dim);
      double a = (double)p * inv;
      cos_t[(size_t)p * half + i] = (float)cos(a);
      sin_t[(size_t)p * half + i] = (float)sin(a);
    }
}

static void rope_head(const orc_ctx* c, double* v, int pos) {
  const int half = c->d.head_dim / 2;
  for (int i = 0; i < half; ++i) {
    double cs = c->cos_t[(size_t)pos * half + i], sn = c->sin_t[(size_t)pos * half + i];
    double a = v[i], b = v[i + half];
    v[i] = a * cs - b * sn;
    v[i + half] = b * cs + a * sn;
  }
}

/* ------------------------------------------------------------------------ */
/* Stage 1: patch cosine similarity between I_t and I_{t-1} (Sec. III-B).    */
/* The patch vector is the raw uint8 RGB values, flattened (y, x, c).        */
/* ------------------------------------------------------------------------ */

static const uint8_t* patch_px(const orc_dims* d, const uint8_t* frame, int v, int e) {
  const int p = d->patch, gw = d->img_w / p, gh = d->img_h / p;
  const int view = v / (gw * gh), r = v % (gw * gh);
  const int py = r / gw, px = r % gw;
  const int ry = e / (3 * p), rx = (e / 3) % p, ch = e % 3;
  const size_t off = (((size_t)view * d->img_h + (size_t)(py * p + ry)) * d->img_w + (size_t)(px * p + rx)) * 3 + ch;
  return frame + off;
}

void orc_patch_stats(const orc_dims* d, const uint8_t* frame, const uint8_t* prev, int v,
                     int64_t* dotp, int64_t* na, int64_t* nb) {
  const int n = d->patch * d->patch * 3;
  int64_t s = 0, a2 = 0, b2 = 0;
  for (int e = 0; e < n; ++e) {
    int64_t a = *patch_px(d, frame, v, e), b = *patch_px(d, prev, v, e);
    s += a * b;
    a2 += a * a;
    b2 += b * b;
  }
  *dotp = s;
  *na = a2;
  *nb = b2;
}

/* cos > num/den, decided exactly.  Both patches all-zero: cos = 1.  Exactly
 * one all-zero: cos = 0.  Otherwise cos = d / sqrt(na*nb) with d >= 0, and
 * cos > num/den  <=>  d > 0  and  d^2 * den^2 > num^2 * na * nb. */
int orc_is_static(int64_t d, int64_t na, int64_t nb, uint32_t num, uint32_t den) {
  typedef unsigned __int128 u128;
  if (den == 0) return 0;
  if (na == 0 && nb == 0) return num < den;
  if (na == 0 || nb == 0) return 0;
  if (d <= 0) return 0;
  u128 lhs = (u128)((uint64_t)d * (uint64_t)d) * ((uint64_t)den * (uint64_t)den);
  u128 rhs = (u128)((uint64_t)num * (uint64_t)num) * ((uint64_t)na * (uint64_t)nb);
  return lhs > rhs;
}

/* cos^2 as a fraction (num2, den2) with den2 > 0. */
static void cos2(int64_t d, int64_t na, int64_t nb, uint64_t* n2, uint64_t* d2) {
  if (na == 0 && nb == 0) { *n2 = 1; *d2 = 1; return; }
  if (na == 0 || nb == 0) { *n2 = 0; *d2 = 1; return; }
  *n2 = (uint64_t)d * (uint64_t)d;
  *d2 = (uint64_t)na * (uint64_t)nb;
}

/* Reuse order: the more similar patch first (higher cosine), ties to the
 * lower patch index.  Cosines of the patches compared here are >= 0, so
 * comparing cos^2 decides. */
int orc_more_similar(int64_t d_i, int64_t na_i, int64_t nb_i, int i,
                     int64_t d_j, int64_t na_j, int64_t nb_j, int j) {
  typedef unsigned __int128 u128;
  uint64_t ni, di, nj, dj;
  cos2(d_i, na_i, nb_i, &ni, &di);
  cos2(d_j, na_j, nb_j, &nj, &dj);
  u128 l = (u128)ni * dj, r = (u128)nj * di;
  if (l != r) return l > r;
  return i < j;
}

static int pos_is_visual(const orc_ctx* c, int pos) { return pos >= 1 && pos <= c->Nv; }
/* Prompt tokens: BOS at 0 and the text after the visual (and proprio) tokens. */
static int pos_is_text(const orc_ctx* c, int pos) {
  return pos == 0 || (pos > c->Nv + (c->d.proprio_dim > 0 ? 1 : 0) && pos < c->P);
}

/* Stage 2's removal set: the top_k entries of rel, ranked by value (higher
 * first), equal values by index (lower first). */
/* Stage 3 from the layers' normalized attention entropy (a reading: the paper
 * names the idea, not the formula).  Low entropy, more reuse: the target of
 * layer l is hi - (hi - lo) * ent[l] per mille; the targets are smoothed over
 * depth, each layer moving `weight` per mille of the way from the previous
 * layer's value to its own target; the result is floored and clamped. */
void orc_entropy_schedule(const double* ent, int n_layers, int lo, int hi, int weight, uint16_t* permille) {
  double r = 0.0;
  for (int l = 0; l < n_layers; ++l) {
    const double t = (double)hi - (double)(hi - lo) * ent[l];
    r = l == 0 ? t : r + ((double)weight / 1000.0) * (t - r);
    double f = floor(r);
    if (f < 0.0) f = 0.0;
    if (f > 1000.0) f = 1000.0;
    permille[l] = (uint16_t)f;
  }
}

void orc_top_k(const double* rel, int n, int top_k, uint8_t* out) {
  for (int v = 0; v < n; ++v) {
    int before = 0;
    for (int u = 0; u < n; ++u)
      if (rel[u] > rel[v] || (rel[u] == rel[v] && u < v)) ++before;
    out[v] = (uint8_t)(before < top_k);
  }
}

/* Stages 1-3 applied: the recompute order idx[0..S) and per-layer row counts
 * M[l] such that the rows recomputed at layer l are idx[0 .. M[l]).
 *   reusable = static patches (Stage 1) that Stage 2 did not mark relevant.
 *   idx = [every position that is not a reusable patch, ascending]
 *         ++ [reusable patches, least similar first].
 *   k_l = floor(permille[l] * |reusable| / 1000) reusable patches (the most
 *   similar) are reused at layer l, so M[l] = S - k_l.
 * The full branch recomputes everything: idx = 0 .. S-1 and M[l] = S.
 * Returns |reusable|. */
int orc_select2(const orc_dims* d, const uint8_t* frame, const uint8_t* prev, int have_prev,
                uint32_t num, uint32_t den, const uint16_t* permille, int full,
                const double* relevance, int top_k, uint8_t* mask, uint8_t* relevant,
                int32_t* idx, int32_t* M) {
  const int Nv = d->n_views * (d->img_h / d->patch) * (d->img_w / d->patch);
  const int P = d->n_text + Nv + (d->proprio_dim > 0 ? 1 : 0);
  const int S = P + (d->parallel ? d->n_action : 0);
  const int L = d->n_layers;
  for (int l = 0; l < L; ++l)
    if (permille[l] > 1000) return ORC_ERR_ARG;
  if (top_k < 0) return ORC_ERR_ARG;
  int64_t* st = (int64_t*)malloc(sizeof(int64_t) * 3 * (size_t)(Nv > 0 ? Nv : 1));
  int* stat = (int*)malloc(sizeof(int) * (size_t)(Nv > 0 ? Nv : 1));
  uint8_t* rel = (uint8_t*)calloc((size_t)(Nv > 0 ? Nv : 1), 1);
  if (relevance && top_k > 0) orc_top_k(relevance, Nv, top_k, rel);
  int nS = 0;
  for (int v = 0; v < Nv; ++v) {
    int s = 0;
    if (have_prev) {
      orc_patch_stats(d, frame, prev, v, &st[3 * v], &st[3 * v + 1], &st[3 * v + 2]);
      s = orc_is_static(st[3 * v], st[3 * v + 1], st[3 * v + 2], num, den);
    }
    if (mask) mask[v] = (uint8_t)s;
    if (relevant) relevant[v] = rel[v];
    if (s && !rel[v]) stat[nS++] = v;
  }
  if (full) {
    for (int i = 0; i < S; ++i) idx[i] = i;
    for (int l = 0; l < L; ++l) M[l] = S;
  } else {
    /* insertion sort of the reusable patches into reuse order */
    for (int a = 1; a < nS; ++a) {
      int key = stat[a], b = a - 1;
      while (b >= 0 && orc_more_similar(st[3 * key], st[3 * key + 1], st[3 * key + 2], key,
                                        st[3 * stat[b]], st[3 * stat[b] + 1], st[3 * stat[b] + 2], stat[b])) {
        stat[b + 1] = stat[b];
        --b;
      }
      stat[b + 1] = key;
    }
    int n = 0;
    for (int pos = 0; pos < S; ++pos) {
      int reusable = 0;
      if (pos >= 1 && pos <= Nv) {
        for (int q = 0; q < nS; ++q)
          if (stat[q] == pos - 1) { reusable = 1; break; }
      }
      if (!reusable) idx[n++] = pos;
    }
    for (int q = nS - 1; q >= 0; --q) idx[n++] = 1 + stat[q];
    for (int l = 0; l < L; ++l) M[l] = S - (int)(((int64_t)permille[l] * nS) / 1000);
  }
  free(st);
  free(stat);
  free(rel);
  return nS;
}

int orc_select(const orc_dims* d, const uint8_t* frame, const uint8_t* prev, int have_prev,
               uint32_t num, uint32_t den, const uint16_t* permille, int full,
               uint8_t* mask, int32_t* idx, int32_t* M) {
  return orc_select2(d, frame, prev, have_prev, num, den, permille, full, NULL, 0, mask, NULL, idx, M);
}

/* ------------------------------------------------------------------------ */
/* Eq. (1) ingredients: top-1 / top-2 of the softmax over the action bins.   */
/* ------------------------------------------------------------------------ */

void orc_margin(const double* lg, int n, int32_t* argmax, double* pmargin, double* lgap) {
  int b1 = 0;
  for (int j = 1; j < n; ++j)
    if (lg[j] > lg[b1]) b1 = j; /* ties keep the lowest bin */
  double l1 = lg[b1], l2 = -INFINITY;
  for (int j = 0; j < n; ++j)
    if (j != b1 && lg[j] > l2) l2 = lg[j];
  double z = 0.0;
  for (int j = 0; j < n; ++j) z += exp(lg[j] - l1);
  *argmax = b1;
  if (n < 2) { *pmargin = 1.0; *lgap = INFINITY; return; }
  /* p1 - p2 with p_j = exp(l_j - l1) / z */
  *pmargin = -expm1(l2 - l1) / z;
  *lgap = l1 - l2;
}

/* Entropy of the softmax p_j = exp(l_j - l1) / z:  -sum p_j ln p_j
 * = ln z - sum p_j (l_j - l1). */
double orc_entropy(const double* lg, int n) {
  double l1 = lg[0];
  for (int j = 1; j < n; ++j)
    if (lg[j] > l1) l1 = lg[j];
  double z = 0.0, s = 0.0;
  for (int j = 0; j < n; ++j) {
    const double e = exp(lg[j] - l1);
    z += e;
    s += e * (lg[j] - l1);
  }
  return log(z) - s / z;
}

/* ------------------------------------------------------------------------ */
/* Context and cache                                                        */
/* ------------------------------------------------------------------------ */

int orc_create(const orc_dims* d, const orc_weights* w, orc_ctx** out) {
  if (!d || !w || !out) return ORC_ERR_ARG;
  if (d->n_layers < 1 || d->hidden < 1 || d->n_heads < 1 || d->head_dim < 2 || (d->head_dim & 1) ||
      d->head_dim > 512 || d->n_heads * d->head_dim != d->hidden || d->ffn < 1 || d->n_bins < 2 || d->vocab < d->n_bins ||
      d->patch < 1 || d->img_h % d->patch || d->img_w % d->patch || d->n_views < 1 || d->n_text < 1 ||
      d->n_action < 1 || d->proprio_dim < 0)
    return ORC_ERR_ARG;
  orc_ctx* c = (orc_ctx*)calloc(1, sizeof(orc_ctx));
  if (!c) return ORC_ERR_OOM;
  c->d = *d;
  c->w = *w;
  const int L = d->n_layers;
  c->layer_ptrs = (const void**)malloc(sizeof(void*) * 9 * (size_t)L);
  const void* const* src[9] = {w->attn_norm, w->wq, w->wk, w->wv, w->wo,
                               w->ffn_norm, w->w_gate, w->w_up, w->w_down};
  for (int a = 0; a < 9; ++a)
    for (int l = 0; l < L; ++l) c->layer_ptrs[a * L + l] = src[a][l];
  c->w.attn_norm = c->layer_ptrs + 0 * L;
  c->w.wq = c->layer_ptrs + 1 * L;
  c->w.wk = c->layer_ptrs + 2 * L;
  c->w.wv = c->layer_ptrs + 3 * L;
  c->w.wo = c->layer_ptrs + 4 * L;
  c->w.ffn_norm = c->layer_ptrs + 5 * L;
  c->w.w_gate = c->layer_ptrs + 6 * L;
  c->w.w_up = c->layer_ptrs + 7 * L;
  c->w.w_down = c->layer_ptrs + 8 * L;
  c->Nv = d->n_views * (d->img_h / d->patch) * (d->img_w / d->patch);
  c->P = d->n_text + c->Nv + (d->proprio_dim > 0 ? 1 : 0);
  c->S = c->P + (d->parallel ? d->n_action : 0);
  c->T = c->S + (d->parallel ? 0 : d->n_action - 1);
  const int half = d->head_dim / 2;
  c->cos_t = (float*)malloc(sizeof(float) * (size_t)c->T * half);
  c->sin_t = (float*)malloc(sizeof(float) * (size_t)c->T * half);
  orc_rope_table(d, c->T, c->cos_t, c->sin_t);
  *out = c;
  return ORC_OK;
}

void orc_destroy(orc_ctx* c) {
  if (!c) return;
  free(c->layer_ptrs);
  free(c->cos_t);
  free(c->sin_t);
  free(c);
}

static size_t frame_bytes(const orc_dims* d) { return (size_t)d->n_views * d->img_h * d->img_w * 3; }

int orc_cache_new(const orc_ctx* c, int batch, orc_cache** out) {
  if (!c || batch < 1 || !out) return ORC_ERR_ARG;
  orc_cache* k = (orc_cache*)calloc(1, sizeof(orc_cache));
  if (!k) return ORC_ERR_OOM;
  const size_t L = c->d.n_layers, Hd = c->d.hidden;
  k->c = c;
  k->B = batch;
  k->K = (float*)calloc((size_t)batch * L * c->T * Hd, sizeof(float));
  k->V = (float*)calloc((size_t)batch * L * c->T * Hd, sizeof(float));
  k->H = (float*)calloc((size_t)batch * L * c->S * Hd, sizeof(float));
  k->prev = (uint8_t*)calloc((size_t)batch * frame_bytes(&c->d), 1);
  k->m_prev = (double*)calloc((size_t)batch, sizeof(double));
  k->valid = (uint8_t*)calloc((size_t)batch, 1);
  k->rel = (double*)calloc((size_t)batch * (c->Nv > 0 ? c->Nv : 1), sizeof(double));
  k->rel_valid = (uint8_t*)calloc((size_t)batch, 1);
  k->prev_ids = (int32_t*)calloc((size_t)batch * c->d.n_action, sizeof(int32_t));
  k->ids_valid = (uint8_t*)calloc((size_t)batch, 1);
  k->ent = (double*)calloc((size_t)batch * L, sizeof(double));
  k->ent_valid = (uint8_t*)calloc((size_t)batch, 1);
  if (!k->K || !k->V || !k->H || !k->prev || !k->m_prev || !k->valid || !k->rel || !k->rel_valid || !k->prev_ids ||
      !k->ids_valid || !k->ent || !k->ent_valid) {
    orc_cache_free(k);
    return ORC_ERR_OOM;
  }
  *out = k;
  return ORC_OK;
}

void orc_cache_free(orc_cache* k) {
  if (!k) return;
  free(k->K);
  free(k->V);
  free(k->H);
  free(k->prev);
  free(k->m_prev);
  free(k->valid);
  free(k->rel);
  free(k->rel_valid);
  free(k->prev_ids);
  free(k->ids_valid);
  free(k->ent);
  free(k->ent_valid);
  free(k);
}

/* Invalidation: the next step runs as if no cache existed (Algorithm 1). */
int orc_reset(orc_cache* k, int seq) {
  if (!k || seq < -1 || seq >= k->B) return ORC_ERR_ARG;
  for (int b = 0; b < k->B; ++b)
    if (seq == -1 || seq == b) k->valid[b] = k->rel_valid[b] = k->ids_valid[b] = k->ent_valid[b] = 0;
  return ORC_OK;
}

int orc_cache_read(const orc_cache* k, int seq, int kind, int layer, float* dst) {
  const orc_ctx* c = k->c;
  if (seq < 0 || seq >= k->B || layer < 0 || layer >= c->d.n_layers || kind < 0 || kind > 2) return ORC_ERR_ARG;
  const size_t Hd = c->d.hidden, L = c->d.n_layers;
  if (kind == 2) {
    memcpy(dst, k->H + (((size_t)seq * L + layer) * c->S) * Hd, sizeof(float) * c->S * Hd);
  } else {
    const float* src = kind == 0 ? k->K : k->V;
    memcpy(dst, src + (((size_t)seq * L + layer) * c->T) * Hd, sizeof(float) * c->T * Hd);
  }
  return ORC_OK;
}

int orc_cache_write(orc_cache* k, int seq, int kind, int layer, const float* src) {
  if (!k || !src) return ORC_ERR_ARG;
  const orc_ctx* c = k->c;
  if (seq < 0 || seq >= k->B || layer < 0 || layer >= c->d.n_layers || kind < 0 || kind > 1) return ORC_ERR_ARG;
  const size_t Hd = c->d.hidden, L = c->d.n_layers;
  float* dst = (kind == 0 ? k->K : k->V) + (((size_t)seq * L + layer) * c->T) * Hd;
  memcpy(dst, src, sizeof(float) * c->T * Hd);
  return ORC_OK;
}

int orc_cache_state(const orc_cache* k, int seq, double* m_prev, int* valid) {
  if (!k || seq < 0 || seq >= k->B) return ORC_ERR_ARG;
  *m_prev = k->m_prev[seq];
  *valid = k->valid[seq];
  return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Transformer layer over a set of rows (Llama-2 block).                    */
/* ------------------------------------------------------------------------ */

/* Keys a query at `pos` attends to: every position j <= pos (causal), except
 * that rows of the parallel action block see the whole prefix and the whole
 * block (bidirectional block). */
static int key_limit(const orc_ctx* c, int pos) {
  if (c->d.parallel && pos >= c->P) return c->P + c->d.n_action; /* exclusive */
  return pos + 1;
}

/* One decoder layer for n rows at positions pos[i]; x holds their fp32
 * residual rows.  Fresh K/V of every row are written to the cache before any
 * row attends, and attention reads the cache (reused + fresh entries).
 * rel (Stage 2, NULL = not wanted) receives, per visual patch v, the softmax
 * probability of key 1 + v summed over the text rows among the n (in row
 * order) and, within a row, over the heads in order.
 * ent (Stage 3 adaptive, NULL = not wanted) receives the layer's normalized
 * attention entropy: over the text rows among the n that attend to two or
 * more keys, and every head, the mean of H / ln(keys), H = -sum_j p_j ln p_j
 * of the row's causal softmax (rows in order, heads in order within a row). */
static void layer_rows(const orc_ctx* c, orc_cache* k, int b, int l, int n, const int32_t* pos, float* x,
                       double* rel, double* ent) {
  const int Hd = c->d.hidden, nh = c->d.n_heads, hd = c->d.head_dim, F = c->d.ffn;
  const size_t T = c->T, L = c->d.n_layers;
  float* Kl = k->K + (((size_t)b * L + l) * T) * Hd;
  float* Vl = k->V + (((size_t)b * L + l) * T) * Hd;
  double* h = (double*)malloc(sizeof(double) * (size_t)n * Hd);
  double* q = (double*)malloc(sizeof(double) * (size_t)n * Hd);
  double* kk = (double*)malloc(sizeof(double) * (size_t)n * Hd);
  double* vv = (double*)malloc(sizeof(double) * (size_t)n * Hd);
  double* att = (double*)malloc(sizeof(double) * (size_t)n * Hd);
  double* y = (double*)malloc(sizeof(double) * (size_t)n * Hd);
  double* g = (double*)malloc(sizeof(double) * (size_t)n * F);
  double* u = (double*)malloc(sizeof(double) * (size_t)n * F);

  /* attention block */
  for (int i = 0; i < n; ++i) rmsnorm_row(c, x + (size_t)i * Hd, c->w.attn_norm[l], h + (size_t)i * Hd);
  linear(c, c->w.wq[l], Hd, Hd, n, h, q);
  linear(c, c->w.wk[l], Hd, Hd, n, h, kk);
  linear(c, c->w.wv[l], Hd, Hd, n, h, vv);
  for (int i = 0; i < n; ++i) {
    for (int hh = 0; hh < nh; ++hh) {
      rope_head(c, q + (size_t)i * Hd + (size_t)hh * hd, pos[i]);
      rope_head(c, kk + (size_t)i * Hd + (size_t)hh * hd, pos[i]);
    }
    for (int e = 0; e < Hd; ++e) {
      q[(size_t)i * Hd + e] = store_act(c, q[(size_t)i * Hd + e]);
      Kl[(size_t)pos[i] * Hd + e] = (float)store_act(c, kk[(size_t)i * Hd + e]);
      Vl[(size_t)pos[i] * Hd + e] = (float)store_act(c, vv[(size_t)i * Hd + e]);
    }
  }
  const double scale = 1.0 / sqrt((double)hd);
  const int Nv = c->Nv;
  /* per (row, head): probability of each visual key (text rows only) */
  double* pv = rel ? (double*)calloc((size_t)n * nh * (Nv > 0 ? Nv : 1), sizeof(double)) : NULL;
  /* per (row, head): normalized entropy, or -1 where the row does not count */
  double* hv = ent ? (double*)malloc(sizeof(double) * (size_t)n * nh) : NULL;
#pragma omp parallel for schedule(dynamic)
  for (int ih = 0; ih < n * nh; ++ih) {
    const int i = ih / nh, hh = ih % nh;
    const int nk = key_limit(c, pos[i]);
    double* sc = (double*)malloc(sizeof(double) * (size_t)nk);
    double kd[512];
    const double* qi = q + (size_t)i * Hd + (size_t)hh * hd;
    double mx = -INFINITY;
    for (int j = 0; j < nk; ++j) {
      for (int e = 0; e < hd; ++e) kd[e] = Kl[(size_t)j * Hd + (size_t)hh * hd + e];
      sc[j] = dot(qi, kd, hd) * scale;
      if (sc[j] > mx) mx = sc[j];
    }
    double z = 0.0, zu = 0.0;
    for (int j = 0; j < nk; ++j) {
      const double u = sc[j] - mx;
      sc[j] = exp(u);
      z += sc[j];
      zu += sc[j] * u;
    }
    /* H = -sum p ln p with p = e^u / z: ln z - sum e^u u / z */
    if (hv) hv[ih] = (pos_is_text(c, pos[i]) && nk >= 2) ? (log(z) - zu / z) / log((double)nk) : -1.0;
    if (pv && pos_is_text(c, pos[i]))
      for (int j = 1; j < nk && j <= Nv; ++j) pv[((size_t)i * nh + hh) * Nv + (j - 1)] = sc[j] / z;
    for (int e = 0; e < hd; ++e) {
      double o = 0.0;
      for (int j = 0; j < nk; ++j) o += sc[j] * (double)Vl[(size_t)j * Hd + (size_t)hh * hd + e];
      att[(size_t)i * Hd + (size_t)hh * hd + e] = store_act(c, o / z);
    }
    free(sc);
  }
  if (hv) {
    double sum = 0.0;
    int cnt = 0;
    for (int q = 0; q < n * nh; ++q)
      if (hv[q] >= 0.0) {
        sum += hv[q];
        ++cnt;
      }
    *ent = cnt ? sum / cnt : 0.0;
    free(hv);
  }
  if (pv) {
    for (int v = 0; v < Nv; ++v) rel[v] = 0.0;
    for (int i = 0; i < n; ++i)
      for (int hh = 0; hh < nh; ++hh)
        for (int v = 0; v < Nv; ++v) rel[v] += pv[((size_t)i * nh + hh) * Nv + v];
    free(pv);
  }
  linear(c, c->w.wo[l], Hd, Hd, n, att, y);
  for (size_t e = 0; e < (size_t)n * Hd; ++e) x[e] = (float)((double)x[e] + y[e]);

  /* MLP block: SwiGLU */
  for (int i = 0; i < n; ++i) rmsnorm_row(c, x + (size_t)i * Hd, c->w.ffn_norm[l], h + (size_t)i * Hd);
  linear(c, c->w.w_gate[l], F, Hd, n, h, g);
  linear(c, c->w.w_up[l], F, Hd, n, h, u);
  for (size_t e = 0; e < (size_t)n * F; ++e) {
    double s = g[e] / (1.0 + exp(-g[e]));
    g[e] = store_act(c, s * u[e]);
  }
  linear(c, c->w.w_down[l], Hd, F, n, g, y);
  for (size_t e = 0; e < (size_t)n * Hd; ++e) x[e] = (float)((double)x[e] + y[e]);

  free(h); free(q); free(kk); free(vv); free(att); free(y); free(g); free(u);
}

int orc_layer(orc_ctx* c, orc_cache* k, int seq, int layer, int n, const int32_t* pos, float* x) {
  if (!c || !k || k->c != c || !pos || !x || seq < 0 || seq >= k->B || layer < 0 || layer >= c->d.n_layers ||
      n < 1 || n > c->S)
    return ORC_ERR_ARG;
  for (int i = 0; i < n; ++i) {
    if (pos[i] < 0 || pos[i] >= c->S) return ORC_ERR_ARG;
    for (int j = 0; j < i; ++j)
      if (pos[j] == pos[i]) return ORC_ERR_ARG;
  }
  layer_rows(c, k, seq, layer, n, pos, x, NULL, NULL);
  return ORC_OK;
}

/* Layer-0 input of the token at `pos` (Sec. III-A layout: BOS, visual
 * patches view-major/row-major, proprio, rest of the text, action block). */
static void embed_row(const orc_ctx* c, int pos, const uint8_t* frame, const int32_t* prompt,
                      const float* proprio, float* x) {
  const int Hd = c->d.hidden;
  const int has_p = c->d.proprio_dim > 0;
  if (pos == 0 || (pos > c->Nv + has_p && pos < c->P)) {
    const int t = pos == 0 ? 0 : pos - c->Nv - has_p;
    const int id = prompt[t];
    for (int e = 0; e < Hd; ++e) x[e] = (float)wget(c, c->w.tok_emb, (size_t)id * Hd + e);
  } else if (pos_is_visual(c, pos)) {
    /* visual token: (W_p . patch bytes) / 255 */
    const int v = pos - 1, n = c->d.patch * c->d.patch * 3;
    double* pv = (double*)malloc(sizeof(double) * n);
    for (int e = 0; e < n; ++e) pv[e] = (double)*patch_px(&c->d, frame, v, e);
    double* wr = (double*)malloc(sizeof(double) * n);
    for (int o = 0; o < Hd; ++o) {
      for (int e = 0; e < n; ++e) wr[e] = wget(c, c->w.patch_w, (size_t)o * n + e);
      x[o] = (float)(dot(pv, wr, n) / 255.0);
    }
    free(pv);
    free(wr);
  } else if (has_p && pos == c->Nv + 1) {
    const int n = c->d.proprio_dim;
    for (int o = 0; o < Hd; ++o) {
      double s = 0.0;
      for (int e = 0; e < n; ++e) s += wget(c, c->w.proprio_w, (size_t)o * n + e) * (double)proprio[e];
      x[o] = (float)s;
    }
  } else { /* parallel action block */
    const int a = pos - c->P;
    for (int e = 0; e < Hd; ++e) x[e] = (float)wget(c, c->w.action_emb, (size_t)a * Hd + e);
  }
}

/* Final norm and the action-bin rows of the LM head -> logits, argmax,
 * margins, and the entropy of the bin softmax.  With vm != NULL also every
 * other row of the LM head: p1 - p2 of the softmax over the whole
 * vocabulary (the two largest probabilities of any tokens). */
static void head_row(const orc_ctx* c, const float* x, double* logits, int32_t* id, double* pm, double* lg,
                     double* ent, double* vm) {
  const int Hd = c->d.hidden, nb = c->d.n_bins, V = c->d.vocab;
  double* h = (double*)malloc(sizeof(double) * Hd);
  double* wr = (double*)malloc(sizeof(double) * Hd);
  rmsnorm_row(c, x, c->w.final_norm, h);
  for (int j = 0; j < nb; ++j) {
    const size_t row = (size_t)(V - nb + j);
    for (int e = 0; e < Hd; ++e) wr[e] = wget(c, c->w.lm_head, row * Hd + e);
    logits[j] = dot(h, wr, Hd);
  }
  orc_margin(logits, nb, id, pm, lg);
  *ent = orc_entropy(logits, nb);
  if (vm) {
    double* all = (double*)malloc(sizeof(double) * V);
    for (int r = 0; r < V - nb; ++r) {
      for (int e = 0; e < Hd; ++e) wr[e] = wget(c, c->w.lm_head, (size_t)r * Hd + e);
      all[r] = dot(h, wr, Hd);
    }
    memcpy(all + (V - nb), logits, sizeof(double) * nb);
    int32_t top;
    double gap;
    orc_margin(all, V, &top, vm, &gap);
    free(all);
  }
  free(h);
  free(wr);
}

/* ------------------------------------------------------------------------ */
/* Algorithm 1 for one sequence.                                            */
/* ------------------------------------------------------------------------ */

static int step_seq(orc_ctx* c, orc_cache* k, int b, const uint8_t* frame, const int32_t* prompt,
                    const float* proprio, uint32_t num, uint32_t den, double tau_m,
                    const uint16_t* permille, const orc_opts* o, orc_out* out) {
  const int L = c->d.n_layers, Hd = c->d.hidden, S = c->S, D = c->d.n_action, nb = c->d.n_bins;
  const size_t fb = frame_bytes(&c->d);
  uint8_t* prev = k->prev + (size_t)b * fb;

  /* Gate on the margin of step t-1 (strict <); an empty cache runs full. */
  const int gate = !k->valid[b] || k->m_prev[b] < tau_m;
  int full = gate;
  if (o && o->gate_override && o->gate_override[b] >= 0) full = o->gate_override[b] ? 1 : 0;
  if (!k->valid[b]) full = 1;
  out->gate_auto[b] = (uint8_t)gate;
  out->recomputed[b] = (uint8_t)full;

  int32_t* idx = (int32_t*)malloc(sizeof(int32_t) * S);
  int32_t* M = (int32_t*)malloc(sizeof(int32_t) * L);
  uint8_t* mask = (uint8_t*)malloc((size_t)(c->Nv > 0 ? c->Nv : 1));
  uint8_t* relevant = (uint8_t*)malloc((size_t)(c->Nv > 0 ? c->Nv : 1));
  /* Stage 2 uses the relevance the previous step measured */
  const int s2 = o && o->s2_top_k > 0;
  const double* rel_prev = (s2 && k->rel_valid[b]) ? k->rel + (size_t)b * c->Nv : NULL;
  /* Stage 3: the caller's schedule, or the one the previous step's layer
   * entropies give (a lock-step replay may impose the other side's) */
  const int s3 = o && o->s3_adaptive;
  uint16_t* sched = (uint16_t*)malloc(sizeof(uint16_t) * L);
  if (s3 && k->ent_valid[b])
    orc_entropy_schedule(k->ent + (size_t)b * L, L, o->s3_lo, o->s3_hi, o->s3_weight, sched);
  else
    memcpy(sched, permille, sizeof(uint16_t) * L);
  if (out->schedule) memcpy(out->schedule + (size_t)b * L, sched, sizeof(uint16_t) * L);
  const uint16_t* use = (s3 && o->s3_forced) ? o->s3_forced + (size_t)b * L : sched;
  int nS = orc_select2(&c->d, frame, prev, k->valid[b], num, den, use, full, rel_prev, s2 ? o->s2_top_k : 0,
                       mask, relevant, idx, M);
  free(sched);
  if (nS < 0) { free(idx); free(M); free(mask); free(relevant); return ORC_ERR_ARG; }
  if (out->static_mask) memcpy(out->static_mask + (size_t)b * c->Nv, mask, (size_t)c->Nv);
  if (out->relevant) memcpy(out->relevant + (size_t)b * c->Nv, relevant, (size_t)c->Nv);
  free(relevant);
  if (out->idx) memcpy(out->idx + (size_t)b * S, idx, sizeof(int32_t) * S);
  if (out->M) memcpy(out->M + (size_t)b * L, M, sizeof(int32_t) * L);

  /* Partial (or full) forward over the prefix pass. */
  float* x = (float*)malloc(sizeof(float) * (size_t)S * Hd);
  for (int i = 0; i < M[0]; ++i) embed_row(c, idx[i], frame, prompt, proprio, x + (size_t)i * Hd);
  float* Hb = k->H + (size_t)b * L * S * Hd;
  double* rel_now = s2 ? (double*)calloc((size_t)(c->Nv > 0 ? c->Nv : 1), sizeof(double)) : NULL;
  double* ent_now = s3 ? (double*)calloc((size_t)L, sizeof(double)) : NULL;
  for (int l = 0; l < L; ++l) {
    if (l > 0) {
      /* rows computed at layer l-1 record their layer-l input; rows that join
       * at layer l start from the cached layer-l input of that position */
      for (int i = 0; i < M[l - 1]; ++i)
        memcpy(Hb + ((size_t)l * S + idx[i]) * Hd, x + (size_t)i * Hd, sizeof(float) * Hd);
      for (int i = M[l - 1]; i < M[l]; ++i)
        memcpy(x + (size_t)i * Hd, Hb + ((size_t)l * S + idx[i]) * Hd, sizeof(float) * Hd);
    }
    layer_rows(c, k, b, l, M[l], idx, x, (s2 && l == o->s2_layer) ? rel_now : NULL, s3 ? ent_now + l : NULL);
  }
  /* every text row is recomputed at every layer, so the layer entropies are
   * complete too; the next step's Stage 3 reads them */
  if (out->layer_entropy)
    for (int l = 0; l < L; ++l) out->layer_entropy[(size_t)b * L + l] = s3 ? ent_now[l] : 0.0;
  if (s3) memcpy(k->ent + (size_t)b * L, ent_now, sizeof(double) * L);
  k->ent_valid[b] = (uint8_t)s3;
  free(ent_now);
  /* every text row is recomputed at every layer, so this step's relevance is
   * complete; it is what the next step's Stage 2 reads */
  if (out->relevance)
    for (int v = 0; v < c->Nv; ++v) out->relevance[(size_t)b * c->Nv + v] = s2 ? rel_now[v] : 0.0;
  if (s2) memcpy(k->rel + (size_t)b * c->Nv, rel_now, sizeof(double) * c->Nv);
  k->rel_valid[b] = (uint8_t)s2;
  free(rel_now);

  /* Action tokens. */
  double* lg = (double*)malloc(sizeof(double) * nb);
  double sig_sum = 0.0, sig_min = INFINITY;
  int32_t* ids = out->action_ids + (size_t)b * D;
  for (int a = 0; a < D; ++a) {
    int slot = -1, target;
    if (c->d.parallel) {
      target = c->P + a;
    } else if (a == 0) {
      target = c->P - 1;
    } else {
      target = -1;
    }
    float* xr;
    float* xdec = NULL;
    if (target >= 0) {
      for (int i = 0; i < M[L - 1]; ++i)
        if (idx[i] == target) { slot = i; break; }
      if (slot < 0) { free(idx); free(M); free(mask); free(x); free(lg); return ORC_ERR_ARG; }
      xr = x + (size_t)slot * Hd;
    } else {
      /* autoregressive decode: feed bin a-1 at position P + a - 1 */
      const int fed = (o && o->forced_ids) ? o->forced_ids[(size_t)b * D + a - 1] : ids[a - 1];
      const int tok = c->d.vocab - nb + fed;
      int32_t p = c->P + a - 1;
      xdec = (float*)malloc(sizeof(float) * Hd);
      for (int e = 0; e < Hd; ++e) xdec[e] = (float)wget(c, c->w.tok_emb, (size_t)tok * Hd + e);
      for (int l = 0; l < L; ++l) layer_rows(c, k, b, l, 1, &p, xdec, NULL, NULL);
      xr = xdec;
    }
    double pm, gap, ent, vm = 0.0;
    const int want_vm = (o && o->margin_kind == 2) || out->vocab_margin;
    head_row(c, xr, lg, &ids[a], &pm, &gap, &ent, want_vm ? &vm : NULL);
    if (out->logits) memcpy(out->logits + ((size_t)b * D + a) * nb, lg, sizeof(double) * nb);
    out->margins[(size_t)b * D + a] = pm;
    out->logit_gap[(size_t)b * D + a] = gap;
    if (out->entropy) out->entropy[(size_t)b * D + a] = ent;
    if (out->vocab_margin) out->vocab_margin[(size_t)b * D + a] = vm;
    const double sig = (o && o->margin_kind == 1) ? gap : (o && o->margin_kind == 2) ? vm : pm;
    sig_sum += sig;
    if (sig < sig_min) sig_min = sig;
    free(xdec);
  }
  const double m_t = (o && o->reduction == 1) ? sig_min : sig_sum / D;
  out->step_margin[b] = m_t;
  /* action delta against the previous step's bins (Sec. VI) */
  int32_t* pid = k->prev_ids + (size_t)b * D;
  int32_t delta = 0;
  if (k->ids_valid[b])
    for (int a = 0; a < D; ++a) delta += abs(ids[a] - pid[a]);
  if (out->action_delta) out->action_delta[b] = delta;
  memcpy(pid, ids, sizeof(int32_t) * D);
  k->ids_valid[b] = 1;
  k->m_prev[b] = m_t;
  k->valid[b] = 1;
  memcpy(prev, frame, fb);
  free(idx); free(M); free(mask); free(x); free(lg);
  return ORC_OK;
}

int orc_step(orc_ctx* c, orc_cache* k, const uint8_t* frames, const int32_t* prompt_ids,
             const float* proprio, uint32_t tau_num, uint32_t tau_den, double tau_margin,
             const uint16_t* reuse_permille, const orc_opts* opts, orc_out* out) {
  if (!c || !k || k->c != c || !frames || !prompt_ids || !reuse_permille || !out || !out->action_ids ||
      !out->margins || !out->logit_gap || !out->recomputed || !out->gate_auto || !out->step_margin || tau_den == 0)
    return ORC_ERR_ARG;
  if (c->d.proprio_dim > 0 && !proprio) return ORC_ERR_ARG;
  if (opts && (opts->margin_kind < 0 || opts->margin_kind > 2)) return ORC_ERR_ARG;
  if (opts && (opts->s2_top_k < 0 || (opts->s2_top_k > 0 && (opts->s2_layer < 0 || opts->s2_layer >= c->d.n_layers))))
    return ORC_ERR_ARG;
  if (opts && opts->s3_adaptive &&
      (opts->s3_lo < 0 || opts->s3_lo > opts->s3_hi || opts->s3_hi > 1000 || opts->s3_weight < 0 ||
       opts->s3_weight > 1000))
    return ORC_ERR_ARG;
  if (opts && opts->s3_forced)
    for (int q = 0; q < k->B * c->d.n_layers; ++q)
      if (opts->s3_forced[q] > 1000) return ORC_ERR_ARG;
  const size_t fb = frame_bytes(&c->d);
  for (int b = 0; b < k->B; ++b) {
    if (opts && opts->active && !opts->active[b]) {
      /* a sequence that sits the step out: nothing of it changes */
      const size_t D = c->d.n_action, nb = c->d.n_bins, Nv = c->Nv, S = c->S, L = c->d.n_layers;
      memset(out->action_ids + b * D, 0, sizeof(int32_t) * D);
      memset(out->margins + b * D, 0, sizeof(double) * D);
      memset(out->logit_gap + b * D, 0, sizeof(double) * D);
      if (out->logits) memset(out->logits + b * D * nb, 0, sizeof(double) * D * nb);
      out->recomputed[b] = 0;
      out->gate_auto[b] = 0;
      out->step_margin[b] = 0.0;
      if (out->static_mask) memset(out->static_mask + b * Nv, 0, Nv);
      if (out->idx) memset(out->idx + b * S, 0, sizeof(int32_t) * S);
      if (out->M) memset(out->M + b * L, 0, sizeof(int32_t) * L);
      if (out->relevance) memset(out->relevance + b * Nv, 0, sizeof(double) * Nv);
      if (out->relevant) memset(out->relevant + b * Nv, 0, Nv);
      if (out->entropy) memset(out->entropy + b * D, 0, sizeof(double) * D);
      if (out->vocab_margin) memset(out->vocab_margin + b * D, 0, sizeof(double) * D);
      if (out->action_delta) out->action_delta[b] = 0;
      if (out->layer_entropy) memset(out->layer_entropy + b * L, 0, sizeof(double) * L);
      if (out->schedule) memset(out->schedule + b * L, 0, sizeof(uint16_t) * L);
      continue;
    }
    int r = step_seq(c, k, b, frames + (size_t)b * fb, prompt_ids + (size_t)b * c->d.n_text,
                     proprio ? proprio + (size_t)b * c->d.proprio_dim : NULL, tau_num, tau_den, tau_margin,
                     reuse_permille, opts, out);
    if (r) return r;
  }
  return ORC_OK;
}
