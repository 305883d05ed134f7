// C-ABI of libvlac: context (repacked weights, TMA descriptors, workspace),
// caller-owned caches and the step of Algorithm 1.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

#include "internal.cuh"

using namespace vlac;

namespace vlac {
bool g_pdl = true;
}

namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

constexpr uint32_t kDefaultWaitLimit = 1u << 24;

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// A bump allocator over one device allocation.
struct Carve {
  size_t off = 0;
  template <typename P>
  void take(P*& p, size_t bytes, char* base) {
    off = align_up(off, 256);
    p = base ? reinterpret_cast<P*>(base + off) : nullptr;
    off += bytes;
  }
};

}  // namespace

struct vlac_ctx {
  vlac_dims d;
  int P, S, Tc, Nv, pdim, kpad, has_p, rows_cap;
  bool bf16;
  size_t esz;
  int dev;
  int n_sm = 1;
  int gemv_ns = 4;  // decode-GEMV weight ring stages (32 KB each)
  int gemv_pf_kb = 0;  // decode-GEMV L2 prefetch of the next projection, KB per CTA (measured: off is best)
  int dpass_bar = 1;  // persistent pass: grid barrier kind (VLAC_DPASS_BAR: 1 release/acquire, 0 fences)
  bool dpass_kv = true;  // persistent pass: attention K/V staged in shared memory (VLAC_DPASS_KV)
  bool fuse_rows = true;  // prefix: a layer's down residual and the next layer's input norm in one launch (VLAC_FUSE_ROWS)
  bool use_dpass = true;  // decode passes as one persistent cooperative launch (k_dpass.cu) where supported
  int dpass_attn_chunks = 0;  // its key ranges per (sequence, head); 0 = chosen from the SM count
  void** dp_ptrs = nullptr;  // device: per-layer pointers [w_qkv | w_o | w_gu | w_d | g_attn | g_ffn][L]
  unsigned* dp_bar = nullptr;  // device: the persistent pass's grid-barrier counter
  char* dmem = nullptr;  // decode-streaming copies of the projections
  std::vector<void*> dqkv, dwo, dgu, dwd;
  // weights
  char* wmem = nullptr;
  void *tok_emb, *patch_w, *proprio_w, *action_emb, *final_norm, *head_w;
  void* head_full;  // the whole LM head [vocab][hidden]; head_w is its last n_bins rows
  std::vector<void*> attn_norm, ffn_norm, wqkv, wo, wgu, wd;
  float *rope_cos, *rope_sin;
  // TMA descriptors (bf16 only)
  std::vector<CUtensorMap> tm_qkv, tm_o, tm_gu, tm_d;
  CUtensorMap tm_patch;
  ActMaps tm_A, tm_AO, tm_G, tm_col;
  int split_qkv = 1, split_o = 1, split_gu = 1, split_d = 1;
  // where each projection's K-split partials go (uniform splits, or whole
  // tiles plus K-split tail tiles when the tiles exceed one wave of SMs)
  SplitPlan sp_qkv{}, sp_o{}, sp_gu{}, sp_d{};
  float* part_tail = nullptr;  // compact partials of the tail tiles' later splits
  size_t part_tail_elems = 0;
  // workspace
  char* wsmem = nullptr;
  float *X, *Xd, *part;
  size_t part_elems = 0;
  void *A, *Q, *AO, *G, *col;
  StepParams* prm;
  int3* stats;
  uint8_t *mask, *full;
  int *idx, *M, *off, *emit_slot, *off_dec, *idx_dec, *err;
  float *logits_ws, *attn_part, *ssq_a, *ssq_b;
  unsigned* attn_cnt;  // decode attention: finished key chunks per (sequence, head); zero between launches
  // staged per-step inputs and outputs (fixed addresses, so a step can be a graph)
  uint8_t* in_frames;
  int32_t* in_prompt;
  float* in_proprio;
  int8_t* in_override;
  int32_t* in_forced;
  uint8_t* in_active;
  uint8_t* in_s2_forced;
  int32_t* o_ids;
  float *o_margins, *o_gaps, *o_step_margin, *o_logits;
  uint8_t *o_recomputed, *o_gate_auto, *o_mask;
  int32_t *o_idx, *o_M;
  float* o_rel;         // Stage-2 relevance of the step [B][Nv]
  uint8_t* o_relevant;  // Stage-2 removal set of the step [B][Nv]
  float* rel_part;      // Stage-2 relevance per (sequence, head) [B][n_heads][Nv]
  bool s2_on = false;   // this step measures and applies Stage 2
  int s2_layer = 0;
  float *o_entropy, *o_vm;  // per action token: bin-softmax entropy, whole-vocabulary margin
  int32_t* o_delta;         // per sequence: action delta
  void* vh_rows;            // whole-vocabulary margin: normed action rows [rows][hidden] (T)
  float* vh_logits;         // and their logits over the non-bin rows [rows][vocab - n_bins]
  bool vm_on = false;       // this step computes the whole-vocabulary margin
  // Stage 3 adaptive: per-layer entropies per (sequence, head, text row)
  // [L][B][n_heads][nt], the schedule derived [B][L] and applied [B][L], the
  // replayed schedule [B][L] and the entropies returned [B][L]
  float* ent_part;
  uint16_t *sched_own, *sched_use, *in_s3_forced;
  float* o_lent;
  bool s3_on = false;  // this step measures the layer entropies
  int text_lo = 0, n_textrows = 0;  // text rows after the image: positions text_lo .. P-1
  cudaStream_t cap_stream = nullptr;
  bool use_graph = true;
  bool fatal = false;  // a launch was refused for exceeding a workspace buffer
  int* err_host = nullptr;  // pinned
  uint64_t launches = 0;
  uint32_t wait_limit = kDefaultWaitLimit;
  // optional per-launch timing
  struct ProfRec {
    int kind;
    double bytes;
    cudaEvent_t a, b;
  };
  bool prof_on = false;
  std::vector<ProfRec> prof;
  std::vector<cudaEvent_t> ev_pool;
};

struct vlac_cache {
  vlac_ctx* ctx;
  int B;
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t gexec = nullptr;
  int eager_steps = 0;
  uint64_t graph_launches = 0;
  int graph_sig = 0;  // what the graph was captured with: Stage 2 (0 off, 1 + layer), the vocabulary margin, Stage 3
  void *K, *V;
  float* H;
  uint8_t *prev, *valid;
  float* m_prev;
  float* rel;          // [B][Nv] the last step's Stage-2 relevance
  uint8_t* rel_valid;  // [B] rel holds one
  float* ent;          // [B][L] the last step's per-layer attention entropy (Stage 3 adaptive)
  uint8_t* ent_valid;  // [B] ent holds it
  int32_t* prev_ids;   // [B][n_action] the previous step's action bins
  uint8_t* ids_valid;  // [B] prev_ids holds them
  size_t kv_seq_stride, h_seq_stride;  // elements per sequence
  KvMaps kvm;                          // TMA maps of K and V (bf16)
};

#define CK(x)                                  \
  do {                                         \
    if ((x) != cudaSuccess) {                  \
      (void)cudaGetLastError();                \
      return VLAC_ERR_CUDA;                    \
    }                                          \
  } while (0)

// ---- dims ------------------------------------------------------------------

int vlac::check_dims(const vlac_dims* d) {
  if (!d) return VLAC_ERR_INVALID_ARG;
  if (d->n_layers < 1 || d->n_layers > kMaxLayers || d->n_heads < 1 || d->n_heads * d->head_dim != d->hidden ||
      d->ffn < 1 || d->vocab < 1 || d->n_bins < 2 || d->n_bins > d->vocab || d->n_bins > 4096 || d->patch < 1 ||
      d->img_h < d->patch || d->img_w < d->patch || d->img_h % d->patch || d->img_w % d->patch || d->n_views < 1 ||
      d->n_text < 1 || d->n_action < 1 || d->proprio_dim < 0 || d->proprio_dim > 256 || d->max_batch < 1 ||
      d->max_batch > 8 || (d->parallel != 0 && d->parallel != 1) || (!d->parallel && d->n_text < 2) ||
      d->n_bins % 16 ||
      !(d->rms_eps >= 0.f) || !(d->rope_theta > 0.f))
    return VLAC_ERR_INVALID_ARG;
  if (d->dtype != VLAC_F32 && d->dtype != VLAC_BF16) return VLAC_ERR_INVALID_ARG;
  if (d->head_dim != 64 && d->head_dim != 128) return VLAC_ERR_UNSUPPORTED;
  const int nv = d->n_views * (d->img_h / d->patch) * (d->img_w / d->patch);
  if (nv > 4096) return VLAC_ERR_UNSUPPORTED;
  if (d->dtype == VLAC_BF16) {
    if (d->hidden % 128 || d->ffn % 64) return VLAC_ERR_UNSUPPORTED;
  } else {
    if (d->hidden % 4 || d->ffn % 4) return VLAC_ERR_UNSUPPORTED;
  }
  return VLAC_OK;
}

static EncodeTiledFn get_encode() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 2D bf16 tensor [rows][cols] (cols contiguous), box = 64 columns x box_rows, 128B swizzle.
static bool make_map(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  EncodeTiledFn enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D bf16 tensor {cols, rows, planes} (cols contiguous, planes of rows x
// cols), box = 64 columns x box_rows x 1, 128B swizzle; reads outside it are zeros.
static bool make_map3(CUtensorMap* m, const void* base, uint64_t planes, uint64_t rows, uint64_t cols,
                      uint32_t box_rows) {
  EncodeTiledFn enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[3] = {cols, rows, planes};
  cuuint64_t strides[2] = {cols * 2, rows * cols * 2};
  cuuint32_t box[3] = {64, box_rows, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// ---- create / destroy -----------------------------------------------------------

extern "C" int vlac_destroy(vlac_ctx* c) {
  if (!c) return VLAC_ERR_INVALID_ARG;
  for (auto& r : c->prof) {
    cudaEventDestroy(r.a);
    cudaEventDestroy(r.b);
  }
  for (auto e : c->ev_pool) cudaEventDestroy(e);
  if (c->cap_stream) cudaStreamDestroy(c->cap_stream);
  if (c->wmem) cudaFree(c->wmem);
  if (c->dmem) cudaFree(c->dmem);
  if (c->wsmem) cudaFree(c->wsmem);
  if (c->err_host) cudaFreeHost(c->err_host);
  delete c;
  return VLAC_OK;
}

extern "C" int vlac_create(const vlac_dims* dims, const vlac_weights* w, vlac_ctx** out) {
  int rc = check_dims(dims);
  if (rc) return rc;
  if (!w || !out || !w->tok_emb || !w->patch_w || !w->attn_norm || !w->wq || !w->wk || !w->wv || !w->wo ||
      !w->ffn_norm || !w->w_gate || !w->w_up || !w->w_down || !w->final_norm || !w->lm_head)
    return VLAC_ERR_INVALID_ARG;
  if (dims->proprio_dim > 0 && !w->proprio_w) return VLAC_ERR_INVALID_ARG;
  if (dims->parallel && !w->action_emb) return VLAC_ERR_INVALID_ARG;
  for (int l = 0; l < dims->n_layers; ++l)
    if (!w->attn_norm[l] || !w->wq[l] || !w->wk[l] || !w->wv[l] || !w->wo[l] || !w->ffn_norm[l] || !w->w_gate[l] ||
        !w->w_up[l] || !w->w_down[l])
      return VLAC_ERR_INVALID_ARG;

  vlac_ctx* c = new (std::nothrow) vlac_ctx();
  if (!c) return VLAC_ERR_OOM;
  // test hook (fault injection on the host): VLAC_FAIL_ALLOC=n makes the
  // n-th allocation of this call fail as cudaMalloc would, without calling it
  int alloc_no = 0, fail_at = 0;
  if (const char* e = std::getenv("VLAC_FAIL_ALLOC")) fail_at = std::atoi(e);
  auto dev_alloc = [&](void** ptr, size_t bytes, bool host) {
    if (++alloc_no == fail_at) return cudaErrorMemoryAllocation;
    return host ? cudaMallocHost(ptr, bytes) : cudaMalloc(ptr, bytes);
  };
  if (const char* e = std::getenv("VLAC_PDL")) g_pdl = std::atoi(e) != 0;
  if (const char* e = std::getenv("VLAC_GRAPH")) c->use_graph = std::atoi(e) != 0;
  if (const char* e = std::getenv("VLAC_GEMV_NS")) c->gemv_ns = std::max(2, std::min(24, std::atoi(e)));
  if (const char* e = std::getenv("VLAC_GEMV_PF_KB")) c->gemv_pf_kb = std::max(0, std::atoi(e));
  if (const char* e = std::getenv("VLAC_DPASS")) c->use_dpass = std::atoi(e) != 0;
  if (const char* e = std::getenv("VLAC_DPASS_BAR")) c->dpass_bar = std::atoi(e) != 0 ? 1 : 0;
  if (const char* e = std::getenv("VLAC_DPASS_KV")) c->dpass_kv = std::atoi(e) != 0;
  if (const char* e = std::getenv("VLAC_FUSE_ROWS")) c->fuse_rows = std::atoi(e) != 0;
  if (const char* e = std::getenv("VLAC_DPASS_ATTN_CHUNKS")) c->dpass_attn_chunks = std::max(0, std::atoi(e));
  c->d = *dims;
  const vlac_dims& d = c->d;
  c->bf16 = d.dtype == VLAC_BF16;
  c->esz = c->bf16 ? 2 : 4;
  c->Nv = d.n_views * (d.img_h / d.patch) * (d.img_w / d.patch);
  c->has_p = d.proprio_dim > 0;
  c->P = d.n_text + c->Nv + c->has_p;
  c->text_lo = 1 + c->Nv + c->has_p;
  c->n_textrows = c->P - c->text_lo;
  c->S = c->P + (d.parallel ? d.n_action : 0);
  c->Tc = c->S + (d.parallel ? 0 : d.n_action - 1);
  c->pdim = d.patch * d.patch * 3;
  c->kpad = c->bf16 ? (int)align_up(c->pdim, 64) : c->pdim;
  c->rows_cap = d.max_batch * c->S;
  if (cudaGetDevice(&c->dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&c->n_sm, cudaDevAttrMultiProcessorCount, c->dev) != cudaSuccess) {
    delete c;
    return VLAC_ERR_CUDA;
  }
  const size_t L = d.n_layers, Hd = d.hidden, F = d.ffn, E = c->esz;

  // ---- weights: one allocation, fused [q|k|v] and [gate|up] projections ----
  Carve wc;
  auto plan_w = [&](char* base) {
    wc = Carve();
    wc.take(c->tok_emb, (size_t)d.vocab * Hd * E, base);
    wc.take(c->patch_w, Hd * c->kpad * E, base);
    wc.take(c->proprio_w, Hd * std::max(d.proprio_dim, 1) * E, base);
    wc.take(c->action_emb, (size_t)d.n_action * Hd * E, base);
    wc.take(c->final_norm, Hd * E, base);
    wc.take(c->head_full, (size_t)d.vocab * Hd * E, base);
    if (base) c->head_w = static_cast<char*>(c->head_full) + (size_t)(d.vocab - d.n_bins) * Hd * E;
    c->attn_norm.resize(L); c->ffn_norm.resize(L); c->wqkv.resize(L); c->wo.resize(L); c->wgu.resize(L); c->wd.resize(L);
    for (size_t l = 0; l < L; ++l) {
      wc.take(c->attn_norm[l], Hd * E, base);
      wc.take(c->wqkv[l], 3 * Hd * Hd * E, base);
      wc.take(c->wo[l], Hd * Hd * E, base);
      wc.take(c->ffn_norm[l], Hd * E, base);
      wc.take(c->wgu[l], 2 * F * Hd * E, base);
      wc.take(c->wd[l], Hd * F * E, base);
    }
    const size_t half = d.head_dim / 2;
    wc.take(c->rope_cos, (size_t)c->Tc * half * 4, base);
    wc.take(c->rope_sin, (size_t)c->Tc * half * 4, base);
  };
  plan_w(nullptr);
  if (dev_alloc(reinterpret_cast<void**>(&c->wmem), wc.off, false) != cudaSuccess) {
    (void)cudaGetLastError();
    delete c;
    return VLAC_ERR_OOM;
  }
  plan_w(c->wmem);
  auto fail = [&](int code) {
    vlac_destroy(c);
    return code;
  };
  auto cp = [&](void* dst, const void* src, size_t bytes) {
    return cudaMemcpy(dst, src, bytes, cudaMemcpyDeviceToDevice) == cudaSuccess;
  };
  bool ok = cp(c->tok_emb, w->tok_emb, (size_t)d.vocab * Hd * E);
  ok = ok && cudaMemset(c->patch_w, 0, Hd * c->kpad * E) == cudaSuccess;
  ok = ok && cudaMemcpy2D(c->patch_w, c->kpad * E, w->patch_w, c->pdim * E, c->pdim * E, Hd,
                          cudaMemcpyDeviceToDevice) == cudaSuccess;
  if (d.proprio_dim) ok = ok && cp(c->proprio_w, w->proprio_w, Hd * d.proprio_dim * E);
  if (d.parallel) ok = ok && cp(c->action_emb, w->action_emb, (size_t)d.n_action * Hd * E);
  ok = ok && cp(c->final_norm, w->final_norm, Hd * E);
  ok = ok && cp(c->head_full, w->lm_head, (size_t)d.vocab * Hd * E);
  for (size_t l = 0; l < L && ok; ++l) {
    char* qkv = static_cast<char*>(c->wqkv[l]);
    char* gu = static_cast<char*>(c->wgu[l]);
    ok = cp(c->attn_norm[l], w->attn_norm[l], Hd * E) && cp(qkv, w->wq[l], Hd * Hd * E) &&
         cp(qkv + Hd * Hd * E, w->wk[l], Hd * Hd * E) && cp(qkv + 2 * Hd * Hd * E, w->wv[l], Hd * Hd * E) &&
         cp(c->wo[l], w->wo[l], Hd * Hd * E) && cp(c->ffn_norm[l], w->ffn_norm[l], Hd * E) &&
         cp(gu, w->w_gate[l], F * Hd * E) && cp(gu + F * Hd * E, w->w_up[l], F * Hd * E) &&
         cp(c->wd[l], w->w_down[l], Hd * F * E);
  }
  if (!ok) return fail(VLAC_ERR_CUDA);
  {  // decode-streaming copies: pair-grouped, K-chunked tiles (one bulk copy per pipeline stage)
    const size_t e_qkv = tiled_decode_elems(Hd, 3 * Hd / 2), e_o = tiled_decode_elems(Hd, Hd / 2);
    const size_t e_gu = tiled_decode_elems(Hd, F), e_d = tiled_decode_elems(F, Hd / 2);
    Carve dc;
    auto plan_d = [&](char* base) {
      dc = Carve();
      c->dqkv.resize(L); c->dwo.resize(L); c->dgu.resize(L); c->dwd.resize(L);
      for (size_t l = 0; l < L; ++l) {
        dc.take(c->dqkv[l], e_qkv * E, base);
        dc.take(c->dwo[l], e_o * E, base);
        dc.take(c->dgu[l], e_gu * E, base);
        dc.take(c->dwd[l], e_d * E, base);
      }
    };
    plan_d(nullptr);
    if (dev_alloc(reinterpret_cast<void**>(&c->dmem), dc.off, false) != cudaSuccess) {
      (void)cudaGetLastError();
      return fail(VLAC_ERR_OOM);
    }
    plan_d(c->dmem);
    for (size_t l = 0; l < L; ++l) {
      if (c->bf16) {
        launch_tile_decode_weights<bf16>((const bf16*)c->wqkv[l], Hd, 3 * Hd / 2, kEpiQkvRope, d.n_heads, d.head_dim, F,
                                         (bf16*)c->dqkv[l], 0);
        launch_tile_decode_weights<bf16>((const bf16*)c->wo[l], Hd, Hd / 2, kEpiResid, d.n_heads, d.head_dim, F,
                                         (bf16*)c->dwo[l], 0);
        launch_tile_decode_weights<bf16>((const bf16*)c->wgu[l], Hd, F, kEpiSwiglu, d.n_heads, d.head_dim, F,
                                         (bf16*)c->dgu[l], 0);
        launch_tile_decode_weights<bf16>((const bf16*)c->wd[l], F, Hd / 2, kEpiResid, d.n_heads, d.head_dim, F,
                                         (bf16*)c->dwd[l], 0);
      } else {
        launch_tile_decode_weights<float>((const float*)c->wqkv[l], Hd, 3 * Hd / 2, kEpiQkvRope, d.n_heads,
                                          d.head_dim, F, (float*)c->dqkv[l], 0);
        launch_tile_decode_weights<float>((const float*)c->wo[l], Hd, Hd / 2, kEpiResid, d.n_heads, d.head_dim, F,
                                          (float*)c->dwo[l], 0);
        launch_tile_decode_weights<float>((const float*)c->wgu[l], Hd, F, kEpiSwiglu, d.n_heads, d.head_dim, F,
                                          (float*)c->dgu[l], 0);
        launch_tile_decode_weights<float>((const float*)c->wd[l], F, Hd / 2, kEpiResid, d.n_heads, d.head_dim, F,
                                          (float*)c->dwd[l], 0);
      }
    }
    if (cudaGetLastError() != cudaSuccess || cudaDeviceSynchronize() != cudaSuccess) return fail(VLAC_ERR_CUDA);
  }
  {  // RoPE tables: angle pos * theta^(-2i/head_dim) in fp64, stored fp32
    const int half = d.head_dim / 2;
    std::vector<float> cs((size_t)c->Tc * half), sn((size_t)c->Tc * half);
    for (int p = 0; p < c->Tc; ++p)
      for (int i = 0; i < half; ++i) {
        const double a = (double)p * std::pow((double)d.rope_theta, -2.0 * i / d.head_dim);
        cs[(size_t)p * half + i] = (float)std::cos(a);
        sn[(size_t)p * half + i] = (float)std::sin(a);
      }
    if (cudaMemcpy(c->rope_cos, cs.data(), cs.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess ||
        cudaMemcpy(c->rope_sin, sn.data(), sn.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess)
      return fail(VLAC_ERR_CUDA);
  }

  // ---- split-K of the prefix GEMMs: balance CTA waves (one CTA per SM)
  // against the fp32 partial traffic of every extra split ----
  if (c->bf16) {
    // Every CTA re-reads the whole activation tile from L2, so extra splits of
    // the wide projections cost more than their better wave fill gains; only
    // the narrow ones (fewer tiles than half the SMs) are split.
    auto pick = [&](int N, int K) {
      const int tiles = N / 128, kch = K / 64;
      if (2 * tiles > c->n_sm) return 1;
      const int sp = std::max(1, std::min({8, kch, c->n_sm / tiles}));
      const int cps = (kch + sp - 1) / sp;  // chunks per split; every split must get some
      return (kch + cps - 1) / cps;
    };
    c->split_qkv = pick(3 * (int)Hd, (int)Hd);
    c->split_o = pick((int)Hd, (int)Hd);
    c->split_gu = pick(2 * (int)F, (int)Hd);
    c->split_d = pick((int)Hd, (int)F);
    if (const char* e = std::getenv("VLAC_SPLITS")) {  // "qkv,o,gu,down" override for sweeps
      int a[4];
      if (std::sscanf(e, "%d,%d,%d,%d", &a[0], &a[1], &a[2], &a[3]) == 4) {
        c->split_qkv = a[0];
        c->split_o = a[1];
        c->split_gu = a[2];
        c->split_d = a[3];
      }
    }
  }

  // ---- tail tiles: a projection with more weight tiles than one wave of
  // CTAs (one per SM) runs whole tiles for every full wave and cuts each
  // remaining tile's K range over the SMs the last wave would leave idle;
  // only those tiles have more than one partial ----
  {
    int plan_sms = c->n_sm;
    if (const char* e = std::getenv("VLAC_PLAN_SMS")) plan_sms = std::max(1, std::atoi(e));  // tests and sweeps
    bool tail_on = c->bf16;
    if (const char* e = std::getenv("VLAC_GEMM_TAIL")) tail_on = tail_on && std::atoi(e) != 0;
    const size_t rcap = c->rows_cap;
    auto plan = [&](int N, int K, int split) {
      const int tiles = N / 128, kch = K / 64;
      if (tail_on && tiles > plan_sms) {
        const int full = (tiles / plan_sms) * plan_sms, rem = tiles - full;
        int tail = rem ? std::min({8, kch, plan_sms / rem}) : 1;
        if (tail >= 2) {
          const int cps = (kch + tail - 1) / tail;
          tail = (kch + cps - 1) / cps;  // every split gets some K
          const int ld = rem * 128;
          c->part_tail_elems = std::max(c->part_tail_elems, (size_t)(tail - 1) * rcap * ld);
          return SplitPlan{full * 128, tail, rcap * (size_t)N, nullptr, rcap * (size_t)ld, ld};
        }
      }
      return uniform_splits(split, rcap * (size_t)N);
    };
    c->sp_qkv = plan(3 * (int)Hd, (int)Hd, c->split_qkv);
    c->sp_o = plan((int)Hd, (int)Hd, c->split_o);
    c->sp_gu = plan(2 * (int)F, (int)Hd, c->split_gu);
    c->sp_d = plan((int)Hd, (int)F, c->split_d);
  }

  // ---- workspace ----
  const size_t rc_ = c->rows_cap, Bm = d.max_batch;
  // every GEMM writes splits x rows_cap x N fp32 partials into `part`
  const size_t part_n = std::max({(size_t)c->split_qkv * 3 * Hd, (size_t)c->split_o * Hd, (size_t)c->split_gu * 2 * F,
                                  (size_t)c->split_d * Hd, Hd});
  c->part_elems = rc_ * part_n;
  Carve sc;
  auto plan_s = [&](char* base) {
    sc = Carve();
    sc.take(c->X, rc_ * Hd * 4, base);
    sc.take(c->Xd, Bm * Hd * 4, base);
    sc.take(c->part, rc_ * part_n * 4, base);
    sc.take(c->part_tail, std::max(c->part_tail_elems, (size_t)4) * 4, base);
    sc.take(c->A, rc_ * Hd * E, base);
    sc.take(c->Q, rc_ * Hd * E, base);
    sc.take(c->AO, rc_ * Hd * E, base);
    sc.take(c->G, rc_ * F * E, base);
    sc.take(c->col, rc_ * c->kpad * E, base);
    sc.take(c->prm, sizeof(StepParams), base);
    sc.take(c->stats, Bm * c->Nv * sizeof(int3), base);
    sc.take(c->mask, Bm * c->Nv, base);
    sc.take(c->full, Bm, base);
    sc.take(c->idx, Bm * c->S * 4, base);
    sc.take(c->M, Bm * L * 4, base);
    sc.take(c->off, L * (Bm + 1) * 4, base);
    sc.take(c->emit_slot, Bm * 4, base);
    sc.take(c->off_dec, (Bm + 1) * 4, base);
    sc.take(c->idx_dec, Bm * 4, base);
    sc.take(c->err, 4, base);
    sc.take(c->logits_ws, Bm * (d.parallel ? d.n_action : 1) * d.n_bins * 4, base);
    sc.take(c->attn_part, Bm * d.n_heads * ((c->Tc + 31) / 32) * (d.head_dim + 2) * 4, base);
    sc.take(c->attn_cnt, Bm * d.n_heads * sizeof(unsigned), base);
    sc.take(c->ssq_a, Bm * std::max((size_t)c->n_sm, Hd / kDecodeRowsPerCta) * 4, base);
    sc.take(c->ssq_b, Bm * std::max((size_t)c->n_sm, Hd / kDecodeRowsPerCta) * 4, base);
    sc.take(c->dp_ptrs, 6 * L * sizeof(void*), base);
    sc.take(c->dp_bar, sizeof(unsigned), base);
    const size_t fbytes = (size_t)d.n_views * d.img_h * d.img_w * 3;
    sc.take(c->in_frames, Bm * fbytes, base);
    sc.take(c->in_prompt, Bm * d.n_text * 4, base);
    sc.take(c->in_proprio, Bm * std::max(d.proprio_dim, 1) * 4, base);
    sc.take(c->in_override, Bm, base);
    sc.take(c->in_forced, Bm * d.n_action * 4, base);
    sc.take(c->in_active, Bm, base);
    sc.take(c->in_s2_forced, Bm * c->Nv, base);
    sc.take(c->in_s3_forced, Bm * L * 2, base);
    sc.take(c->sched_own, Bm * L * 2, base);
    sc.take(c->sched_use, Bm * L * 2, base);
    sc.take(c->o_lent, Bm * L * 4, base);
    sc.take(c->ent_part, L * Bm * d.n_heads * std::max(c->n_textrows, 1) * 4, base);
    sc.take(c->o_ids, Bm * d.n_action * 4, base);
    sc.take(c->o_margins, Bm * d.n_action * 4, base);
    sc.take(c->o_gaps, Bm * d.n_action * 4, base);
    sc.take(c->o_step_margin, Bm * 4, base);
    sc.take(c->o_logits, Bm * d.n_action * d.n_bins * 4, base);
    sc.take(c->o_recomputed, Bm, base);
    sc.take(c->o_gate_auto, Bm, base);
    sc.take(c->o_mask, Bm * c->Nv, base);
    sc.take(c->o_idx, Bm * c->S * 4, base);
    sc.take(c->o_M, Bm * L * 4, base);
    sc.take(c->o_rel, Bm * c->Nv * 4, base);
    sc.take(c->o_relevant, Bm * c->Nv, base);
    sc.take(c->rel_part, Bm * d.n_heads * c->Nv * 4, base);
    sc.take(c->o_entropy, Bm * d.n_action * 4, base);
    sc.take(c->o_vm, Bm * d.n_action * 4, base);
    sc.take(c->o_delta, Bm * 4, base);
    const size_t head_rows = Bm * (d.parallel ? d.n_action : 1);
    sc.take(c->vh_rows, head_rows * Hd * E, base);
    sc.take(c->vh_logits, head_rows * std::max(d.vocab - d.n_bins, 1) * 4, base);
  };
  plan_s(nullptr);
  if (dev_alloc(reinterpret_cast<void**>(&c->wsmem), sc.off, false) != cudaSuccess) {
    (void)cudaGetLastError();
    return fail(VLAC_ERR_OOM);
  }
  plan_s(c->wsmem);
  if (cudaMemset(c->wsmem, 0, sc.off) != cudaSuccess) return fail(VLAC_ERR_CUDA);
  {
    std::vector<int> od(Bm + 1);
    for (size_t b = 0; b <= Bm; ++b) od[b] = (int)b;
    if (cudaMemcpy(c->off_dec, od.data(), od.size() * 4, cudaMemcpyHostToDevice) != cudaSuccess)
      return fail(VLAC_ERR_CUDA);
  }
  if (c->bf16 && !c->dqkv.empty()) {  // per-layer pointers of the persistent decode pass
    std::vector<void*> pp(6 * L);
    for (size_t l = 0; l < L; ++l) {
      pp[l] = c->dqkv[l];
      pp[L + l] = c->dwo[l];
      pp[2 * L + l] = c->dgu[l];
      pp[3 * L + l] = c->dwd[l];
      pp[4 * L + l] = c->attn_norm[l];
      pp[5 * L + l] = c->ffn_norm[l];
    }
    if (cudaMemcpy(c->dp_ptrs, pp.data(), pp.size() * sizeof(void*), cudaMemcpyHostToDevice) != cudaSuccess)
      return fail(VLAC_ERR_CUDA);
  }
  if (dev_alloc(reinterpret_cast<void**>(&c->err_host), sizeof(int), true) != cudaSuccess) {
    (void)cudaGetLastError();
    c->err_host = nullptr;
    return fail(VLAC_ERR_OOM);
  }
  *c->err_host = 0;
  if (cudaStreamCreateWithFlags(&c->cap_stream, cudaStreamNonBlocking) != cudaSuccess) return fail(VLAC_ERR_CUDA);

  // ---- TMA descriptors ----
  if (c->bf16) {
    c->tm_qkv.resize(L); c->tm_o.resize(L); c->tm_gu.resize(L); c->tm_d.resize(L);
    auto act = [&](ActMaps* am, const void* base, size_t cols) {
      bool r = true;
      for (int i = 0; i < 4; ++i) r = r && make_map(&am->m[i], base, rc_, cols, 32u << i);
      return r;
    };
    bool mok = make_map(&c->tm_patch, c->patch_w, Hd, c->kpad, 128) && act(&c->tm_A, c->A, Hd) &&
               act(&c->tm_AO, c->AO, Hd) && act(&c->tm_G, c->G, F) && act(&c->tm_col, c->col, c->kpad);
    for (size_t l = 0; l < L && mok; ++l)
      mok = make_map(&c->tm_qkv[l], c->wqkv[l], 3 * Hd, Hd, 128) && make_map(&c->tm_o[l], c->wo[l], Hd, Hd, 128) &&
            make_map(&c->tm_gu[l], c->wgu[l], 2 * F, Hd, 128) && make_map(&c->tm_d[l], c->wd[l], Hd, F, 128);
    if (!mok) return fail(VLAC_ERR_CUDA);
  }
  if (cudaDeviceSynchronize() != cudaSuccess) return fail(VLAC_ERR_CUDA);
  *out = c;
  return VLAC_OK;
}

// ---- caches -----------------------------------------------------------------------

static size_t cache_layout(const vlac_ctx* c, int B, char* base, vlac_cache* k) {
  const vlac_dims& d = c->d;
  Carve cv;
  void* K;
  void* V;
  float* H;
  uint8_t *prev, *valid, *rel_valid, *ids_valid, *ent_valid;
  float *m_prev, *rel, *ent;
  int32_t* prev_ids;
  const size_t kv = (size_t)d.n_layers * d.n_heads * c->Tc * d.head_dim;
  const size_t hs = (size_t)d.n_layers * c->S * d.hidden;
  cv.take(K, B * kv * c->esz, base);
  cv.take(V, B * kv * c->esz, base);
  cv.take(H, B * hs * 4, base);
  cv.take(prev, (size_t)B * d.n_views * d.img_h * d.img_w * 3, base);
  cv.take(m_prev, (size_t)B * 4, base);
  cv.take(valid, (size_t)B, base);
  cv.take(rel, (size_t)B * c->Nv * 4, base);
  cv.take(rel_valid, (size_t)B, base);
  cv.take(prev_ids, (size_t)B * d.n_action * 4, base);
  cv.take(ids_valid, (size_t)B, base);
  cv.take(ent, (size_t)B * d.n_layers * 4, base);
  cv.take(ent_valid, (size_t)B, base);
  if (k) {
    k->ent = ent; k->ent_valid = ent_valid;
    k->K = K; k->V = V; k->H = H; k->prev = prev; k->m_prev = m_prev; k->valid = valid;
    k->rel = rel; k->rel_valid = rel_valid;
    k->prev_ids = prev_ids; k->ids_valid = ids_valid;
    k->kv_seq_stride = kv;
    k->h_seq_stride = hs;
  }
  return align_up(cv.off, 256);
}

extern "C" int vlac_cache_bytes(const vlac_ctx* c, int batch, size_t* bytes) {
  if (!c || !bytes || batch < 1 || batch > c->d.max_batch) return VLAC_ERR_INVALID_ARG;
  *bytes = cache_layout(c, batch, nullptr, nullptr);
  return VLAC_OK;
}

extern "C" int vlac_cache_init(vlac_ctx* c, void* mem, size_t bytes, int batch, vlac_cache** out) {
  if (!c || !mem || !out || batch < 1 || batch > c->d.max_batch) return VLAC_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(mem) % 256) return VLAC_ERR_INVALID_ARG;
  const size_t need = cache_layout(c, batch, nullptr, nullptr);
  if (bytes < need) return VLAC_ERR_INVALID_ARG;
  vlac_cache* k = new (std::nothrow) vlac_cache();
  if (!k) return VLAC_ERR_OOM;
  k->ctx = c;
  k->B = batch;
  cache_layout(c, batch, static_cast<char*>(mem), k);
  if (c->bf16) {
    // the prefix attention's K/V tiles: rows of head_dim, Tc positions per (sequence, layer, head)
    const uint64_t planes = (uint64_t)batch * c->d.n_layers * c->d.n_heads;
    if (!make_map3(&k->kvm.k, k->K, planes, c->Tc, c->d.head_dim, 64) ||
        !make_map3(&k->kvm.v, k->V, planes, c->Tc, c->d.head_dim, 64)) {
      delete k;
      return VLAC_ERR_CUDA;
    }
  }
  if (cudaMemset(mem, 0, need) != cudaSuccess || cudaDeviceSynchronize() != cudaSuccess) {
    (void)cudaGetLastError();
    delete k;
    return VLAC_ERR_CUDA;
  }
  *out = k;
  return VLAC_OK;
}

extern "C" int vlac_cache_destroy(vlac_cache* k) {
  if (!k) return VLAC_ERR_INVALID_ARG;
  if (k->gexec) cudaGraphExecDestroy(k->gexec);
  if (k->graph) cudaGraphDestroy(k->graph);
  delete k;
  return VLAC_OK;
}

extern "C" int vlac_reset(vlac_cache* k, int seq, void* stream) {
  if (!k || seq < -1 || seq >= k->B) return VLAC_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (seq < 0) {
    CK(cudaMemsetAsync(k->valid, 0, (size_t)k->B, st));
    CK(cudaMemsetAsync(k->rel_valid, 0, (size_t)k->B, st));
    CK(cudaMemsetAsync(k->ids_valid, 0, (size_t)k->B, st));
    CK(cudaMemsetAsync(k->ent_valid, 0, (size_t)k->B, st));
  } else {
    CK(cudaMemsetAsync(k->valid + seq, 0, 1, st));
    CK(cudaMemsetAsync(k->rel_valid + seq, 0, 1, st));
    CK(cudaMemsetAsync(k->ids_valid + seq, 0, 1, st));
    CK(cudaMemsetAsync(k->ent_valid + seq, 0, 1, st));
  }
  return VLAC_OK;
}

// ---- the step ------------------------------------------------------------------

namespace {

cudaEvent_t prof_event(vlac_ctx* c) {
  if (!c->ev_pool.empty()) {
    cudaEvent_t e = c->ev_pool.back();
    c->ev_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

// Records events around one launch of a profiled kernel kind.
struct ProfScope {
  vlac_ctx* c;
  cudaStream_t st;
  vlac_ctx::ProfRec rec;
  ProfScope(vlac_ctx* c_, int kind, double bytes, cudaStream_t s) : c(c_), st(s) {
    if (!c->prof_on) return;
    rec.kind = kind;
    rec.bytes = bytes;
    rec.a = prof_event(c);
    rec.b = prof_event(c);
    cudaEventRecord(rec.a, st);
  }
  ~ProfScope() {
    if (!c->prof_on) return;
    cudaEventRecord(rec.b, st);
    c->prof.push_back(rec);
  }
};

template <typename T>
void dgemv(vlac_ctx* c, const DGemv& a_in, int epi, int nb, cudaStream_t st) {
  DGemv a = a_in;
  a.ns = c->gemv_ns;
  a.wait_limit = c->wait_limit;
  // the stage ring must fit next to the input vector in shared memory
  const size_t xs = ((size_t)nb * a.K * sizeof(T) + 1023) / 1024 * 1024;
  while (a.ns > 2 && (size_t)a.ns * dgemv_stage_bytes() + (xs > 64 * 1024 ? 0 : xs) > 200 * 1024) --a.ns;
  ProfScope ps(c, VLAC_PROF_DECODE_GEMV,
               (double)2 * a.n_pairs * a.K * sizeof(T) + (double)nb * a.K * sizeof(T) + (double)nb * 2 * a.n_pairs * 4,
               st);
  launch_dgemv<T>(a, epi, nb, c->n_sm, st);
  c->launches += 1;
}

template <typename T>
void gemm(vlac_ctx* c, const ActMaps* tmA, const CUtensorMap* tmW, const T* A, const void* W, const int* m_ptr,
          int N, int K, const SplitPlan& sp, cudaStream_t st) {
  const int kch = c->bf16 ? K / 64 : 1, cps = (kch + sp.tail - 1) / sp.tail;
  const bool compact = sp.tail_ld != 0;
  const size_t slots = compact ? 1 : (size_t)sp.tail;
  if (slots * c->rows_cap * N > c->part_elems ||  // never launch a GEMM whose partials do not fit,
      (compact && (size_t)(sp.tail - 1) * c->rows_cap * sp.tail_ld > c->part_tail_elems) ||
      (sp.tail - 1) * cps >= kch || (!c->bf16 && (sp.tail != 1 || sp.full_cols))) {  // or a split without K
    c->fatal = true;
    return;
  }
  ProfScope ps(c, VLAC_PROF_PREFIX_GEMM, (double)N * K * sizeof(T), st);
  if constexpr (sizeof(T) == 2) {
    launch_gemm_tc(tmA, tmW, m_ptr, c->rows_cap, N, K, sp, c->part, c->err, c->wait_limit, st);
  } else {
    launch_gemm_simt<T>(A, static_cast<const T*>(W), m_ptr, c->rows_cap, N, K, c->part, st);
  }
  c->launches += 1;
}

// One decoder layer of the prefix pass for the rows `rl` of B sequences:
// the input norm (rows joining at this layer start from H, rows computed at
// the previous layer record their input there; H NULL at layer 0), q/k/v
// with RoPE and the K/V scatter into Kc_l / Vc_l (this layer of the cache),
// the mixed-cache attention, o-projection + residual, the MLP norm, gate/up +
// SwiGLU and down + residual.  The bf16 attention reads the K/V tiles through
// the cache's maps kvm; seq0 is the batch's first sequence in the cache.
// do_in: this layer's input norm runs here (else the previous layer's last
// launch ran it); rl_next / H_next: the next layer's rows and H slice, whose
// input norm then runs fused with this layer's down residual.
template <typename T>
void prefix_layer(vlac_ctx* c, const Rows& rl, const int* off_prev, int B, int l, float* H, size_t h_seq_stride,
                  T* Kc_l, T* Vc_l, size_t kv_seq_stride, const KvMaps* kvm, int seq0, cudaStream_t st,
                  bool do_in = true, const Rows* rl_next = nullptr, float* H_next = nullptr) {
  const vlac_dims& d = c->d;
  const int S = c->S, Hd = d.hidden, F = d.ffn, nh = d.n_heads, hd = d.head_dim;
  const float eps = d.rms_eps;
  T* A = static_cast<T*>(c->A);
  T* Q = static_cast<T*>(c->Q);
  T* AO = static_cast<T*>(c->AO);
  T* G = static_cast<T*>(c->G);
  auto W = [](void* p) { return static_cast<const T*>(p); };
  auto with_tail = [&](SplitPlan p) {
    p.tail_p = c->part_tail;
    return p;
  };
  const SplitPlan sq = with_tail(c->sp_qkv), so = with_tail(c->sp_o), sg = with_tail(c->sp_gu), sd = with_tail(c->sp_d);
  const int* ml = rl.off + B;
  if (do_in) {
    ProfScope ps_(c, VLAC_PROF_ROWS, 0, st);
    launch_layer_in<T>(rl, off_prev, B, S, Hd, H, h_seq_stride, W(c->attn_norm[l]), eps, A, st);
  }
  gemm<T>(c, &c->tm_A, c->bf16 ? &c->tm_qkv[l] : nullptr, A, c->wqkv[l], ml, 3 * Hd, Hd, sq, st);
  {
    ProfScope ps_(c, VLAC_PROF_ROWS, 0, st);
    launch_qkv_epilogue<T>(rl, B, S, nh, hd, c->part, sq, c->rope_cos, c->rope_sin, Q, Kc_l, Vc_l, kv_seq_stride,
                           c->Tc, st);
  }
  {
    ProfScope ps_(c, VLAC_PROF_PREFIX_ATTN, 0, st);
    launch_attention<T>(rl, B, S, nh, hd, Q, Kc_l, Vc_l, kv_seq_stride, c->Tc, c->P, d.parallel, d.n_action, AO, kvm,
                        d.n_layers * nh, (seq0 * d.n_layers + l) * nh, c->err, c->wait_limit, st);
  }
  gemm<T>(c, &c->tm_AO, c->bf16 ? &c->tm_o[l] : nullptr, AO, c->wo[l], ml, Hd, Hd, so, st);
  {
    ProfScope ps_(c, VLAC_PROF_ROWS, 0, st);
    launch_residual_norm<T>(rl, B, S, Hd, c->part, so, W(c->ffn_norm[l]), eps, A, st);
  }
  gemm<T>(c, &c->tm_A, c->bf16 ? &c->tm_gu[l] : nullptr, A, c->wgu[l], ml, 2 * F, Hd, sg, st);
  {
    ProfScope ps_(c, VLAC_PROF_ROWS, 0, st);
    launch_swiglu<T>(rl, B, S, F, c->part, sg, G, st);
  }
  gemm<T>(c, &c->tm_G, c->bf16 ? &c->tm_d[l] : nullptr, G, c->wd[l], ml, Hd, F, sd, st);
  {
    ProfScope ps_(c, VLAC_PROF_ROWS, 0, st);
    if (rl_next)
      launch_residual_layer_in<T>(*rl_next, rl.off, B, S, Hd, c->part, sd, H_next, h_seq_stride,
                                  W(c->attn_norm[l + 1]), eps, A, st);
    else
      launch_residual(rl, B, S, Hd, c->part, sd, st);
  }
  c->launches += do_in ? 6 : 5;
}

// The step body: reads only the staged inputs and writes only the context's
// output buffers, so its launches can be captured once and replayed.
template <typename T>
int step_impl(vlac_ctx* c, vlac_cache* k, cudaStream_t st) {
  vlac_step_out outv{c->o_ids,   c->o_margins, c->o_gaps, c->o_recomputed, c->o_step_margin, c->o_gate_auto,
                     c->o_logits, c->o_mask,    c->o_idx,  c->o_M,         c->o_rel,         c->o_relevant,
                     c->o_entropy, c->o_vm,    c->o_delta};
  VocabHead vh{c->head_full, c->d.vocab - c->d.n_bins, c->vh_rows, c->vh_logits, c->o_vm};
  const VocabHead* vhp = c->vm_on ? &vh : nullptr;
  const int head_launches = c->vm_on ? (vh.n_rows ? 4 : 3) : 1;
  const vlac_step_out* out = &outv;
  const uint8_t* frames = c->in_frames;
  const int32_t* prompt = c->in_prompt;
  const float* proprio = c->in_proprio;
  const vlac_dims& d = c->d;
  const int B = k->B, S = c->S, L = d.n_layers, Hd = d.hidden, F = d.ffn, D = d.n_action, nb = d.n_bins;
  const int nh = d.n_heads, hd = d.head_dim;
  const float eps = d.rms_eps;
  T* A = static_cast<T*>(c->A);
  T* Q = static_cast<T*>(c->Q);
  T* AO = static_cast<T*>(c->AO);
  T* G = static_cast<T*>(c->G);
  T* col = static_cast<T*>(c->col);
  T* Kc = static_cast<T*>(k->K);
  T* Vc = static_cast<T*>(k->V);
  const size_t kv_layer = (size_t)nh * c->Tc * hd;
  const int8_t* ovr = c->in_override;
  const int32_t* forced = c->in_forced;
  auto W = [](void* p) { return static_cast<const T*>(p); };

  // Stage 1 and the gate + Stage-3 plan
  {
    ProfScope ps_(c, VLAC_PROF_OTHER, 0, st);
    launch_patch_stats(frames, k->prev, k->valid, c->prm, B, d.n_views, d.img_h, d.img_w, d.patch, c->stats, c->mask,
                       out->static_mask, st);
  }
  {
    // Stage 3's per-sequence schedule (the caller's unless adaptive)
    ProfScope ps_(c, VLAC_PROF_OTHER, 0, st);
    launch_schedule(c->prm, k->ent, k->ent_valid, c->in_s3_forced, c->in_active, B, L, c->sched_own, c->sched_use,
                    c->o_lent, st);
  }
  {
    ProfScope ps_(c, VLAC_PROF_OTHER, 0, st);
    launch_select(c->stats, c->mask, k->valid, k->m_prev, c->prm, ovr, B, c->Nv, S, L, c->P, d.parallel, D, c->full,
                  c->idx, c->M, c->off, c->emit_slot, out->recomputed, out->gate_auto, out->idx, out->M,
                  c->in_active, k->rel, k->rel_valid, c->in_s2_forced, out->relevant, out->relevance, c->sched_use,
                  st);
  }
  c->launches += 4;

  // layer-0 inputs of the recomputed rows
  Rows r0{c->off, c->idx, S, c->X};
  const int* m0 = c->off + B;
  {
    ProfScope ps_(c, VLAC_PROF_ROWS, 0, st);
    launch_im2col<T>(r0, B, S, frames, d.n_views, d.img_h, d.img_w, d.patch, c->kpad, col, st);
  }
  gemm<T>(c, &c->tm_col, &c->tm_patch, col, c->patch_w, m0, Hd, c->kpad, uniform_splits(1, c->rows_cap * Hd), st);
  {
    ProfScope ps_(c, VLAC_PROF_ROWS, 0, st);
    launch_embed<T>(r0, B, S, Hd, c->Nv, c->P, c->has_p, d.proprio_dim, d.n_text, d.vocab, prompt, proprio,
                    W(c->tok_emb), c->part, W(c->proprio_w), W(c->action_emb), c->err, st);
  }
  c->launches += 2;

  for (int l = 0; l < L; ++l) {
    Rows rl{c->off + (size_t)l * (B + 1), c->idx, S, c->X};
    const int* off_prev = l == 0 ? rl.off : c->off + (size_t)(l - 1) * (B + 1);
    // the next layer's input norm runs with this layer's down residual
    const Rows rl_next{c->off + (size_t)(l + 1) * (B + 1), c->idx, S, c->X};
    const bool fuse_next = c->fuse_rows && l + 1 < L;
    prefix_layer<T>(c, rl, off_prev, B, l, l == 0 ? nullptr : k->H + (size_t)l * S * Hd, k->h_seq_stride,
                    Kc + l * kv_layer, Vc + l * kv_layer, k->kv_seq_stride, &k->kvm, 0, st,
                    l == 0 || !c->fuse_rows, fuse_next ? &rl_next : nullptr,
                    fuse_next ? k->H + (size_t)(l + 1) * S * Hd : nullptr);
    if (c->s2_on && l == c->s2_layer) {
      // Stage 2: the text rows' attention on the visual keys of this layer (Q
      // still holds this layer's rows)
      ProfScope ps_(c, VLAC_PROF_PREFIX_ATTN, 0, st);
      if (launch_relevance<T>(rl, B, nh, hd, Q, Kc + l * kv_layer, k->kv_seq_stride, c->Tc, c->Nv,
                              1 + c->Nv + c->has_p, c->P, c->rel_part, k->rel, out->relevance, k->rel_valid,
                              c->prm, c->in_active, st))
        c->fatal = true;
      c->launches += 2;
    }
    if (c->s3_on) {
      // Stage 3 adaptive: this layer's attention entropy of the text rows
      ProfScope ps_(c, VLAC_PROF_PREFIX_ATTN, 0, st);
      if (launch_layer_entropy<T>(rl, B, nh, hd, Q, Kc + l * kv_layer, k->kv_seq_stride, c->Tc, c->text_lo, c->P,
                                  c->ent_part + (size_t)l * B * nh * c->n_textrows, st))
        c->fatal = true;
      c->launches += 1;
    }
  }
  if (c->s3_on) {
    ProfScope ps_(c, VLAC_PROF_OTHER, 0, st);
    launch_entropy_finish(c->ent_part, L, B, nh, c->n_textrows, k->ent, k->ent_valid, c->o_lent, c->prm,
                          c->in_active, st);
    c->launches += 1;
  }
  // action head on the prefix pass: the last text row, or the parallel action block
  {
    ProfScope ps_(c, VLAC_PROF_HEAD, 0, st);
    launch_head2<T>(c->X, c->emit_slot, (size_t)S * Hd, d.parallel ? D : 1, B, Hd, nb, W(c->final_norm),
                    W(c->head_w), eps, c->logits_ws, D, 0, out->action_ids, out->margins, out->logit_gap, out->logits,
                    out->entropy, vhp, st);
  }
  c->launches += head_launches;

  if (!d.parallel) {
    // autoregressive decode: one row per sequence, fused GEMVs
    for (int a = 1; a < D; ++a) {
      const int pos = c->P + a - 1;
      {
        ProfScope ps_(c, VLAC_PROF_OTHER, 0, st);
        launch_decode_embed<T>(B, a, D, c->P, Hd, d.vocab, nb, W(c->tok_emb), out->action_ids, forced, c->prm, c->Xd,
                               c->idx_dec, c->ssq_b, c->err, st);
      }
      c->launches += 1;
      // optional prefetch chain (VLAC_GEMV_PF_KB, off by default): each GEMV
      // pulls the start of the next one's weights into L2
      auto set_pf = [&](DGemv& g, const void* Wn, int Kn, int pairs) {
        g.pf_W = Wn;
        g.pf_K = Kn;
        g.pf_pairs = pairs;
        g.pf_grid = dgemv_grid(pairs, c->n_sm);
        g.pf_bytes = (uint32_t)c->gemv_pf_kb * 1024;
        if (!g.pf_bytes) g.pf_W = nullptr;
      };
      // all layers as one persistent cooperative launch (VLAC_DPASS=1, bf16,
      // head_dim 128, up to two sequences); else one launch per projection
      bool dp_done = false;
      if constexpr (sizeof(T) == 2) {
        if (c->use_dpass && dpass_supported((int)Hd, (int)F, nh, hd, B, c->gemv_ns)) {
          DPass p{};
          const bf16* const* pp = reinterpret_cast<const bf16* const*>(c->dp_ptrs);
          p.w_qkv = pp;
          p.w_o = pp + L;
          p.w_gu = pp + 2 * L;
          p.w_d = pp + 3 * L;
          p.g_attn = pp + 4 * L;
          p.g_ffn = pp + 5 * L;
          p.L = L;
          p.hidden = (int)Hd;
          p.ffn = (int)F;
          p.n_heads = nh;
          p.Tc = c->Tc;
          p.pos = pos;
          p.ns = c->gemv_ns;
          p.n_ssq0 = (int)Hd / kDecodeRowsPerCta;
          p.eps = eps;
          p.scale = 1.0f / sqrtf((float)hd);
          p.rope_cos = c->rope_cos;
          p.rope_sin = c->rope_sin;
          p.X = c->Xd;
          p.Q = Q;
          p.AO = AO;
          p.G = G;
          p.Kc = Kc;
          p.Vc = Vc;
          p.kv_layer = kv_layer;
          p.kv_seq_stride = k->kv_seq_stride;
          p.ssq0 = c->ssq_b;
          p.ssq = c->ssq_a;
          p.bar = c->dp_bar;
          p.err = c->err;
          p.bar_mode = c->dpass_bar;
          p.wait_limit = c->wait_limit;
          {
            // key ranges per (sequence, head): enough items for the SMs, at
            // most one per 32 keys (the partial buffer's capacity) and 8
            const int cap = std::min(8, (c->Tc + 31) / 32);
            int chunks = std::max(1, std::min(cap, c->n_sm / std::max(1, B * nh)));
            if (c->dpass_attn_chunks > 0) chunks = std::min(cap, c->dpass_attn_chunks);
            p.attn_chunks = chunks;
            // the first item's K/V rows staged in shared memory, as many as
            // fit next to the ring
            p.kv_keys = 0;
            if (c->dpass_kv)
              p.kv_keys = std::min((c->Tc + chunks - 1) / chunks, dpass_kv_fit((int)Hd, (int)F, B, c->gemv_ns));
            p.part_stride = (size_t)((c->Tc + 31) / 32) * (hd + 2);
            p.attn_part = c->attn_part;
            p.attn_cnt = c->attn_cnt;
          }
          int rc_dp;
          {
            ProfScope ps_(c, VLAC_PROF_DECODE_GEMV, (double)L * (4.0 * Hd * Hd + 3.0 * F * Hd) * 2, st);
            rc_dp = launch_dpass(p, B, c->n_sm, st);
          }
          if (rc_dp == VLAC_OK) {
            c->launches += 1;
            dp_done = true;
          } else if (rc_dp == VLAC_ERR_UNSUPPORTED) {
            (void)cudaGetLastError();  // one CTA per SM does not fit: the per-projection chain runs instead
          } else {
            c->fatal = true;
          }
        }
      }
      for (int l = 0; l < L && !dp_done; ++l) {
        DGemv g{};
        g.eps = eps;
        g.n_heads = nh;
        g.head_dim = hd;
        // q, k, v with the attention RMSNorm prologue, RoPE and the K/V scatter
        g.W = c->dqkv[l];
        g.n_pairs = 3 * Hd / 2;
        g.K = Hd;
        g.X = c->Xd;
        g.gain = c->attn_norm[l];
        g.Q = Q;
        g.Kc = Kc + l * kv_layer;
        g.Vc = Vc + l * kv_layer;
        g.kv_seq_stride = k->kv_seq_stride;
        g.Tc = c->Tc;
        g.pos = pos;
        g.rope_cos = c->rope_cos;
        g.rope_sin = c->rope_sin;
        g.ssq_in = c->ssq_b;
        g.n_ssq = l == 0 ? Hd / kDecodeRowsPerCta : dgemv_grid(Hd / 2, c->n_sm);  // embedding or down-projection
        g.err = c->err;
        set_pf(g, c->dwo[l], Hd, Hd / 2);
        dgemv<T>(c, g, kEpiQkvRope, B, st);
        {
          ProfScope ps_(c, VLAC_PROF_DECODE_ATTN, 0, st);
          launch_dec_attention<T>(B, nh, hd, Q, Kc + l * kv_layer, Vc + l * kv_layer, k->kv_seq_stride, c->Tc, pos,
                                  c->attn_part, c->attn_cnt, AO, st);
        }
        c->launches += 1;
        // o-projection + residual
        DGemv o{};
        o.W = c->dwo[l];
        o.n_pairs = Hd / 2;
        o.K = Hd;
        o.xin = AO;
        o.Xres = c->Xd;
        o.n_out = Hd;
        o.ssq_out = c->ssq_a;
        o.err = c->err;
        set_pf(o, c->dgu[l], Hd, F);
        dgemv<T>(c, o, kEpiResid, B, st);
        // gate/up with the MLP RMSNorm prologue and SwiGLU
        DGemv u{};
        u.W = c->dgu[l];
        u.n_pairs = F;
        u.K = Hd;
        u.X = c->Xd;
        u.gain = c->ffn_norm[l];
        u.eps = eps;
        u.G = G;
        u.ffn = F;
        u.ssq_in = c->ssq_a;
        u.n_ssq = dgemv_grid(Hd / 2, c->n_sm);  // o-projection
        u.err = c->err;
        set_pf(u, c->dwd[l], F, Hd / 2);
        dgemv<T>(c, u, kEpiSwiglu, B, st);
        // down-projection + residual
        DGemv dn{};
        dn.W = c->dwd[l];
        dn.n_pairs = Hd / 2;
        dn.K = F;
        dn.xin = G;
        dn.Xres = c->Xd;
        dn.n_out = Hd;
        dn.ssq_out = c->ssq_b;
        dn.err = c->err;
        if (l + 1 < L) set_pf(dn, c->dqkv[l + 1], Hd, 3 * Hd / 2);
        else if (a + 1 < D) set_pf(dn, c->dqkv[0], Hd, 3 * Hd / 2);
        dgemv<T>(c, dn, kEpiResid, B, st);
      }
      {
        ProfScope ps_(c, VLAC_PROF_HEAD, 0, st);
        launch_head2<T>(c->Xd, nullptr, Hd, 1, B, Hd, nb, W(c->final_norm), W(c->head_w), eps, c->logits_ws, D, a,
                        out->action_ids, out->margins, out->logit_gap, out->logits, out->entropy, vhp, st);
      }
      c->launches += head_launches;
    }
  }
  {
    ProfScope ps_(c, VLAC_PROF_OTHER, 0, st);
    launch_finish(B, D, c->prm, out->margins, out->logit_gap, out->vocab_margin, k->m_prev, k->valid, out->step_margin,
                  out->action_ids, k->prev_ids, k->ids_valid, out->action_delta, c->in_active, st);
  }
  {
    ProfScope ps_(c, VLAC_PROF_OTHER, 0, st);
    const StepOutputs so{out->action_ids, out->margins,   out->logit_gap,   out->logits, out->step_margin,
                         out->recomputed, out->gate_auto, out->static_mask, out->idx,    out->M,
                         out->relevance,  out->relevant,  out->entropy,     out->vocab_margin,
                         out->action_delta};
    launch_commit(B, D, nb, c->Nv, S, L, (size_t)d.n_views * d.img_h * d.img_w * 3, frames, k->prev, c->prm,
                  c->in_active, so, st);
  }
  c->launches += 2;
  CK(cudaMemcpyAsync(c->err_host, c->err, sizeof(int), cudaMemcpyDeviceToHost, st));
  CK(cudaGetLastError());
  return VLAC_OK;
}

int run_body(vlac_ctx* c, vlac_cache* k, cudaStream_t st) {
  const int rc = c->bf16 ? step_impl<bf16>(c, k, st) : step_impl<float>(c, k, st);
  return c->fatal ? VLAC_ERR_INVALID_ARG : rc;
}

// First step of a cache runs eagerly (lazy per-kernel set-up happens there);
// the second captures the body into a graph, which every later step replays.
int run_step(vlac_ctx* c, vlac_cache* k, cudaStream_t st) {
  if (!c->use_graph || c->prof_on) return run_body(c, k, st);
  const int sig = ((c->s2_on ? 1 + c->s2_layer : 0) * 2 + (c->vm_on ? 1 : 0)) * 2 + (c->s3_on ? 1 : 0);
  if (k->gexec && k->graph_sig != sig) {
    // Stage 2, Stage 3 adaptive or the whole-vocabulary margin switched on or
    // off, or Stage 2 moved to another layer: the launch list
    // differs, so the graph is captured again (after one eager step)
    cudaGraphExecDestroy(k->gexec);
    cudaGraphDestroy(k->graph);
    k->gexec = nullptr;
    k->graph = nullptr;
    k->eager_steps = 0;
  }
  if (!k->gexec) {
    if (k->eager_steps++ == 0) return run_body(c, k, st);
    const uint64_t n0 = c->launches;
    CK(cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeThreadLocal));
    const int rc = run_body(c, k, c->cap_stream);
    cudaGraph_t g = nullptr;
    const cudaError_t e = cudaStreamEndCapture(c->cap_stream, &g);
    if (rc != VLAC_OK || e != cudaSuccess) {
      if (g) cudaGraphDestroy(g);
      (void)cudaGetLastError();
      return rc != VLAC_OK ? rc : VLAC_ERR_CUDA;
    }
    if (cudaGraphInstantiate(&k->gexec, g, 0) != cudaSuccess) {
      cudaGraphDestroy(g);
      k->gexec = nullptr;
      (void)cudaGetLastError();
      return VLAC_ERR_CUDA;
    }
    k->graph = g;
    k->graph_sig = sig;
    k->graph_launches = c->launches - n0;
    c->launches = n0;
  }
  CK(cudaGraphLaunch(k->gexec, st));
  c->launches += k->graph_launches;
  return VLAC_OK;
}

}  // namespace

extern "C" int vlac_step(vlac_ctx* c, vlac_cache* k, const uint8_t* frames, const int32_t* prompt_ids,
                         const float* proprio, vlac_rational tau_sim, float tau_margin,
                         const uint16_t* reuse_permille, const vlac_step_opts* opts, const vlac_step_out* out,
                         void* stream) {
  if (!c || !k || !frames || !prompt_ids || !reuse_permille || !out || !out->action_ids || !out->margins ||
      !out->logit_gap || !out->recomputed || !out->step_margin || tau_sim.den == 0)
    return VLAC_ERR_INVALID_ARG;
  if (k->ctx != c) return VLAC_ERR_STATE;
  if (c->d.proprio_dim > 0 && !proprio) return VLAC_ERR_INVALID_ARG;
  if (tau_margin != tau_margin) return VLAC_ERR_INVALID_ARG;
  StepParams p;
  std::memset(&p, 0, sizeof(p));
  for (int l = 0; l < c->d.n_layers; ++l) {
    if (reuse_permille[l] > 1000) return VLAC_ERR_INVALID_ARG;
    p.permille[l] = reuse_permille[l];
  }
  int mk = opts ? opts->margin_kind : VLAC_MARGIN_PROB;
  int red = opts ? opts->reduction : VLAC_REDUCE_DEFAULT;
  if (mk != VLAC_MARGIN_PROB && mk != VLAC_MARGIN_LOGIT && mk != VLAC_MARGIN_VOCAB) return VLAC_ERR_INVALID_ARG;
  if (red == VLAC_REDUCE_DEFAULT) red = c->d.parallel ? VLAC_REDUCE_MIN : VLAC_REDUCE_MEAN;
  if (red != VLAC_REDUCE_MEAN && red != VLAC_REDUCE_MIN) return VLAC_ERR_INVALID_ARG;
  p.tau_num = tau_sim.num;
  p.tau_den = tau_sim.den;
  p.tau_margin = tau_margin;
  p.margin_kind = mk;
  p.reduction = red;
  p.has_override = (opts && opts->gate_override) ? 1 : 0;
  p.has_forced = (opts && opts->forced_ids) ? 1 : 0;
  p.has_active = (opts && opts->active) ? 1 : 0;
  const int s2_k = opts ? opts->s2_top_k : 0, s2_l = opts ? opts->s2_layer : 0;
  if (s2_k < 0 || (s2_k > 0 && (s2_l < 0 || s2_l >= c->d.n_layers))) return VLAC_ERR_INVALID_ARG;
  p.s2_top_k = s2_k;
  p.s2_layer = s2_k > 0 ? s2_l : 0;
  p.has_s2_forced = (s2_k > 0 && opts->s2_forced) ? 1 : 0;
  p.s3_adaptive = (opts && opts->s3_adaptive) ? 1 : 0;
  if (p.s3_adaptive) {
    if (opts->s3_lo < 0 || opts->s3_lo > opts->s3_hi || opts->s3_hi > 1000 || opts->s3_weight < 0 ||
        opts->s3_weight > 1000)
      return VLAC_ERR_INVALID_ARG;
    p.s3_lo = opts->s3_lo;
    p.s3_hi = opts->s3_hi;
    p.s3_weight = opts->s3_weight;
    p.has_s3_forced = opts->s3_forced ? 1 : 0;
    if (c->n_textrows < 1) return VLAC_ERR_UNSUPPORTED;  // no text rows after the image to measure
  }
  // an error latched by an earlier step on this context is reported first
  if (*c->err_host) {
    const int e = *c->err_host;
    *c->err_host = 0;
    cudaMemsetAsync(c->err, 0, sizeof(int), static_cast<cudaStream_t>(stream));
    return e;
  }
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const vlac_dims& d = c->d;
  const int B = k->B, D = d.n_action;
  const size_t fb = (size_t)d.n_views * d.img_h * d.img_w * 3;
  CopyList in{};
  auto add = [](CopyList& l, const void* src, void* dst, size_t bytes) {
    if (src && dst && bytes && l.n < kMaxSpans) l.span[l.n++] = CopySpan{src, dst, bytes};
  };
  add(in, frames, c->in_frames, (size_t)B * fb);
  add(in, prompt_ids, c->in_prompt, (size_t)B * d.n_text * 4);
  if (d.proprio_dim) add(in, proprio, c->in_proprio, (size_t)B * d.proprio_dim * 4);
  if (p.has_override) add(in, opts->gate_override, c->in_override, (size_t)B);
  if (p.has_forced) add(in, opts->forced_ids, c->in_forced, (size_t)B * D * 4);
  if (p.has_active) add(in, opts->active, c->in_active, (size_t)B);
  if (p.has_s2_forced) add(in, opts->s2_forced, c->in_s2_forced, (size_t)B * c->Nv);
  if (p.has_s3_forced) add(in, opts->s3_forced, c->in_s3_forced, (size_t)B * d.n_layers * 2);
  {
    ProfScope ps_(c, VLAC_PROF_OTHER, 0, st);
    launch_stage(p, c->prm, in, st);
  }
  c->launches += 1;
  c->s2_on = p.s2_top_k > 0;
  c->s2_layer = p.s2_layer;
  c->s3_on = p.s3_adaptive != 0;
  c->vm_on = mk == VLAC_MARGIN_VOCAB || out->vocab_margin != nullptr;
  int rc = run_step(c, k, st);
  if (rc) return rc;
  CopyList o{};
  add(o, c->o_ids, out->action_ids, (size_t)B * D * 4);
  add(o, c->o_margins, out->margins, (size_t)B * D * 4);
  add(o, c->o_gaps, out->logit_gap, (size_t)B * D * 4);
  add(o, c->o_recomputed, out->recomputed, (size_t)B);
  add(o, c->o_step_margin, out->step_margin, (size_t)B * 4);
  add(o, c->o_gate_auto, out->gate_auto, (size_t)B);
  add(o, c->o_logits, out->logits, (size_t)B * D * d.n_bins * 4);
  add(o, c->o_mask, out->static_mask, (size_t)B * c->Nv);
  add(o, c->o_idx, out->idx, (size_t)B * c->S * 4);
  add(o, c->o_M, out->M, (size_t)B * d.n_layers * 4);
  add(o, c->o_rel, out->relevance, (size_t)B * c->Nv * 4);
  add(o, c->o_relevant, out->relevant, (size_t)B * c->Nv);
  add(o, c->o_entropy, out->entropy, (size_t)B * D * 4);
  if (c->vm_on) add(o, c->o_vm, out->vocab_margin, (size_t)B * D * 4);
  add(o, c->o_delta, out->action_delta, (size_t)B * 4);
  add(o, c->o_lent, out->layer_entropy, (size_t)B * d.n_layers * 4);
  add(o, c->sched_own, out->schedule, (size_t)B * d.n_layers * 2);
  {
    ProfScope ps_(c, VLAC_PROF_OTHER, 0, st);
    launch_copies(o, st);
  }
  c->launches += 1;
  CK(cudaGetLastError());
  return VLAC_OK;
}

// ---- the one-layer workload -----------------------------------------------------

namespace {
template <typename T>
int layer_bench_impl(vlac_ctx* c, vlac_cache* k, int seq, int layer, const int32_t* pos, int M, float* x,
                     cudaStream_t st) {
  const vlac_dims& d = c->d;
  const size_t Hd = d.hidden, kv_layer = (size_t)d.n_heads * c->Tc * d.head_dim;
  launch_layer_setup(pos, M, c->S, c->idx, c->off, c->err, st);
  c->launches += 1;
  CK(cudaMemcpyAsync(c->X, x, (size_t)M * Hd * sizeof(float), cudaMemcpyDeviceToDevice, st));
  Rows rl{c->off, c->idx, c->S, c->X};
  T* Kc = static_cast<T*>(k->K) + (size_t)seq * k->kv_seq_stride + (size_t)layer * kv_layer;
  T* Vc = static_cast<T*>(k->V) + (size_t)seq * k->kv_seq_stride + (size_t)layer * kv_layer;
  prefix_layer<T>(c, rl, rl.off, 1, layer, nullptr, 0, Kc, Vc, k->kv_seq_stride, &k->kvm, seq, st);
  CK(cudaMemcpyAsync(x, c->X, (size_t)M * Hd * sizeof(float), cudaMemcpyDeviceToDevice, st));
  CK(cudaGetLastError());
  return c->fatal ? VLAC_ERR_INVALID_ARG : VLAC_OK;
}
}  // namespace

extern "C" int vlac_layer_bench(vlac_ctx* c, vlac_cache* k, int seq, int layer, const int32_t* pos, int M, float* x,
                                void* stream) {
  if (!c || !k || !pos || !x || k->ctx != c || seq < 0 || seq >= k->B || layer < 0 || layer >= c->d.n_layers ||
      M < 1 || M > c->S)
    return VLAC_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  return c->bf16 ? layer_bench_impl<bf16>(c, k, seq, layer, pos, M, x, st)
                 : layer_bench_impl<float>(c, k, seq, layer, pos, M, x, st);
}

namespace {
int kv_move(const vlac_cache* k, int seq, int layer, void* K, void* V, bool to_cache, void* stream) {
  if (!k || !K || !V || seq < 0 || seq >= k->B || layer < 0 || layer >= k->ctx->d.n_layers ||
      (reinterpret_cast<uintptr_t>(K) | reinterpret_cast<uintptr_t>(V)) % 4)
    return VLAC_ERR_INVALID_ARG;
  const vlac_ctx* c = k->ctx;
  const vlac_dims& d = c->d;
  const size_t kv_layer = (size_t)d.n_heads * c->Tc * d.head_dim;
  const size_t off = ((size_t)seq * k->kv_seq_stride + (size_t)layer * kv_layer) * c->esz;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  launch_kv_copy(static_cast<char*>(k->K) + off, K, d.n_heads, c->Tc, d.head_dim, (int)c->esz, to_cache, st);
  launch_kv_copy(static_cast<char*>(k->V) + off, V, d.n_heads, c->Tc, d.head_dim, (int)c->esz, to_cache, st);
  CK(cudaGetLastError());
  return VLAC_OK;
}
}  // namespace

extern "C" int vlac_cache_load(vlac_cache* k, int seq, int layer, const void* K, const void* V, void* stream) {
  return kv_move(k, seq, layer, const_cast<void*>(K), const_cast<void*>(V), true, stream);
}
extern "C" int vlac_cache_store(const vlac_cache* k, int seq, int layer, void* K, void* V, void* stream) {
  return kv_move(k, seq, layer, K, V, false, stream);
}

extern "C" int vlac_sync_error(vlac_ctx* c) {
  if (!c) return VLAC_ERR_INVALID_ARG;
  CK(cudaDeviceSynchronize());
  int e = 0;
  CK(cudaMemcpy(&e, c->err, sizeof(int), cudaMemcpyDeviceToHost));
  CK(cudaMemset(c->err, 0, sizeof(int)));
  *c->err_host = 0;
  return e;
}

extern "C" uint64_t vlac_launch_count(const vlac_ctx* c) { return c ? c->launches : 0; }

extern "C" int vlac_selftest_wait(vlac_ctx* c, uint32_t spin_limit) {
  if (!c) return VLAC_ERR_INVALID_ARG;
  CK(cudaDeviceSynchronize());
  CK(cudaMemset(c->err, 0, sizeof(int)));
  if (launch_wait_selftest(c->err, spin_limit, 0)) return VLAC_ERR_CUDA;
  c->launches += 1;
  CK(cudaDeviceSynchronize());
  int e = 0;
  CK(cudaMemcpy(&e, c->err, sizeof(int), cudaMemcpyDeviceToHost));
  CK(cudaMemset(c->err, 0, sizeof(int)));
  return e;
}

extern "C" int vlac_set_wait_limit(vlac_ctx* c, uint32_t polls) {
  if (!c) return VLAC_ERR_INVALID_ARG;
  c->wait_limit = polls;
  return VLAC_OK;
}

extern "C" int vlac_prof_enable(vlac_ctx* c, int on) {
  if (!c) return VLAC_ERR_INVALID_ARG;
  c->prof_on = on != 0;
  return VLAC_OK;
}

extern "C" int vlac_prof_read(vlac_ctx* c, int kind, double* total_ms, uint64_t* launches, double* bytes) {
  if (!c || !total_ms || !launches || !bytes) return VLAC_ERR_INVALID_ARG;
  double ms = 0, by = 0;
  uint64_t n = 0;
  if (kind < 0 || kind >= VLAC_PROF_KINDS) return VLAC_ERR_INVALID_ARG;
  std::vector<vlac_ctx::ProfRec> keep;
  for (auto& r : c->prof) {
    if (r.kind != kind) {
      keep.push_back(r);
      continue;
    }
    float t = 0.f;
    if (cudaEventSynchronize(r.b) != cudaSuccess || cudaEventElapsedTime(&t, r.a, r.b) != cudaSuccess) {
      (void)cudaGetLastError();
      return VLAC_ERR_CUDA;
    }
    ms += t;
    by += r.bytes;
    ++n;
    c->ev_pool.push_back(r.a);
    c->ev_pool.push_back(r.b);
  }
  c->prof.swap(keep);
  *total_ms = ms;
  *launches = n;
  *bytes = by;
  return VLAC_OK;
}

extern "C" const char* vlac_strerror(int code) {
  switch (code) {
    case VLAC_OK: return "ok";
    case VLAC_ERR_INVALID_ARG: return "invalid argument";
    case VLAC_ERR_CUDA: return "CUDA runtime error";
    case VLAC_ERR_OOM: return "out of memory";
    case VLAC_ERR_TIMEOUT: return "a bounded device wait gave up";
    case VLAC_ERR_DEVICE_CHECK: return "a device-side bounds check rejected an input";
    case VLAC_ERR_STATE: return "cache does not belong to this context";
    case VLAC_ERR_UNSUPPORTED: return "dims not supported by this build";
    default: return "unknown error";
  }
}
