// Row-wise kernels of the layer loop: layer-0 inputs (Sec. III-A: patches
// projected to token embeddings and concatenated with the language tokens),
// the layer-input gather/record of the cached representations, RMSNorm, the
// GEMM epilogues (RoPE + K/V scatter, residual adds, SwiGLU) and the Eq. (1)
// action head.  Every kernel handles rows (b, i), i < count_b, on a
// (rows, batch) grid; the compacted row index is off[b] + i.
#include "internal.cuh"

namespace vlac {

// ---- layer-0 inputs ----------------------------------------------------------

// im2col of the visual rows of layer 0: row r holds the patch bytes (y, x, c)
// as T, zero-padded to kpad columns; non-visual rows are zero.
template <typename T>
__global__ void im2col_kernel(Rows rows, const uint8_t* __restrict__ frames, int n_views, int img_h, int img_w,
                              int patch, int kpad, T* __restrict__ col) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.y, i = blockIdx.x;
  const int cnt = rows.off[b + 1] - rows.off[b];
  if (i >= cnt) return;
  const int r = rows.off[b] + i;
  const int pos = rows.idx[(size_t)b * rows.idx_stride + i];
  const int gw = img_w / patch, gh = img_h / patch, Nv = n_views * gw * gh;
  T* dst = col + (size_t)r * kpad;
  const int n = patch * patch * 3, row_bytes = patch * 3;
  if (pos >= 1 && pos <= Nv) {
    const int v = pos - 1, view = v / (gw * gh), rr = v % (gw * gh), py = rr / gw, px = rr % gw;
    const uint8_t* f = frames + (size_t)b * n_views * img_h * img_w * 3;
    for (int e = threadIdx.x; e < kpad; e += blockDim.x) {
      float val = 0.f;
      if (e < n) {
        const int ry = e / row_bytes, rem = e - ry * row_bytes;
        val = (float)f[((size_t)(view * img_h + py * patch + ry) * img_w + (size_t)px * patch) * 3 + rem];
      }
      dst[e] = from_f<T>(val);
    }
  } else {
    for (int e = threadIdx.x; e < kpad; e += blockDim.x) dst[e] = from_f<T>(0.f);
  }
}

// Layer-0 residual rows: text -> token embedding, visual -> (W_p . patch) / 255
// (the GEMM output in patch_part), proprio -> W_pr . proprio, parallel action
// positions -> their learned embedding.
template <typename T>
__global__ void embed_kernel(Rows rows, int hidden, int Nv, int P, int has_proprio, int proprio_dim, int n_text,
                             int vocab, const int32_t* __restrict__ prompt, const float* __restrict__ proprio,
                             const T* __restrict__ tok_emb, const float* __restrict__ patch_part,
                             const T* __restrict__ proprio_w, const T* __restrict__ action_emb, int* err) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.y, i = blockIdx.x;
  const int cnt = rows.off[b + 1] - rows.off[b];
  if (i >= cnt) return;
  const int r = rows.off[b] + i;
  const int pos = rows.idx[(size_t)b * rows.idx_stride + i];
  float* x = rows.X + ((size_t)b * rows.idx_stride + i) * hidden;
  const bool is_text = pos == 0 || (pos > Nv + has_proprio && pos < P);
  if (is_text) {
    const int t = pos == 0 ? 0 : pos - Nv - has_proprio;
    int id = prompt[(size_t)b * n_text + t];
    if (id < 0 || id >= vocab) {
      if (threadIdx.x == 0) set_error(err, VLAC_ERR_DEVICE_CHECK);
      id = 0;
    }
    const T* e = tok_emb + (size_t)id * hidden;
    for (int k = threadIdx.x; k < hidden; k += blockDim.x) x[k] = to_f(e[k]);
  } else if (pos >= 1 && pos <= Nv) {
    const float* p = patch_part + (size_t)r * hidden;
    for (int k = threadIdx.x; k < hidden; k += blockDim.x) x[k] = p[k] / 255.0f;
  } else if (has_proprio && pos == Nv + 1) {
    const float* pr = proprio + (size_t)b * proprio_dim;
    for (int k = threadIdx.x; k < hidden; k += blockDim.x) {
      float s = 0.f;
      for (int j = 0; j < proprio_dim; ++j) s = fmaf(to_f(proprio_w[(size_t)k * proprio_dim + j]), pr[j], s);
      x[k] = s;
    }
  } else {
    const T* e = action_emb + (size_t)(pos - P) * hidden;
    for (int k = threadIdx.x; k < hidden; k += blockDim.x) x[k] = to_f(e[k]);
  }
}

// ---- RMSNorm ----------------------------------------------------------------

// y = T((x * r) * g), r = 1 / sqrt(mean(x^2) + eps).  One block per row.
template <typename T>
__device__ __forceinline__ void rmsnorm_row(const float* __restrict__ x, const T* __restrict__ g, int hidden,
                                            float eps, T* __restrict__ y, float* red) {
  float ss = 0.f;
  for (int k = threadIdx.x; k < hidden; k += blockDim.x) ss = fmaf(x[k], x[k], ss);
  ss = block_sum(ss, red);
  const float r = 1.0f / sqrtf(ss / (float)hidden + eps);
  for (int k = threadIdx.x; k < hidden; k += blockDim.x) y[k] = from_f<T>((x[k] * r) * to_f(g[k]));
}

// Layer input: rows computed at the previous layer record their layer-l input
// in the H cache; rows that join at layer l start from the cached layer-l
// input of their position; every row of this layer is normalised into A.
template <typename T>
__global__ void layer_in_kernel(Rows rows, const int* __restrict__ off_prev, int hidden, float* __restrict__ H,
                                size_t h_seq_stride, const T* __restrict__ gain, float eps, T* __restrict__ A) {
  pdl_wait();
  pdl_trigger();
  __shared__ float red[32];
  const int b = blockIdx.y, i = blockIdx.x;
  const int cnt = rows.off[b + 1] - rows.off[b];
  const int cnt_prev = off_prev[b + 1] - off_prev[b];
  if (i >= cnt && (H == nullptr || i >= cnt_prev)) return;
  const int pos = rows.idx[(size_t)b * rows.idx_stride + i];
  float* x = rows.X + ((size_t)b * rows.idx_stride + i) * hidden;
  if (H) {
    float* h = H + (size_t)b * h_seq_stride + (size_t)pos * hidden;
    const float4* s4 = reinterpret_cast<const float4*>(i < cnt_prev ? x : h);
    float4* d4 = reinterpret_cast<float4*>(i < cnt_prev ? h : x);
    for (int k = threadIdx.x; k < hidden / 4; k += blockDim.x) d4[k] = s4[k];
    __syncthreads();
  }
  if (i >= cnt) return;
  rmsnorm_row<T>(x, gain, hidden, eps, A + (size_t)(rows.off[b] + i) * hidden, red);
}

// ---- GEMM epilogues ------------------------------------------------------------

__device__ __forceinline__ float sum_splits(const float* __restrict__ part, int splits, size_t stride, size_t o) {
  float v = part[o];
  for (int s = 1; s < splits; ++s) v += part[o + (size_t)s * stride];
  return v;
}

// q, k, v from the fused projection [q | k | v]; RoPE (rotate-half) on q and k
// at the row's absolute position; Q to its row, K and V scattered into the
// cache at that position (layout [b][head][position][head_dim]).
template <typename T>
__global__ void qkv_epilogue_kernel(Rows rows, int n_heads, int head_dim, const float* __restrict__ part,
                                    int splits, size_t split_stride, const float* __restrict__ rope_cos,
                                    const float* __restrict__ rope_sin, T* __restrict__ Q, T* __restrict__ Kc,
                                    T* __restrict__ Vc, size_t kv_seq_stride, int Tc) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.y, i = blockIdx.x;
  const int cnt = rows.off[b + 1] - rows.off[b];
  if (i >= cnt) return;
  const int r = rows.off[b] + i;
  const int pos = rows.idx[(size_t)b * rows.idx_stride + i];
  const int hidden = n_heads * head_dim, half = head_dim / 2, N = 3 * hidden;
  const float* pr = part + (size_t)r * N;
  T* q_out = Q + (size_t)r * hidden;
  for (int t = threadIdx.x; t < n_heads * half; t += blockDim.x) {
    const int h = t / half, e = t - h * half;
    const float c = rope_cos[(size_t)pos * half + e], s = rope_sin[(size_t)pos * half + e];
    const size_t base = (size_t)h * head_dim + e;
    const float q1 = sum_splits(pr, splits, split_stride, base);
    const float q2 = sum_splits(pr, splits, split_stride, base + half);
    const float k1 = sum_splits(pr, splits, split_stride, hidden + base);
    const float k2 = sum_splits(pr, splits, split_stride, hidden + base + half);
    const float v1 = sum_splits(pr, splits, split_stride, 2 * hidden + base);
    const float v2 = sum_splits(pr, splits, split_stride, 2 * hidden + base + half);
    q_out[base] = from_f<T>(q1 * c - q2 * s);
    q_out[base + half] = from_f<T>(q2 * c + q1 * s);
    const size_t kv = (size_t)b * kv_seq_stride + ((size_t)h * Tc + pos) * head_dim + e;
    Kc[kv] = from_f<T>(k1 * c - k2 * s);
    Kc[kv + half] = from_f<T>(k2 * c + k1 * s);
    Vc[kv] = from_f<T>(v1);
    Vc[kv + half] = from_f<T>(v2);
  }
}

// x += o-projection (summed over splits), then A = T(RMSNorm(x) * g).
template <typename T>
__global__ void residual_norm_kernel(Rows rows, int hidden, const float* __restrict__ part, int splits,
                                     size_t split_stride, const T* __restrict__ gain, float eps, T* __restrict__ A) {
  pdl_wait();
  pdl_trigger();
  __shared__ float red[32];
  const int b = blockIdx.y, i = blockIdx.x;
  const int cnt = rows.off[b + 1] - rows.off[b];
  if (i >= cnt) return;
  const int r = rows.off[b] + i;
  float* x = rows.X + ((size_t)b * rows.idx_stride + i) * hidden;
  const float* pr = part + (size_t)r * hidden;
  for (int k = threadIdx.x; k < hidden; k += blockDim.x) x[k] = x[k] + sum_splits(pr, splits, split_stride, k);
  __syncthreads();
  rmsnorm_row<T>(x, gain, hidden, eps, A + (size_t)r * hidden, red);
}

// G = T(silu(g) * u) from the fused projection [gate | up].
template <typename T>
__global__ void swiglu_kernel(Rows rows, int ffn, const float* __restrict__ part, int splits, size_t split_stride,
                              T* __restrict__ G) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.y, i = blockIdx.x;
  const int cnt = rows.off[b + 1] - rows.off[b];
  if (i >= cnt) return;
  const int r = rows.off[b] + i;
  const float* pr = part + (size_t)r * 2 * ffn;
  for (int j = threadIdx.x; j < ffn; j += blockDim.x) {
    const float g = sum_splits(pr, splits, split_stride, j);
    const float u = sum_splits(pr, splits, split_stride, (size_t)ffn + j);
    G[(size_t)r * ffn + j] = from_f<T>((g / (1.0f + expf(-g))) * u);
  }
}

// x += down-projection (summed over splits).
__global__ void residual_kernel(Rows rows, int hidden, const float* __restrict__ part, int splits,
                                size_t split_stride) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.y, i = blockIdx.x;
  const int cnt = rows.off[b + 1] - rows.off[b];
  if (i >= cnt) return;
  const int r = rows.off[b] + i;
  float* x = rows.X + ((size_t)b * rows.idx_stride + i) * hidden;
  const float* pr = part + (size_t)r * hidden;
  for (int k = threadIdx.x; k < hidden; k += blockDim.x) x[k] = x[k] + sum_splits(pr, splits, split_stride, k);
}

// Autoregressive decode input: the bin fed back (argmax, or the forced replay
// bin) selects token vocab - n_bins + bin at position P + d - 1.
template <typename T>
__global__ void decode_embed_kernel(int d, int D, int P, int hidden, int vocab, int n_bins,
                                    const T* __restrict__ tok_emb, const int32_t* __restrict__ ids,
                                    const int32_t* __restrict__ forced, const StepParams* __restrict__ prm,
                                    float* __restrict__ Xd, int* __restrict__ idx_dec, float* __restrict__ ssq_out,
                                    int* err) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.x;
  int bin = (prm->has_forced && forced) ? forced[(size_t)b * D + d - 1] : ids[(size_t)b * D + d - 1];
  if (bin < 0 || bin >= n_bins) {
    if (threadIdx.x == 0) set_error(err, VLAC_ERR_DEVICE_CHECK);
    bin = 0;
  }
  const T* e = tok_emb + (size_t)(vocab - n_bins + bin) * hidden;
  for (int k = threadIdx.x; k < hidden; k += blockDim.x) Xd[(size_t)b * hidden + k] = to_f(e[k]);
  // sums of squares of the new residual row, in the decode GEMVs' groups of rows
  const int ng = hidden / kDecodeRowsPerCta;
  for (int g = threadIdx.x; g < ng; g += blockDim.x) {
    float t = 0.f;
    for (int r = 0; r < kDecodeRowsPerCta; ++r) {
      const float v = to_f(e[g * kDecodeRowsPerCta + r]);
      t = fmaf(v, v, t);
    }
    ssq_out[(size_t)b * ng + g] = t;
  }
  if (threadIdx.x == 0) idx_dec[b] = P + d - 1;
}

// m_t = mean (Eq. 1) or min of the per-token signals; the cache keeps it for
// the next step's gate and becomes valid.
__global__ void finish_kernel(int B, int D, const StepParams* __restrict__ prm, const float* __restrict__ margins,
                              const float* __restrict__ gaps, float* __restrict__ m_prev, uint8_t* __restrict__ valid,
                              float* __restrict__ user_step_margin) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const float* sig = (prm->margin_kind == VLAC_MARGIN_LOGIT ? gaps : margins) + (size_t)b * D;
  float m;
  if (prm->reduction == VLAC_REDUCE_MIN) {
    m = sig[0];
    for (int a = 1; a < D; ++a) m = fminf(m, sig[a]);
  } else {
    float s = 0.f;
    for (int a = 0; a < D; ++a) s += sig[a];
    m = s / (float)D;
  }
  m_prev[b] = m;
  valid[b] = 1;
  user_step_margin[b] = m;
}

// ---- per-step staging -------------------------------------------------------------

// Block-strided byte copies of every span (16-byte vectors when both ends are
// aligned); block 0 also writes the step scalars.
__global__ void copy_spans_kernel(CopyList list, StepParams p, StepParams* prm) {
  pdl_wait();
  pdl_trigger();
  if (prm && blockIdx.x == 0 && threadIdx.x == 0) *prm = p;
  for (int s = 0; s < list.n; ++s) {
    const CopySpan c = list.span[s];
    const uint8_t* src = static_cast<const uint8_t*>(c.src);
    uint8_t* dst = static_cast<uint8_t*>(c.dst);
    const size_t tid = (size_t)blockIdx.x * blockDim.x + threadIdx.x, nth = (size_t)gridDim.x * blockDim.x;
    if (((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15) == 0) {
      const size_t nv = c.bytes / 16;
      for (size_t i = tid; i < nv; i += nth)
        reinterpret_cast<uint4*>(dst)[i] = reinterpret_cast<const uint4*>(src)[i];
      for (size_t i = nv * 16 + tid; i < c.bytes; i += nth) dst[i] = src[i];
    } else {
      for (size_t i = tid; i < c.bytes; i += nth) dst[i] = src[i];
    }
  }
}

void launch_stage(const StepParams& p, StepParams* prm, const CopyList& list, cudaStream_t st) {
  launch_k(copy_spans_kernel, dim3(64), dim3(256), 0, st, list, p, prm);
}
void launch_copies(const CopyList& list, cudaStream_t st) {
  StepParams none{};
  launch_k(copy_spans_kernel, dim3(8), dim3(256), 0, st, list, none, (StepParams*)nullptr);
}

// ---- launchers -----------------------------------------------------------------

template <typename T>
void launch_im2col(Rows rows, int B, int S, const uint8_t* frames, int n_views, int img_h, int img_w, int patch,
                   int kpad, T* col, cudaStream_t st) {
  launch_k(im2col_kernel<T>, dim3(S, B), dim3(128), 0, st, rows, frames, n_views, img_h, img_w, patch, kpad, col);
}
template <typename T>
void launch_embed(Rows rows, int B, int S, int hidden, int Nv, int P, int has_proprio, int proprio_dim, int n_text,
                  int vocab, const int32_t* prompt, const float* proprio, const T* tok_emb, const float* patch_part,
                  const T* proprio_w, const T* action_emb, int* err, cudaStream_t st) {
  launch_k(embed_kernel<T>, dim3(S, B), dim3(256), 0, st, rows, hidden, Nv, P, has_proprio, proprio_dim, n_text,
           vocab, prompt, proprio, tok_emb, patch_part, proprio_w, action_emb, err);
}
template <typename T>
void launch_layer_in(Rows rows, const int* off_prev, int B, int S, int hidden, float* H, size_t h_seq_stride,
                     const T* gain, float eps, T* A, cudaStream_t st) {
  launch_k(layer_in_kernel<T>, dim3(S, B), dim3(256), 0, st, rows, off_prev, hidden, H, h_seq_stride, gain, eps, A);
}
template <typename T>
void launch_qkv_epilogue(Rows rows, int B, int S, int n_heads, int head_dim, const float* part, int splits,
                         size_t split_stride, const float* rope_cos, const float* rope_sin, T* Q, T* Kc, T* Vc,
                         size_t kv_seq_stride, int Tc, cudaStream_t st) {
  launch_k(qkv_epilogue_kernel<T>, dim3(S, B), dim3(256), 0, st, rows, n_heads, head_dim, part, splits, split_stride,
           rope_cos, rope_sin, Q, Kc, Vc, kv_seq_stride, Tc);
}
template <typename T>
void launch_residual_norm(Rows rows, int B, int S, int hidden, const float* part, int splits, size_t split_stride,
                          const T* gain, float eps, T* A, cudaStream_t st) {
  launch_k(residual_norm_kernel<T>, dim3(S, B), dim3(256), 0, st, rows, hidden, part, splits, split_stride, gain, eps,
           A);
}
template <typename T>
void launch_swiglu(Rows rows, int B, int S, int ffn, const float* part, int splits, size_t split_stride, T* G,
                   cudaStream_t st) {
  launch_k(swiglu_kernel<T>, dim3(S, B), dim3(256), 0, st, rows, ffn, part, splits, split_stride, G);
}
void launch_residual(Rows rows, int B, int S, int hidden, const float* part, int splits, size_t split_stride,
                     cudaStream_t st) {
  launch_k(residual_kernel, dim3(S, B), dim3(256), 0, st, rows, hidden, part, splits, split_stride);
}
template <typename T>
void launch_decode_embed(int B, int d, int D, int P, int hidden, int vocab, int n_bins, const T* tok_emb,
                         const int32_t* ids, const int32_t* forced, const StepParams* prm, float* Xd, int* idx_dec,
                         float* ssq_out, int* err, cudaStream_t st) {
  launch_k(decode_embed_kernel<T>, dim3(B), dim3(256), 0, st, d, D, P, hidden, vocab, n_bins, tok_emb, ids, forced,
           prm, Xd, idx_dec, ssq_out, err);
}
void launch_finish(int B, int D, const StepParams* prm, const float* margins, const float* gaps, float* m_prev,
                   uint8_t* valid, float* user_step_margin, cudaStream_t st) {
  launch_k(finish_kernel, dim3((B + 63) / 64), dim3(64), 0, st, B, D, prm, margins, gaps, m_prev, valid,
           user_step_margin);
}

#define VLAC_INST(T)                                                                                              \
  template void launch_im2col<T>(Rows, int, int, const uint8_t*, int, int, int, int, int, T*, cudaStream_t);     \
  template void launch_embed<T>(Rows, int, int, int, int, int, int, int, int, int, const int32_t*, const float*, \
                                const T*, const float*, const T*, const T*, int*, cudaStream_t);                 \
  template void launch_layer_in<T>(Rows, const int*, int, int, int, float*, size_t, const T*, float, T*,          \
                                   cudaStream_t);                                                                 \
  template void launch_qkv_epilogue<T>(Rows, int, int, int, int, const float*, int, size_t, const float*,         \
                                       const float*, T*, T*, T*, size_t, int, cudaStream_t);                      \
  template void launch_residual_norm<T>(Rows, int, int, int, const float*, int, size_t, const T*, float, T*,      \
                                        cudaStream_t);                                                            \
  template void launch_swiglu<T>(Rows, int, int, int, const float*, int, size_t, T*, cudaStream_t);               \
  template void launch_decode_embed<T>(int, int, int, int, int, int, int, const T*, const int32_t*,               \
                                       const int32_t*, const StepParams*, float*, int*, float*, int*, cudaStream_t);
VLAC_INST(float)
VLAC_INST(bf16)

}  // namespace vlac
