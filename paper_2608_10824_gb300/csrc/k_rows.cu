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

// ---- vector helpers (4 consecutive elements; row lengths are multiples of 4) ----

template <typename T> __device__ __forceinline__ float4 load4(const T* p);
template <> __device__ __forceinline__ float4 load4<float>(const float* p) { return *reinterpret_cast<const float4*>(p); }
template <> __device__ __forceinline__ float4 load4<bf16>(const bf16* p) {
  const uint2 w = *reinterpret_cast<const uint2*>(p);
  return make_float4(__uint_as_float(w.x << 16), __uint_as_float(w.x & 0xFFFF0000u), __uint_as_float(w.y << 16),
                     __uint_as_float(w.y & 0xFFFF0000u));
}
template <typename T> __device__ __forceinline__ void store4(T* p, float4 v);
template <> __device__ __forceinline__ void store4<float>(float* p, float4 v) { *reinterpret_cast<float4*>(p) = v; }
template <> __device__ __forceinline__ void store4<bf16>(bf16* p, float4 v) {
  const __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y), hi = __floats2bfloat162_rn(v.z, v.w);
  *reinterpret_cast<uint2*>(p) =
      make_uint2(*reinterpret_cast<const uint32_t*>(&lo), *reinterpret_cast<const uint32_t*>(&hi));
}
__device__ __forceinline__ float4 add4(float4 a, float4 b) {
  return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}
__device__ __forceinline__ float sq4(float4 a, float acc) {
  return fmaf(a.w, a.w, fmaf(a.z, a.z, fmaf(a.y, a.y, fmaf(a.x, a.x, acc))));
}
// Sum over the GEMM's K splits of column o of compacted row r (pr = that
// row of split 0), in split order; see SplitPlan for the layout.
__device__ __forceinline__ float4 sum_splits4(const float* __restrict__ pr, const SplitPlan& sp, int r, size_t o) {
  float4 v = *reinterpret_cast<const float4*>(pr + o);
  if ((long long)o < sp.full_cols) return v;
  if (sp.tail_ld) {
    const float* t = sp.tail_p + (size_t)r * sp.tail_ld + (o - sp.full_cols);
    for (int s = 1; s < sp.tail; ++s) v = add4(v, *reinterpret_cast<const float4*>(t + (size_t)(s - 1) * sp.tail_stride));
  } else {
    for (int s = 1; s < sp.tail; ++s) v = add4(v, *reinterpret_cast<const float4*>(pr + o + (size_t)s * sp.stride));
  }
  return v;
}

// ---- RMSNorm ----------------------------------------------------------------

// Threads of a row-normalising block: one float4 of a 4096-wide row each, so
// that all of a row's loads are in flight at once.
constexpr int kNormThreads = 1024;

// y = T((x * r) * g), r = 1 / sqrt(mean(x^2) + eps); `ss` is this thread's part
// of sum(x^2).  One block per row.
template <typename T>
__device__ __forceinline__ void rmsnorm_row(const float* __restrict__ x, float ss, const T* __restrict__ g, int hidden,
                                            float eps, T* __restrict__ y, float* red) {
  ss = block_sum(ss, red);
  const float r = 1.0f / sqrtf(ss / (float)hidden + eps);
#pragma unroll 4
  for (int c = threadIdx.x; c < hidden / 4; c += blockDim.x) {
    const float4 xv = reinterpret_cast<const float4*>(x)[c], gv = load4<T>(g + 4 * c);
    store4<T>(y + 4 * c, make_float4((xv.x * r) * gv.x, (xv.y * r) * gv.y, (xv.z * r) * gv.z, (xv.w * r) * gv.w));
  }
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
  float ss = 0.f;
  if (H) {
    float* h = H + (size_t)b * h_seq_stride + (size_t)pos * hidden;
    const float4* s4 = reinterpret_cast<const float4*>(i < cnt_prev ? x : h);
    float4* d4 = reinterpret_cast<float4*>(i < cnt_prev ? h : x);
#pragma unroll 4
    for (int k = threadIdx.x; k < hidden / 4; k += blockDim.x) {
      const float4 v = s4[k];
      d4[k] = v;
      ss = sq4(v, ss);
    }
  } else {
#pragma unroll 4
    for (int k = threadIdx.x; k < hidden / 4; k += blockDim.x) ss = sq4(reinterpret_cast<const float4*>(x)[k], ss);
  }
  if (i >= cnt) return;
  rmsnorm_row<T>(x, ss, gain, hidden, eps, A + (size_t)(rows.off[b] + i) * hidden, red);
}

// The down-projection residual of layer l fused with layer l+1's input: rows
// computed at layer l add their down-projection (summed over splits), and
// the sum is their layer-(l+1) input, recorded in the H cache; rows that join
// at layer l+1 start from H; every row of layer l+1 is normalised into A.
// The same arithmetic, element for element, as residual_kernel followed by
// layer_in_kernel.  rows: layer l+1's; off_prev: layer l's row offsets.
template <typename T>
__global__ void residual_layer_in_kernel(Rows rows, const int* __restrict__ off_prev, int hidden,
                                         const float* __restrict__ part, SplitPlan sp, float* __restrict__ H,
                                         size_t h_seq_stride, const T* __restrict__ gain, float eps,
                                         T* __restrict__ A) {
  pdl_wait();
  pdl_trigger();
  __shared__ float red[32];
  const int b = blockIdx.y, i = blockIdx.x;
  const int cnt = rows.off[b + 1] - rows.off[b];
  const int cnt_prev = off_prev[b + 1] - off_prev[b];
  if (i >= cnt && i >= cnt_prev) return;
  const int pos = rows.idx[(size_t)b * rows.idx_stride + i];
  float* x = rows.X + ((size_t)b * rows.idx_stride + i) * hidden;
  float4* x4 = reinterpret_cast<float4*>(x);
  float4* h4 = reinterpret_cast<float4*>(H + (size_t)b * h_seq_stride + (size_t)pos * hidden);
  float ss = 0.f;
  if (i < cnt_prev) {
    const int r = off_prev[b] + i;
    const float* pr = part + (size_t)r * hidden;
#pragma unroll 4
    for (int k = threadIdx.x; k < hidden / 4; k += blockDim.x) {
      const float4 v = add4(x4[k], sum_splits4(pr, sp, r, 4 * (size_t)k));
      x4[k] = v;
      h4[k] = v;
      ss = sq4(v, ss);
    }
  } else {
#pragma unroll 4
    for (int k = threadIdx.x; k < hidden / 4; k += blockDim.x) {
      const float4 v = h4[k];
      x4[k] = v;
      ss = sq4(v, ss);
    }
  }
  if (i >= cnt) return;
  rmsnorm_row<T>(x, ss, gain, hidden, eps, A + (size_t)(rows.off[b] + i) * hidden, red);
}

// ---- GEMM epilogues ------------------------------------------------------------

// q, k, v from the fused projection [q | k | v]; RoPE (rotate-half) on q and k
// at the row's absolute position; Q to its row, K and V scattered into the
// cache at that position (layout [b][head][position][head_dim]).  A thread
// takes four consecutive e of one head and their partners e + half.
template <typename T>
__global__ void qkv_epilogue_kernel(Rows rows, int n_heads, int head_dim, const float* __restrict__ part,
                                    SplitPlan sp, const float* __restrict__ rope_cos,
                                    const float* __restrict__ rope_sin, T* __restrict__ Q, T* __restrict__ Kc,
                                    T* __restrict__ Vc, size_t kv_seq_stride, int Tc) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.y, i = blockIdx.x;
  const int cnt = rows.off[b + 1] - rows.off[b];
  if (i >= cnt) return;
  const int r = rows.off[b] + i;
  const int pos = rows.idx[(size_t)b * rows.idx_stride + i];
  const int hidden = n_heads * head_dim, half = head_dim / 2, N = 3 * hidden, q4 = half / 4;
  const float* pr = part + (size_t)r * N;
  T* q_out = Q + (size_t)r * hidden;
  // gridDim.z blocks share a row
  const int nt = n_heads * q4, t0 = (int)(((long long)nt * blockIdx.z) / gridDim.z);
  const int t1 = (int)(((long long)nt * (blockIdx.z + 1)) / gridDim.z);
  for (int t = t0 + threadIdx.x; t < t1; t += blockDim.x) {
    const int h = t / q4, e = 4 * (t - h * q4);
    const float4 c = *reinterpret_cast<const float4*>(rope_cos + (size_t)pos * half + e);
    const float4 s = *reinterpret_cast<const float4*>(rope_sin + (size_t)pos * half + e);
    const size_t base = (size_t)h * head_dim + e;
    const float4 q1 = sum_splits4(pr, sp, r, base);
    const float4 q2 = sum_splits4(pr, sp, r, base + half);
    const float4 k1 = sum_splits4(pr, sp, r, hidden + base);
    const float4 k2 = sum_splits4(pr, sp, r, hidden + base + half);
    const float4 v1 = sum_splits4(pr, sp, r, 2 * hidden + base);
    const float4 v2 = sum_splits4(pr, sp, r, 2 * hidden + base + half);
    store4<T>(q_out + base, make_float4(q1.x * c.x - q2.x * s.x, q1.y * c.y - q2.y * s.y, q1.z * c.z - q2.z * s.z,
                                        q1.w * c.w - q2.w * s.w));
    store4<T>(q_out + base + half, make_float4(q2.x * c.x + q1.x * s.x, q2.y * c.y + q1.y * s.y,
                                               q2.z * c.z + q1.z * s.z, q2.w * c.w + q1.w * s.w));
    const size_t kv = (size_t)b * kv_seq_stride + ((size_t)h * Tc + pos) * head_dim + e;
    store4<T>(Kc + kv, make_float4(k1.x * c.x - k2.x * s.x, k1.y * c.y - k2.y * s.y, k1.z * c.z - k2.z * s.z,
                                   k1.w * c.w - k2.w * s.w));
    store4<T>(Kc + kv + half, make_float4(k2.x * c.x + k1.x * s.x, k2.y * c.y + k1.y * s.y, k2.z * c.z + k1.z * s.z,
                                          k2.w * c.w + k1.w * s.w));
    store4<T>(Vc + kv, v1);
    store4<T>(Vc + kv + half, v2);
  }
}

// x += o-projection (summed over splits), then A = T(RMSNorm(x) * g).
template <typename T>
__global__ void residual_norm_kernel(Rows rows, int hidden, const float* __restrict__ part, SplitPlan sp,
                                     const T* __restrict__ gain, float eps, T* __restrict__ A) {
  pdl_wait();
  pdl_trigger();
  __shared__ float red[32];
  const int b = blockIdx.y, i = blockIdx.x;
  const int cnt = rows.off[b + 1] - rows.off[b];
  if (i >= cnt) return;
  const int r = rows.off[b] + i;
  float* x = rows.X + ((size_t)b * rows.idx_stride + i) * hidden;
  const float* pr = part + (size_t)r * hidden;
  float ss = 0.f;
#pragma unroll 4
  for (int c = threadIdx.x; c < hidden / 4; c += blockDim.x) {
    const float4 v = add4(reinterpret_cast<const float4*>(x)[c], sum_splits4(pr, sp, r, 4 * (size_t)c));
    reinterpret_cast<float4*>(x)[c] = v;
    ss = sq4(v, ss);
  }
  rmsnorm_row<T>(x, ss, gain, hidden, eps, A + (size_t)r * hidden, red);
}

// G = T(silu(g) * u) from the fused projection [gate | up].
template <typename T>
__global__ void swiglu_kernel(Rows rows, int ffn, const float* __restrict__ part, SplitPlan sp, T* __restrict__ G) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.y, i = blockIdx.x;
  const int cnt = rows.off[b + 1] - rows.off[b];
  if (i >= cnt) return;
  const int r = rows.off[b] + i;
  const float* pr = part + (size_t)r * 2 * ffn;
  // gridDim.z blocks share a row, so that enough loads are in flight
  const int n4 = ffn / 4, c0 = (int)(((long long)n4 * blockIdx.z) / gridDim.z);
  const int c1 = (int)(((long long)n4 * (blockIdx.z + 1)) / gridDim.z);
#pragma unroll 4
  for (int c = c0 + threadIdx.x; c < c1; c += blockDim.x) {
    const float4 g = sum_splits4(pr, sp, r, 4 * (size_t)c);
    const float4 u = sum_splits4(pr, sp, r, (size_t)ffn + 4 * c);
    store4<T>(G + (size_t)r * ffn + 4 * c,
              make_float4((g.x / (1.0f + expf(-g.x))) * u.x, (g.y / (1.0f + expf(-g.y))) * u.y,
                          (g.z / (1.0f + expf(-g.z))) * u.z, (g.w / (1.0f + expf(-g.w))) * u.w));
  }
}

// x += down-projection (summed over splits).
__global__ void residual_kernel(Rows rows, int hidden, const float* __restrict__ part, SplitPlan sp) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.y, i = blockIdx.x;
  const int cnt = rows.off[b + 1] - rows.off[b];
  if (i >= cnt) return;
  const int r = rows.off[b] + i;
  float* x = rows.X + ((size_t)b * rows.idx_stride + i) * hidden;
  const float* pr = part + (size_t)r * hidden;
  // gridDim.z blocks share a row, so that enough loads are in flight
  const int n4 = hidden / 4, c0 = (int)(((long long)n4 * blockIdx.z) / gridDim.z);
  const int c1 = (int)(((long long)n4 * (blockIdx.z + 1)) / gridDim.z);
#pragma unroll 4
  for (int c = c0 + threadIdx.x; c < c1; c += blockDim.x)
    reinterpret_cast<float4*>(x)[c] =
        add4(reinterpret_cast<const float4*>(x)[c], sum_splits4(pr, sp, r, 4 * (size_t)c));
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
// the next step's gate and becomes valid.  The action delta (Sec. VI) is the
// L1 distance in bins to the previous step's ids on the sequence.
__global__ void finish_kernel(int B, int D, const StepParams* __restrict__ prm, const float* __restrict__ margins,
                              const float* __restrict__ gaps, const float* __restrict__ vms,
                              float* __restrict__ m_prev, uint8_t* __restrict__ valid,
                              float* __restrict__ user_step_margin, const int32_t* __restrict__ ids,
                              int32_t* __restrict__ prev_ids, uint8_t* __restrict__ ids_valid,
                              int32_t* __restrict__ delta, const uint8_t* __restrict__ active) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  if (prm->has_active && active && !active[b]) {  // sat the step out: the gate state and ids stay
    user_step_margin[b] = 0.f;
    delta[b] = 0;
    return;
  }
  const float* sig = (prm->margin_kind == VLAC_MARGIN_LOGIT   ? gaps
                      : prm->margin_kind == VLAC_MARGIN_VOCAB ? vms
                                                              : margins) +
                     (size_t)b * D;
  int dl = 0;
  for (int a = 0; a < D; ++a) {
    const int v = ids[(size_t)b * D + a];
    if (ids_valid[b]) dl += abs(v - prev_ids[(size_t)b * D + a]);
    prev_ids[(size_t)b * D + a] = v;
  }
  ids_valid[b] = 1;
  delta[b] = dl;
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

// ---- the one-layer entry ----------------------------------------------------------

__global__ void layer_setup_kernel(const int32_t* __restrict__ pos, int M, int S, int* __restrict__ idx,
                                   int* __restrict__ off, int* err) {
  pdl_wait();
  pdl_trigger();
  for (int i = threadIdx.x; i < M; i += blockDim.x) {
    int p = pos[i];
    if (p < 0 || p >= S) {
      set_error(err, VLAC_ERR_DEVICE_CHECK);
      p = 0;
    }
    idx[i] = p;
  }
  if (threadIdx.x == 0) {
    off[0] = 0;
    off[1] = M;
  }
}

// One block per (position, head): head_dim elements, copied as 4-byte words.
__global__ void kv_copy_kernel(uint8_t* __restrict__ cache, uint8_t* __restrict__ flat, int n_heads, int Tc,
                               int row_bytes, bool to_cache) {
  pdl_wait();
  pdl_trigger();
  const int t = blockIdx.x, h = blockIdx.y;
  uint32_t* cw = reinterpret_cast<uint32_t*>(cache + ((size_t)h * Tc + t) * row_bytes);
  uint32_t* fw = reinterpret_cast<uint32_t*>(flat + ((size_t)t * n_heads + h) * row_bytes);
  for (int w = threadIdx.x; w < row_bytes / 4; w += blockDim.x) {
    if (to_cache)
      cw[w] = fw[w];
    else
      fw[w] = cw[w];
  }
}

void launch_layer_setup(const int32_t* pos, int M, int S, int* idx, int* off, int* err, cudaStream_t st) {
  launch_k(layer_setup_kernel, dim3(1), dim3(256), 0, st, pos, M, S, idx, off, err);
}
void launch_kv_copy(void* cache, void* flat, int n_heads, int Tc, int head_dim, int esz, bool to_cache,
                    cudaStream_t st) {
  launch_k(kv_copy_kernel, dim3(Tc, n_heads), dim3(64), 0, st, static_cast<uint8_t*>(cache),
           static_cast<uint8_t*>(flat), n_heads, Tc, head_dim * esz, to_cache);
}

cudaError_t launch_stage(const StepParams& p, StepParams* prm, const CopyList& list, cudaStream_t st) {
  return launch_k(copy_spans_kernel, dim3(64), dim3(256), 0, st, list, p, prm);
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
  launch_k(layer_in_kernel<T>, dim3(S, B), dim3(kNormThreads), 0, st, rows, off_prev, hidden, H, h_seq_stride, gain, eps, A);
}
template <typename T>
void launch_residual_layer_in(Rows rows, const int* off_prev, int B, int S, int hidden, const float* part,
                              const SplitPlan& sp, float* H, size_t h_seq_stride, const T* gain, float eps, T* A,
                              cudaStream_t st) {
  launch_k(residual_layer_in_kernel<T>, dim3(S, B), dim3(kNormThreads), 0, st, rows, off_prev, hidden, part, sp, H,
           h_seq_stride, gain, eps, A);
}
template <typename T>
void launch_qkv_epilogue(Rows rows, int B, int S, int n_heads, int head_dim, const float* part, const SplitPlan& sp,
                         const float* rope_cos, const float* rope_sin, T* Q, T* Kc, T* Vc, size_t kv_seq_stride,
                         int Tc, cudaStream_t st) {
  launch_k(qkv_epilogue_kernel<T>, dim3(S, B, 2), dim3(256), 0, st, rows, n_heads, head_dim, part, sp, rope_cos,
           rope_sin, Q, Kc, Vc, kv_seq_stride, Tc);
}
template <typename T>
void launch_residual_norm(Rows rows, int B, int S, int hidden, const float* part, const SplitPlan& sp, const T* gain,
                          float eps, T* A, cudaStream_t st) {
  launch_k(residual_norm_kernel<T>, dim3(S, B), dim3(kNormThreads), 0, st, rows, hidden, part, sp, gain, eps, A);
}
template <typename T>
void launch_swiglu(Rows rows, int B, int S, int ffn, const float* part, const SplitPlan& sp, T* G, cudaStream_t st) {
  launch_k(swiglu_kernel<T>, dim3(S, B, 4), dim3(256), 0, st, rows, ffn, part, sp, G);
}
void launch_residual(Rows rows, int B, int S, int hidden, const float* part, const SplitPlan& sp, cudaStream_t st) {
  launch_k(residual_kernel, dim3(S, B, 4), dim3(256), 0, st, rows, hidden, part, sp);
}
template <typename T>
void launch_decode_embed(int B, int d, int D, int P, int hidden, int vocab, int n_bins, const T* tok_emb,
                         const int32_t* ids, const int32_t* forced, const StepParams* prm, float* Xd, int* idx_dec,
                         float* ssq_out, int* err, cudaStream_t st) {
  launch_k(decode_embed_kernel<T>, dim3(B), dim3(256), 0, st, d, D, P, hidden, vocab, n_bins, tok_emb, ids, forced,
           prm, Xd, idx_dec, ssq_out, err);
}
void launch_finish(int B, int D, const StepParams* prm, const float* margins, const float* gaps, const float* vms,
                   float* m_prev, uint8_t* valid, float* user_step_margin, const int32_t* ids, int32_t* prev_ids,
                   uint8_t* ids_valid, int32_t* delta, const uint8_t* active, cudaStream_t st) {
  launch_k(finish_kernel, dim3((B + 63) / 64), dim3(64), 0, st, B, D, prm, margins, gaps, vms, m_prev, valid,
           user_step_margin, ids, prev_ids, ids_valid, delta, active);
}

// Grid (chunks, B): sequence b's previous frame becomes this step's frame (16-byte
// words where both ends allow, bytes otherwise), or, for a sequence that sat
// the step out, its outputs are zeroed.
__global__ void commit_kernel(int D, int n_bins, int Nv, int S, int L, size_t frame_bytes,
                              const uint8_t* __restrict__ frames, uint8_t* __restrict__ prev,
                              const StepParams* __restrict__ prm, const uint8_t* __restrict__ active, StepOutputs o) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.y;
  const size_t tid = (size_t)blockIdx.x * blockDim.x + threadIdx.x, nth = (size_t)gridDim.x * blockDim.x;
  if (!(prm->has_active && active && !active[b])) {
    const uint8_t* src = frames + (size_t)b * frame_bytes;
    uint8_t* dst = prev + (size_t)b * frame_bytes;
    if (((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15) == 0) {
      const size_t nv = frame_bytes / 16;
      for (size_t i = tid; i < nv; i += nth) reinterpret_cast<uint4*>(dst)[i] = reinterpret_cast<const uint4*>(src)[i];
      for (size_t i = nv * 16 + tid; i < frame_bytes; i += nth) dst[i] = src[i];
    } else {
      for (size_t i = tid; i < frame_bytes; i += nth) dst[i] = src[i];
    }
    return;
  }
  for (size_t i = tid; i < (size_t)D; i += nth) {
    o.ids[(size_t)b * D + i] = 0;
    o.margins[(size_t)b * D + i] = 0.f;
    o.gaps[(size_t)b * D + i] = 0.f;
    if (o.entropy) o.entropy[(size_t)b * D + i] = 0.f;
    if (o.vocab_margin) o.vocab_margin[(size_t)b * D + i] = 0.f;
  }
  for (size_t i = tid; i < (size_t)D * n_bins; i += nth) o.logits[(size_t)b * D * n_bins + i] = 0.f;
  for (size_t i = tid; i < (size_t)Nv; i += nth) o.mask[(size_t)b * Nv + i] = 0;
  for (size_t i = tid; i < (size_t)S; i += nth) o.idx[(size_t)b * S + i] = 0;
  for (size_t i = tid; i < (size_t)L; i += nth) o.M[(size_t)b * L + i] = 0;
  for (size_t i = tid; i < (size_t)Nv; i += nth) {
    if (o.relevance) o.relevance[(size_t)b * Nv + i] = 0.f;
    if (o.relevant) o.relevant[(size_t)b * Nv + i] = 0;
  }
  if (tid == 0) {
    o.recomputed[b] = 0;
    o.gate_auto[b] = 0;
    o.step_margin[b] = 0.f;
  }
}

void launch_commit(int B, int D, int n_bins, int Nv, int S, int L, size_t frame_bytes, const uint8_t* frames,
                   uint8_t* prev, const StepParams* prm, const uint8_t* active, const StepOutputs& o,
                   cudaStream_t st) {
  launch_k(commit_kernel, dim3(16, B), dim3(256), 0, st, D, n_bins, Nv, S, L, frame_bytes, frames, prev, prm, active,
           o);
}

#define VLAC_INST(T)                                                                                              \
  template void launch_im2col<T>(Rows, int, int, const uint8_t*, int, int, int, int, int, T*, cudaStream_t);     \
  template void launch_embed<T>(Rows, int, int, int, int, int, int, int, int, int, const int32_t*, const float*, \
                                const T*, const float*, const T*, const T*, int*, cudaStream_t);                 \
  template void launch_layer_in<T>(Rows, const int*, int, int, int, float*, size_t, const T*, float, T*,          \
                                   cudaStream_t);                                                                 \
  template void launch_residual_layer_in<T>(Rows, const int*, int, int, int, const float*, const SplitPlan&,     \
                                            float*, size_t, const T*, float, T*, cudaStream_t);                   \
  template void launch_qkv_epilogue<T>(Rows, int, int, int, int, const float*, const SplitPlan&, const float*,  \
                                       const float*, T*, T*, T*, size_t, int, cudaStream_t);                      \
  template void launch_residual_norm<T>(Rows, int, int, int, const float*, const SplitPlan&, const T*, float, T*, \
                                        cudaStream_t);                                                            \
  template void launch_swiglu<T>(Rows, int, int, int, const float*, const SplitPlan&, T*, cudaStream_t);          \
  template void launch_decode_embed<T>(int, int, int, int, int, int, int, const T*, const int32_t*,               \
                                       const int32_t*, const StepParams*, float*, int*, float*, int*, cudaStream_t);
VLAC_INST(float)
VLAC_INST(bf16)

}  // namespace vlac
