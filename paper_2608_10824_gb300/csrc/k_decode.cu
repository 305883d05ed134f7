// Decode passes of the autoregressive action tokens (Algorithm 1, "decode
// action tokens"): one new row per sequence per pass, so every projection is
// a weight-streaming GEMV.  The GEMVs carry the row-wise work of the layer:
//   - RMSNorm prologue: each CTA normalises the (<= 8) fp32 residual rows
//     into shared memory (the same fixed reduction order in every CTA);
//   - epilogues: RoPE + K/V scatter into the cache, residual add, SwiGLU.
// Attention of the single query per head is split over key chunks and
// combined in a fixed order.  The action head (final norm, bin logits) is a
// multi-CTA GEMV followed by a one-warp top-2 / margin reduction per row.
#include "internal.cuh"

namespace vlac {

namespace {

__device__ __forceinline__ uint4 ld_stream(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

template <typename T> struct Vec;
template <> struct Vec<bf16> { static constexpr int n = 8; };
template <> struct Vec<float> { static constexpr int n = 4; };

template <typename T>
__device__ __forceinline__ void unpack(const uint4& u, float* f) {
  if constexpr (sizeof(T) == 2) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      f[2 * i] = __uint_as_float(w[i] << 16);
      f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
  } else {
    f[0] = __uint_as_float(u.x);
    f[1] = __uint_as_float(u.y);
    f[2] = __uint_as_float(u.z);
    f[3] = __uint_as_float(u.w);
  }
}

__device__ __forceinline__ float warp_allsum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Normalises NB fp32 rows of width K into shared memory as T:
// xs[b][k] = T((x * r_b) * g[k]),  r_b = 1 / sqrt(mean(x_b^2) + eps).
template <typename T, int NB>
__device__ __forceinline__ void norm_rows_to_smem(const float* __restrict__ X, const T* __restrict__ g, int K,
                                                  float eps, T* xs) {
  __shared__ float red[32][NB];
  __shared__ float rr[NB];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  float ss[NB];
#pragma unroll
  for (int b = 0; b < NB; ++b) ss[b] = 0.f;
  for (int k = threadIdx.x; k < K; k += blockDim.x)
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      const float x = X[(size_t)b * K + k];
      ss[b] = fmaf(x, x, ss[b]);
    }
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    const float s = warp_allsum(ss[b]);
    if (lane == 0) red[w][b] = s;
  }
  __syncthreads();
  if (threadIdx.x < NB) {
    float t = 0.f;
    for (int i = 0; i < nw; ++i) t += red[i][threadIdx.x];
    rr[threadIdx.x] = 1.0f / sqrtf(t / (float)K + eps);
  }
  __syncthreads();
  for (int k = threadIdx.x; k < K; k += blockDim.x) {
    const float gk = to_f(g[k]);
#pragma unroll
    for (int b = 0; b < NB; ++b) xs[(size_t)b * K + k] = from_f<T>((X[(size_t)b * K + k] * rr[b]) * gk);
  }
  __syncthreads();
}

}  // namespace

// ---- fused decode GEMV ----------------------------------------------------------

template <typename T, int NB, int EPI, bool NORM, int UNROLL>
__global__ void __launch_bounds__(256) dgemv_kernel(DGemv a) {
  constexpr int V = Vec<T>::n;
  extern __shared__ __align__(16) uint8_t dsm[];
  T* xs = reinterpret_cast<T*>(dsm);
  const int K = a.K;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int p = blockIdx.x * (blockDim.x >> 5) + warp;
  int r1 = 0, r2 = 0;
  int sec = 0, h = 0, e = 0;
  const int hd = a.head_dim, half = hd >> 1;
  if constexpr (EPI == kEpiQkvRope) {
    const int hidden = a.n_heads * hd;
    sec = p / (hidden / 2);
    const int within = p - sec * (hidden / 2);
    h = within / half;
    e = within - h * half;
    r1 = sec * hidden + h * hd + e;
    r2 = r1 + half;
  } else if constexpr (EPI == kEpiSwiglu) {
    r1 = p;
    r2 = a.ffn + p;
  } else {
    r1 = 2 * p;
    r2 = 2 * p + 1;
  }
  // the weight rows do not depend on earlier kernels: start pulling them into
  // L2 while the previous kernel of the stream drains
  if (p < a.n_pairs && lane == 0) {
    prefetch_l2(static_cast<const T*>(a.W) + (size_t)r1 * K, (uint32_t)(K * sizeof(T)));
    prefetch_l2(static_cast<const T*>(a.W) + (size_t)r2 * K, (uint32_t)(K * sizeof(T)));
  }
  pdl_wait();
  pdl_trigger();
  if constexpr (NORM) norm_rows_to_smem<T, NB>(a.X, static_cast<const T*>(a.gain), K, a.eps, xs);
  if (p >= a.n_pairs) return;
  const T* W = static_cast<const T*>(a.W);
  const int kv = K / V;
  const uint4* w1 = reinterpret_cast<const uint4*>(W + (size_t)r1 * K);
  const uint4* w2 = reinterpret_cast<const uint4*>(W + (size_t)r2 * K);
  const uint4* xv = reinterpret_cast<const uint4*>(NORM ? (const T*)xs : static_cast<const T*>(a.xin));
  float acc1[NB], acc2[NB];
#pragma unroll
  for (int b = 0; b < NB; ++b) acc1[b] = acc2[b] = 0.f;
  for (int k0 = lane; k0 < kv; k0 += 32 * UNROLL) {
    uint4 q1[UNROLL], q2[UNROLL];
#pragma unroll
    for (int u = 0; u < UNROLL; ++u) {
      const int k = k0 + u * 32;
      if (k < kv) {
        q1[u] = ld_stream(w1 + k);
        q2[u] = ld_stream(w2 + k);
      }
    }
#pragma unroll
    for (int u = 0; u < UNROLL; ++u) {
      const int k = k0 + u * 32;
      if (k >= kv) break;
      float f1[V], f2[V];
      unpack<T>(q1[u], f1);
      unpack<T>(q2[u], f2);
#pragma unroll
      for (int b = 0; b < NB; ++b) {
        float xf[V];
        uint4 xu;
        if constexpr (NORM) xu = xv[(size_t)b * kv + k];
        else xu = __ldg(xv + (size_t)b * kv + k);
        unpack<T>(xu, xf);
#pragma unroll
        for (int i = 0; i < V; ++i) {
          acc1[b] = fmaf(f1[i], xf[i], acc1[b]);
          acc2[b] = fmaf(f2[i], xf[i], acc2[b]);
        }
      }
    }
  }
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    acc1[b] = warp_allsum(acc1[b]);
    acc2[b] = warp_allsum(acc2[b]);
  }
  if (lane >= NB) return;
  // lane b writes sequence b
  float y1 = acc1[0], y2 = acc2[0];
#pragma unroll
  for (int b = 1; b < NB; ++b)
    if (lane == b) {
      y1 = acc1[b];
      y2 = acc2[b];
    }
  const int b = lane;
  if constexpr (EPI == kEpiQkvRope) {
    const int hidden = a.n_heads * hd;
    float o1 = y1, o2 = y2;
    if (sec < 2) {
      const float c = a.rope_cos[(size_t)a.pos * half + e], s = a.rope_sin[(size_t)a.pos * half + e];
      o1 = y1 * c - y2 * s;
      o2 = y2 * c + y1 * s;
    }
    if (sec == 0) {
      T* q = static_cast<T*>(a.Q) + (size_t)b * hidden + (size_t)h * hd;
      q[e] = from_f<T>(o1);
      q[e + half] = from_f<T>(o2);
    } else {
      T* c = static_cast<T*>(sec == 1 ? a.Kc : a.Vc) + (size_t)b * a.kv_seq_stride +
             ((size_t)h * a.Tc + a.pos) * hd;
      c[e] = from_f<T>(o1);
      c[e + half] = from_f<T>(o2);
    }
  } else if constexpr (EPI == kEpiSwiglu) {
    static_cast<T*>(a.G)[(size_t)b * a.ffn + p] = from_f<T>((y1 / (1.0f + expf(-y1))) * y2);
  } else {
    float* x = a.Xres + (size_t)b * a.n_out;
    x[r1] += y1;
    x[r2] += y2;
  }
}

template <typename T, int NB, int EPI, bool NORM>
static void dgemv_nb(const DGemv& a, cudaStream_t st) {
  const int warps = 8;
  const int blocks = (a.n_pairs + warps - 1) / warps;
  const size_t smem = NORM ? (size_t)NB * a.K * sizeof(T) : 0;
  constexpr int U = NB <= 2 ? 4 : 2;
  static size_t smem_set = 48 * 1024;  // raised once per instantiation, before any graph capture of it
  if (smem > smem_set) {
    cudaFuncSetAttribute(dgemv_kernel<T, NB, EPI, NORM, U>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    smem_set = smem;
  }
  launch_k(dgemv_kernel<T, NB, EPI, NORM, U>, dim3(blocks), dim3(warps * 32), smem, st, a);
}

template <typename T, int EPI, bool NORM>
static void dgemv_dispatch(const DGemv& a, int nb, cudaStream_t st) {
  switch (nb) {
    case 1: dgemv_nb<T, 1, EPI, NORM>(a, st); break;
    case 2: dgemv_nb<T, 2, EPI, NORM>(a, st); break;
    case 3: dgemv_nb<T, 3, EPI, NORM>(a, st); break;
    case 4: dgemv_nb<T, 4, EPI, NORM>(a, st); break;
    case 5: dgemv_nb<T, 5, EPI, NORM>(a, st); break;
    case 6: dgemv_nb<T, 6, EPI, NORM>(a, st); break;
    case 7: dgemv_nb<T, 7, EPI, NORM>(a, st); break;
    default: dgemv_nb<T, 8, EPI, NORM>(a, st); break;
  }
}

template <typename T>
void launch_dgemv(const DGemv& a, int epi, int nb, cudaStream_t st) {
  switch (epi) {
    case kEpiQkvRope: dgemv_dispatch<T, kEpiQkvRope, true>(a, nb, st); break;
    case kEpiSwiglu: dgemv_dispatch<T, kEpiSwiglu, true>(a, nb, st); break;
    default: dgemv_dispatch<T, kEpiResid, false>(a, nb, st); break;
  }
}
template void launch_dgemv<float>(const DGemv&, int, int, cudaStream_t);
template void launch_dgemv<bf16>(const DGemv&, int, int, cudaStream_t);

// ---- decode attention: one query per (sequence, head) ----------------------------

// Partial softmax of one 32-key chunk: m = max score, l = sum exp(s - m),
// acc = sum exp(s - m) * v.  Lane holds elements [lane*EPL, lane*EPL + EPL).
template <typename T, int HD>
__global__ void __launch_bounds__(32) dec_attn_partial_kernel(const T* __restrict__ Q, const T* __restrict__ Kc,
                                                              const T* __restrict__ Vc, size_t kv_seq_stride, int Tc,
                                                              int pos, int n_heads, float scale,
                                                              float* __restrict__ part, int nchunk) {
  pdl_wait();
  pdl_trigger();
  constexpr int EPL = HD / 32;
  const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z, lane = threadIdx.x;
  const int hidden = n_heads * HD;
  float q[EPL];
#pragma unroll
  for (int i = 0; i < EPL; ++i) q[i] = to_f(Q[(size_t)b * hidden + (size_t)h * HD + lane * EPL + i]);
  const T* Kh = Kc + (size_t)b * kv_seq_stride + (size_t)h * Tc * HD;
  const T* Vh = Vc + (size_t)b * kv_seq_stride + (size_t)h * Tc * HD;
  const int j0 = c * 32, j1 = min(j0 + 32, pos + 1);
  float s_mine = -INFINITY;  // lane j keeps the score of key j0 + j
  for (int j = j0; j < j1; ++j) {
    float d = 0.f;
#pragma unroll
    for (int i = 0; i < EPL; ++i) d = fmaf(q[i], to_f(Kh[(size_t)j * HD + lane * EPL + i]), d);
    d = warp_allsum(d) * scale;
    if (lane == j - j0) s_mine = d;
  }
  float m = s_mine;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  const float pj = (s_mine == -INFINITY) ? 0.f : expf(s_mine - m);
  const float l = warp_allsum(pj);
  float acc[EPL];
#pragma unroll
  for (int i = 0; i < EPL; ++i) acc[i] = 0.f;
  for (int j = j0; j < j1; ++j) {
    const float p = __shfl_sync(0xffffffffu, pj, j - j0);
#pragma unroll
    for (int i = 0; i < EPL; ++i) acc[i] = fmaf(p, to_f(Vh[(size_t)j * HD + lane * EPL + i]), acc[i]);
  }
  float* o = part + (((size_t)b * n_heads + h) * nchunk + c) * (HD + 2);
#pragma unroll
  for (int i = 0; i < EPL; ++i) o[lane * EPL + i] = acc[i];
  if (lane == 0) {
    o[HD] = m;
    o[HD + 1] = l;
  }
}

// Combines the chunks of one (sequence, head) in chunk order.
template <typename T, int HD>
__global__ void __launch_bounds__(HD) dec_attn_combine_kernel(const float* __restrict__ part, int nchunk,
                                                              int n_heads, T* __restrict__ O) {
  pdl_wait();
  pdl_trigger();
  const int h = blockIdx.x, b = blockIdx.y, e = threadIdx.x;
  const float* base = part + ((size_t)b * n_heads + h) * nchunk * (HD + 2);
  float M = -INFINITY;
  for (int c = 0; c < nchunk; ++c) M = fmaxf(M, base[(size_t)c * (HD + 2) + HD]);
  float L = 0.f, acc = 0.f;
  for (int c = 0; c < nchunk; ++c) {
    const float* pc = base + (size_t)c * (HD + 2);
    const float f = expf(pc[HD] - M);
    L = fmaf(pc[HD + 1], f, L);
    acc = fmaf(pc[e], f, acc);
  }
  O[(size_t)b * n_heads * HD + (size_t)h * HD + e] = from_f<T>(acc / L);
}

template <typename T>
void launch_dec_attention(int B, int n_heads, int head_dim, const T* Q, const T* Kc, const T* Vc, size_t kv_seq_stride,
                          int Tc, int pos, float* part, T* O, cudaStream_t st) {
  const int nchunk = (pos + 1 + 31) / 32;
  const float scale = 1.0f / sqrtf((float)head_dim);
  if (head_dim == 128) {
    launch_k(dec_attn_partial_kernel<T, 128>, dim3(nchunk, n_heads, B), dim3(32), 0, st, Q, Kc, Vc, kv_seq_stride,
             Tc, pos, n_heads, scale, part, nchunk);
    launch_k(dec_attn_combine_kernel<T, 128>, dim3(n_heads, B), dim3(128), 0, st, part, nchunk, n_heads, O);
  } else {
    launch_k(dec_attn_partial_kernel<T, 64>, dim3(nchunk, n_heads, B), dim3(32), 0, st, Q, Kc, Vc, kv_seq_stride,
             Tc, pos, n_heads, scale, part, nchunk);
    launch_k(dec_attn_combine_kernel<T, 64>, dim3(n_heads, B), dim3(64), 0, st, part, nchunk, n_heads, O);
  }
}
template void launch_dec_attention<float>(int, int, int, const float*, const float*, const float*, size_t, int, int,
                                          float*, float*, cudaStream_t);
template void launch_dec_attention<bf16>(int, int, int, const bf16*, const bf16*, const bf16*, size_t, int, int,
                                         float*, bf16*, cudaStream_t);

// ---- action head -------------------------------------------------------------------

// Bin logits of one action row: final RMSNorm (into shared memory as T), then
// 16 bins per CTA, two per warp.  Rows of sequence b are
// X + b * x_seq_stride + (row_of_seq[b] + j) * hidden (row_of_seq NULL = row j).
template <typename T>
__global__ void __launch_bounds__(256) head_logits_kernel(const float* __restrict__ X, const int* __restrict__ row_of_seq,
                                                          size_t x_seq_stride, int hidden, int n_bins,
                                                          const T* __restrict__ final_norm,
                                                          const T* __restrict__ head_w, float eps,
                                                          float* __restrict__ logits_ws) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ __align__(16) uint8_t dsm[];
  T* xs = reinterpret_cast<T*>(dsm);
  const int j = blockIdx.y, b = blockIdx.z;
  const int row = row_of_seq ? row_of_seq[b] + j : j;
  const float* x = X + (size_t)b * x_seq_stride + (size_t)row * hidden;
  norm_rows_to_smem<T, 1>(x, final_norm, hidden, eps, xs);
  constexpr int V = Vec<T>::n;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c1 = blockIdx.x * 16 + warp * 2, c2 = c1 + 1;
  const int kv = hidden / V;
  const uint4* w1 = reinterpret_cast<const uint4*>(head_w + (size_t)c1 * hidden);
  const uint4* w2 = reinterpret_cast<const uint4*>(head_w + (size_t)c2 * hidden);
  const uint4* xv = reinterpret_cast<const uint4*>(xs);
  float a1 = 0.f, a2 = 0.f;
  for (int k = lane; k < kv; k += 32) {
    float f1[V], f2[V], xf[V];
    unpack<T>(__ldg(w1 + k), f1);
    unpack<T>(__ldg(w2 + k), f2);
    unpack<T>(xv[k], xf);
#pragma unroll
    for (int i = 0; i < V; ++i) {
      a1 = fmaf(f1[i], xf[i], a1);
      a2 = fmaf(f2[i], xf[i], a2);
    }
  }
  a1 = warp_allsum(a1);
  a2 = warp_allsum(a2);
  if (lane == 0) {
    float* lg = logits_ws + ((size_t)b * gridDim.y + j) * n_bins;
    lg[c1] = a1;
    lg[c2] = a2;
  }
}

// argmax (lowest bin on ties), top-2 logit gap and p1 - p2 of one row.
__global__ void __launch_bounds__(32) head_margin_kernel(const float* __restrict__ logits_ws, int n_bins, int D, int tok0,
                                                         int32_t* __restrict__ ids, float* __restrict__ margins,
                                                         float* __restrict__ gaps, float* __restrict__ logits) {
  pdl_wait();
  pdl_trigger();
  const int j = blockIdx.x, b = blockIdx.y, lane = threadIdx.x;
  const float* lg = logits_ws + ((size_t)b * gridDim.x + j) * n_bins;
  float bv = -INFINITY;
  int bi = 0x7fffffff;
  for (int c = lane; c < n_bins; c += 32)
    if (lg[c] > bv) {
      bv = lg[c];
      bi = c;
    }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
    const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
    if (ov > bv || (ov == bv && oi < bi)) {
      bv = ov;
      bi = oi;
    }
  }
  float v2 = -INFINITY, z = 0.f;
  for (int c = lane; c < n_bins; c += 32) {
    if (c != bi) v2 = fmaxf(v2, lg[c]);
    z += expf(lg[c] - bv);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v2 = fmaxf(v2, __shfl_xor_sync(0xffffffffu, v2, o));
  z = warp_allsum(z);
  const size_t t = (size_t)b * D + tok0 + j;
  if (lane == 0) {
    ids[t] = bi;
    margins[t] = -expm1f(v2 - bv) / z;
    gaps[t] = bv - v2;
  }
  if (logits)
    for (int c = lane; c < n_bins; c += 32) logits[t * n_bins + c] = lg[c];
}

template <typename T>
void launch_head2(const float* X, const int* row_of_seq, size_t x_seq_stride, int rows_per_seq, int B, int hidden,
                  int n_bins, const T* final_norm, const T* head_w, float eps, float* logits_ws, int D, int tok0,
                  int32_t* ids, float* margins, float* gaps, float* logits, cudaStream_t st) {
  const size_t smem = (size_t)hidden * sizeof(T);
  launch_k(head_logits_kernel<T>, dim3(n_bins / 16, rows_per_seq, B), dim3(256), smem, st, X, row_of_seq,
           x_seq_stride, hidden, n_bins, final_norm, head_w, eps, logits_ws);
  launch_k(head_margin_kernel, dim3(rows_per_seq, B), dim3(32), 0, st, logits_ws, n_bins, D, tok0, ids, margins, gaps,
           logits);
}
template void launch_head2<float>(const float*, const int*, size_t, int, int, int, int, const float*, const float*,
                                  float, float*, int, int, int32_t*, float*, float*, float*, cudaStream_t);
template void launch_head2<bf16>(const float*, const int*, size_t, int, int, int, int, const bf16*, const bf16*,
                                 float, float*, int, int, int32_t*, float*, float*, float*, cudaStream_t);

}  // namespace vlac
