// Causal attention of the recomputed rows over the mixed (reused + fresh) KV
// cache of their layer: Algorithm 1's partial forward attends every cached
// position j <= pos, whether the K/V of j were reused from an earlier frame or
// recomputed this step.  Rows of a parallel action block see the whole prefix
// and the whole block.
//
// One block per (16 query rows of one sequence, head).  K/V tiles of 32 keys,
// aligned to absolute positions, are staged in shared memory; each warp runs
// an online softmax (fp32) for two query rows.  A row's result depends only
// on its own query and the cache, never on which other rows share the block.
#include "internal.cuh"

namespace vlac {

template <typename T, int HD>
__global__ void __launch_bounds__(256) attn_kernel(Rows rows, int n_heads, const T* __restrict__ Q,
                                                   const T* __restrict__ Kc, const T* __restrict__ Vc,
                                                   size_t kv_seq_stride, int Tc, int P, int parallel, int n_action,
                                                   float scale, T* __restrict__ O) {
  pdl_wait();
  pdl_trigger();
  constexpr int QT = 16, KT = 32, NC = HD / 32;
  __shared__ float Kt[HD][KT + 1];  // padded: conflict-free transposed stores
  __shared__ float Vs[KT][HD];
  __shared__ float Qs[QT][HD];
  __shared__ int lim[QT];
  __shared__ int s_maxlim;
  const int qt = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int cnt = rows.off[b + 1] - rows.off[b];
  const int i0 = qt * QT;
  if (i0 >= cnt) return;
  const int nq = min(QT, cnt - i0);
  const int hidden = n_heads * HD;
  const int r0 = rows.off[b] + i0;
  for (int t = threadIdx.x; t < QT * HD; t += blockDim.x) {
    const int qi = t / HD, e = t - qi * HD;
    Qs[qi][e] = qi < nq ? to_f(Q[(size_t)(r0 + qi) * hidden + (size_t)h * HD + e]) : 0.f;
  }
  if (threadIdx.x < QT) {
    const int qi = threadIdx.x;
    int l = 0;
    if (qi < nq) {
      const int pos = rows.idx[(size_t)b * rows.idx_stride + i0 + qi];
      l = (parallel && pos >= P) ? P + n_action : pos + 1;
      l = min(l, Tc);
    }
    lim[qi] = l;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int m = 0;
    for (int q = 0; q < QT; ++q) m = max(m, lim[q]);
    s_maxlim = m;
  }
  __syncthreads();
  const int maxlim = s_maxlim;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const T* Kh = Kc + (size_t)b * kv_seq_stride + (size_t)h * Tc * HD;
  const T* Vh = Vc + (size_t)b * kv_seq_stride + (size_t)h * Tc * HD;

  float m_run[2], l_run[2], acc[2][NC];
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    m_run[s] = -INFINITY;
    l_run[s] = 0.f;
#pragma unroll
    for (int c = 0; c < NC; ++c) acc[s][c] = 0.f;
  }

  for (int t0 = 0; t0 < maxlim; t0 += KT) {
    for (int t = threadIdx.x; t < KT * HD; t += blockDim.x) {
      const int j = t / HD, e = t - j * HD;
      const int key = t0 + j;
      float kv = 0.f, vv = 0.f;
      if (key < Tc) {
        kv = to_f(Kh[(size_t)key * HD + e]);
        vv = to_f(Vh[(size_t)key * HD + e]);
      }
      Kt[e][j] = kv;
      Vs[j][e] = vv;
    }
    __syncthreads();
#pragma unroll
    for (int s = 0; s < 2; ++s) {
      const int q = warp * 2 + s;
      if (q >= nq) continue;
      float sc = 0.f;
#pragma unroll 8
      for (int e = 0; e < HD; ++e) sc = fmaf(Qs[q][e], Kt[e][lane], sc);
      sc *= scale;
      if (t0 + lane >= lim[q]) sc = -INFINITY;
      const float mt = warp_max(sc);
      const float m_new = fmaxf(m_run[s], mt);
      const float p = (sc == -INFINITY) ? 0.f : expf(sc - m_new);
      const float corr = (m_run[s] == -INFINITY) ? 0.f : expf(m_run[s] - m_new);
      l_run[s] = l_run[s] * corr + warp_sum(p);
#pragma unroll
      for (int c = 0; c < NC; ++c) acc[s][c] *= corr;
#pragma unroll 4
      for (int jj = 0; jj < KT; ++jj) {
        const float pj = __shfl_sync(0xffffffffu, p, jj);
#pragma unroll
        for (int c = 0; c < NC; ++c) acc[s][c] = fmaf(pj, Vs[jj][lane + 32 * c], acc[s][c]);
      }
      m_run[s] = m_new;
    }
    __syncthreads();
  }
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    const int q = warp * 2 + s;
    if (q >= nq) continue;
    T* o = O + (size_t)(r0 + q) * hidden + (size_t)h * HD;
#pragma unroll
    for (int c = 0; c < NC; ++c) o[lane + 32 * c] = from_f<T>(acc[s][c] / l_run[s]);
  }
}

template <typename T>
void launch_attention(Rows rows, int B, int S, int n_heads, int head_dim, const T* Q, const T* Kc, const T* Vc,
                      size_t kv_seq_stride, int Tc, int P, int parallel, int n_action, T* O, cudaStream_t st) {
  dim3 grid((S + 15) / 16, n_heads, B);
  const float scale = 1.0f / sqrtf((float)head_dim);
  if (head_dim == 128)
    launch_k(attn_kernel<T, 128>, grid, dim3(256), 0, st, rows, n_heads, Q, Kc, Vc, kv_seq_stride, Tc, P, parallel,
             n_action, scale, O);
  else
    launch_k(attn_kernel<T, 64>, grid, dim3(256), 0, st, rows, n_heads, Q, Kc, Vc, kv_seq_stride, Tc, P, parallel,
             n_action, scale, O);
}

template void launch_attention<float>(Rows, int, int, int, int, const float*, const float*, const float*, size_t,
                                      int, int, int, int, float*, cudaStream_t);
template void launch_attention<bf16>(Rows, int, int, int, int, const bf16*, const bf16*, const bf16*, size_t, int,
                                     int, int, int, bf16*, cudaStream_t);

}  // namespace vlac
