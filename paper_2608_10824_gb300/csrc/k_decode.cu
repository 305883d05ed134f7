// Decode passes of the autoregressive action tokens (Algorithm 1, "decode
// action tokens"): one new row per sequence per pass, so every projection is
// a weight-streaming GEMV.  The GEMVs carry the row-wise work of the layer:
//   - RMSNorm prologue: each CTA normalises the (<= 8) fp32 residual rows
//     into shared memory (the same fixed reduction order in every CTA);
//   - epilogues: RoPE + K/V scatter into the cache, residual add, SwiGLU.
// Attention of the single query per head is split over key chunks and
// combined in a fixed order.  The action head (final norm, bin logits) is a
// multi-CTA GEMV followed by a one-warp top-2 / margin reduction per row.
#include <cooperative_groups.h>

#include <algorithm>
#include <type_traits>

#include "internal.cuh"

namespace vlac {

namespace {

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
//
// Weight layout for decode streaming (built once at create time): output row
// pairs are grouped 4 at a time (8 weight rows); a group's K range is cut into
// chunks of kDecTileB bytes per row; the tile [8 rows][chunk] is contiguous,
// and the tiles of a group follow each other, then the next group.  Pair p's
// rows:
//   QKV:     (i, i + head_dim/2) of one head of q, k or v;
//   SwiGLU:  (gate j, up j);
//   other:   (2p, 2p + 1).
// Inside a bf16 tile the 8 rows are interleaved in steps of 8 elements
// ([k/8][row][k%8]): the 8 rows of one 8-element K step are 128 contiguous
// bytes, so one ldmatrix.x4 reads 8 rows x 32 K without bank conflicts and
// hands every lane its B fragment of two m16n8k16 products.  fp32 tiles stay
// row-major ([row][k]).
//
// Persistent GEMV: one CTA per SM owns a contiguous, balanced range of groups
// and so one contiguous region of the tiled weights.  A producer warp streams
// it tile by tile into a ring of shared-memory stages with 1-D bulk copies;
// the producer starts before the dependency wait (weights are constant), so a
// kernel's first stages stream in while its predecessor drains.
//
// bf16 consumers (8 warps): warp w takes the w-th eighth of every tile's K
// range, for all 8 rows, on the tensor pipe: the weights are the B operand
// (n = row), the input vectors the A operand (m = sequence, rows >= NB zero),
// so D[b][row] accumulates y_b over the warp's K range in fp32.  The products
// are exact and the adds are fp32, as in a scalar dot product; the tensor
// path only removes the unpacking and multiply-add instructions that
// otherwise bound the consumers below the stream rate.  At the end of a group
// the 8 warps' partials are added in warp (K) order by one warp, which
// rotates from group to group, and it runs the epilogue.  fp32 consumers run
// the scalar loop: warp w handles pair w/2 over one half of each tile's K.
//
// RMSNorm without a second pass over the row: every residual-writing GEMV
// (and the decode embedding) stores per CTA and sequence the sum of squares
// of the residual elements it produced; a normalising GEMV sums those
// partials in index order for the mean square and normalises the input
// vector once into shared memory (x * r * g rounded to T).  bf16 vectors are
// kept in A-fragment order: per 32-element K step and lane t the elements
// (2t, 2t+1, 2t+8, 2t+9, 2t+16, 2t+17, 2t+24, 2t+25), one 16-byte load.
//
// Every ring wait is bounded (a.wait_limit polls).  A wait that gives up
// latches VLAC_ERR_TIMEOUT and raises the CTA's give-up flag: the producer
// stops issuing; the consumers run out their loops without computing or
// handing stages back, so they stay in step at the named barriers; and a
// consumer that gave up waits (bounded) for the producer's copies still
// landing before the CTA exits.

constexpr int kNC = 8;          // consumer warps
constexpr int kGP = kDecGroupPairs;      // row pairs per group
constexpr int kMaxNS = 24;               // stage ring capacity
constexpr int kDecTileB = kDecTileBytes; // bytes of one tile row (K chunk)

__host__ __device__ inline size_t sgemv_xs_bytes(int nb, int K, int esz) {
  return ((size_t)nb * K * esz + 1023) / 1024 * 1024;
}


template <int EPI>
__host__ __device__ __forceinline__ void dec_pair_rows(int p, int n_heads, int head_dim, int ffn, int& r1, int& r2) {
  if (EPI == kEpiQkvRope) {
    const int half = head_dim >> 1, hidden = n_heads * head_dim;
    const int sec = p / (hidden / 2), within = p - sec * (hidden / 2);
    const int h = within / half, e = within - h * half;
    r1 = sec * hidden + h * head_dim + e;
    r2 = r1 + half;
  } else if (EPI == kEpiSwiglu) {
    r1 = p;
    r2 = ffn + p;
  } else {
    r1 = 2 * p;
    r2 = 2 * p + 1;
  }
}

// Builds the tiled copy: one block per (group, tile row).
template <typename T, int EPI>
__global__ void tile_decode_weights_kernel(const T* __restrict__ W, int K, int n_pairs, int n_heads, int head_dim,
                                           int ffn, T* __restrict__ out) {
  constexpr int TR = 2 * kGP;
  const int KC = kDecTileB / (int)sizeof(T);
  const int g = blockIdx.x, r = blockIdx.y;  // r: 0 .. TR-1
  const int p = g * kGP + r / 2;
  int r1 = 0, r2 = 0;
  if (p < n_pairs) dec_pair_rows<EPI>(p, n_heads, head_dim, ffn, r1, r2);
  const T* src = W + (size_t)((r & 1) ? r2 : r1) * K;
  T* base = out + (size_t)g * TR * K;
  for (int k = threadIdx.x; k < K; k += blockDim.x) {
    const int c = k / KC, kk = k - c * KC, kn = min(KC, K - c * KC);
    const size_t at = sizeof(T) == 2 ? (size_t)((kk >> 3) * TR + r) * 8 + (kk & 7) : (size_t)r * kn + kk;
    base[(size_t)TR * c * KC + at] = p < n_pairs ? src[k] : from_f<T>(0.f);
  }
}

template <typename T>
void launch_tile_decode_weights(const T* W, int K, int n_pairs, int epi, int n_heads, int head_dim, int ffn, T* out,
                                cudaStream_t st) {
  const int n_groups = (n_pairs + kGP - 1) / kGP;
  dim3 grid(n_groups, 2 * kGP);
  if (epi == kEpiQkvRope)
    tile_decode_weights_kernel<T, kEpiQkvRope><<<grid, 256, 0, st>>>(W, K, n_pairs, n_heads, head_dim, ffn, out);
  else if (epi == kEpiSwiglu)
    tile_decode_weights_kernel<T, kEpiSwiglu><<<grid, 256, 0, st>>>(W, K, n_pairs, n_heads, head_dim, ffn, out);
  else
    tile_decode_weights_kernel<T, kEpiResid><<<grid, 256, 0, st>>>(W, K, n_pairs, n_heads, head_dim, ffn, out);
}
template void launch_tile_decode_weights<float>(const float*, int, int, int, int, int, int, float*, cudaStream_t);
template void launch_tile_decode_weights<bf16>(const bf16*, int, int, int, int, int, int, bf16*, cudaStream_t);
size_t tiled_decode_elems(int K, int n_pairs) { return (size_t)((n_pairs + kGP - 1) / kGP) * 2 * kGP * K; }
size_t dgemv_stage_bytes() { return (size_t)2 * kGP * kDecTileB; }

// Epilogue of one output row pair (p) of sequence b: y1, y2 are the two rows'
// dot products; e1, e2 the operands loaded ahead (RoPE cos/sin, or the two
// residual elements).  Returns the residual epilogue's sum of squares.
template <typename T, int EPI>
__device__ __forceinline__ float dgemv_epilogue(const DGemv& a, int p, int b, float y1, float y2, float e1, float e2) {
  if constexpr (EPI == kEpiQkvRope) {
    const int hd = a.head_dim, half = hd >> 1, hidden = a.n_heads * hd;
    const int sec = p / (hidden / 2), within = p - sec * (hidden / 2);
    const int h = within / half, e = within - h * half;
    float o1 = y1, o2 = y2;
    if (sec < 2) {
      o1 = y1 * e1 - y2 * e2;  // (cos, sin) of the pair's RoPE angle
      o2 = y2 * e1 + y1 * e2;
    }
    T* dst = sec == 0 ? static_cast<T*>(a.Q) + (size_t)b * hidden + (size_t)h * hd
                      : static_cast<T*>(sec == 1 ? a.Kc : a.Vc) + (size_t)b * a.kv_seq_stride +
                            ((size_t)h * a.Tc + a.pos) * hd;
    dst[e] = from_f<T>(o1);
    dst[e + half] = from_f<T>(o2);
    return 0.f;
  } else if constexpr (EPI == kEpiSwiglu) {
    static_cast<T*>(a.G)[(size_t)b * a.ffn + p] = from_f<T>((y1 / (1.0f + expf(-y1))) * y2);
    return 0.f;
  } else {
    float* x = a.Xres + (size_t)b * a.n_out;
    const float n1 = e1 + y1, n2 = e2 + y2;
    x[2 * p] = n1;
    x[2 * p + 1] = n2;
    return fmaf(n1, n1, n2 * n2);
  }
}

template <typename T, int EPI>
__device__ __forceinline__ void dgemv_epilogue_operands(const DGemv& a, int p, int b, float& e1, float& e2) {
  e1 = e2 = 0.f;
  if constexpr (EPI == kEpiQkvRope) {
    const int hd = a.head_dim, half = hd >> 1, hidden = a.n_heads * hd;
    const int sec = p / (hidden / 2), within = p - sec * (hidden / 2);
    const int e = within - (within / half) * half;
    if (sec < 2) {
      e1 = a.rope_cos[(size_t)a.pos * half + e];
      e2 = a.rope_sin[(size_t)a.pos * half + e];
    }
  } else if constexpr (EPI == kEpiResid) {
    e1 = a.Xres[(size_t)b * a.n_out + 2 * p];
    e2 = a.Xres[(size_t)b * a.n_out + 2 * p + 1];
  }
}

__device__ __forceinline__ uint32_t ldg_u32(const void* p) { return __ldg(static_cast<const unsigned int*>(p)); }

template <typename T, int NB, int EPI, bool NORM, bool XG>
__global__ void __launch_bounds__((kNC + 1) * 32, 1) dgemv_kernel(DGemv a) {
  constexpr bool kMma = sizeof(T) == 2;
  constexpr int V = Vec<T>::n;
  constexpr int KC = kDecTileB / (int)sizeof(T);
  constexpr int TR = 2 * kGP;  // tile rows
  const int NS = a.ns;
  const size_t stage_b = (size_t)TR * kDecTileB;
  extern __shared__ __align__(1024) uint8_t dsm[];
  __shared__ __align__(8) uint64_t full_bar[kMaxNS];
  __shared__ __align__(8) uint64_t empty_bar[kMaxNS];
  __shared__ float red[kNC][32];
  __shared__ float rr[NB];
  __shared__ __align__(8) float2 pacc[2][kNC][32];  // bf16 path: per-warp partials, two groups in flight
  __shared__ float half_acc[kGP][2][NB];            // fp32 path: the second K half of every pair
  __shared__ int abort_flag;
  __shared__ __align__(8) uint64_t done_bar;  // the producer has issued its last copy
  __shared__ uint32_t prod_end[3];             // its ring stage, phase and copy count at that point
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int K = a.K, nchunk = (K + KC - 1) / KC;
  const int G = (a.n_pairs + kGP - 1) / kGP;
  int g0, g1;
  dgemv_group_range(G, gridDim.x, blockIdx.x, g0, g1);
  T* xs = reinterpret_cast<T*>(dsm);
  uint8_t* stages = dsm + (XG ? 0 : sgemv_xs_bytes(NB, K, (int)sizeof(T)));
  const T* Wt = static_cast<const T*>(a.W);
  if (threadIdx.x == 0) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], kNC);
    }
    mbar_init(&done_bar, 1);
    abort_flag = 0;
    mbar_fence_init();
  }
  __syncthreads();
  volatile int* abort = &abort_flag;

  if (warp == kNC) {
    // ---- producer: weights only, so it runs ahead of the dependency wait ----
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, issued = 0;
      for (int g = g0; g < g1 && !*abort; ++g) {
        const T* gbase = Wt + (size_t)g * TR * K;
        for (int c = 0; c < nchunk; ++c) {
          const int kn = min(KC, K - c * KC);
          if (!mbar_wait(&empty_bar[stage], phase ^ 1u, a.wait_limit, abort)) {
            set_error(a.err, VLAC_ERR_TIMEOUT);
            *abort = 1;
            break;
          }
          const uint32_t bytes = (uint32_t)(TR * kn * sizeof(T));
          mbar_expect_tx(&full_bar[stage], bytes);
          bulk_g2s(stages + (size_t)stage * stage_b, gbase + (size_t)TR * c * KC, bytes, &full_bar[stage]);
          ++issued;
          if (++stage == NS) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      prod_end[0] = (uint32_t)stage;
      prod_end[1] = phase;
      prod_end[2] = issued;
      mbar_arrive(&done_bar);  // release: the consumers that gave up read prod_end after it
      // the next GEMV's weights do not depend on anything: pull the start of
      // the region its CTA of this index will stream into L2 now
      if (a.pf_W && (int)blockIdx.x < a.pf_grid) {
        const int Gn = (a.pf_pairs + kGP - 1) / kGP;
        int n0, n1;
        dgemv_group_range(Gn, a.pf_grid, blockIdx.x, n0, n1);
        const size_t gbytes = (size_t)TR * a.pf_K * sizeof(T);
        const uint8_t* base = static_cast<const uint8_t*>(a.pf_W) + (size_t)n0 * gbytes;
        size_t left = min((size_t)a.pf_bytes, (size_t)(n1 - n0) * gbytes);
        for (size_t off = 0; left > 0;) {
          const uint32_t piece = (uint32_t)min(left, (size_t)65536);
          prefetch_l2(base + off, piece);
          off += piece;
          left -= piece;
        }
      }
    }
    pdl_wait();
    pdl_trigger();
    return;
  }

  // ---- consumers ----
  pdl_wait();
  pdl_trigger();
  const int tid = threadIdx.x;  // 0 .. kNC*32-1
  if constexpr (NORM) {
    const T* gn = static_cast<const T*>(a.gain);
    // bf16: the first items of the vector are loaded together with the
    // sums-of-squares partials, so that the prologue costs one round trip
    constexpr int kPre = 2;  // items (8 elements) per thread loaded ahead
    const int n8 = K / 8;
    uint4 pg[kPre];
    float4 px0[kPre], px1[kPre];
    if constexpr (kMma) {
#pragma unroll
      for (int j = 0; j < kPre; ++j) {
        const int m = tid + j * kNC * 32;
        if (m < NB * n8) {
          const int b = m / n8, k = (m - b * n8) * 8;
          pg[j] = *reinterpret_cast<const uint4*>(gn + k);
          px0[j] = *reinterpret_cast<const float4*>(a.X + (size_t)b * K + k);
          px1[j] = *reinterpret_cast<const float4*>(a.X + (size_t)b * K + k + 4);
        }
      }
    }
    float sacc[NB];
#pragma unroll
    for (int b = 0; b < NB; ++b) sacc[b] = 0.f;
    for (int c = tid; c < a.n_ssq; c += kNC * 32)
#pragma unroll
      for (int b = 0; b < NB; ++b) sacc[b] += a.ssq_in[(size_t)b * a.n_ssq + c];
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      const float t = warp_allsum(sacc[b]);
      if (lane == 0) red[warp][b] = t;
    }
    asm volatile("bar.sync 1, %0;" ::"r"(kNC * 32));
    if (tid < NB) {
      float t = 0.f;
      for (int w = 0; w < kNC; ++w) t += red[w][tid];
      rr[tid] = 1.0f / sqrtf(t / (float)K + a.eps);
    }
    asm volatile("bar.sync 1, %0;" ::"r"(kNC * 32));
    if constexpr (kMma) {
      // 8 elements per item; the first kPre items of a thread were loaded above
#pragma unroll 4
      for (int m = tid; m < NB * n8; m += kNC * 32) {
        const int b = m / n8, k = (m - b * n8) * 8, j = (m - tid) / (kNC * 32);
        uint4 gv;
        float4 x0, x1;
        if (j < kPre) {
          gv = pg[0];
          x0 = px0[0];
          x1 = px1[0];
#pragma unroll
          for (int jj = 1; jj < kPre; ++jj)
            if (jj == j) {
              gv = pg[jj];
              x0 = px0[jj];
              x1 = px1[jj];
            }
        } else {
          gv = *reinterpret_cast<const uint4*>(gn + k);
          x0 = *reinterpret_cast<const float4*>(a.X + (size_t)b * K + k);
          x1 = *reinterpret_cast<const float4*>(a.X + (size_t)b * K + k + 4);
        }
        float gf[8];
        unpack<T>(gv, gf);
        const float r = rr[b];
        const float xv[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
        uint32_t* row = reinterpret_cast<uint32_t*>(xs + (size_t)b * K);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const __nv_bfloat162 v = __floats2bfloat162_rn((xv[2 * j] * r) * gf[2 * j], (xv[2 * j + 1] * r) * gf[2 * j + 1]);
          row[afrag_pos(k + 2 * j) >> 1] = *reinterpret_cast<const uint32_t*>(&v);
        }
      }
    } else {
      for (int k = tid; k < K; k += kNC * 32) {
        const float gk = to_f(gn[k]);
#pragma unroll
        for (int b = 0; b < NB; ++b) xs[(size_t)b * K + k] = from_f<T>((a.X[(size_t)b * K + k] * rr[b]) * gk);
      }
    }
  } else if constexpr (!XG) {
    if constexpr (kMma) {
      const int n8 = K / 8;
#pragma unroll 4
      for (int m = tid; m < NB * n8; m += kNC * 32) {
        const int b = m / n8, k = (m - b * n8) * 8;
        const uint4 v = *reinterpret_cast<const uint4*>(static_cast<const T*>(a.xin) + (size_t)b * K + k);
        uint32_t* row = reinterpret_cast<uint32_t*>(xs + (size_t)b * K);
        row[afrag_pos(k) >> 1] = v.x;
        row[afrag_pos(k + 2) >> 1] = v.y;
        row[afrag_pos(k + 4) >> 1] = v.z;
        row[afrag_pos(k + 6) >> 1] = v.w;
      }
    } else {
      const uint4* src = reinterpret_cast<const uint4*>(static_cast<const T*>(a.xin));
      uint4* dst = reinterpret_cast<uint4*>(xs);
      for (int i = tid; i < NB * K / V; i += kNC * 32) dst[i] = src[i];
    }
  }
  asm volatile("bar.sync 1, %0;" ::"r"(kNC * 32));

  float ssq = 0.f;  // residual epilogue: this thread's sum of squares (sequence per lane, see below)
  bool aborted = false;
  int stage = 0;
  uint32_t phase = 0;
  if constexpr (kMma) {
    const int gq = lane >> 2, tq = lane & 3;  // fragment row (sequence) and column pair
    const uint32_t st_lane = smem_u32(stages) + (uint32_t)lane * 16;
    for (int g = g0; g < g1; ++g) {
      const int pb = (g - g0) & 1, ew = (g - g0) % kNC;  // partial buffer, epilogue warp
      const int p = g * kGP + tq;
      const bool epi = warp == ew && gq < NB && p < a.n_pairs;
      float e1 = 0.f, e2 = 0.f;
      if (epi) dgemv_epilogue_operands<T, EPI>(a, p, gq, e1, e2);  // latency hidden by the tiles
      // four accumulator sets, so that consecutive products do not wait on
      // each other; added in a fixed order at the end of the group
      float d[4][4];
#pragma unroll
      for (int u = 0; u < 4; ++u) d[u][0] = d[u][1] = d[u][2] = d[u][3] = 0.f;
      for (int c = 0; c < nchunk; ++c) {
        const int k0 = c * KC, n32 = min(KC, K - k0) >> 5;
        const int i0 = n32 * warp / kNC, i1 = n32 * (warp + 1) / kNC;
        bool ok = true;
        if (lane == 0) ok = mbar_wait(&full_bar[stage], phase, a.wait_limit, abort);
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) {
          if (lane == 0) {
            set_error(a.err, VLAC_ERR_TIMEOUT);
            *abort = 1;
          }
          // the warp stays in the group loop, in step with the others' named
          // barriers; the stage is not handed back, so it is never refilled
          aborted = true;
          if (++stage == NS) {
            stage = 0;
            phase ^= 1u;
          }
          continue;
        }
        const uint32_t st = st_lane + (uint32_t)(stage * stage_b);
        const T* xrow = XG ? static_cast<const T*>(a.xin) + (size_t)gq * K + k0 + 2 * tq : xs + (size_t)gq * K + k0 + tq * 8;
        int i = i0;
        // blocks of four 32-element K steps: all fragments are loaded before
        // the first product, one accumulator set per step
        for (; i + 4 <= i1; i += 4) {
          uint32_t bf[4][4];
          uint4 xa[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            ldsm_x4(st + (uint32_t)(i + u) * 512u, bf[u][0], bf[u][1], bf[u][2], bf[u][3]);
            xa[u] = make_uint4(0u, 0u, 0u, 0u);
          }
          if (gq < NB) {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              if constexpr (XG) {
                const T* xr = xrow + (i + u) * 32;
                xa[u] = make_uint4(ldg_u32(xr), ldg_u32(xr + 8), ldg_u32(xr + 16), ldg_u32(xr + 24));
              } else {
                xa[u] = *reinterpret_cast<const uint4*>(xrow + (i + u) * 32);
              }
            }
          }
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            mma_bf16(d[u], xa[u].x, 0u, xa[u].y, 0u, bf[u][0], bf[u][1]);
            mma_bf16(d[u], xa[u].z, 0u, xa[u].w, 0u, bf[u][2], bf[u][3]);
          }
        }
        for (; i < i1; ++i) {
          uint32_t b0, b1, b2, b3;
          ldsm_x4(st + (uint32_t)i * 512u, b0, b1, b2, b3);
          uint4 xv = make_uint4(0u, 0u, 0u, 0u);
          if (gq < NB) {
            if constexpr (XG) {
              const T* xr = xrow + i * 32;
              xv = make_uint4(ldg_u32(xr), ldg_u32(xr + 8), ldg_u32(xr + 16), ldg_u32(xr + 24));
            } else {
              xv = *reinterpret_cast<const uint4*>(xrow + i * 32);
            }
          }
          mma_bf16(d[0], xv.x, 0u, xv.y, 0u, b0, b1);
          mma_bf16(d[0], xv.z, 0u, xv.w, 0u, b2, b3);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty_bar[stage]);
        if (++stage == NS) {
          stage = 0;
          phase ^= 1u;
        }
      }
      // D[gq][2tq], D[gq][2tq+1]: this warp's share of pair tq of sequence gq
      if (gq < NB)
        pacc[pb][warp][lane] = make_float2(((d[0][0] + d[1][0]) + d[2][0]) + d[3][0], ((d[0][1] + d[1][1]) + d[2][1]) + d[3][1]);
      // after this barrier every warp has also finished the previous group's
      // epilogue, so the other buffer is free for the next group
      asm volatile("bar.sync 1, %0;" ::"r"(kNC * 32));
      if (epi) {
        float y1 = 0.f, y2 = 0.f;
#pragma unroll
        for (int w = 0; w < kNC; ++w) {
          const float2 v = pacc[pb][w][lane];
          y1 += v.x;
          y2 += v.y;
        }
        ssq += dgemv_epilogue<T, EPI>(a, p, gq, y1, y2, e1, e2);
      }
    }
  } else {
    const int q = warp >> 1, hk = warp & 1;  // pair within the group, K half
    const T* xsrc = XG ? static_cast<const T*>(a.xin) : xs;
    for (int g = g0; g < g1; ++g) {
      const int p = g * kGP + q;
      const bool epi = hk == 0 && lane < NB && p < a.n_pairs;
      float e1 = 0.f, e2 = 0.f;
      if (epi) dgemv_epilogue_operands<T, EPI>(a, p, lane, e1, e2);
      float acc1[NB], acc2[NB];
#pragma unroll
      for (int b = 0; b < NB; ++b) acc1[b] = acc2[b] = 0.f;
      for (int c = 0; c < nchunk; ++c) {
        const int k0 = c * KC, kn = min(KC, K - k0), nv = kn / V;
        const int v0 = hk ? nv / 2 : 0, v1 = hk ? nv : nv / 2;  // this warp's 16-byte vectors of the rows
        bool ok = true;
        if (lane == 0) ok = mbar_wait(&full_bar[stage], phase, a.wait_limit, abort);
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) {
          if (lane == 0) {
            set_error(a.err, VLAC_ERR_TIMEOUT);
            *abort = 1;
          }
          // the warp stays in the group loop, in step with the others' named
          // barriers; the stage is not handed back, so it is never refilled
          aborted = true;
          if (++stage == NS) {
            stage = 0;
            phase ^= 1u;
          }
          continue;
        }
        const T* st = reinterpret_cast<const T*>(stages + (size_t)stage * stage_b);
        const uint4* w1 = reinterpret_cast<const uint4*>(st + (size_t)(2 * q) * kn);
        const uint4* w2 = reinterpret_cast<const uint4*>(st + (size_t)(2 * q + 1) * kn);
        for (int v = v0 + lane; v < v1; v += 32) {
          float f1[V], f2[V];
          unpack<T>(w1[v], f1);
          unpack<T>(w2[v], f2);
#pragma unroll
          for (int b = 0; b < NB; ++b) {
            float xf[V];
            unpack<T>(reinterpret_cast<const uint4*>(xsrc + (size_t)b * K + k0)[v], xf);
#pragma unroll
            for (int i = 0; i < V; ++i) {
              acc1[b] = fmaf(f1[i], xf[i], acc1[b]);
              acc2[b] = fmaf(f2[i], xf[i], acc2[b]);
            }
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty_bar[stage]);
        if (++stage == NS) {
          stage = 0;
          phase ^= 1u;
        }
      }
      // add the two K halves of every pair in order, then the epilogue
#pragma unroll
      for (int b = 0; b < NB; ++b) {
        const float t1 = warp_allsum(acc1[b]), t2 = warp_allsum(acc2[b]);
        if (hk == 1 && lane == 0) {
          half_acc[q][0][b] = t1;
          half_acc[q][1][b] = t2;
        }
        acc1[b] = t1;
        acc2[b] = t2;
      }
      asm volatile("bar.sync 1, %0;" ::"r"(kNC * 32));
      if (epi) {
        float y1 = 0.f, y2 = 0.f;
#pragma unroll
        for (int bb = 0; bb < NB; ++bb)
          if (bb == lane) {
            y1 = acc1[bb] + half_acc[q][0][bb];
            y2 = acc2[bb] + half_acc[q][1][bb];
          }
        ssq += dgemv_epilogue<T, EPI>(a, p, lane, y1, y2, e1, e2);
      }
      asm volatile("bar.sync 1, %0;" ::"r"(kNC * 32));  // half_acc is reused by the next group
    }
  }
  if constexpr (EPI == kEpiResid) {
    // per thread: sequence gq = lane/4 (bf16) or lane (fp32); summed over the
    // warps and then the lanes of a sequence in a fixed order
    red[warp][lane] = ssq;
    asm volatile("bar.sync 1, %0;" ::"r"(kNC * 32));
    if (tid < NB) {
      float t = 0.f;
      for (int w = 0; w < kNC; ++w) {
        if constexpr (kMma) {
          for (int j = 0; j < 4; ++j) t += red[w][tid * 4 + j];
        } else {
          t += red[w][tid];
        }
      }
      a.ssq_out[(size_t)tid * gridDim.x + blockIdx.x] = t;
    }
  }
  // A warp that gave up skipped waits, so copies may still be landing in this
  // CTA's shared memory; a warp that did not saw every copy land.
  if (aborted && lane == 0) {
    bool ended = false;
    for (uint32_t it = 0; it < kWaitLimit && !ended; ++it) ended = mbar_test(&done_bar, 0);
    if (ended) ring_drain(full_bar, NS, (int)prod_end[0], prod_end[1], prod_end[2]);
  }
}

template <typename T, int NB, int EPI, bool NORM>
static void dgemv_nb(const DGemv& a, int grid, cudaStream_t st) {
  // the input vector lives in shared memory unless it is large (then it is read through L1)
  const bool xg = !NORM && (size_t)NB * a.K * sizeof(T) > 64 * 1024;
  const size_t smem = (xg ? 0 : sgemv_xs_bytes(NB, a.K, (int)sizeof(T))) + (size_t)a.ns * 2 * kGP * kDecTileB;
  auto kern = xg ? dgemv_kernel<T, NB, EPI, NORM, true> : dgemv_kernel<T, NB, EPI, NORM, false>;
  static size_t smem_set[2] = {48 * 1024, 48 * 1024};  // raised once per kernel, before any graph capture of it
  if (smem > smem_set[xg]) {
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    smem_set[xg] = smem;
  }
  launch_k(kern, dim3(grid), dim3((kNC + 1) * 32), smem, st, a);
}

template <typename T, int EPI, bool NORM>
static void dgemv_dispatch(const DGemv& a, int nb, int grid, cudaStream_t st) {
  switch (nb) {
    case 1: dgemv_nb<T, 1, EPI, NORM>(a, grid, st); break;
    case 2: dgemv_nb<T, 2, EPI, NORM>(a, grid, st); break;
    case 3: dgemv_nb<T, 3, EPI, NORM>(a, grid, st); break;
    case 4: dgemv_nb<T, 4, EPI, NORM>(a, grid, st); break;
    case 5: dgemv_nb<T, 5, EPI, NORM>(a, grid, st); break;
    case 6: dgemv_nb<T, 6, EPI, NORM>(a, grid, st); break;
    case 7: dgemv_nb<T, 7, EPI, NORM>(a, grid, st); break;
    default: dgemv_nb<T, 8, EPI, NORM>(a, grid, st); break;
  }
}

int dgemv_grid(int n_pairs, int n_sm) { return std::min((n_pairs + kGP - 1) / kGP, n_sm); }

template <typename T>
void launch_dgemv(const DGemv& a, int epi, int nb, int n_sm, cudaStream_t st) {
  const int grid = dgemv_grid(a.n_pairs, n_sm);
  switch (epi) {
    case kEpiQkvRope: dgemv_dispatch<T, kEpiQkvRope, true>(a, nb, grid, st); break;
    case kEpiSwiglu: dgemv_dispatch<T, kEpiSwiglu, true>(a, nb, grid, st); break;
    default: dgemv_dispatch<T, kEpiResid, false>(a, nb, grid, st); break;
  }
}
template void launch_dgemv<float>(const DGemv&, int, int, int, cudaStream_t);
template void launch_dgemv<bf16>(const DGemv&, int, int, int, cudaStream_t);

// ---- decode attention: one query per (sequence, head) ----------------------------
//
// The keys 0..pos of every (sequence, head) are cut into chunks of 64; one
// block of two warps per (chunk, head, sequence), one warp per 32-key tile.
// A warp issues all loads of its tile at once -- lane j reads key j's K row,
// and the V rows go to shared memory by cp.async -- so a tile costs one memory
// round trip.  Each block leaves its partial (max, sum, output row) in `part`;
// the last block of a (sequence, head) to finish (a counter that it resets)
// adds the partials in chunk order and writes the output.
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(smem))),
               "l"(gmem)
               : "memory");
}

constexpr int kDecKeys = 64;  // keys per block

template <typename T, int HD>
__global__ void __launch_bounds__(64) dec_attn_kernel(const T* __restrict__ Q, const T* __restrict__ Kc,
                                                      const T* __restrict__ Vc, size_t kv_seq_stride, int Tc, int pos,
                                                      int n_heads, float scale, float* __restrict__ part,
                                                      unsigned* __restrict__ counters, T* __restrict__ O) {
  constexpr int EPL = HD / 32, V = Vec<T>::n, CPR = HD * (int)sizeof(T) / 16;  // 16-byte chunks per row
  constexpr int NW = kDecKeys / 32;
  __shared__ __align__(16) T vbuf_all[NW][32][HD];
  __shared__ float qs[HD];
  __shared__ float wm[NW], wl[NW];
  __shared__ float wacc[NW][HD];
  __shared__ int is_last;
  pdl_wait();
  pdl_trigger();
  const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z, n_kc = gridDim.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int hidden = n_heads * HD;
  T* vbuf = &vbuf_all[warp][0][0];
  const T* Kh = Kc + (size_t)b * kv_seq_stride + (size_t)h * Tc * HD;
  const T* Vh = Vc + (size_t)b * kv_seq_stride + (size_t)h * Tc * HD;
  const int nkeys = min(pos + 1, Tc);
  const int k0 = c * kDecKeys, k1 = min(nkeys, k0 + kDecKeys);
  for (int e = threadIdx.x; e < HD; e += blockDim.x) qs[e] = to_f(Q[(size_t)b * hidden + (size_t)h * HD + e]);
  __syncthreads();
  float m_run = -INFINITY, l_run = 0.f, acc[EPL];
#pragma unroll
  for (int e = 0; e < EPL; ++e) acc[e] = 0.f;
  const int j0 = k0 + warp * 32;
  if (j0 < k1) {
    const int j = j0 + lane, jn = min(32, k1 - j0);
    // the tile's V rows go to shared memory asynchronously, its K rows to registers
    for (int q = lane; q < jn * CPR; q += 32) {
      const int jj = q / CPR, r = q - jj * CPR;
      cp_async16(vbuf + (size_t)jj * HD + r * (16 / sizeof(T)), Vh + (size_t)(j0 + jj) * HD + r * (16 / sizeof(T)));
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    uint4 kr[HD / V];
    if (j < k1) {
      const uint4* src = reinterpret_cast<const uint4*>(Kh + (size_t)j * HD);
#pragma unroll
      for (int v = 0; v < HD / V; ++v) kr[v] = src[v];
    }
    float sc = -INFINITY;
    if (j < k1) {
      float d = 0.f;
#pragma unroll
      for (int v = 0; v < HD / V; ++v) {
        float f[V];
        unpack<T>(kr[v], f);
#pragma unroll
        for (int i = 0; i < V; ++i) d = fmaf(f[i], qs[v * V + i], d);
      }
      sc = d * scale;
    }
    m_run = warp_max(sc);
    const float p = (sc == -INFINITY) ? 0.f : expf(sc - m_run);
    l_run = warp_sum(p);
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncwarp();
#pragma unroll 8
    for (int jj = 0; jj < jn; ++jj) {
      const float pj = __shfl_sync(0xffffffffu, p, jj);
      const T* vr = vbuf + (size_t)jj * HD + lane * EPL;
#pragma unroll
      for (int e = 0; e < EPL; ++e) acc[e] = fmaf(pj, to_f(vr[e]), acc[e]);
    }
  }
  if (lane == 0) {
    wm[warp] = m_run;
    wl[warp] = l_run;
  }
#pragma unroll
  for (int e = 0; e < EPL; ++e) wacc[warp][lane * EPL + e] = acc[e];
  __syncthreads();
  // this block's partial: the warps' tiles combined in tile order
  float* mine = part + ((size_t)(b * n_heads + h) * n_kc + c) * (HD + 2);
  {
    float M = -INFINITY;
    for (int w = 0; w < NW; ++w) M = fmaxf(M, wm[w]);
    for (int e = threadIdx.x; e < HD; e += blockDim.x) {
      float L = 0.f, o = 0.f;
      for (int w = 0; w < NW; ++w) {
        const float f = (wm[w] == -INFINITY) ? 0.f : expf(wm[w] - M);
        L = fmaf(wl[w], f, L);
        o = fmaf(wacc[w][e], f, o);
      }
      mine[2 + e] = o;
      if (e == 0) {
        mine[0] = M;
        mine[1] = L;
      }
    }
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const unsigned prev = atomicAdd(counters + b * n_heads + h, 1u);
    is_last = prev == (unsigned)(n_kc - 1);
  }
  __syncthreads();
  if (!is_last) return;
  // the last block: every chunk's partial, in chunk order
  __threadfence();
  const float* all = part + (size_t)(b * n_heads + h) * n_kc * (HD + 2);
  float M = -INFINITY;
  for (int q = 0; q < n_kc; ++q) M = fmaxf(M, __ldcg(all + (size_t)q * (HD + 2)));
  for (int e = threadIdx.x; e < HD; e += blockDim.x) {
    float L = 0.f, o = 0.f;
    for (int q = 0; q < n_kc; ++q) {
      const float mq = __ldcg(all + (size_t)q * (HD + 2));
      const float f = (mq == -INFINITY) ? 0.f : expf(mq - M);
      L = fmaf(__ldcg(all + (size_t)q * (HD + 2) + 1), f, L);
      o = fmaf(__ldcg(all + (size_t)q * (HD + 2) + 2 + e), f, o);
    }
    O[(size_t)b * hidden + (size_t)h * HD + e] = from_f<T>(o / L);
  }
  if (threadIdx.x == 0) counters[b * n_heads + h] = 0u;  // ready for the next launch
}

// Cluster variant (bf16, up to 8 blocks of 128 keys): the blocks of one
// (sequence, head) form a thread-block cluster.  K and V rows of the keys
// before `pos` were written by earlier passes, so they are requested before
// the dependency wait and arrive while the preceding QKV projection drains;
// only Q and the new key's row wait for it.  Each block leaves its partial
// in its own shared memory; block 0 of the cluster reads them over
// distributed shared memory in chunk order and writes the output.
constexpr int kDcW = 4;             // warps per block, 32 keys each
constexpr int kDcKeys = kDcW * 32;  // keys per block
constexpr int kDcMaxCluster = 8;    // portable cluster size

template <int HD>
__global__ void __launch_bounds__(kDcW * 32) dec_attn_cluster_kernel(const bf16* __restrict__ Q,
                                                                     const bf16* __restrict__ Kc,
                                                                     const bf16* __restrict__ Vc,
                                                                     size_t kv_seq_stride, int Tc, int pos,
                                                                     int n_heads, float scale, bf16* __restrict__ O) {
  using T = bf16;
  constexpr int EPL = HD / 32, V = Vec<T>::n, CPR = HD * (int)sizeof(T) / 16;  // 16-byte chunks per row
  __shared__ __align__(16) T vbuf_all[kDcW][32][HD];
  __shared__ float qs[HD];
  __shared__ float wm[kDcW], wl[kDcW];
  __shared__ float wacc[kDcW][HD];
  __shared__ float cpart[HD + 2];  // this block's (max, sum, output row)
  namespace cg = cooperative_groups;
  cg::cluster_group cluster = cg::this_cluster();
  const int c = blockIdx.x, h = blockIdx.y, b = blockIdx.z, n_kc = gridDim.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int hidden = n_heads * HD;
  T* vbuf = &vbuf_all[warp][0][0];
  const T* Kh = Kc + (size_t)b * kv_seq_stride + (size_t)h * Tc * HD;
  const T* Vh = Vc + (size_t)b * kv_seq_stride + (size_t)h * Tc * HD;
  const int nkeys = min(pos + 1, Tc);
  const int k1 = min(nkeys, (c + 1) * kDcKeys);
  const int j0 = c * kDcKeys + warp * 32, jn = max(0, min(32, k1 - j0)), j = j0 + lane;
  // ---- before the dependency wait: the rows of the older keys ----
  for (int q = lane; q < jn * CPR; q += 32) {
    const int jj = q / CPR, r = q - jj * CPR;
    if (j0 + jj != pos)
      cp_async16(vbuf + (size_t)jj * HD + r * (16 / sizeof(T)), Vh + (size_t)(j0 + jj) * HD + r * (16 / sizeof(T)));
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
  uint4 kr[HD / V];
  if (lane < jn && j != pos) {
    const uint4* src = reinterpret_cast<const uint4*>(Kh + (size_t)j * HD);
#pragma unroll
    for (int v = 0; v < HD / V; ++v) kr[v] = src[v];
  }
  pdl_wait();
  pdl_trigger();
  // ---- the query and the new key's row ----
  if (lane < jn && j == pos) {
    const uint4* src = reinterpret_cast<const uint4*>(Kh + (size_t)j * HD);
#pragma unroll
    for (int v = 0; v < HD / V; ++v) kr[v] = src[v];
  }
  if (pos >= j0 && pos < j0 + jn)
    for (int r = lane; r < CPR; r += 32)
      cp_async16(vbuf + (size_t)(pos - j0) * HD + r * (16 / sizeof(T)), Vh + (size_t)pos * HD + r * (16 / sizeof(T)));
  asm volatile("cp.async.commit_group;" ::: "memory");
  for (int e = threadIdx.x; e < HD; e += blockDim.x) qs[e] = to_f(Q[(size_t)b * hidden + (size_t)h * HD + e]);
  __syncthreads();
  float m_run = -INFINITY, l_run = 0.f, acc[EPL];
#pragma unroll
  for (int e = 0; e < EPL; ++e) acc[e] = 0.f;
  if (jn > 0) {
    float sc = -INFINITY;
    if (lane < jn) {
      float d = 0.f;
#pragma unroll
      for (int v = 0; v < HD / V; ++v) {
        float f[V];
        unpack<T>(kr[v], f);
#pragma unroll
        for (int i = 0; i < V; ++i) d = fmaf(f[i], qs[v * V + i], d);
      }
      sc = d * scale;
    }
    m_run = warp_max(sc);
    const float p = (sc == -INFINITY) ? 0.f : expf(sc - m_run);
    l_run = warp_sum(p);
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncwarp();
#pragma unroll 8
    for (int jj = 0; jj < jn; ++jj) {
      const float pj = __shfl_sync(0xffffffffu, p, jj);
      const T* vr = vbuf + (size_t)jj * HD + lane * EPL;
#pragma unroll
      for (int e = 0; e < EPL; ++e) acc[e] = fmaf(pj, to_f(vr[e]), acc[e]);
    }
  }
  if (lane == 0) {
    wm[warp] = m_run;
    wl[warp] = l_run;
  }
#pragma unroll
  for (int e = 0; e < EPL; ++e) wacc[warp][lane * EPL + e] = acc[e];
  __syncthreads();
  {
    float M = -INFINITY;
    for (int w = 0; w < kDcW; ++w) M = fmaxf(M, wm[w]);
    for (int e = threadIdx.x; e < HD; e += blockDim.x) {
      float L = 0.f, o = 0.f;
      for (int w = 0; w < kDcW; ++w) {
        const float f = (wm[w] == -INFINITY) ? 0.f : expf(wm[w] - M);
        L = fmaf(wl[w], f, L);
        o = fmaf(wacc[w][e], f, o);
      }
      cpart[2 + e] = o;
      if (e == 0) {
        cpart[0] = M;
        cpart[1] = L;
      }
    }
  }
  cluster.sync();
  if (cluster.block_rank() == 0) {
    float M = -INFINITY;
    for (int q = 0; q < n_kc; ++q) M = fmaxf(M, *cluster.map_shared_rank(&cpart[0], q));
    for (int e = threadIdx.x; e < HD; e += blockDim.x) {
      float L = 0.f, o = 0.f;
      for (int q = 0; q < n_kc; ++q) {
        const float* rp = cluster.map_shared_rank(&cpart[0], q);
        const float f = (rp[0] == -INFINITY) ? 0.f : expf(rp[0] - M);
        L = fmaf(rp[1], f, L);
        o = fmaf(rp[2 + e], f, o);
      }
      O[(size_t)b * hidden + (size_t)h * HD + e] = from_f<T>(o / L);
    }
  }
  cluster.sync();  // every block's partial stays in place until block 0 has read it
}

template <int HD>
void launch_dec_attn_cluster(int B, int n_heads, int n_kc, const bf16* Q, const bf16* Kc, const bf16* Vc,
                             size_t kv_seq_stride, int Tc, int pos, float scale, bf16* O, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_kc, n_heads, B);
  cfg.blockDim = dim3(kDcW * 32);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = n_kc;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = g_pdl ? 2 : 1;
  cudaLaunchKernelEx(&cfg, dec_attn_cluster_kernel<HD>, Q, Kc, Vc, kv_seq_stride, Tc, pos, n_heads, scale, O);
}

template <typename T>
void launch_dec_attention(int B, int n_heads, int head_dim, const T* Q, const T* Kc, const T* Vc, size_t kv_seq_stride,
                          int Tc, int pos, float* part, unsigned* counters, T* O, cudaStream_t st) {
  const float scale = 1.0f / sqrtf((float)head_dim);
  const int nkeys = std::min(pos + 1, Tc);
  if constexpr (sizeof(T) == 2) {
    const int n_kc = (nkeys + kDcKeys - 1) / kDcKeys;
    if (n_kc <= kDcMaxCluster && (head_dim == 128 || head_dim == 64)) {
      if (head_dim == 128)
        launch_dec_attn_cluster<128>(B, n_heads, n_kc, Q, Kc, Vc, kv_seq_stride, Tc, pos, scale, O, st);
      else
        launch_dec_attn_cluster<64>(B, n_heads, n_kc, Q, Kc, Vc, kv_seq_stride, Tc, pos, scale, O, st);
      return;
    }
  }
  const int n_kc = (nkeys + kDecKeys - 1) / kDecKeys;
  const dim3 grid(n_kc, n_heads, B);
  if (head_dim == 128)
    launch_k(dec_attn_kernel<T, 128>, grid, dim3(kDecKeys), 0, st, Q, Kc, Vc, kv_seq_stride, Tc, pos, n_heads, scale,
             part, counters, O);
  else
    launch_k(dec_attn_kernel<T, 64>, grid, dim3(kDecKeys), 0, st, Q, Kc, Vc, kv_seq_stride, Tc, pos, n_heads, scale,
             part, counters, O);
}
template void launch_dec_attention<float>(int, int, int, const float*, const float*, const float*, size_t, int, int,
                                          float*, unsigned*, float*, cudaStream_t);
template void launch_dec_attention<bf16>(int, int, int, const bf16*, const bf16*, const bf16*, size_t, int, int,
                                         float*, unsigned*, bf16*, cudaStream_t);

// ---- action head -------------------------------------------------------------------

// Action head of one action row, fused (Eq. 1): the final RMSNorm, the
// logits of the n_bins action-bin rows of the LM head, and the top-2 / margin
// reduction.  One thread-block cluster of kHeadCluster blocks per (row,
// sequence) splits the bins: each block norms the row into its shared memory
// as T and computes n_bins / kHeadCluster logits, four bins per warp at a time
// (lanes over K, fp32 FMA, warp sum); block 0 then collects every logit over
// distributed shared memory and one warp reduces them: argmax (lowest bin on
// ties), l1 - l2, p1 - p2 = (1 - exp(l2 - l1)) / z and the entropy
// ln z - sum_c p_c (l_c - l1), z = sum_c exp(l_c - l1).  The cluster
// barriers are the hardware's; no block waits on a flag.
constexpr int kHeadCluster = 8;
template <typename T>
__global__ void __launch_bounds__(256) head_fused_kernel(const float* __restrict__ X, const int* __restrict__ row_of_seq,
                                                         size_t x_seq_stride, int hidden, int n_bins,
                                                         const T* __restrict__ final_norm,
                                                         const T* __restrict__ head_w, float eps,
                                                         float* __restrict__ logits_ws, int D, int tok0,
                                                         int32_t* __restrict__ ids, float* __restrict__ margins,
                                                         float* __restrict__ gaps, float* __restrict__ logits,
                                                         float* __restrict__ entropy) {
  namespace cg = cooperative_groups;
  cg::cluster_group cluster = cg::this_cluster();
  pdl_wait();
  pdl_trigger();
  extern __shared__ __align__(1024) uint8_t dsm[];
  T* xs = reinterpret_cast<T*>(dsm);                                     // [hidden]
  const int per = n_bins / kHeadCluster;
  float* lg_own = reinterpret_cast<float*>(dsm + (size_t)hidden * sizeof(T));  // [per]
  float* lg_all = lg_own + per;                                          // [n_bins], block 0 only
  const int rank = (int)cluster.block_rank();
  const int j = blockIdx.y, b = blockIdx.z;
  const int row = row_of_seq ? row_of_seq[b] + j : j;
  const float* x = X + (size_t)b * x_seq_stride + (size_t)row * hidden;
  norm_rows_to_smem<T, 1>(x, final_norm, hidden, eps, xs);
  constexpr int V = Vec<T>::n;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kv = hidden / V;
  const uint4* xv = reinterpret_cast<const uint4*>(xs);
  // four bins per warp at a time (their weight rows streamed side by side);
  // per bin the same order: lanes over K, fp32 FMA, then the warp sum
  for (int c = 4 * warp; c < per; c += 32) {
    const uint4* w[4];
    float a[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      w[q] = reinterpret_cast<const uint4*>(head_w + (size_t)(rank * per + min(c + q, per - 1)) * hidden);
      a[q] = 0.f;
    }
    // a lane's K steps k = lane, lane + 32, ... in order; the loads of four
    // steps are issued before their products
    for (int k0 = lane; k0 < kv; k0 += 128) {
      uint4 wr[4][4];
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int q = 0; q < 4; ++q) wr[u][q] = k0 + 32 * u < kv ? __ldg(w[q] + k0 + 32 * u) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if (k0 + 32 * u >= kv) break;
        float xf[V];
        unpack<T>(xv[k0 + 32 * u], xf);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          float f[V];
          unpack<T>(wr[u][q], f);
#pragma unroll
          for (int i = 0; i < V; ++i) a[q] = fmaf(f[i], xf[i], a[q]);
        }
      }
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      a[q] = warp_allsum(a[q]);
      if (lane == 0 && c + q < per) lg_own[c + q] = a[q];
    }
  }
  cluster.sync();
  if (rank == 0 && warp == 0) {
    for (int c = lane; c < n_bins; c += 32) lg_all[c] = *cluster.map_shared_rank(&lg_own[c % per], c / per);
    __syncwarp();
    const float* lg = lg_all;
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
    float v2 = -INFINITY, z = 0.f, zl = 0.f;
    for (int c = lane; c < n_bins; c += 32) {
      if (c != bi) v2 = fmaxf(v2, lg[c]);
      const float e = expf(lg[c] - bv);
      z += e;
      zl = fmaf(e, lg[c] - bv, zl);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v2 = fmaxf(v2, __shfl_xor_sync(0xffffffffu, v2, o));
    z = warp_allsum(z);
    zl = warp_allsum(zl);
    const size_t t = (size_t)b * D + tok0 + j;
    if (lane == 0) {
      ids[t] = bi;
      margins[t] = -expm1f(v2 - bv) / z;
      gaps[t] = bv - v2;
      if (entropy) entropy[t] = logf(z) - zl / z;
    }
    float* ws = logits_ws + ((size_t)b * gridDim.y + j) * n_bins;  // the vocabulary margin reads them
    for (int c = lane; c < n_bins; c += 32) {
      ws[c] = lg[c];
      if (logits) logits[t * n_bins + c] = lg[c];
    }
  }
  cluster.sync();  // every block's logits stay in place until block 0 has read them
}

// ---- margin over the whole vocabulary (Sec. IV-A, VLAC_MARGIN_VOCAB) ------------

// The final-norm rows of the action positions, stored as T for the vocabulary
// GEMV: row (b, j) at xh + (b * rows_per_seq + j) * hidden, rounded exactly as
// the bin head rounds them.
template <typename T>
__global__ void __launch_bounds__(256) head_rows_kernel(const float* __restrict__ X, const int* __restrict__ row_of_seq,
                                                        size_t x_seq_stride, int hidden, const T* __restrict__ final_norm,
                                                        float eps, T* __restrict__ xh) {
  pdl_wait();
  pdl_trigger();
  const int j = blockIdx.x, b = blockIdx.y;
  const int row = row_of_seq ? row_of_seq[b] + j : j;
  norm_rows_to_smem<T, 1>(X + (size_t)b * x_seq_stride + (size_t)row * hidden, final_norm, hidden, eps,
                          xh + ((size_t)b * gridDim.x + j) * hidden);
}

// Logits of the LM-head rows outside the action bins (r < n_rows) for NR
// normed action rows at once: a CTA takes 64 weight rows, 8 per warp, lanes
// over K; every weight element read is used for the NR rows.
// vl[(g * NR + i) * n_rows + r] for input row g * NR + i < n_in.
constexpr int kVocRowsPerCta = 64;

template <typename T, int NR>
__global__ void __launch_bounds__(256) vocab_logits_kernel(const T* __restrict__ W, int n_rows, int hidden,
                                                           const T* __restrict__ xh, int n_in,
                                                           float* __restrict__ vl) {
  pdl_wait();
  pdl_trigger();
  constexpr int V = Vec<T>::n;
  extern __shared__ __align__(16) uint8_t vsm[];
  T* xs = reinterpret_cast<T*>(vsm);  // [NR][hidden]
  const int g = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int kv = hidden / V;
  for (int m = threadIdx.x; m < NR * kv; m += blockDim.x) {
    const int i = m / kv, k = m - i * kv;
    const int row = g * NR + i;
    reinterpret_cast<uint4*>(xs)[m] =
        row < n_in ? reinterpret_cast<const uint4*>(xh + (size_t)row * hidden)[k] : make_uint4(0u, 0u, 0u, 0u);
  }
  __syncthreads();
  const int r0 = blockIdx.x * kVocRowsPerCta + warp * 8;
  float acc[8][NR];
#pragma unroll
  for (int q = 0; q < 8; ++q)
#pragma unroll
    for (int i = 0; i < NR; ++i) acc[q][i] = 0.f;
  for (int k = lane; k < kv; k += 32) {
    float xf[NR][V];
#pragma unroll
    for (int i = 0; i < NR; ++i) unpack<T>(reinterpret_cast<const uint4*>(xs + (size_t)i * hidden)[k], xf[i]);
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      float wf[V];
      const uint4 wv = r0 + q < n_rows ? __ldg(reinterpret_cast<const uint4*>(W + (size_t)(r0 + q) * hidden) + k)
                                       : make_uint4(0u, 0u, 0u, 0u);
      unpack<T>(wv, wf);
#pragma unroll
      for (int i = 0; i < NR; ++i)
#pragma unroll
        for (int e = 0; e < V; ++e) acc[q][i] = fmaf(wf[e], xf[i][e], acc[q][i]);
    }
  }
#pragma unroll
  for (int q = 0; q < 8; ++q)
#pragma unroll
    for (int i = 0; i < NR; ++i) {
      const float s = warp_allsum(acc[q][i]);
      const int row = g * NR + i;
      if (lane == 0 && r0 + q < n_rows && row < n_in) vl[(size_t)row * n_rows + r0 + q] = s;
    }
}

// p1 - p2 of the softmax over all vocab logits of one action row: the two
// largest (a value present twice counts twice) and sum exp(l - l1), from the
// non-bin logits vl and the bin logits of logits_ws; fixed reduction order.
__global__ void __launch_bounds__(256) vocab_margin_kernel(const float* __restrict__ vl, int n_rows,
                                                           const float* __restrict__ logits_ws, int n_bins, int D,
                                                           int tok0, float* __restrict__ vm) {
  pdl_wait();
  pdl_trigger();
  __shared__ float s1[8], s2[8], sz[8];
  const int j = blockIdx.x, b = blockIdx.y, rows_per_seq = gridDim.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const size_t rix = (size_t)b * rows_per_seq + j;
  const float* a = vl + rix * n_rows;
  const float* bl = logits_ws + rix * n_bins;
  const int n = n_rows + n_bins;
  float t1 = -INFINITY, t2 = -INFINITY;
  for (int c = threadIdx.x; c < n; c += blockDim.x) {
    const float v = c < n_rows ? a[c] : bl[c - n_rows];
    if (v > t1) {
      t2 = t1;
      t1 = v;
    } else if (v > t2) {
      t2 = v;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float u1 = __shfl_xor_sync(0xffffffffu, t1, o), u2 = __shfl_xor_sync(0xffffffffu, t2, o);
    const float n2 = fmaxf(fminf(t1, u1), fmaxf(t2, u2));
    t1 = fmaxf(t1, u1);
    t2 = n2;
  }
  if (lane == 0) {
    s1[warp] = t1;
    s2[warp] = t2;
  }
  __syncthreads();
  t1 = s1[0];
  t2 = s2[0];
  for (int w = 1; w < 8; ++w) {
    const float n2 = fmaxf(fminf(t1, s1[w]), fmaxf(t2, s2[w]));
    t1 = fmaxf(t1, s1[w]);
    t2 = n2;
  }
  float z = 0.f;
  for (int c = threadIdx.x; c < n; c += blockDim.x) z += expf((c < n_rows ? a[c] : bl[c - n_rows]) - t1);
  z = warp_allsum(z);
  if (lane == 0) sz[warp] = z;
  __syncthreads();
  if (threadIdx.x == 0) {
    float zt = 0.f;
    for (int w = 0; w < 8; ++w) zt += sz[w];
    vm[(size_t)b * D + tok0 + j] = -expm1f(t2 - t1) / zt;
  }
}

template <typename T, int NR>
static void vocab_logits_launch(const T* W, int n_rows, int hidden, const T* xh, int n_in, float* vl,
                                cudaStream_t st) {
  const size_t smem = (size_t)NR * hidden * sizeof(T);
  static size_t smem_set = 48 * 1024;  // raised once per kernel, before any graph capture of it
  if (smem > smem_set) {
    cudaFuncSetAttribute(vocab_logits_kernel<T, NR>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    smem_set = smem;
  }
  const dim3 grid((n_rows + kVocRowsPerCta - 1) / kVocRowsPerCta, (n_in + NR - 1) / NR);
  launch_k(vocab_logits_kernel<T, NR>, grid, dim3(256), smem, st, W, n_rows, hidden, xh, n_in, vl);
}

template <typename T>
void launch_head2(const float* X, const int* row_of_seq, size_t x_seq_stride, int rows_per_seq, int B, int hidden,
                  int n_bins, const T* final_norm, const T* head_w, float eps, float* logits_ws, int D, int tok0,
                  int32_t* ids, float* margins, float* gaps, float* logits, float* entropy, const VocabHead* vh,
                  cudaStream_t st) {
  const size_t smem = (size_t)hidden * sizeof(T) + (size_t)(n_bins / kHeadCluster + n_bins) * sizeof(float);
  static size_t smem_set = 48 * 1024;  // raised once per kernel, before any graph capture of it
  if (smem > smem_set) {
    cudaFuncSetAttribute(head_fused_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    smem_set = smem;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kHeadCluster, rows_per_seq, B);
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kHeadCluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = g_pdl ? 2 : 1;
  cudaLaunchKernelEx(&cfg, head_fused_kernel<T>, X, row_of_seq, x_seq_stride, hidden, n_bins, final_norm, head_w, eps,
                     logits_ws, D, tok0, ids, margins, gaps, logits, entropy);
  if (!vh) return;
  // the other rows of the LM head: every weight row read once per group of <= 8 action rows
  T* xh = static_cast<T*>(vh->xh);
  const T* Wv = static_cast<const T*>(vh->W);
  launch_k(head_rows_kernel<T>, dim3(rows_per_seq, B), dim3(256), 0, st, X, row_of_seq, x_seq_stride, hidden,
           final_norm, eps, xh);
  const int n_in = rows_per_seq * B;
  if (vh->n_rows == 0) {  // every token is an action bin
  } else if (n_in == 1)
    vocab_logits_launch<T, 1>(Wv, vh->n_rows, hidden, xh, n_in, vh->vl, st);
  else if (n_in == 2)
    vocab_logits_launch<T, 2>(Wv, vh->n_rows, hidden, xh, n_in, vh->vl, st);
  else if (n_in <= 4)
    vocab_logits_launch<T, 4>(Wv, vh->n_rows, hidden, xh, n_in, vh->vl, st);
  else
    vocab_logits_launch<T, 8>(Wv, vh->n_rows, hidden, xh, n_in, vh->vl, st);
  launch_k(vocab_margin_kernel, dim3(rows_per_seq, B), dim3(256), 0, st, (const float*)vh->vl, vh->n_rows,
           (const float*)logits_ws, n_bins, D, tok0, vh->vm);
}
template void launch_head2<float>(const float*, const int*, size_t, int, int, int, int, const float*, const float*,
                                  float, float*, int, int, int32_t*, float*, float*, float*, float*, const VocabHead*,
                                  cudaStream_t);
template void launch_head2<bf16>(const float*, const int*, size_t, int, int, int, int, const bf16*, const bf16*,
                                 float, float*, int, int, int32_t*, float*, float*, float*, float*, const VocabHead*,
                                 cudaStream_t);

}  // namespace vlac
