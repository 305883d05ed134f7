// Persistent decode pass: every layer of one autoregressive decode token in
// one cooperative launch (Algorithm 1, the decode of the action tokens),
// bf16 weights, head_dim 128, up to two sequences.
//
// The per-projection chain (k_decode.cu) loses time at every launch
// boundary: the release after the previous grid, the input-vector prologue
// and the whole-group imbalance, while its weight ring sits full.  Here one
// CTA per SM runs all layers.  A producer warp streams this CTA's share of
// every projection of every layer through the ring and never waits on
// another CTA (the weights are constant); eight consumer warps run the
// projections and the attention, separated by grid-wide barriers, while the
// ring keeps filling.
//
// Per layer: q/k/v (RMSNorm prologue, RoPE, Q and the K/V rows at pos) |
// barrier | attention, one (sequence, head, key range) per CTA, the CTA's
// older K/V rows staged in shared memory during the layer before | barrier |
// o-projection + residual | barrier | gate/up (RMSNorm prologue, SwiGLU) |
// barrier | down + residual | barrier (before the next layer).
//
// Data one CTA writes and another reads inside the launch (Q, the K/V rows at
// pos, the attention output and partials, the residual rows, the SwiGLU
// output, the sums of squares) is published by the barrier (a release add at
// GPU scope after a CTA barrier; an acquire poll, then a CTA barrier) and
// read through L2 (ld.global.cg).  Every wait is bounded (the context's wait
// limit; drains before exit keep a fixed one); a CTA that gives up latches
// VLAC_ERR_TIMEOUT, stops waiting and still arrives at every later barrier,
// so the others finish.
#include <algorithm>

#include "internal.cuh"

namespace vlac {

namespace {

constexpr int kPC = 8;                                      // consumer warps
constexpr int kPTR = 2 * kDecGroupPairs;                    // tile rows
constexpr int kPKC = kDecTileBytes / 2;                     // bf16 elements per K chunk
constexpr size_t kPStage = (size_t)kPTR * kDecTileBytes;    // bytes per ring stage
constexpr int kPMaxNS = 8;                                  // ring capacity
constexpr int kPHD = 128;                                   // head_dim

__device__ __forceinline__ float p_allsum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float p_allmax(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ void bf16x8(const uint4& u, float* f) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}
__device__ __forceinline__ void consumers_sync() { asm volatile("bar.sync 1, %0;" ::"r"(kPC * 32) : "memory"); }

// One projection of one layer: 0 q/k/v, 1 o, 2 gate/up, 3 down.
struct Proj {
  const bf16* W;
  int K, n_pairs;
};
__device__ __forceinline__ Proj proj_of(const DPass& a, int l, int j) {
  if (j == 0) return {a.w_qkv[l], a.hidden, 3 * a.hidden / 2};
  if (j == 1) return {a.w_o[l], a.hidden, a.hidden / 2};
  if (j == 2) return {a.w_gu[l], a.hidden, a.ffn};
  return {a.w_d[l], a.ffn, a.hidden / 2};
}

// Grid-wide barrier number `epoch` (1, 2, ...): every CTA arrives once.
// bar_mode 1: the arrival is a release add at GPU scope (it orders the
// CTA's writes before it, which the CTA barrier before it collects) and the
// poll an acquire load; bar_mode 0: full fences around a relaxed add and a
// volatile poll.
__device__ __forceinline__ void grid_sync(const DPass& a, unsigned epoch, volatile int* abort) {
  consumers_sync();
  if (threadIdx.x == 0) {
    const unsigned target = epoch * gridDim.x;
    uint32_t it = 0;
    if (a.bar_mode == 1) {
      asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(a.bar) : "memory");
      if (!*abort) {
        for (;;) {
          unsigned v;
          asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(a.bar) : "memory");
          if (v >= target) break;
          if (++it > a.wait_limit) {
            set_error(a.err, VLAC_ERR_TIMEOUT);
            *abort = 1;
            break;
          }
          __nanosleep(20);
        }
      }
    } else {
      __threadfence();
      atomicAdd(a.bar, 1u);
      if (!*abort) {
        while (*reinterpret_cast<volatile unsigned*>(a.bar) < target) {
          if (++it > a.wait_limit) {
            set_error(a.err, VLAC_ERR_TIMEOUT);
            *abort = 1;
            break;
          }
          __nanosleep(32);
        }
      }
      __threadfence();
    }
  }
  consumers_sync();
}

// The producer's walk over its ring stages: layer l, projection j, this
// CTA's groups g of it, K chunks c, in the order the consumers take them.
struct StageCursor {
  int l, j, g, g1, c, nchunk, K, bx, nx;
  const bf16* W;
  bool done;
  __device__ __forceinline__ StageCursor(const DPass& a, int bx_, int nx_)
      : l(0), j(0), g(0), g1(0), c(0), nchunk(1), K(0), bx(bx_), nx(nx_), W(nullptr), done(a.L <= 0) {
    if (!done) {
      load(a);
      skip(a);
    }
  }
  __device__ __forceinline__ void load(const DPass& a) {
    const Proj P = proj_of(a, l, j);
    int g0;
    dgemv_group_range((P.n_pairs + kDecGroupPairs - 1) / kDecGroupPairs, nx, bx, g0, g1);
    g = g0;
    c = 0;
    K = P.K;
    W = P.W;
    nchunk = (P.K + kPKC - 1) / kPKC;
  }
  // past projections that give this CTA no group
  __device__ __forceinline__ void skip(const DPass& a) {
    while (!done && g >= g1) {
      if (++j == 4) {
        j = 0;
        if (++l == a.L) {
          done = true;
          break;
        }
      }
      load(a);
    }
  }
  __device__ __forceinline__ void next(const DPass& a) {
    if (++c == nchunk) {
      c = 0;
      ++g;
      skip(a);
    }
  }
  __device__ __forceinline__ const bf16* src() const { return W + (size_t)g * kPTR * K + (size_t)kPTR * c * kPKC; }
  __device__ __forceinline__ uint32_t bytes() const { return (uint32_t)(kPTR * min(kPKC, K - c * kPKC) * 2); }
};

// xs[b] = bf16(RMSNorm(X[b]) * g) in A-fragment order; the mean square from
// the producers' sums-of-squares partials (ssq_in[b][n_ssq], in index order).
constexpr int kNormIt = 2;  // items (8 elements) per thread the norm prologue holds in registers

// The gains a thread's first kNormIt prologue items use: constant, so they are
// loaded before the grid barrier that precedes the prologue.
template <int NB>
__device__ __forceinline__ void load_gain(const bf16* gain, int K, uint4 (&pg)[kNormIt]) {
  const int tid = threadIdx.x, n8 = K / 8;
#pragma unroll
  for (int j = 0; j < kNormIt; ++j) {
    const int m = tid + j * kPC * 32;
    pg[j] = make_uint4(0u, 0u, 0u, 0u);
    if (m < NB * n8) pg[j] = *reinterpret_cast<const uint4*>(gain + (m - (m / n8) * n8) * 8);
  }
}

template <int NB>
__device__ void prologue_norm(const DPass& a, const float* ssq_in, int n_ssq, const bf16* gain, int K, bf16* xs,
                              float (*red)[32], float* rr, const uint4 (&pg)[kNormIt]) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // the rows are loaded with the sums of squares, so that the prologue waits
  // on one round trip to L2 (up to kNormIt items per thread)
  constexpr int kIt = kNormIt;
  const int n8 = K / 8, items = NB * n8;
  const bool held = items <= kIt * kPC * 32;
  float4 px0[kIt], px1[kIt];
  if (held) {
#pragma unroll
    for (int j = 0; j < kIt; ++j) {
      const int m = tid + j * kPC * 32;
      if (m < items) {
        const int b = m / n8, k = (m - b * n8) * 8;
        px0[j] = __ldcg(reinterpret_cast<const float4*>(a.X + (size_t)b * K + k));
        px1[j] = __ldcg(reinterpret_cast<const float4*>(a.X + (size_t)b * K + k + 4));
      }
    }
  }
  float sacc[NB];
#pragma unroll
  for (int b = 0; b < NB; ++b) sacc[b] = 0.f;
  for (int c = tid; c < n_ssq; c += kPC * 32)
#pragma unroll
    for (int b = 0; b < NB; ++b) sacc[b] += __ldcg(ssq_in + (size_t)b * n_ssq + c);
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    const float t = p_allsum(sacc[b]);
    if (lane == 0) red[warp][b] = t;
  }
  consumers_sync();
  if (tid < NB) {
    float t = 0.f;
    for (int w = 0; w < kPC; ++w) t += red[w][tid];
    rr[tid] = 1.0f / sqrtf(t / (float)K + a.eps);
  }
  consumers_sync();
  if (held) {
#pragma unroll
    for (int j = 0; j < kIt; ++j) {
      const int m = tid + j * kPC * 32;
      if (m < items) {
        const int b = m / n8, k = (m - b * n8) * 8;
        float gf[8];
        bf16x8(pg[j], gf);
        const float r = rr[b];
        const float xv[8] = {px0[j].x, px0[j].y, px0[j].z, px0[j].w, px1[j].x, px1[j].y, px1[j].z, px1[j].w};
        uint32_t* row = reinterpret_cast<uint32_t*>(xs + (size_t)b * K);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const __nv_bfloat162 v =
              __floats2bfloat162_rn((xv[2 * q] * r) * gf[2 * q], (xv[2 * q + 1] * r) * gf[2 * q + 1]);
          row[afrag_pos(k + 2 * q) >> 1] = *reinterpret_cast<const uint32_t*>(&v);
        }
      }
    }
    consumers_sync();
    return;
  }
#pragma unroll 2
  for (int m = tid; m < NB * n8; m += kPC * 32) {
    const int b = m / n8, k = (m - b * n8) * 8;
    const uint4 gv = *reinterpret_cast<const uint4*>(gain + k);
    const float4 x0 = __ldcg(reinterpret_cast<const float4*>(a.X + (size_t)b * K + k));
    const float4 x1 = __ldcg(reinterpret_cast<const float4*>(a.X + (size_t)b * K + k + 4));
    float gf[8];
    bf16x8(gv, gf);
    const float r = rr[b];
    const float xv[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
    uint32_t* row = reinterpret_cast<uint32_t*>(xs + (size_t)b * K);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const __nv_bfloat162 v = __floats2bfloat162_rn((xv[2 * j] * r) * gf[2 * j], (xv[2 * j + 1] * r) * gf[2 * j + 1]);
      row[afrag_pos(k + 2 * j) >> 1] = *reinterpret_cast<const uint32_t*>(&v);
    }
  }
  consumers_sync();
}

// xs[b] = src[b] (bf16 rows of width K) in A-fragment order.
template <int NB>
__device__ void prologue_copy(const bf16* src, int K, bf16* xs) {
  const int tid = threadIdx.x, n8 = K / 8, items = NB * n8;
  // batches of kIt items per thread, every load of a batch issued before its
  // first store (a 9-warp block has 168 registers per thread)
  constexpr int kIt = 4;
  for (int base = 0; base < items; base += kIt * kPC * 32) {
    uint4 v[kIt];
#pragma unroll
    for (int j = 0; j < kIt; ++j) {
      const int m = base + tid + j * kPC * 32;
      if (m < items) {
        const int b = m / n8, k = (m - b * n8) * 8;
        v[j] = __ldcg(reinterpret_cast<const uint4*>(src + (size_t)b * K + k));
      }
    }
#pragma unroll
    for (int j = 0; j < kIt; ++j) {
      const int m = base + tid + j * kPC * 32;
      if (m < items) {
        const int b = m / n8, k = (m - b * n8) * 8;
        uint32_t* row = reinterpret_cast<uint32_t*>(xs + (size_t)b * K);
        row[afrag_pos(k) >> 1] = v[j].x;
        row[afrag_pos(k + 2) >> 1] = v[j].y;
        row[afrag_pos(k + 4) >> 1] = v[j].z;
        row[afrag_pos(k + 6) >> 1] = v[j].w;
      }
    }
  }
  consumers_sync();
}

struct Ring {
  uint8_t* stages;
  uint64_t* full;
  uint64_t* empty;
  int ns, stage;
  uint32_t phase;
};

// One projection of layer l over this CTA's groups [g0, g1): the products on
// the tensor pipe (weights as B, the NB input vectors as A), the 8 warps'
// shares added in warp order by a rotating warp, which runs the epilogue.
// Returns this thread's residual sum of squares (sequence lane / 4).
template <int NB, int J>
__device__ float consume(const DPass& a, int l, const Proj& P, int g0, int g1, const bf16* xs, Ring& R,
                         float2 (*pacc)[kPC][32], volatile int* ring_dead) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gq = lane >> 2, tq = lane & 3;
  const int K = P.K, nchunk = (K + kPKC - 1) / kPKC;
  const int hidden = a.hidden, half = kPHD / 2;
  const uint32_t st_lane = smem_u32(R.stages) + (uint32_t)lane * 16;
  float ssq = 0.f;
  for (int g = g0; g < g1; ++g) {
    const int pb = (g - g0) & 1, ew = (g - g0) % kPC;
    const int p = g * kDecGroupPairs + tq;
    const bool epi = warp == ew && gq < NB && p < P.n_pairs;
    float e1 = 0.f, e2 = 0.f;  // epilogue operands, loaded ahead
    if (epi) {
      if constexpr (J == 0) {
        const int sec = p / (hidden / 2), within = p - sec * (hidden / 2), e = within % half;
        if (sec < 2) {
          e1 = a.rope_cos[(size_t)a.pos * half + e];
          e2 = a.rope_sin[(size_t)a.pos * half + e];
        }
      } else if constexpr (J == 1 || J == 3) {
        e1 = __ldcg(a.X + (size_t)gq * hidden + 2 * p);
        e2 = __ldcg(a.X + (size_t)gq * hidden + 2 * p + 1);
      }
    }
    float d[4][4];
#pragma unroll
    for (int u = 0; u < 4; ++u) d[u][0] = d[u][1] = d[u][2] = d[u][3] = 0.f;
    for (int c = 0; c < nchunk; ++c) {
      const int k0 = c * kPKC, n32 = min(kPKC, K - k0) >> 5;
      const int i0 = n32 * warp / kPC, i1 = n32 * (warp + 1) / kPC;
      // ring waits ignore the grid barrier's give-up flag: a stage is handed
      // back only after its copy landed; once one ring wait times out the
      // ring is dead and the others return at once
      bool ok = true;
      if (lane == 0) ok = mbar_wait(&R.full[R.stage], R.phase, a.wait_limit, ring_dead);
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (ok) {
        const uint32_t st = st_lane + (uint32_t)((size_t)R.stage * kPStage);
        const bf16* xrow = xs + (size_t)gq * K + k0 + tq * 8;
        int i = i0;
        for (; i + 4 <= i1; i += 4) {
          uint32_t bf[4][4];
          uint4 xa[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            ldsm_x4(st + (uint32_t)(i + u) * 512u, bf[u][0], bf[u][1], bf[u][2], bf[u][3]);
            xa[u] = gq < NB ? *reinterpret_cast<const uint4*>(xrow + (i + u) * 32) : make_uint4(0u, 0u, 0u, 0u);
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
          const uint4 xv = gq < NB ? *reinterpret_cast<const uint4*>(xrow + i * 32) : make_uint4(0u, 0u, 0u, 0u);
          mma_bf16(d[0], xv.x, 0u, xv.y, 0u, b0, b1);
          mma_bf16(d[0], xv.z, 0u, xv.w, 0u, b2, b3);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&R.empty[R.stage]);
      } else if (lane == 0) {
        // a stage whose wait failed is not handed back, so it is never
        // refilled; the producer sees the flag and stops
        set_error(a.err, VLAC_ERR_TIMEOUT);
        *ring_dead = 1;
      }
      if (++R.stage == R.ns) {
        R.stage = 0;
        R.phase ^= 1u;
      }
    }
    if (gq < NB)
      pacc[pb][warp][lane] =
          make_float2(((d[0][0] + d[1][0]) + d[2][0]) + d[3][0], ((d[0][1] + d[1][1]) + d[2][1]) + d[3][1]);
    consumers_sync();  // also: every warp has finished the previous group's epilogue
    if (epi) {
      float y1 = 0.f, y2 = 0.f;
#pragma unroll
      for (int w = 0; w < kPC; ++w) {
        const float2 v = pacc[pb][w][lane];
        y1 += v.x;
        y2 += v.y;
      }
      const int b = gq;
      if constexpr (J == 0) {
        const int sec = p / (hidden / 2), within = p - sec * (hidden / 2);
        const int h = within / half, e = within - h * half;
        float o1 = y1, o2 = y2;
        if (sec < 2) {
          o1 = y1 * e1 - y2 * e2;
          o2 = y2 * e1 + y1 * e2;
        }
        bf16* dst = sec == 0 ? a.Q + (size_t)b * hidden + (size_t)h * kPHD
                             : (sec == 1 ? a.Kc : a.Vc) + (size_t)l * a.kv_layer + (size_t)b * a.kv_seq_stride +
                                   ((size_t)h * a.Tc + a.pos) * kPHD;
        dst[e] = __float2bfloat16_rn(o1);
        dst[e + half] = __float2bfloat16_rn(o2);
      } else if constexpr (J == 2) {
        a.G[(size_t)b * a.ffn + p] = __float2bfloat16_rn((y1 / (1.0f + expf(-y1))) * y2);
      } else {
        const float n1 = e1 + y1, n2 = e2 + y2;
        a.X[(size_t)b * hidden + 2 * p] = n1;
        a.X[(size_t)b * hidden + 2 * p + 1] = n2;
        ssq += fmaf(n1, n1, n2 * n2);
      }
    }
  }
  return ssq;
}

// This CTA's sums of squares of the residual elements it wrote, per sequence.
template <int NB>
__device__ void write_ssq(const DPass& a, float ssq, float (*red)[32]) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  red[warp][lane] = ssq;
  consumers_sync();
  if (tid < NB) {
    float t = 0.f;
    for (int w = 0; w < kPC; ++w)
      for (int j = 0; j < 4; ++j) t += red[w][tid * 4 + j];
    a.ssq[(size_t)tid * gridDim.x + blockIdx.x] = t;
  }
  consumers_sync();
}

// Single-query attention of layer l: items (sequence, head, key range) spread
// over the CTAs.  The item's keys are cut evenly over the eight warps, a key
// per lane (online softmax per warp), and the eight warps are combined in
// order.  With one range per head the CTA writes the output row; with
// several, it writes its range's partial and the last range to finish
// combines the ranges in order (no CTA waits for another).
// The key range [k0, k1) of attention item `item` (sequence, head, range).
__device__ __forceinline__ void item_keys(const DPass& a, int item, int& b, int& h, int& ch, int& k0, int& k1) {
  const int nkeys = min(a.pos + 1, a.Tc), nch = a.attn_chunks;
  const int bh = item / nch;
  ch = item - bh * nch;
  b = bh / a.n_heads;
  h = bh - b * a.n_heads;
  k0 = (int)(((long long)nkeys * ch) / nch);
  k1 = (int)(((long long)nkeys * (ch + 1)) / nch);
}

// Staging of the first item's K and V rows for layer l into shared memory
// (thread 0): the keys before pos were written by earlier passes, so their
// rows can be on their way a layer ahead.  [*lo, *hi): the staged keys.
__device__ __forceinline__ void stage_kv(const DPass& a, int NBxH, int l, bf16* kvK, bf16* kvV, uint64_t* bar,
                                         int* lo, int* hi) {
  *lo = *hi = 0;
  if (a.kv_keys <= 0 || (int)blockIdx.x >= NBxH * a.attn_chunks) return;
  int b, h, ch, k0, k1;
  item_keys(a, blockIdx.x, b, h, ch, k0, k1);
  const int kend = min(k1, min(a.pos, k0 + a.kv_keys));
  if (kend <= k0) return;
  const size_t off = (size_t)l * a.kv_layer + (size_t)b * a.kv_seq_stride + ((size_t)h * a.Tc + k0) * kPHD;
  const uint32_t bytes = (uint32_t)(kend - k0) * kPHD * 2;
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // after the generic reads of the last layer
  mbar_expect_tx(bar, 2 * bytes);
  bulk_g2s(kvK, a.Kc + off, bytes, bar);
  bulk_g2s(kvV, a.Vc + off, bytes, bar);
  *lo = k0;
  *hi = kend;
}

template <int NB>
__device__ void attention(const DPass& a, int l, float* qs, float* wm, float* wl, float (*wacc)[kPHD],
                          volatile int* s_last, const bf16* kvK, const bf16* kvV, int kv_lo, int kv_hi) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int hidden = a.hidden, nkeys = min(a.pos + 1, a.Tc), nch = a.attn_chunks;
  for (int item = blockIdx.x; item < NB * a.n_heads * nch; item += gridDim.x) {
    if (item != (int)blockIdx.x) kv_lo = kv_hi = 0;  // only the first item is staged
    const int bh = item / nch, ch = item - bh * nch;
    const int b = bh / a.n_heads, h = bh - b * a.n_heads;
    const int k0 = (int)(((long long)nkeys * ch) / nch), k1 = (int)(((long long)nkeys * (ch + 1)) / nch);
    const bf16* Kh = a.Kc + (size_t)l * a.kv_layer + (size_t)b * a.kv_seq_stride + (size_t)h * a.Tc * kPHD;
    const bf16* Vh = a.Vc + (size_t)l * a.kv_layer + (size_t)b * a.kv_seq_stride + (size_t)h * a.Tc * kPHD;
    if (tid < kPHD) qs[tid] = __bfloat162float(__ldcg(a.Q + (size_t)b * hidden + (size_t)h * kPHD + tid));
    consumers_sync();
    float m_run = -INFINITY, l_run = 0.f, acc[4] = {0.f, 0.f, 0.f, 0.f};
    // the range's keys cut evenly over the eight warps (a key per lane)
    const int kw = (k1 - k0 + kPC - 1) / kPC, w0 = k0 + warp * kw, w1 = min(k1, w0 + kw);
    for (int j0 = w0; j0 < w1; j0 += 32) {
      const int jn = min(32, w1 - j0), j = j0 + lane;
      float s = -INFINITY;
      if (lane < jn) {
        uint4 kv[kPHD / 8];
        if (j >= kv_lo && j < kv_hi) {
          const uint4* kr = reinterpret_cast<const uint4*>(kvK + (size_t)(j - kv_lo) * kPHD);
#pragma unroll
          for (int v = 0; v < kPHD / 8; ++v) kv[v] = kr[v];
        } else {
          const uint4* kr = reinterpret_cast<const uint4*>(Kh + (size_t)j * kPHD);
#pragma unroll
          for (int v = 0; v < kPHD / 8; ++v) kv[v] = __ldcg(kr + v);
        }
        // four partial sums over the head dimension (element i mod 4),
        // added in a fixed order
        float dp[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int v = 0; v < kPHD / 8; ++v) {
          float f[8];
          bf16x8(kv[v], f);
#pragma unroll
          for (int i = 0; i < 8; ++i) dp[i & 3] = fmaf(f[i], qs[v * 8 + i], dp[i & 3]);
        }
        s = ((dp[0] + dp[1]) + (dp[2] + dp[3])) * a.scale;
      }
      const float m_new = fmaxf(m_run, p_allmax(s));
      const float corr = m_run == -INFINITY ? 0.f : expf(m_run - m_new);
      const float pr = s == -INFINITY ? 0.f : expf(s - m_new);
      l_run = l_run * corr + p_allsum(pr);
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[e] *= corr;
#pragma unroll 8
      for (int jj = 0; jj < jn; ++jj) {
        const float pj = __shfl_sync(0xffffffffu, pr, jj);
        const int jr = j0 + jj;
        const uint2 vv = (jr >= kv_lo && jr < kv_hi)
                             ? *reinterpret_cast<const uint2*>(kvV + (size_t)(jr - kv_lo) * kPHD + lane * 4)
                             : __ldcg(reinterpret_cast<const uint2*>(Vh + (size_t)jr * kPHD + lane * 4));
        acc[0] = fmaf(pj, __uint_as_float(vv.x << 16), acc[0]);
        acc[1] = fmaf(pj, __uint_as_float(vv.x & 0xFFFF0000u), acc[1]);
        acc[2] = fmaf(pj, __uint_as_float(vv.y << 16), acc[2]);
        acc[3] = fmaf(pj, __uint_as_float(vv.y & 0xFFFF0000u), acc[3]);
      }
      m_run = m_new;
    }
    if (lane == 0) {
      wm[warp] = m_run;
      wl[warp] = l_run;
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) wacc[warp][lane * 4 + e] = acc[e];
    consumers_sync();
    // this item's (max, sum, unnormalised output), warps in order
    float M = -INFINITY, L = 0.f, o = 0.f;
    if (tid < kPHD) {
      for (int w = 0; w < kPC; ++w) M = fmaxf(M, wm[w]);
      for (int w = 0; w < kPC; ++w) {
        const float f = wm[w] == -INFINITY ? 0.f : expf(wm[w] - M);
        L = fmaf(wl[w], f, L);
        o = fmaf(wacc[w][tid], f, o);
      }
    }
    if (nch == 1) {
      if (tid < kPHD) a.AO[(size_t)b * hidden + (size_t)h * kPHD + tid] = __float2bfloat16_rn(o / L);
      consumers_sync();
      continue;
    }
    float* part = a.attn_part + (size_t)bh * a.part_stride;
    if (tid < kPHD) {
      part[(size_t)ch * (kPHD + 2) + 2 + tid] = o;
      if (tid == 0) {
        part[(size_t)ch * (kPHD + 2)] = M;
        part[(size_t)ch * (kPHD + 2) + 1] = L;
      }
    }
    // the CTA barrier collects the partial's stores; thread 0's ticket
    // releases them at GPU scope and acquires the other ranges' partials
    consumers_sync();
    if (tid == 0) {
      unsigned t;
      asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(t) : "l"(a.attn_cnt + bh) : "memory");
      *s_last = t == (unsigned)(nch - 1);
    }
    consumers_sync();
    if (*s_last) {
      if (tid < kPHD) {
        float Mx = -INFINITY;
        for (int c = 0; c < nch; ++c) Mx = fmaxf(Mx, __ldcg(part + (size_t)c * (kPHD + 2)));
        float Lt = 0.f, ot = 0.f;
        for (int c = 0; c < nch; ++c) {
          const float mc = __ldcg(part + (size_t)c * (kPHD + 2));
          const float f = mc == -INFINITY ? 0.f : expf(mc - Mx);
          Lt = fmaf(__ldcg(part + (size_t)c * (kPHD + 2) + 1), f, Lt);
          ot = fmaf(__ldcg(part + (size_t)c * (kPHD + 2) + 2 + tid), f, ot);
        }
        a.AO[(size_t)b * hidden + (size_t)h * kPHD + tid] = __float2bfloat16_rn(ot / Lt);
      }
      if (tid == 0) a.attn_cnt[bh] = 0u;  // ready for the next layer (after the grid barriers)
    }
    consumers_sync();
  }
}

template <int NB>
__global__ void __launch_bounds__((kPC + 1) * 32, 1) dpass_kernel(const __grid_constant__ DPass a) {
  extern __shared__ uint8_t dsm_raw[];
  __shared__ __align__(8) uint64_t full_bar[kPMaxNS];
  __shared__ __align__(8) uint64_t empty_bar[kPMaxNS];
  __shared__ float red[kPC][32];
  __shared__ float rr[NB];
  __shared__ __align__(8) float2 pacc[2][kPC][32];
  __shared__ float qs[kPHD], wm[kPC], wl[kPC];
  __shared__ float wacc[kPC][kPHD];
  __shared__ int abort_flag, ring_flag, last_flag;
  __shared__ __align__(8) uint64_t kv_bar;  // the staged K/V rows of the layer in flight
  __shared__ int kv_lo, kv_hi, kv_dead;
  uint8_t* dsm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dsm_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int xs_bytes = ((NB * max(a.hidden, a.ffn) * 2 + 1023) / 1024) * 1024;
  bf16* xs = reinterpret_cast<bf16*>(dsm);
  Ring R{dsm + xs_bytes, full_bar, empty_bar, a.ns, 0, 0u};
  bf16* kvK = reinterpret_cast<bf16*>(dsm + xs_bytes + (size_t)a.ns * kPStage);
  bf16* kvV = kvK + (size_t)a.kv_keys * kPHD;
  if (threadIdx.x == 0) {
    for (int s = 0; s < a.ns; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], kPC);
    }
    mbar_init(&kv_bar, 1);
    abort_flag = 0;
    ring_flag = 0;
    kv_dead = 0;
    mbar_fence_init();
  }
  __syncthreads();
  volatile int* abort = &abort_flag;  // a grid barrier gave up: stop waiting on other CTAs
  volatile int* ring_dead = &ring_flag;  // a ring wait timed out: the weight ring is abandoned

  if (warp == kPC) {
    // ---- producer: every projection of every layer, in consumption order ----
    if (lane == 0) {
      uint32_t issued = 0;
      StageCursor cur(a, blockIdx.x, gridDim.x);
      while (!cur.done) {
        if (!mbar_wait(&R.empty[R.stage], R.phase ^ 1u, a.wait_limit, ring_dead)) {
          // the consumers stopped releasing stages: nothing more is issued
          set_error(a.err, VLAC_ERR_TIMEOUT);
          *ring_dead = 1;
          break;
        }
        const uint32_t bytes = cur.bytes();
        mbar_expect_tx(&R.full[R.stage], bytes);
        bulk_g2s(R.stages + (size_t)R.stage * kPStage, cur.src(), bytes, &R.full[R.stage]);
        ++issued;
        if (++R.stage == R.ns) {
          R.stage = 0;
          R.phase ^= 1u;
        }
        cur.next(a);
      }
      // no bulk copy may still be landing in this CTA's shared memory when it
      // exits; on the normal path the consumers waited for every one already
      ring_drain(R.full, R.ns, R.stage, R.phase, issued);
    }
    return;
  }

  // ---- consumers ----
  unsigned epoch = 0;
  if (threadIdx.x == 0) stage_kv(a, NB * a.n_heads, 0, kvK, kvV, &kv_bar, &kv_lo, &kv_hi);
  int kv_issued = -1;  // the last layer whose staging copy was issued (thread 0's view is what counts)
  if (threadIdx.x == 0 && kv_hi > kv_lo) kv_issued = 0;
  for (int l = 0; l < a.L; ++l) {
    int g0, g1;
    // q/k/v: RMSNorm of the residual rows (sums of squares from the decode
    // embedding for layer 0, else from the previous down-projection)
    uint4 pga[kNormIt];
    load_gain<NB>(a.g_attn[l], a.hidden, pga);  // constant: before the barrier
    if (l > 0) grid_sync(a, ++epoch, abort);
    if (threadIdx.x == 0) {
      // this CTA's attention items: their older K/V rows (written by earlier
      // passes) start on their way into L2 while the q/k/v projection runs
      for (int item = blockIdx.x; item < NB * a.n_heads; item += gridDim.x) {
        const int b = item / a.n_heads, h = item - b * a.n_heads;
        const size_t off = (size_t)l * a.kv_layer + (size_t)b * a.kv_seq_stride + (size_t)h * a.Tc * kPHD;
        const uint32_t bytes = (uint32_t)(min(a.pos, a.Tc) * kPHD * 2);
        if (bytes >= 16) {
          prefetch_l2(a.Kc + off, bytes & ~15u);
          prefetch_l2(a.Vc + off, bytes & ~15u);
        }
      }
    }
    {
      const Proj P = proj_of(a, l, 0);
      prologue_norm<NB>(a, l == 0 ? a.ssq0 : a.ssq, l == 0 ? a.n_ssq0 : (int)gridDim.x, a.g_attn[l], P.K, xs, red, rr,
                        pga);
      dgemv_group_range((P.n_pairs + kDecGroupPairs - 1) / kDecGroupPairs, gridDim.x, blockIdx.x, g0, g1);
      consume<NB, 0>(a, l, P, g0, g1, xs, R, pacc, ring_dead);
    }
    grid_sync(a, ++epoch, abort);
    {
      // the staged rows of this layer (the CTA barrier inside the attention
      // phase orders thread 0's flags before the other threads' reads)
      int lo = 0, hi = 0;
      if (threadIdx.x == 0 && kv_hi > kv_lo && !kv_dead) {
        if (mbar_wait(&kv_bar, (uint32_t)l & 1u, a.wait_limit, ring_dead)) {
          lo = kv_lo;
          hi = kv_hi;
        } else {
          set_error(a.err, VLAC_ERR_TIMEOUT);
          kv_dead = 1;  // read from global from now on; the copy is waited for at exit
        }
      }
      if (threadIdx.x == 0) {
        kv_lo = lo;
        kv_hi = hi;
      }
      consumers_sync();
      lo = kv_lo;
      hi = kv_hi;
      // every reader observes the copy's completion itself (it completed: no wait)
      if (threadIdx.x != 0 && hi > lo) mbar_wait(&kv_bar, (uint32_t)l & 1u, kWaitLimit, ring_dead);
      attention<NB>(a, l, qs, wm, wl, wacc, &last_flag, kvK, kvV, lo, hi);
      // attention ended with a CTA barrier: the buffer is free for the next layer
      if (threadIdx.x == 0 && !kv_dead && l + 1 < a.L) {
        stage_kv(a, NB * a.n_heads, l + 1, kvK, kvV, &kv_bar, &kv_lo, &kv_hi);
        if (kv_hi > kv_lo) kv_issued = l + 1;
      }
    }
    grid_sync(a, ++epoch, abort);
    {  // o-projection + residual
      const Proj P = proj_of(a, l, 1);
      prologue_copy<NB>(a.AO, P.K, xs);
      dgemv_group_range((P.n_pairs + kDecGroupPairs - 1) / kDecGroupPairs, gridDim.x, blockIdx.x, g0, g1);
      write_ssq<NB>(a, consume<NB, 1>(a, l, P, g0, g1, xs, R, pacc, ring_dead), red);
    }
    uint4 pgf[kNormIt];
    load_gain<NB>(a.g_ffn[l], a.hidden, pgf);
    grid_sync(a, ++epoch, abort);
    {  // gate/up with the MLP RMSNorm, SwiGLU
      const Proj P = proj_of(a, l, 2);
      prologue_norm<NB>(a, a.ssq, (int)gridDim.x, a.g_ffn[l], P.K, xs, red, rr, pgf);
      dgemv_group_range((P.n_pairs + kDecGroupPairs - 1) / kDecGroupPairs, gridDim.x, blockIdx.x, g0, g1);
      consume<NB, 2>(a, l, P, g0, g1, xs, R, pacc, ring_dead);
    }
    grid_sync(a, ++epoch, abort);
    {  // down + residual
      const Proj P = proj_of(a, l, 3);
      prologue_copy<NB>(a.G, P.K, xs);
      dgemv_group_range((P.n_pairs + kDecGroupPairs - 1) / kDecGroupPairs, gridDim.x, blockIdx.x, g0, g1);
      write_ssq<NB>(a, consume<NB, 3>(a, l, P, g0, g1, xs, R, pacc, ring_dead), red);
    }
  }
  // a staging copy whose wait gave up may still be landing: wait for it
  // (bounded, deaf to the give-up flags) before the CTA exits
  if (threadIdx.x == 0 && kv_dead && kv_issued >= 0) {
    int never = 0;
    mbar_wait(&kv_bar, (uint32_t)kv_issued & 1u, kWaitLimit, &never);
  }
}

template <int NB>
int dpass_launch(const DPass& a, int n_sm, cudaStream_t st) {
  const size_t smem = 1024 + ((size_t)NB * std::max(a.hidden, a.ffn) * 2 + 1023) / 1024 * 1024 + (size_t)a.ns * kPStage +
                      dpass_kv_bytes(a.kv_keys);
  static size_t smem_set = 0;
  if (smem > smem_set) {
    if (cudaFuncSetAttribute(dpass_kernel<NB>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
      return VLAC_ERR_UNSUPPORTED;  // more than a block may have: the per-projection chain runs instead
    smem_set = smem;
  }
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, dpass_kernel<NB>, (kPC + 1) * 32, smem) != cudaSuccess ||
      per_sm < 1)
    return VLAC_ERR_UNSUPPORTED;
  if (cudaMemsetAsync(a.bar, 0, sizeof(unsigned), st) != cudaSuccess) return VLAC_ERR_CUDA;
  if (a.attn_chunks > 1 && cudaMemsetAsync(a.attn_cnt, 0, (size_t)NB * a.n_heads * sizeof(unsigned), st) != cudaSuccess)
    return VLAC_ERR_CUDA;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_sm);
  cfg.blockDim = dim3((kPC + 1) * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, dpass_kernel<NB>, a) == cudaSuccess ? VLAC_OK : VLAC_ERR_CUDA;
}

}  // namespace

size_t dpass_kv_bytes(int kv_keys) { return (size_t)2 * std::max(kv_keys, 0) * kPHD * 2; }
size_t dpass_smem_bytes(int hidden, int ffn, int nb, int ns, int kv_keys) {
  return 1024 + ((size_t)nb * std::max(hidden, ffn) * 2 + 1023) / 1024 * 1024 + (size_t)ns * kPStage +
         dpass_kv_bytes(kv_keys);
}

int dpass_kv_fit(int hidden, int ffn, int nb, int ns) {
  // what the device lets one block have, less the kernel's static shared
  // memory and the dynamic part without staging
  int dev = 0, optin = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
    return 0;
  cudaFuncAttributes fa{};
  if (cudaFuncGetAttributes(&fa, nb == 1 ? dpass_kernel<1> : dpass_kernel<2>) != cudaSuccess) return 0;
  const long long room = (long long)optin - (long long)fa.sharedSizeBytes - (long long)dpass_smem_bytes(hidden, ffn, nb, ns, 0);
  return room > 0 ? (int)(room / (long long)dpass_kv_bytes(1)) : 0;
}

bool dpass_supported(int hidden, int ffn, int n_heads, int head_dim, int nb, int ns) {
  return head_dim == kPHD && n_heads * head_dim == hidden && nb >= 1 && nb <= 2 && hidden % 64 == 0 && ffn % 64 == 0 &&
         ns >= 2 && ns <= kPMaxNS && (size_t)nb * std::max(hidden, ffn) * 2 + (size_t)ns * kPStage + 1024 <= 200 * 1024;
}

int launch_dpass(const DPass& a, int nb, int n_sm, cudaStream_t st) {
  return nb == 1 ? dpass_launch<1>(a, n_sm, st) : dpass_launch<2>(a, n_sm, st);
}

}  // namespace vlac
