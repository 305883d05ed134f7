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

// ---- bf16 path: tensor cores (mma.m16n8k16), flash-attention style ----------------
//
// One block of 4 warps per (64 query rows of one sequence, head); warp w owns
// 16 rows.  Key tiles of 64 positions (aligned to absolute positions) are
// double-buffered in shared memory by TMA (cp.async.bulk.tensor) from the
// cache's 3-D tensor maps {head_dim, position, sequence x layer x head}: one
// 64 x 64 box per 64 dimensions of K and of V, 128-byte swizzled, completing
// on the buffer's mbarrier; keys at or past Tc lie outside the map and arrive
// as zeros.  Per tile: S = Q K^T on the tensor cores (fp32 accumulators),
// scale, causal mask by the row's absolute position, online softmax in fp32,
// P rounded to bf16 and O += P V on the tensor cores.  Masked keys contribute
// exact zeros and a fully masked tile leaves a row's state unchanged, so a
// row's result does not depend on the other rows of its block.  The waits
// are bounded: a wait that gives up latches VLAC_ERR_TIMEOUT, the block
// stops, and thread 0 lets the copies still in flight land before it exits.
namespace {

constexpr int kAQ = 64;   // query rows per block
constexpr int kAK = 64;   // keys per tile
constexpr int kAW = 4;    // warps per block

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* tm, int x, int y, int z, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
      "[%5];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tm)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
      : "memory");
}
// Byte offset of (key r, dimension e) in a tile of 64-dimension boxes, each
// box 64 rows of 128 bytes with the 16-byte chunks of row r XOR-ed by r % 8.
__device__ __forceinline__ uint32_t sw_off(int r, int e) {
  return (uint32_t)((e >> 6) * (kAK * 128) + r * 128 + ((((e & 63) >> 3) ^ (r & 7)) << 4));
}

template <int HD>
__global__ void __launch_bounds__(kAW * 32) attn_mma_kernel(Rows rows, int n_heads, const bf16* __restrict__ Q,
                                                            const __grid_constant__ KvMaps kvm, int z_seq,
                                                            int z_layer, int Tc, int P, int parallel, int n_action,
                                                            float scale, bf16* __restrict__ O,
                                                            int* __restrict__ err, uint32_t wait_limit) {
  pdl_wait();
  pdl_trigger();
  constexpr int KS = HD / 16;       // k-steps of S = Q K^T
  constexpr int ND = HD / 8;        // 8-column tiles of O
  constexpr uint32_t kTile = (uint32_t)kAK * HD * 2;  // bytes of one K (or V) tile
  extern __shared__ __align__(1024) uint8_t dsm[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dsm) + 1023) & ~uintptr_t(1023));
  // [buf][K | V][tile]
  __shared__ __align__(8) uint64_t full[2];
  __shared__ int lim_s[kAQ];
  __shared__ int maxlim_s, abort_s, never_s;
  const int qt = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int cnt = rows.off[b + 1] - rows.off[b];
  const int i0 = qt * kAQ;
  if (i0 >= cnt) return;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, t = lane & 3;
  const int hidden = n_heads * HD, r0 = rows.off[b] + i0;
  if (tid < kAQ) {
    int lim = 0;
    if (i0 + tid < cnt) {
      const int pos = rows.idx[(size_t)b * rows.idx_stride + i0 + tid];
      lim = (parallel && pos >= P) ? P + n_action : pos + 1;
      lim = min(lim, Tc);
    }
    lim_s[tid] = lim;
  }
  if (tid == 0) {
    mbar_init(&full[0], 1);
    mbar_init(&full[1], 1);
    abort_s = 0;
    never_s = 0;
    mbar_fence_init();
  }
  __syncthreads();
  if (tid == 0) {
    int m = 0;
    for (int q = 0; q < kAQ; ++q) m = max(m, lim_s[q]);
    maxlim_s = m;
  }
  const int z = b * z_seq + z_layer + h;
  const uint32_t sm_base = smem_u32(sm);
  auto ks_of = [&](int buf) { return sm_base + (uint32_t)(2 * buf) * kTile; };
  auto vs_of = [&](int buf) { return sm_base + (uint32_t)(2 * buf + 1) * kTile; };
  // issued by thread 0 only
  auto load_tile = [&](int tile, int buf) {
    mbar_expect_tx(&full[buf], 2 * kTile);
#pragma unroll
    for (int hh = 0; hh < HD / 64; ++hh) {
      tma_load_3d(ks_of(buf) + (uint32_t)hh * (kAK * 128), &kvm.k, hh * 64, tile * kAK, z, &full[buf]);
      tma_load_3d(vs_of(buf) + (uint32_t)hh * (kAK * 128), &kvm.v, hh * 64, tile * kAK, z, &full[buf]);
    }
  };
  __syncthreads();
  const int n_tiles = (maxlim_s + kAK - 1) / kAK;
  if (tid == 0 && n_tiles > 0) load_tile(0, 0);
  // this warp's Q rows as A fragments (rows past the block's rows are zero)
  const int ra = warp * 16 + g, rb = ra + 8;  // rows of the block held by this thread
  uint32_t qa[KS][4];
  {
    const bool va = i0 + ra < cnt, vb = i0 + rb < cnt;
    const bf16* qpa = Q + (size_t)(r0 + (va ? ra : 0)) * hidden + (size_t)h * HD;
    const bf16* qpb = Q + (size_t)(r0 + (vb ? rb : 0)) * hidden + (size_t)h * HD;
#pragma unroll
    for (int ks = 0; ks < KS; ++ks) {
      const int e = 16 * ks + 2 * t;
      qa[ks][0] = va ? *reinterpret_cast<const uint32_t*>(qpa + e) : 0u;
      qa[ks][1] = vb ? *reinterpret_cast<const uint32_t*>(qpb + e) : 0u;
      qa[ks][2] = va ? *reinterpret_cast<const uint32_t*>(qpa + e + 8) : 0u;
      qa[ks][3] = vb ? *reinterpret_cast<const uint32_t*>(qpb + e + 8) : 0u;
    }
  }
  const int lim_a = lim_s[ra], lim_b = lim_s[rb];
  float o[ND][4];
#pragma unroll
  for (int nd = 0; nd < ND; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;
  float m_a = -INFINITY, m_b = -INFINITY, l_a = 0.f, l_b = 0.f;  // per-thread partial row sums
  int tile = 0;
  for (; tile < n_tiles; ++tile) {
    const int buf = tile & 1;
    // buffer buf ^ 1 was released by the previous tile's closing barrier
    if (tid == 0 && tile + 1 < n_tiles) load_tile(tile + 1, buf ^ 1);
    if (!mbar_wait(&full[buf], (uint32_t)(tile >> 1) & 1u, wait_limit, &abort_s)) {
      set_error(err, VLAC_ERR_TIMEOUT);
      abort_s = 1;
    }
    __syncthreads();
    if (abort_s) break;
    // S = Q K^T for 64 keys: 8 n-tiles of 8 keys
    float sc[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) sc[nt][0] = sc[nt][1] = sc[nt][2] = sc[nt][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < KS; ++ks) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {  // n-tiles 2np, 2np + 1
        // matrices: (keys 16np + 0..7, dims 16ks), (same keys, dims 16ks + 8), next 8 keys likewise
        const int mi = lane >> 3, rr = lane & 7;
        const int key = 16 * np + (mi >> 1) * 8 + rr, dim = 16 * ks + (mi & 1) * 8;
        uint32_t k0, k1, k2, k3;
        ldsm_x4(ks_of(buf) + sw_off(key, dim), k0, k1, k2, k3);
        mma_bf16(sc[2 * np], qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3], k0, k1);
        mma_bf16(sc[2 * np + 1], qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3], k2, k3);
      }
    }
    // scale, mask, online softmax (rows ra: elements 0, 1; rb: elements 2, 3)
    const int t0 = tile * kAK;
    float mx_a = m_a, mx_b = m_b;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const int key = t0 + nt * 8 + 2 * t;
      sc[nt][0] = key < lim_a ? sc[nt][0] * scale : -INFINITY;
      sc[nt][1] = key + 1 < lim_a ? sc[nt][1] * scale : -INFINITY;
      sc[nt][2] = key < lim_b ? sc[nt][2] * scale : -INFINITY;
      sc[nt][3] = key + 1 < lim_b ? sc[nt][3] * scale : -INFINITY;
      mx_a = fmaxf(mx_a, fmaxf(sc[nt][0], sc[nt][1]));
      mx_b = fmaxf(mx_b, fmaxf(sc[nt][2], sc[nt][3]));
    }
    mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, 1));
    mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, 2));
    mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, 1));
    mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, 2));
    const float base_a = mx_a == -INFINITY ? 0.f : mx_a, base_b = mx_b == -INFINITY ? 0.f : mx_b;
    const float corr_a = m_a == -INFINITY ? 0.f : expf(m_a - base_a);
    const float corr_b = m_b == -INFINITY ? 0.f : expf(m_b - base_b);
    m_a = mx_a;
    m_b = mx_b;
    l_a *= corr_a;
    l_b *= corr_b;
#pragma unroll
    for (int nd = 0; nd < ND; ++nd) {
      o[nd][0] *= corr_a;
      o[nd][1] *= corr_a;
      o[nd][2] *= corr_b;
      o[nd][3] *= corr_b;
    }
    uint32_t pa[4][4];  // P as A fragments of the 4 key k-steps
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const float p0 = expf(sc[nt][0] - base_a), p1 = expf(sc[nt][1] - base_a);
      const float p2 = expf(sc[nt][2] - base_b), p3 = expf(sc[nt][3] - base_b);
      l_a += p0 + p1;
      l_b += p2 + p3;
      pa[nt >> 1][(nt & 1) * 2 + 0] = pack_bf16(p0, p1);
      pa[nt >> 1][(nt & 1) * 2 + 1] = pack_bf16(p2, p3);
    }
    // O += P V: k-steps of 16 keys, 8-column tiles of V (transposed loads)
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
      for (int np = 0; np < ND / 2; ++np) {  // column tiles 2np, 2np + 1
        const int mi = lane >> 3, rr = lane & 7;
        const int key = 16 * kk + (mi & 1) * 8 + rr, dim = 16 * np + (mi >> 1) * 8;
        uint32_t v0, v1, v2, v3;
        ldsm_x4_t(vs_of(buf) + sw_off(key, dim), v0, v1, v2, v3);
        mma_bf16(o[2 * np], pa[kk][0], pa[kk][1], pa[kk][2], pa[kk][3], v0, v1);
        mma_bf16(o[2 * np + 1], pa[kk][0], pa[kk][1], pa[kk][2], pa[kk][3], v2, v3);
      }
    }
    __syncthreads();  // the buffer is refilled next
  }
  if (abort_s) {
    // tiles tile and tile + 1 may have been issued and not consumed: let
    // their copies land (bounded, deaf to the give-up flag) before exit
    if (tid == 0)
      for (int u = tile; u < min(tile + 2, n_tiles); ++u)
        (void)mbar_wait(&full[u & 1], (uint32_t)(u >> 1) & 1u, kWaitLimit, &never_s);
    return;
  }
  // full row sums over the quad, then O / l
  l_a += __shfl_xor_sync(0xffffffffu, l_a, 1);
  l_a += __shfl_xor_sync(0xffffffffu, l_a, 2);
  l_b += __shfl_xor_sync(0xffffffffu, l_b, 1);
  l_b += __shfl_xor_sync(0xffffffffu, l_b, 2);
  const float ia = l_a > 0.f ? 1.0f / l_a : 0.f, ib = l_b > 0.f ? 1.0f / l_b : 0.f;
  if (i0 + ra < cnt) {
    bf16* op = O + (size_t)(r0 + ra) * hidden + (size_t)h * HD;
#pragma unroll
    for (int nd = 0; nd < ND; ++nd)
      *reinterpret_cast<uint32_t*>(op + nd * 8 + 2 * t) = pack_bf16(o[nd][0] * ia, o[nd][1] * ia);
  }
  if (i0 + rb < cnt) {
    bf16* op = O + (size_t)(r0 + rb) * hidden + (size_t)h * HD;
#pragma unroll
    for (int nd = 0; nd < ND; ++nd)
      *reinterpret_cast<uint32_t*>(op + nd * 8 + 2 * t) = pack_bf16(o[nd][2] * ib, o[nd][3] * ib);
  }
}

template <int HD>
void attn_mma_launch(Rows rows, int B, int S, int n_heads, const bf16* Q, const KvMaps& kvm, int z_seq, int z_layer,
                     int Tc, int P, int parallel, int n_action, float scale, bf16* O, int* err, uint32_t wait_limit,
                     cudaStream_t st) {
  const size_t smem = (size_t)4 * kAK * HD * sizeof(bf16) + 1024;  // K and V, two buffers, 1024-byte aligned
  static bool smem_set = false;  // raised once, before any graph capture of the kernel
  if (!smem_set) {
    cudaFuncSetAttribute(attn_mma_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    smem_set = true;
  }
  const dim3 grid((S + kAQ - 1) / kAQ, n_heads, B);
  launch_k(attn_mma_kernel<HD>, grid, dim3(kAW * 32), smem, st, rows, n_heads, Q, kvm, z_seq, z_layer, Tc, P,
           parallel, n_action, scale, O, err, wait_limit);
}

}  // namespace

template <typename T>
void launch_attention(Rows rows, int B, int S, int n_heads, int head_dim, const T* Q, const T* Kc, const T* Vc,
                      size_t kv_seq_stride, int Tc, int P, int parallel, int n_action, T* O, const KvMaps* kvm,
                      int z_seq, int z_layer, int* err, uint32_t wait_limit, cudaStream_t st) {
  const float scale = 1.0f / sqrtf((float)head_dim);
  if constexpr (sizeof(T) == 2) {
    if (head_dim == 128)
      attn_mma_launch<128>(rows, B, S, n_heads, Q, *kvm, z_seq, z_layer, Tc, P, parallel, n_action, scale, O, err,
                           wait_limit, st);
    else
      attn_mma_launch<64>(rows, B, S, n_heads, Q, *kvm, z_seq, z_layer, Tc, P, parallel, n_action, scale, O, err,
                          wait_limit, st);
    return;
  }
  dim3 grid((S + 15) / 16, n_heads, B);
  if (head_dim == 128)
    launch_k(attn_kernel<T, 128>, grid, dim3(256), 0, st, rows, n_heads, Q, Kc, Vc, kv_seq_stride, Tc, P, parallel,
             n_action, scale, O);
  else
    launch_k(attn_kernel<T, 64>, grid, dim3(256), 0, st, rows, n_heads, Q, Kc, Vc, kv_seq_stride, Tc, P, parallel,
             n_action, scale, O);
}

// ---- Stage 2 relevance (Sec. III-B, task-relevant filtering) ----------------
//
// For one layer: the softmax probability that each text row puts on each
// visual key (positions 1 .. Nv), summed over the text rows.  One block per
// (head, sequence).  Warp w takes the text rows w, w + 8, ... in row order:
// the lanes compute the row's scores over its keys (kept in shared memory),
// the warp reduces the maximum and the sum, and the lanes add the visual
// probabilities into the warp's own sums.  The warps' sums are then added in
// warp order.  The exact causal softmax of each row, sinks included, as in the
// prefix attention.
constexpr int kRelWarps = 8;

template <typename T, int HD>
__global__ void __launch_bounds__(kRelWarps * 32)
    relevance_kernel(Rows rows, int n_heads, const T* __restrict__ Q, const T* __restrict__ Kc,
                     size_t kv_seq_stride, int Tc, int Nv, int text_lo, int P, float scale,
                     float* __restrict__ part) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ __align__(16) float rsm[];
  const int h = blockIdx.x, b = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* qs = rsm + warp * HD;                                        // [kRelWarps][HD]
  float* sc = rsm + kRelWarps * HD + (size_t)warp * Tc;               // [kRelWarps][Tc]
  float* acc = rsm + (size_t)kRelWarps * (HD + Tc) + (size_t)warp * Nv;  // [kRelWarps][Nv]
  for (int v = lane; v < Nv; v += 32) acc[v] = 0.f;
  const int cnt = rows.off[b + 1] - rows.off[b];
  const int hidden = n_heads * HD;
  const T* Kh = Kc + (size_t)b * kv_seq_stride + (size_t)h * Tc * HD;
  for (int i = warp; i < cnt; i += kRelWarps) {
    const int pos = rows.idx[(size_t)b * rows.idx_stride + i];
    if (pos < text_lo || pos >= P) continue;  // not a text row after the image
    const int nk = min(pos + 1, Tc);
    const T* q = Q + (size_t)(rows.off[b] + i) * hidden + (size_t)h * HD;
    for (int e = lane; e < HD; e += 32) qs[e] = to_f(q[e]);
    __syncwarp();
    float mx = -INFINITY;
    for (int j = lane; j < nk; j += 32) {
      const T* kr = Kh + (size_t)j * HD;
      float dot = 0.f;
      if constexpr (sizeof(T) == 2) {
        const uint4* k4 = reinterpret_cast<const uint4*>(kr);
#pragma unroll 4
        for (int c8 = 0; c8 < HD / 8; ++c8) {
          const uint4 u = k4[c8];
          const uint32_t wv[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            dot = fmaf(__uint_as_float(wv[t] << 16), qs[c8 * 8 + 2 * t], dot);
            dot = fmaf(__uint_as_float(wv[t] & 0xFFFF0000u), qs[c8 * 8 + 2 * t + 1], dot);
          }
        }
      } else {
        const float4* k4 = reinterpret_cast<const float4*>(kr);
#pragma unroll 4
        for (int c4 = 0; c4 < HD / 4; ++c4) {
          const float4 u = k4[c4];
          dot = fmaf(u.x, qs[c4 * 4 + 0], dot);
          dot = fmaf(u.y, qs[c4 * 4 + 1], dot);
          dot = fmaf(u.z, qs[c4 * 4 + 2], dot);
          dot = fmaf(u.w, qs[c4 * 4 + 3], dot);
        }
      }
      const float sv = dot * scale;
      sc[j] = sv;
      mx = fmaxf(mx, sv);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float z = 0.f;
    for (int j = lane; j < nk; j += 32) {
      const float pj = expf(sc[j] - mx);
      sc[j] = pj;
      z += pj;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
    const float inv = 1.0f / z;
    __syncwarp();  // every lane's probabilities are in sc
    for (int v = lane; v < Nv && v + 1 < nk; v += 32) acc[v] += sc[v + 1] * inv;
    __syncwarp();  // before the next row overwrites qs and sc
  }
  __syncthreads();
  const float* acc0 = rsm + (size_t)kRelWarps * (HD + Tc);
  for (int v = threadIdx.x; v < Nv; v += blockDim.x) {
    float t = 0.f;
    for (int w = 0; w < kRelWarps; ++w) t += acc0[(size_t)w * Nv + v];
    part[((size_t)b * n_heads + h) * Nv + v] = t;
  }
}

// The heads' relevance added in head order; the step's relevance is kept for
// the next step's selection and returned.
__global__ void relevance_sum_kernel(const float* __restrict__ part, int n_heads, int Nv, float* __restrict__ rel,
                                     float* __restrict__ rel_out, uint8_t* __restrict__ rel_valid,
                                     const StepParams* __restrict__ prm, const uint8_t* __restrict__ active) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.x;
  if (prm->has_active && active && !active[b]) {  // sat the step out: its relevance stays
    for (int v = threadIdx.x; v < Nv; v += blockDim.x) rel_out[(size_t)b * Nv + v] = 0.f;
    return;
  }
  for (int v = threadIdx.x; v < Nv; v += blockDim.x) {
    float t = 0.f;
    for (int h = 0; h < n_heads; ++h) t += part[((size_t)b * n_heads + h) * Nv + v];
    rel[(size_t)b * Nv + v] = t;
    rel_out[(size_t)b * Nv + v] = t;
  }
  if (threadIdx.x == 0) rel_valid[b] = 1;
}

template <typename T, int HD>
void relevance_launch(Rows rows, int B, int n_heads, const T* Q, const T* Kc, size_t kv_seq_stride, int Tc, int Nv,
                      int text_lo, int P, size_t smem, float* part, cudaStream_t st) {
  static size_t smem_set = 48 * 1024;  // raised once per kernel, before any graph capture of it
  if (smem > smem_set) {
    cudaFuncSetAttribute(relevance_kernel<T, HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    smem_set = smem;
  }
  launch_k(relevance_kernel<T, HD>, dim3(n_heads, B), dim3(kRelWarps * 32), smem, st, rows, n_heads, Q, Kc,
           kv_seq_stride, Tc, Nv, text_lo, P, 1.0f / sqrtf((float)HD), part);
}

template <typename T>
int launch_relevance(Rows rows, int B, int n_heads, int head_dim, const T* Q, const T* Kc, size_t kv_seq_stride,
                     int Tc, int Nv, int text_lo, int P, float* part, float* rel, float* rel_out, uint8_t* rel_valid,
                     const StepParams* prm, const uint8_t* active, cudaStream_t st) {
  const size_t smem = (size_t)kRelWarps * (head_dim + Tc + Nv) * sizeof(float);
  if (smem > 200 * 1024) return 1;
  if (head_dim == 128)
    relevance_launch<T, 128>(rows, B, n_heads, Q, Kc, kv_seq_stride, Tc, Nv, text_lo, P, smem, part, st);
  else
    relevance_launch<T, 64>(rows, B, n_heads, Q, Kc, kv_seq_stride, Tc, Nv, text_lo, P, smem, part, st);
  launch_k(relevance_sum_kernel, dim3(B), dim3(256), 0, st, (const float*)part, n_heads, Nv, rel, rel_out, rel_valid,
           prm, active);
  return 0;
}

// ---- Stage 3 layer entropy (Sec. III-B, entropy-adaptive layer-wise reuse) --
//
// For one layer: per text row that sees two or more keys (positions
// text_lo .. P-1; BOS sees one) and head, the normalized entropy
// H / ln(keys) of the row's exact causal softmax, H = ln z - sum_j e^u_j u_j / z
// with u_j = s_j - max_j s_j and z = sum_j e^u_j.  One block per (head,
// sequence), warp w taking the text rows w, w + 8, ...; part[b][h][pos -
// text_lo].
template <typename T, int HD>
__global__ void __launch_bounds__(kRelWarps * 32)
    entropy_kernel(Rows rows, int n_heads, const T* __restrict__ Q, const T* __restrict__ Kc, size_t kv_seq_stride,
                   int Tc, int text_lo, int P, float scale, float* __restrict__ part) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ __align__(16) float esm[];
  const int h = blockIdx.x, b = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* qs = esm + warp * HD;                           // [kRelWarps][HD]
  float* sc = esm + kRelWarps * HD + (size_t)warp * Tc;  // [kRelWarps][Tc]
  const int cnt = rows.off[b + 1] - rows.off[b];
  const int hidden = n_heads * HD, nt = P - text_lo;
  const T* Kh = Kc + (size_t)b * kv_seq_stride + (size_t)h * Tc * HD;
  for (int i = warp; i < cnt; i += kRelWarps) {
    const int pos = rows.idx[(size_t)b * rows.idx_stride + i];
    if (pos < text_lo || pos >= P) continue;
    const int nk = min(pos + 1, Tc);
    const T* q = Q + (size_t)(rows.off[b] + i) * hidden + (size_t)h * HD;
    for (int e = lane; e < HD; e += 32) qs[e] = to_f(q[e]);
    __syncwarp();
    float mx = -INFINITY;
    for (int j = lane; j < nk; j += 32) {
      const T* kr = Kh + (size_t)j * HD;
      float dot = 0.f;
#pragma unroll 8
      for (int e = 0; e < HD; ++e) dot = fmaf(to_f(kr[e]), qs[e], dot);
      sc[j] = dot * scale;
      mx = fmaxf(mx, sc[j]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float z = 0.f, zu = 0.f;
    for (int j = lane; j < nk; j += 32) {
      const float u = sc[j] - mx, e = expf(u);
      z += e;
      zu = fmaf(e, u, zu);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      z += __shfl_xor_sync(0xffffffffu, z, o);
      zu += __shfl_xor_sync(0xffffffffu, zu, o);
    }
    if (lane == 0) part[((size_t)b * n_heads + h) * nt + (pos - text_lo)] = (logf(z) - zu / z) / logf((float)nk);
    __syncwarp();  // before the next row overwrites qs and sc
  }
}

// Per sequence and layer: the mean of the layer's normalized entropies over
// text rows (in position order) and heads, summed in fp64; kept in the cache
// for the next step's schedule and returned.  A sequence that sat the step
// out keeps its entropies.
__global__ void entropy_finish_kernel(const float* __restrict__ part, int L, int B, int n_heads, int nt,
                                      float* __restrict__ ent, uint8_t* __restrict__ ent_valid,
                                      float* __restrict__ ent_out, const StepParams* __restrict__ prm,
                                      const uint8_t* __restrict__ active) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.x;
  const bool sat_out = prm->has_active && active && !active[b];
  for (int l = threadIdx.x; l < L; l += blockDim.x) {
    if (sat_out) {
      ent_out[(size_t)b * L + l] = 0.f;
      continue;
    }
    const float* pl = part + ((size_t)l * B + b) * n_heads * nt;
    double sum = 0.0;
    for (int r = 0; r < nt; ++r)
      for (int h = 0; h < n_heads; ++h) sum += (double)pl[(size_t)h * nt + r];
    const float e = (float)(sum / (double)(nt * n_heads));
    ent[(size_t)b * L + l] = e;
    ent_out[(size_t)b * L + l] = e;
  }
  if (threadIdx.x == 0 && !sat_out) ent_valid[b] = 1;
}

template <typename T>
int launch_layer_entropy(Rows rows, int B, int n_heads, int head_dim, const T* Q, const T* Kc, size_t kv_seq_stride,
                         int Tc, int text_lo, int P, float* part, cudaStream_t st) {
  const size_t smem = (size_t)kRelWarps * (head_dim + Tc) * sizeof(float);
  if (smem > 200 * 1024 || P <= text_lo) return 1;
  static size_t smem_set[2] = {48 * 1024, 48 * 1024};  // raised once per kernel, before any graph capture of it
  const float scale = 1.0f / sqrtf((float)head_dim);
  if (head_dim == 128) {
    if (smem > smem_set[0]) {
      cudaFuncSetAttribute(entropy_kernel<T, 128>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      smem_set[0] = smem;
    }
    launch_k(entropy_kernel<T, 128>, dim3(n_heads, B), dim3(kRelWarps * 32), smem, st, rows, n_heads, Q, Kc,
             kv_seq_stride, Tc, text_lo, P, scale, part);
  } else {
    if (smem > smem_set[1]) {
      cudaFuncSetAttribute(entropy_kernel<T, 64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      smem_set[1] = smem;
    }
    launch_k(entropy_kernel<T, 64>, dim3(n_heads, B), dim3(kRelWarps * 32), smem, st, rows, n_heads, Q, Kc,
             kv_seq_stride, Tc, text_lo, P, scale, part);
  }
  return 0;
}
void launch_entropy_finish(const float* part, int L, int B, int n_heads, int nt, float* ent, uint8_t* ent_valid,
                           float* ent_out, const StepParams* prm, const uint8_t* active, cudaStream_t st) {
  launch_k(entropy_finish_kernel, dim3(B), dim3(64), 0, st, part, L, B, n_heads, nt, ent, ent_valid, ent_out, prm,
           active);
}
template int launch_layer_entropy<float>(Rows, int, int, int, const float*, const float*, size_t, int, int, int,
                                         float*, cudaStream_t);
template int launch_layer_entropy<bf16>(Rows, int, int, int, const bf16*, const bf16*, size_t, int, int, int, float*,
                                        cudaStream_t);

template int launch_relevance<float>(Rows, int, int, int, const float*, const float*, size_t, int, int, int, int,
                                     float*, float*, float*, uint8_t*, const StepParams*, const uint8_t*,
                                     cudaStream_t);
template int launch_relevance<bf16>(Rows, int, int, int, const bf16*, const bf16*, size_t, int, int, int, int,
                                    float*, float*, float*, uint8_t*, const StepParams*, const uint8_t*,
                                    cudaStream_t);

template void launch_attention<float>(Rows, int, int, int, int, const float*, const float*, const float*, size_t,
                                      int, int, int, int, float*, const KvMaps*, int, int, int*, uint32_t,
                                      cudaStream_t);
template void launch_attention<bf16>(Rows, int, int, int, int, const bf16*, const bf16*, const bf16*, size_t, int,
                                     int, int, int, bf16*, const KvMaps*, int, int, int*, uint32_t, cudaStream_t);

}  // namespace vlac
