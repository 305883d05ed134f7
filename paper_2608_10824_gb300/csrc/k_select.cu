// Stage 1 (static patch detection) and the gate + Stage-3 selection.
//
// Sec. III-B, Stage 1: cosine similarity between corresponding patches of
// I_t and I_{t-1}; a patch is static when the similarity is above tau.  The
// similarity vector is the raw uint8 RGB values of the patch, and the
// comparison against tau = num/den is decided exactly in integers.
// Sec. III-B, Stage 2 (optional): the top_k patches by the previous step's
// text-to-vision relevance are taken out of the static set; the rest is the
// reusable set.
// Algorithm 1: m_{t-1} < theta_m (strict) invalidates the cache and runs the
// full pass; otherwise Stage 3 reuses, at layer l, the floor(s_l * |R| / 1000)
// most similar reusable patches and recomputes the rest.
#include <mutex>

#include "internal.cuh"

namespace vlac {

typedef unsigned __int128 u128;

constexpr int kMaxSelectDevices = 64;

// cos > num/den, exact.  Both patches all-zero: cos = 1; exactly one: cos = 0.
__device__ __forceinline__ bool cos_above(uint32_t d, uint32_t na, uint32_t nb, uint32_t num, uint32_t den) {
  if (den == 0) return false;
  if (na == 0 && nb == 0) return num < den;
  if (na == 0 || nb == 0 || d == 0) return false;
  const u128 lhs = (u128)((uint64_t)d * d) * (u128)((uint64_t)den * den);
  const u128 rhs = (u128)((uint64_t)num * num) * (u128)((uint64_t)na * nb);
  return lhs > rhs;
}

// cos^2 as a fraction with a positive denominator.
__device__ __forceinline__ void cos2_frac(int3 s, uint64_t& n2, uint64_t& d2) {
  const uint32_t d = (uint32_t)s.x, na = (uint32_t)s.y, nb = (uint32_t)s.z;
  if (na == 0 && nb == 0) { n2 = 1; d2 = 1; return; }
  if (na == 0 || nb == 0) { n2 = 0; d2 = 1; return; }
  n2 = (uint64_t)d * d;
  d2 = (uint64_t)na * nb;
}

// Reuse order: patch u precedes patch v when its cosine is higher, ties by index.
__device__ __forceinline__ bool more_similar(int3 su, int u, int3 sv, int v) {
  uint64_t nu, du, nv, dv;
  cos2_frac(su, nu, du);
  cos2_frac(sv, nv, dv);
  const u128 l = (u128)nu * dv, r = (u128)nv * du;
  if (l != r) return l > r;
  return u < v;
}

// One warp per (sequence, patch): integer dot product and squared norms.
__global__ void patch_stats_kernel(const uint8_t* __restrict__ frames, const uint8_t* __restrict__ prev,
                                   const uint8_t* __restrict__ valid, const StepParams* __restrict__ prm,
                                   int n_views, int img_h, int img_w, int patch, int Nv, int3* __restrict__ stats,
                                   uint8_t* __restrict__ mask, uint8_t* __restrict__ user_mask) {
  pdl_wait();
  pdl_trigger();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int v = blockIdx.x * (blockDim.x >> 5) + warp;
  const int b = blockIdx.y;
  if (v >= Nv) return;
  const size_t fb = (size_t)n_views * img_h * img_w * 3;
  const uint8_t* fa = frames + (size_t)b * fb;
  const uint8_t* fp = prev + (size_t)b * fb;
  const int gw = img_w / patch, gh = img_h / patch;
  const int view = v / (gw * gh), r = v % (gw * gh), py = r / gw, px = r % gw;
  const int n = patch * patch * 3, row_bytes = patch * 3;
  uint32_t d = 0, na = 0, nb = 0;
  for (int e = lane; e < n; e += 32) {
    const int ry = e / row_bytes, rem = e - ry * row_bytes;
    const size_t o = ((size_t)(view * img_h + py * patch + ry) * img_w + (size_t)px * patch) * 3 + rem;
    const uint32_t a = fa[o], c = fp[o];
    d += a * c;
    na += a * a;
    nb += c * c;
  }
  d = __reduce_add_sync(0xffffffffu, d);
  na = __reduce_add_sync(0xffffffffu, na);
  nb = __reduce_add_sync(0xffffffffu, nb);
  if (lane == 0) {
    const bool st = valid[b] && cos_above(d, na, nb, prm->tau_num, prm->tau_den);
    stats[(size_t)b * Nv + v] = make_int3((int)d, (int)na, (int)nb);
    mask[(size_t)b * Nv + v] = st;
    if (user_mask) user_mask[(size_t)b * Nv + v] = st;
  }
}

// One block per sequence: gate decision, Stage-2 removal, reuse ranking and
// the ordered recompute list.  idx = [positions that are not reusable,
// ascending] ++ [reusable patches, least similar first], so the rows
// recomputed at layer l are idx[0 .. M[l]).
__global__ void select_kernel(const int3* __restrict__ stats, const uint8_t* __restrict__ mask,
                              const uint8_t* __restrict__ valid, const float* __restrict__ m_prev,
                              const StepParams* __restrict__ prm, const int8_t* __restrict__ override_,
                              int Nv, int S, int L, int P, int parallel, int n_action, uint8_t* __restrict__ full_out,
                              int* __restrict__ idx, int* __restrict__ M, int* __restrict__ emit_slot,
                              uint8_t* __restrict__ user_recomputed, uint8_t* __restrict__ user_gate_auto,
                              int* __restrict__ user_idx, int* __restrict__ user_M,
                              const uint8_t* __restrict__ active, const float* __restrict__ rel,
                              uint8_t* __restrict__ rel_valid, const uint8_t* __restrict__ s2_forced,
                              uint8_t* __restrict__ relevant, float* __restrict__ rel_out,
                              const uint16_t* __restrict__ sched) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ uint8_t smem[];
  int3* s_st = reinterpret_cast<int3*>(smem);
  int* s_rank = reinterpret_cast<int*>(s_st + Nv);
  uint8_t* s_stat = reinterpret_cast<uint8_t*>(s_rank + Nv);
  __shared__ int s_full;
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  if (prm->has_active && active && !active[b]) {
    // the sequence sits this step out: no rows at any layer
    if (tid == 0) {
      full_out[b] = 0;
      emit_slot[b] = 0;
      if (user_recomputed) user_recomputed[b] = 0;
      if (user_gate_auto) user_gate_auto[b] = 0;
    }
    for (int l = tid; l < L; l += blockDim.x) M[(size_t)b * L + l] = 0;
    return;
  }
  if (tid == 0) {
    const bool ok = valid[b] != 0;
    const bool gate = !ok || m_prev[b] < prm->tau_margin;
    bool full = gate;
    if (prm->has_override && override_ && override_[b] >= 0) full = override_[b] != 0;
    if (!ok) full = true;
    s_full = full;
    full_out[b] = full;
    if (user_recomputed) user_recomputed[b] = full;
    if (user_gate_auto) user_gate_auto[b] = gate;
  }
  for (int v = tid; v < Nv; v += blockDim.x) {
    s_st[v] = stats[(size_t)b * Nv + v];
    s_stat[v] = mask[(size_t)b * Nv + v];
  }
  // Stage 2: patch v is relevant when fewer than top_k patches rank before it
  // (higher relevance, or equal relevance and lower index)
  const int top_k = prm->s2_top_k;
  const bool s2 = top_k > 0 && rel && rel_valid[b];
  for (int v = tid; v < Nv; v += blockDim.x) {
    bool r = false;
    if (s2) {
      const float* rb = rel + (size_t)b * Nv;
      const float rv = rb[v];
      int before = 0;
      for (int u = 0; u < Nv; ++u) {
        const float ru = rb[u];
        before += (ru > rv || (ru == rv && u < v)) ? 1 : 0;
      }
      r = before < top_k;
    }
    // lock-step replay: the caller's set is applied, the own one reported
    const bool apply = (top_k > 0 && prm->has_s2_forced && s2_forced) ? s2_forced[(size_t)b * Nv + v] != 0 : r;
    if (apply) s_stat[v] = 0;
    if (relevant) relevant[(size_t)b * Nv + v] = r;
    if (top_k == 0 && rel_out) rel_out[(size_t)b * Nv + v] = 0.f;
  }
  if (top_k == 0 && rel_valid && tid == 0) rel_valid[b] = 0;  // nothing measured this step
  __syncthreads();
  const bool full = s_full != 0;
  int* idx_b = idx + (size_t)b * S;
  if (full) {
    for (int i = tid; i < S; i += blockDim.x) idx_b[i] = i;
    for (int l = tid; l < L; l += blockDim.x) M[(size_t)b * L + l] = S;
    if (tid == 0) emit_slot[b] = parallel ? P : P - 1;
  }
  __syncthreads();
  if (!full) {
    // |S| and the reuse rank of every static patch (0 = most similar)
    __shared__ int s_ns;
    if (tid == 0) s_ns = 0;
    __syncthreads();
    int local = 0;
    for (int v = tid; v < Nv; v += blockDim.x) local += s_stat[v];  // |R|
    if (local) atomicAdd(&s_ns, local);
    for (int v = tid; v < Nv; v += blockDim.x) {
      if (!s_stat[v]) continue;
      int rank = 0;
      const int3 sv = s_st[v];
      for (int u = 0; u < Nv; ++u)
        if (u != v && s_stat[u] && more_similar(s_st[u], u, sv, v)) ++rank;
      s_rank[v] = rank;
    }
    __syncthreads();
    const int nS = s_ns, n_always = S - nS;
    if (warp == 0) {
      int base = 0;
      for (int p0 = 0; p0 < S; p0 += 32) {
        const int p = p0 + lane;
        const bool always = p < S && !(p >= 1 && p <= Nv && s_stat[p - 1]);
        const unsigned bal = __ballot_sync(0xffffffffu, always);
        if (always) idx_b[base + __popc(bal & ((1u << lane) - 1u))] = p;
        base += __popc(bal);
      }
    }
    for (int v = tid; v < Nv; v += blockDim.x)
      if (s_stat[v]) idx_b[n_always + (nS - 1 - s_rank[v])] = 1 + v;
    for (int l = tid; l < L; l += blockDim.x)
      M[(size_t)b * L + l] =
          S - (int)(((uint32_t)(sched ? sched[(size_t)b * L + l] : prm->permille[l]) * (uint32_t)nS) / 1000u);
    if (tid == 0) emit_slot[b] = parallel ? n_always - n_action : n_always - 1;
  }
  __syncthreads();
  if (user_idx)
    for (int i = tid; i < S; i += blockDim.x) user_idx[(size_t)b * S + i] = idx_b[i];
  if (user_M)
    for (int l = tid; l < L; l += blockDim.x) user_M[(size_t)b * L + l] = M[(size_t)b * L + l];
}

// Stage 3's per-sequence schedule (Sec. III-B, entropy-adaptive layer-wise
// reuse, this library's reading): with the option on and the previous step's
// layer entropies e_l in the cache, t_l = hi - (hi - lo) * e_l per mille,
// smoothed over depth (r_0 = t_0, r_l = r_{l-1} + weight/1000 * (t_l - r_{l-1}),
// in fp64) and floored; otherwise the caller's schedule.  `own` receives the
// derived schedule, `use` the one the selection applies (a lock-step replay
// may impose another).
__global__ void schedule_kernel(const StepParams* __restrict__ prm, const float* __restrict__ ent,
                                uint8_t* __restrict__ ent_valid, const uint16_t* __restrict__ forced, int L,
                                const uint8_t* __restrict__ active, uint16_t* __restrict__ own,
                                uint16_t* __restrict__ use, float* __restrict__ ent_out) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.x;
  if (threadIdx.x != 0) return;
  if (prm->has_active && active && !active[b]) {  // sat the step out: its state stays, its outputs are zero
    for (int l = 0; l < L; ++l) {
      own[(size_t)b * L + l] = 0;
      use[(size_t)b * L + l] = prm->permille[l];
      ent_out[(size_t)b * L + l] = 0.f;
    }
    return;
  }
  const bool adaptive = prm->s3_adaptive && ent_valid[b];
  const double lo = prm->s3_lo, hi = prm->s3_hi, w = prm->s3_weight / 1000.0;
  double r = 0.0;
  for (int l = 0; l < L; ++l) {
    uint16_t v = prm->permille[l];
    if (adaptive) {
      const double t = hi - (hi - lo) * (double)ent[(size_t)b * L + l];
      r = l == 0 ? t : r + w * (t - r);
      v = (uint16_t)fmin(1000.0, fmax(0.0, floor(r)));
    }
    own[(size_t)b * L + l] = v;
    use[(size_t)b * L + l] = (prm->s3_adaptive && prm->has_s3_forced && forced) ? forced[(size_t)b * L + l] : v;
    if (!prm->s3_adaptive) ent_out[(size_t)b * L + l] = 0.f;  // nothing measured this step
  }
  if (!prm->s3_adaptive) ent_valid[b] = 0;
}

// Row offsets of every layer: off[l][b] = sum of M[b'][l] over b' < b.
__global__ void plan_kernel(const int* __restrict__ M, int B, int L, int* __restrict__ off) {
  pdl_wait();
  pdl_trigger();
  for (int l = threadIdx.x; l < L; l += blockDim.x) {
    int acc = 0;
    off[(size_t)l * (B + 1)] = 0;
    for (int b = 0; b < B; ++b) {
      acc += M[(size_t)b * L + l];
      off[(size_t)l * (B + 1) + b + 1] = acc;
    }
  }
}

cudaError_t launch_patch_stats(const uint8_t* frames, const uint8_t* prev, const uint8_t* valid,
                               const StepParams* prm, int B, int n_views, int img_h, int img_w, int patch,
                               int3* stats, uint8_t* mask, uint8_t* user_mask, cudaStream_t st) {
  const int Nv = n_views * (img_h / patch) * (img_w / patch);
  dim3 grid((Nv + 7) / 8, B);
  return launch_k(patch_stats_kernel, grid, dim3(256), 0, st, frames, prev, valid, prm, n_views, img_h, img_w, patch, Nv,
           stats, mask, user_mask);
}

// Shared memory of select_kernel for Nv patches: the int3 statistics, the
// reuse ranks and the static flags.  Above 48 KB (Nv > 2890) the kernel needs
// the opt-in limit, raised once per device for the largest Nv the dims
// accept (4096 patches).
static size_t select_smem(int Nv) { return (size_t)Nv * (sizeof(int3) + sizeof(int) + 1) + 16; }
static cudaError_t select_smem_attr(size_t smem) {
  if (smem <= 48u * 1024u) return cudaSuccess;
  static std::mutex mu;
  static bool done[kMaxSelectDevices] = {};
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxSelectDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (!done[dev]) {
    e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)select_smem(4096));
    if (e != cudaSuccess) return e;
    done[dev] = true;
  }
  return cudaSuccess;
}

void launch_schedule(const StepParams* prm, const float* ent, uint8_t* ent_valid, const uint16_t* forced,
                     const uint8_t* active, int B, int L, uint16_t* own, uint16_t* use, float* ent_out,
                     cudaStream_t st) {
  launch_k(schedule_kernel, dim3(B), dim3(32), 0, st, prm, ent, ent_valid, forced, L, active, own, use, ent_out);
}

cudaError_t launch_select(const int3* stats, const uint8_t* mask, const uint8_t* valid, const float* m_prev,
                          const StepParams* prm, const int8_t* override_, int B, int Nv, int S, int L, int P,
                          int parallel, int n_action, uint8_t* full, int* idx, int* M, int* off, int* emit_slot,
                          uint8_t* user_recomputed, uint8_t* user_gate_auto, int* user_idx, int* user_M,
                          const uint8_t* active, const float* rel, uint8_t* rel_valid, const uint8_t* s2_forced,
                          uint8_t* relevant, float* rel_out, const uint16_t* sched, cudaStream_t st) {
  const size_t smem = select_smem(Nv);
  cudaError_t e = select_smem_attr(smem);
  if (e != cudaSuccess) return e;
  e = launch_k(select_kernel, dim3(B), dim3(512), smem, st, stats, mask, valid, m_prev, prm, override_, Nv, S, L, P,
           parallel, n_action, full, idx, M, emit_slot, user_recomputed, user_gate_auto, user_idx, user_M, active, rel,
           rel_valid, s2_forced, relevant, rel_out, sched);
  if (e != cudaSuccess) return e;
  return launch_k(plan_kernel, dim3(1), dim3(256), 0, st, M, B, L, off);
}

}  // namespace vlac
