// Allocation-free variant of the selection stage (Stage-1 patch similarity,
// the gate and the Stage-3 recompute order) for callers that may not allocate
// device memory at run time: real-time control loops whose memory is fixed
// up front, and host frameworks that own every device allocation themselves.
//
// The kernels are the ones vlac_step runs; only their scratch (the per-patch
// integer statistics, the step scalars, the per-layer row offsets) lives in a
// file-scope device array instead of a context workspace.
#include <cstring>
#include <mutex>

#include "internal.cuh"

namespace {

// Scratch shared by every call on a device; it keeps whatever the last call
// left in it.  256 KiB: the int3 statistics of up to 20,000 (sequence, patch)
// pairs plus the step scalars and per-layer row offsets.
constexpr size_t kNoallocScratchBytes = 256u << 10;
static __device__ __align__(256) unsigned char g_select_scratch[kNoallocScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
unsigned char* g_scratch_dev[kMaxDevices] = {};

size_t round256(size_t v) { return (v + 255) / 256 * 256; }

// Device address of the scratch array for the current device.  The symbol's
// name in host code is only a stand-in, so the address is looked up once per
// device with that device current.
int scratch_for_current_device(unsigned char** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    (void)cudaGetLastError();
    return VLAC_ERR_CUDA;
  }
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_dev[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_select_scratch) != cudaSuccess || !p) {
      (void)cudaGetLastError();
      return VLAC_ERR_CUDA;
    }
    g_scratch_dev[dev] = static_cast<unsigned char*>(p);
  }
  *out = g_scratch_dev[dev];
  return VLAC_OK;
}

}  // namespace

extern "C" int vlac_select_noalloc(const vlac_dims* d, int batch, const uint8_t* frames, const uint8_t* prev_frames,
                                   const uint8_t* valid, const float* m_prev, vlac_rational tau_sim,
                                   float tau_margin, const uint16_t* reuse_permille, const int8_t* gate_override,
                                   uint8_t* static_mask, int32_t* idx, int32_t* M, uint8_t* recomputed,
                                   void* stream) {
  using namespace vlac;
  if (!d || vlac::check_dims(d) != VLAC_OK || batch < 1 || batch > d->max_batch || !frames || !prev_frames ||
      !valid || !m_prev || !reuse_permille || !static_mask || !idx || !M || !recomputed || tau_sim.den == 0 ||
      tau_margin != tau_margin)
    return VLAC_ERR_INVALID_ARG;
  const int Nv = d->n_views * (d->img_h / d->patch) * (d->img_w / d->patch);
  const int has_p = d->proprio_dim > 0 ? 1 : 0;
  const int P = d->n_text + Nv + has_p;
  const int S = P + (d->parallel ? d->n_action : 0);
  const int L = d->n_layers;
  // scratch layout: step scalars | int3 stats [B][Nv] | full [B] | offsets [L][B+1] | emit slot [B]
  const size_t o_prm = 0;
  const size_t o_stats = round256(o_prm + sizeof(StepParams));
  const size_t o_full = round256(o_stats + sizeof(int3) * (size_t)batch * Nv);
  const size_t o_off = round256(o_full + (size_t)batch);
  const size_t o_emit = round256(o_off + sizeof(int) * (size_t)L * (batch + 1));
  const size_t need = round256(o_emit + sizeof(int) * (size_t)batch);
  if (need > kNoallocScratchBytes) return VLAC_ERR_UNSUPPORTED;  // valid dims, beyond the fixed scratch
  StepParams p;
  memset(&p, 0, sizeof(p));
  for (int l = 0; l < L; ++l) {
    if (reuse_permille[l] > 1000) return VLAC_ERR_INVALID_ARG;
    p.permille[l] = reuse_permille[l];
  }
  p.tau_num = tau_sim.num;
  p.tau_den = tau_sim.den;
  p.tau_margin = tau_margin;
  p.has_override = gate_override ? 1 : 0;
  unsigned char* base = nullptr;
  int rc = scratch_for_current_device(&base);
  if (rc) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  StepParams* prm = reinterpret_cast<StepParams*>(base + o_prm);
  int3* stats = reinterpret_cast<int3*>(base + o_stats);
  uint8_t* full = base + o_full;
  int* off = reinterpret_cast<int*>(base + o_off);
  int* emit = reinterpret_cast<int*>(base + o_emit);
  // every scratch entry a kernel reads is written earlier in this call, so
  // nothing has to be cleared first
  // each launch's own status: an error left over from the caller's earlier
  // work is neither reported as this call's nor cleared
  CopyList none{};
  if (launch_stage(p, prm, none, st) != cudaSuccess) return VLAC_ERR_CUDA;
  if (launch_patch_stats(frames, prev_frames, valid, prm, batch, d->n_views, d->img_h, d->img_w, d->patch, stats,
                         static_mask, nullptr, st) != cudaSuccess)
    return VLAC_ERR_CUDA;
  if (launch_select(stats, static_mask, valid, m_prev, prm, gate_override, batch, Nv, S, L, P, d->parallel,
                    d->n_action, full, idx, M, off, emit, recomputed, nullptr, nullptr, nullptr, nullptr, nullptr,
                    nullptr, nullptr, nullptr, nullptr, nullptr, st) != cudaSuccess)
    return VLAC_ERR_CUDA;
  return VLAC_OK;
}
