// Internal declarations shared by the CUDA translation units of libvlac.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/vlac.h"

namespace vlac {

typedef __nv_bfloat16 bf16;

constexpr int kMaxLayers = 256;

// Per-step scalars, written to device memory before the step's kernels run.
struct StepParams {
  uint32_t tau_num, tau_den;
  float tau_margin;
  int32_t margin_kind;
  int32_t reduction;  // resolved: 0 mean, 1 min
  int32_t has_override;
  int32_t has_forced;
  int32_t has_active;
  int32_t s2_top_k;  // Stage 2: 0 = off
  int32_t s2_layer;
  int32_t has_s2_forced;
  int32_t s3_adaptive;  // Stage 3 from the previous step's layer entropies: 0 = the permille below
  int32_t s3_lo, s3_hi, s3_weight;
  int32_t has_s3_forced;
  uint16_t permille[kMaxLayers];
};

// Where the K-split partial sums of a prefix GEMM live (out[s][m][n] of
// launch_gemm_tc).  Columns below full_cols come from CTAs that ran the whole
// K range: one partial, at part.  The other columns have `tail` partials: the
// first at part, split s >= 1 either at part + s * stride (the uniform
// layout, tail_ld == 0) or compactly at
// tail_p + (s - 1) * tail_stride + row * tail_ld + (col - full_cols).
struct SplitPlan {
  int full_cols;
  int tail;
  size_t stride;
  float* tail_p;
  size_t tail_stride;
  int tail_ld;
};
inline SplitPlan uniform_splits(int splits, size_t stride) { return SplitPlan{0, splits, stride, nullptr, 0, 0}; }

// A set of rows processed by one layer: per sequence b, rows i < count_b with
// count_b = off[b+1] - off[b]; the compacted row index is off[b] + i, the
// token position is idx[b * idx_stride + i], and the fp32 residual row lives at
// X + (b * idx_stride + i) * hidden.
struct Rows {
  const int* off;
  const int* idx;
  int idx_stride;
  float* X;
};

// Arguments of the fused decode GEMV (one new row per sequence).  Output row
// pairs: QKV -> (i, i + head_dim/2) of one head of q, k or v; SwiGLU ->
// (gate j, up j); residual -> (2p, 2p + 1).
enum { kEpiQkvRope = 0, kEpiResid = 1, kEpiSwiglu = 2 };
struct DGemv {
  const void* W;  // [rows][K] weights (T)
  int n_pairs;
  int K;
  const float* X;     // RMSNorm prologue: fp32 residual rows [nb][K]
  const void* gain;   // RMSNorm gains (T)
  float eps;
  const void* xin;    // plain input rows [nb][K] (T) when there is no prologue
  float* Xres;        // residual epilogue: Xres[b][n] += y
  int n_out;          // row stride of Xres
  void* Q;            // QKV epilogue
  void* Kc;
  void* Vc;
  size_t kv_seq_stride;
  int Tc, pos, n_heads, head_dim;
  const float* rope_cos;
  const float* rope_sin;
  void* G;            // SwiGLU epilogue: G[b][j]
  int ffn;
  const float* ssq_in;  // normalising GEMV: per-producer-CTA sums of squares [nb][n_ssq]
  int n_ssq;
  float* ssq_out;       // residual GEMV: this launch's per-CTA sums of squares [nb][grid]
  int* err;             // device error word (bounded waits)
  uint32_t wait_limit;  // polls of a ring wait before it gives up (drains keep kWaitLimit)
  int ns;               // stages of the weight ring
  // optional (pf_W null: off): the next decode GEMV of the stream; this CTA
  // pulls the start of that kernel's CTA region into L2 once its own loads
  // are issued
  const void* pf_W;
  int pf_K, pf_pairs, pf_grid;
  uint32_t pf_bytes;
};
constexpr int kDecodeRowsPerCta = 4;  // residual rows per decode-GEMV CTA (2 row pairs)

// Tiled decode weights (built at create, streamed by the decode GEMV and the
// persistent decode pass): groups of kDecGroupPairs output row pairs, K cut
// into chunks of kDecTileBytes per row, bf16 tiles interleaved in 8-element K
// steps ([k/8][row][k%8]).
constexpr int kDecGroupPairs = 4;
constexpr int kDecTileBytes = 4096;

// Groups [g0, g1) of CTA b when G groups are cut over n CTAs: the first
// G mod n CTAs take one group more.  CTAs are placed on SMs in index order as
// the previous kernel's CTAs leave, so the low indices start first and fill
// their weight ring earliest; they are the ones given the extra group.
__host__ __device__ inline void dgemv_group_range(int G, int n, int b, int& g0, int& g1) {
  const int q = G / n, r = G - q * n;
  g0 = b * q + (b < r ? b : r);
  g1 = g0 + q + (b < r ? 1 : 0);
}

// Position (in elements, within its row) of element k of a bf16 input vector
// in the A-fragment order of mma.m16n8k16: per 32-element K step and lane t
// the elements 2t, 2t+1, 2t+8, 2t+9, 2t+16, 2t+17, 2t+24, 2t+25.
__device__ __forceinline__ int afrag_pos(int k) {
  const int i = k >> 5, w = k & 31, s = w >> 3, t = (w & 7) >> 1;
  return ((i * 4 + t) * 8) + s * 2 + (w & 1);
}

// ---- scalar helpers --------------------------------------------------------
template <typename T> __device__ __forceinline__ float to_f(T v);
template <> __device__ __forceinline__ float to_f<float>(float v) { return v; }
template <> __device__ __forceinline__ float to_f<bf16>(bf16 v) { return __bfloat162float(v); }
template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }

// Programmatic dependent launch.  Every kernel of the step calls pdl_wait()
// before it touches data written by an earlier kernel of the stream (a no-op
// when the launch did not allow early start), and pdl_trigger() once its
// dependents may be scheduled.  Work that reads only constant data (weight
// prefetches) may run before pdl_wait().
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
// Starts pulling [p, p + bytes) into L2 (bytes: multiple of 16, p 16-byte aligned).
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// ---- mbarrier and bulk-copy helpers ------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// Bounded wait for the phase with `parity`; false after `limit` polls or once
// another role raised *abort.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, uint32_t limit, volatile int* abort) {
  for (uint32_t i = 0; i < limit; ++i) {
    if (mbar_test(bar, parity)) return true;
    if (*abort) return false;
  }
  return false;
}
// 1-D bulk copy global -> shared completing on `bar` (16-byte aligned, bytes % 16 == 0).
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(src), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}
constexpr uint32_t kWaitLimit = 1u << 24;

// Give-up path of a bulk-copy ring: before its CTA exits, wait (bounded, deaf
// to any give-up flag) until the producer's last min(issued, ns) copies have
// landed.  A stage is refilled only after every consumer waited for its
// previous copy, so these are the only copies that can still be in flight;
// (stage, phase) is the producer's ring position after its last issue.
__device__ __forceinline__ void ring_drain(uint64_t* full, int ns, int stage, uint32_t phase, uint32_t issued) {
  const int n_last = (int)min(issued, (uint32_t)ns);
  for (int q = 0; q < n_last; ++q) {
    int s = stage - 1 - q;
    uint32_t ph = phase;
    if (s < 0) {
      s += ns;
      ph ^= 1u;
    }
    for (uint32_t it = 0; it < kWaitLimit && !mbar_test(&full[s], ph); ++it) {
    }
  }
}

__device__ __forceinline__ void set_error(int* err, int code) {
  if (err) atomicCAS(err, 0, code);
}

// ldmatrix: four 8x8 b16 matrices; lane l gives the row address of row l%8 of matrix l/8
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
// D += A * B on the legacy tensor path, m16n8k16, bf16 operands, fp32 accumulators
__device__ __forceinline__ void mma_bf16(float* d, uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Block-wide sum in a fixed order (warp butterflies, then warp 0 over the
// per-warp partials).  `red` holds >= 32 floats.  All threads get the result.
__device__ __forceinline__ float block_sum(float v, float* red) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) red[w] = v;
  __syncthreads();
  float t = (threadIdx.x < (unsigned)nw) ? red[threadIdx.x] : 0.f;
  if (w == 0) {
    t = warp_sum(t);
    if (lane == 0) red[0] = t;
  }
  __syncthreads();
  float r = red[0];
  __syncthreads();
  return r;
}

// Launch with optional programmatic stream serialization (the kernel may
// start while its predecessor drains; it must call pdl_wait()).  Returns the
// launch's own status.
extern bool g_pdl;
template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = g_pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

}  // namespace vlac

// ---- launchers (defined in the kernel translation units) -------------------
namespace vlac {

int check_dims(const vlac_dims* d);  // VLAC_OK or the error vlac_create would return

cudaError_t launch_patch_stats(const uint8_t* frames, const uint8_t* prev, const uint8_t* valid,
                        const StepParams* prm, int B, int n_views, int img_h, int img_w, int patch,
                        int3* stats, uint8_t* mask, uint8_t* user_mask, cudaStream_t st);
// Stage 2 state (all NULL = Stage 2 unavailable): rel [B][Nv] the previous
// step's relevance and rel_valid [B] whether it holds one (cleared here on a
// step with Stage 2 off); s2_forced [B][Nv] (with prm->has_s2_forced) is
// applied instead of the kernel's own removal set; relevant [B][Nv] receives
// the own set and rel_out [B][Nv] is zeroed on a step with Stage 2 off.
cudaError_t launch_select(const int3* stats, const uint8_t* mask, const uint8_t* valid, const float* m_prev,
                   const StepParams* prm, const int8_t* override_, int B, int Nv, int S, int L, int P,
                   int parallel, int n_action, uint8_t* full, int* idx, int* M, int* off, int* emit_slot,
                   uint8_t* user_recomputed, uint8_t* user_gate_auto, int* user_idx, int* user_M,
                   const uint8_t* active, const float* rel, uint8_t* rel_valid, const uint8_t* s2_forced,
                   uint8_t* relevant, float* rel_out, const uint16_t* sched, cudaStream_t st);
// Stage 3's schedule per sequence ([B][L]): own = derived (or the caller's),
// use = what the selection applies (sched of launch_select).  With Stage 3
// adaptive off it clears ent_valid and zeroes ent_out; a sequence that sits
// the step out keeps its state and gets zero outputs.
void launch_schedule(const StepParams* prm, const float* ent, uint8_t* ent_valid, const uint16_t* forced,
                     const uint8_t* active, int B, int L, uint16_t* own, uint16_t* use, float* ent_out,
                     cudaStream_t st);

template <typename T>
void launch_im2col(Rows rows, int B, int S, const uint8_t* frames, int n_views, int img_h, int img_w,
                   int patch, int kpad, T* col, cudaStream_t st);
template <typename T>
void launch_embed(Rows rows, int B, int S, int hidden, int Nv, int P, int has_proprio, int proprio_dim,
                  int n_text, int vocab, const int32_t* prompt, const float* proprio, const T* tok_emb,
                  const float* patch_part, const T* proprio_w, const T* action_emb, int* err,
                  cudaStream_t st);
template <typename T>
void launch_layer_in(Rows rows, const int* off_prev, int B, int S, int hidden, float* H, size_t h_seq_stride,
                     const T* gain, float eps, T* A, cudaStream_t st);
template <typename T>
void launch_qkv_epilogue(Rows rows, int B, int S, int n_heads, int head_dim, const float* part, const SplitPlan& sp,
                         const float* rope_cos, const float* rope_sin, T* Q, T* Kc, T* Vc, size_t kv_seq_stride,
                         int Tc, cudaStream_t st);
template <typename T>
void launch_residual_norm(Rows rows, int B, int S, int hidden, const float* part, const SplitPlan& sp, const T* gain,
                          float eps, T* A, cudaStream_t st);
template <typename T>
void launch_swiglu(Rows rows, int B, int S, int ffn, const float* part, const SplitPlan& sp, T* G, cudaStream_t st);
void launch_residual(Rows rows, int B, int S, int hidden, const float* part, const SplitPlan& sp, cudaStream_t st);
// residual_kernel of layer l and layer_in_kernel of layer l+1 in one launch
// (rows: layer l+1's; off_prev: layer l's offsets; H: layer l+1's H slice)
template <typename T>
void launch_residual_layer_in(Rows rows, const int* off_prev, int B, int S, int hidden, const float* part,
                              const SplitPlan& sp, float* H, size_t h_seq_stride, const T* gain, float eps, T* A,
                              cudaStream_t st);
// TMA maps of a cache's K and V (bf16 caches): 3-D {head_dim, Tc, batch x
// layers x heads}, boxes of 64 dimensions x 64 positions, 128-byte swizzle,
// positions past Tc read as zeros.  The box of (sequence b, layer l, head h)
// is at z = b * layers * heads + l * heads + h.
struct KvMaps {
  CUtensorMap k, v;
};
// Mixed-cache attention of one layer.  bf16: the K/V tiles come through kvm
// (z_seq = layers x heads, z_layer = l x heads); fp32: from Kc / Vc (this
// layer's slice, kv_seq_stride elements per sequence).
template <typename T>
void launch_attention(Rows rows, int B, int S, int n_heads, int head_dim, const T* Q, const T* Kc, const T* Vc,
                      size_t kv_seq_stride, int Tc, int P, int parallel, int n_action, T* O, const KvMaps* kvm,
                      int z_seq, int z_layer, int* err, uint32_t wait_limit, cudaStream_t st);
// Stage 2 relevance of one layer (rows as for launch_attention; text rows are
// positions text_lo .. P-1): part [B][n_heads][Nv] per head, then rel and
// rel_out [B][Nv] summed over the heads in order, and rel_valid[b] = 1.
// Returns nonzero if the shared-memory need exceeds a block's.
template <typename T>
int launch_relevance(Rows rows, int B, int n_heads, int head_dim, const T* Q, const T* Kc, size_t kv_seq_stride,
                     int Tc, int Nv, int text_lo, int P, float* part, float* rel, float* rel_out, uint8_t* rel_valid,
                     const StepParams* prm, const uint8_t* active, cudaStream_t st);
// Stage 3: one layer's normalized attention entropy per (sequence, head, text
// row) into part [B][n_heads][P - text_lo] (returns 1 if it cannot run);
// then, after the prefix pass, the per-layer means from part [L][B][...]
// into the cache (ent [B][L], ent_valid [B]) and ent_out.
template <typename T>
int launch_layer_entropy(Rows rows, int B, int n_heads, int head_dim, const T* Q, const T* Kc, size_t kv_seq_stride,
                         int Tc, int text_lo, int P, float* part, cudaStream_t st);
void launch_entropy_finish(const float* part, int L, int B, int n_heads, int nt, float* ent, uint8_t* ent_valid,
                           float* ent_out, const StepParams* prm, const uint8_t* active, cudaStream_t st);
template <typename T>
void launch_decode_embed(int B, int d, int D, int P, int hidden, int vocab, int n_bins, const T* tok_emb,
                         const int32_t* ids, const int32_t* forced, const StepParams* prm, float* Xd,
                         int* idx_dec, float* ssq_out, int* err, cudaStream_t st);
// m_t from the per-token signals (margins, gaps or vocabulary margins vms by
// prm->margin_kind); also the action delta against prev_ids (kept in the
// cache, with ids_valid) into delta.  A sequence that sat the step out
// (prm->has_active, active[b] == 0) keeps its gate state and previous ids.
void launch_finish(int B, int D, const StepParams* prm, const float* margins, const float* gaps, const float* vms,
                   float* m_prev, uint8_t* valid, float* user_step_margin, const int32_t* ids, int32_t* prev_ids,
                   uint8_t* ids_valid, int32_t* delta, const uint8_t* active, cudaStream_t st);
// End of a step: the previous frame of every sequence that stepped becomes
// this step's frame, and the outputs of the sequences that sat the step out
// are zeroed (with prm->has_active; active NULL = all stepped).
struct StepOutputs {
  int32_t* ids;
  float *margins, *gaps, *logits, *step_margin;
  uint8_t *recomputed, *gate_auto, *mask;
  int32_t *idx, *M;
  float* relevance;   // Stage 2 outputs [B][Nv]
  uint8_t* relevant;
  float *entropy, *vocab_margin;  // [B][D]
  int32_t* action_delta;          // [B]
};
void launch_commit(int B, int D, int n_bins, int Nv, int S, int L, size_t frame_bytes, const uint8_t* frames,
                   uint8_t* prev, const StepParams* prm, const uint8_t* active, const StepOutputs& o,
                   cudaStream_t st);

// Copies of the caller's per-step inputs into the context's staging buffers
// (and the step scalars into device memory), and of the step's outputs back
// to the caller's buffers.  A NULL source (or destination) is skipped.
struct CopySpan {
  const void* src;
  void* dst;
  size_t bytes;
};
constexpr int kMaxSpans = 24;
struct CopyList {
  CopySpan span[kMaxSpans];
  int n;
};
cudaError_t launch_stage(const StepParams& p, StepParams* prm, const CopyList& list, cudaStream_t st);
// One-layer entry: idx[i] = pos[i] for i < M (an index outside [0, S) latches
// VLAC_ERR_DEVICE_CHECK and is replaced by 0, so no access leaves the cache),
// off = {0, M}.
void launch_layer_setup(const int32_t* pos, int M, int S, int* idx, int* off, int* err, cudaStream_t st);
// K or V of one layer of one sequence between the cache layout
// [head][position][head_dim] (cache) and [position][head * head_dim] (flat),
// elements of esz bytes; to_cache selects the direction.
void launch_kv_copy(void* cache, void* flat, int n_heads, int Tc, int head_dim, int esz, bool to_cache,
                    cudaStream_t st);
void launch_copies(const CopyList& list, cudaStream_t st);

// Tensor maps of one activation buffer with boxes of 32, 64, 128 and 256 rows.
struct ActMaps {
  CUtensorMap m[4];
};
// GEMMs: out[s][m][n] = sum over split s of A[m][k] * W[n][k]; rows m < *m_ptr.
// Split plan sp: CTAs for the first sp.full_cols / 128 weight tiles run the
// whole K range; every other tile is cut into sp.tail K ranges (see SplitPlan
// for where each partial goes).
void launch_gemm_tc(const ActMaps* tmA, const CUtensorMap* tmW, const int* m_ptr, int m_cap, int N, int K,
                    const SplitPlan& sp, float* out, int* err, uint32_t wait_limit, cudaStream_t st);
template <typename T>
void launch_gemm_simt(const T* A, const T* W, const int* m_ptr, int m_cap, int N, int K, float* out,
                      cudaStream_t st);
int launch_wait_selftest(int* err, uint32_t spin_limit, cudaStream_t st);
template <typename T>
void launch_dgemv(const DGemv& a, int epi, int nb, int n_sm, cudaStream_t st);
int dgemv_grid(int n_pairs, int n_sm);  // CTAs (and sum-of-squares partials) of one decode GEMV

// Persistent decode pass (k_dpass.cu): all layers of one decode token in one
// cooperative launch, one CTA per SM.  Per-layer arrays are device arrays of L
// pointers (tiled decode weights, RMSNorm gains); K/V of layer l at
// Kc/Vc + l * kv_layer.  `ssq0` holds the decode embedding's sums of squares
// ([nb][n_ssq0]); `ssq` ([nb][grid]) and `bar` (zeroed by the launcher) are
// the launch's own workspace.
struct DPass {
  const bf16* const* w_qkv;
  const bf16* const* w_o;
  const bf16* const* w_gu;
  const bf16* const* w_d;
  const bf16* const* g_attn;
  const bf16* const* g_ffn;
  int L, hidden, ffn, n_heads, Tc, pos, ns, n_ssq0;
  float eps, scale;
  const float* rope_cos;
  const float* rope_sin;
  float* X;
  bf16* Q;
  bf16* AO;
  bf16* G;
  bf16* Kc;
  bf16* Vc;
  size_t kv_layer, kv_seq_stride;
  const float* ssq0;
  float* ssq;
  unsigned* bar;
  int* err;
  // attention: each (sequence, head) cut into attn_chunks key ranges; with
  // more than one, every range's partial (max, sum, unnormalised output) goes
  // to attn_part + (b * n_heads + h) * part_stride + chunk * (head_dim + 2) and
  // the last range to finish (counted in attn_cnt, zero between uses) combines
  int attn_chunks;
  size_t part_stride;
  float* attn_part;
  unsigned* attn_cnt;
  // grid barrier: 0 fence + atomic add + poll; 1 release add + acquire poll
  int bar_mode;
  // attention: up to kv_keys keys of the CTA's first item staged in shared
  // memory a layer ahead (0: read from global)
  int kv_keys;
  uint32_t wait_limit;  // polls of a ring, staging or grid-barrier wait before it gives up (drains keep kWaitLimit)
};
size_t dpass_kv_bytes(int kv_keys);
size_t dpass_smem_bytes(int hidden, int ffn, int nb, int ns, int kv_keys);
int dpass_kv_fit(int hidden, int ffn, int nb, int ns);  // K/V rows the staging buffer can hold on this device
bool dpass_supported(int hidden, int ffn, int n_heads, int head_dim, int nb, int ns);
int launch_dpass(const DPass& a, int nb, int n_sm, cudaStream_t st);
// Decode-streaming copy of a projection (W: [rows][K]); see k_decode.cu for the layout.
template <typename T>
void launch_tile_decode_weights(const T* W, int K, int n_pairs, int epi, int n_heads, int head_dim, int ffn, T* out,
                                cudaStream_t st);
size_t tiled_decode_elems(int K, int n_pairs);
size_t dgemv_stage_bytes();  // bytes of one weight-ring stage of the decode GEMV
template <typename T>
void launch_dec_attention(int B, int n_heads, int head_dim, const T* Q, const T* Kc, const T* Vc, size_t kv_seq_stride,
                          int Tc, int pos, float* part, unsigned* counters, T* O, cudaStream_t st);
// Margin over the whole vocabulary: W the LM-head rows outside the bins
// ([n_rows][hidden], T), xh scratch for the normed action rows ([rows][hidden],
// T), vl scratch for their logits ([rows][n_rows] fp32), vm the margins [B][D].
struct VocabHead {
  const void* W;
  int n_rows;
  void* xh;
  float* vl;
  float* vm;
};
// Action head of rows_per_seq rows per sequence: bin logits, ids, margins,
// gaps, entropy (may be NULL) and, with vh, the whole-vocabulary margin.
template <typename T>
void launch_head2(const float* X, const int* row_of_seq, size_t x_seq_stride, int rows_per_seq, int B, int hidden,
                  int n_bins, const T* final_norm, const T* head_w, float eps, float* logits_ws, int D, int tok0,
                  int32_t* ids, float* margins, float* gaps, float* logits, float* entropy, const VocabHead* vh,
                  cudaStream_t st);

}  // namespace vlac
