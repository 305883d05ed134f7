// Projections of the prefix pass: out[s][m][n] = sum_k A[m][k] * W[n][k] over
// the k range of split s.  Two kernels:
//   - gemm_tc:   bf16 (M = recomputed rows, device-resident), tcgen05 MMA
//                with fp32 accumulators in TMEM, operands staged by TMA into
//                128B-swizzled shared memory.  The weight tile is the 128-row
//                MMA operand and the token rows are the N side ("swap-AB"), so
//                one weight tile feeds every recomputed row.
//   - gemm_simt: the fp32 tiny model.
// The decode passes (M = batch <= 8) use the fused weight-streaming GEMV in
// k_decode.cu.
#include <cstdlib>

#include "internal.cuh"

namespace vlac {

// =============================================================================
// tcgen05 GEMM
// =============================================================================
namespace tc {

constexpr int kBM = 128;        // weight rows per CTA (MMA M)
constexpr int kBK = 64;         // K elements per stage = one 128-byte swizzle row
constexpr int kBoxRows = 32;    // granularity of the activation operand's token rows (boxes of 32..256 rows)
constexpr int kMaxTok = 256;    // token columns per pass when several passes are needed
constexpr int kOnePass = 384;   // up to this many tokens run in one pass (split accumulator chains)
constexpr int kMaxStages = 8;
constexpr int kWTileBytes = kBM * kBK * 2;  // 16 KB
constexpr int kSmemBytes = 212 * 1024;      // dynamic shared memory (tiles only)
constexpr int kThreads = 192;               // warp 0 TMA, warp 1 MMA, warps 2..5 epilogue
constexpr int kPrefetchChunks = 16;         // weight K-chunks pulled into L2 before the dependency wait

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* tm, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
          "r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(tm)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}
__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot)), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D[tmem] (+)= A[smem] * B[smem]^T, bf16 inputs, fp32 accumulate.
__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrives on `bar` once every MMA issued so far by this thread has completed.
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int j = 0; j < 16; ++j) v[j] = __uint_as_float(r[j]);
}

// Shared-memory matrix descriptor of a K-major operand in 128B-swizzled rows
// (8-row groups 1024 bytes apart).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);        // start address
  d |= (uint64_t)1 << 16;                          // leading byte offset (unused for swizzled K-major)
  d |= (uint64_t)((1024u >> 4) & 0x3FFFu) << 32;   // stride byte offset: next 8-row group
  d |= (uint64_t)1 << 46;                          // descriptor version
  d |= (uint64_t)2 << 61;                          // 128-byte swizzle
  return d;
}
// Instruction descriptor: bf16 x bf16 -> fp32, both operands K-major, M = 128.
__device__ __forceinline__ uint32_t idesc_bf16(int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);
}

__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ ActMaps tmA, const __grid_constant__ CUtensorMap tmW,
                   const int* __restrict__ m_ptr, int m_cap, int N, int k_chunks, int chunks_per_split,
                   float* __restrict__ out, size_t split_stride, int full_tiles, int tail,
                   float* __restrict__ tail_out, size_t tail_stride, int tail_ld, int chain_mode,
                   int* __restrict__ err, uint32_t wait_limit) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[kMaxStages];
  __shared__ __align__(8) uint64_t empty_bar[kMaxStages];
  __shared__ __align__(8) uint64_t acc_full, acc_empty;
  __shared__ uint32_t tmem_slot;
  __shared__ __align__(8) uint64_t drain_bar;
  __shared__ int abort_flag, never;
  __shared__ int prod_cnt[kMaxStages], cons_cnt[kMaxStages];
  __shared__ uint32_t last_par[kMaxStages];

  uint8_t* tiles = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // this CTA's weight tile and K range: the first full_tiles CTAs run a whole
  // tile; the rest cut the remaining tiles into `tail` K ranges each (with
  // full_tiles == 0 in the order of a (tiles x splits) grid)
  const int n_tiles = N / kBM;
  const int bx = blockIdx.x, by = blockIdx.y, ny = gridDim.y;
  int tile, sidx;  // sidx -1: the whole K range
  if (bx < full_tiles) {
    tile = bx;
    sidx = -1;
  } else if (full_tiles == 0) {
    tile = bx % n_tiles;
    sidx = bx / n_tiles;
  } else {
    const int j = bx - full_tiles;
    tile = full_tiles + j / tail;
    sidx = j - (j / tail) * tail;
  }
  const int n0 = tile * kBM;
  const int kc0 = sidx < 0 ? 0 : sidx * chunks_per_split;
  const int kc1 = sidx < 0 ? k_chunks : min(kc0 + chunks_per_split, k_chunks);
  if (threadIdx.x == 0) {
    // the weight tiles do not depend on earlier kernels: start pulling the
    // first ones into L2 while the previous kernel drains
    const int k1 = min(kc1, kc0 + kPrefetchChunks);
    for (int kc = kc0; kc < k1; ++kc)
      asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];" ::"l"(
                       reinterpret_cast<uint64_t>(&tmW)),
                   "r"(kc * kBK), "r"(n0)
                   : "memory");
  }
  pdl_wait();
  pdl_trigger();
  const int M_all = min(*m_ptr, m_cap);
  if (M_all <= 0) return;
  // token blocks (gridDim.y > 1): above one pass of rows every CTA takes one
  // block of kMaxTok rows, so the blocks of a tile run side by side instead
  // of as passes of one CTA; at or below it block 0 takes every row
  const int one_pass = chain_mode == 1 ? kMaxTok : kOnePass;
  int row_base = 0, M = M_all;
  if (ny > 1) {
    if (M_all <= one_pass) {
      if (by > 0) return;
    } else {
      row_base = by * kMaxTok;
      if (row_base >= M_all) return;
      M = min(M_all - row_base, kMaxTok);
    }
  }
  const int nk = kc1 - kc0;
  if (nk <= 0) return;
  // token passes: one pass up to one_pass tokens, else passes of kMaxTok
  // (every pass streams the weight tile again)
  const int pass_tok = M <= one_pass ? M : kMaxTok;
  const int tok_layout = ((min(M, pass_tok) + kBoxRows - 1) / kBoxRows) * kBoxRows;
  const uint32_t stage_bytes = kWTileBytes + (uint32_t)tok_layout * 128u;
  const int n_stages = min(kMaxStages, (int)((kSmemBytes - 1024) / stage_bytes));
  const int n_pass = (M + pass_tok - 1) / pass_tok;
  // Independent accumulator chains: consecutive MMAs into one accumulator
  // serialise, so the K steps of 16 alternate between C accumulators, added
  // in order by the epilogue.  chain_mode 1 (the default): always C = 2, at
  // most 256 tokens per pass (2 x 256 TMEM columns), so a token's fp32
  // summation order does not depend on which other tokens share the pass.
  // chain_mode 0: C = 4 for up to 128 tokens, 2 for up to 256, and above 256
  // the first `split` tokens get two chains and the rest one (split +
  // tok_layout <= 512 columns): one pass up to 384 tokens, not row-invariant.
  const int C = chain_mode == 1 ? 2 : tok_layout <= 128 ? 4 : tok_layout <= 256 ? 2 : 1;
  const int split = (C == 1 && chain_mode == 0) ? ((512 - tok_layout) / kBoxRows) * kBoxRows : 0;
  const uint32_t ncols = 512;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kMaxStages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
      prod_cnt[s] = 0;
      cons_cnt[s] = 0;
      last_par[s] = 0;
    }
    mbar_init(&acc_full, 1);
    mbar_init(&acc_empty, 4);
    mbar_init(&drain_bar, 1);
    abort_flag = 0;
    never = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    tmem_alloc(&tmem_slot, ncols);
    tmem_relinquish();
  }
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem_base = tmem_slot;
  volatile int* abort = &abort_flag;

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      for (int pass = 0; pass < n_pass && !*abort; ++pass) {
        const int row0 = pass * pass_tok;
        const int rows = min(M - row0, pass_tok);
        const int nbox = (rows + kBoxRows - 1) / kBoxRows;
        for (int kc = kc0; kc < kc1; ++kc) {
          if (!mbar_wait(&empty_bar[stage], phase ^ 1u, wait_limit, abort)) {
            set_error(err, VLAC_ERR_TIMEOUT);
            *abort = 1;
            break;
          }
          uint8_t* wt = tiles + (size_t)stage * stage_bytes;
          uint8_t* at = wt + kWTileBytes;
          mbar_expect_tx(&full_bar[stage], kWTileBytes + (uint32_t)nbox * kBoxRows * 128u);
          tma_load_2d(wt, &tmW, kc * kBK, n0, &full_bar[stage]);
          // the token rows in as few boxes as possible: 256, 128, 64 and 32 rows
          for (int done = 0, left = nbox; left > 0;) {
            const int lg = left >= 8 ? 3 : left >= 4 ? 2 : left >= 2 ? 1 : 0;
            tma_load_2d(at + (size_t)done * kBoxRows * 128, &tmA.m[lg], kc * kBK, row_base + row0 + done * kBoxRows,
                        &full_bar[stage]);
            done += 1 << lg;
            left -= 1 << lg;
          }
          prod_cnt[stage] += 1;
          last_par[stage] = phase;
          if (++stage == n_stages) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      for (int pass = 0; pass < n_pass && !*abort; ++pass) {
        const int rows = min(M - pass * pass_tok, pass_tok);
        if (pass > 0 && !mbar_wait(&acc_empty, (uint32_t)(pass - 1) & 1u, wait_limit, abort)) {
          set_error(err, VLAC_ERR_TIMEOUT);
          *abort = 1;
          break;
        }
        fence_after();
        for (int i = 0; i < nk; ++i) {
          if (!mbar_wait(&full_bar[stage], phase, wait_limit, abort)) {
            set_error(err, VLAC_ERR_TIMEOUT);
            *abort = 1;
            break;
          }
          cons_cnt[stage] += 1;
          fence_after();
          const uint32_t wt = smem_u32(tiles + (size_t)stage * stage_bytes);
          const uint32_t at = wt + kWTileBytes;
#pragma unroll
          for (int k16 = 0; k16 < kBK / 16; ++k16) {
            const uint64_t adesc = sw128_desc(wt + k16 * 32);
            if (split > 0) {
              // tokens [0, split): chain k16 % 2; tokens [split, rows): one chain
              umma_bf16(tmem_base + (k16 & 1) * split, adesc, sw128_desc(at + k16 * 32), idesc_bf16(split),
                        (i > 0 || k16 >= 2) ? 1u : 0u);
              const int nr = ((rows - split + 15) / 16) * 16;
              umma_bf16(tmem_base + 2 * split, adesc, sw128_desc(at + split * 128 + k16 * 32), idesc_bf16(nr),
                        (i > 0 || k16 > 0) ? 1u : 0u);
            } else if (C > 1) {
              // chain k16 % C accumulates every C-th K step
              const int n = ((rows + 15) / 16) * 16;
              const uint64_t bdesc = sw128_desc(at + k16 * 32);
              umma_bf16(tmem_base + (k16 % C) * tok_layout, adesc, bdesc, idesc_bf16(n),
                        (i > 0 || k16 >= C) ? 1u : 0u);
            } else {
              for (int sub = 0; sub * 256 < rows; ++sub) {
                const int n = min(256, ((rows - sub * 256 + 15) / 16) * 16);
                const uint64_t bdesc = sw128_desc(at + sub * 256 * 128 + k16 * 32);
                umma_bf16(tmem_base + sub * 256, adesc, bdesc, idesc_bf16(n), (i > 0 || k16 > 0) ? 1u : 0u);
              }
            }
          }
          umma_commit(&empty_bar[stage]);
          if (++stage == n_stages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        umma_commit(&acc_full);
      }
      if (*abort) {
        // every MMA issued so far must finish before TMEM and the tiles go away
        umma_commit(&drain_bar);
        mbar_wait(&drain_bar, 0, kWaitLimit, &never);
      }
    }
  } else {
    // ---------------- epilogue: TMEM -> fp32 partials ----------------
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    // where this CTA's partial goes: split 0 (or a whole tile) into out, a
    // later split into its uniform slot or the compact tail slots
    float* dst = out;
    int ld = N, n = n0 + q * 32 + lane;
    if (sidx > 0) {
      if (tail_ld) {
        dst = tail_out + (size_t)(sidx - 1) * tail_stride;
        ld = tail_ld;
        n -= full_tiles * kBM;
      } else {
        dst = out + (size_t)sidx * split_stride;
      }
    }
    for (int pass = 0; pass < n_pass; ++pass) {
      const int row0 = pass * pass_tok;
      const int rows = min(M - row0, pass_tok);
      bool ok = true;
      if (lane == 0) ok = mbar_wait(&acc_full, (uint32_t)pass & 1u, wait_limit, abort);
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) {
        if (lane == 0) {
          set_error(err, VLAC_ERR_TIMEOUT);
          *abort = 1;
        }
        break;
      }
      fence_after();
      for (int c0 = 0; c0 < rows; c0 += 16) {
        float v[16];
        const uint32_t lane_base = tmem_base + ((uint32_t)(q * 32) << 16);
        if (split > 0) {
          if (c0 < split) {  // the two chains, in order
            float w[16];
            tmem_ld16(lane_base + (uint32_t)c0, v);
            tmem_ld16(lane_base + (uint32_t)(split + c0), w);
#pragma unroll
            for (int j = 0; j < 16; ++j) v[j] += w[j];
          } else {
            tmem_ld16(lane_base + (uint32_t)(2 * split + (c0 - split)), v);
          }
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const int m = row0 + c0 + j;
            if (m < M) dst[(size_t)(row_base + m) * ld + n] = v[j];
          }
          continue;
        }
        tmem_ld16(lane_base + (uint32_t)c0, v);
        for (int ch = 1; ch < C; ++ch) {  // chains added in order
          float w[16];
          tmem_ld16(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(ch * tok_layout + c0), w);
#pragma unroll
          for (int j = 0; j < 16; ++j) v[j] += w[j];
        }
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const int m = row0 + c0 + j;
          if (m < M) dst[(size_t)(row_base + m) * ld + n] = v[j];
        }
      }
      fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty);
    }
  }

  __syncthreads();
  if (threadIdx.x == 0 && abort_flag) {
    // let every bulk copy that was issued but not consumed land before exit
    for (int s = 0; s < n_stages; ++s)
      if (prod_cnt[s] > cons_cnt[s]) mbar_wait(&full_bar[s], last_par[s], kWaitLimit, &never);
  }
  fence_before();
  __syncthreads();
  fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, ncols);
}

}  // namespace tc

void launch_gemm_tc(const ActMaps* tmA, const CUtensorMap* tmW, const int* m_ptr, int m_cap, int N, int K,
                    const SplitPlan& sp, float* out, int* err, uint32_t wait_limit, cudaStream_t st) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaFuncSetAttribute(tc::gemm_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, tc::kSmemBytes);
    attr_set = true;
  }
  const int k_chunks = K / tc::kBK;
  const int cps = (k_chunks + sp.tail - 1) / sp.tail;
  const int full_tiles = sp.full_cols / tc::kBM, n_tiles = N / tc::kBM;
  // token blocks side by side when the rows can exceed one pass (the CTAs of
  // blocks a step does not need return at once)
  // VLAC_GEMM_TOKEN_BLOCKS: 0 never, 1 whenever the rows exceed one pass.
  // Two passes inside one CTA stream the weight tile twice; blocks side by
  // side run the second pass on another SM at the same time, which pays off
  // where the extra CTAs find idle SMs and costs a wave where they do not.
  static const int token_blocks = [] {
    const char* e = std::getenv("VLAC_GEMM_TOKEN_BLOCKS");
    return e ? (std::atoi(e) != 0 ? 1 : 0) : -1;
  }();
  // accumulator chains (see gemm_tc_kernel): 1 (default) keeps every row's
  // summation order independent of the row count; VLAC_GEMM_CHAINS=0 selects
  // the row-count-dependent chains (faster for 257-384 rows, not
  // row-invariant), kept for measurement
  static const int chain_mode = [] {
    const char* e = std::getenv("VLAC_GEMM_CHAINS");
    return (e && std::atoi(e) == 0) ? 0 : 1;
  }();
  const int one_pass = chain_mode == 1 ? tc::kMaxTok : tc::kOnePass;
  const int nx = full_tiles + (n_tiles - full_tiles) * sp.tail;
  const int nb = (m_cap + tc::kMaxTok - 1) / tc::kMaxTok;
  // unset: side by side above two passes, or where all the blocks' CTAs fit
  // in about one and a third waves of SMs
  static const int n_sm = [] {
    int dev = 0, v = 152;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
    return v;
  }();
  const bool tb_on = m_cap > one_pass && (token_blocks == 1 ||
                                          (token_blocks < 0 && (m_cap > 2 * tc::kMaxTok || 3 * nx * nb <= 4 * n_sm)));
  const int tb = tb_on ? nb : 1;
  dim3 grid(nx, tb);
  launch_k(tc::gemm_tc_kernel, grid, dim3(tc::kThreads), tc::kSmemBytes, st, *tmA, *tmW, m_ptr, m_cap, N, k_chunks,
           cps, out, sp.stride, full_tiles, sp.tail, sp.tail_p, sp.tail_stride, sp.tail_ld, chain_mode, err,
           wait_limit);
}

// =============================================================================
// SIMT GEMM (fp32 tiny model): 64x64 output tile, 4x4 per thread.
// =============================================================================
template <typename T>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const T* __restrict__ A, const T* __restrict__ W,
                                                        const int* __restrict__ m_ptr, int m_cap, int N, int K,
                                                        float* __restrict__ out) {
  pdl_wait();
  pdl_trigger();
  __shared__ float As[16][64 + 1];
  __shared__ float Ws[16][64 + 1];
  const int M = min(*m_ptr, m_cap);
  const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
  if (m0 >= M) return;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += 16) {
    for (int t = threadIdx.x; t < 16 * 64; t += 256) {
      const int kk = t & 15, rr = t >> 4;
      const int m = m0 + rr, n = n0 + rr, k = k0 + kk;
      As[kk][rr] = (m < M && k < K) ? to_f(A[(size_t)m * K + k]) : 0.f;
      Ws[kk][rr] = (n < N && k < K) ? to_f(W[(size_t)n * K + k]) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float a[4], w[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a[i] = As[kk][ty * 4 + i];
        w[i] = Ws[kk][tx * 4 + i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], w[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int m = m0 + ty * 4 + i, n = n0 + tx * 4 + j;
      if (m < M && n < N) out[(size_t)m * N + n] = acc[i][j];
    }
}

template <typename T>
void launch_gemm_simt(const T* A, const T* W, const int* m_ptr, int m_cap, int N, int K, float* out,
                      cudaStream_t st) {
  dim3 grid((N + 63) / 64, (m_cap + 63) / 64);
  launch_k(gemm_simt_kernel<T>, grid, dim3(256), 0, st, A, W, m_ptr, m_cap, N, K, out);
}
template void launch_gemm_simt<float>(const float*, const float*, const int*, int, int, int, float*, cudaStream_t);

// =============================================================================
// Bounded-wait self-test: waits on an mbarrier that nothing completes.
// =============================================================================
__global__ void wait_selftest_kernel(int* err, uint32_t limit) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  if (threadIdx.x == 0 && !mbar_wait(&bar, 0, limit, &abort_flag)) set_error(err, VLAC_ERR_TIMEOUT);
}

int launch_wait_selftest(int* err, uint32_t spin_limit, cudaStream_t st) {
  wait_selftest_kernel<<<1, 32, 0, st>>>(err, spin_limit);
  return cudaGetLastError() == cudaSuccess ? 0 : -1;
}

}  // namespace vlac
