// bf16 LM-head path of pair_grad on the 5th-generation tensor cores
// (tcgen05 + TMEM + TMA, sm_103a).
//
// Objective (Sec. 4.5): J = sum_t c_t logp_t over compacted active tokens,
// logp_t = z_{t,y_t} - lse_t, z = W h. Its gradients split into an exact
// one-hot part (added in fp32 by grad_onehot) and a softmax part that is a
// pair of dense contractions through the logit gradient
//     Gs_tv = -c_t exp(z_tv - lse_t)      (bf16):
//     dH_t += sum_v Gs_tv W_v,     dW_v += sum_t Gs_tv h_t.
//
// Kernels (persistent, warp-specialised: a TMA producer warp, a TMEM-owning
// warp whose elected thread issues the MMAs, four epilogue warps on the four
// TMEM lane quadrants, one tile row per thread):
//   lse_kernel     : 128-token x 256-vocab tiles, K = d in 64-wide
//                    SWIZZLE_128B atoms, fp32 accumulators double-buffered in
//                    TMEM; the epilogue folds each 32-column chunk into an
//                    online (max, sum-exp) per token, picks the target logit
//                    and keeps the chunk's terms 2^(z log2 e - m_c) in fp16
//                    with m_c for the backward.
//   g_image_kernel : the bf16 Gs tiles (the logit-gradient image) from the
//                    kept terms, once, in the swizzled MMA-operand layout.
//   dh_gemm_kernel : dH = Gs . W, image tiles as the K-major A operand.
//   dw_gemm_kernel : dW = Gs^T . Hc, the same tiles read as the MN-major A
//                    operand.
// Without room for the image (no-alloc path, minimum workspace) the logits
// are recomputed: bwd_cluster_kernel (8-CTA clusters sharing each Gs tile
// through an L2 ring) for d = 512 A, else bwd_kernel (one CTA per row
// block and 256-wide d-slice).
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "pair_common.cuh"
#include "tc_ptx.cuh"

namespace pairk {
namespace {

using namespace tc;

constexpr int kThreads = 192;
constexpr int kAtom128 = 128 * 64 * 2;  // 128 rows x 64 bf16 (16 KB)

// ------------------------------------------------------------------ LSE
constexpr int kLseBN = 256;
constexpr int kLseStages = 4;
constexpr uint32_t kLseStageTx = (128 + kLseBN) * 64 * 2;
constexpr int kLsePair = 2;  // CTAs per cluster sharing each vocabulary tile
constexpr uint32_t kIdescLse = idesc_bf16(128, kLseBN, 0, 0);

struct LseSmem {
  uint8_t a[kLseStages][kAtom128];
  uint8_t b[kLseStages][2 * kAtom128];
  uint8_t stg[2][128 * 128];  // kept-term staging: per warp 32 rows x 64 fp16, SWIZZLE_128B
  uint64_t full[kLseStages], empty[kLseStages];
  uint64_t acc_full[2], acc_empty[2];
  uint64_t mma_done;
  uint32_t tmem_base;
  int abort;
};

// Named barrier of the four epilogue warps (128 threads).
__device__ __forceinline__ void epi_sync() {
  asm volatile("bar.sync 1, 128;" ::: "memory");
}

__device__ __forceinline__ uint8_t *align1k(uint8_t *p) {
  return reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(p) + 1023) &
                                     ~static_cast<uintptr_t>(1023));
}

// CTA pairs (2-CTA clusters) work on two token blocks of the same vocabulary
// split in lockstep: each CTA fetches its own token atom and one half (128
// rows) of the shared 256-row vocabulary atom, multicast into both CTAs'
// stage. A stage is refilled only after both CTAs' MMAs released it (each
// MMA warp commits to the empty barrier of both CTAs). This halves the
// vocabulary bytes each SM's copy engine requests, which is what limits the
// loads here (the engine's outstanding requests wait on DRAM-latency tiles).
__global__ void __cluster_dims__(kLsePair, 1, 1) __launch_bounds__(kThreads, 1)
    lse_kernel(const __grid_constant__ CUtensorMap tmH,
               const __grid_constant__ CUtensorMap tmW,
               const __grid_constant__ CUtensorMap tmS, int d, int V,
               int nsplit, int64_t Tpad, const int32_t *counters,
               const int32_t *tok_y, float2 *part, float *zy, int rb0, int cap,
               const void *sbuf, float4 *mbuf, int s_blocks, int32_t *dev_err) {
  extern __shared__ uint8_t smem_raw[];
  LseSmem &sm = *reinterpret_cast<LseSmem *>(align1k(smem_raw));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Teff = counters[0];
  // Token blocks [rb0, rb0 + n_tb) of this launch. With sbuf, the logits of
  // its first s_blocks blocks are also kept, per 32-column chunk c of a row
  // as P_j = 2^(z_j log2 e - m_c) in fp16 (in [0, 1]) with the chunk maximum
  // m_c = max_j z_j log2 e in fp32: 128 x 128 tiles, tile (b, vt) at
  // ((b * n_vt128 + vt) * 128 + row) * 128 + col of sbuf (written through
  // tmS, a [rows][128] fp16 view: each epilogue warp stages its 32 rows of
  // two chunks in shared memory and writes them with one TMA store), and
  // the row's four maxima as one float4 at mbuf[(b * n_vt128 + vt) * 128 +
  // row]. The same per-chunk terms P_j make up the log-sum-exp sum.
  const int n_tb = min(max((Teff + 127) / 128 - rb0, 0), cap);
  const int n_vt128 = (V + 127) / 128;
  const int s_lim = min(n_tb, s_blocks);
  const int n_vt = (V + kLseBN - 1) / kLseBN;
  // Work unit = (pair of token blocks, vocabulary split); CTA r of the pair
  // takes token block 2 * pair + r (past the last block for an odd count:
  // in-bounds padding rows whose results are never written).
  // Units (pair of token blocks, vocabulary split), split index fastest.
  // (Split-major order, which lets the pairs running at once share each W
  // split in L2, measured 4 % slower.)
  const int n_pairs = (n_tb + 1) / 2;
  const int n_units = n_pairs * nsplit;
  const int nk = d / 64;
  const int r = (int)cluster_rank();
  const int pid = (int)cluster_id_x(), npairs = (int)num_clusters_x();

  if (threadIdx.x == 0) {
    for (int s = 0; s < kLseStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kLsePair);  // both CTAs' MMAs done with the stage
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sm.acc_full[s], 1);
      mbar_init(&sm.acc_empty[s], 128);
    }
    mbar_init(&sm.mma_done, 1);
    sm.abort = 0;
    fence_mbar_init();
    prefetch_tmap(&tmH);
    prefetch_tmap(&tmW);
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // the peer's barriers exist before any multicast lands
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  volatile int *abort = &sm.abort;

  if (warp == 0) {
    {  // whole warp: uniform loop state; elected lane issues
      int stage = 0;
      uint32_t ph = 0;
      int last_ph[kLseStages];
      for (int s = 0; s < kLseStages; ++s) last_ph[s] = -1;
      bool ok = true;
      for (int u = pid; u < n_units && ok; u += npairs) {
        const int tb = rb0 + 2 * (u / nsplit) + r, sp = u % nsplit;
        const int vt0 = (int)((int64_t)sp * n_vt / nsplit);
        const int vt1 = (int)((int64_t)(sp + 1) * n_vt / nsplit);
        for (int vt = vt0; vt < vt1 && ok; ++vt) {
          for (int k = 0; k < nk; ++k) {
            if (!(ok = wait_cluster(&sm.empty[stage], ph ^ 1, abort, dev_err))) break;
            if (elect_one()) {
              mbar_expect_tx(&sm.full[stage], kLseStageTx);
              tma_load_2d(sm.a[stage], &tmH, &sm.full[stage], k * 64, tb * 128);
              tma_load_2d_mc(sm.b[stage] + r * (kLseBN / 2) * 128, &tmW, &sm.full[stage],
                             k * 64, vt * kLseBN + r * (kLseBN / 2), (uint16_t)3);
            }
            __syncwarp();
            last_ph[stage] = (int)ph;
            if (++stage == kLseStages) { stage = 0; ph ^= 1; }
          }
        }
      }
      // Never leave a copy in flight: wait (bounded) for the last one issued
      // on every stage.
      for (int s = 0; s < kLseStages; ++s)
        if (last_ph[s] >= 0) {
          volatile int never = 0;
          wait(&sm.full[s], (uint32_t)last_ph[s], &never, dev_err);
        }
    }
  } else if (warp == 1) {
    {  // whole warp: uniform loop state; elected lane issues
      int stage = 0, acc = 0;
      uint32_t ph = 0, acc_ph = 0;
      const uint64_t da0 = sdesc_sw128(smem_u32(sm.a[0]), 16, 1024);
      const uint64_t db0 = sdesc_sw128(smem_u32(sm.b[0]), 16, 1024);
      bool ok = true;
      for (int u = pid; u < n_units && ok; u += npairs) {
        const int sp = u % nsplit;
        const int vt0 = (int)((int64_t)sp * n_vt / nsplit);
        const int vt1 = (int)((int64_t)(sp + 1) * n_vt / nsplit);
        for (int vt = vt0; vt < vt1 && ok; ++vt) {
          if (!(ok = wait(&sm.acc_empty[acc], acc_ph ^ 1, abort, dev_err))) break;
          tc_fence_after();
          const uint32_t dt = tmem + acc * kLseBN;
          for (int k = 0; k < nk; ++k) {
            if (!(ok = wait(&sm.full[stage], ph, abort, dev_err))) break;
            const uint64_t da = da0 + (uint64_t)stage * (kAtom128 >> 4);
            const uint64_t db = db0 + (uint64_t)stage * ((2 * kAtom128) >> 4);
            if (elect_one()) {
#pragma unroll
              for (int kk = 0; kk < 4; ++kk)
                mma_bf16(dt, da + 2 * kk, db + 2 * kk, kIdescLse, (k | kk) != 0);
              mma_commit_multicast(&sm.empty[stage], (uint16_t)3);
            }
            __syncwarp();
            if (++stage == kLseStages) { stage = 0; ph ^= 1; }
          }
          if (!ok) break;
          if (elect_one()) mma_commit(&sm.acc_full[acc]);
          __syncwarp();
          if (++acc == 2) { acc = 0; acc_ph ^= 1; }
        }
      }
      if (elect_one()) mma_commit(&sm.mma_done);
      __syncwarp();
      volatile int never = 0;
      wait(&sm.mma_done, 0, &never, dev_err);
    }
  } else {
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_addr = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    int acc = 0, sbuf_i = 0;
    uint32_t acc_ph = 0;
    bool ok = true;
    for (int u = pid; u < n_units && ok; u += npairs) {
      const int tbl = 2 * (u / nsplit) + r, sp = u % nsplit;
      const int tb = rb0 + tbl;
      const int vt0 = (int)((int64_t)sp * n_vt / nsplit);
      const int vt1 = (int)((int64_t)(sp + 1) * n_vt / nsplit);
      const int p = tb * 128 + row;
      const bool valid = p < Teff;
      const bool keep = sbuf && tbl < s_lim;  // uniform over the CTA
      float mrow[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
      const int yt = valid ? tok_y[p] : -1;
      float m2 = -INFINITY, l = 0.f, zt = 0.f;
      bool found = false;
      for (int vt = vt0; vt < vt1; ++vt) {
        if (!(ok = wait_sleepy(&sm.acc_full[acc], acc_ph, abort, dev_err))) break;
        tc_fence_after();
#pragma unroll 1
        for (int c = 0; c < kLseBN / 32; ++c) {
          float v[32];
          tmem_ld32(lane_addr + acc * kLseBN + c * 32, v);
          const int col0 = vt * kLseBN + c * 32;
          const int off = yt - col0;
          if (off >= 0 && off < 32) {
            found = true;
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (j == off) zt = v[j];
          }
          const int nvalid = V - col0;  // columns >= V are padding
          float mc = -INFINITY;
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            v[j] = (j < nvalid) ? v[j] * kLog2e : -INFINITY;
            mc = fmaxf(mc, v[j]);
          }
          if (mc == -INFINITY) continue;  // the whole chunk lies past V
          // Chunk terms relative to the chunk maximum, then folded into the
          // running (max, sum): v[j] becomes P_j.
          float s = 0.f;
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            v[j] = ex2_approx(v[j] - mc);
            s += v[j];
          }
          if (mc > m2) {
            l = l * ex2_approx(m2 - mc) + s;
            m2 = mc;
          } else {
            l += s * ex2_approx(mc - m2);
          }
          if (keep) {
            // Per warp: its 32 rows x 64 columns (two chunks) in fp16, in its
            // own 4 KB buffer, stored by its lane 0 once both halves (or the
            // last chunk before V) are in. The store that last read this
            // buffer is done before the first half is written.
            const int half = c & 1;
            if (half == 0) {
              if (lane == 0) bulk_wait_group_read<1>();
              __syncwarp();
            }
            uint8_t *buf = sm.stg[sbuf_i] + quad * 4096;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              uint32_t pk[4];
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                __half2 h2 = __floats2half2_rn(v[8 * e + 2 * q], v[8 * e + 2 * q + 1]);
                pk[q] = *reinterpret_cast<uint32_t *>(&h2);
              }
              *reinterpret_cast<uint4 *>(buf + lane * 128 + (((half * 4 + e) ^ (lane & 7)) << 4)) =
                  make_uint4(pk[0], pk[1], pk[2], pk[3]);
            }
            mrow[c & 3] = mc;
            const bool last = col0 + 32 >= V;
            if (half == 1 || last) {
              fence_async_smem();
              __syncwarp();
              if (lane == 0) {
                tma_store_2d_evict_first(&tmS, buf, col0 & 64,
                                         (tbl * n_vt128 + (col0 >> 7)) * 128 + quad * 32);
                bulk_commit_group();
              }
              sbuf_i ^= 1;
            }
            if ((c & 3) == 3 || last) {
              mbuf[((int64_t)tbl * n_vt128 + (col0 >> 7)) * 128 + row] =
                  make_float4(mrow[0], mrow[1], mrow[2], mrow[3]);
              mrow[0] = mrow[1] = mrow[2] = mrow[3] = -INFINITY;
            }
          }
        }
        tc_fence_before();
        mbar_arrive(&sm.acc_empty[acc]);
        if (++acc == 2) { acc = 0; acc_ph ^= 1; }
      }
      if (!ok) break;
      if (valid) {
        part[(int64_t)sp * Tpad + p] = make_float2(m2, l);
        if (found) zy[p] = zt;
      }
    }
    // Every kept-logit store has completed before the CTA leaves.
    if (lane == 0) bulk_wait_group<0>();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no CTA leaves while its peer may still signal or fill it
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// lse_t = ln 2 * (M + log2 sum_s l_s 2^(m_s - M)) over the vocabulary splits.
// Tokens [128 rb0, 128 (rb0 + cap)) of the active ones.
__global__ void lse_combine_kernel(int nsplit, int64_t Tpad,
                                   const int32_t *counters, const float2 *part,
                                   float *lse, int rb0, int cap) {
  const int Teff = counters[0];
  const int64_t hi64 = (int64_t)(rb0 + (int64_t)cap) * 128;
  const int p1 = (int)(hi64 < Teff ? hi64 : Teff);
  for (int p = rb0 * 128 + blockIdx.x * blockDim.x + threadIdx.x; p < p1;
       p += gridDim.x * blockDim.x) {
    float M = -INFINITY;
    for (int s = 0; s < nsplit; ++s) M = fmaxf(M, part[(int64_t)s * Tpad + p].x);
    float L = 0.f;
    for (int s = 0; s < nsplit; ++s) {
      const float2 q = part[(int64_t)s * Tpad + p];
      if (q.y > 0.f) L += q.y * exp2f(q.x - M);
    }
    lse[p] = (M + log2f(L)) * 0.6931471805599453f;
  }
}

// ------------------------------------------------------------- backward
constexpr int kBwdBN = 128;     // S tile columns
constexpr int kSlice = 256;     // output columns held in TMEM per unit
constexpr int kBwdStages = 3;
constexpr uint32_t kBwdStageTx = 2 * kAtom128;
constexpr uint32_t kIdescS = idesc_bf16(128, kBwdBN, 0, 0);

struct BwdSmem {
  uint8_t a[kBwdStages][kAtom128];   // rows-operand atoms (128 x 64)
  uint8_t b[kBwdStages][kAtom128];   // cols-operand atoms (128 x 64)
  uint8_t cs[kSlice / 64][kAtom128]; // cols operand, d-slice (MN-major B)
  uint8_t g[kBwdBN / 64][kAtom128];  // Gs tile, K-major A (2 atoms along K)
  float col_c[kBwdBN], col_l[kBwdBN];
  uint64_t full[kBwdStages], empty[kBwdStages];
  uint64_t s_full[2], s_empty[2];
  uint64_t g_full, g_empty, cs_full, cs_empty, o_full, o_empty, mma_done;
  uint32_t tmem_base;
  int abort;
};

// kTokenRows: rows = tokens (output dH), cols = vocabulary.
// otherwise : rows = vocabulary (output dW), cols = tokens.
template <bool kTokenRows>
__global__ void __launch_bounds__(kThreads, 1)
    bwd_kernel(const __grid_constant__ CUtensorMap tmR,
               const __grid_constant__ CUtensorMap tmC, int d, int V,
               const int32_t *counters, const int32_t *tok_idx,
               const float *tok_c, const float *lse, float *out,
               int32_t *dev_err) {
  extern __shared__ uint8_t smem_raw[];
  BwdSmem &sm = *reinterpret_cast<BwdSmem *>(align1k(smem_raw));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Teff = counters[0];
  const int nsl = (d + kSlice - 1) / kSlice;
  const int n_rb = kTokenRows ? (Teff + 127) / 128 : (V + 127) / 128;
  const int n_ct = kTokenRows ? (V + kBwdBN - 1) / kBwdBN : (Teff + kBwdBN - 1) / kBwdBN;
  const int n_units = n_rb * nsl;
  const int nk = d / 64;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kBwdStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sm.s_full[s], 1);
      mbar_init(&sm.s_empty[s], 128);
    }
    mbar_init(&sm.g_full, 128);
    mbar_init(&sm.g_empty, 1);
    mbar_init(&sm.cs_full, 1);
    mbar_init(&sm.cs_empty, 1);
    mbar_init(&sm.o_full, 1);
    mbar_init(&sm.o_empty, 128);
    mbar_init(&sm.mma_done, 1);
    sm.abort = 0;
    fence_mbar_init();
    prefetch_tmap(&tmR);
    prefetch_tmap(&tmC);
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  const uint32_t tmem_o = tmem + 2 * kBwdBN;  // columns [256, 512)
  volatile int *abort = &sm.abort;

  if (warp == 0) {
    {  // whole warp: uniform loop state; elected lane issues
      int stage = 0;
      uint32_t ph = 0, cs_ph = 0;
      int last_ph[kBwdStages];
      for (int s = 0; s < kBwdStages; ++s) last_ph[s] = -1;
      int cs_last = -1;
      bool ok = true;
      auto load_s = [&](int rb, int ct) {
        for (int k = 0; k < nk && ok; ++k) {
          if (!(ok = wait(&sm.empty[stage], ph ^ 1, abort, dev_err))) break;
          if (elect_one()) {
            mbar_expect_tx(&sm.full[stage], kBwdStageTx);
            tma_load_2d(sm.a[stage], &tmR, &sm.full[stage], k * 64, rb * 128);
            tma_load_2d(sm.b[stage], &tmC, &sm.full[stage], k * 64, ct * kBwdBN);
          }
          __syncwarp();
          last_ph[stage] = (int)ph;
          if (++stage == kBwdStages) { stage = 0; ph ^= 1; }
        }
      };
      auto load_cs = [&](int sl, int w, int ct) {
        if (!ok) return;
        if (!(ok = wait(&sm.cs_empty, cs_ph ^ 1, abort, dev_err))) return;
        if (elect_one()) {
          mbar_expect_tx(&sm.cs_full, (uint32_t)(w / 64) * kAtom128);
          for (int j = 0; j < w / 64; ++j)
            tma_load_2d(sm.cs[j], &tmC, &sm.cs_full, sl * kSlice + j * 64, ct * kBwdBN);
        }
        __syncwarp();
        cs_last = (int)cs_ph;
        cs_ph ^= 1;
      };
      for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
        const int rb = u / nsl, sl = u % nsl;
        const int w = min(kSlice, d - sl * kSlice);
        if (n_ct == 0) continue;
        load_s(rb, 0);
        for (int ct = 1; ct < n_ct && ok; ++ct) {
          load_s(rb, ct);
          load_cs(sl, w, ct - 1);
        }
        load_cs(sl, w, n_ct - 1);
      }
      volatile int never = 0;
      for (int s = 0; s < kBwdStages; ++s)
        if (last_ph[s] >= 0) wait(&sm.full[s], (uint32_t)last_ph[s], &never, dev_err);
      if (cs_last >= 0) wait(&sm.cs_full, (uint32_t)cs_last, &never, dev_err);
    }
  } else if (warp == 1) {
    {  // whole warp: uniform loop state; elected lane issues
      int stage = 0;
      uint32_t ph = 0, s_ph[2] = {0, 0}, g_ph = 0, cs_ph = 0, o_ph = 0;
      bool ok = true;
      auto issue_s = [&](int ct) {
        const int buf = ct & 1;
        if (!(ok = wait(&sm.s_empty[buf], s_ph[buf] ^ 1, abort, dev_err))) return;
        tc_fence_after();
        const uint32_t dt = tmem + buf * kBwdBN;
        for (int k = 0; k < nk; ++k) {
          if (!(ok = wait(&sm.full[stage], ph, abort, dev_err))) return;
          const uint32_t sa = smem_u32(sm.a[stage]), sb = smem_u32(sm.b[stage]);
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              mma_bf16(dt, sdesc_sw128(sa + kk * 32, 16, 1024),
                       sdesc_sw128(sb + kk * 32, 16, 1024), kIdescS,
                       (k | kk) != 0);
            mma_commit(&sm.empty[stage]);
          }
          __syncwarp();
          if (++stage == kBwdStages) { stage = 0; ph ^= 1; }
        }
        if (elect_one()) mma_commit(&sm.s_full[buf]);
        __syncwarp();
        s_ph[buf] ^= 1;
      };
      auto issue_o = [&](int ct, int w) {
        if (!ok) return;
        if (!(ok = wait(&sm.g_full, g_ph, abort, dev_err))) return;
        if (!(ok = wait(&sm.cs_full, cs_ph, abort, dev_err))) return;
        if (ct == 0 && !(ok = wait(&sm.o_empty, o_ph ^ 1, abort, dev_err))) return;
        tc_fence_after();
        const uint32_t idesc = idesc_bf16(128, w, 0, 1);
        const uint32_t sg = smem_u32(sm.g[0]), sc = smem_u32(sm.cs[0]);
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < kBwdBN / 16; ++kk) {
            const uint64_t ad = sdesc_sw128(sg + (kk >> 2) * kAtom128 + (kk & 3) * 32, 16, 1024);
            const uint64_t bd = sdesc_sw128(sc + kk * 2048, kAtom128, 1024);
            mma_bf16(tmem_o, ad, bd, idesc, (ct | kk) != 0);
          }
          mma_commit(&sm.g_empty);
          mma_commit(&sm.cs_empty);
        }
        __syncwarp();
        g_ph ^= 1;
        cs_ph ^= 1;
      };
      for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
        const int sl = u % nsl;
        const int w = min(kSlice, d - sl * kSlice);
        if (n_ct == 0) continue;
        issue_s(0);
        for (int ct = 0; ct < n_ct && ok; ++ct) {
          if (ct + 1 < n_ct) issue_s(ct + 1);
          issue_o(ct, w);
        }
        if (!ok) break;
        if (elect_one()) mma_commit(&sm.o_full);
        __syncwarp();
        o_ph ^= 1;
      }
      if (elect_one()) mma_commit(&sm.mma_done);
      __syncwarp();
      volatile int never = 0;
      wait(&sm.mma_done, 0, &never, dev_err);
    }
  } else {
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    uint32_t s_ph[2] = {0, 0}, g_ph = 0, o_ph = 0;
    bool ok = true;
    for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
      const int rb = u / nsl, sl = u % nsl;
      const int w = min(kSlice, d - sl * kSlice);
      const int rid = rb * 128 + row;  // token position or vocabulary id
      float rc = 0.f, rl = 0.f;
      if (kTokenRows && rid < Teff) {
        rc = tok_c[rid];
        rl = lse[rid] * kLog2e;
      }
      for (int ct = 0; ct < n_ct; ++ct) {
        if (!kTokenRows) {
          epi_sync();
          const int p = ct * kBwdBN + row;
          sm.col_c[row] = p < Teff ? tok_c[p] : 0.f;
          sm.col_l[row] = p < Teff ? lse[p] * kLog2e : 0.f;
          epi_sync();
        }
        const int buf = ct & 1;
        if (!(ok = wait(&sm.s_full[buf], s_ph[buf], abort, dev_err))) break;
        s_ph[buf] ^= 1;
        if (!(ok = wait(&sm.g_empty, g_ph ^ 1, abort, dev_err))) break;
        tc_fence_after();
#pragma unroll 1
        for (int c = 0; c < kBwdBN / 32; ++c) {
          float v[32];
          tmem_ld32(tmem + lane_off + buf * kBwdBN + c * 32, v);
          uint32_t pk[16];
#pragma unroll
          for (int j = 0; j < 32; j += 2) {
            float g2[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int col = c * 32 + j + e;
              float cc, ll;
              bool live;
              if (kTokenRows) {
                cc = rc; ll = rl;
                live = (rc != 0.f) && (ct * kBwdBN + col < V);
              } else {
                cc = sm.col_c[col]; ll = sm.col_l[col];
                live = cc != 0.f;
              }
              g2[e] = live ? -cc * ex2_approx(fmaf(v[j + e], kLog2e, -ll)) : 0.f;
            }
            __nv_bfloat162 b2 = __floats2bfloat162_rn(g2[0], g2[1]);
            pk[j >> 1] = *reinterpret_cast<uint32_t *>(&b2);
          }
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const int k = c * 32 + q * 8;  // first column of this 16-byte piece
            uint8_t *dst = sm.g[k >> 6] + sw128_offset(row, k & 63);
            *reinterpret_cast<uint4 *>(dst) =
                make_uint4(pk[q * 4], pk[q * 4 + 1], pk[q * 4 + 2], pk[q * 4 + 3]);
          }
        }
        tc_fence_before();
        mbar_arrive(&sm.s_empty[buf]);
        fence_async_smem();
        mbar_arrive(&sm.g_full);
        g_ph ^= 1;
      }
      if (!ok) break;
      const bool valid = kTokenRows ? (rid < Teff) : (rid < V);
      float *dst = nullptr;
      if (valid)
        dst = out + (kTokenRows ? (int64_t)tok_idx[rid] : (int64_t)rid) * d + sl * kSlice;
      if (n_ct == 0) {
        if (valid)
          for (int k = 0; k < w; ++k) dst[k] = 0.f;
        continue;
      }
      if (!(ok = wait(&sm.o_full, o_ph, abort, dev_err))) break;
      o_ph ^= 1;
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < w / 32; ++c) {
        float v[32];
        tmem_ld32(tmem_o + lane_off + c * 32, v);
        if (valid) {
#pragma unroll
          for (int q = 0; q < 8; ++q)
            reinterpret_cast<float4 *>(dst + c * 32)[q] =
                make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        }
      }
      tc_fence_before();
      mbar_arrive(&sm.o_empty);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// ------------------------------------------------- backward, cluster form
//
// One 8-CTA cluster owns a row block (128 tokens for dH, 128 vocabulary rows
// for dW); CTA k of the cluster keeps out[rows, k*w : (k+1)*w] (w = d/8) in
// TMEM for the whole unit, so each logit-gradient tile Gs is formed once per
// cluster instead of once per d-slice.
//
// Tile ownership rotates: the owner of column tile g (g mod 8) accumulates
// the full-depth S tile in TMEM, spread evenly over the 8 slots that end
// kClLag slots before the tile is used (d/512 K-atoms per slot), converts it
// to bf16 Gs and publishes the 32 KB tile (already in the swizzled K-major
// layout of the MMA operand) once, to a per-cluster ring in global memory,
// then signals every CTA of the cluster through its pub[owner][m & 1]
// mbarrier (m = g / 8, the owner's tile count). Every CTA pulls Gs(s) into
// shared memory with a bulk copy and updates out += Gs(s) . C[s, slice].
// The ring holds two tiles per owner, and an owner overwrites its slot of
// tile g - 16 only after every CTA is done with that tile; with two pub
// barriers per owner this also keeps any consumer's parity wait unambiguous,
// and it leaves 16 slots (not 8) for the round trip consume -> convert ->
// publish -> load. The exchange goes through L2
// because distributed shared memory sustains far less per-SM egress than a
// broadcast of a 32 KB tile to 7 peers per slot needs. In every slot every
// CTA issues the same tensor work: a share of one S accumulation plus one
// output update. The slot counter runs across units, so the staggered S
// schedule never drains at unit boundaries.
//
// The column tile is BN wide (BN = 128 for d <= 2048, 96 for d = 2560, 64
// for d = 3072): TMEM holds two BN-column S buffers plus the d/8-column
// output slice, 2 BN + d/8 <= 512.
constexpr int kCl = 8;          // cluster size (power of two)
constexpr int kClStages = 4;    // S operand stages
constexpr int kClLag = 3;       // slots between an S tile's completion and its use
constexpr int kClJ = kCl + kClLag;
constexpr int kGSlots = 1;      // Gs tiles staged in shared memory
constexpr int kClThreads = 256; // + warp 6: loads of C[s, slice] and Gs; warp 7: output MMAs

template <int BN>
struct ClTile {
  static constexpr uint32_t kColAtom = BN * 64 * 2;         // BN rows x 64 bf16
  static constexpr int kGsAtoms = (BN + 63) / 64;           // Gs K-major atoms
  static constexpr uint32_t kGsBytes = kGsAtoms * kAtom128; // one Gs tile
  static constexpr int kCsAtoms = (512 - 2 * BN) / 64;      // max output-slice atoms
  static constexpr uint32_t kIdescS = idesc_bf16(128, BN, 0, 0);
};

template <int BN>
struct ClSmem {
  using T = ClTile<BN>;
  uint8_t a[kClStages][kAtom128];                 // rows operand atoms (128 x 64)
  uint8_t b[kClStages][T::kColAtom];              // column operand atoms (BN x 64)
  uint8_t cs[T::kCsAtoms][T::kColAtom];           // C[s, slice]: MN-major B
  uint8_t g[kGSlots][T::kGsAtoms][kAtom128];      // Gs tiles: 128 x BN bf16, K-major A
  float col_c[BN], col_l[BN];
  uint64_t full[kClStages], empty[kClStages];
  uint64_t s_full[2], s_empty[2];
  uint64_t g_full[kGSlots], gs_empty[kGSlots];
  uint64_t cs_full[2], cs_empty[2];  // C[s, slice] in two column parts
  uint64_t pub[kCl][2];              // owner o published its tile m (by m & 1)
  uint64_t gfree[2];                 // (owner) all CTAs done with its tile m (by m & 1)
  uint64_t o_full, o_empty, mma_done;
  uint32_t tmem_base;
  int abort;
};

// Bulk copy global -> this CTA's shared memory, completing on `bar`.
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes,
                                          uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1], %2, [%3];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// The tiles of one cluster, in processing order: first its F = n_rb / ncl
// full row blocks (cid, cid + ncl, ...), each with all n_ct column tiles;
// then an even share [t0, t1) of the row-major tiles of the remaining
// R = n_rb mod ncl row blocks, so that all clusters finish within a tile of
// each other. A unit (run of tiles with one row block) in that tail may cover
// only part of its row block. Since R < ncl, a cluster's share has at most
// n_ct tiles and so at most two tail units; each is stored to the cluster's
// scratch slot (cid, u) and tail_reduce_kernel sums the slots of every tail
// row in cluster order (deterministic, no atomics).
struct TileMap {
  int n_ct, ncl, cid, gT, t0, rbT, N;
  __device__ void setup(int n_rb, int n_ct_, int cid_, int ncl_) {
    n_ct = n_ct_;
    ncl = ncl_;
    cid = cid_;
    const int F = n_ct ? n_rb / ncl : 0;
    const int R = n_ct ? n_rb - F * ncl : 0;
    const int64_t T = (int64_t)R * n_ct;
    gT = F * n_ct;
    rbT = F * ncl;
    t0 = (int)(T * cid / ncl);
    N = gT + (int)(T * (cid + 1) / ncl) - t0;
  }
  __device__ bool tail(int g) const { return g >= gT; }
};

// Walks tile indices g = 0, 1, 2, ... of a TileMap as (row block, column
// tile) pairs without divisions in the loop.
struct TileCursor {
  int ct, rb, g;
  __device__ void init(const TileMap &mp, int g_) {
    g = g_;
    if (mp.n_ct == 0) {
      ct = 0;
      rb = mp.cid;
    } else if (g < mp.gT) {
      ct = g % mp.n_ct;
      rb = mp.cid + (g / mp.n_ct) * mp.ncl;
    } else {
      const int t = mp.t0 + (g - mp.gT);
      ct = t % mp.n_ct;
      rb = mp.rbT + t / mp.n_ct;
    }
  }
  __device__ void next(const TileMap &mp) {
    ++g;
    if (g == mp.gT) {
      ct = mp.t0 % mp.n_ct;
      rb = mp.rbT + mp.t0 / mp.n_ct;
    } else if (++ct == mp.n_ct) {
      ct = 0;
      rb += g < mp.gT ? mp.ncl : 1;
    }
  }
  __device__ bool unit_start(const TileMap &mp) const { return ct == 0 || g == mp.gT; }
  __device__ bool unit_end(const TileMap &mp) const { return ct == mp.n_ct - 1 || g == mp.N - 1; }
};

// Final values of the tail rows (see TileMap) of the chunk of row blocks
// [rb0, rb0 + cap): for each row, the sum in cluster order of the partial
// units the clusters stored to their scratch slots.
template <bool kTokenRows, int BN>
__global__ void tail_reduce_kernel(int d, int V, int ncl, int rb0, int cap,
                                   const int32_t *counters, const int32_t *tok_idx,
                                   const float *tailbuf, float *out) {
  const int Teff = counters[0];
  const int n_rows = kTokenRows ? Teff : V;
  const int n_ct = kTokenRows ? (V + BN - 1) / BN : (Teff + BN - 1) / BN;
  const int n_rb = min(max((n_rows + 127) / 128 - rb0, 0), cap);
  if (n_ct == 0) return;
  const int F = n_rb / ncl, R = n_rb - F * ncl;
  if (R == 0) return;
  const int64_t Tt = (int64_t)R * n_ct;
  const int r0 = (rb0 + F * ncl) * 128;
  const int r1 = min(n_rows, (rb0 + n_rb) * 128);
  const int vec = d / 4;
  const float4 *src = reinterpret_cast<const float4 *>(tailbuf);
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
       i < (int64_t)(r1 - r0) * vec; i += (int64_t)gridDim.x * blockDim.x) {
    const int off = (int)(i / vec);           // row offset from r0
    const int rl = off >> 7, rr = off & 127;  // tail row block, row within it
    const int c4 = (int)(i % vec);
    const int64_t lo = (int64_t)rl * n_ct, hi = lo + n_ct;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int c = 0; c < ncl; ++c) {
      const int64_t a = Tt * c / ncl, b = Tt * (c + 1) / ncl;
      if ((a > lo ? a : lo) < (b < hi ? b : hi)) {
        const int u = rl - (int)(a / n_ct);  // this row block's unit in cluster c
        const float4 p = src[((int64_t)(c * 2 + u) * 128 + rr) * vec + c4];
        acc.x += p.x; acc.y += p.y; acc.z += p.z; acc.w += p.w;
      }
    }
    const int rid = r0 + off;
    const int64_t row = kTokenRows ? (int64_t)tok_idx[rid] : (int64_t)rid;
    reinterpret_cast<float4 *>(out + row * d)[c4] = acc;
  }
}

template <bool kTokenRows, int BN>
__global__ void __cluster_dims__(kCl, 1, 1) __launch_bounds__(kClThreads, 1)
    bwd_cluster_kernel(const __grid_constant__ CUtensorMap tmR,
                       const __grid_constant__ CUtensorMap tmC,
                       const __grid_constant__ CUtensorMap tmC64, int d, int V,
                       const int32_t *counters, const int32_t *tok_idx,
                       const float *tok_c, const float *lse, float *out,
                       uint8_t *gring, uint8_t *gimg, float *tailbuf, int rb0, int cap,
                       int32_t *dev_err) {
  extern __shared__ uint8_t smem_raw[];
  ClSmem<BN> &sm = *reinterpret_cast<ClSmem<BN> *>(align1k(smem_raw));
  using Tl = ClTile<BN>;
  constexpr uint32_t kGsBytes = Tl::kGsBytes, kColAtom = Tl::kColAtom;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int k = (int)cluster_rank();
  const int cid = (int)cluster_id_x(), ncl = (int)num_clusters_x();
  const int Teff = counters[0];
  const int A = d / (64 * kCl);            // K-atoms per slot (d / 512)
  const int w = 64 * A;                    // this CTA's d-slice width
  const int nk = d / 64;
  // The output update runs in two parts with their own operand barriers, so
  // part 0's operands of the next slot load while part 1 still computes.
  // With a 128-wide tile and a slice of at most 256 columns (d <= 2048) the
  // parts are the two 64-row K halves of the tile (Gs atom p with rows
  // [64p, 64p + 64) of C[s, slice]; 256-wide MMAs); otherwise they are two
  // column parts of A0 and A - A0 atoms of the slice.
  const bool ksplit = BN == 128 && A <= 4;
  const int A0 = ksplit ? A : (A + 1) >> 1, A1 = ksplit ? A : A - A0;
  // Row blocks [rb0, rb0 + n_rb) of this launch (one chunk); TileMap and
  // TileCursor count them from 0.
  const int n_rb = min(max((kTokenRows ? (Teff + 127) / 128 : (V + 127) / 128) - rb0, 0), cap);
  const int n_ct = kTokenRows ? (V + BN - 1) / BN : (Teff + BN - 1) / BN;
  const int n_my = cid < n_rb ? (n_rb - cid + ncl - 1) / ncl : 0;
  TileMap mp;
  mp.setup(n_rb, n_ct, cid, ncl);
  const int N = mp.N;                      // tiles of this cluster
  // Ring of published Gs tiles: [owner][job parity] for this cluster.
  uint8_t *ring = gring + (size_t)cid * kCl * 2 * kGsBytes;
  // Where tile g (chunk row block rb, column tile ct) is published: its own
  // slot of the logit-gradient image when the launch keeps one (a later pass
  // reads it again), else the ring slot.
  auto gs_tile = [&](int g, int rb, int ct) {
    return gimg ? gimg + ((size_t)rb * n_ct + ct) * kGsBytes
                : ring + ((size_t)(g & (kCl - 1)) * 2 + (size_t)((g >> 3) & 1)) * kGsBytes;
  };
  // The tile whose S this CTA accumulates during slot s (may be < 0 or >= N).
  auto job_of = [&](int s) {
    const int g0 = s + kClLag + 1;
    return g0 + ((k - g0) & (kCl - 1));
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < kClStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sm.s_full[s], 1);
      mbar_init(&sm.s_empty[s], 128);
      mbar_init(&sm.gfree[s], kCl);
    }
    for (int s = 0; s < kGSlots; ++s) {
      mbar_init(&sm.g_full[s], 1);
      mbar_init(&sm.gs_empty[s], 1);
    }
    for (int p = 0; p < 2; ++p) {
      mbar_init(&sm.cs_full[p], 1);
      mbar_init(&sm.cs_empty[p], 1);
    }
    for (int o = 0; o < kCl; ++o) {
      mbar_init(&sm.pub[o][0], 1);
      mbar_init(&sm.pub[o][1], 1);
    }
    mbar_init(&sm.o_full, 1);
    mbar_init(&sm.o_empty, 128);
    mbar_init(&sm.mma_done, 2);  // one final commit per MMA-issuing warp
    sm.abort = 0;
    fence_mbar_init();
    prefetch_tmap(&tmR);
    prefetch_tmap(&tmC);
    prefetch_tmap(&tmC64);
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // every CTA's barriers exist before anyone signals them
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  const uint32_t tmem_o = tmem + 2 * BN;
  volatile int *abort = &sm.abort;

  if (warp == 0) {
    // Producer of the S operands (this CTA's share of its owned tiles).
    {  // whole warp: uniform loop state; elected lane issues
      int stage = 0;
      uint32_t ph = 0;
      int last_ph[kClStages];
      for (int s = 0; s < kClStages; ++s) last_ph[s] = -1;
      bool ok = true;
      int job_rb = 0, job_ct = 0, job_g = -1;
      for (int s = -kClJ; s < N && ok; ++s) {
        const int gj = job_of(s);
        if (gj < 0 || gj >= N) continue;
        if (gj != job_g) {
          TileCursor c;
          c.init(mp, gj);
          job_rb = c.rb; job_ct = c.ct; job_g = gj;
        }
        const int a0 = (s - (gj - kClJ)) * A;
        for (int a = a0; a < a0 + A; ++a) {
          if (!(ok = wait(&sm.empty[stage], ph ^ 1, abort, dev_err))) break;
          if (elect_one()) {
            mbar_expect_tx(&sm.full[stage], kAtom128 + kColAtom);
            tma_load_2d(sm.a[stage], &tmR, &sm.full[stage], a * 64, (rb0 + job_rb) * 128);
            tma_load_2d(sm.b[stage], &tmC, &sm.full[stage], a * 64, job_ct * BN);
          }
          __syncwarp();
          last_ph[stage] = (int)ph;
          if (++stage == kClStages) { stage = 0; ph ^= 1; }
        }
      }
      volatile int never = 0;
      for (int s = 0; s < kClStages; ++s)
        if (last_ph[s] >= 0) wait(&sm.full[s], (uint32_t)last_ph[s], &never, dev_err);
    }
  } else if (warp == 6) {
    // Producer of the output-update operands: C[s, slice] and Gs(s).
    {  // whole warp: uniform loop state; elected lane issues
      uint32_t cs_ph[2] = {0, 0}, ge_ph[kGSlots] = {};
      int cs_last[2] = {-1, -1}, g_last[kGSlots];
      for (int i = 0; i < kGSlots; ++i) g_last[i] = -1;
      bool ok = true;
      TileCursor cur;
      cur.init(mp, 0);
      // Output operand C[s, slice], column part p (atoms [j0, j0 + na)).
      auto load_cs = [&](int p, int j0, int na, int ct) {
        if (!(ok = wait(&sm.cs_empty[p], cs_ph[p] ^ 1, abort, dev_err))) return;
        if (elect_one()) {
          mbar_expect_tx(&sm.cs_full[p], (uint32_t)na * kColAtom);
          for (int j = j0; j < j0 + na; ++j)
            tma_load_2d(sm.cs[j], &tmC, &sm.cs_full[p], k * w + j * 64, ct * BN);
        }
        __syncwarp();
        cs_last[p] = (int)cs_ph[p];
        cs_ph[p] ^= 1;
      };
      // K-split: part p = Gs atom p and rows [64p, 64p + 64) of every slice
      // atom, on one barrier.
      auto load_khalf = [&](int p, int s, int rb, int ct) {
        if (!(ok = wait(&sm.cs_empty[p], cs_ph[p] ^ 1, abort, dev_err))) return;
        if (p == 0) {
          // pub[o][b] completes once per two tiles of owner o: parity (m >> 1) & 1.
          if (!(ok = wait_cluster(&sm.pub[s & (kCl - 1)][(s >> 3) & 1], (uint32_t)((s >> 4) & 1),
                                  abort, dev_err)))
            return;
          fence_proxy_async_global();
        }
        if (elect_one()) {
          mbar_expect_tx(&sm.cs_full[p], kAtom128 + (uint32_t)A * (kColAtom / 2));
          bulk_load(sm.g[0][p], gs_tile(s, rb, ct) + p * kAtom128, kAtom128, &sm.cs_full[p]);
          for (int j = 0; j < A; ++j)
            tma_load_2d(sm.cs[j] + p * (kColAtom / 2), &tmC64, &sm.cs_full[p], k * w + j * 64,
                        ct * BN + 64 * p);
        }
        __syncwarp();
        cs_last[p] = (int)cs_ph[p];
        cs_ph[p] ^= 1;
      };
      for (int s = 0; s < N && ok && ksplit; ++s, cur.next(mp)) {
        load_khalf(0, s, cur.rb, cur.ct);
        if (!ok) break;
        load_khalf(1, s, cur.rb, cur.ct);
      }
      for (int s = 0; s < N && ok && !ksplit; ++s, cur.next(mp)) {
        load_cs(0, 0, A0, cur.ct);
        if (!ok) break;
        // Gs(s) from its owner's ring slot.
        const int gb = s & (kGSlots - 1);
        // pub[o][b] completes once per two tiles of owner o: parity (m >> 1) & 1.
        if (!(ok = wait_cluster(&sm.pub[s & (kCl - 1)][(s >> 3) & 1], (uint32_t)((s >> 4) & 1), abort,
                                dev_err)))
          break;
        fence_proxy_async_global();
        if (!(ok = wait(&sm.gs_empty[gb], ge_ph[gb] ^ 1, abort, dev_err))) break;
        if (elect_one()) {
          mbar_expect_tx(&sm.g_full[gb], kGsBytes);
          bulk_load(sm.g[gb][0], gs_tile(s, cur.rb, cur.ct), kGsBytes, &sm.g_full[gb]);
        }
        __syncwarp();
        g_last[gb] = (int)ge_ph[gb];
        ge_ph[gb] ^= 1;
        if (A1 > 0) load_cs(1, A0, A1, cur.ct);
      }
      volatile int never = 0;
      for (int p = 0; p < 2; ++p)
        if (cs_last[p] >= 0) wait(&sm.cs_full[p], (uint32_t)cs_last[p], &never, dev_err);
      for (int i = 0; i < kGSlots; ++i)
        if (g_last[i] >= 0) wait(&sm.g_full[i], (uint32_t)g_last[i], &never, dev_err);
    }
  } else if (warp == 1 || warp == 7) {
    // Two MMA issuers with independent instruction streams: warp 1 the S
    // accumulations (TMEM columns [0, 256)), warp 7 the output update
    // (columns [256, 512)). tcgen05.mma issue runs only about one instruction
    // ahead of execution, so the bookkeeping between one warp's MMAs (barrier
    // polls, loop state) would otherwise leave the tensor pipe idle; with two
    // streams the other warp's MMAs fill those gaps. Each warp's commits
    // track its own MMAs only.
    {  // whole warp: uniform loop state; elected lane issues
      // Descriptors of every buffer, built once; K steps add to the start
      // address field (16-byte units). Buffers of one kind are contiguous,
      // so buffer i adds i times its size (in 16-byte units) to the base.
      const uint64_t da0 = sdesc_sw128(smem_u32(sm.a[0]), 16, 1024);
      const uint64_t db0 = sdesc_sw128(smem_u32(sm.b[0]), 16, 1024);
      const uint64_t dg0 = sdesc_sw128(smem_u32(sm.g[0][0]), 16, 1024);
      const uint64_t dc = sdesc_sw128(smem_u32(sm.cs[0]), kColAtom, 1024);
      constexpr uint32_t kAtomU = kAtom128 >> 4, kColU = kColAtom >> 4, kGsU = kGsBytes >> 4;
      bool ok = true;
      if (warp == 1) {
        int stage = 0;
        uint32_t ph = 0, s_ph[2] = {0, 0};
        for (int s = -kClJ; s < N && ok; ++s) {
          const int gj = job_of(s);
          if (gj < 0 || gj >= N) continue;
          const int buf = (gj >> 3) & 1;
          const int a0 = (s - (gj - kClJ)) * A;
          if (a0 == 0) {
            if (!(ok = wait(&sm.s_empty[buf], s_ph[buf] ^ 1, abort, dev_err))) break;
            tc_fence_after();
          }
          const uint32_t dt = tmem + buf * BN;
          for (int a = a0; a < a0 + A; ++a) {
            if (!(ok = wait(&sm.full[stage], ph, abort, dev_err))) break;
            const uint64_t da = da0 + stage * kAtomU, db = db0 + stage * kColU;
            if (elect_one()) {
#pragma unroll
              for (int kk = 0; kk < 4; ++kk)
                mma_bf16(dt, da + 2 * kk, db + 2 * kk, Tl::kIdescS, (a | kk) != 0);
              mma_commit(&sm.empty[stage]);
              if (a + 1 == nk) mma_commit(&sm.s_full[buf]);
            }
            __syncwarp();
            if (++stage == kClStages) { stage = 0; ph ^= 1; }
          }
          if (a0 + A == nk) s_ph[buf] ^= 1;
        }
      } else {
        uint32_t o_ph = 0, cs_ph[2] = {0, 0}, g_ph[kGSlots] = {};
        const uint32_t idesc_o0 = idesc_bf16(128, 64 * A0, 0, 1);
        const uint32_t idesc_o1 = idesc_bf16(128, 64 * (A1 > 0 ? A1 : 1), 0, 1);
        const uint64_t dc1 = dc + (uint64_t)A0 * kColU;
        TileCursor cur;  // tile of slot s
        cur.init(mp, 0);
        const uint32_t idesc_w = idesc_bf16(128, 64 * A, 0, 1);
        for (int s = 0; s < N && ok && ksplit; ++s, cur.next(mp)) {
          const bool unit_start = cur.unit_start(mp);
          const bool unit_end = cur.unit_end(mp);
          if (unit_start && !(ok = wait(&sm.o_empty, o_ph ^ 1, abort, dev_err))) break;
          for (int p = 0; p < 2 && ok; ++p) {
            if (!(ok = wait(&sm.cs_full[p], cs_ph[p], abort, dev_err))) break;
            cs_ph[p] ^= 1;
            tc_fence_after();
            if (elect_one()) {
#pragma unroll
              for (int q = 0; q < 4; ++q)
                mma_bf16(tmem_o, dg0 + p * kAtomU + q * 2,
                         dc + p * (kColU / 2) + q * (2048 >> 4), idesc_w,
                         !(unit_start && p == 0 && q == 0));
              mma_commit(&sm.cs_empty[p]);
              if (p == 1) {
                // Tell the owner of s that this CTA is done with tile s (see below).
                if (s + 2 * kCl < N)
                  mma_commit_multicast(&sm.gfree[(s >> 3) & 1], (uint16_t)(1u << (s & (kCl - 1))));
                if (unit_end) mma_commit(&sm.o_full);
              }
            }
            __syncwarp();
          }
          if (ok && unit_end) o_ph ^= 1;
        }
        for (int s = 0; s < N && ok && !ksplit; ++s, cur.next(mp)) {
          const int gb = s & (kGSlots - 1);
          const bool unit_start = cur.unit_start(mp);
          const bool unit_end = cur.unit_end(mp);
          if (unit_start && !(ok = wait(&sm.o_empty, o_ph ^ 1, abort, dev_err))) break;
          if (!(ok = wait(&sm.g_full[gb], g_ph[gb], abort, dev_err))) break;
          g_ph[gb] ^= 1;
          if (!(ok = wait(&sm.cs_full[0], cs_ph[0], abort, dev_err))) break;
          cs_ph[0] ^= 1;
          tc_fence_after();
          const uint64_t dg = dg0 + gb * kGsU;
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < BN / 16; ++kk)
              mma_bf16(tmem_o, dg + (kk >> 2) * kAtomU + (kk & 3) * 2, dc + kk * (2048 >> 4),
                       idesc_o0, !(unit_start && kk == 0));
            mma_commit(&sm.cs_empty[0]);
          }
          __syncwarp();
          if (A1 > 0) {
            if (!(ok = wait(&sm.cs_full[1], cs_ph[1], abort, dev_err))) break;
            cs_ph[1] ^= 1;
            tc_fence_after();
          }
          // Tell the owner of s that this CTA is done with tile s. The owner
          // publishes tile s + 16 (same ring slot, same pub barrier) only after
          // all 8 CTAs are, so no pub phase can run ahead of a consumer still
          // waiting on an earlier one.
          const bool notify = s + 2 * kCl < N;
          if (elect_one()) {
            if (A1 > 0) {
#pragma unroll
              for (int kk = 0; kk < BN / 16; ++kk)
                mma_bf16(tmem_o + 64 * A0, dg + (kk >> 2) * kAtomU + (kk & 3) * 2,
                         dc1 + kk * (2048 >> 4), idesc_o1, !(unit_start && kk == 0));
              mma_commit(&sm.cs_empty[1]);
            }
            mma_commit(&sm.gs_empty[gb]);
            if (notify)
              mma_commit_multicast(&sm.gfree[(s >> 3) & 1], (uint16_t)(1u << (s & (kCl - 1))));
            if (unit_end) mma_commit(&sm.o_full);
          }
          __syncwarp();
          if (unit_end) o_ph ^= 1;
        }
      }
      if (elect_one()) mma_commit(&sm.mma_done);
      __syncwarp();
      volatile int never = 0;
      wait(&sm.mma_done, 0, &never, dev_err);
    }
  } else {
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    uint32_t sf_ph[2] = {0, 0}, free_ph[2] = {0, 0}, o_ph = 0;
    bool ok = true;
    TileCursor cur;  // tile of slot s (s >= 0), for unit drains
    cur.init(mp, 0);
    for (int s = -kClJ; s < N && ok; ++s) {
      const int g = s + kClLag + 1;  // tile whose S completes in slot s
      if (g >= 0 && g < N && (g & (kCl - 1)) == k) {
        const int m = g >> 3;
        const int buf = m & 1;
        TileCursor gt;
        gt.init(mp, g);
        const int rb = gt.rb, ct = gt.ct;
        float rc = 0.f, rl = 0.f;
        if (kTokenRows) {
          const int p = (rb0 + rb) * 128 + row;
          if (p < Teff) { rc = tok_c[p]; rl = lse[p] * kLog2e; }
        } else {
          epi_sync();
          const int p = ct * BN + row;
          if (row < BN) {
            sm.col_c[row] = p < Teff ? tok_c[p] : 0.f;
            sm.col_l[row] = p < Teff ? lse[p] * kLog2e : 0.f;
          }
          epi_sync();
        }
        if (!(ok = wait_sleepy(&sm.s_full[buf], sf_ph[buf], abort, dev_err))) break;
        sf_ph[buf] ^= 1;
        if (m >= 2) {
          // Every CTA has finished with this owner's tile g - 16.
          const int pb = m & 1;
          if (!(ok = wait_cluster(&sm.gfree[pb], free_ph[pb], abort, dev_err))) break;
          free_ph[pb] ^= 1;
        }
        tc_fence_after();
        uint8_t *dst_tile = gs_tile(g, rb, ct);
#pragma unroll 1
        for (int c = 0; c < BN / 32; ++c) {
          float v[32];
          tmem_ld32(tmem + lane_off + buf * BN + c * 32, v);
          uint32_t pk[16];
#pragma unroll
          for (int j = 0; j < 32; j += 2) {
            float g2[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int col = c * 32 + j + e;
              float cc, ll;
              bool live;
              if (kTokenRows) {
                cc = rc; ll = rl;
                live = (rc != 0.f) && (ct * BN + col < V);
              } else {
                cc = sm.col_c[col]; ll = sm.col_l[col];
                live = cc != 0.f;
              }
              g2[e] = live ? -cc * ex2_approx(fmaf(v[j + e], kLog2e, -ll)) : 0.f;
            }
            __nv_bfloat162 b2 = __floats2bfloat162_rn(g2[0], g2[1]);
            pk[j >> 1] = *reinterpret_cast<uint32_t *>(&b2);
          }
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const int kc = c * 32 + q * 8;
            *reinterpret_cast<uint4 *>(dst_tile + (kc >> 6) * kAtom128 +
                                       sw128_offset(row, kc & 63)) =
                make_uint4(pk[q * 4], pk[q * 4 + 1], pk[q * 4 + 2], pk[q * 4 + 3]);
          }
        }
        tc_fence_before();
        mbar_arrive(&sm.s_empty[buf]);
        // The CTA barrier orders every epilogue thread's stores before the
        // elected thread's cluster-scope release (cumulativity); readers
        // fence the async proxy after acquiring pub[].
        epi_sync();
        if (warp == 2 && lane < kCl) {
          // One lane per destination CTA, in parallel: fence, then a relaxed
          // arrive (a release pattern per lane).
          fence_acq_rel_cluster();
          mbar_arrive_cluster_relaxed(mapa(smem_u32(&sm.pub[k][m & 1]), (uint32_t)lane));
        }
      }
      if (s < 0) continue;
      const bool unit_end = cur.unit_end(mp);
      const bool tail = mp.tail(cur.g);
      const int rb = cur.rb;
      // A tail unit's slot: its row block's place among this cluster's tail units.
      const int tu = tail ? (rb - mp.rbT) - mp.t0 / mp.n_ct : 0;
      cur.next(mp);
      if (unit_end) {
        // Drain the finished unit: out[rows, k*w : (k+1)*w].
        if (!(ok = wait_sleepy(&sm.o_full, o_ph, abort, dev_err))) break;
        o_ph ^= 1;
        tc_fence_after();
        const int rid = (rb0 + rb) * 128 + row;
        const bool valid = kTokenRows ? (rid < Teff) : (rid < V);
        float *dst = nullptr;
        if (tail)
          dst = tailbuf + ((int64_t)(cid * 2 + tu) * 128 + row) * d + k * w;
        else if (valid)
          dst = out + (kTokenRows ? (int64_t)tok_idx[rid] : (int64_t)rid) * d + k * w;
#pragma unroll 1
        for (int c = 0; c < w / 32; ++c) {
          float v[32];
          tmem_ld32(tmem_o + lane_off + c * 32, v);
          if (dst) {
#pragma unroll
            for (int q = 0; q < 8; ++q)
              reinterpret_cast<float4 *>(dst + c * 32)[q] =
                  make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          }
        }
        tc_fence_before();
        mbar_arrive(&sm.o_empty);
      }
    }
    // No column tiles at all (no active token): the slice is zero.
    if (ok && n_ct == 0) {
      for (int j = 0; j < n_my; ++j) {
        const int rid = (rb0 + cid + j * ncl) * 128 + row;
        if (!kTokenRows && rid < V)
          for (int c = 0; c < w; ++c) out[(int64_t)rid * d + k * w + c] = 0.f;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no CTA leaves while a peer may still signal its barriers
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// ------------------------------------------ logit-gradient image from S
//
// Gs_tv = -c_t exp(z_tv - lse_t) in bf16 for every tile of a chunk of token
// blocks, from the chunk-relative terms the LSE pass kept (fp16 P_v =
// 2^(z_v log2 e - m) and the fp32 chunk maximum m, per 32 columns):
// Gs = -c_t 2^(m - lse_t log2 e) P_v, one exponential per 8 columns. One
// 32 KB image tile per 128 tokens x 128 vocabulary rows, two K-major
// SWIZZLE_128B atoms of 64 vocabulary columns (the layout both backward
// GEMMs read). Columns >= V, rows >= T_eff and tokens with c_t = 0 give
// exact zeros. Streaming kernel: 34 KB read and 32 KB written per tile.
__global__ void __launch_bounds__(256) g_image_kernel(int V, int rb0, int cap,
                                                      const int32_t *counters,
                                                      const float *__restrict__ tok_c,
                                                      const float *__restrict__ lse,
                                                      const __half *__restrict__ sbuf,
                                                      const float4 *__restrict__ mbuf,
                                                      uint8_t *__restrict__ gimg) {
  const int Teff = counters[0];
  const int nrb = min(max((Teff + 127) / 128 - rb0, 0), cap);
  const int n_vt = (V + 127) / 128;
  const int64_t n_tiles = (int64_t)nrb * n_vt;
  // Thread t of the block handles 8-column chunk (t & 15) of rows
  // (t >> 4) + 16 k, k < 8; all eight loads are issued before any use.
  const int ch = threadIdx.x & 15, r0 = threadIdx.x >> 4;
  for (int64_t tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
    const int b = (int)(tile / n_vt), vt = (int)(tile - (int64_t)b * n_vt);
    const __half *src = sbuf + tile * (128 * 128);
    const float4 *mt = mbuf + tile * 128;
    uint8_t *dst = gimg + tile * kGImgTileBytes;
    const int col0 = vt * 128 + ch * 8;
    uint4 h[8];
    float4 m4[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int row = r0 + 16 * k;
      h[k] = *reinterpret_cast<const uint4 *>(src + row * 128 + ch * 8);
      m4[k] = mt[row];
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const int row = r0 + 16 * k;
      const int p = (rb0 + b) * 128 + row;
      float sc = 0.f;
      if (p < Teff && col0 < V) {
        const float cc = tok_c[p];
        const int q = ch >> 2;
        const float m = q == 0 ? m4[k].x : q == 1 ? m4[k].y : q == 2 ? m4[k].z : m4[k].w;
        if (cc != 0.f) sc = -cc * ex2_approx(m - lse[p] * kLog2e);
      }
      const uint32_t hw[4] = {h[k].x, h[k].y, h[k].z, h[k].w};
      uint32_t pk[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 f = __half22float2(*reinterpret_cast<const __half2 *>(&hw[e]));
        const float g0 = col0 + 2 * e < V ? sc * f.x : 0.f;
        const float g1 = col0 + 2 * e + 1 < V ? sc * f.y : 0.f;
        __nv_bfloat162 b2 = __floats2bfloat162_rn(g0, g1);
        pk[e] = *reinterpret_cast<uint32_t *>(&b2);
      }
      *reinterpret_cast<uint4 *>(dst + (ch >> 3) * kAtom128 + sw128_offset(row, (ch & 7) * 8)) =
          make_uint4(pk[0], pk[1], pk[2], pk[3]);
    }
  }
}

// ---------------------------------------------- dH from the stored image
//
// Softmax part of dH as the plain GEMM dH[t, :] = sum_v Gs[t, v] W[v, :],
// with the image tiles as the K-major A operand (64 vocabulary rows per
// stage, one 16 KB atom, copied verbatim) and W as the MN-major B operand.
// CTA pairs (2-CTA clusters) take two token blocks of the same 256-column
// chunk of d and share its W stage by multicast (each CTA fetches two of the
// four 64-column atoms). Work unit = (token block pair, 256-column chunk);
// the fp32 accumulator (128 x 256) is double-buffered in TMEM so the drain of
// one unit overlaps the next. Each (token, column) is owned by one CTA and
// summed over all of V in one fixed order: deterministic, no atomics. An odd
// last block is computed twice (the pair's other CTA repeats it) and stored
// once.
constexpr int kDhN = 256;                              // output columns per unit
constexpr int kDhStages = 4;
constexpr uint32_t kDhABytes = kAtom128;               // 128 tokens x 64 vocabulary
constexpr uint32_t kDhBBytes = (kDhN / 64) * 64 * 128; // 4 column atoms x 64 rows
constexpr uint32_t kIdescDh = idesc_bf16(128, kDhN, 0, 1);

struct DhSmem {
  uint8_t a[kDhStages][kDhABytes];
  uint8_t b[kDhStages][kDhBBytes];
  uint64_t full[kDhStages], empty[kDhStages];
  uint64_t acc_full[2], acc_empty[2], mma_done;
  uint32_t tmem_base;
  int abort;
};

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    dh_gemm_kernel(const __grid_constant__ CUtensorMap tmW, int d, int V, int rb0, int cap,
                   const int32_t *counters, const int32_t *tok_idx, const uint8_t *gimg,
                   float *dH, int32_t *dev_err) {
  const int Teff = counters[0];
  const int nrb = min(max((Teff + 127) / 128 - rb0, 0), cap);
  if (nrb == 0) return;  // no token in this chunk
  extern __shared__ uint8_t smem_raw[];
  DhSmem &sm = *reinterpret_cast<DhSmem *>(align1k(smem_raw));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = (int)cluster_rank();
  const int pid = (int)cluster_id_x(), npairs = (int)num_clusters_x();
  const int n_vt = (V + 127) / 128;
  const int nks = 2 * n_vt;  // 64-wide vocabulary steps (image atoms)
  const int nq = d / kDhN;
  const int n_units = (nrb + 1) / 2 * nq;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kDhStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 2);  // both CTAs' MMAs done with the stage
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sm.acc_full[s], 1);
      mbar_init(&sm.acc_empty[s], 128);
    }
    mbar_init(&sm.mma_done, 1);
    sm.abort = 0;
    fence_mbar_init();
    prefetch_tmap(&tmW);
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // the peer's barriers exist before any multicast lands
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  volatile int *abort = &sm.abort;

  if (warp == 0) {
    {  // whole warp: uniform loop state; elected lane issues
      int stage = 0;
      uint32_t ph = 0;
      int last_ph[kDhStages];
      for (int s = 0; s < kDhStages; ++s) last_ph[s] = -1;
      bool ok = true;
      for (int u = pid; u < n_units && ok; u += npairs) {
        const int tp = u / nq, q = u - tp * nq;
        const int b = min(2 * tp + r, nrb - 1);
        const uint8_t *arow = gimg + (size_t)b * n_vt * kGImgTileBytes;
        for (int ks = 0; ks < nks; ++ks) {
          if (!(ok = wait_cluster(&sm.empty[stage], ph ^ 1, abort, dev_err))) break;
          if (elect_one()) {
            mbar_expect_tx(&sm.full[stage], kDhABytes + kDhBBytes);
            bulk_load(sm.a[stage], arow + (size_t)ks * kAtom128, kAtom128, &sm.full[stage]);
            tma_load_3d_mc(sm.b[stage] + r * (kDhBBytes / 2), &tmW, &sm.full[stage], 0, 64 * ks,
                           q * (kDhN / 64) + r * (kDhN / 128), (uint16_t)3);
          }
          __syncwarp();
          last_ph[stage] = (int)ph;
          if (++stage == kDhStages) { stage = 0; ph ^= 1; }
        }
      }
      for (int s = 0; s < kDhStages; ++s)
        if (last_ph[s] >= 0) {
          volatile int never = 0;
          wait(&sm.full[s], (uint32_t)last_ph[s], &never, dev_err);
        }
    }
  } else if (warp == 1) {
    {  // whole warp: uniform loop state; elected lane issues
      // A: K-major atom, 16 tokens of K = 32 bytes along the swizzled row.
      // B: 4 column atoms of 64 vocabulary rows (LBO 8 KB), row groups of 8
      // (SBO 1 KB); 16 vocabulary rows = 2 KB.
      const uint64_t da0 = sdesc_sw128(smem_u32(sm.a[0]), 16, 1024);
      const uint64_t db0 = sdesc_sw128(smem_u32(sm.b[0]), 64 * 128, 1024);
      int stage = 0, acc = 0;
      uint32_t ph = 0, acc_ph = 0;
      bool ok = true;
      for (int u = pid; u < n_units && ok; u += npairs) {
        if (!(ok = wait(&sm.acc_empty[acc], acc_ph ^ 1, abort, dev_err))) break;
        tc_fence_after();
        const uint32_t dt = tmem + acc * kDhN;
        for (int ks = 0; ks < nks; ++ks) {
          if (!(ok = wait(&sm.full[stage], ph, abort, dev_err))) break;
          const uint64_t da = da0 + (uint64_t)stage * (kDhABytes >> 4);
          const uint64_t db = db0 + (uint64_t)stage * (kDhBBytes >> 4);
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              mma_bf16(dt, da + 2 * kk, db + kk * (2048 >> 4), kIdescDh, (ks | kk) != 0);
            mma_commit_multicast(&sm.empty[stage], (uint16_t)3);
          }
          __syncwarp();
          if (++stage == kDhStages) { stage = 0; ph ^= 1; }
        }
        if (!ok) break;
        if (elect_one()) mma_commit(&sm.acc_full[acc]);
        __syncwarp();
        if (++acc == 2) { acc = 0; acc_ph ^= 1; }
      }
      if (elect_one()) mma_commit(&sm.mma_done);
      __syncwarp();
      volatile int never = 0;
      wait(&sm.mma_done, 0, &never, dev_err);
    }
  } else {
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    int acc = 0;
    uint32_t acc_ph = 0;
    bool ok = true;
    for (int u = pid; u < n_units && ok; u += npairs) {
      const int tp = u / nq, q = u - tp * nq;
      const int t = (rb0 + 2 * tp + r) * 128 + row;
      const bool valid = 2 * tp + r < nrb && t < Teff;
      float4 *dst =
          valid ? reinterpret_cast<float4 *>(dH + (int64_t)tok_idx[t] * d + q * kDhN) : nullptr;
      if (!(ok = wait_sleepy(&sm.acc_full[acc], acc_ph, abort, dev_err))) break;
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < kDhN / 32; ++c) {
        float x[32];
        tmem_ld32(tmem + lane_off + acc * kDhN + c * 32, x);
        if (valid) {
#pragma unroll
          for (int e = 0; e < 8; ++e)
            dst[c * 8 + e] = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
        }
      }
      tc_fence_before();
      mbar_arrive(&sm.acc_empty[acc]);
      if (++acc == 2) { acc = 0; acc_ph ^= 1; }
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no CTA leaves while its peer may still signal or fill it
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// ------------------------------------- dW from the stored logit gradient
//
// With 128-wide column tiles the dH pass keeps every bf16 tile Gs it forms
// (128 tokens x 128 vocabulary rows, one 32 KB image per tile in the
// K-major SWIZZLE_128B layout of its own MMA operand) for a chunk of token
// blocks. Read with the token index as K, the same bytes are the MN-major
// SWIZZLE_128B layout of Gs^T (64 vocabulary rows per 128-byte line, one
// line per token), so the softmax part of dW is the plain GEMM
//     dW[v, :] (+)= sum_t Gs[t, v] Hc[t, :]
// with no logit recomputation.
//
// CTA pairs (2-CTA clusters) share one 512-column chunk of Hc: CTA r of the
// pair fetches half of each Hc stage and multicasts it into both CTAs; each
// CTA fetches the Gs^T stage of its own 128 vocabulary rows. Work unit =
// (vocabulary block pair, 512-column chunk of d); CTA r accumulates
// dW[block 2 p + r, chunk] (128 x 512 fp32 = all of TMEM) over the chunk's
// tokens, 32 token rows per stage, and drains it with plain stores (first
// chunk) or read-add-writes (later chunks; this CTA owns those rows).
// An odd last block is computed twice (the pair's other CTA repeats the
// last block) so both CTAs run the same stage sequence; only one stores it.
constexpr int kDwKS = 32;                                 // token rows per stage
constexpr int kDwStages = 5;
constexpr int kDwN = 512;                                 // output columns per CTA
constexpr uint32_t kDwGBytes = 2 * kDwKS * 128;           // 2 vocabulary atoms x 32 rows
constexpr uint32_t kDwHBytes = (kDwN / 64) * kDwKS * 128; // 8 column atoms x 32 rows
constexpr uint32_t kIdescDw = idesc_bf16(128, 256, 1, 1); // both operands MN-major

struct DwSmem {
  uint8_t g[kDwStages][kDwGBytes];  // Gs^T: MN-major A, atoms 4 KB apart
  uint8_t h[kDwStages][kDwHBytes];  // Hc[t, chunk]: MN-major B, atoms 4 KB apart
  uint64_t full[kDwStages], empty[kDwStages];
  uint64_t acc_full, acc_empty, mma_done;
  uint32_t tmem_base;
  int abort;
};

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    dw_gemm_kernel(const __grid_constant__ CUtensorMap tmG,
                   const __grid_constant__ CUtensorMap tmH, int d, int V, int rb0, int cap,
                   int accumulate, const int32_t *counters, float *dW, int32_t *dev_err) {
  const int Teff = counters[0];
  const int nrb = min(max((Teff + 127) / 128 - rb0, 0), cap);
  // A chunk past the last token adds nothing (the first chunk always runs:
  // with no tokens at all it writes the zero softmax part).
  if (nrb == 0 && accumulate) return;
  extern __shared__ uint8_t smem_raw[];
  DwSmem &sm = *reinterpret_cast<DwSmem *>(align1k(smem_raw));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = (int)cluster_rank();
  const int pid = (int)cluster_id_x(), npairs = (int)num_clusters_x();
  const int n_vb = (V + 127) / 128;
  const int nq = d / kDwN;
  const int n_units = (n_vb + 1) / 2 * nq;
  const int nks = nrb * (128 / kDwKS);

  if (threadIdx.x == 0) {
    for (int s = 0; s < kDwStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 2);  // both CTAs' MMAs done with the stage
    }
    mbar_init(&sm.acc_full, 1);
    mbar_init(&sm.acc_empty, 128);
    mbar_init(&sm.mma_done, 1);
    sm.abort = 0;
    fence_mbar_init();
    prefetch_tmap(&tmG);
    prefetch_tmap(&tmH);
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // the peer's barriers exist before any multicast lands
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  volatile int *abort = &sm.abort;

  if (warp == 0) {
    {  // whole warp: uniform loop state; elected lane issues
      int stage = 0;
      uint32_t ph = 0;
      int last_ph[kDwStages];
      for (int s = 0; s < kDwStages; ++s) last_ph[s] = -1;
      bool ok = true;
      for (int u = pid; u < n_units && ok; u += npairs) {
        const int vp = u / nq, q = u - vp * nq;
        const int vb = min(2 * vp + r, n_vb - 1);
        for (int ks = 0; ks < nks; ++ks) {
          const int rbl = ks >> 2, j = ks & 3;
          if (!(ok = wait_cluster(&sm.empty[stage], ph ^ 1, abort, dev_err))) break;
          if (elect_one()) {
            mbar_expect_tx(&sm.full[stage], kDwGBytes + kDwHBytes);
            tma_load_3d(sm.g[stage], &tmG, &sm.full[stage], 0, kDwKS * j,
                        2 * (rbl * n_vb + vb));
            tma_load_3d_mc(sm.h[stage] + r * (kDwHBytes / 2), &tmH, &sm.full[stage], 0,
                           (rb0 + rbl) * 128 + kDwKS * j, q * (kDwN / 64) + r * (kDwN / 128),
                           (uint16_t)3);
          }
          __syncwarp();
          last_ph[stage] = (int)ph;
          if (++stage == kDwStages) { stage = 0; ph ^= 1; }
        }
      }
      // Never leave a copy in flight: wait (bounded) for the last one issued
      // on every stage.
      for (int s = 0; s < kDwStages; ++s)
        if (last_ph[s] >= 0) {
          volatile int never = 0;
          wait(&sm.full[s], (uint32_t)last_ph[s], &never, dev_err);
        }
    }
  } else if (warp == 1) {
    {  // whole warp: uniform loop state; elected lane issues
      // A: 2 vocabulary atoms (LBO 4 KB), token groups of 8 rows (SBO 1 KB);
      // B: 8 column atoms (LBO 4 KB), the same token groups. One K step of 16
      // tokens advances both by 2 KB; B's second 256-column half is 16 KB on.
      const uint64_t dg0 = sdesc_sw128(smem_u32(sm.g[0]), kDwKS * 128, 1024);
      const uint64_t dh0 = sdesc_sw128(smem_u32(sm.h[0]), kDwKS * 128, 1024);
      int stage = 0;
      uint32_t ph = 0, acc_ph = 0;
      bool ok = true;
      for (int u = pid; u < n_units && ok && nks > 0; u += npairs) {
        if (!(ok = wait(&sm.acc_empty, acc_ph ^ 1, abort, dev_err))) break;
        acc_ph ^= 1;
        tc_fence_after();
        for (int ks = 0; ks < nks; ++ks) {
          if (!(ok = wait(&sm.full[stage], ph, abort, dev_err))) break;
          const uint64_t dg = dg0 + (uint64_t)stage * (kDwGBytes >> 4);
          const uint64_t dh = dh0 + (uint64_t)stage * (kDwHBytes >> 4);
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < kDwKS / 16; ++kk)
#pragma unroll
              for (int nh = 0; nh < 2; ++nh)
                mma_bf16(tmem + nh * 256, dg + kk * (2048 >> 4),
                         dh + nh * ((kDwHBytes / 2) >> 4) + kk * (2048 >> 4), kIdescDw,
                         (ks | kk) != 0);
            mma_commit_multicast(&sm.empty[stage], (uint16_t)3);
          }
          __syncwarp();
          if (++stage == kDwStages) { stage = 0; ph ^= 1; }
        }
        if (!ok) break;
        if (elect_one()) mma_commit(&sm.acc_full);
        __syncwarp();
      }
      if (elect_one()) mma_commit(&sm.mma_done);
      __syncwarp();
      volatile int never = 0;
      wait(&sm.mma_done, 0, &never, dev_err);
    }
  } else {
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    uint32_t acc_ph = 0;
    bool ok = true;
    for (int u = pid; u < n_units && ok; u += npairs) {
      const int vp = u / nq, q = u - vp * nq;
      const int v = (2 * vp + r) * 128 + row;
      const bool valid = 2 * vp + r < n_vb && v < V;
      float4 *dst = valid ? reinterpret_cast<float4 *>(dW + (int64_t)v * d + q * kDwN) : nullptr;
      if (nks == 0) {
        if (valid)
          for (int c = 0; c < kDwN / 4; ++c) dst[c] = make_float4(0.f, 0.f, 0.f, 0.f);
        continue;
      }
      if (!(ok = wait_sleepy(&sm.acc_full, acc_ph, abort, dev_err))) break;
      acc_ph ^= 1;
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < kDwN / 32; ++c) {
        float x[32];
        tmem_ld32(tmem + lane_off + c * 32, x);
        if (valid) {
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            float4 o = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
            if (accumulate) {
              const float4 p = dst[c * 8 + e];
              o.x += p.x; o.y += p.y; o.z += p.z; o.w += p.w;
            }
            dst[c * 8 + e] = o;
          }
        }
      }
      tc_fence_before();
      mbar_arrive(&sm.acc_empty);
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no CTA leaves while its peer may still signal or fill it
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// --------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D bf16 row-major [rows][cols] map with 64 x box_rows SWIZZLE_128B boxes.
bool make_map(CUtensorMap *m, const void *ptr, int64_t rows, int64_t cols,
              int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr),
            dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D bf16 map: dims (innermost first) with byte strides of dims 1 and 2,
// box `box`, swizzle `sw`.
bool make_map3(CUtensorMap *m, const void *ptr, const cuuint64_t (&dims)[3],
               const cuuint64_t (&strides)[2], const cuuint32_t (&box)[3],
               CUtensorMapSwizzle sw) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t d[3] = {dims[0], dims[1], dims[2]};
  cuuint64_t st[2] = {strides[0], strides[1]};
  cuuint32_t b[3] = {box[0], box[1], box[2]};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(ptr), d, st, b, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// fp16 [rows][128] map with 64-column x 32-row SWIZZLE_128B boxes (the
// kept chunk-relative terms, stored by the LSE pass one warp's rows at a
// time).
bool make_map_s(CUtensorMap *m, const void *ptr, int64_t rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {128, (cuuint64_t)rows};
  cuuint64_t strides[1] = {128 * 2};
  cuuint32_t box[2] = {64, 32};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void *>(ptr), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int num_sms();

// CTAs of the LSE grid: every 2-CTA cluster that fits at once (persistent).
int lse_grid(size_t smem) {
  static int cached = 0;
  if (cached) return cached;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kLsePair * 64, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, (const void *)lse_kernel, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    n = num_sms() / kLsePair;
  }
  cached = kLsePair * (n > 0 ? n : 1);
  return cached;
}

int num_sms() {
  static int n = 0;
  if (!n) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

// CTAs of a persistent grid of 2-CTA clusters: every pair that fits at once
// (from the occupancy API; cached per kernel in *cache).
int pair_grid(const void *kernel, size_t smem, int *cache) {
  if (*cache) return *cache;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * 64, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    n = num_sms() / 2;
  }
  *cache = 2 * (n > 0 ? n : 1);
  return *cache;
}

// The cluster backward needs d = 8 * 64 * A with 1 <= A <= 6: each CTA's
// output slice of 64 * A columns stays in TMEM beside two S buffers of the
// column-tile width BN (2 BN + 64 A <= 512).
bool use_cluster_path(int d) { return grad_cluster_path(d); }
int cluster_tile_width(int d) { return d <= 2048 ? 128 : d <= 2560 ? 96 : 64; }

// Clusters that fit at once (persistent grid), from the occupancy API.
template <int BN>
int cluster_grid(const void *kernel, size_t smem) {
  static int cached = 0;
  if (cached) return cached;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kCl * 64, 1, 1);
  cfg.blockDim = dim3(kClThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    n = num_sms() / kCl;
  }
  if (n > kMaxClusters) n = kMaxClusters;
  cached = n > 0 ? n : 1;
  return cached;
}

// dH and dW by the cluster kernels with BN-wide column tiles. Row operands
// use 128-row boxes (mH for dH, mW128 for dW); column operands BN-row boxes.
template <int BN>
pair_status grad_bwd_cluster(const GradArgs &g, const GradWorkspace &w, cudaStream_t s,
                             const CUtensorMap &mH, const CUtensorMap &mW128) {
  CUtensorMap mHc, mWc, mHc64, mWc64;
  if (!make_map(&mHc, w.Hc, w.Tpad, g.d, BN) || !make_map(&mWc, g.W, g.V, g.d, BN) ||
      !make_map(&mHc64, w.Hc, w.Tpad, g.d, 64) || !make_map(&mWc64, g.W, g.V, g.d, 64))
    return PAIR_ERR_CUDA;
  const int nsm = num_sms();
  const size_t cl_smem = sizeof(ClSmem<BN>) + 1024;
  PAIR_CUDA_TRY(cudaFuncSetAttribute(bwd_cluster_kernel<true, BN>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)cl_smem));
  PAIR_CUDA_TRY(cudaFuncSetAttribute(bwd_cluster_kernel<false, BN>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)cl_smem));
  const int ncl = cluster_grid<BN>((const void *)bwd_cluster_kernel<true, BN>, cl_smem);
  uint8_t *gring = static_cast<uint8_t *>(w.gring);
  constexpr int kAll = 0x7fffffff;
  PAIR_BEGIN("bwd_dh_tc", s);
  bwd_cluster_kernel<true, BN><<<ncl * kCl, kClThreads, cl_smem, s>>>(
      mH, mWc, mWc64, g.d, g.V, w.counters, w.tok_idx, w.tok_c, w.lse, g.dH, gring, nullptr,
      w.tailbuf, 0, kAll, g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("tail_dh", s);
  tail_reduce_kernel<true, BN><<<nsm, 256, 0, s>>>(g.d, g.V, ncl, 0, kAll, w.counters,
                                                   w.tok_idx, w.tailbuf, g.dH);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("bwd_dw_tc", s);
  bwd_cluster_kernel<false, BN><<<ncl * kCl, kClThreads, cl_smem, s>>>(
      mW128, mHc, mHc64, g.d, g.V, w.counters, w.tok_idx, w.tok_c, w.lse, g.dW, gring, nullptr,
      w.tailbuf, 0, kAll, g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("tail_dw", s);
  tail_reduce_kernel<false, BN><<<nsm, 256, 0, s>>>(g.d, g.V, ncl, 0, kAll, w.counters,
                                                    w.tok_idx, w.tailbuf, g.dW);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

constexpr int kAllBlocks = 0x7fffffff;

// Log-sum-exp pass over token blocks [rb0, rb0 + cap) (clipped to the active
// ones), then lse for those tokens. With keep, the chunk-relative logit terms
// of the first s_blocks of those blocks are kept in w.sbuf / w.mbuf.
pair_status launch_lse(const GradArgs &g, const GradWorkspace &w, cudaStream_t s, int rb0,
                       int cap, bool keep, int s_blocks) {
  void *sbuf = keep ? w.sbuf : nullptr;
  CUtensorMap mH, mW128, mS = {};
  if (!make_map(&mH, w.Hc, w.Tpad, g.d, 128) || !make_map(&mW128, g.W, g.V, g.d, 128))
    return PAIR_ERR_CUDA;
  if (sbuf && !make_map_s(&mS, sbuf, (int64_t)w.gimg_rb * ((g.V + 127) / 128) * 128))
    return PAIR_ERR_CUDA;
  const int nsm = num_sms();
  const size_t lse_smem = sizeof(LseSmem) + 1024;
  PAIR_CUDA_TRY(cudaFuncSetAttribute(lse_kernel,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)lse_smem));
  PAIR_BEGIN("lse_tc", s);
  lse_kernel<<<lse_grid(lse_smem), kThreads, lse_smem, s>>>(
      mH, mW128, mS, g.d, g.V, w.nsplit, w.Tpad, w.counters, w.tok_y, w.part, w.zy, rb0, cap, sbuf,
      keep ? w.mbuf : nullptr, s_blocks, g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("lse_combine", s);
  lse_combine_kernel<<<nsm * 4, 256, 0, s>>>(w.nsplit, w.Tpad, w.counters, w.part, w.lse, rb0,
                                             cap);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

// The backward through the logit-gradient image runs whenever the workspace
// holds one: token blocks in chunks of w.gimg_rb, and for each chunk
//   g_image   Gs (bf16 tiles) from the kept fp32 logits, lse and c_t,
//   dh_gemm   dH rows of the chunk = Gs . W,
//   dw_gemm   dW (+)= Gs^T . Hc (the first chunk stores, later ones add).
// The number of chunks follows from T, so the launch sequence needs no
// device-to-host read; chunks past the last active token exit at once.
bool image_path(const GradWorkspace &w) { return w.gimg && w.sbuf && w.gimg_rb > 0; }

int64_t image_chunks(const GradArgs &g, const GradWorkspace &w) {
  return ((g.T + 127) / 128 + w.gimg_rb - 1) / w.gimg_rb;
}

pair_status launch_chunk_bwd(const GradArgs &g, const GradWorkspace &w, cudaStream_t s,
                             int64_t c) {
  const int cap = w.gimg_rb;
  const int rb0 = (int)(c * cap);
  const int n_vt = (g.V + 127) / 128;
  CUtensorMap mG, mH3, mW3;
  if (!make_map3(&mG, w.gimg, {64, 128, (cuuint64_t)2 * cap * n_vt}, {128, 16384}, {64, 32, 2},
                 CU_TENSOR_MAP_SWIZZLE_NONE) ||
      !make_map3(&mH3, w.Hc, {64, (cuuint64_t)w.Tpad, (cuuint64_t)g.d / 64},
                 {(cuuint64_t)g.d * 2, 128}, {64, (cuuint32_t)kDwKS, 4},
                 CU_TENSOR_MAP_SWIZZLE_128B) ||
      !make_map3(&mW3, g.W, {64, (cuuint64_t)g.V, (cuuint64_t)g.d / 64},
                 {(cuuint64_t)g.d * 2, 128}, {64, 64, 2}, CU_TENSOR_MAP_SWIZZLE_128B))
    return PAIR_ERR_CUDA;
  const size_t dh_smem = sizeof(DhSmem) + 1024, dw_smem = sizeof(DwSmem) + 1024;
  PAIR_CUDA_TRY(cudaFuncSetAttribute(dh_gemm_kernel,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dh_smem));
  PAIR_CUDA_TRY(cudaFuncSetAttribute(dw_gemm_kernel,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dw_smem));
  static int dh_cache = 0, dw_cache = 0;
  uint8_t *gimg = static_cast<uint8_t *>(w.gimg);
  PAIR_BEGIN("g_image", s);
  g_image_kernel<<<num_sms() * 3, 256, 0, s>>>(g.V, rb0, cap, w.counters, w.tok_c, w.lse,
                                               static_cast<const __half *>(w.sbuf), w.mbuf, gimg);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("dh_gemm_tc", s);
  dh_gemm_kernel<<<pair_grid((const void *)dh_gemm_kernel, dh_smem, &dh_cache), kThreads,
                   dh_smem, s>>>(mW3, g.d, g.V, rb0, cap, w.counters, w.tok_idx, gimg, g.dH,
                                 g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("dw_gemm_tc", s);
  dw_gemm_kernel<<<pair_grid((const void *)dw_gemm_kernel, dw_smem, &dw_cache), kThreads,
                   dw_smem, s>>>(mG, mH3, g.d, g.V, rb0, cap, c > 0 ? 1 : 0, w.counters, g.dW,
                                 g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

}  // namespace

// Forward half: per-token log-sum-exp and target logit over every active
// token (with an image, the first chunk's logits are kept for the backward).
pair_status grad_lse_tc(const GradArgs &g, const GradWorkspace &w, cudaStream_t s) {
  if (image_path(w)) return launch_lse(g, w, s, 0, kAllBlocks, true, w.gimg_rb);
  return launch_lse(g, w, s, 0, kAllBlocks, false, 0);
}

// Backward half: softmax parts of dH and dW from the token coefficients,
// after grad_lse_tc (chunks after the first recompute their logits).
pair_status grad_bwd_tc(const GradArgs &g, const GradWorkspace &w, cudaStream_t s) {
  if (image_path(w)) {
    const int64_t nc = image_chunks(g, w);
    for (int64_t c = 0; c < nc; ++c) {
      if (c > 0) {
        const pair_status st = launch_lse(g, w, s, (int)(c * w.gimg_rb), w.gimg_rb, true,
                                          w.gimg_rb);
        if (st != PAIR_OK) return st;
      }
      const pair_status st = launch_chunk_bwd(g, w, s, c);
      if (st != PAIR_OK) return st;
    }
    return PAIR_OK;
  }
  CUtensorMap mH, mW128;
  if (!make_map(&mH, w.Hc, w.Tpad, g.d, 128) || !make_map(&mW128, g.W, g.V, g.d, 128))
    return PAIR_ERR_CUDA;
  if (use_cluster_path(g.d)) {
    switch (cluster_tile_width(g.d)) {
      case 128: return grad_bwd_cluster<128>(g, w, s, mH, mW128);
      case 96: return grad_bwd_cluster<96>(g, w, s, mH, mW128);
      default: return grad_bwd_cluster<64>(g, w, s, mH, mW128);
    }
  }
  const int nsm = num_sms();
  const size_t bwd_smem = sizeof(BwdSmem) + 1024;
  PAIR_CUDA_TRY(cudaFuncSetAttribute(bwd_kernel<true>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bwd_smem));
  PAIR_CUDA_TRY(cudaFuncSetAttribute(bwd_kernel<false>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bwd_smem));
  PAIR_BEGIN("bwd_dh_tc", s);
  bwd_kernel<true><<<nsm, kThreads, bwd_smem, s>>>(
      mH, mW128, g.d, g.V, w.counters, w.tok_idx, w.tok_c, w.lse, g.dH, g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("bwd_dw_tc", s);
  bwd_kernel<false><<<nsm, kThreads, bwd_smem, s>>>(
      mW128, mH, g.d, g.V, w.counters, w.tok_idx, w.tok_c, w.lse, g.dW, g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

// Memory the backward may use for kept logit terms (fp16 terms and fp32
// chunk maxima) and bf16 logit-gradient tiles, 66 KB per 128 x 128 tile;
// larger problems run in token chunks.
constexpr int64_t kImageBudget = int64_t(24) << 30;
constexpr size_t kImageTileBytes = kGImgTileBytes + 128 * 128 * 2 + 128 * 16;

int grad_gimg_rows(int64_t T, int32_t d, int32_t V, pair_dtype dt) {
  if (dt != PAIR_BF16 || d < 512 || d % kDwN != 0) return 0;
  const int64_t n_rb = (T + 127) / 128;
  const int64_t per_rb = (int64_t)((V + 127) / 128) * (int64_t)kImageTileBytes;
  int64_t cap = kImageBudget / per_rb;
  if (cap < 32) cap = 32;
  return (int)(n_rb < cap ? n_rb : cap);
}

size_t grad_image_block_bytes(int32_t V) {
  return (size_t)((V + 127) / 128) * kImageTileBytes;
}

// Whole head: with an image, each chunk's log-sum-exp pass keeps its logits
// for that chunk's backward (no recomputation); otherwise forward, then the
// recomputing backward.
pair_status grad_head_tc(const GradArgs &g, const GradWorkspace &w, cudaStream_t s) {
  if (image_path(w)) {
    const int64_t nc = image_chunks(g, w);
    for (int64_t c = 0; c < nc; ++c) {
      pair_status st = launch_lse(g, w, s, (int)(c * w.gimg_rb), w.gimg_rb, true, w.gimg_rb);
      if (st == PAIR_OK) st = launch_chunk_bwd(g, w, s, c);
      if (st != PAIR_OK) return st;
    }
    return PAIR_OK;
  }
  const pair_status st = grad_lse_tc(g, w, s);
  return st != PAIR_OK ? st : grad_bwd_tc(g, w, s);
}

}  // namespace pairk
