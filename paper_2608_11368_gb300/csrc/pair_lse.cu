// Log-sum-exp pass of the bf16 LM-head path (Sec. 4.5 forward): per active
// token the log-sum-exp of its logits z = W h and its target logit, on the
// 5th-generation tensor cores. With a workspace that keeps them, the softmax
// terms of a chunk of token blocks, relative to each token's target logit,
// are stored for the backward as the bf16 image the dH and dW GEMMs read.
#include "tc_kernels.cuh"

namespace pairk {
namespace {

using namespace tc;
using namespace tck;

// ------------------------------------------------------------------ LSE
constexpr int kLseBN = 256;     // vocabulary rows per tile (N of the pair MMA)
constexpr int kLseStages = 5;
constexpr int kLsePair = 2;     // CTAs per cluster: one M = 256 MMA per K step
// Bytes that complete one stage, counted on the even CTA's barrier: each CTA
// lands its token atom and its 128 vocabulary rows.
constexpr uint32_t kLseStageTx = kLsePair * 2 * kAtom128;
constexpr uint32_t kIdescLse = idesc_bf16(256, kLseBN, 0, 0);

struct LseSmem {
  uint8_t a[kLseStages][kAtom128];  // this CTA's token block, one K-atom (128 x 64)
  uint8_t b[kLseStages][kAtom128];  // this CTA's half of the vocabulary tile (128 x 64)
  uint8_t stg[2][128 * 128];  // kept-term staging: per warp 32 rows x 64 fp16, SWIZZLE_128B
  uint64_t full[kLseStages], empty[kLseStages];
  uint64_t acc_full[2], acc_empty[2];
  uint64_t mma_done;
  uint32_t tmem_base;
  int abort;
};

// Work unit u -> (pair of token blocks, vocabulary split). Units come in
// groups of kLseSplitGroup splits: every pair over the group's splits (split
// fastest), then the next group. The CTAs running at once then share the W
// rows of two splits (78 MB for the 152k vocabulary) and their token blocks
// in L2, instead of streaming all of W from DRAM once per few pairs as a
// split-fastest order over all splits does.
constexpr int kLseSplitGroup = 2;
__device__ __forceinline__ void lse_unit(int u, int n_pairs, int nsplit, int &pair, int &sp) {
  const int sg = (nsplit % kLseSplitGroup == 0) ? kLseSplitGroup : 1;
  const int gsize = n_pairs * sg;
  const int gi = u / gsize, w = u - gi * gsize;
  pair = w / sg;
  sp = gi * sg + (w - pair * sg);
}

// CTA pairs (2-CTA clusters) work on two token blocks of the same vocabulary
// split in lockstep, as one M = 256 tile: the even CTA issues every MMA of
// the pair (cta_group::2), over the 256 token rows of both CTAs' A stages and
// the 256 vocabulary rows of their B stages (128 in each CTA), and each CTA's
// TMEM receives the logits of its own token block. Each CTA fetches only its
// own token atom and its own half of the vocabulary atom, so a stage is 32 KB
// per CTA; the even CTA's full barrier counts both CTAs' bytes, and the MMA's
// commits release the stage and publish the accumulator in both CTAs. The
// odd CTA's epilogue returns each accumulator buffer to the even CTA's
// acc_empty barrier. Five stages: a sixth fits beside the staging buffers but
// measured slower over the whole step (deeper pipelines let the pairs drift
// apart in the vocabulary, so fewer of them share W rows in L2), four starve
// the MMA.
template <bool kImage>
__global__ void __cluster_dims__(kLsePair, 1, 1) __launch_bounds__(kThreads, 1)
    lse_kernel(const __grid_constant__ CUtensorMap tmH,
               const __grid_constant__ CUtensorMap tmW, int d, int V,
               int nsplit, int64_t Tpad, const int32_t *counters,
               const int32_t *tok_y, const float *ref, float2 *part, float *zy, int rb0,
               int cap, uint8_t *gimg, int s_blocks, int fix, int32_t *dev_err) {
  // The fix-up launch redoes the pass only if the first one flagged a row
  // (the same value for every CTA: uniform exit before any cluster step).
  if (kImage && fix && counters[2] == 0) return;
  extern __shared__ uint8_t smem_raw[];
  LseSmem &sm = *reinterpret_cast<LseSmem *>(align1k(smem_raw));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Teff = counters[0];
  // Token blocks [rb0, rb0 + n_tb) of this launch. Per split, part holds
  // (maximum, sum of terms) of each token's logits z (log2 units). Without
  // kImage the terms are relative to the running maximum. With kImage they
  // are P_v = 2^(z_v log2 e - R_t) for the token's reference R_t (ref), and
  // the bf16 P of the first s_blocks blocks form the image: 128 x 128 tiles,
  // tile (b, vt) at (b * n_vt128 + vt) * 32 KB of gimg as two K-major
  // SWIZZLE_128B atoms of 64 columns (each epilogue warp stages 32 rows x 64
  // columns in that layout and writes the 4 KB with one bulk copy). Columns
  // in [V, 128 n_vt128) and rows past T_eff are exact zeros.
  const int n_tb = min(max((Teff + 127) / 128 - rb0, 0), cap);
  const int n_vt128 = (V + 127) / 128;
  const int s_lim = min(n_tb, s_blocks);
  const int n_vt = (V + kLseBN - 1) / kLseBN;
  // Work unit = (pair of token blocks, vocabulary split); CTA r of the pair
  // takes token block 2 * pair + r (past the last block for an odd count:
  // in-bounds padding rows whose results are never written).
  // Units (pair of token blocks, vocabulary split) in groups of splits (see
  // lse_unit). (A split-major order, where every pair running at once reads
  // the same split, measured 4 % slower.)
  const int n_pairs = (n_tb + 1) / 2;
  const int n_units = n_pairs * nsplit;
  const int nk = d / 64;
  const int r = (int)cluster_rank();
  const int pid = (int)cluster_id_x(), npairs = (int)num_clusters_x();

  if (threadIdx.x == 0) {
    for (int s = 0; s < kLseStages; ++s) {
      mbar_init(&sm.full[s], 1);   // the even CTA's expect_tx (both CTAs' bytes)
      mbar_init(&sm.empty[s], 1);  // the pair MMA's commit
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sm.acc_full[s], 1);
      mbar_init(&sm.acc_empty[s], kLsePair * 128);  // both CTAs' epilogue threads
    }
    mbar_init(&sm.mma_done, 1);
    sm.abort = 0;
    fence_mbar_init();
    prefetch_tmap(&tmH);
    prefetch_tmap(&tmW);
  }
  if (warp == 1) {
    tmem_alloc_pair(&sm.tmem_base, 512);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // the pair's barriers exist before any copy or commit lands
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
        int pr, sp;
        lse_unit(u, n_pairs, nsplit, pr, sp);
        const int tb = rb0 + 2 * pr + r;
        const int vt0 = (int)((int64_t)sp * n_vt / nsplit);
        const int vt1 = (int)((int64_t)(sp + 1) * n_vt / nsplit);
        for (int vt = vt0; vt < vt1 && ok; ++vt) {
          for (int k = 0; k < nk; ++k) {
            if (!(ok = wait_cluster(&sm.empty[stage], ph ^ 1, abort, dev_err))) break;
            if (elect_one()) {
              if (r == 0) mbar_expect_tx(&sm.full[stage], kLseStageTx);
              const uint32_t fb = mapa(smem_u32(&sm.full[stage]), 0);
              tma_load_2d_pair(sm.a[stage], &tmH, fb, k * 64, tb * 128);
              tma_load_2d_pair(sm.b[stage], &tmW, fb, k * 64, vt * kLseBN + r * (kLseBN / 2));
            }
            __syncwarp();
            last_ph[stage] = (int)ph;
            if (++stage == kLseStages) { stage = 0; ph ^= 1; }
          }
        }
      }
      // Never leave a copy in flight: wait (bounded) for the last one issued
      // on every stage: its completion on the even CTA, its consumption by
      // the pair MMA on the odd one (both CTAs issue the same sequence).
      for (int s = 0; s < kLseStages; ++s)
        if (last_ph[s] >= 0) {
          volatile int never = 0;
          if (r == 0)
            wait_cluster(&sm.full[s], (uint32_t)last_ph[s], &never, dev_err);
          else
            wait_cluster(&sm.empty[s], (uint32_t)last_ph[s], &never, dev_err);
        }
    }
  } else if (warp == 1) {
    if (r == 0) {  // whole warp: uniform loop state; elected lane issues
      int stage = 0, acc = 0;
      uint32_t ph = 0, acc_ph = 0;
      const uint64_t da0 = sdesc_sw128(smem_u32(sm.a[0]), 16, 1024);
      const uint64_t db0 = sdesc_sw128(smem_u32(sm.b[0]), 16, 1024);
      bool ok = true;
      for (int u = pid; u < n_units && ok; u += npairs) {
        int pr, sp;
        lse_unit(u, n_pairs, nsplit, pr, sp);
        const int vt0 = (int)((int64_t)sp * n_vt / nsplit);
        const int vt1 = (int)((int64_t)(sp + 1) * n_vt / nsplit);
        for (int vt = vt0; vt < vt1 && ok; ++vt) {
          if (!(ok = wait_cluster(&sm.acc_empty[acc], acc_ph ^ 1, abort, dev_err))) break;
          tc_fence_after();
          const uint32_t dt = tmem + acc * kLseBN;
          for (int k = 0; k < nk; ++k) {
            if (!(ok = wait_cluster(&sm.full[stage], ph, abort, dev_err))) break;
            tc_fence_after();
            const uint64_t da = da0 + (uint64_t)stage * (kAtom128 >> 4);
            const uint64_t db = db0 + (uint64_t)stage * (kAtom128 >> 4);
            if (elect_one()) {
#pragma unroll
              for (int kk = 0; kk < 4; ++kk)
                mma_bf16_pair(dt, da + 2 * kk, db + 2 * kk, kIdescLse, (k | kk) != 0);
              mma_commit_pair(&sm.empty[stage], (uint16_t)3);
            }
            __syncwarp();
            if (++stage == kLseStages) { stage = 0; ph ^= 1; }
          }
          if (!ok) break;
          if (elect_one()) mma_commit_pair(&sm.acc_full[acc], (uint16_t)3);
          __syncwarp();
          if (++acc == 2) { acc = 0; acc_ph ^= 1; }
        }
      }
      if (elect_one()) mma_commit_pair(&sm.mma_done, (uint16_t)1);
      __syncwarp();
      volatile int never = 0;
      wait(&sm.mma_done, 0, &never, dev_err);
    }
  } else {
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_addr = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    const int img_cols = n_vt128 * 128;  // image columns: V rounded up to a tile
    int acc = 0, sbuf_i = 0;
    uint32_t acc_ph = 0;
    bool ok = true;
    for (int u = pid; u < n_units && ok; u += npairs) {
      int pr, sp;
      lse_unit(u, n_pairs, nsplit, pr, sp);
      const int tbl = 2 * pr + r;
      const int tb = rb0 + tbl;
      const int vt0 = (int)((int64_t)sp * n_vt / nsplit);
      const int vt1 = (int)((int64_t)(sp + 1) * n_vt / nsplit);
      const int p = tb * 128 + row;
      const bool valid = p < Teff;
      const bool keep = kImage && tbl < s_lim;  // uniform over the CTA
      const float R = (kImage && valid) ? ref[p] : 0.f;
      const int yt = valid ? tok_y[p] : -1;
      float m2 = -INFINITY, l = 0.f, zt = 0.f;
      bool found = false;
      for (int vt = vt0; vt < vt1; ++vt) {
        if (!(ok = wait_sleepy_cluster(&sm.acc_full[acc], acc_ph, abort, dev_err))) break;
        tc_fence_after();
#pragma unroll 1
        for (int c = 0; c < kLseBN / 32; ++c) {
          const int col0 = vt * kLseBN + c * 32;
          if (kImage ? col0 >= img_cols : col0 >= V) break;  // the rest lies past V
          float v[32];
          tmem_ld32(lane_addr + acc * kLseBN + c * 32, v);
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
          if (kImage) {
            // Terms relative to the token's reference: v[j] becomes P_j.
            m2 = fmaxf(m2, mc);
            float sum = 0.f;
#pragma unroll
            for (int j = 0; j < 32; ++j) {
              v[j] = valid ? ex2_approx(v[j] - R) : 0.f;
              sum += v[j];
            }
            l += sum;
          } else {
            if (mc == -INFINITY) continue;
            // Chunk terms relative to the chunk maximum, folded into the
            // running (maximum, sum).
            float sum = 0.f;
#pragma unroll
            for (int j = 0; j < 32; ++j) sum += ex2_approx(v[j] - mc);
            if (mc > m2) {
              l = l * ex2_approx(m2 - mc) + sum;
              m2 = mc;
            } else {
              l += sum * ex2_approx(mc - m2);
            }
          }
          if (keep) {
            // Per warp: its 32 rows x 64 columns (two chunks) as bf16 in the
            // image atom's swizzled layout, in its own 4 KB buffer, stored by
            // its lane 0 once both halves are in (the image width is a
            // multiple of 64 columns). The store that last read this buffer
            // is done before the first half is written.
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
                __nv_bfloat162 b2 = __floats2bfloat162_rn(v[8 * e + 2 * q], v[8 * e + 2 * q + 1]);
                pk[q] = *reinterpret_cast<uint32_t *>(&b2);
              }
              *reinterpret_cast<uint4 *>(buf + lane * 128 + (((half * 4 + e) ^ (lane & 7)) << 4)) =
                  make_uint4(pk[0], pk[1], pk[2], pk[3]);
            }
            if (half == 1) {
              fence_async_smem();
              __syncwarp();
              if (lane == 0) {
                const int acol = col0 & ~63;  // the atom's first column
                uint8_t *dst = gimg +
                               (((size_t)tbl * n_vt128 + (acol >> 7)) * 2 + ((acol >> 6) & 1)) *
                                   kAtom128 +
                               quad * 4096;
                bulk_store_evict_first(dst, buf, 4096);
                bulk_commit_group();
              }
              sbuf_i ^= 1;
            }
          }
        }
        tc_fence_before();
        mbar_arrive_cluster(mapa(smem_u32(&sm.acc_empty[acc]), 0));
        if (++acc == 2) { acc = 0; acc_ph ^= 1; }
      }
      if (!ok) break;
      if (valid) {
        part[(int64_t)sp * Tpad + p] = make_float2(m2, l);
        if (found) zy[p] = zt;
      }
    }
    // Every image store has completed before the CTA leaves.
    if (lane == 0) bulk_wait_group<0>();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no CTA leaves while its peer may still signal or fill it
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, 512);
  }
}

// Largest distance (log2 units) of a row's maximum logit above its reference
// that the image pass keeps: the terms stay below 2^64, their sums far from
// the fp32 range. Rows beyond it are redone with the maximum as reference.
constexpr float kImgFixLog2 = 64.f;

// lse of tokens [128 rb0, 128 (rb0 + cap)) of the active ones, over the
// vocabulary splits. Without kImage: lse = ln 2 (M + log2 sum_s l_s 2^(m_s -
// M)). With kImage (terms relative to R_t): lsum_t = sum_s l_s and lse =
// ln 2 (R_t + log2 lsum_t); in the first pass (fix = 0), a row whose maximum
// m exceeds R_t by more than kImgFixLog2 instead gets R_t = m and is counted
// in counters[2] for the fix-up pass; the fix-up pass (fix = 1) runs only if
// some row was counted.
template <bool kImage>
__global__ void lse_combine_kernel(int nsplit, int64_t Tpad, int32_t *counters,
                                   const float2 *part, float *lse, float *ref, float *lsum,
                                   int rb0, int cap, int fix) {
  if (kImage && fix && counters[2] == 0) return;
  const int Teff = counters[0];
  const int64_t hi64 = (int64_t)(rb0 + (int64_t)cap) * 128;
  const int p1 = (int)(hi64 < Teff ? hi64 : Teff);
  for (int p = rb0 * 128 + blockIdx.x * blockDim.x + threadIdx.x; p < p1;
       p += gridDim.x * blockDim.x) {
    float M = -INFINITY;
    for (int s = 0; s < nsplit; ++s) M = fmaxf(M, part[(int64_t)s * Tpad + p].x);
    float L = 0.f;
    if (kImage) {
      for (int s = 0; s < nsplit; ++s) L += part[(int64_t)s * Tpad + p].y;
      const float R = ref[p];
      if (!fix && M - R > kImgFixLog2) {
        ref[p] = M;
        atomicAdd(&counters[2], 1);
      } else {
        lsum[p] = L;
        lse[p] = (R + log2f(L)) * 0.6931471805599453f;
      }
    } else {
      for (int s = 0; s < nsplit; ++s) {
        const float2 q = part[(int64_t)s * Tpad + p];
        if (q.y > 0.f) L += q.y * exp2f(q.x - M);
      }
      lse[p] = (M + log2f(L)) * 0.6931471805599453f;
    }
  }
}

// Reference of the image pass: R_p = z_p[y_p] log2 e for every compacted
// active token p (target_logit_dot).
__global__ void ref_logit_kernel(int d, const int32_t *counters, const int32_t *tok_y,
                                 const __nv_bfloat16 *Hc, const __nv_bfloat16 *W, float *ref) {
  const int Teff = counters[0];
  const int lane = threadIdx.x & 31;
  const int nw = (gridDim.x * blockDim.x) >> 5;
  for (int p = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; p < Teff; p += nw) {
    const float z = target_logit_dot(d, Hc + (int64_t)p * d, W + (int64_t)tok_y[p] * d, lane);
    if (lane == 0) ref[p] = z * kLog2e;
  }
}

// CTAs of the LSE grid: every 2-CTA cluster that fits at once (persistent).
int lse_grid(size_t smem) {
  static int cached = 0;
  if (cached) return cached;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kLsePair * 64, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, (const void *)lse_kernel<true>, &cfg) != cudaSuccess ||
      n <= 0) {
    cudaGetLastError();
    n = num_sms() / kLsePair;
  }
  cached = kLsePair * (n > 0 ? n : 1);
  return cached;
}

}  // namespace

namespace tck {

pair_status launch_ref(const GradArgs &g, const GradWorkspace &w, cudaStream_t s) {
  PAIR_BEGIN("ref_logit", s);
  ref_logit_kernel<<<num_sms() * 8, 256, 0, s>>>(
      g.d, w.counters, w.tok_y, static_cast<const __nv_bfloat16 *>(w.Hc),
      static_cast<const __nv_bfloat16 *>(g.W), w.ref);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

// Log-sum-exp pass over token blocks [rb0, rb0 + cap) (clipped to the active
// ones), then lse for those tokens. With image, the terms are relative to
// w.ref, the bf16 terms of the first s_blocks of those blocks are kept in
// w.gimg, and a fix-up pass redoes the blocks (only if some row was flagged).
pair_status launch_lse(const GradArgs &g, const GradWorkspace &w, cudaStream_t s, int rb0,
                       int cap, bool image, int s_blocks) {
  CUtensorMap mH, mW128;
  if (!make_map(&mH, w.Hc, w.Tpad, g.d, 128) || !make_map(&mW128, g.W, g.V, g.d, 128))
    return PAIR_ERR_CUDA;
  const int nsm = num_sms();
  const size_t lse_smem = sizeof(LseSmem) + 1024;
  PAIR_CUDA_TRY(cudaFuncSetAttribute(lse_kernel<true>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)lse_smem));
  PAIR_CUDA_TRY(cudaFuncSetAttribute(lse_kernel<false>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)lse_smem));
  const int grid = lse_grid(lse_smem);
  if (!image) {
    PAIR_BEGIN("lse_tc", s);
    lse_kernel<false><<<grid, kThreads, lse_smem, s>>>(
        mH, mW128, g.d, g.V, w.nsplit, w.Tpad, w.counters, w.tok_y, nullptr, w.part, w.zy, rb0,
        cap, nullptr, 0, 0, g.dev_err);
    PAIR_LAUNCH_CHECK(s);
    PAIR_BEGIN("lse_combine", s);
    lse_combine_kernel<false><<<nsm * 4, 256, 0, s>>>(w.nsplit, w.Tpad, w.counters, w.part,
                                                      w.lse, nullptr, nullptr, rb0, cap, 0);
    PAIR_LAUNCH_CHECK(s);
    return PAIR_OK;
  }
  uint8_t *gimg = static_cast<uint8_t *>(w.gimg);
  PAIR_CUDA_TRY(cudaMemsetAsync(w.counters + 2, 0, sizeof(int32_t), s));
  for (int fix = 0; fix < 2; ++fix) {
    PAIR_BEGIN(fix ? "lse_fix" : "lse_tc", s);
    lse_kernel<true><<<grid, kThreads, lse_smem, s>>>(
        mH, mW128, g.d, g.V, w.nsplit, w.Tpad, w.counters, w.tok_y, w.ref, w.part, w.zy, rb0,
        cap, gimg, s_blocks, fix, g.dev_err);
    PAIR_LAUNCH_CHECK(s);
    PAIR_BEGIN("lse_combine", s);
    lse_combine_kernel<true><<<nsm * 4, 256, 0, s>>>(w.nsplit, w.Tpad, w.counters, w.part,
                                                     w.lse, w.ref, w.lsum, rb0, cap, fix);
    PAIR_LAUNCH_CHECK(s);
  }
  return PAIR_OK;
}

}  // namespace tck
}  // namespace pairk
