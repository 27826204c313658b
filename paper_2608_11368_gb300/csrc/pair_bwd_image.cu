// Backward of the bf16 LM-head path through the image the log-sum-exp pass
// keeps: bf16 tiles of the softmax terms P_tv = 2^(z_tv log2 e - R_t)
// relative to each token's reference R_t, whose row sums lsum_t the pass
// also returns. With s_t = -c_t / lsum_t the softmax part of the logit
// gradient is Gs_tv = s_t P_tv, so
//     dH[t, :] = s_t sum_v P_tv W[v, :]     (dh_gemm, s_t in the epilogue)
//     dW[v, :] = sum_t P_tv (s_t Hc[t, :])   (dw_gemm on pre-scaled rows)
// as plain tcgen05 GEMMs (no logit recomputation, no pass over the image
// between them), one token chunk at a time.
#include "tc_kernels.cuh"

namespace pairk {
namespace {

using namespace tc;
using namespace tck;

// --------------------------------------------- scaled rows for dW
//
// Hs[i, :] = s_t Hc[t, :] in bf16 for the chunk's token rows t = 128 rb0 + i,
// s_t = -c_t / lsum_t (0 for c_t = 0); rows past T_eff are exact zeros.
// Streaming kernel, 8 columns per thread.
__global__ void __launch_bounds__(256)
    scale_rows_kernel(int d, int rb0, int cap, const int32_t *counters,
                      const float *__restrict__ tok_c, const float *__restrict__ lsum,
                      const __nv_bfloat16 *__restrict__ Hc, __nv_bfloat16 *__restrict__ Hs) {
  const int Teff = counters[0];
  const int nrb = min(max((Teff + 127) / 128 - rb0, 0), cap);
  const int d8 = d / 8;
  const int64_t n8 = (int64_t)nrb * 128 * d8;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n8;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = e / d8;
    const int k8 = (int)(e - i * d8);
    const int64_t t = (int64_t)rb0 * 128 + i;
    uint4 out = make_uint4(0u, 0u, 0u, 0u);
    if (t < Teff) {
      const float c = tok_c[t];
      if (c != 0.f) {
        const float sc = -c / lsum[t];
        const uint4 h = reinterpret_cast<const uint4 *>(Hc + t * d)[k8];
        const uint32_t hw[4] = {h.x, h.y, h.z, h.w};
        uint32_t pk[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float2 f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162 *>(&hw[q]));
          __nv_bfloat162 b2 = __floats2bfloat162_rn(sc * f.x, sc * f.y);
          pk[q] = *reinterpret_cast<uint32_t *>(&b2);
        }
        out = make_uint4(pk[0], pk[1], pk[2], pk[3]);
      }
    }
    reinterpret_cast<uint4 *>(Hs + i * d)[k8] = out;
  }
}

// Row scale of the softmax part of dH: s_t = -c_t / lsum_t.
__device__ __forceinline__ float row_scale(const float *tok_c, const float *lsum, int t) {
  const float c = tok_c[t];
  return c != 0.f ? -c / lsum[t] : 0.f;
}

// ---------------------------------------------- dH from the stored image
//
// Softmax part of dH as the plain GEMM dH[t, :] = s_t sum_v P[t, v] W[v, :],
// with the image tiles as the K-major A operand (64 vocabulary rows per
// stage, one 16 KB atom, copied verbatim), W as the MN-major B operand and
// the row scale s_t applied when the accumulator is drained.
// CTA pairs (2-CTA clusters) take two token blocks of the same 512-column
// chunk of d as two M = 256 tiles of 256 columns each: the even CTA issues
// every MMA of the pair (cta_group::2) over both CTAs' image atoms and each
// 256-column half's four W column atoms, two in each CTA, and each CTA's TMEM
// receives its own token block's rows (128 x 512 fp32, all of TMEM; a unit
// runs long enough that its drain, not overlapped with the next unit, costs
// well under 1 %). Work unit = (token block pair, 512-column chunk): the
// units of one token pair read its image rows, and with d = 2048 the 76
// pairs of a GB300 hold 19 token pairs' four units at once, so no token
// pair's units straddle two rounds. Each (token, column) is owned by one CTA
// and summed over all of V in one fixed order: deterministic, no atomics. An
// odd last block is computed twice (the pair's other CTA repeats it) and
// stored once.
constexpr int kDhN = 512;                              // output columns per unit
constexpr int kDhStages = 4;
constexpr uint32_t kDhABytes = kAtom128;               // 128 tokens x 64 vocabulary
constexpr uint32_t kDhBBytes = (kDhN / 128) * 64 * 128; // this CTA's 4 column atoms x 64 rows
constexpr uint32_t kIdescDh = idesc_bf16(256, 256, 0, 1);

// Work list of the persistent backward GEMMs (dh_gemm_kernel,
// dw_gemm_kernel): the units that fill whole rounds of the grid (ncl
// clusters) run over all of their K extent; the R < ncl units left for the
// last round are cut into S parts of K each (R S <= ncl, at most `cap`
// partial tiles of scratch), so that round takes a part's time instead of a
// unit's. Work item i < full_end is unit i; item full_end + j is part j % S
// of unit full_end + j / S, over K steps [part nks / S, (part + 1) nks / S);
// its fp32 tile goes to scratch slot j and the kernel's tail-combine pass
// adds the S parts in order (deterministic).
struct TailSplit {
  int full_end, R, S;
};
__host__ __device__ __forceinline__ TailSplit tail_split(int n_units, int ncl, int cap, int nks) {
  const int rem = n_units % ncl;
  int S = rem ? ncl / rem : 1;
  if (rem && S * rem > cap) S = cap / rem;
  if (S > nks) S = nks;
  if (S < 2) return TailSplit{n_units, 0, 1};
  return TailSplit{n_units - rem, rem, S};
}
// Work item i of a TailSplit -> unit u, its K steps [k0, k1) and scratch
// slot (-1: a whole unit).
__device__ __forceinline__ void tail_item(const TailSplit &tl, int nks, int i, int &u, int &k0,
                                          int &k1, int &slot) {
  if (i < tl.full_end) {
    u = i; k0 = 0; k1 = nks; slot = -1;
  } else {
    const int j = i - tl.full_end, part = j % tl.S;
    u = tl.full_end + j / tl.S;
    k0 = (int)((int64_t)part * nks / tl.S);
    k1 = (int)((int64_t)(part + 1) * nks / tl.S);
    slot = j;
  }
}

// Pacing of dh_gemm_kernel's whole units: the CTA pairs of a round read the
// same W rows (all of them read all of W, in step order) and four at a time
// the same image rows, so they share those rows in L2 only while they stay
// close in the vocabulary. Every kPaceEvery K steps the even CTA's producer
// publishes its position (round * nks + step) and, while it is more than
// kPaceLead steps ahead of the slowest pair still on a whole unit, waits
// (at most kPaceCycles per check, then it goes on: the pacing only affects
// speed, never results). A pair that has left its whole units publishes
// INT_MAX. (The log-sum-exp pass and the dW GEMM run K steps a third as
// long: there the check itself stalls their producers, whose stages hold
// under 2 us of work, and pacing them measured 9-14 % slower.)
constexpr int kPaceEvery = 16;
constexpr int kPaceLead = 64;
constexpr long long kPaceCycles = 40000;

__device__ __forceinline__ void pace_publish(int32_t *prog, int pid, int pos) {
  *reinterpret_cast<volatile int32_t *>(prog + pid) = pos;
}
// Whole warp: bounded wait until every pair's position is at least pos - kPaceLead.
__device__ __forceinline__ void pace_wait(const int32_t *prog, int ncl, int pos, int lane) {
  const long long t0 = clock64();
  while (true) {
    int mn = 0x7fffffff;
    for (int c = lane; c < ncl; c += 32)
      mn = min(mn, *reinterpret_cast<const volatile int32_t *>(prog + c));
    for (int o = 16; o > 0; o >>= 1) mn = min(mn, __shfl_xor_sync(0xffffffffu, mn, o));
    if (mn >= pos - kPaceLead || clock64() - t0 > kPaceCycles) break;
    __nanosleep(256);
  }
}

struct DhSmem {
  uint8_t a[kDhStages][kDhABytes];
  uint8_t b[kDhStages][kDhBBytes];
  uint64_t full[kDhStages], empty[kDhStages];
  uint64_t acc_full, acc_empty, mma_done;
  uint32_t tmem_base;
  int abort;
};

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    dh_gemm_kernel(const __grid_constant__ CUtensorMap tmG, const __grid_constant__ CUtensorMap tmW,
                   int d, int V, int rb0, int cap, const int32_t *counters,
                   const int32_t *tok_idx, const float *tok_c, const float *lsum, float *dH,
                   float *scratch, int scratch_cap, int32_t *prog, int32_t *dev_err) {
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
  const TailSplit tl = tail_split(n_units, npairs, scratch_cap, nks);
  const int n_items = tl.full_end + tl.R * tl.S;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kDhStages; ++s) {
      mbar_init(&sm.full[s], 1);   // the even CTA's expect_tx (both CTAs' bytes)
      mbar_init(&sm.empty[s], 1);  // the pair MMA's commit
    }
    mbar_init(&sm.acc_full, 1);
    mbar_init(&sm.acc_empty, 2 * 128);  // both CTAs' epilogue threads
    mbar_init(&sm.mma_done, 1);
    sm.abort = 0;
    fence_mbar_init();
    prefetch_tmap(&tmG);
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
      int last_ph[kDhStages];
      for (int s = 0; s < kDhStages; ++s) last_ph[s] = -1;
      bool ok = true;
      const bool pacing = prog != nullptr && r == 0 && npairs <= kMaxPairs;
      if (pacing && lane == 0) pace_publish(prog, pid, 0);
      for (int i = pid; i < n_items && ok; i += npairs) {
        int u, k0, k1, slot;
        tail_item(tl, nks, i, u, k0, k1, slot);
        const int tp = u / nq, q = u - tp * nq;
        const int b = min(2 * tp + r, nrb - 1);
        const int atom0 = b * nks;  // the block's first image atom
        const bool whole = pacing && slot < 0;
        if (pacing && !whole && lane == 0) pace_publish(prog, pid, 0x7fffffff);
        for (int ks = k0; ks < k1; ++ks) {
          if (whole && (ks & (kPaceEvery - 1)) == 0) {
            const int pos = (i / npairs) * nks + ks;
            if (lane == 0) pace_publish(prog, pid, pos);
            pace_wait(prog, npairs, pos, lane);
          }
          if (!(ok = wait_cluster(&sm.empty[stage], ph ^ 1, abort, dev_err))) break;
          if (elect_one()) {
            if (r == 0) mbar_expect_tx(&sm.full[stage], 2 * (kDhABytes + kDhBBytes));
            const uint32_t fb = mapa(smem_u32(&sm.full[stage]), 0);
            tma_load_3d_pair(sm.a[stage], &tmG, fb, 0, 0, atom0 + ks);
            // Column atoms 2r, 2r + 1 of each 256-column half of the chunk.
            tma_load_3d_pair(sm.b[stage], &tmW, fb, 0, 64 * ks, q * (kDhN / 64) + 2 * r);
            tma_load_3d_pair(sm.b[stage] + kDhBBytes / 2, &tmW, fb, 0, 64 * ks,
                             q * (kDhN / 64) + 4 + 2 * r);
          }
          __syncwarp();
          last_ph[stage] = (int)ph;
          if (++stage == kDhStages) { stage = 0; ph ^= 1; }
        }
      }
      if (pacing && lane == 0) pace_publish(prog, pid, 0x7fffffff);
      // The last copy of every stage: completed on the even CTA, consumed by
      // the pair MMA on the odd one (both CTAs issue the same sequence).
      for (int s = 0; s < kDhStages; ++s)
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
      // A: K-major atom, 16 tokens of K = 32 bytes along the swizzled row.
      // B: per 256-column half, this CTA's 2 column atoms of 64 vocabulary
      // rows (LBO 8 KB), row groups of 8 (SBO 1 KB); 16 vocabulary rows =
      // 2 KB; the second half is 16 KB on.
      const uint64_t da0 = sdesc_sw128(smem_u32(sm.a[0]), 16, 1024);
      const uint64_t db0 = sdesc_sw128(smem_u32(sm.b[0]), 64 * 128, 1024);
      int stage = 0;
      uint32_t ph = 0, acc_ph = 0;
      bool ok = true;
      for (int i = pid; i < n_items && ok; i += npairs) {
        int u, k0, k1, slot;
        tail_item(tl, nks, i, u, k0, k1, slot);
        if (!(ok = wait_cluster(&sm.acc_empty, acc_ph ^ 1, abort, dev_err))) break;
        acc_ph ^= 1;
        tc_fence_after();
        for (int ks = k0; ks < k1; ++ks) {
          if (!(ok = wait_cluster(&sm.full[stage], ph, abort, dev_err))) break;
          tc_fence_after();
          const uint64_t da = da0 + (uint64_t)stage * (kDhABytes >> 4);
          const uint64_t db = db0 + (uint64_t)stage * (kDhBBytes >> 4);
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
#pragma unroll
              for (int nh = 0; nh < 2; ++nh)
                mma_bf16_pair(tmem + nh * 256, da + 2 * kk,
                              db + nh * ((kDhBBytes / 2) >> 4) + kk * (2048 >> 4), kIdescDh,
                              (ks != k0) | (kk != 0));
            mma_commit_pair(&sm.empty[stage], (uint16_t)3);
          }
          __syncwarp();
          if (++stage == kDhStages) { stage = 0; ph ^= 1; }
        }
        if (!ok) break;
        if (elect_one()) mma_commit_pair(&sm.acc_full, (uint16_t)3);
        __syncwarp();
      }
      if (elect_one()) mma_commit_pair(&sm.mma_done, (uint16_t)1);
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
    for (int i = pid; i < n_items && ok; i += npairs) {
      int u, k0, k1, slot;
      tail_item(tl, nks, i, u, k0, k1, slot);
      const int tp = u / nq, q = u - tp * nq;
      const int t = (rb0 + 2 * tp + r) * 128 + row;
      const bool valid = 2 * tp + r < nrb && t < Teff;
      float4 *dst =
          slot >= 0
              ? reinterpret_cast<float4 *>(scratch + (((int64_t)slot * 2 + r) * 128 + row) * kDhN)
          : valid ? reinterpret_cast<float4 *>(dH + (int64_t)tok_idx[t] * d + q * kDhN)
                  : nullptr;
      // Partial tiles stay unscaled (the combine pass scales their sum).
      const float sc = (slot < 0 && valid) ? row_scale(tok_c, lsum, t) : 1.f;
      if (!(ok = wait_sleepy_cluster(&sm.acc_full, acc_ph, abort, dev_err))) break;
      acc_ph ^= 1;
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < kDhN / 32; ++c) {
        float x[32];
        tmem_ld32(tmem + lane_off + c * 32, x);
        if (dst) {
#pragma unroll
          for (int e = 0; e < 8; ++e)
            dst[c * 8 + e] = make_float4(sc * x[4 * e], sc * x[4 * e + 1], sc * x[4 * e + 2],
                                         sc * x[4 * e + 3]);
        }
      }
      tc_fence_before();
      mbar_arrive_cluster(mapa(smem_u32(&sm.acc_empty), 0));
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no CTA leaves while its peer may still signal or fill it
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, 512);
  }
}

// dH of the units dh_gemm_kernel split into vocabulary parts (see TailSplit):
// the sum of their S partial tiles in part order, times the row scale.
__global__ void __launch_bounds__(256)
    dh_tail_combine_kernel(int d, int V, int rb0, int cap, int ncl, int scratch_cap,
                           const int32_t *counters, const int32_t *tok_idx,
                           const float *__restrict__ tok_c, const float *__restrict__ lsum,
                           const float *__restrict__ scratch, float *dH) {
  const int Teff = counters[0];
  const int nrb = min(max((Teff + 127) / 128 - rb0, 0), cap);
  if (nrb == 0) return;
  const int nks = 2 * ((V + 127) / 128);
  const int nq = d / kDhN;
  const TailSplit tl = tail_split((nrb + 1) / 2 * nq, ncl, scratch_cap, nks);
  constexpr int kQ = kDhN / 4;  // float4 per tile row
  const int64_t n4 = (int64_t)tl.R * 2 * 128 * kQ;
  const float4 *src = reinterpret_cast<const float4 *>(scratch);
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n4;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int c4 = (int)(e % kQ);
    const int row = (int)((e / kQ) % 128);
    const int r = (int)((e / (kQ * 128)) % 2);
    const int uj = (int)(e / (kQ * 256));
    const int u = tl.full_end + uj;
    const int tp = u / nq, q = u - tp * nq;
    const int t = (rb0 + 2 * tp + r) * 128 + row;
    if (2 * tp + r >= nrb || t >= Teff) continue;
    float4 acc = src[(((int64_t)uj * tl.S * 2 + r) * 128 + row) * kQ + c4];
    for (int p = 1; p < tl.S; ++p) {
      const float4 v = src[((((int64_t)uj * tl.S + p) * 2 + r) * 128 + row) * kQ + c4];
      acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
    }
    const float sc = row_scale(tok_c, lsum, t);
    reinterpret_cast<float4 *>(dH + (int64_t)tok_idx[t] * d + q * kDhN)[c4] =
        make_float4(sc * acc.x, sc * acc.y, sc * acc.z, sc * acc.w);
  }
}

// ------------------------------------- dW from the stored softmax terms
//
// The image keeps every bf16 tile P of a chunk of token blocks (128 tokens x
// 128 vocabulary rows, 32 KB, in the K-major SWIZZLE_128B layout of the dH
// GEMM's A operand). Read with the token index as K, the same bytes are the
// MN-major SWIZZLE_128B layout of P^T (64 vocabulary rows per 128-byte line,
// one line per token), so with the pre-scaled rows Hs = s_t Hc[t, :] of the
// chunk the softmax part of dW is the plain GEMM
//     dW[v, :] (+)= sum_t P[t, v] Hs[t, :]
// with no logit recomputation.
//
// CTA pairs (2-CTA clusters) share one 512-column chunk of Hs as two M = 256
// tiles of 256 columns each: the even CTA issues every MMA of the pair
// (cta_group::2) over both CTAs' P^T stages (each CTA fetches the one of its
// own 128 vocabulary rows) and each 256-column half's four Hs column atoms,
// two in each CTA. Work unit = (vocabulary block pair, 512-column chunk of
// d); CTA r accumulates dW[block 2 p + r, chunk] (128 x 512 fp32 = all of
// TMEM) over the chunk's tokens, 32 token rows per stage, and drains it with
// plain stores (first chunk) or read-add-writes (later chunks; this CTA owns
// those rows). An odd last block is computed twice (the pair's other CTA
// repeats the last block) so both CTAs run the same stage sequence; only one
// stores it.
constexpr int kDwKS = 32;                                 // token rows per stage
constexpr int kDwStages = 5;
constexpr int kDwN = 512;                                 // output columns per CTA
constexpr uint32_t kDwGBytes = 2 * kDwKS * 128;           // 2 vocabulary atoms x 32 rows
constexpr uint32_t kDwHBytes = (kDwN / 128) * kDwKS * 128; // this CTA's 4 column atoms x 32 rows
constexpr uint32_t kIdescDw = idesc_bf16(256, 256, 1, 1); // both operands MN-major

struct DwSmem {
  uint8_t g[kDwStages][kDwGBytes];  // P^T: MN-major A, atoms 4 KB apart
  uint8_t h[kDwStages][kDwHBytes];  // Hs[t, chunk]: MN-major B, atoms 4 KB apart
  uint64_t full[kDwStages], empty[kDwStages];
  uint64_t acc_full, acc_empty, mma_done;
  uint32_t tmem_base;
  int abort;
};

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    dw_gemm_kernel(const __grid_constant__ CUtensorMap tmG,
                   const __grid_constant__ CUtensorMap tmH, int d, int V, int rb0, int cap,
                   int accumulate, const int32_t *counters, float *dW, float *scratch,
                   int scratch_cap, int32_t *dev_err) {
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
  const TailSplit tl = tail_split(n_units, npairs, scratch_cap, nks);
  const int n_items = tl.full_end + tl.R * tl.S;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kDwStages; ++s) {
      mbar_init(&sm.full[s], 1);   // the even CTA's expect_tx (both CTAs' bytes)
      mbar_init(&sm.empty[s], 1);  // the pair MMA's commit
    }
    mbar_init(&sm.acc_full, 1);
    mbar_init(&sm.acc_empty, 2 * 128);  // both CTAs' epilogue threads
    mbar_init(&sm.mma_done, 1);
    sm.abort = 0;
    fence_mbar_init();
    prefetch_tmap(&tmG);
    prefetch_tmap(&tmH);
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
      int last_ph[kDwStages];
      for (int s = 0; s < kDwStages; ++s) last_ph[s] = -1;
      bool ok = true;
      for (int i = pid; i < n_items && ok; i += npairs) {
        int u, k0, k1, slot;
        tail_item(tl, nks, i, u, k0, k1, slot);
        const int vp = u / nq, q = u - vp * nq;
        const int vb = min(2 * vp + r, n_vb - 1);
        for (int ks = k0; ks < k1; ++ks) {
          const int rbl = ks >> 2, j = ks & 3;
          if (!(ok = wait_cluster(&sm.empty[stage], ph ^ 1, abort, dev_err))) break;
          if (elect_one()) {
            if (r == 0) mbar_expect_tx(&sm.full[stage], 2 * (kDwGBytes + kDwHBytes));
            const uint32_t fb = mapa(smem_u32(&sm.full[stage]), 0);
            const int t0 = rbl * 128 + kDwKS * j;  // chunk row of Hs
            tma_load_3d_pair(sm.g[stage], &tmG, fb, 0, kDwKS * j, 2 * (rbl * n_vb + vb));
            // Column atoms 2r, 2r + 1 of each 256-column half of the chunk.
            tma_load_3d_pair(sm.h[stage], &tmH, fb, 0, t0, q * (kDwN / 64) + 2 * r);
            tma_load_3d_pair(sm.h[stage] + kDwHBytes / 2, &tmH, fb, 0, t0,
                             q * (kDwN / 64) + 4 + 2 * r);
          }
          __syncwarp();
          last_ph[stage] = (int)ph;
          if (++stage == kDwStages) { stage = 0; ph ^= 1; }
        }
      }
      // Never leave a copy in flight: wait (bounded) for the last one issued
      // on every stage: completed on the even CTA, consumed by the pair MMA
      // on the odd one (both CTAs issue the same sequence).
      for (int s = 0; s < kDwStages; ++s)
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
      // A: 2 vocabulary atoms (LBO 4 KB), token groups of 8 rows (SBO 1 KB);
      // B: this CTA's 2 column atoms of each half (LBO 4 KB), the same token
      // groups. One K step of 16 tokens advances both by 2 KB; B's second
      // 256-column half is 8 KB on.
      const uint64_t dg0 = sdesc_sw128(smem_u32(sm.g[0]), kDwKS * 128, 1024);
      const uint64_t dh0 = sdesc_sw128(smem_u32(sm.h[0]), kDwKS * 128, 1024);
      int stage = 0;
      uint32_t ph = 0, acc_ph = 0;
      bool ok = true;
      for (int i = pid; i < n_items && ok && nks > 0; i += npairs) {
        int u, k0, k1, slot;
        tail_item(tl, nks, i, u, k0, k1, slot);
        if (!(ok = wait_cluster(&sm.acc_empty, acc_ph ^ 1, abort, dev_err))) break;
        acc_ph ^= 1;
        tc_fence_after();
        for (int ks = k0; ks < k1; ++ks) {
          if (!(ok = wait_cluster(&sm.full[stage], ph, abort, dev_err))) break;
          tc_fence_after();
          const uint64_t dg = dg0 + (uint64_t)stage * (kDwGBytes >> 4);
          const uint64_t dh = dh0 + (uint64_t)stage * (kDwHBytes >> 4);
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < kDwKS / 16; ++kk)
#pragma unroll
              for (int nh = 0; nh < 2; ++nh)
                mma_bf16_pair(tmem + nh * 256, dg + kk * (2048 >> 4),
                              dh + nh * ((kDwHBytes / 2) >> 4) + kk * (2048 >> 4), kIdescDw,
                              (ks != k0) | (kk != 0));
            mma_commit_pair(&sm.empty[stage], (uint16_t)3);
          }
          __syncwarp();
          if (++stage == kDwStages) { stage = 0; ph ^= 1; }
        }
        if (!ok) break;
        if (elect_one()) mma_commit_pair(&sm.acc_full, (uint16_t)3);
        __syncwarp();
      }
      if (elect_one()) mma_commit_pair(&sm.mma_done, (uint16_t)1);
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
    for (int i = pid; i < n_items && ok; i += npairs) {
      int u, k0, k1, slot;
      tail_item(tl, nks, i, u, k0, k1, slot);
      const int vp = u / nq, q = u - vp * nq;
      const int v = (2 * vp + r) * 128 + row;
      const bool valid = 2 * vp + r < n_vb && v < V;
      float4 *dst = valid ? reinterpret_cast<float4 *>(dW + (int64_t)v * d + q * kDwN) : nullptr;
      float4 *part_dst =
          slot >= 0
              ? reinterpret_cast<float4 *>(scratch + (((int64_t)slot * 2 + r) * 128 + row) * kDwN)
              : nullptr;
      if (nks == 0) {
        if (valid)
          for (int c = 0; c < kDwN / 4; ++c) dst[c] = make_float4(0.f, 0.f, 0.f, 0.f);
        continue;
      }
      if (!(ok = wait_sleepy_cluster(&sm.acc_full, acc_ph, abort, dev_err))) break;
      acc_ph ^= 1;
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < kDwN / 32; ++c) {
        float x[32];
        tmem_ld32(tmem + lane_off + c * 32, x);
        if (part_dst) {
#pragma unroll
          for (int e = 0; e < 8; ++e)
            part_dst[c * 8 + e] = make_float4(x[4 * e], x[4 * e + 1], x[4 * e + 2], x[4 * e + 3]);
        } else if (valid) {
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
      mbar_arrive_cluster(mapa(smem_u32(&sm.acc_empty), 0));
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no CTA leaves while its peer may still signal or fill it
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, 512);
  }
}

// dW rows of the units dw_gemm_kernel split into token parts (see
// TailSplit): the sum of their S partial tiles in part order, stored or
// (later token chunks) added.
__global__ void __launch_bounds__(256)
    dw_tail_combine_kernel(int d, int V, int rb0, int cap, int accumulate, int ncl,
                           int scratch_cap, const int32_t *counters,
                           const float *__restrict__ scratch, float *dW) {
  const int Teff = counters[0];
  const int nrb = min(max((Teff + 127) / 128 - rb0, 0), cap);
  const int n_vb = (V + 127) / 128;
  const int nq = d / kDwN;
  const TailSplit tl = tail_split((n_vb + 1) / 2 * nq, ncl, scratch_cap, nrb * (128 / kDwKS));
  constexpr int kQ = kDwN / 4;  // float4 per tile row
  const int64_t n4 = (int64_t)tl.R * 2 * 128 * kQ;
  const float4 *src = reinterpret_cast<const float4 *>(scratch);
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n4;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int c4 = (int)(e % kQ);
    const int row = (int)((e / kQ) % 128);
    const int r = (int)((e / (kQ * 128)) % 2);
    const int uj = (int)(e / (kQ * 256));
    const int u = tl.full_end + uj;
    const int vp = u / nq, q = u - vp * nq;
    const int v = (2 * vp + r) * 128 + row;
    if (2 * vp + r >= n_vb || v >= V) continue;
    float4 acc = src[(((int64_t)uj * tl.S * 2 + r) * 128 + row) * kQ + c4];
    for (int p = 1; p < tl.S; ++p) {
      const float4 x = src[((((int64_t)uj * tl.S + p) * 2 + r) * 128 + row) * kQ + c4];
      acc.x += x.x; acc.y += x.y; acc.z += x.z; acc.w += x.w;
    }
    float4 *dst = reinterpret_cast<float4 *>(dW + (int64_t)v * d + q * kDwN) + c4;
    if (accumulate) {
      const float4 o = *dst;
      acc.x += o.x; acc.y += o.y; acc.z += o.z; acc.w += o.w;
    }
    *dst = acc;
  }
}

}  // namespace

namespace tck {

pair_status launch_chunk_bwd(const GradArgs &g, const GradWorkspace &w, cudaStream_t s,
                             int64_t c) {
  const int cap = w.gimg_rb;
  const int rb0 = (int)(c * cap);
  const int n_vt = (g.V + 127) / 128;
  CUtensorMap mG, mGA, mH3, mW3;
  if (!make_map3(&mG, w.gimg, {64, 128, (cuuint64_t)2 * cap * n_vt}, {128, 16384}, {64, 32, 2},
                 CU_TENSOR_MAP_SWIZZLE_NONE) ||
      !make_map3(&mGA, w.gimg, {64, 128, (cuuint64_t)2 * cap * n_vt}, {128, 16384}, {64, 128, 1},
                 CU_TENSOR_MAP_SWIZZLE_NONE) ||
      !make_map3(&mH3, w.hs, {64, (cuuint64_t)cap * 128, (cuuint64_t)g.d / 64},
                 {(cuuint64_t)g.d * 2, 128}, {64, (cuuint32_t)kDwKS, 2},
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
  PAIR_BEGIN("scale_rows", s);
  scale_rows_kernel<<<num_sms() * 4, 256, 0, s>>>(
      g.d, rb0, cap, w.counters, w.tok_c, w.lsum, static_cast<const __nv_bfloat16 *>(w.Hc),
      static_cast<__nv_bfloat16 *>(w.hs));
  PAIR_LAUNCH_CHECK(s);
  // Scratch for the split last round of dH: the cluster path's tail rows
  // (unused by this path), in 2 x 128 x kDhN fp32 tiles.
  const int dh_grid = pair_grid((const void *)dh_gemm_kernel, dh_smem, &dh_cache);
  const int scratch_cap =
      w.tailbuf ? (int)((int64_t)kMaxClusters * 2 * 128 * g.d / (2 * 128 * kDhN)) : 0;
  PAIR_BEGIN("dh_gemm_tc", s);
  dh_gemm_kernel<<<dh_grid, kThreads, dh_smem, s>>>(mGA, mW3, g.d, g.V, rb0, cap, w.counters,
                                                    w.tok_idx, w.tok_c, w.lsum, g.dH, w.tailbuf,
                                                    scratch_cap, w.prog, g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  if (scratch_cap > 0) {
    PAIR_BEGIN("dh_tail", s);
    dh_tail_combine_kernel<<<num_sms() * 2, 256, 0, s>>>(g.d, g.V, rb0, cap, dh_grid / 2,
                                                         scratch_cap, w.counters, w.tok_idx,
                                                         w.tok_c, w.lsum, w.tailbuf, g.dH);
    PAIR_LAUNCH_CHECK(s);
  }
  const int dw_grid = pair_grid((const void *)dw_gemm_kernel, dw_smem, &dw_cache);
  const int dw_scratch_cap =
      w.tailbuf ? (int)((int64_t)kMaxClusters * 2 * 128 * g.d / (2 * 128 * kDwN)) : 0;
  PAIR_BEGIN("dw_gemm_tc", s);
  dw_gemm_kernel<<<dw_grid, kThreads, dw_smem, s>>>(mG, mH3, g.d, g.V, rb0, cap, c > 0 ? 1 : 0,
                                                    w.counters, g.dW, w.tailbuf, dw_scratch_cap,
                                                    g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  if (dw_scratch_cap > 0) {
    PAIR_BEGIN("dw_tail", s);
    dw_tail_combine_kernel<<<num_sms() * 2, 256, 0, s>>>(g.d, g.V, rb0, cap, c > 0 ? 1 : 0,
                                                         dw_grid / 2, dw_scratch_cap, w.counters,
                                                         w.tailbuf, g.dW);
    PAIR_LAUNCH_CHECK(s);
  }
  return PAIR_OK;
}


}  // namespace tck

// Memory the backward may use for the image of softmax terms (32 KB per
// 128 x 128 tile) and the scaled hidden rows of a chunk (128 d bf16 per token
// block); larger problems run in token chunks.
constexpr int64_t kImageBudget = int64_t(24) << 30;

int grad_gimg_rows(int64_t T, int32_t d, int32_t V, pair_dtype dt) {
  if (dt != PAIR_BF16 || d < 512 || d % kDwN != 0) return 0;
  const int64_t n_rb = (T + 127) / 128;
  const int64_t per_rb = (int64_t)grad_image_block_bytes(d, V);
  int64_t cap = kImageBudget / per_rb;
  if (cap < 32) cap = 32;
  return (int)(n_rb < cap ? n_rb : cap);
}

size_t grad_image_block_bytes(int32_t d, int32_t V) {
  return (size_t)((V + 127) / 128) * kGImgTileBytes + (size_t)128 * d * 2;
}

}  // namespace pairk
