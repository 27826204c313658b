// fp32 LM-head path of pair_grad on the CUDA cores (PAIR_F32 inputs).
//
// The objective of Sec. 4.5, sum_i a_i log pi(o_i|q), over compacted active
// tokens t (coefficient c_t = a of its rollout):
//   z_tv = <h_t, W_v>, lse_t = log sum_v exp z_tv, logp_t = z_{t,y_t} - lse_t
//   dJ/dh_t = sum_v G_tv W_v,  dJ/dW_v = sum_t G_tv h_t,
//   G_tv = c_t (1[v = y_t] - exp(z_tv - lse_t)).
// Logits are recomputed where needed and never stored. Every reduction runs
// in a fixed order (warp xor-tree, then warps in index order), so results
// are bit-reproducible. fp32 throughout (the one-hot term is exact in G).
#include "pair_common.cuh"

namespace pairk {
namespace {

constexpr int kWarps = 8;

__device__ __forceinline__ float warp_sum(float v) {
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// lse and target logit of every active token: one block per token, one warp
// per vocabulary row (coalesced W reads), online max / sum-exp per warp.
__global__ void __launch_bounds__(kWarps * 32) simt_lse_kernel(
    int d, int V, const int32_t *counters, const float *Hc, const float *W,
    const int32_t *tok_y, float *lse, float *zy) {
  extern __shared__ float hs[];
  __shared__ float wm[kWarps], wl[kWarps], wz[kWarps];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Teff = counters[0];
  for (int p = blockIdx.x; p < Teff; p += gridDim.x) {
    for (int k = threadIdx.x; k < d; k += blockDim.x) hs[k] = Hc[(int64_t)p * d + k];
    __syncthreads();
    const int yt = tok_y[p];
    float m = -INFINITY, l = 0.f, zt = 0.f;
    for (int v = warp; v < V; v += kWarps) {
      const float *w = W + (int64_t)v * d;
      float z = 0.f;
      for (int k = lane; k < d; k += 32) z = fmaf(hs[k], w[k], z);
      z = warp_sum(z);
      const float mn = fmaxf(m, z);
      l = l * expf(m - mn) + expf(z - mn);
      m = mn;
      if (v == yt) zt = z;
    }
    if (lane == 0) { wm[warp] = m; wl[warp] = l; wz[warp] = zt; }
    __syncthreads();
    if (threadIdx.x == 0) {
      float M = -INFINITY;
      for (int k = 0; k < kWarps; ++k) M = fmaxf(M, wm[k]);
      float L = 0.f, Z = 0.f;
      for (int k = 0; k < kWarps; ++k) {
        L += wl[k] * expf(wm[k] - M);
        if ((yt % kWarps) == k) Z = wz[k];
      }
      lse[p] = M + logf(L);
      zy[p] = Z;
    }
    __syncthreads();
  }
}

// dJ/dh_t for every active token: one block per token; warp w accumulates
// vocabulary rows v = w mod kWarps into its own shared-memory row.
__global__ void __launch_bounds__(kWarps * 32) simt_dh_kernel(
    int d, int V, const int32_t *counters, const int32_t *tok_idx,
    const float *Hc, const float *W, const int32_t *tok_y, const float *tok_c,
    const float *lse, float *dH) {
  extern __shared__ float sm[];
  float *hs = sm;            // [d]
  float *acc = sm + d;       // [kWarps][d]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Teff = counters[0];
  for (int p = blockIdx.x; p < Teff; p += gridDim.x) {
    for (int k = threadIdx.x; k < d; k += blockDim.x) hs[k] = Hc[(int64_t)p * d + k];
    for (int k = threadIdx.x; k < kWarps * d; k += blockDim.x) acc[k] = 0.f;
    __syncthreads();
    const int yt = tok_y[p];
    const float c = tok_c[p], ls = lse[p];
    float *my = acc + warp * d;
    for (int v = warp; v < V; v += kWarps) {
      const float *w = W + (int64_t)v * d;
      float z = 0.f;
      for (int k = lane; k < d; k += 32) z = fmaf(hs[k], w[k], z);
      z = warp_sum(z);
      const float g = c * ((v == yt ? 1.f : 0.f) - expf(z - ls));
      for (int k = lane; k < d; k += 32) my[k] = fmaf(g, w[k], my[k]);
    }
    __syncthreads();
    float *row = dH + (int64_t)tok_idx[p] * d;
    for (int k = threadIdx.x; k < d; k += blockDim.x) {
      float s = 0.f;
      for (int q = 0; q < kWarps; ++q) s += acc[q * d + k];
      row[k] = s;
    }
    __syncthreads();
  }
}

// dJ/dW_v for every vocabulary row: one block per row; warp w accumulates
// active tokens p = w mod kWarps.
__global__ void __launch_bounds__(kWarps * 32) simt_dw_kernel(
    int d, int V, const int32_t *counters, const float *Hc, const float *W,
    const int32_t *tok_y, const float *tok_c, const float *lse, float *dW) {
  extern __shared__ float sm[];
  float *ws = sm;            // [d]
  float *acc = sm + d;       // [kWarps][d]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Teff = counters[0];
  for (int v = blockIdx.x; v < V; v += gridDim.x) {
    for (int k = threadIdx.x; k < d; k += blockDim.x) ws[k] = W[(int64_t)v * d + k];
    for (int k = threadIdx.x; k < kWarps * d; k += blockDim.x) acc[k] = 0.f;
    __syncthreads();
    float *my = acc + warp * d;
    for (int p = warp; p < Teff; p += kWarps) {
      const float *h = Hc + (int64_t)p * d;
      float z = 0.f;
      for (int k = lane; k < d; k += 32) z = fmaf(ws[k], h[k], z);
      z = warp_sum(z);
      const float g = tok_c[p] * ((tok_y[p] == v ? 1.f : 0.f) - expf(z - lse[p]));
      for (int k = lane; k < d; k += 32) my[k] = fmaf(g, h[k], my[k]);
    }
    __syncthreads();
    float *row = dW + (int64_t)v * d;
    for (int k = threadIdx.x; k < d; k += blockDim.x) {
      float s = 0.f;
      for (int q = 0; q < kWarps; ++q) s += acc[q * d + k];
      row[k] = s;
    }
    __syncthreads();
  }
}

}  // namespace

pair_status grad_lse_simt(const GradArgs &g, const GradWorkspace &w, cudaStream_t s) {
  const float *Hc = static_cast<const float *>(w.Hc);
  const float *W = static_cast<const float *>(g.W);
  const int grid = 152 * 8;
  const size_t sm1 = (size_t)g.d * 4;
  PAIR_CUDA_TRY(cudaFuncSetAttribute(simt_lse_kernel,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm1));
  PAIR_BEGIN("simt_lse", s);
  simt_lse_kernel<<<grid, kWarps * 32, sm1, s>>>(g.d, g.V, w.counters, Hc, W, w.tok_y, w.lse,
                                                 w.zy);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

pair_status grad_bwd_simt(const GradArgs &g, const GradWorkspace &w, cudaStream_t s) {
  const float *Hc = static_cast<const float *>(w.Hc);
  const float *W = static_cast<const float *>(g.W);
  const int grid = 152 * 8;
  const size_t sm2 = (size_t)(kWarps + 1) * g.d * 4;
  PAIR_CUDA_TRY(cudaFuncSetAttribute(simt_dh_kernel,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm2));
  PAIR_CUDA_TRY(cudaFuncSetAttribute(simt_dw_kernel,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm2));
  PAIR_BEGIN("simt_dh", s);
  simt_dh_kernel<<<grid, kWarps * 32, sm2, s>>>(g.d, g.V, w.counters, w.tok_idx, Hc, W, w.tok_y,
                                                w.tok_c, w.lse, g.dH);
  PAIR_LAUNCH_CHECK(s);
  const int gridv = (int)(g.V < 152 * 16 ? g.V : 152 * 16);
  PAIR_BEGIN("simt_dw", s);
  simt_dw_kernel<<<gridv, kWarps * 32, sm2, s>>>(g.d, g.V, w.counters, Hc, W, w.tok_y, w.tok_c,
                                                 w.lse, g.dW);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

pair_status grad_head_simt(const GradArgs &g, const GradWorkspace &w, cudaStream_t s) {
  const pair_status st = grad_lse_simt(g, w, s);
  return st != PAIR_OK ? st : grad_bwd_simt(g, w, s);
}

}  // namespace pairk
