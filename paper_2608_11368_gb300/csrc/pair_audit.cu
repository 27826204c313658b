// pair_audit: the frozen-population estimator audit (Sec. 5, "Frozen-policy
// estimator audit"; App. D metrics) over many design draws of one candidate
// group with explicit score vectors s_i in R^D.
//
// Target: the complete-pair gradient g = scale * sum_{i<j} h_ij over all G
// candidates (Eq. pair-kernel), i.e. g = sum_i abar_i s_i with
// abar_i = scale * 1/2 sum_{j != i} (r_i - r_j). Every draw's estimate is
// ghat_b = sum_i a_bi s_i (the coefficient collapse of Eq. pair-ht, under any
// weighting of pair_coeffs_weighted), so with the Gram matrix K = S S^T all
// statistics are G-dimensional quadratic forms:
//   ||ghat_b - g||^2 = e_b^T K e_b,  e_b = a_b - abar,
//   <ghat_b, g> = a_b^T K abar,  ||ghat_b||^2 = a_b^T K a_b,
//   E[ghat] - g = (E[a] - abar) S.
// K, abar and the quadratic forms are accumulated in fp64; the coefficients
// are the fp32 pair_coeffs_weighted values of each draw.
#include "pair_coeffs_dev.cuh"

namespace pairk {
namespace {

constexpr int kAuditBlocks = 4096;  // partial-sum slots (draw b -> block b mod grid), at most
constexpr int kAuditStats = 8;

// Deterministic block sum of one double per thread (all threads call).
__device__ double block_sum_double(double v, double *red) {
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[w] = v;
  __syncthreads();
  double s = 0.0;
  for (int k = 0; k < nw; ++k) s += red[k];
  return s;
}

// K[i][j] = sum_d S[i][d] S[j][d] in fp64; block i computes row i.
__global__ void audit_gram_kernel(int G, int D, const float *__restrict__ S, double *K) {
  __shared__ double red[32];
  const int i = blockIdx.x;
  const float *si = S + (size_t)i * D;
  for (int j = 0; j < G; ++j) {
    const float *sj = S + (size_t)j * D;
    double acc = 0.0;
    for (int d = threadIdx.x; d < D; d += blockDim.x) acc += (double)si[d] * (double)sj[d];
    const double t = block_sum_double(acc, red);
    if (threadIdx.x == 0) K[(size_t)i * G + j] = t;
  }
}

// abar, u = K abar and ||g||^2 = abar^T K abar (one block of >= G threads).
__global__ void audit_target_kernel(int G, const float *__restrict__ r, float scale,
                                    const double *__restrict__ K, double *abar, double *u,
                                    double *gg) {
  __shared__ double sa[128];
  __shared__ double red[32];
  const int i = threadIdx.x;
  if (i < G) {
    double s = 0.0;
    for (int j = 0; j < G; ++j) s += (double)r[i] - (double)r[j];
    sa[i] = (double)scale * 0.5 * s;
    abar[i] = sa[i];
  }
  __syncthreads();
  double ui = 0.0;
  if (i < G) {
    for (int j = 0; j < G; ++j) ui += K[(size_t)i * G + j] * sa[j];
    u[i] = ui;
  }
  const double t = block_sum_double(i < G ? sa[i] * ui : 0.0, red);
  if (i == 0) *gg = t;
}

template <int GP>
struct AuditSmem {
  GroupSmemW<GP> grp;
  double K[GP * GP];
  double abar[GP], u[GP], e[GP], a[GP];
  double red[32];
};

// Persistent: block q handles draws b = q, q + grid, ... in order and writes
// its partial sums [stats..., sum_b w_b a_b (G)] to part[q].
template <int GP>
__global__ void __launch_bounds__(GP, 1) audit_draws_kernel(
    int N, int G, const float *__restrict__ r, const float *__restrict__ rho,
    const uint8_t *__restrict__ Jd, const double *__restrict__ wd, float scale, int center,
    int wmode, float w_max, const double *__restrict__ K, const double *__restrict__ abar,
    const double *__restrict__ u, const double *__restrict__ gg_p, double *part,
    int32_t *dev_err) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  AuditSmem<GP> &sm = *reinterpret_cast<AuditSmem<GP> *>(smem_raw);
  const int tid = threadIdx.x;
  for (int k = tid; k < G * G; k += GP) {
    const int i = k / G, j = k % G;
    sm.K[i * GP + j] = K[k];
  }
  if (tid < GP) {
    const bool in = tid < G;
    sm.abar[tid] = in ? abar[tid] : 0.0;
    sm.u[tid] = in ? u[tid] : 0.0;
    sm.grp.r[tid] = in ? r[tid] : 0.f;
    sm.grp.pi[tid] = (in && wmode == PAIR_W_MARGINAL) ? rho[(size_t)tid * G + tid] : 1.f;
  }
  const double gg = *gg_p;
  // rho is the same for every draw: its triangle is read once per block.
  float v[GP / 2];
  load_upper<GP>(rho, G, weighting_reads_rho(wmode), v);
  double acc[6] = {0, 0, 0, 0, 0, 0};  // mse, cos, vertices, edges, ess, weight
  double a_acc = 0.0;
  for (int b = blockIdx.x; b < N; b += gridDim.x) {
    __syncthreads();
    sm.grp.J[tid] = (tid < G) ? (Jd[(size_t)b * G + tid] != 0) : 0;
    __syncthreads();
    const WeightedOut o =
        group_coeffs_w<GP>(sm.grp, v, G, scale, (uint32_t)center, wmode, w_max, dev_err);
    const double ai = (double)o.a;
    const double ei = ai - sm.abar[tid];
    sm.e[tid] = ei;
    sm.a[tid] = ai;
    __syncthreads();
    double Ke = 0.0;
    if (tid < G)
      for (int j = 0; j < G; ++j) Ke += sm.K[tid * GP + j] * sm.e[j];
    const double q_ee = block_sum_double(ei * Ke, sm.red);
    const double q_au = block_sum_double(ai * sm.u[tid], sm.red);
    const double q_aa = block_sum_double(ai * (Ke + sm.u[tid]), sm.red);
    const double w = wd ? wd[b] : 1.0 / (double)N;
    if (tid == 0) {
      const double cosb = (q_aa > 0.0 && gg > 0.0) ? q_au / sqrt(q_aa * gg) : 0.0;
      const double ess = o.W2 > 0.f ? (double)o.W * (double)o.W / (double)o.W2 : 0.0;
      acc[0] += w * q_ee;
      acc[1] += w * cosb;
      acc[2] += w * (double)o.K;
      acc[3] += w * (double)(o.K * (o.K - 1) / 2);
      acc[4] += w * ess;
      acc[5] += w;
    }
    a_acc += w * ai;
  }
  double *pq = part + (size_t)blockIdx.x * (kAuditStats + GP);
  if (tid == 0)
    for (int k = 0; k < 6; ++k) pq[k] = acc[k];
  if (tid < GP) pq[kAuditStats + tid] = a_acc;
}

// Sums the partials in block order, normalises by the total weight, and forms
// the bias E[a] - abar, its norm through K and (optionally) the vector (E[a] -
// abar) S. One block of 256 threads.
__global__ void audit_finish_kernel(int nblk, int G, int GP, int D, const float *__restrict__ S,
                                    const double *__restrict__ K, const double *__restrict__ abar,
                                    const double *__restrict__ gg_p,
                                    const double *__restrict__ part, double *stats, double *bias) {
  __shared__ double em[128];
  __shared__ double red[32];
  __shared__ double tot[6];
  const int tid = threadIdx.x;
  // Each column of the partials (6 statistics, then G coefficient sums) is
  // summed by every thread over a strided share of the blocks, then by the
  // block reduction: a fixed order, and the loads of a column in flight
  // together.
  for (int k = 0; k < 6 + G; ++k) {
    const int col = k < 6 ? k : kAuditStats + (k - 6);
    double s = 0.0;
    for (int q = tid; q < nblk; q += blockDim.x) s += part[(size_t)q * (kAuditStats + GP) + col];
    const double t = block_sum_double(s, red);
    if (tid == 0) {
      if (k < 6) tot[k] = t;
      else em[k - 6] = t;
    }
  }
  __syncthreads();
  const double W = tot[5];
  if (tid < G) em[tid] = (W > 0.0 ? em[tid] / W : 0.0) - abar[tid];
  __syncthreads();
  double Ke = 0.0;
  if (tid < G)
    for (int j = 0; j < G; ++j) Ke += K[(size_t)tid * G + j] * em[j];
  const double bb = block_sum_double(tid < G ? em[tid] * Ke : 0.0, red);
  if (tid == 0) {
    stats[0] = sqrt(bb > 0.0 ? bb : 0.0);
    for (int k = 0; k < 5; ++k) stats[1 + k] = W > 0.0 ? tot[k] / W : 0.0;
    stats[6] = *gg_p;
    stats[7] = W;
  }
  if (bias)
    for (int d = tid; d < D; d += blockDim.x) {
      double s = 0.0;
      for (int i = 0; i < G; ++i) s += em[i] * (double)S[(size_t)i * D + d];
      bias[d] = s;
    }
}

template <int GP>
pair_status launch_audit_gp(int N, int G, int D, const float *r, const float *rho,
                            const float *S, const uint8_t *Jd, const double *wd, float scale,
                            uint32_t flags, int wmode, float w_max, double *stats, double *bias,
                            double *ws, int32_t *dev_err, cudaStream_t s) {
  double *K = ws, *abar = K + (size_t)G * G, *u = abar + G, *gg = u + G;
  double *part = gg + 2;
  PAIR_BEGIN("audit_gram", s);
  audit_gram_kernel<<<G, 256, 0, s>>>(G, D, S, K);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("audit_target", s);
  audit_target_kernel<<<1, 128, 0, s>>>(G, r, scale, K, abar, u, gg);
  PAIR_LAUNCH_CHECK(s);
  // As many blocks as the SMs hold at once (the draws loop is latency bound,
  // one group per block), at most the kAuditBlocks partial slots.
  const size_t smem = sizeof(AuditSmem<GP>);
  PAIR_CUDA_TRY(cudaFuncSetAttribute(audit_draws_kernel<GP>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  int dev = 0, nsm = 0, per_sm = 0;
  PAIR_CUDA_TRY(cudaGetDevice(&dev));
  PAIR_CUDA_TRY(cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev));
  PAIR_CUDA_TRY(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, audit_draws_kernel<GP>, GP,
                                                              smem));
  int nblk = (nsm > 0 ? nsm : 1) * (per_sm > 0 ? per_sm : 1);
  if (nblk > kAuditBlocks) nblk = kAuditBlocks;
  if (nblk > N) nblk = N;
  PAIR_BEGIN("audit_draws", s);
  audit_draws_kernel<GP><<<nblk, GP, smem, s>>>(N, G, r, rho, Jd, wd, scale,
                                                (int)flags, wmode, w_max, K,
                                                abar, u, gg, part, dev_err);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("audit_finish", s);
  audit_finish_kernel<<<1, 256, 0, s>>>(nblk, G, GP, D, S, K, abar, gg, part, stats, bias);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

}  // namespace
}  // namespace pairk

using namespace pairk;

extern "C" size_t pair_audit_workspace_size(int32_t N, int32_t G, int32_t D) {
  if (N < 1 || G < 2 || G > PAIR_MAX_G || D < 1) return 0;
  const int GP = G <= 32 ? 32 : G <= 64 ? 64 : 128;
  const size_t nblk = N < kAuditBlocks ? (size_t)N : (size_t)kAuditBlocks;
  return sizeof(double) * ((size_t)G * G + 2 * (size_t)G + 2 + nblk * (kAuditStats + GP));
}

extern "C" pair_status pair_audit(int32_t N, int32_t G, int32_t D, const float *r,
                                  const float *rho, const float *S, const uint8_t *Jdraws,
                                  const double *draw_weight, float scale, uint32_t flags,
                                  pair_weighting wmode, float w_max, double *stats, double *bias,
                                  void *ws, size_t ws_bytes, int32_t *dev_err,
                                  pair_stream_t stream) {
  reset_launches();
  const size_t need = pair_audit_workspace_size(N, G, D);
  if (need == 0 || !r || !S || !Jdraws || !stats ||
      (flags & ~(PAIR_CENTER | PAIR_STANDARDIZE)) != 0)
    return PAIR_ERR_INVALID_ARG;
  const int wm = (int)wmode;
  if (wm < PAIR_W_HT || wm > PAIR_W_HAJEK) return PAIR_ERR_INVALID_ARG;
  if (wm != PAIR_W_UNWEIGHTED && !rho) return PAIR_ERR_INVALID_ARG;
  if (wm == PAIR_W_CLIPPED && !(w_max > 0.f && w_max <= 3.0e38f)) return PAIR_ERR_INVALID_ARG;
  if (!ws || ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 15u)) return PAIR_ERR_WORKSPACE;
  const pair_status dv = check_device();
  if (dv != PAIR_OK) return dv;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  double *w = static_cast<double *>(ws);
  if (G <= 32)
    return launch_audit_gp<32>(N, G, D, r, rho, S, Jdraws, draw_weight, scale, flags, wm, w_max,
                               stats, bias, w, dev_err, s);
  if (G <= 64)
    return launch_audit_gp<64>(N, G, D, r, rho, S, Jdraws, draw_weight, scale, flags, wm, w_max,
                               stats, bias, w, dev_err, s);
  return launch_audit_gp<128>(N, G, D, r, rho, S, Jdraws, draw_weight, scale, flags, wm, w_max,
                              stats, bias, w, dev_err, s);
}
