// Device building blocks of the group coefficient kernels, shared by
// pair_coeffs.cu and pair_audit.cu: deterministic block reductions, the fixed
// pairwise tree, and the weighted coefficients of one group.
#pragma once

#include "pair_common.cuh"

namespace pairk {
namespace {

// Row-major offset of (i, j), i < j, in the packed strict upper triangle.
template <int GP>
__device__ __forceinline__ int upper_off(int i, int j) {
  return i * (2 * GP - i - 1) / 2 + (j - i - 1);
}

// Deterministic block sum of one int per thread (all threads call).
__device__ int block_sum_int(int v, int *red) {
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[w] = v;
  __syncthreads();
  int s = 0;
  for (int k = 0; k < nw; ++k) s += red[k];
  return s;
}

// Deterministic block sum of one float per thread in a fixed tree order.
__device__ float block_sum_float(float v, float *red) {
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[w] = v;
  __syncthreads();
  float s = 0.f;
  for (int k = 0; k < nw; ++k) s += red[k];
  return s;
}

// Deterministic block maximum of one float per thread (all threads call).
__device__ float block_max_float(float v, float *red) {
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  const int w = threadIdx.x >> 5, nw = (blockDim.x + 31) >> 5;
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[w] = v;
  __syncthreads();
  float m = 0.f;
  for (int k = 0; k < nw; ++k) m = fmaxf(m, red[k]);
  return m;
}

// Sum of the 2^l-blocked pairwise tree over x_0 .. x_{GP-1} (the same fixed
// order the HT kernel uses for its row sums).
template <int GP>
struct PairwiseSum {
  float p[8];
  __device__ __forceinline__ void add(int k, float x) {
    float c = x;
    int m = k;
#pragma unroll
    for (int l = 0; l < 8; ++l) {
      if (m & 1) { c = p[l] + c; m >>= 1; }
      else { p[l] = c; break; }
    }
  }
  __device__ __forceinline__ float total() const { return p[(GP == 32) ? 5 : (GP == 64) ? 6 : 7]; }
};

template <int GP>
struct GroupSmemW {
  float U[GP * (GP - 1) / 2];  // strict upper triangle of terms (r_i - r_j) w_ij
  float r[GP];
  float pi[GP];                // marginals (rho diagonal) or 1/p (product path)
  int8_t J[GP];
  int red_i[32];
  float red_f[32];
};

// Reward standardisation (App. "Practical departures"): v divided by the
// sample standard deviation (n - 1) of the completed rewards, two-pass. With
// fewer than two completed vertices or equal rewards there is no contrast
// edge and v is already 0. All threads call.
__device__ __forceinline__ float standardize_by_rewards(float v, float r, bool completed, int K,
                                                       float *red) {
  if (K < 2) return v;
  const float mean = block_sum_float(completed ? r : 0.f, red) / (float)K;
  const float dv = completed ? r - mean : 0.f;
  const float ss = block_sum_float(dv * dv, red);
  const float sd = sqrtf(ss / (float)(K - 1));
  return sd > 0.f ? __fdiv_rn(v, sd) : 0.f;
}

// Result of one group's weighted coefficients (per thread: its vertex).
struct WeightedOut {
  float a;          // this vertex's coefficient (scale applied)
  uint8_t active;
  int K, C;         // completed vertices, contrast edges
  float W, W2, Wmax;  // sum, sum of squares and max of the completed-edge weights
};

// The upper-triangle entries of rho_g that thread tid owns, read by row
// pairs (step k covers rows k and GP-1-k), all loads in flight at once; every
// entry with j < G is loaded (its line is fetched anyway), so the loads need
// not wait for J. Entries of edges that are not completed are never used.
template <int GP>
__device__ __forceinline__ void load_upper(const float *rho_g, int G, bool needs_rho,
                                           float (&v)[GP / 2]) {
  const int tid = threadIdx.x;
#pragma unroll
  for (int k = 0; k < GP / 2; ++k) {
    const int n1 = GP - 1 - k;
    int i, j;
    if (tid < n1) { i = k; j = k + 1 + tid; }
    else { i = GP - 1 - k; j = i + 1 + (tid - n1); }
    v[k] = (needs_rho && tid < GP - 1 && j < G) ? __ldg(rho_g + (size_t)i * G + j) : 1.f;
  }
}

__device__ __forceinline__ bool weighting_reads_rho(int wmode) {
  return wmode == PAIR_W_HT || wmode == PAIR_W_CLIPPED || wmode == PAIR_W_HAJEK;
}

// Coefficients of one group under a weighting variant (see
// pair_coeffs_weighted), from the entries load_upper fetched. The caller has
// placed r, J (and, for the marginal weighting, the marginals) in shared
// memory. Every term is placed once, every vertex summed by the fixed
// pairwise tree. All GP threads call.
template <int GP>
__device__ WeightedOut group_coeffs_w(GroupSmemW<GP> &sm, const float (&v)[GP / 2], int G,
                                      float scale, uint32_t flags, int wmode, float w_max,
                                      int32_t *dev_err) {
  const int tid = threadIdx.x;
  int my_contrast = 0, bad = 0;
  float sw = 0.f, sw2 = 0.f, mw = 0.f;
  if (tid < GP - 1) {
#pragma unroll
    for (int k = 0; k < GP / 2; ++k) {
      const int n1 = GP - 1 - k;
      int i, j;
      if (tid < n1) { i = k; j = k + 1 + tid; }
      else { i = GP - 1 - k; j = i + 1 + (tid - n1); }
      const bool live = (j < G) && sm.J[i] && sm.J[j];
      float t = 0.f;
      if (live) {
        const float dr = sm.r[i] - sm.r[j];
        float w = 1.f;
        bool okw = true;
        if (wmode == PAIR_W_UNWEIGHTED) {
          t = dr;
        } else if (wmode == PAIR_W_MARGINAL) {
          const float pi = sm.pi[i], pj = sm.pi[j];
          okw = (pi > 0.f) && (pj > 0.f);
          const float den = pi * pj;
          t = okw ? __fdiv_rn(dr, den) : 0.f;
          w = okw ? __frcp_rn(den) : 0.f;
        } else {
          const float rij = v[k];
          okw = rij > 0.f;
          w = okw ? __frcp_rn(rij) : 0.f;
          if (wmode == PAIR_W_CLIPPED && w > w_max) {
            w = w_max;
            t = dr * w_max;
          } else {
            t = okw ? __fdiv_rn(dr, rij) : 0.f;
          }
        }
        if (!okw) {
          bad = 1;
        } else {
          my_contrast += (sm.r[i] != sm.r[j]);
          sw += w;
          sw2 = fmaf(w, w, sw2);
          mw = fmaxf(mw, w);
        }
      }
      sm.U[upper_off<GP>(i, j)] = t;
    }
  }
  if (bad) flag_error(dev_err, PAIR_DEV_ERR_NONPOSITIVE_INCLUSION);
  WeightedOut o;
  o.W = block_sum_float(sw, sm.red_f);
  o.W2 = block_sum_float(sw2, sm.red_f);
  o.Wmax = block_max_float(mw, sm.red_f);
  __syncthreads();

  PairwiseSum<GP> ps;
  bool nz = false;
#pragma unroll
  for (int k = 0; k < GP; ++k) {
    float x = 0.f;
    if (k < tid) x = -sm.U[upper_off<GP>(k, tid)];
    else if (k > tid) x = sm.U[upper_off<GP>(tid, k)];
    nz |= (x != 0.f);
    ps.add(k, x);
  }
  const float sum = ps.total();
  float av = (sum == 0.f) ? 0.f : 0.5f * sum;
  if (wmode == PAIR_W_HAJEK) av = o.W > 0.f ? __fdiv_rn(av, o.W) : 0.f;
  o.active = (tid < G && sm.J[tid] && nz) ? 1 : 0;
  const int packed = block_sum_int((int)sm.J[tid] | (my_contrast << 16), sm.red_i);
  o.K = packed & 0xffff;
  o.C = packed >> 16;
  if (flags & PAIR_STANDARDIZE) av = standardize_by_rewards(av, sm.r[tid], sm.J[tid] != 0, o.K,
                                                           sm.red_f);
  if ((flags & PAIR_CENTER) && o.K > 0) {
    const float s2 = block_sum_float(sm.J[tid] ? av : 0.f, sm.red_f);
    const float mean = s2 / (float)o.K;
    if (sm.J[tid]) av -= mean;
  }
  o.a = (tid < G) ? av * scale : 0.f;
  __syncthreads();  // U is reused by the caller's next group
  return o;
}

}  // namespace
}  // namespace pairk
