// Per-group coefficient collapse and the dense estimator.
//
// Sec. 4.5, Eq. (pair-advantage): a_i = scale * 1/2 sum_{j != i} J_iJ_j
// (r_i - r_j) / rho_ij, and Eq. (pair-ht) collapsed to g = sum_i a_i s_i.
// Algorithm 1 enumerates the observed induced edges; here every edge (i<j)
// is read once from the upper triangle of rho and its antisymmetric term is
// placed at (i, j) and (j, i) of a shared-memory matrix, after which each
// vertex sums its row with a fixed binary tree (deterministic, error
// O(log2 G) ulp of sum_j |term_j|).
//
// Memory: the upper triangle is read by "row pairs": rows k and GP-1-k
// together hold exactly GP-1 upper entries, so a block of >= GP threads reads
// them as two contiguous runs per step, fully unrolled to keep every load
// of the group in flight at once.
#include "pair_coeffs_stream.cuh"

namespace pairk {
namespace {

template <int GP>
struct GroupSmem {
  float U[GP * (GP - 1) / 2];  // strict upper triangle t_ij (i < j), row-major
  float r[GP];
  float a[GP];
  int8_t J[GP];
  int red_i[32];
  float red_f[32];
};

// Computes the coefficients of group `b` into sm.a[0..G) (scale applied).
// Requires blockDim.x >= GP. Returns K and the contrast count (all threads).
template <int GP>
__device__ void group_coeffs(GroupSmem<GP> &sm, int b, int G, const float *r,
                             const uint8_t *J, const float *rho, float scale,
                             bool center, int32_t *dev_err, int &K_out,
                             int &contrast_out, uint8_t &active_out) {
  const int tid = threadIdx.x;
  const size_t gbase = (size_t)b * G;
  const float *rho_g = rho + (size_t)b * G * G;
  // Load phase: every upper entry this thread owns, issued together with r
  // and J so the group pays one memory latency (the lines of the triangle
  // are fetched in any case; entries of edges that are not completed are
  // loaded but never used). Step k covers rows k (first GP-1-k threads) and
  // GP-1-k (the rest).
  float v[GP / 2];
  if (tid < GP - 1) {
#pragma unroll
    for (int k = 0; k < GP / 2; ++k) {
      const int n1 = GP - 1 - k;
      int i, j;
      if (tid < n1) { i = k; j = k + 1 + tid; }
      else { i = GP - 1 - k; j = i + 1 + (tid - n1); }
      v[k] = (j < G) ? __ldg(rho_g + (size_t)i * G + j) : 1.f;
    }
  }
  if (tid < GP) {
    const bool in = tid < G;
    sm.r[tid] = in ? r[gbase + tid] : 0.f;
    sm.J[tid] = in ? (J[gbase + tid] != 0) : 0;
  }
  __syncthreads();

  int my_contrast = 0, bad = 0;
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
        const float rij = v[k];
        if (!(rij > 0.f)) {
          bad = 1;
        } else {
          t = __fdiv_rn(sm.r[i] - sm.r[j], rij);
          my_contrast += (sm.r[i] != sm.r[j]);
        }
      }
      sm.U[upper_off<GP>(i, j)] = t;
    }
  }
  if (bad) flag_error(dev_err, PAIR_DEV_ERR_NONPOSITIVE_INCLUSION);
  __syncthreads();

  // Row sum of the antisymmetric terms by a fixed pairwise tree, streamed:
  // partial p[l] holds the sum of the last complete block of 2^l terms.
  float a = 0.f;
  uint8_t act = 0;
  if (tid < GP) {
    float p[8];
    bool nz = false;
#pragma unroll
    for (int k = 0; k < GP; ++k) {
      float x = 0.f;
      if (k < tid) x = -sm.U[upper_off<GP>(k, tid)];
      else if (k > tid) x = sm.U[upper_off<GP>(tid, k)];
      nz |= (x != 0.f);
      float c = x;
      int m = k;
#pragma unroll
      for (int l = 0; l < 8; ++l) {
        if (m & 1) { c = p[l] + c; m >>= 1; }
        else { p[l] = c; break; }
      }
    }
    // GP is a power of two: the final carry landed in p[log2 GP].
    const float sum = p[(GP == 32) ? 5 : (GP == 64) ? 6 : 7];
    a = (sum == 0.f) ? 0.f : 0.5f * sum;
    act = (tid < G && sm.J[tid] && nz) ? 1 : 0;
  }
  // K (low 16 bits) and contrast edges (high bits) in one reduction.
  const int packed = block_sum_int(((tid < GP) ? (int)sm.J[tid] : 0) | (my_contrast << 16),
                                   sm.red_i);
  const int K = packed & 0xffff, C = packed >> 16;
  if (center && K > 0) {
    // App. C: centre across the observed endpoints.
    const float s = block_sum_float((tid < GP && sm.J[tid]) ? a : 0.f, sm.red_f);
    const float mean = s / (float)K;
    if (tid < GP && sm.J[tid]) a -= mean;
  }
  if (tid < GP) sm.a[tid] = (tid < G) ? a * scale : 0.f;
  __syncthreads();
  K_out = K;
  contrast_out = C;
  active_out = act;
}

template <int GP>
__global__ void __launch_bounds__(GP, 1024 / GP) coeffs_kernel(
    int B, int G, const float *__restrict__ r, const uint8_t *__restrict__ J,
    const float *__restrict__ rho, float scale, int center,
    float *__restrict__ a, uint8_t *__restrict__ active,
    int32_t *__restrict__ edges, int32_t *__restrict__ contrast,
    int32_t *dev_err) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  GroupSmem<GP> &sm = *reinterpret_cast<GroupSmem<GP> *>(smem_raw);
  const int b = blockIdx.x;
  int K, C;
  uint8_t act;
  group_coeffs<GP>(sm, b, G, r, J, rho, scale, center != 0, dev_err, K, C, act);
  const int tid = threadIdx.x;
  if (tid < G) {
    a[(size_t)b * G + tid] = sm.a[tid];
    if (active) active[(size_t)b * G + tid] = act;
  }
  if (tid == 0) {
    if (edges) edges[b] = K * (K - 1) / 2;
    if (contrast) contrast[b] = C;
  }
}

// g_b = sum_i a_i s_{b,i} for one group, given its coefficients a_s[0..G) in
// shared memory (block-wide call): the nonzero coefficients are listed, then
// S is streamed over D with 16-byte loads; rows with a_i == 0 are never read.
template <int GP>
__device__ __forceinline__ void dense_rows(int b, int G, int D, const float *a_s,
                                           const float *__restrict__ S,
                                           float *__restrict__ g) {
  __shared__ int rows[GP];
  __shared__ float coef[GP];
  __shared__ int n_rows;
  const int tid = threadIdx.x;
  if (tid == 0) {
    int n = 0;
    for (int i = 0; i < G; ++i)
      if (a_s[i] != 0.f) { rows[n] = i; coef[n] = a_s[i]; ++n; }
    n_rows = n;
  }
  __syncthreads();
  const int n = n_rows;
  const float *Sb = S + (size_t)b * G * D;
  float *gb = g + (size_t)b * D;
  const bool vec = ((D & 3) == 0) && ((reinterpret_cast<uintptr_t>(S) & 15) == 0) &&
                   ((reinterpret_cast<uintptr_t>(g) & 15) == 0);
  if (vec) {
    const int D4 = D >> 2;
    for (int c0 = tid; c0 < D4; c0 += 4 * blockDim.x) {
      float4 acc[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) acc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      int q = 0;
      for (; q + 1 < n; q += 2) {
        float4 x0[4], x1[4];
        const float4 *p0 = reinterpret_cast<const float4 *>(Sb + (size_t)rows[q] * D);
        const float4 *p1 = reinterpret_cast<const float4 *>(Sb + (size_t)rows[q + 1] * D);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int c = c0 + u * blockDim.x;
          x0[u] = c < D4 ? __ldcs(p0 + c) : make_float4(0.f, 0.f, 0.f, 0.f);
          x1[u] = c < D4 ? __ldcs(p1 + c) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        const float w0 = coef[q], w1 = coef[q + 1];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          acc[u].x = fmaf(w0, x0[u].x, acc[u].x); acc[u].y = fmaf(w0, x0[u].y, acc[u].y);
          acc[u].z = fmaf(w0, x0[u].z, acc[u].z); acc[u].w = fmaf(w0, x0[u].w, acc[u].w);
          acc[u].x = fmaf(w1, x1[u].x, acc[u].x); acc[u].y = fmaf(w1, x1[u].y, acc[u].y);
          acc[u].z = fmaf(w1, x1[u].z, acc[u].z); acc[u].w = fmaf(w1, x1[u].w, acc[u].w);
        }
      }
      if (q < n) {
        const float4 *p0 = reinterpret_cast<const float4 *>(Sb + (size_t)rows[q] * D);
        const float w0 = coef[q];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int c = c0 + u * blockDim.x;
          if (c < D4) {
            const float4 x = __ldcs(p0 + c);
            acc[u].x = fmaf(w0, x.x, acc[u].x); acc[u].y = fmaf(w0, x.y, acc[u].y);
            acc[u].z = fmaf(w0, x.z, acc[u].z); acc[u].w = fmaf(w0, x.w, acc[u].w);
          }
        }
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int c = c0 + u * blockDim.x;
        if (c < D4) __stcs(reinterpret_cast<float4 *>(gb) + c, acc[u]);
      }
    }
  } else {
    for (int c = tid; c < D; c += blockDim.x) {
      float acc = 0.f;
      for (int q = 0; q < n; ++q) acc = fmaf(coef[q], Sb[(size_t)rows[q] * D + c], acc);
      gb[c] = acc;
    }
  }
}

// One block per group: coefficients (general form), then dense_rows.
template <int GP>
__global__ void __launch_bounds__(256, 4) dense_kernel(
    int B, int G, int D, const float *__restrict__ r,
    const uint8_t *__restrict__ J, const float *__restrict__ rho,
    const float *__restrict__ S, float scale, float *__restrict__ g,
    float *__restrict__ a_out, int32_t *dev_err) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  GroupSmem<GP> &sm = *reinterpret_cast<GroupSmem<GP> *>(smem_raw);
  const int b = blockIdx.x, tid = threadIdx.x;
  int K, C;
  uint8_t act;
  group_coeffs<GP>(sm, b, G, r, J, rho, scale, false, dev_err, K, C, act);
  if (a_out && tid < G) a_out[(size_t)b * G + tid] = sm.a[tid];
  dense_rows<GP>(b, G, D, sm.a, S, g);
}

// The same for groups the streaming coefficient kernel takes (G <= 64, G a
// multiple of 4, aligned inputs): warp 0 stages the group and collapses it
// with warp_group_coeffs, so the coefficients are bit-identical to
// pair_coeffs'.
struct DenseStagedSmem {
  int Qt[kGMax];
  float a[kGMax];
  __align__(16) unsigned char stage[kStageBytes];
  __align__(16) unsigned char aux[kWarpAux];
};

__global__ void __launch_bounds__(256, 4) dense_staged_kernel(
    int B, int G, int D, const float *__restrict__ r, const uint8_t *__restrict__ J,
    const float *__restrict__ rho, const float *__restrict__ S, float scale,
    float *__restrict__ g, float *__restrict__ a_out, int32_t *dev_err, const StreamGeom geom) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  DenseStagedSmem &sm = *reinterpret_cast<DenseStagedSmem *>(smem_raw);
  const int b = blockIdx.x, tid = threadIdx.x;
  stream_qt(geom, sm.Qt);
  __syncthreads();
  if (tid < 32) {
    uint64_t *bar = reinterpret_cast<uint64_t *>(sm.aux + 64 * 4 * 3);
    volatile int *abort = reinterpret_cast<volatile int *>(bar + 2);
    stream_init_gaps(sm.stage, G, sm.Qt);
    if (tid == 0) {
      tc::mbar_init(bar, 1);
      *abort = 0;
      tc::fence_mbar_init();
    }
    __syncwarp();
    issue_group(sm.stage, bar, rho, r, load_j_word(J, b, B, G), b, G,
                stream_rows(G, sm.Qt, geom.group_bytes));
    const bool ok = __all_sync(0xffffffffu, tc::wait(bar, 0u, abort, dev_err));
    if (!ok) drain_wait(bar, 0u);
    __syncwarp();
    WarpCoeffs o = {};
    if (ok)
      o = warp_group_coeffs<PAIR_W_HT, false>(sm.stage, sm.Qt, stream_diag(G, sm.Qt), G, scale,
                                              0u, 0.f, sm.aux, dev_err);
    sm.a[tid] = o.a0;
    sm.a[tid + 32] = o.a1;
  }
  __syncthreads();
  if (a_out && tid < G) a_out[(size_t)b * G + tid] = sm.a[tid];
  dense_rows<kGMax>(b, G, D, sm.a, S, g);
}

// Coefficients under a weighting variant (see pair_coeffs_weighted), plus
// the ESS and largest weight of the group's completed edges. One block of GP
// threads per group.
template <int GP>
__global__ void __launch_bounds__(GP, 1024 / GP) coeffs_w_kernel(
    int B, int G, const float *__restrict__ r, const uint8_t *__restrict__ J,
    const float *__restrict__ rho, float scale, int center, int wmode, float w_max,
    float *__restrict__ a, uint8_t *__restrict__ active, int32_t *__restrict__ edges,
    int32_t *__restrict__ contrast, float *__restrict__ ess, float *__restrict__ max_w,
    int32_t *dev_err) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  GroupSmemW<GP> &sm = *reinterpret_cast<GroupSmemW<GP> *>(smem_raw);
  const int b = blockIdx.x, tid = threadIdx.x;
  const size_t gbase = (size_t)b * G;
  const float *rho_g = rho + (size_t)b * G * G;
  float v[GP / 2];
  load_upper<GP>(rho_g, G, weighting_reads_rho(wmode), v);
  {
    const bool in = tid < G;
    sm.r[tid] = in ? r[gbase + tid] : 0.f;
    sm.J[tid] = in ? (J[gbase + tid] != 0) : 0;
    sm.pi[tid] = (in && wmode == PAIR_W_MARGINAL) ? rho_g[(size_t)tid * G + tid] : 1.f;
  }
  __syncthreads();
  const WeightedOut o = group_coeffs_w<GP>(sm, v, G, scale, (uint32_t)center, wmode, w_max,
                                           dev_err);
  if (tid < G) {
    a[gbase + tid] = o.a;
    if (active) active[gbase + tid] = o.active;
  }
  if (tid == 0) {
    if (edges) edges[b] = o.K * (o.K - 1) / 2;
    if (contrast) contrast[b] = o.C;
    if (ess) ess[b] = o.W2 > 0.f ? __fdiv_rn(o.W * o.W, o.W2) : 0.f;
    if (max_w) max_w[b] = o.Wmax;
  }
}

// Independent (product) design: rho_ij = p_i p_j, so the coefficients need
// only the marginals p [B][G]: a_i = 1/2 (J_i / p_i) sum_{j != i} J_j
// (r_i - r_j) / p_j, summed per vertex by the fixed pairwise tree (the same
// terms as the joint form, without reading a G x G matrix).
template <int GP>
__global__ void __launch_bounds__(GP, 4) coeffs_product_kernel(
    int B, int G, const float *__restrict__ r, const uint8_t *__restrict__ J,
    const float *__restrict__ p, float scale, int center, float *__restrict__ a,
    uint8_t *__restrict__ active, int32_t *__restrict__ edges, int32_t *__restrict__ contrast,
    float *__restrict__ ess, float *__restrict__ max_w, int32_t *dev_err) {
  __shared__ float sr[GP], sq[GP];
  __shared__ int8_t sJ[GP];
  __shared__ int red_i[32];
  __shared__ float red_f[32];
  const int b = blockIdx.x, tid = threadIdx.x;
  const size_t gbase = (size_t)b * G;
  int bad = 0;
  {
    const bool in = tid < G;
    const bool j = in && J[gbase + tid] != 0;
    const float pv = in ? p[gbase + tid] : 1.f;
    if (j && !(pv > 0.f)) bad = 1;
    sr[tid] = in ? r[gbase + tid] : 0.f;
    sJ[tid] = (j && pv > 0.f) ? 1 : 0;
    sq[tid] = (j && pv > 0.f) ? __frcp_rn(pv) : 0.f;
  }
  if (bad) flag_error(dev_err, PAIR_DEV_ERR_NONPOSITIVE_INCLUSION);
  __syncthreads();
  PairwiseSum<GP> ps;
  bool nz = false;
  int my_contrast = 0;
  float sw = 0.f, sw2 = 0.f, mw = 0.f;
  const float ri = sr[tid], qi = sq[tid];
  const bool Ji = sJ[tid] != 0;
#pragma unroll
  for (int k = 0; k < GP; ++k) {
    const float x = (k != tid && Ji && sJ[k]) ? (ri - sr[k]) * sq[k] : 0.f;
    nz |= (x != 0.f);
    ps.add(k, x);
    if (k > tid && Ji && sJ[k]) {
      const float w = qi * sq[k];
      sw += w;
      sw2 = fmaf(w, w, sw2);
      mw = fmaxf(mw, w);
      my_contrast += (ri != sr[k]);
    }
  }
  const float sum = ps.total();
  float av = (sum == 0.f) ? 0.f : 0.5f * qi * sum;
  const float W = block_sum_float(sw, red_f);
  const float W2 = block_sum_float(sw2, red_f);
  const float Wmax = block_max_float(mw, red_f);
  const int packed = block_sum_int((int)sJ[tid] | (my_contrast << 16), red_i);
  const int K = packed & 0xffff, C = packed >> 16;
  if (center & PAIR_STANDARDIZE) av = standardize_by_rewards(av, ri, Ji, K, red_f);
  if ((center & PAIR_CENTER) && K > 0) {
    const float s2 = block_sum_float(Ji ? av : 0.f, red_f);
    const float mean = s2 / (float)K;
    if (Ji) av -= mean;
  }
  if (tid < G) {
    a[gbase + tid] = av * scale;
    if (active) active[gbase + tid] = (Ji && nz) ? 1 : 0;
  }
  if (tid == 0) {
    if (edges) edges[b] = K * (K - 1) / 2;
    if (contrast) contrast[b] = C;
    if (ess) ess[b] = W2 > 0.f ? __fdiv_rn(W * W, W2) : 0.f;
    if (max_w) max_w[b] = Wmax;
  }
}

template <int GP>
pair_status launch_coeffs_w_gp(int32_t B, int32_t G, const float *r, const uint8_t *J,
                               const float *rho, float scale, uint32_t flags, int wmode,
                               float w_max, float *a, uint8_t *active, int32_t *edges,
                               int32_t *contrast, float *ess, float *max_w, int32_t *dev_err,
                               cudaStream_t s) {
  const size_t smem = sizeof(GroupSmemW<GP>);
  PAIR_CUDA_TRY(cudaFuncSetAttribute(coeffs_w_kernel<GP>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  PAIR_BEGIN("coeffs_w", s);
  coeffs_w_kernel<GP><<<B, GP, smem, s>>>(B, G, r, J, rho, scale, (int)flags, wmode, w_max, a,
                                          active, edges, contrast, ess, max_w, dev_err);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

// Product design for G <= 64: one warp per group. Lane c holds vertices c
// and c + 32; the completed ones are packed (vertex order) into the warp's
// shared lists of r and q = 1/p (IEEE reciprocal, as the block form), and
// each completed vertex i sums its terms (r_i - r_j) q_j over every packed
// partner (its own slot adds an exact 0) in a fixed order: four interleaved
// partial sums combined pairwise. a_i = 1/2 q_i sum; the weight diagnostics
// sum q_i q_j over the pairs i < j of packed slots.
template <bool DIAG>
__global__ void __launch_bounds__(128) coeffs_product_warp_kernel(
    int B, int G, const float *__restrict__ r, const uint8_t *__restrict__ J,
    const float *__restrict__ p, float scale, uint32_t flags, float *__restrict__ a,
    uint8_t *__restrict__ active, int32_t *__restrict__ edges, int32_t *__restrict__ contrast,
    float *__restrict__ ess, float *__restrict__ max_w, int32_t *dev_err) {
  __shared__ float pr[4][64], pq[4][64];
  const int lane = threadIdx.x & 31, wi = threadIdx.x >> 5;
  const int b = blockIdx.x * 4 + wi;
  if (b >= B) return;  // warp-uniform; the warps of a block never synchronise
  const size_t gb = (size_t)b * G;
  float rv[2], qv[2];
  bool cv[2];
  int bad = 0;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int v = lane + 32 * h;
    const bool in = v < G;
    const bool j = in && J[gb + v] != 0;
    const float pv = in ? p[gb + v] : 1.f;
    if (j && !(pv > 0.f)) bad = 1;
    cv[h] = j && pv > 0.f;
    rv[h] = in ? r[gb + v] : 0.f;
    qv[h] = cv[h] ? __frcp_rn(pv) : 0.f;
  }
  if (__any_sync(0xffffffffu, bad) && lane == 0)
    flag_error(dev_err, PAIR_DEV_ERR_NONPOSITIVE_INCLUSION);
  const unsigned m0 = __ballot_sync(0xffffffffu, cv[0]), m1 = __ballot_sync(0xffffffffu, cv[1]);
  const unsigned lt = (1u << lane) - 1u;
  const int K0 = __popc(m0), K = K0 + __popc(m1);
  const int slot[2] = {__popc(m0 & lt), K0 + __popc(m1 & lt)};
#pragma unroll
  for (int h = 0; h < 2; ++h)
    if (cv[h]) {
      pr[wi][slot[h]] = rv[h];
      pq[wi][slot[h]] = qv[h];
    }
  __syncwarp();
  float av[2] = {0.f, 0.f};
  int diff[2] = {0, 0};
  float sw = 0.f, sw2 = 0.f, mw = 0.f;
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    if (!cv[h]) continue;
    float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
    int nd = 0;
    int kk = 0;
    for (; kk + 4 <= K; kk += 4) {
      const float r0 = pr[wi][kk], r1 = pr[wi][kk + 1], r2 = pr[wi][kk + 2], r3 = pr[wi][kk + 3];
      s0 += (rv[h] - r0) * pq[wi][kk];
      s1 += (rv[h] - r1) * pq[wi][kk + 1];
      s2 += (rv[h] - r2) * pq[wi][kk + 2];
      s3 += (rv[h] - r3) * pq[wi][kk + 3];
      nd += (r0 != rv[h]) + (r1 != rv[h]) + (r2 != rv[h]) + (r3 != rv[h]);
    }
    for (; kk < K; ++kk) {
      const float rk = pr[wi][kk];
      const float x = (rv[h] - rk) * pq[wi][kk];
      if ((kk & 3) == 0) s0 += x; else if ((kk & 3) == 1) s1 += x; else s2 += x;
      nd += rk != rv[h];
    }
    const float sum = (s0 + s1) + (s2 + s3);
    av[h] = (sum == 0.f) ? 0.f : 0.5f * qv[h] * sum;
    diff[h] = nd;
    if (DIAG)
      for (int k2 = slot[h] + 1; k2 < K; ++k2) {
        const float w = qv[h] * pq[wi][k2];
        sw += w;
        sw2 = fmaf(w, w, sw2);
        mw = fmaxf(mw, w);
      }
  }
  if ((flags & PAIR_STANDARDIZE) && K >= 2) {
    // Sample standard deviation (n - 1) of the completed rewards, two-pass.
    const float mean = warp_sum((cv[0] ? rv[0] : 0.f) + (cv[1] ? rv[1] : 0.f)) / (float)K;
    const float d0 = cv[0] ? rv[0] - mean : 0.f, d1 = cv[1] ? rv[1] - mean : 0.f;
    const float sd = sqrtf(warp_sum(d0 * d0 + d1 * d1) / (float)(K - 1));
    av[0] = sd > 0.f ? __fdiv_rn(av[0], sd) : 0.f;
    av[1] = sd > 0.f ? __fdiv_rn(av[1], sd) : 0.f;
  }
  if ((flags & PAIR_CENTER) && K > 0) {
    const float mean = warp_sum(av[0] + av[1]) / (float)K;
    if (cv[0]) av[0] -= mean;
    if (cv[1]) av[1] -= mean;
  }
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int v = lane + 32 * h;
    if (v < G) {
      a[gb + v] = av[h] * scale;
      if (active) active[gb + v] = (cv[h] && diff[h] > 0) ? 1 : 0;
    }
  }
  int nd_all = diff[0] + diff[1];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) nd_all += __shfl_xor_sync(0xffffffffu, nd_all, o);
  float W = 0.f, W2 = 0.f, Wmax = 0.f;
  if (DIAG) {
    W = warp_sum(sw);
    W2 = warp_sum(sw2);
    Wmax = warp_max(mw);
  }
  if (lane == 0) {
    if (edges) edges[b] = K * (K - 1) / 2;
    if (contrast) contrast[b] = nd_all / 2;
    if (DIAG) {
      if (ess) ess[b] = W2 > 0.f ? __fdiv_rn(W * W, W2) : 0.f;
      if (max_w) max_w[b] = Wmax;
    }
  }
}

template <int GP>
pair_status launch_coeffs_product_gp(int32_t B, int32_t G, const float *r, const uint8_t *J,
                                     const float *p, float scale, uint32_t flags, float *a,
                                     uint8_t *active, int32_t *edges, int32_t *contrast,
                                     float *ess, float *max_w, int32_t *dev_err, cudaStream_t s) {
  PAIR_BEGIN("coeffs_product", s);
  coeffs_product_kernel<GP><<<B, GP, 0, s>>>(B, G, r, J, p, scale, (int)flags, a, active, edges,
                                             contrast, ess, max_w, dev_err);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

template <int GP>
pair_status launch_coeffs_gp(int32_t B, int32_t G, const float *r,
                             const uint8_t *J, const float *rho, float scale,
                             uint32_t flags, float *a, uint8_t *active,
                             int32_t *edges, int32_t *contrast,
                             int32_t *dev_err, cudaStream_t s) {
  const size_t smem = sizeof(GroupSmem<GP>);
  PAIR_CUDA_TRY(cudaFuncSetAttribute(coeffs_kernel<GP>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)smem));
  PAIR_BEGIN("coeffs", s);
  coeffs_kernel<GP><<<B, GP, smem, s>>>(B, G, r, J, rho, scale,
                                        (flags & PAIR_CENTER) ? 1 : 0, a,
                                        active, edges, contrast, dev_err);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

template <int GP>
pair_status launch_dense_gp(int32_t B, int32_t G, int32_t D, const float *r,
                            const uint8_t *J, const float *rho, const float *S,
                            float scale, float *g, float *a, int32_t *dev_err,
                            cudaStream_t s) {
  const size_t smem = sizeof(GroupSmem<GP>);
  PAIR_CUDA_TRY(cudaFuncSetAttribute(dense_kernel<GP>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)smem));
  PAIR_BEGIN("dense", s);
  dense_kernel<GP><<<B, 256, smem, s>>>(B, G, D, r, J, rho, S, scale, g, a,
                                        dev_err);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

}  // namespace

pair_status launch_coeffs(int32_t B, int32_t G, const float *r,
                          const uint8_t *J, const float *rho, float scale,
                          uint32_t flags, float *a, uint8_t *active,
                          int32_t *edges, int32_t *contrast, int32_t *dev_err,
                          cudaStream_t s) {
  if (coeffs_stream_applies(G, r, J, rho))
    return launch_coeffs_stream(B, G, r, J, rho, scale, flags, PAIR_W_HT, false, 0.f, a, active,
                                edges, contrast, nullptr, nullptr, dev_err, s);
  if (flags & PAIR_STANDARDIZE)  // HT through the weighted kernel (bit-identical HT terms)
    return launch_coeffs_weighted(B, G, r, J, rho, scale, flags, PAIR_W_HT, 0.f, a, active, edges,
                                  contrast, nullptr, nullptr, dev_err, s);
  if (G <= 32)
    return launch_coeffs_gp<32>(B, G, r, J, rho, scale, flags, a, active,
                                edges, contrast, dev_err, s);
  if (G <= 64)
    return launch_coeffs_gp<64>(B, G, r, J, rho, scale, flags, a, active,
                                edges, contrast, dev_err, s);
  return launch_coeffs_gp<128>(B, G, r, J, rho, scale, flags, a, active,
                               edges, contrast, dev_err, s);
}

pair_status launch_coeffs_weighted(int32_t B, int32_t G, const float *r, const uint8_t *J,
                                   const float *rho, float scale, uint32_t flags, int wmode,
                                   float w_max, float *a, uint8_t *active, int32_t *edges,
                                   int32_t *contrast, float *ess, float *max_w,
                                   int32_t *dev_err, cudaStream_t s) {
  if ((wmode == PAIR_W_HT || wmode == PAIR_W_CLIPPED || wmode == PAIR_W_HAJEK) &&
      coeffs_stream_applies(G, r, J, rho))
    return launch_coeffs_stream(B, G, r, J, rho, scale, flags, wmode, true, w_max, a, active,
                                edges, contrast, ess, max_w, dev_err, s);
  if (G <= 32)
    return launch_coeffs_w_gp<32>(B, G, r, J, rho, scale, flags, wmode, w_max, a, active, edges,
                                  contrast, ess, max_w, dev_err, s);
  if (G <= 64)
    return launch_coeffs_w_gp<64>(B, G, r, J, rho, scale, flags, wmode, w_max, a, active, edges,
                                  contrast, ess, max_w, dev_err, s);
  return launch_coeffs_w_gp<128>(B, G, r, J, rho, scale, flags, wmode, w_max, a, active, edges,
                                 contrast, ess, max_w, dev_err, s);
}

pair_status launch_coeffs_product(int32_t B, int32_t G, const float *r, const uint8_t *J,
                                  const float *p, float scale, uint32_t flags, float *a,
                                  uint8_t *active, int32_t *edges, int32_t *contrast, float *ess,
                                  float *max_w, int32_t *dev_err, cudaStream_t s) {
  if (G <= 64) {
    const int blocks = (int)ceil_div(B, 4);
    PAIR_BEGIN("coeffs_product", s);
    if (ess || max_w)
      coeffs_product_warp_kernel<true><<<blocks, 128, 0, s>>>(
          B, G, r, J, p, scale, flags, a, active, edges, contrast, ess, max_w, dev_err);
    else
      coeffs_product_warp_kernel<false><<<blocks, 128, 0, s>>>(
          B, G, r, J, p, scale, flags, a, active, edges, contrast, ess, max_w, dev_err);
    PAIR_LAUNCH_CHECK(s);
    return PAIR_OK;
  }
  return launch_coeffs_product_gp<128>(B, G, r, J, p, scale, flags, a, active, edges, contrast,
                                       ess, max_w, dev_err, s);
}

pair_status launch_estimate_dense(int32_t B, int32_t G, int32_t D,
                                  const float *r, const uint8_t *J,
                                  const float *rho, const float *S,
                                  float scale, float *g, float *a,
                                  int32_t *dev_err, cudaStream_t s) {
  if (coeffs_stream_applies(G, r, J, rho)) {
    const size_t smem = sizeof(DenseStagedSmem);
    PAIR_CUDA_TRY(cudaFuncSetAttribute(dense_staged_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    PAIR_BEGIN("dense", s);
    dense_staged_kernel<<<B, 256, smem, s>>>(B, G, D, r, J, rho, S, scale, g, a, dev_err,
                                              make_stream_geom(G));
    PAIR_LAUNCH_CHECK(s);
    return PAIR_OK;
  }
  if (G <= 32)
    return launch_dense_gp<32>(B, G, D, r, J, rho, S, scale, g, a, dev_err, s);
  if (G <= 64)
    return launch_dense_gp<64>(B, G, D, r, J, rho, S, scale, g, a, dev_err, s);
  return launch_dense_gp<128>(B, G, D, r, J, rho, S, scale, g, a, dev_err, s);
}

}  // namespace pairk
