// pair_allocate: the allocation step before the path (Sec. 4.3-4.4). For
// every group, the contrast graph (Eq. disagreement / Eq. edge-proxy), the
// shared-vertex surrogate b_i (Sec. 4.4) and the continuation probabilities
// of the convex program of Eqs. (convex-objective)-(budget):
//     min_x  Phi(x) = sum_{i<j} a_ij e^(x_i + x_j) + sum_i b_i e^(x_i)
//     s.t.   sum_i c_i e^(-x_i) <= budget,   0 <= x_i <= -log pi_min,
// with pi_i = e^(-x_i).
//
// Solver (one CTA per group, fp64): a log-barrier path-following method,
//     F_t(x) = t Phi(x) - log(budget - sum c e^-x) - sum log x_i - sum log(X - x_i),
// Newton steps on F_t (gradient and Hessian in closed form, the G x G system
// factorised by Cholesky in shared memory, backtracking line search kept
// strictly feasible), t multiplied by 32 (G <= 24) or 16 after each centring,
// with a predictor step along the central path's tangent from the factor of
// the centred point, until the duality-gap bound (2G + 1) / t is below
// 1e-12 Phi. The paper solves the
// same program with SLSQP on the CPU (App. C); any method reaching its
// unique optimum is equivalent, and a barrier method maps onto one CTA with
// a fixed, small number of dense factorisations. Cases the program leaves
// without an interior (budget >= sum c: pi = 1; budget = pi_min sum c:
// pi = pi_min; budget below that: infeasible) and the flat objective (all
// a_ij = b_i = 0) are classified first, from the fp64 sum of c in index
// order. If Newton does not converge within its iteration cap, the group
// falls back to the uniform pi = budget / sum c of the same expected cost
// (the paper's fallback).
#include <math.h>
#include <stdint.h>

#include "pair_common.cuh"

namespace pairk {
namespace {

constexpr int kAllocMaxNewton = 600;    // total Newton steps per group
constexpr int kAllocMaxBacktrack = 80;  // halvings per line search
constexpr double kGapRel = 1e-12;       // stop at (2G + 1) / t <= kGapRel * Phi
// Barrier parameter growth per centring: 32 for groups of up to 24 (fewer
// Newton steps in all: about 59 against 66 per group of 16), 16 above (at 64,
// 32 costs more steps than it saves).
__host__ __device__ constexpr double barrier_growth(int G) { return G <= 24 ? 32.0 : 16.0; }
// Newton decrement^2 / 2 of a centred point. lambda^2 / 2 bounds F_t - min F_t,
// so centring adds at most about lambda^2 / t to Phi, far below the gap
// bound (2G + 1) / t >= 5 / t; a tighter threshold only adds Newton steps
// (on 64 groups of 16, 1e-6 takes about 68 steps per group and 1e-3 about
// 65, with pi as close to the KKT point).
constexpr double kCentred = 1e-3;
// A line search stops once the decrease its step could bring, step * lambda^2,
// is below this many fp64 units of |F_t|: such a decrease cannot be told from
// rounding, so halving further only repeats function evaluations (the point
// is then treated as centred, as after a failed search).
constexpr double kResolution = 16.0 * 2.220446049250313e-16;

// Groups of up to 64 keep the edge proxies a_ij in shared memory (fp64, as
// computed on the fly otherwise); the 128-candidate form has no room for them.
template <int GP>
constexpr bool kEdgeTable = GP <= 64;

template <int GP>
struct AllocSmem {
  double H[GP][GP + 1];  // Newton system, factorised in place (lower triangle)
  double A[kEdgeTable<GP> ? GP : 1][kEdgeTable<GP> ? GP + 1 : 1];  // a_ij (see kEdgeTable)
  double c[GP], b[GP], dx[GP];
  double dinv[GP];       // 1 / L_kk of the current factorisation
  float p[GP], m[GP];
  double red[GP / 32];
  double sum_c;
  int any;
};

// Sum over the CTA (all GP threads call it; returns the total to every thread).
template <int GP>
__device__ double block_sum(AllocSmem<GP> &sm, double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) sm.red[threadIdx.x >> 5] = v;
  __syncthreads();
  double t = 0.0;
#pragma unroll
  for (int w = 0; w < GP / 32; ++w) t += sm.red[w];
  return t;
}

// Solves H y = r in place in sm.dx with the Cholesky factor in sm.H (lower
// triangle) and the pivot inverses in sm.dinv (all GP threads call; thread i
// holds r_i on entry and reads y_i after the call).
template <int GP>
__device__ void chol_solve(AllocSmem<GP> &sm, int G, bool act, double r) {
  const int i = threadIdx.x;
  __syncthreads();
  sm.dx[i] = act ? r : 0.0;
  for (int k = 0; k < G; ++k) {
    __syncthreads();
    if (i == k) sm.dx[k] *= sm.dinv[k];
    __syncthreads();
    if (i > k && act) sm.dx[i] -= sm.H[i][k] * sm.dx[k];
  }
  for (int k = G - 1; k >= 0; --k) {
    __syncthreads();
    if (i == k) sm.dx[k] *= sm.dinv[k];
    __syncthreads();
    if (i < k) sm.dx[i] -= sm.H[k][i] * sm.dx[k];
  }
  __syncthreads();
}

// Largest step along d keeping every coordinate strictly inside the box
// (0, X), shared by all threads (min over the group, 1e300 if unbounded).
template <int GP>
__device__ double box_step(AllocSmem<GP> &sm, int G, bool act, double x, double d, double X) {
  double smax = 1.0e300;
  if (act && d < 0.0) smax = -x / d;
  if (act && d > 0.0) smax = (X - x) / d;
  __syncthreads();
  sm.dx[threadIdx.x] = smax;
  __syncthreads();
  if (threadIdx.x == 0) {
    double mn = 1.0e300;
    for (int k = 0; k < G; ++k) mn = fmin(mn, sm.dx[k]);
    sm.red[0] = mn;
  }
  __syncthreads();
  const double r = sm.red[0];
  __syncthreads();
  return r;
}

struct AllocIn {
  int G;
  const float *p_hat, *m_hat, *a;
  int g;
};

// Edge proxy a_ij: the explicit array, else Eq. (disagreement) from p_hat,
// times ((m_i + m_j) / 2)^2 with score-norm predictions (Eq. edge-proxy).
template <int GP>
__device__ __forceinline__ double edge(const AllocIn &in, const AllocSmem<GP> &sm, int i,
                                       int j) {
  if (i == j) return 0.0;
  if (in.a) return (double)in.a[((size_t)in.g * in.G + i) * in.G + j];
  const double pi = sm.p[i], pj = sm.p[j];
  double d = pi * (1.0 - pj) + (1.0 - pi) * pj;
  if (in.m_hat) {
    const double h = 0.5 * ((double)sm.m[i] + (double)sm.m[j]);
    d *= h * h;
  }
  return d;
}

// a_ij from the table where there is one (same fp64 value as edge()).
template <int GP>
__device__ __forceinline__ double edge_at(const AllocIn &in, const AllocSmem<GP> &sm, int i,
                                          int j) {
  if constexpr (kEdgeTable<GP>) return sm.A[i][j];
  else return edge<GP>(in, sm, i, j);
}

// Phi, the budget slack and this coordinate's S_i = sum_j a_ij u_j at x_i
// (u_i = e^x_i held by thread i, shared through sm.dx as scratch).
template <int GP>
__device__ void eval(const AllocIn &in, AllocSmem<GP> &sm, bool act, double x, double budget,
                     double &u, double &e, double &S, double &phi, double &slack) {
  u = act ? exp(x) : 0.0;
  e = act ? sm.c[threadIdx.x] / u : 0.0;  // c e^-x without a second exp
  __syncthreads();
  sm.dx[threadIdx.x] = u;
  __syncthreads();
  S = 0.0;
  if (act)
    for (int j = 0; j < in.G; ++j) S += edge_at<GP>(in, sm, threadIdx.x, j) * sm.dx[j];
  phi = block_sum<GP>(sm, act ? u * (0.5 * S + sm.b[threadIdx.x]) : 0.0);
  slack = budget - block_sum<GP>(sm, e);
}

template <int GP>
__global__ void __launch_bounds__(GP, 1) alloc_kernel(int G, const float *p_hat, const float *m_hat,
                                                   const float *a, const float *c_hat,
                                                   const float *budget_in, float pi_min,
                                                   float *pi_out, double *stats,
                                                   int32_t *dev_err) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  AllocSmem<GP> &sm = *reinterpret_cast<AllocSmem<GP> *>(smem_raw);
  const int i = threadIdx.x, g = blockIdx.x;
  const bool act = i < G;
  const AllocIn in{G, p_hat, m_hat, a, g};

  // ---- inputs and their validity
  bool bad = false;
  double ci = 1.0;
  if (act) {
    ci = (double)c_hat[(size_t)g * G + i];
    bad |= !(ci > 0.0 && ci <= 3.0e38);
    if (!a) {
      const float pf = p_hat[(size_t)g * G + i];
      bad |= !(pf >= 0.f && pf <= 1.f);
      sm.p[i] = pf;
      if (m_hat) {
        const float mf = m_hat[(size_t)g * G + i];
        bad |= !(mf >= 0.f && mf <= 3.0e38f);
        sm.m[i] = mf;
      }
    } else {
      for (int j = 0; j < G; ++j) {
        const float v = a[((size_t)g * G + i) * G + j];
        bad |= (j != i) && !(v >= 0.f && v <= 3.0e38f);
      }
    }
  }
  sm.c[i] = act ? ci : 0.0;
  const double budget = (double)budget_in[g];
  bad |= !(budget > 0.0 && budget <= 3.0e38);
  if (i == 0) sm.any = 0;
  __syncthreads();
  if (bad) atomicOr(&sm.any, 1);
  // The sum of c in index order (the classification is bit-identical to a
  // sequential fp64 sum on the host).
  if (i == 0) {
    double s = 0.0;
    for (int k = 0; k < G; ++k) s += sm.c[k];
    sm.sum_c = s;
  }
  __syncthreads();
  const bool invalid = sm.any != 0;
  const double sc = sm.sum_c, pmin = (double)pi_min, X = -log(pmin);
  if constexpr (kEdgeTable<GP>) {
    if (act && !invalid)
      for (int j = 0; j < G; ++j) sm.A[i][j] = edge<GP>(in, sm, i, j);
    __syncthreads();
  }

  // ---- b_i = (sum_{j != i} sqrt a_ij)^2 - sum_{j != i} a_ij
  double bi = 0.0, asum = 0.0;
  if (act && !invalid) {
    double sq = 0.0;
    for (int j = 0; j < G; ++j) {
      const double v = edge_at<GP>(in, sm, i, j);
      sq += sqrt(v);
      asum += v;
    }
    bi = sq * sq - asum;
  }
  sm.b[i] = bi;
  __syncthreads();
  const bool flat = block_sum<GP>(sm, asum + bi) == 0.0;

  int status;
  if (invalid) status = PAIR_ALLOC_INVALID;
  else if (budget >= sc) status = PAIR_ALLOC_SLACK;
  else if (budget == pmin * sc) status = PAIR_ALLOC_FLOOR;
  else if (budget < pmin * sc) status = PAIR_ALLOC_INFEASIBLE;
  else if (flat) status = PAIR_ALLOC_FLAT;
  else status = PAIR_ALLOC_OK;

  double x = 0.0, t = 0.0, gap = 0.0;
  int newton = 0;
  if (status == PAIR_ALLOC_SLACK) {
    x = 0.0;
  } else if (status == PAIR_ALLOC_FLOOR || status == PAIR_ALLOC_INFEASIBLE) {
    x = X;
  } else if (status == PAIR_ALLOC_FLAT) {
    x = -log(budget / sc);
  } else if (status == PAIR_ALLOC_OK) {
    const int m = 2 * G + 1;
    const double tmul = barrier_growth(G);
    x = -log(0.5 * (budget / sc + pmin));  // strictly feasible start
    double u, e, S, phi, slack;
    eval<GP>(in, sm, act, x, budget, u, e, S, phi, slack);
    t = (double)m / phi;
    bool done = false;
    while (newton < kAllocMaxNewton && !done) {
      ++newton;
      // Gradient and Hessian of F_t at x.
      // 1/x and 1/(X - x) from one division; 1/slack once per step.
      const double rr = act ? 1.0 / (x * (X - x)) : 0.0;
      const double bnd_lo = act ? (X - x) * rr : 0.0, bnd_hi = act ? x * rr : 0.0;
      const double inv_s = 1.0 / slack;
      const double gi =
          act ? t * u * (S + sm.b[i]) - e * inv_s - bnd_lo + bnd_hi : 0.0;
      // u_j and e_j for the Hessian rows (e_j in H's spare column).
      __syncthreads();
      sm.dx[i] = u;
      if (act) sm.H[i][GP] = e;
      __syncthreads();
      if (act) {
        const double inv_s2 = inv_s * inv_s;
        for (int j = 0; j <= i; ++j) {
          double h = e * sm.H[j][GP] * inv_s2;
          if (j == i)
            h += t * u * (S + sm.b[i]) + e * inv_s + bnd_lo * bnd_lo + bnd_hi * bnd_hi;
          else
            h += t * edge_at<GP>(in, sm, i, j) * u * sm.dx[j];
          sm.H[i][j] = h;
        }
      }
      // Cholesky (lower triangle, in place); each pivot's inverse is formed
      // once, so the column scaling and both substitutions multiply. One
      // reciprocal square root per pivot gives both 1/L_kk and L_kk = d/sqrt(d).
      bool spd = true;
      for (int k = 0; k < G; ++k) {
        __syncthreads();
        if (i == k) {
          const double d = sm.H[k][k];
          const double rs = d > 0.0 ? rsqrt(d) : 0.0;
          sm.H[k][k] = d * rs;
          sm.dinv[k] = rs;
        }
        __syncthreads();
        if (sm.H[k][k] == 0.0) spd = false;
        if (!spd) break;
        if (i > k && act) sm.H[i][k] *= sm.dinv[k];
        __syncthreads();
        if (i > k && act) {
          const double lik = sm.H[i][k];
          for (int j = k + 1; j <= i; ++j) sm.H[i][j] -= lik * sm.H[j][k];
        }
      }
      if (!spd) break;
      // Solve H dx = -g (forward, then backward substitution).
      chol_solve<GP>(sm, G, act, -gi);
      const double d = act ? sm.dx[i] : 0.0;
      const double lam2 = -block_sum<GP>(sm, gi * d);
      if (lam2 * 0.5 <= kCentred) {
        // Centred: stop once the gap bound is small, else raise t.
        if ((double)m / t <= kGapRel * phi) {
          done = true;
          break;
        }
        // Predictor: the central path x*(t) has grad F_t = 0, so
        // dx*/dt = -H^-1 grad Phi with the Hessian just factorised; move
        // along it to the next t (kept strictly inside the box and the
        // budget, halving the step otherwise), then let Newton correct.
        chol_solve<GP>(sm, G, act, act ? -u * (S + sm.b[i]) : 0.0);
        const double v = act ? (tmul - 1.0) * t * sm.dx[i] : 0.0;
        double pstep = fmin(1.0, 0.99 * box_step<GP>(sm, G, act, x, v, X));
        for (int ls = 0; ls < 8; ++ls) {
          const double xt = x + pstep * v;
          double ut, et, St, phit, slackt;
          eval<GP>(in, sm, act, xt, budget, ut, et, St, phit, slackt);
          // slackt is the same in every thread: the exit is uniform.
          if (slackt > 0.0) {
            x = xt; u = ut; e = et; S = St; phi = phit; slack = slackt;
            break;
          }
          pstep *= 0.5;
        }
        t *= tmul;
        continue;
      }
      // Largest step keeping every coordinate strictly inside the box.
      double step = fmin(1.0, 0.99 * box_step<GP>(sm, G, act, x, d, X));
      const double F0 = t * phi - log(slack) -
                        block_sum<GP>(sm, act ? log(x * (X - x)) : 0.0);
      bool moved = false;
      for (int ls = 0; ls < kAllocMaxBacktrack; ++ls) {
        // step, lam2 and F0 are the same in every thread: the exit is uniform.
        if (step * lam2 < kResolution * fabs(F0)) break;
        const double xt = x + step * d;
        double ut, et, St, phit, slackt;
        eval<GP>(in, sm, act, xt, budget, ut, et, St, phit, slackt);
        bool ok = slackt > 0.0;
        if (ok) {
          const double Ft = t * phit - log(slackt) -
                            block_sum<GP>(sm, act ? log(xt * (X - xt)) : 0.0);
          // Strict decrease as well: at fp64 resolution of F_t a step can
          // pass Armijo without changing anything.
          ok = Ft < F0 && Ft <= F0 - 0.01 * step * lam2;
        }
        if (ok) {
          x = xt; u = ut; e = et; S = St; phi = phit; slack = slackt;
          moved = true;
          break;
        }
        step *= 0.5;
      }
      if (!moved) {
        // No descent at fp64 resolution: the point is as centred as it gets.
        if ((double)m / t <= kGapRel * phi) {
          done = true;
          break;
        }
        t *= tmul;
      }
    }
    gap = (double)m / t;
    if (!done) {
      status = PAIR_ALLOC_FALLBACK;
      x = -log(budget / sc);
    }
  }

  // ---- outputs
  double u_out = 0.0, e_out = 0.0, S_out = 0.0, phi_out = 0.0, slack_out = 0.0;
  if (status != PAIR_ALLOC_INVALID)
    eval<GP>(in, sm, act, x, budget, u_out, e_out, S_out, phi_out, slack_out);
  if (act)
    pi_out[(size_t)g * G + i] = status == PAIR_ALLOC_INVALID ? __int_as_float(0x7fc00000)
                                                             : (float)exp(-x);
  if (i == 0) {
    if (status == PAIR_ALLOC_INVALID) atomicOr(dev_err, PAIR_DEV_ERR_ALLOC_INPUT);
    if (status == PAIR_ALLOC_INFEASIBLE) atomicOr(dev_err, PAIR_DEV_ERR_ALLOC_INFEASIBLE);
    if (stats) {
      double *st = stats + (size_t)g * PAIR_ALLOC_NSTATS;
      st[PAIR_ALLOC_PHI] = status == PAIR_ALLOC_INVALID ? 0.0 : phi_out;
      st[PAIR_ALLOC_SPENT] = status == PAIR_ALLOC_INVALID ? 0.0 : budget - slack_out;
      st[PAIR_ALLOC_GAP] = gap;
      st[PAIR_ALLOC_NEWTON] = (double)newton;
      st[PAIR_ALLOC_STATUS] = (double)status;
    }
  }
}

template <int GP>
pair_status launch_alloc(int32_t B, int32_t G, const float *p_hat, const float *m_hat,
                         const float *a, const float *c_hat, const float *budget, float pi_min,
                         float *pi, double *stats, int32_t *dev_err, cudaStream_t s) {
  const size_t smem = sizeof(AllocSmem<GP>);
  PAIR_CUDA_TRY(cudaFuncSetAttribute(alloc_kernel<GP>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  PAIR_BEGIN("allocate", s);
  alloc_kernel<GP><<<B, GP, smem, s>>>(G, p_hat, m_hat, a, c_hat, budget, pi_min, pi, stats,
                                       dev_err);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

}  // namespace
}  // namespace pairk

using namespace pairk;

extern "C" pair_status pair_allocate(int32_t B, int32_t G, const float *p_hat,
                                     const float *m_hat, const float *a, const float *c_hat,
                                     const float *budget, float pi_min, float *pi,
                                     double *stats, int32_t *dev_err, pair_stream_t stream) {
  reset_launches();
  if (B < 1 || G < 2 || G > PAIR_MAX_G || !c_hat || !budget || !pi || !dev_err)
    return PAIR_ERR_INVALID_ARG;
  if (!a && !p_hat) return PAIR_ERR_INVALID_ARG;
  if (!(pi_min > 0.f && pi_min <= 1.f)) return PAIR_ERR_INVALID_ARG;
  const pair_status dv = check_device();
  if (dv != PAIR_OK) return dv;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (G <= 32)
    return launch_alloc<32>(B, G, p_hat, m_hat, a, c_hat, budget, pi_min, pi, stats, dev_err, s);
  if (G <= 64)
    return launch_alloc<64>(B, G, p_hat, m_hat, a, c_hat, budget, pi_min, pi, stats, dev_err, s);
  return launch_alloc<128>(B, G, p_hat, m_hat, a, c_hat, budget, pi_min, pi, stats, dev_err, s);
}
