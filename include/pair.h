/*
 * pair.h -- C ABI of the GB300 (sm_103a) hot path of the Pair estimator
 * (Pairwise-Aware Inclusion Reweighting for adaptive rollout allocation).
 *
 * Problem statement (Sec. 3): a prompt has G candidate rollouts with
 * verifiable rewards r_i and sequence scores s_i = d log pi(o_i|q) / d theta.
 * An adaptive continuation design completes rollout i iff J_i = 1; the
 * sampler logs the joint inclusion probabilities rho_ij = P(J_i = J_j = 1)
 * > 0 (Sec. 3.3). With the pair kernel h_ij = 1/2 (r_i - r_j)(s_i - s_j)
 * (Sec. 3.2, Eq. pair-kernel) the design-unbiased estimator is
 *     g = (1/M) sum_{i<j} J_i J_j h_ij / rho_ij,      M = C(G, 2)
 * (Sec. 4.5, Eq. pair-ht), which collapses to g = sum_i A_i s_i with
 *     A_i = 1/(2M) sum_{j != i} J_i J_j (r_i - r_j) / rho_ij
 * (Eq. pair-advantage); the policy is updated through the objective
 * sum_i A_i log pi(o_i | q) (Sec. 4.5, Algorithm 1).
 *
 * Normalisation: every entry point takes `scale`. The coefficient computed
 * is a_i = scale * 1/2 sum_{j != i} J_i J_j (r_i - r_j) / rho_ij, so
 * scale = 1 gives the plain completed-edge sum and scale = 1/C(G,2) gives
 * the paper's A_i (M counts all G candidates, not the completed ones).
 *
 * Conventions shared by all calls:
 *  - All array pointers are caller-owned DEVICE memory unless stated.
 *    Outputs are overwritten (never accumulated). The library never
 *    allocates, frees or synchronises inside a compute call; every call is
 *    asynchronous on `stream` (0 = legacy default stream).
 *  - Row-major layouts; group b, candidate i is element b*G + i.
 *  - rho [B][G][G] float32: only the strict upper triangle (i < j) is read;
 *    the diagonal and lower triangle are ignored (rho is symmetric by
 *    definition, Sec. 3.3).
 *  - Host-detected argument errors return immediately, before any launch.
 *  - Device-detected data errors (rho_ij <= 0 or NaN on a completed edge;
 *    a target id outside [0, V) at a mask = 1 token) never trap: the kernel
 *    finishes, the affected outputs are unspecified, and a bit is OR-ed into
 *    the caller's device word `dev_err`, which `pair_status_sync` decodes.
 *  - Requires a compute capability 10.3 device (GB300). Other devices get
 *    PAIR_ERR_UNSUPPORTED.
 *  - Single-GPU library: every call runs on the current device only, and
 *    every array it is given must live on that device. The tensor-core head
 *    kernels (the log-sum-exp pass and the two backward GEMMs) run one MMA
 *    per pair of CTAs of a 2-CTA cluster; their tensor maps cover only the
 *    caller's buffers and the workspace on the current device, never another
 *    GPU's memory, and no kernel issues TMA multicast loads. A multi-GPU
 *    trainer runs one independent call per GPU (whole prompt groups per GPU)
 *    and does its own exchange of dW outside the library.
 */
#ifndef PAIR_H_
#define PAIR_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define PAIR_API __attribute__((visibility("default")))
#else
#define PAIR_API
#endif

/* Opaque CUDA stream handle (a cudaStream_t). */
typedef struct CUstream_st *pair_stream_t;

typedef enum {
  PAIR_OK = 0,
  PAIR_ERR_INVALID_ARG = 1,           /* null pointer, bad size or layout   */
  PAIR_ERR_UNSUPPORTED = 2,           /* device or shape not supported      */
  PAIR_ERR_WORKSPACE = 3,             /* workspace missing or too small     */
  PAIR_ERR_NONPOSITIVE_INCLUSION = 4, /* rho_ij <= 0 or NaN, completed edge */
  PAIR_ERR_TARGET_RANGE = 5,          /* y_t outside [0, V) at a mask=1 token */
  PAIR_ERR_CUDA = 6,                  /* a CUDA runtime call failed         */
  PAIR_ERR_DEVICE_TIMEOUT = 7,        /* a bounded on-device wait gave up;
                                         outputs of that call are invalid  */
  PAIR_ERR_ALLOC_INPUT = 8,           /* pair_allocate: invalid input value */
  PAIR_ERR_ALLOC_INFEASIBLE = 9       /* pair_allocate: budget < pi_min sum c */
} pair_status;

typedef enum { PAIR_F32 = 0, PAIR_BF16 = 1 } pair_dtype;

/* Bits of the device error word written by the kernels. */
#define PAIR_DEV_ERR_NONPOSITIVE_INCLUSION 1
#define PAIR_DEV_ERR_TARGET_RANGE 2
#define PAIR_DEV_ERR_TIMEOUT 4 /* a pipeline wait exceeded its limit (~2 s) */
#define PAIR_DEV_ERR_ALLOC_INPUT 8       /* pair_allocate: invalid input value */
#define PAIR_DEV_ERR_ALLOC_INFEASIBLE 16 /* pair_allocate: budget < pi_min sum c */

/* pair_coeffs flags. */
#define PAIR_CENTER 1u /* subtract the mean of a over completed vertices
                          (App. C, numerical stability). Off by default:
                          in exact arithmetic the sum is already zero. */
#define PAIR_STANDARDIZE 2u /* divide the coefficients of each group by the
                          sample standard deviation (n - 1) of its completed
                          rewards (the practical reward standardisation of
                          App. "Practical departures"; biased, see there).
                          Groups with equal completed rewards stay 0. */

/* Largest group size G accepted by pair_coeffs / pair_estimate_dense. */
#define PAIR_MAX_G 128

/*
 * pair_coeffs -- per-rollout coefficients of Eq. (pair-advantage) and the
 * observed-edge bookkeeping of Algorithm 1 (enumerate induced edges,
 * accumulate each edge term into both endpoints).
 *
 * In:  B >= 1 groups of G candidates, 2 <= G <= PAIR_MAX_G.
 *      r      [B][G] float32  rewards (any real value; binary in RLVR).
 *      J      [B][G] uint8    completion indicators (0 or nonzero).
 *      rho    [B][G][G] float32 logged joint inclusion probabilities.
 *      scale  multiplies every coefficient (see the header comment).
 *      flags  0 or PAIR_CENTER | PAIR_STANDARDIZE.
 * Out: a      [B][G] float32  a_i = scale * 1/2 sum_{j != i} J_iJ_j
 *                             (r_i - r_j)/rho_ij; exactly 0 where J_i = 0
 *                             or no completed partner has another reward.
 *      active [B][G] uint8    1 iff J_i = 1 and some completed j != i has
 *                             r_j != r_i (nullable).
 *      edges  [B] int32       number of observed edges C(K_b, 2),
 *                             K_b = sum_i J_i (nullable).
 *      contrast_edges [B] int32 observed edges with r_i != r_j (nullable).
 *      dev_err: device int32 error word (nullable; if null, device data
 *               errors are not reported).
 * Arithmetic: fp32, fixed-order tree summation over the partners;
 * deterministic (bit-identical reruns). For G <= 64 with G a multiple of 4
 * and 16-byte aligned r and rho (4-byte aligned J) each term is
 * (r_i - r_j) times the hardware reciprocal of rho_ij (within 1.5 ulp of the
 * quotient; exactly 0 when r_i = r_j and exactly antisymmetric), and a rho
 * below 2^-126 on a completed edge is reported like rho <= 0; otherwise the
 * term is the IEEE quotient. Either way the error of a_i is a few ulp of
 * 1/2 sum_j |term_j|.
 */
PAIR_API pair_status pair_coeffs(int32_t B, int32_t G, const float *r, const uint8_t *J,
                        const float *rho, float scale, uint32_t flags,
                        float *a, uint8_t *active, int32_t *edges,
                        int32_t *contrast_edges, int32_t *dev_err,
                        pair_stream_t stream);

/*
 * Edge weightings of pair_coeffs_weighted (App. "Estimated and stabilized
 * propensities"; the ablation variants of Sec. 5). For a completed edge
 * (i, j) the coefficient term is 1/2 (r_i - r_j) w_ij with
 *   PAIR_W_HT          w = 1/rho_ij                  (Eq. pair-ht; exact)
 *   PAIR_W_UNWEIGHTED  w = 1                         (no pair correction)
 *   PAIR_W_MARGINAL    w = 1/(pi_i pi_j), pi_i = rho_ii (marginal-only)
 *   PAIR_W_CLIPPED     w = min(1/rho_ij, w_max)
 *   PAIR_W_HAJEK       w = 1/rho_ij, and the group's coefficients divided by
 *                      the sum of w over its completed edges (self-normalised
 *                      ratio form; 0 when there is no completed edge).
 * Only PAIR_W_HT is unbiased for the complete-pair target (Thm. 2); the
 * others are the paper's biased comparison variants.
 */
typedef enum {
  PAIR_W_HT = 0,
  PAIR_W_UNWEIGHTED = 1,
  PAIR_W_MARGINAL = 2,
  PAIR_W_CLIPPED = 3,
  PAIR_W_HAJEK = 4
} pair_weighting;

/*
 * pair_coeffs_weighted -- pair_coeffs under a weighting variant, with the
 * per-group diagnostics of App. D: ESS = (sum_e w_e)^2 / sum_e w_e^2 and the
 * largest weight over the completed edges (both 0 without one).
 *
 * In:  as pair_coeffs, plus wmode (pair_weighting) and w_max (> 0 and finite
 *      for PAIR_W_CLIPPED, ignored otherwise). rho's strict upper triangle
 *      is read for the joint probabilities (not at all for
 *      PAIR_W_UNWEIGHTED); its diagonal only for PAIR_W_MARGINAL.
 *      PAIR_CENTER centres after the weighting (and the Hajek division).
 * Out: a, active, edges, contrast_edges as pair_coeffs (active and the edge
 *      counts do not depend on the weighting);
 *      ess [B], max_w [B] float32 (nullable).
 * Errors: PAIR_ERR_INVALID_ARG for the pair_coeffs conditions, an unknown
 *      wmode, or a non-positive / non-finite w_max with PAIR_W_CLIPPED;
 *      device: rho_ij <= 0 or NaN on a completed edge (pi_i, pi_j for
 *      PAIR_W_MARGINAL) -> PAIR_DEV_ERR_NONPOSITIVE_INCLUSION.
 * Arithmetic: fp32, fixed tree sums; the weights of HT, clipped and
 * self-normalised weighting as pair_coeffs' terms (the hardware reciprocal
 * where pair_coeffs uses it, IEEE division and reciprocal otherwise).
 */
PAIR_API pair_status pair_coeffs_weighted(int32_t B, int32_t G, const float *r,
                                          const uint8_t *J, const float *rho, float scale,
                                          uint32_t flags, pair_weighting wmode, float w_max,
                                          float *a, uint8_t *active, int32_t *edges,
                                          int32_t *contrast_edges, float *ess, float *max_w,
                                          int32_t *dev_err, pair_stream_t stream);

/*
 * pair_coeffs_product -- the coefficients of pair_coeffs for the independent
 * (product) design, rho_ij = p_i p_j (Sec. 4: independent Bernoulli
 * continuation), from the marginals alone:
 *     a_i = scale * 1/2 (J_i / p_i) sum_{j != i} J_j (r_i - r_j) / p_j,
 * reading 9 bytes per candidate instead of a G x G matrix per group.
 *
 * In:  r, J as pair_coeffs; p [B][G] float32 marginal inclusion probabilities
 *      (read where J_i = 1); scale, flags as pair_coeffs.
 * Out: a, active, edges, contrast_edges as pair_coeffs; ess, max_w as
 *      pair_coeffs_weighted for the weights 1/(p_i p_j) (nullable).
 * Errors: as pair_coeffs; device: p_i <= 0 or NaN where J_i = 1 ->
 *      PAIR_DEV_ERR_NONPOSITIVE_INCLUSION.
 */
PAIR_API pair_status pair_coeffs_product(int32_t B, int32_t G, const float *r,
                                         const uint8_t *J, const float *p, float scale,
                                         uint32_t flags, float *a, uint8_t *active,
                                         int32_t *edges, int32_t *contrast_edges, float *ess,
                                         float *max_w, int32_t *dev_err,
                                         pair_stream_t stream);

/*
 * pair_audit -- the frozen-population estimator audit (Sec. 5; metrics of
 * App. D) of one candidate group: r [G], rho [G][G] (as pair_coeffs_weighted),
 * explicit scores S [G][D], and N design draws Jdraws [N][G] (uint8). Each
 * draw's estimate is ghat_b = sum_i a_bi s_i with a_b the
 * pair_coeffs_weighted coefficients of that draw (wmode, w_max, scale,
 * flags); the target is the complete-pair gradient g = scale * sum_{i<j}
 * h_ij over all G candidates (Eq. pair-kernel). With draw weights w_b
 * (draw_weight [N] double, nullable = 1/N each; e.g. exact design
 * probabilities of an enumeration) and W = sum_b w_b, stats [8] (double) gets
 *   [PAIR_AUDIT_BIAS_NORM]  || sum_b w_b ghat_b / W - g ||
 *   [PAIR_AUDIT_MSE]        sum_b w_b || ghat_b - g ||^2 / W
 *   [PAIR_AUDIT_COS]        sum_b w_b cos(ghat_b, g) / W (0 where ghat_b = 0)
 *   [PAIR_AUDIT_VERTICES]   mean completed vertices, [PAIR_AUDIT_EDGES] mean
 *                           completed edges, [PAIR_AUDIT_ESS] mean ESS
 *   [PAIR_AUDIT_TARGET_SQ]  || g ||^2,  [PAIR_AUDIT_WEIGHT] W
 * and bias [D] (double, nullable) the vector sum_b w_b ghat_b / W - g.
 * Everything is formed through the Gram matrix S S^T in fp64 (the
 * coefficients themselves are fp32); deterministic. ws: device workspace of
 * pair_audit_workspace_size(N, G, D) bytes, 16-byte aligned, no initial
 * contents needed.
 * Errors: as pair_coeffs_weighted; PAIR_ERR_WORKSPACE.
 */
#define PAIR_AUDIT_BIAS_NORM 0
#define PAIR_AUDIT_MSE 1
#define PAIR_AUDIT_COS 2
#define PAIR_AUDIT_VERTICES 3
#define PAIR_AUDIT_EDGES 4
#define PAIR_AUDIT_ESS 5
#define PAIR_AUDIT_TARGET_SQ 6
#define PAIR_AUDIT_WEIGHT 7
#define PAIR_AUDIT_NSTATS 8

PAIR_API size_t pair_audit_workspace_size(int32_t N, int32_t G, int32_t D);
PAIR_API pair_status pair_audit(int32_t N, int32_t G, int32_t D, const float *r,
                                const float *rho, const float *S, const uint8_t *Jdraws,
                                const double *draw_weight, float scale, uint32_t flags,
                                pair_weighting wmode, float w_max, double *stats, double *bias,
                                void *ws, size_t ws_bytes, int32_t *dev_err,
                                pair_stream_t stream);

/*
 * pair_estimate_dense -- Eq. (pair-ht) for explicit score vectors:
 *     g_b = scale * sum_{i<j} J_iJ_j h_ij / rho_ij = sum_i a_i s_{b,i}
 * (the coefficient collapse of Eq. pair-advantage; rows with a_i = 0 are
 * never read).
 *
 * In:  r, J, rho, scale as for pair_coeffs (flags = 0);
 *      S [B][G][D] float32 score vectors, D >= 1.
 * Out: g [B][D] float32; exactly 0 for a group without an active vertex.
 *      a [B][G] float32 coefficients (nullable).
 *      dev_err as for pair_coeffs.
 */
PAIR_API pair_status pair_estimate_dense(int32_t B, int32_t G, int32_t D,
                                const float *r, const uint8_t *J,
                                const float *rho, const float *S, float scale,
                                float *g, float *a, int32_t *dev_err,
                                pair_stream_t stream);

/*
 * pair_allocate -- the allocation step before the path (Sec. 4.3-4.4): for
 * each of B groups of G candidates, the contrast graph, the shared-vertex
 * surrogate and the continuation probabilities pi of the convex program of
 * Eqs. (convex-objective)-(budget):
 *     min_x  sum_{i<j} a_ij e^(x_i + x_j) + sum_i b_i e^(x_i)
 *     s.t.   sum_i c_i e^(-x_i) <= budget,  0 <= x_i <= -log pi_min,
 * pi_i = e^(-x_i), b_i = (sum_{j != i} sqrt a_ij)^2 - sum_{j != i} a_ij.
 * The edge proxy a_ij (Eq. edge-proxy) is the explicit a when given, else
 * the disagreement p_i (1 - p_j) + (1 - p_i) p_j of the predicted success
 * probabilities (Eq. disagreement), times ((m_i + m_j) / 2)^2 when score-norm
 * predictions m are given. Solved per group in fp64 to a duality-gap bound
 * of 1e-12 Phi (log-barrier Newton, one CTA per group); the group's case is
 * classified first from the fp64 sum of c in index order:
 *     PAIR_ALLOC_SLACK       budget >= sum c: pi = 1 (x = 0 minimises Phi)
 *     PAIR_ALLOC_FLOOR       budget == pi_min sum c: pi = pi_min
 *     PAIR_ALLOC_INFEASIBLE  budget < pi_min sum c: pi = pi_min, and
 *                            PAIR_DEV_ERR_ALLOC_INFEASIBLE is raised
 *     PAIR_ALLOC_FLAT        every a_ij and b_i is 0: pi = budget / sum c
 *     PAIR_ALLOC_OK          solved
 *     PAIR_ALLOC_FALLBACK    Newton did not converge: pi = budget / sum c
 *                            (uniform, same expected cost; App. C)
 *     PAIR_ALLOC_INVALID     a non-finite or out-of-range input: pi = NaN,
 *                            PAIR_DEV_ERR_ALLOC_INPUT is raised.
 * In:  B >= 1, 2 <= G <= PAIR_MAX_G; p_hat [B][G] float in [0, 1] (nullable
 *      when a is given); m_hat [B][G] float >= 0 (nullable); a [B][G][G]
 *      float >= 0, symmetric, diagonal ignored (nullable); c_hat [B][G]
 *      float > 0 (predicted suffix costs); budget [B] float > 0 (budget on
 *      the expected suffix cost); 0 < pi_min <= 1. All device pointers.
 * Out: pi [B][G] float; stats [B][PAIR_ALLOC_NSTATS] double (nullable):
 *      [PAIR_ALLOC_PHI] objective at pi, [PAIR_ALLOC_SPENT] sum c pi,
 *      [PAIR_ALLOC_GAP] duality-gap bound (2G + 1) / t, [PAIR_ALLOC_NEWTON]
 *      Newton steps, [PAIR_ALLOC_STATUS] the status above.
 * dev_err required. Deterministic. No workspace, no allocation.
 */
#define PAIR_ALLOC_OK 0
#define PAIR_ALLOC_SLACK 1
#define PAIR_ALLOC_FLOOR 2
#define PAIR_ALLOC_INFEASIBLE 3
#define PAIR_ALLOC_FALLBACK 4
#define PAIR_ALLOC_FLAT 5
#define PAIR_ALLOC_INVALID 6
#define PAIR_ALLOC_PHI 0
#define PAIR_ALLOC_SPENT 1
#define PAIR_ALLOC_GAP 2
#define PAIR_ALLOC_NEWTON 3
#define PAIR_ALLOC_STATUS 4
#define PAIR_ALLOC_NSTATS 5
PAIR_API pair_status pair_allocate(int32_t B, int32_t G, const float *p_hat, const float *m_hat,
                                   const float *a, const float *c_hat, const float *budget,
                                   float pi_min, float *pi, double *stats, int32_t *dev_err,
                                   pair_stream_t stream);

/*
 * pair_grad_workspace_size -- bytes of device workspace pair_grad (and
 * pair_grad_clipped) should be given for T packed tokens, hidden size d,
 * vocabulary V, R rollouts and dtype dt. Returns 0 for arguments pair_grad
 * would reject.
 * For PAIR_BF16 with d a multiple of 512 this includes the image of the
 * backward: the log-sum-exp pass keeps the bf16 softmax terms
 * 2^(z_tv log2 e - R_t) relative to each token's target logit R_t, 32 KB per
 * 128 tokens x 128 vocabulary rows, which the dH and dW GEMMs read instead of
 * recomputing the logits, plus the chunk's hidden rows scaled by
 * -c_t / sum_v 2^(z_tv log2 e - R_t) (128 d bf16 per token block). It holds
 * min(ceil(T/128), max(32, 24 GiB / per_block)) token blocks, per_block =
 * ceil(V/128) * 32768 + 256 d bytes (at most about 24 GiB); longer batches
 * run the backward in token chunks of that many blocks.
 */
PAIR_API size_t pair_grad_workspace_size(int64_t T, int32_t d, int32_t V, int32_t R,
                                pair_dtype dt);

/*
 * pair_grad_workspace_min_size -- the smallest workspace pair_grad accepts:
 * pair_grad_workspace_size without the image. Any size from here up to
 * pair_grad_workspace_size is valid; the image then holds the token blocks
 * that fit (more chunks), and with none no logit-sized tensor is kept at all
 * (the on-chip form: the log-sum-exp pass is fused with dH, and dW
 * recomputes the logits). Results agree to bf16/fp32 rounding across sizes
 * (the sums run in a different order), and are bit-identical for the same
 * size.
 */
PAIR_API size_t pair_grad_workspace_min_size(int64_t T, int32_t d, int32_t V, int32_t R,
                                    pair_dtype dt);

/*
 * pair_grad -- the policy objective of Sec. 4.5, sum_i a_i log pi(o_i | q),
 * realised on an LM output head over a packed variable-length batch, with
 * its exact gradients (ascent convention: derivatives OF the objective; a
 * trainer minimising a loss negates them):
 *     z_t = W h_t,  logp_t = z_t[y_t] - logsumexp(z_t),
 *     Jobj = sum_i a_i sum_{t in rollout i, mask_t = 1} logp_t,
 *     dH = dJobj/dH  [T][d],   dW = dJobj/dW  [V][d].
 * The sequence score of Sec. 3.1 is the per-rollout sum over tokens (no
 * length normalisation). Rollouts with a_i == 0 (+0 or -0) are skipped
 * entirely; their tokens' dH rows, like those of mask = 0 tokens, are
 * written as exact zeros. No logit-sized tensor is written in fp32: with the
 * default workspace the log-sum-exp pass keeps the bf16 softmax terms once
 * for the dH and dW GEMMs (see pair_grad_workspace_size); with the minimum
 * workspace nothing logit-sized is written.
 *
 * In:  T >= 1 packed tokens; d hidden size; V vocabulary size; dt dtype of
 *      H and W (PAIR_BF16: fp32 accumulation on the tensor cores, requires
 *      d % 64 == 0; PAIR_F32: fp32 CUDA-core path).
 *      Shapes: T >= 1, R >= 1, V >= 1, d % 16 == 0 (PAIR_F32) or
 *      d % 64 == 0 (PAIR_BF16); H, W 16-byte aligned.
 *      H [T][d] (dt)     hidden state that predicts y_t (targets are NOT
 *                        shifted by the library).
 *      W [V][d] (dt)     head weight (nn.Linear layout).
 *      y [T] int32       target ids; read only where mask_t = 1.
 *      mask [T] uint8    1 = response token, 0 = padding (padding rows of H
 *                        and y may hold anything, NaN included).
 *      cu_seqlens [R+1] int32  rollout i owns tokens [cu[i], cu[i+1]);
 *                        cu[0] = 0, non-decreasing, cu[R] = T (R >= 1).
 *      a [R] float32     per-rollout coefficients (e.g. from pair_coeffs,
 *                        group-major b*G + i).
 * Out: dH [T][d] float32, dW [V][d] float32,
 *      Jobj [1] double   (device pointer),
 *      logp_seq [R] float32 (nullable): sum of logp_t over the rollout's
 *                        mask = 1 tokens where a_i != 0, 0 elsewhere.
 * Workspace: ws (device, >= pair_grad_workspace_min_size bytes, normally
 *      pair_grad_workspace_size; any contents, 256-byte aligned). dev_err as
 *      for pair_coeffs (target-range and pipeline-timeout errors).
 * Deterministic: repeated calls with the same ws_bytes give bit-identical
 * outputs.
 */
PAIR_API pair_status pair_grad(int64_t T, int32_t d, int32_t V, pair_dtype dt,
                      const void *H, const void *W, const int32_t *y,
                      const uint8_t *mask, const int32_t *cu_seqlens,
                      int32_t R, const float *a, float *dH, float *dW,
                      double *Jobj, float *logp_seq, void *ws,
                      size_t ws_bytes, int32_t *dev_err, pair_stream_t stream);

/*
 * pair_grad_token_logp -- the per-token log-probabilities of the most recent
 * pair_grad (or pair_grad_clipped) call that used workspace ws:
 *     logp_tok[t] = z_t[y_t] - logsumexp(z_t)        (Sec. 4.5, log pi per token)
 * for every token t with mask_t = 1 in a rollout with a_i != 0, and 0 at every
 * other token. This is what a PPO trainer keeps as the old log-probabilities
 * of the next epochs (App. "Practical departures"); summed over a rollout it
 * is that call's logp_seq. The workspace holds them until the next call that
 * uses it.
 * In:  T, d, V, R, dt, ws and ws_bytes exactly as given to that call, on the
 *      same stream after it (stream order is the only synchronisation).
 * Out: logp_tok [T] float32 (device).
 * Errors: PAIR_ERR_INVALID_ARG (null logp_tok or shapes pair_grad rejects),
 *      PAIR_ERR_WORKSPACE (ws null, misaligned or below the minimum size).
 */
PAIR_API pair_status pair_grad_token_logp(int64_t T, int32_t d, int32_t V, int32_t R,
                                          pair_dtype dt, const void *ws, size_t ws_bytes,
                                          float *logp_tok, pair_stream_t stream);

/*
 * pair_grad_clipped -- the clipped trajectory-ratio surrogate of the practical
 * PPO epochs (Sec. 4.5; App. "Practical departures"), on the same LM-head
 * realisation as pair_grad. With the detached coefficients A_i = a[i] and the
 * trajectory ratio rho_i = exp(logp_seq_i - logp_old[i]) of every rollout
 * (logp_seq_i this call's summed log-probability, formed in fp64),
 *     J = sum_i min(rho_i A_i, clip(rho_i, 1 - clip_eps, 1 + clip_eps) A_i),
 * and dH, dW are its gradients: those of sum_i c_i logp_seq_i with
 * c_i = A_i rho_i where the unclipped term is the minimum (A_i > 0:
 * rho_i <= 1 + eps; A_i < 0: rho_i >= 1 - eps) and c_i = 0 where the clip
 * binds. At logp_old = logp_seq every ratio is 1 and the result is
 * pair_grad's gradient (J = sum_i A_i). The paper marks this as a
 * trust-region surrogate, not the design-unbiased gradient.
 * In:  as pair_grad, plus logp_old [R] float32 (device; read where a_i != 0)
 *      and clip_eps >= 0 (finite).
 * Out: as pair_grad (Jobj = the surrogate J); coef [R] float32 (nullable):
 *      the c_i used.
 * Workspace: as pair_grad (>= pair_grad_workspace_min_size, normally
 * pair_grad_workspace_size). With more than one token chunk, chunks after
 * the first recompute their log-sum-exp pass (the first keeps its logit
 * terms from the full pass that forms the ratios). Errors: as pair_grad.
 */
PAIR_API pair_status pair_grad_clipped(int64_t T, int32_t d, int32_t V, pair_dtype dt,
                                       const void *H, const void *W, const int32_t *y,
                                       const uint8_t *mask, const int32_t *cu_seqlens, int32_t R,
                                       const float *a, const float *logp_old, float clip_eps,
                                       float *dH, float *dW, double *Jobj, float *logp_seq,
                                       float *coef, void *ws, size_t ws_bytes, int32_t *dev_err,
                                       pair_stream_t stream);

/*
 * pair_grad_noalloc -- pair_grad without a caller-provided workspace, for
 * callers that cannot allocate device memory: for example a plug-in that
 * runs inside a host application which owns every device allocation and
 * exposes no allocator to it, or code that must not call cudaMalloc
 * because of the device-wide synchronisation and the out-of-memory failure
 * mode that an allocation brings. The paper has no counterpart; this is a
 * deployment convenience around the same kernels.
 *
 * Arguments, outputs and numerics are those of pair_grad, minus ws and
 * ws_bytes. The workspace is a file-scope device array of
 * PAIR_NOALLOC_MAX_WORKSPACE bytes that every GPU loading this library
 * holds until the process exits. It keeps no image of softmax terms (the
 * backward recomputes the logits); a problem is accepted iff
 * pair_grad_workspace_min_size(T, d, V, R, dt) <= PAIR_NOALLOC_MAX_WORKSPACE
 * and rejected with PAIR_ERR_WORKSPACE before any launch otherwise. That
 * size grows with T * d (the compacted hidden rows) plus, for bf16, a fixed
 * exchange buffer and, for d a multiple of 512, per-cluster partial rows of
 * width d. In this build the accepted range is, roughly: PAIR_F32, T (4 d +
 * 152) <= 33 MB (T <= 28,000 at d = 256); PAIR_BF16 with d a multiple of 512,
 * only d = 512 with T <= 6,000 (larger d need more than the array for the
 * partial rows alone); other PAIR_BF16 d, T (2 d + 152) <= 20.9 MB. Larger
 * heads (the Qwen3 shapes) need pair_grad with a caller-provided workspace.
 * The call allocates nothing.
 * The first call on each device looks up the array's device address (with
 * that device current) and caches it per device and CUDA context; make that
 * first call before any stream capture. A device reset (cudaDeviceReset)
 * unloads the array but may leave the context handle unchanged, so a process
 * that resets a device must not call pair_grad_noalloc on it afterwards.
 * All calls on a device share the one array, which keeps
 * the previous call's contents (pair_grad needs no zeroed workspace): calls
 * whose executions overlap on the GPU (different streams, or host threads
 * without ordering) race on it and must be serialised by the caller.
 */
#define PAIR_NOALLOC_MAX_WORKSPACE (32u << 20)
PAIR_API pair_status pair_grad_noalloc(int64_t T, int32_t d, int32_t V,
                                       pair_dtype dt, const void *H,
                                       const void *W, const int32_t *y,
                                       const uint8_t *mask,
                                       const int32_t *cu_seqlens, int32_t R,
                                       const float *a, float *dH, float *dW,
                                       double *Jobj, float *logp_seq,
                                       int32_t *dev_err, pair_stream_t stream);

/*
 * pair_status_sync -- synchronise `stream`, read the device error word
 * (if non-null), reset it to 0, and return the status it encodes
 * (PAIR_ERR_DEVICE_TIMEOUT, then PAIR_ERR_NONPOSITIVE_INCLUSION, then
 * PAIR_ERR_TARGET_RANGE), or
 * PAIR_ERR_CUDA if the stream reports an error. Not for hot loops.
 */
PAIR_API pair_status pair_status_sync(pair_stream_t stream, int32_t *dev_err);

/* Static description of a status code. */
PAIR_API const char *pair_status_string(pair_status st);

/* Kernel launches issued by the most recent compute call on this thread
 * (used to report how many of this library's kernels ran). */
PAIR_API int32_t pair_last_launch_count(void);

/*
 * Optional per-kernel timing (tracing). While enabled on a host thread,
 * every kernel this library launches from that thread is bracketed by CUDA
 * events recorded on the launch stream (at most 4096 launches are kept).
 * pair_timing_enable(1) starts a fresh record; pair_timing_read waits for
 * the recorded events, writes up to `max` durations in milliseconds and
 * static kernel names (either array may be null), clears the record and
 * returns the number written. Off by default; costs two event records per
 * launch when on.
 */
PAIR_API void pair_timing_enable(int32_t on);
PAIR_API int32_t pair_timing_read(int32_t max, float *ms, const char **names);

/*
 * pair_selftest_wait_timeout -- exercises the failure path of the pipeline
 * waits (a diagnostic for tests; no counterpart in the paper).
 * Launches one block that waits on an mbarrier nothing ever arrives on,
 * through the same bounded-wait code every tensor-core kernel uses, with a
 * limit of limit_cycles SM clocks (1 .. 4e9). The wait gives up, raises the
 * block's abort flag (a second role then stops waiting at once) and ORs
 * PAIR_DEV_ERR_TIMEOUT into *dev_err; the kernel then returns normally, so
 * the context stays usable. seen (2 int32, device) receives bit 0 = the wait
 * gave up, bit 1 = the abort flag was raised, and seen[1] = 1 when the second
 * role saw the flag. Asynchronous on `stream`; follow with pair_status_sync,
 * which then returns PAIR_ERR_DEVICE_TIMEOUT.
 * Errors: PAIR_ERR_INVALID_ARG (null pointer, limit out of range),
 * PAIR_ERR_UNSUPPORTED, PAIR_ERR_CUDA.
 */
PAIR_API pair_status pair_selftest_wait_timeout(int64_t limit_cycles, int32_t *dev_err,
                                                int32_t *seen, pair_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* PAIR_H_ */
