// Shared definitions for the Pair estimator CUDA library (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "pair.h"

namespace pairk {

// Clusters the cluster backward may run at once (ring buffers are sized for
// this many); each ring holds 8 owners x 2 tiles x 32 KB.
constexpr int kMaxClusters = 24;
constexpr int kMaxPairs = 256;  // 2-CTA clusters of a persistent grid, at most
constexpr int kOneHotBucket = 16;  // vocabulary rows per bucket of the one-hot dW part
constexpr size_t kRingBytesPerCluster = 8 * 2 * 32768;

constexpr float kLog2e = 1.4426950408889634f;

// Launch bookkeeping (per host thread): counts the kernels of the current
// entry-point call and, when timing is enabled, brackets each launch with
// CUDA events on its stream.
void launch_begin(const char *name, cudaStream_t s);
void launch_end(cudaStream_t s);
void reset_launches();
// PAIR_OK on a compute-capability 10.3 device, else PAIR_ERR_UNSUPPORTED.
pair_status check_device();

__device__ __forceinline__ void flag_error(int32_t *err, int bit) {
  if (err) atomicOr(err, bit);
}

__host__ __device__ __forceinline__ int64_t ceil_div(int64_t a, int64_t b) {
  return (a + b - 1) / b;
}

// Group coefficient kernels (pair_coeffs.cu).
pair_status launch_coeffs(int32_t B, int32_t G, const float *r,
                          const uint8_t *J, const float *rho, float scale,
                          uint32_t flags, float *a, uint8_t *active,
                          int32_t *edges, int32_t *contrast, int32_t *dev_err,
                          cudaStream_t s);
pair_status launch_estimate_dense(int32_t B, int32_t G, int32_t D,
                                  const float *r, const uint8_t *J,
                                  const float *rho, const float *S,
                                  float scale, float *g, float *a,
                                  int32_t *dev_err, cudaStream_t s);
pair_status launch_coeffs_weighted(int32_t B, int32_t G, const float *r, const uint8_t *J,
                                   const float *rho, float scale, uint32_t flags, int wmode,
                                   float w_max, float *a, uint8_t *active, int32_t *edges,
                                   int32_t *contrast, float *ess, float *max_w,
                                   int32_t *dev_err, cudaStream_t s);
// Streaming coefficient kernel (pair_coeffs_stream.cu): G <= 64, G % 4 == 0,
// 16-byte aligned r and rho, 4-byte aligned J. Weightings HT (diag = whether
// ess / max_w are written), clipped and self-normalised.
bool coeffs_stream_applies(int32_t G, const float *r, const uint8_t *J, const float *rho);
pair_status launch_coeffs_stream(int32_t B, int32_t G, const float *r, const uint8_t *J,
                                 const float *rho, float scale, uint32_t flags, int wmode,
                                 bool diag, float w_max, float *a, uint8_t *active,
                                 int32_t *edges, int32_t *contrast, float *ess, float *max_w,
                                 int32_t *dev_err, cudaStream_t s);
pair_status launch_coeffs_product(int32_t B, int32_t G, const float *r, const uint8_t *J,
                                  const float *p, float scale, uint32_t flags, float *a,
                                  uint8_t *active, int32_t *edges, int32_t *contrast, float *ess,
                                  float *max_w, int32_t *dev_err, cudaStream_t s);

// pair_grad pieces (pair_grad_prep.cu, pair_grad_simt.cu, pair_grad_tc.cu).
struct GradWorkspace {
  int32_t *counters;   // [0] = number of active tokens T_eff
  int32_t *seg_cnt;    // [R] active tokens per rollout
  int32_t *seg_off;    // [R+1] exclusive prefix of seg_cnt
  int32_t *tok_idx;    // [T] packed position of each active token
  int32_t *tok_y;      // [T] its target id
  float *tok_c;        // [T] its coefficient c_t = a_seg(t)
  float *lse;          // [Tpad] log-sum-exp of the active token's logits
  float *zy;           // [Tpad] target logit
  float2 *part;        // [nsplit][Tpad] partial (max, sum-exp) per split
  double *seg_logp;    // [R] per-rollout sum of logp (fp64)
  float *ppo_c;        // [R] clipped-surrogate coefficients (pair_grad_clipped)
  double *ppo_L;       // [R] clipped-surrogate terms (pair_grad_clipped)
  void *Hc;            // [Tpad][d] compacted hidden rows (dt), zero tail
  int32_t *bkt;        // [3][nb + 1] one-hot part of dW: per target bucket of
                       // kOneHotBucket rows, token counts, offsets, fill counters
  int32_t *blist;      // [Tpad] active tokens grouped by target bucket
  void *gring;         // per-cluster ring of published Gs tiles
  float *tailbuf;      // [kMaxClusters][2][128][d] partial tail units (cluster path)
  // Fused log-sum-exp + dH pass (cluster path; null otherwise).
  float *ref;          // [Tpad] per-token reference of the softmax terms (log2 units)
  float *mrow;         // [Tpad] row maximum of the logits (log2 units)
  float *lsum;         // [Tpad] image path: sum of 2^(z log2 e - ref) over the vocabulary
  int32_t *prog;       // [kMaxPairs] image path: per-CTA-pair progress of the dH GEMM
  int32_t *rbflag;     // [n_rbmax] row block needs the fix-up pass
  int32_t *rb_list;    // [n_rbmax] row blocks of the fix-up pass (count in counters[1])
  int32_t *ready;      // [n_slots] per-unit publication counters
  float *lpart;        // [n_slots][8][2][128] per-CTA row partials (l, maximum)
  float *tail_l;       // [kMaxClusters][2][2][128] tail units' row partials
  int n_rbmax, n_slots;
  void *gimg;          // bf16 softmax-term tiles 2^(z log2 e - ref) of gimg_rb token blocks
  void *hs;            // [gimg_rb * 128][d] bf16 rows s_t Hc_t of a chunk (s_t = -c_t / lsum_t)
  int gimg_rb;         // token blocks (128 rows) per backward chunk; 0 = no image
  int64_t Tpad;
  int nsplit;
};

// Whether the bf16 backward runs as 8-CTA clusters: d = 512 A, 1 <= A <= 6.
inline bool grad_cluster_path(int d) { return d % 512 == 0 && d >= 512 && d <= 3072; }

// Token blocks per backward chunk for which the bf16 path keeps the image of
// softmax terms and the scaled hidden rows (0 where that path does not apply:
// fp32, or d not a multiple of 512), and the bytes one block of both takes.
int grad_gimg_rows(int64_t T, int32_t d, int32_t V, pair_dtype dt);
size_t grad_image_block_bytes(int32_t d, int32_t V);
constexpr uint32_t kGImgTileBytes = 128 * 128 * 2;  // one 128 x 128 bf16 tile

// Workspace layout with gimg_rb token blocks of image and scaled rows (0 =
// none; at most grad_gimg_rows). Returns its size in bytes.
size_t grad_workspace_bytes(int64_t T, int32_t d, int32_t V, int32_t R,
                            pair_dtype dt, GradWorkspace *out, void *base, int gimg_rb);
// Image token blocks that fit in ws_bytes (at most grad_gimg_rows), or -1 if
// ws_bytes is below the size without an image.
int grad_gimg_rows_fit(int64_t T, int32_t d, int32_t V, int32_t R, pair_dtype dt,
                       size_t ws_bytes);

struct GradArgs {
  int64_t T;
  int32_t d, V, R;
  pair_dtype dt;
  const void *H, *W;
  const int32_t *y;
  const uint8_t *mask;
  const int32_t *cu;
  const float *a;
  float *dH, *dW;
  double *Jobj;
  float *logp_seq;
  int32_t *dev_err;
};

pair_status grad_prepare(const GradArgs &g, const GradWorkspace &w,
                         cudaStream_t s);
pair_status grad_finalize(const GradArgs &g, const GradWorkspace &w,
                          cudaStream_t s);
pair_status grad_head_simt(const GradArgs &g, const GradWorkspace &w,
                           cudaStream_t s);
pair_status grad_head_tc(const GradArgs &g, const GradWorkspace &w,
                         cudaStream_t s);
// Forward (log-sum-exp) and backward halves of the two head paths.
pair_status grad_lse_tc(const GradArgs &g, const GradWorkspace &w, cudaStream_t s);
pair_status grad_bwd_tc(const GradArgs &g, const GradWorkspace &w, cudaStream_t s);
pair_status grad_lse_simt(const GradArgs &g, const GradWorkspace &w, cudaStream_t s);
pair_status grad_bwd_simt(const GradArgs &g, const GradWorkspace &w, cudaStream_t s);
// Clipped trajectory-ratio surrogate between the two halves (pair_grad_prep.cu).
pair_status grad_ppo_coefficients(const GradArgs &g, const GradWorkspace &w,
                                  const float *logp_old, float eps, float *coef_out,
                                  cudaStream_t s);
pair_status grad_ppo_finalize(const GradArgs &g, const GradWorkspace &w, cudaStream_t s);
// Per-token log-probabilities kept in the workspace, scattered to [T].
pair_status grad_token_logp(int64_t T, const GradWorkspace &w, float *logp_tok, cudaStream_t s);
// Exact one-hot parts (added after the tensor-core softmax parts).
pair_status grad_onehot(const GradArgs &g, const GradWorkspace &w,
                        cudaStream_t s);

}  // namespace pairk

#define PAIR_CUDA_TRY(expr)                                   \
  do {                                                        \
    cudaError_t e_ = (expr);                                  \
    if (e_ != cudaSuccess) return PAIR_ERR_CUDA;              \
  } while (0)

#define PAIR_BEGIN(name, s) ::pairk::launch_begin(name, s)

#define PAIR_LAUNCH_CHECK(s)                                  \
  do {                                                        \
    ::pairk::launch_end(s);                                   \
    cudaError_t e_ = cudaGetLastError();                      \
    if (e_ != cudaSuccess) return PAIR_ERR_CUDA;              \
  } while (0)
