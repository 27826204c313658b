// bf16 LM-head path of pair_grad on the 5th-generation tensor cores
// (tcgen05 + TMEM + TMA, sm_103a): the order of its passes and their shared
// host helpers.
//
// Objective (Sec. 4.5): J = sum_t c_t logp_t over compacted active tokens,
// logp_t = z_{t,y_t} - lse_t, z = W h. Its gradients split into an exact
// one-hot part (added in fp32 by grad_onehot) and a softmax part that is a
// pair of dense contractions through the logit gradient
//     Gs_tv = -c_t exp(z_tv - lse_t)      (bf16):
//     dH_t += sum_v Gs_tv W_v,     dW_v += sum_t Gs_tv h_t.
//
// Passes (one file each):
//   pair_lse.cu          log-sum-exp and target logit per token; keeps the
//                        logit terms of a token chunk for the backward.
//   pair_bwd_image.cu    Gs tiles formed once from the kept terms, then
//                        dH = Gs . W and dW = Gs^T . Hc as plain GEMMs.
//   pair_bwd_cluster.cu  without room for the image: the recomputing
//                        backward (8-CTA cluster form, or per d-slice).
#include "tc_kernels.cuh"

namespace pairk {
namespace tck {

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

}  // namespace tck

using namespace tck;

// Forward half: per-token log-sum-exp and target logit over every active
// token (with an image, relative to each token's reference, and the first
// chunk's softmax terms are kept for the backward).
pair_status grad_lse_tc(const GradArgs &g, const GradWorkspace &w, cudaStream_t s) {
  if (image_path(w)) {
    const pair_status st = launch_ref(g, w, s);
    return st != PAIR_OK ? st : launch_lse(g, w, s, 0, kAllBlocks, true, w.gimg_rb);
  }
  return launch_lse(g, w, s, 0, kAllBlocks, false, 0);
}

// Backward half: softmax parts of dH and dW from the token coefficients,
// after grad_lse_tc. With an image, token blocks run in chunks of
// w.gimg_rb: the first chunk uses the softmax terms grad_lse_tc kept, later
// chunks recompute theirs (with the references grad_lse_tc settled).
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
  return grad_bwd_recompute(g, w, s);
}

// The backward through the image runs whenever the workspace holds one:
// token blocks in chunks of w.gimg_rb, and for each chunk
//   scale_rows  Hs = s_t Hc[t, :] in bf16, s_t = -c_t / lsum_t,
//   dh_gemm     dH rows of the chunk = s_t (P . W),
//   dw_gemm     dW (+)= P^T . Hs (the first chunk stores, later ones add),
// P being the bf16 softmax terms 2^(z log2 e - R_t) the chunk's log-sum-exp
// pass kept. The number of chunks follows from T, so the launch sequence
// needs no device-to-host read; chunks past the last active token exit at
// once.
//
// Whole head: with an image, the references R_t, then each chunk's
// log-sum-exp pass keeps its softmax terms for that chunk's backward (no
// recomputation); otherwise, where the cluster kernels apply, the fused
// log-sum-exp + dH pass and the recomputing dW pass (no logit-sized tensor in
// HBM), else forward, then the recomputing backward.
pair_status grad_head_tc(const GradArgs &g, const GradWorkspace &w, cudaStream_t s) {
  if (image_path(w)) {
    const pair_status st = launch_ref(g, w, s);
    if (st != PAIR_OK) return st;
    const int64_t nc = image_chunks(g, w);
    for (int64_t c = 0; c < nc; ++c) {
      pair_status st = launch_lse(g, w, s, (int)(c * w.gimg_rb), w.gimg_rb, true, w.gimg_rb);
      if (st == PAIR_OK) st = launch_chunk_bwd(g, w, s, c);
      if (st != PAIR_OK) return st;
    }
    return PAIR_OK;
  }
  if (onchip_fused_applies(g.d)) return grad_head_onchip(g, w, s);
  const pair_status st = grad_lse_tc(g, w, s);
  return st != PAIR_OK ? st : grad_bwd_tc(g, w, s);
}

}  // namespace pairk
