// Shared pieces of the bf16 LM-head kernels on the 5th-generation tensor
// cores (pair_lse.cu, pair_bwd_image.cu, pair_bwd_cluster.cu) and of their
// host orchestration (pair_grad_tc.cu): the warp-specialised CTA shape,
// small device helpers, tensor-map and grid helpers, and the entry points of
// each stage.
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "pair_common.cuh"
#include "tc_ptx.cuh"

namespace pairk {
namespace tck {

using namespace tc;

// CTA of the head kernels: warp 0 = TMA producer, warp 1 = TMEM owner and
// single-thread MMA issuer, warps 2..5 = epilogue (one TMEM lane quadrant
// each, one tile row per thread).
constexpr int kThreads = 192;
constexpr int kAtom128 = 128 * 64 * 2;  // 128 rows x 64 bf16 (16 KB)
constexpr int kAllBlocks = 0x7fffffff;  // "every token block" for chunked passes

// Named barrier of the four epilogue warps (128 threads).
__device__ __forceinline__ void epi_sync() {
  asm volatile("bar.sync 1, 128;" ::: "memory");
}

__device__ __forceinline__ uint8_t *align1k(uint8_t *p) {
  return reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(p) + 1023) &
                                     ~static_cast<uintptr_t>(1023));
}

// Bulk copy global -> this CTA's shared memory, completing on `bar`.
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes,
                                          uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1], %2, [%3];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// Bulk copy of `bytes` (multiple of 16, both addresses 16-byte aligned) from
// this CTA's shared memory to global memory, tracked by this thread's bulk
// groups, with an L2 evict-first hint.
__device__ __forceinline__ void bulk_store_evict_first(void *dst, const void *src,
                                                       uint32_t bytes) {
  asm volatile(
      "{\n\t.reg .b64 pol;\n\t"
      "createpolicy.fractional.L2::evict_first.b64 pol, 1.0;\n\t"
      "cp.async.bulk.global.shared::cta.bulk_group.L2::cache_hint [%0], [%1], %2, pol;\n\t}" ::"l"(
          reinterpret_cast<uint64_t>(dst)),
      "r"(smem_u32(src)), "r"(bytes)
      : "memory");
}

// <h, w> over d bf16 elements by one warp (d a multiple of 8, rows 16-byte
// aligned): fp32 sums of the products in a fixed order (lane-strided
// 8-element pieces, then the warp's butterfly); every lane gets the sum.
__device__ __forceinline__ float target_logit_dot(int d, const __nv_bfloat16 *h,
                                                  const __nv_bfloat16 *w, int lane) {
  float acc = 0.f;
  for (int k = lane * 8; k < d; k += 256) {
    const uint4 hu = *reinterpret_cast<const uint4 *>(h + k);
    const uint4 wu = *reinterpret_cast<const uint4 *>(w + k);
    const __nv_bfloat162 *hb = reinterpret_cast<const __nv_bfloat162 *>(&hu);
    const __nv_bfloat162 *wb = reinterpret_cast<const __nv_bfloat162 *>(&wu);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 hf = __bfloat1622float2(hb[i]), wf = __bfloat1622float2(wb[i]);
      acc = fmaf(hf.x, wf.x, acc);
      acc = fmaf(hf.y, wf.y, acc);
    }
  }
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  return acc;
}

__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// ---- host helpers (pair_grad_tc.cu)
PFN_cuTensorMapEncodeTiled_v12000 encode_fn();
// 2-D bf16 row-major [rows][cols] map with 64 x box_rows SWIZZLE_128B boxes.
bool make_map(CUtensorMap *m, const void *ptr, int64_t rows, int64_t cols, int box_rows);
// 3-D bf16 map: dims (innermost first), byte strides of dims 1 and 2, box, swizzle.
bool make_map3(CUtensorMap *m, const void *ptr, const cuuint64_t (&dims)[3],
               const cuuint64_t (&strides)[2], const cuuint32_t (&box)[3],
               CUtensorMapSwizzle sw);
int num_sms();
// CTAs of a persistent grid of 2-CTA clusters (occupancy API; cached in *cache).
int pair_grid(const void *kernel, size_t smem, int *cache);

// ---- stages of the head
// Per-token reference of the image path's log-sum-exp pass: R_t = z_t[y_t]
// log2 e for every active token (pair_lse.cu).
pair_status launch_ref(const GradArgs &g, const GradWorkspace &w, cudaStream_t s);
// Log-sum-exp pass over token blocks [rb0, rb0 + cap), then lse of those
// tokens. With image, the softmax terms are taken relative to the reference
// (launch_ref first), the bf16 terms of its first s_blocks blocks are kept as
// the image, and rows too far above their reference are redone (pair_lse.cu).
pair_status launch_lse(const GradArgs &g, const GradWorkspace &w, cudaStream_t s, int rb0,
                       int cap, bool image, int s_blocks);
// One token chunk of the image backward: scaled hidden rows, dh_gemm,
// dw_gemm (pair_bwd_image.cu).
pair_status launch_chunk_bwd(const GradArgs &g, const GradWorkspace &w, cudaStream_t s,
                             int64_t c);
// Backward without an image, recomputing the logits (pair_bwd_cluster.cu).
pair_status grad_bwd_recompute(const GradArgs &g, const GradWorkspace &w, cudaStream_t s);
// Whole head without an image: fused log-sum-exp + dH, then dW (cluster
// form; d = 512 A, A <= 6). lse, zy and dH, dW softmax parts as the
// three-pass sequence leaves them.
bool onchip_fused_applies(int d);
pair_status grad_head_onchip(const GradArgs &g, const GradWorkspace &w, cudaStream_t s);

inline bool image_path(const GradWorkspace &w) { return w.gimg && w.hs && w.gimg_rb > 0; }
inline int64_t image_chunks(const GradArgs &g, const GradWorkspace &w) {
  return ((g.T + 127) / 128 + w.gimg_rb - 1) / w.gimg_rb;
}

}  // namespace tck
}  // namespace pairk
