// pair_grad_noalloc: pair_grad for callers that cannot allocate device
// memory. Its workspace is a fixed array in this library's device data
// instead of a caller-provided buffer; everything else is the pair_grad
// launch sequence, unchanged.
#include <cuda.h>

#include <mutex>

#include "pair_common.cuh"

namespace pairk {
namespace {

constexpr size_t kStaticScratchBytes = PAIR_NOALLOC_MAX_WORKSPACE;

// Workspace shared by every pair_grad_noalloc call on a device. Each GPU
// that loads this library holds one copy until the process exits.
static __device__ __align__(256) unsigned char g_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 128;
std::mutex g_scratch_mu;
struct ScratchSlot {
  CUcontext ctx;  // context the address was looked up in
  void *addr;
};
ScratchSlot g_scratch_slot[kMaxDevices] = {};

using CtxGetCurrentFn = CUresult (*)(CUcontext *);
CtxGetCurrentFn ctx_get_current() {
  static CtxGetCurrentFn fn = nullptr;
  if (!fn) {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<CtxGetCurrentFn>(p);
  }
  return fn;
}

// Device address of g_scratch on the current device. The host-side name of
// a __device__ array is only a stand-in, so the address is looked up (with
// the device current) the first time a device is used, and again whenever
// the current context differs from the one it was looked up in.
pair_status scratch_address(void **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return PAIR_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return PAIR_ERR_UNSUPPORTED;
  CtxGetCurrentFn get = ctx_get_current();
  if (!get) return PAIR_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  ScratchSlot &slot = g_scratch_slot[dev];
  CUcontext ctx = nullptr;
  if (get(&ctx) != CUDA_SUCCESS) return PAIR_ERR_CUDA;
  if (!slot.addr || !ctx || slot.ctx != ctx) {
    void *p = nullptr;
    // The lookup also makes the device's primary context current when no
    // context is yet.
    if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || !p) return PAIR_ERR_CUDA;
    if (get(&ctx) != CUDA_SUCCESS || !ctx) return PAIR_ERR_CUDA;
    slot.ctx = ctx;
    slot.addr = p;
  }
  *out = slot.addr;
  return PAIR_OK;
}

}  // namespace
}  // namespace pairk

using namespace pairk;

extern "C" pair_status pair_grad_noalloc(
    int64_t T, int32_t d, int32_t V, pair_dtype dt, const void *H,
    const void *W, const int32_t *y, const uint8_t *mask,
    const int32_t *cu_seqlens, int32_t R, const float *a, float *dH,
    float *dW, double *Jobj, float *logp_seq, int32_t *dev_err,
    pair_stream_t stream) {
  reset_launches();
  if (!H || !W || !y || !mask || !cu_seqlens || !a || !dH || !dW || !Jobj)
    return PAIR_ERR_INVALID_ARG;
  // This path keeps no image of softmax terms (its dW pass recomputes the
  // logits), so it needs the workspace without one.
  const size_t need = pair_grad_workspace_min_size(T, d, V, R, dt);
  if (need == 0)
    return (dt == PAIR_BF16 && d % 64 != 0 && d % 16 == 0)
               ? PAIR_ERR_UNSUPPORTED
               : PAIR_ERR_INVALID_ARG;
  if (need > kStaticScratchBytes) return PAIR_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(H) & 15u) || (reinterpret_cast<uintptr_t>(W) & 15u) ||
      (reinterpret_cast<uintptr_t>(dH) & 15u) || (reinterpret_cast<uintptr_t>(dW) & 15u))
    return PAIR_ERR_INVALID_ARG;
  const pair_status dv = check_device();
  if (dv != PAIR_OK) return dv;
  void *ws = nullptr;
  const pair_status sa = scratch_address(&ws);
  if (sa != PAIR_OK) return sa;

  // The workspace needs no initial contents: every kernel writes the parts
  // it later reads within the same call.
  GradWorkspace w;
  grad_workspace_bytes(T, d, V, R, dt, &w, ws, 0);
  GradArgs g{T, d, V, R, dt, H, W, y, mask, cu_seqlens, a,
             dH, dW, Jobj, logp_seq, dev_err};
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  pair_status st = grad_prepare(g, w, s);
  if (st != PAIR_OK) return st;
  if (dt == PAIR_BF16) {
    st = grad_head_tc(g, w, s);
    if (st != PAIR_OK) return st;
    st = grad_onehot(g, w, s);
  } else {
    st = grad_head_simt(g, w, s);
  }
  if (st != PAIR_OK) return st;
  return grad_finalize(g, w, s);
}
