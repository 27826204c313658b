// C-ABI entry points of libpair (see include/pair.h for the contract).
//
// Host side only: argument validation, device check, workspace carving and
// the launch sequence. Every compute step runs in this library's kernels.
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "pair_common.cuh"

namespace pairk {

// Per-host-thread launch bookkeeping and the optional per-kernel timer.
namespace {
constexpr int kMaxTimed = 4096;
struct TimedLaunch {
  const char *name;
  cudaEvent_t start, stop;
};
struct LaunchLog {
  int32_t launches = 0;
  bool timing = false;
  int n = 0;           // recorded launches since the last read
  int n_events = 0;    // events created so far (reused across reads)
  TimedLaunch rec[kMaxTimed];
};
thread_local LaunchLog g_log;
}  // namespace

void launch_begin(const char *name, cudaStream_t s) {
  LaunchLog &L = g_log;
  if (!L.timing || L.n >= kMaxTimed) return;
  TimedLaunch &t = L.rec[L.n];
  if (L.n >= L.n_events) {
    if (cudaEventCreate(&t.start) != cudaSuccess ||
        cudaEventCreate(&t.stop) != cudaSuccess)
      return;
    ++L.n_events;
  }
  t.name = name;
  cudaEventRecord(t.start, s);
}

void launch_end(cudaStream_t s) {
  LaunchLog &L = g_log;
  ++L.launches;
  if (!L.timing || L.n >= kMaxTimed || L.n >= L.n_events) return;
  cudaEventRecord(L.rec[L.n].stop, s);
  ++L.n;
}

void reset_launches() { g_log.launches = 0; }

// Compute capability 10.3 (GB300) on the current device; the answer is
// cached per device ordinal (0 = not yet known, 1 = supported, 2 = not), so
// host threads working on different devices never share a slot.
pair_status check_device() {
  constexpr int kMaxDev = 128;
  static std::atomic<int> cache[kMaxDev];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return PAIR_ERR_CUDA;
  const int known = (dev >= 0 && dev < kMaxDev) ? cache[dev].load(std::memory_order_relaxed) : 0;
  if (known) return known == 1 ? PAIR_OK : PAIR_ERR_UNSUPPORTED;
  int major = 0, minor = 0;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
    return PAIR_ERR_CUDA;
  const bool ok = major == 10 && minor == 3;
  if (dev >= 0 && dev < kMaxDev) cache[dev].store(ok ? 1 : 2, std::memory_order_relaxed);
  return ok ? PAIR_OK : PAIR_ERR_UNSUPPORTED;
}

static bool aligned16(const void *p) {
  return (reinterpret_cast<uintptr_t>(p) & 15u) == 0;
}

}  // namespace pairk

using namespace pairk;

extern "C" {

pair_status pair_coeffs(int32_t B, int32_t G, const float *r, const uint8_t *J,
                        const float *rho, float scale, uint32_t flags,
                        float *a, uint8_t *active, int32_t *edges,
                        int32_t *contrast_edges, int32_t *dev_err,
                        pair_stream_t stream) {
  reset_launches();
  if (B < 1 || G < 2 || G > PAIR_MAX_G || !r || !J || !rho || !a ||
      (flags & ~(PAIR_CENTER | PAIR_STANDARDIZE)) != 0)
    return PAIR_ERR_INVALID_ARG;
  const pair_status dv = check_device();
  if (dv != PAIR_OK) return dv;
  return launch_coeffs(B, G, r, J, rho, scale, flags, a, active, edges,
                       contrast_edges, dev_err,
                       reinterpret_cast<cudaStream_t>(stream));
}

pair_status pair_coeffs_weighted(int32_t B, int32_t G, const float *r, const uint8_t *J,
                                 const float *rho, float scale, uint32_t flags,
                                 pair_weighting wmode, float w_max, float *a, uint8_t *active,
                                 int32_t *edges, int32_t *contrast_edges, float *ess,
                                 float *max_w, int32_t *dev_err, pair_stream_t stream) {
  reset_launches();
  if (B < 1 || G < 2 || G > PAIR_MAX_G || !r || !J || !a || (flags & ~(PAIR_CENTER | PAIR_STANDARDIZE)) != 0)
    return PAIR_ERR_INVALID_ARG;
  const int wm = (int)wmode;
  if (wm < PAIR_W_HT || wm > PAIR_W_HAJEK) return PAIR_ERR_INVALID_ARG;
  if (wm != PAIR_W_UNWEIGHTED && !rho) return PAIR_ERR_INVALID_ARG;
  if (wm == PAIR_W_CLIPPED && !(w_max > 0.f && w_max <= 3.0e38f)) return PAIR_ERR_INVALID_ARG;
  const pair_status dv = check_device();
  if (dv != PAIR_OK) return dv;
  return launch_coeffs_weighted(B, G, r, J, rho, scale, flags, wm, w_max, a, active, edges,
                                contrast_edges, ess, max_w, dev_err,
                                reinterpret_cast<cudaStream_t>(stream));
}

pair_status pair_coeffs_product(int32_t B, int32_t G, const float *r, const uint8_t *J,
                                const float *p, float scale, uint32_t flags, float *a,
                                uint8_t *active, int32_t *edges, int32_t *contrast_edges,
                                float *ess, float *max_w, int32_t *dev_err,
                                pair_stream_t stream) {
  reset_launches();
  if (B < 1 || G < 2 || G > PAIR_MAX_G || !r || !J || !p || !a || (flags & ~(PAIR_CENTER | PAIR_STANDARDIZE)) != 0)
    return PAIR_ERR_INVALID_ARG;
  const pair_status dv = check_device();
  if (dv != PAIR_OK) return dv;
  return launch_coeffs_product(B, G, r, J, p, scale, flags, a, active, edges, contrast_edges,
                               ess, max_w, dev_err, reinterpret_cast<cudaStream_t>(stream));
}

pair_status pair_estimate_dense(int32_t B, int32_t G, int32_t D,
                                const float *r, const uint8_t *J,
                                const float *rho, const float *S, float scale,
                                float *g, float *a, int32_t *dev_err,
                                pair_stream_t stream) {
  reset_launches();
  if (B < 1 || G < 2 || G > PAIR_MAX_G || D < 1 || !r || !J || !rho || !S ||
      !g)
    return PAIR_ERR_INVALID_ARG;
  const pair_status dv = check_device();
  if (dv != PAIR_OK) return dv;
  return launch_estimate_dense(B, G, D, r, J, rho, S, scale, g, a, dev_err,
                               reinterpret_cast<cudaStream_t>(stream));
}

pair_status pair_grad_clipped(int64_t T, int32_t d, int32_t V, pair_dtype dt, const void *H,
                              const void *W, const int32_t *y, const uint8_t *mask,
                              const int32_t *cu_seqlens, int32_t R, const float *a,
                              const float *logp_old, float clip_eps, float *dH, float *dW,
                              double *Jobj, float *logp_seq, float *coef, void *ws,
                              size_t ws_bytes, int32_t *dev_err, pair_stream_t stream) {
  reset_launches();
  if (!H || !W || !y || !mask || !cu_seqlens || !a || !logp_old || !dH || !dW || !Jobj)
    return PAIR_ERR_INVALID_ARG;
  if (!(clip_eps >= 0.f && clip_eps <= 1.0e30f)) return PAIR_ERR_INVALID_ARG;
  if (!aligned16(H) || !aligned16(W) || !aligned16(dH) || !aligned16(dW))
    return PAIR_ERR_INVALID_ARG;
  const size_t need = pair_grad_workspace_min_size(T, d, V, R, dt);
  if (need == 0) return (dt == PAIR_BF16 && d % 64 != 0 && d % 16 == 0)
                            ? PAIR_ERR_UNSUPPORTED
                            : PAIR_ERR_INVALID_ARG;
  if (!ws || ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return PAIR_ERR_WORKSPACE;
  const pair_status dv = check_device();
  if (dv != PAIR_OK) return dv;

  GradWorkspace w;
  grad_workspace_bytes(T, d, V, R, dt, &w, ws, grad_gimg_rows_fit(T, d, V, R, dt, ws_bytes));
  GradArgs g{T, d, V, R, dt, H, W, y, mask, cu_seqlens, a,
             dH, dW, Jobj, logp_seq, dev_err};
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // Forward, then the surrogate's coefficients (they depend on this call's
  // log-probabilities), then the backward with those coefficients.
  pair_status st = grad_prepare(g, w, s);
  if (st == PAIR_OK) st = dt == PAIR_BF16 ? grad_lse_tc(g, w, s) : grad_lse_simt(g, w, s);
  if (st == PAIR_OK) st = grad_ppo_coefficients(g, w, logp_old, clip_eps, coef, s);
  if (st == PAIR_OK) st = dt == PAIR_BF16 ? grad_bwd_tc(g, w, s) : grad_bwd_simt(g, w, s);
  if (st == PAIR_OK && dt == PAIR_BF16) st = grad_onehot(g, w, s);
  if (st == PAIR_OK) st = grad_ppo_finalize(g, w, s);
  return st;
}

namespace {
bool grad_shape_ok(int64_t T, int32_t d, int32_t V, int32_t R, pair_dtype dt) {
  if (T < 1 || R < 1 || V < 1 || d < 16 || (d % 16) != 0) return false;
  if (dt != PAIR_F32 && dt != PAIR_BF16) return false;
  if (dt == PAIR_BF16 && (d % 64) != 0) return false;
  return T <= (int64_t)INT32_MAX - 1024;
}
}  // namespace

size_t pair_grad_workspace_size(int64_t T, int32_t d, int32_t V, int32_t R,
                                pair_dtype dt) {
  if (!grad_shape_ok(T, d, V, R, dt)) return 0;
  return grad_workspace_bytes(T, d, V, R, dt, nullptr, nullptr, grad_gimg_rows(T, d, V, dt));
}

size_t pair_grad_workspace_min_size(int64_t T, int32_t d, int32_t V, int32_t R,
                                    pair_dtype dt) {
  if (!grad_shape_ok(T, d, V, R, dt)) return 0;
  return grad_workspace_bytes(T, d, V, R, dt, nullptr, nullptr, 0);
}

pair_status pair_grad(int64_t T, int32_t d, int32_t V, pair_dtype dt,
                      const void *H, const void *W, const int32_t *y,
                      const uint8_t *mask, const int32_t *cu_seqlens,
                      int32_t R, const float *a, float *dH, float *dW,
                      double *Jobj, float *logp_seq, void *ws,
                      size_t ws_bytes, int32_t *dev_err,
                      pair_stream_t stream) {
  reset_launches();
  if (!H || !W || !y || !mask || !cu_seqlens || !a || !dH || !dW || !Jobj)
    return PAIR_ERR_INVALID_ARG;
  if (!aligned16(H) || !aligned16(W) || !aligned16(dH) || !aligned16(dW))
    return PAIR_ERR_INVALID_ARG;
  const size_t need = pair_grad_workspace_min_size(T, d, V, R, dt);
  if (need == 0) return (dt == PAIR_BF16 && d % 64 != 0 && d % 16 == 0)
                            ? PAIR_ERR_UNSUPPORTED
                            : PAIR_ERR_INVALID_ARG;
  if (!ws || ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return PAIR_ERR_WORKSPACE;
  const pair_status dv = check_device();
  if (dv != PAIR_OK) return dv;

  GradWorkspace w;
  grad_workspace_bytes(T, d, V, R, dt, &w, ws, grad_gimg_rows_fit(T, d, V, R, dt, ws_bytes));
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

pair_status pair_grad_token_logp(int64_t T, int32_t d, int32_t V, int32_t R, pair_dtype dt,
                                 const void *ws, size_t ws_bytes, float *logp_tok,
                                 pair_stream_t stream) {
  reset_launches();
  if (!logp_tok) return PAIR_ERR_INVALID_ARG;
  const size_t need = pair_grad_workspace_min_size(T, d, V, R, dt);
  if (need == 0) return PAIR_ERR_INVALID_ARG;
  if (!ws || ws_bytes < need || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return PAIR_ERR_WORKSPACE;
  const pair_status dv = check_device();
  if (dv != PAIR_OK) return dv;
  GradWorkspace w;
  grad_workspace_bytes(T, d, V, R, dt, &w, const_cast<void *>(ws),
                       grad_gimg_rows_fit(T, d, V, R, dt, ws_bytes));
  return grad_token_logp(T, w, logp_tok, reinterpret_cast<cudaStream_t>(stream));
}

pair_status pair_status_sync(pair_stream_t stream, int32_t *dev_err) {
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return PAIR_ERR_CUDA;
  if (!dev_err) return PAIR_OK;
  int32_t h = 0;
  if (cudaMemcpy(&h, dev_err, sizeof(h), cudaMemcpyDeviceToHost) != cudaSuccess)
    return PAIR_ERR_CUDA;
  if (h != 0 && cudaMemset(dev_err, 0, sizeof(h)) != cudaSuccess)
    return PAIR_ERR_CUDA;
  if (h & PAIR_DEV_ERR_TIMEOUT) return PAIR_ERR_DEVICE_TIMEOUT;
  if (h & PAIR_DEV_ERR_NONPOSITIVE_INCLUSION) return PAIR_ERR_NONPOSITIVE_INCLUSION;
  if (h & PAIR_DEV_ERR_TARGET_RANGE) return PAIR_ERR_TARGET_RANGE;
  if (h & PAIR_DEV_ERR_ALLOC_INPUT) return PAIR_ERR_ALLOC_INPUT;
  if (h & PAIR_DEV_ERR_ALLOC_INFEASIBLE) return PAIR_ERR_ALLOC_INFEASIBLE;
  return PAIR_OK;
}

const char *pair_status_string(pair_status st) {
  switch (st) {
    case PAIR_OK: return "ok";
    case PAIR_ERR_INVALID_ARG: return "invalid argument";
    case PAIR_ERR_UNSUPPORTED: return "unsupported device or shape";
    case PAIR_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case PAIR_ERR_NONPOSITIVE_INCLUSION:
      return "joint inclusion probability <= 0 or NaN on a completed edge";
    case PAIR_ERR_TARGET_RANGE: return "target id outside [0, V) at a mask=1 token";
    case PAIR_ERR_CUDA: return "CUDA runtime error";
    case PAIR_ERR_DEVICE_TIMEOUT: return "device pipeline wait timed out";
    case PAIR_ERR_ALLOC_INPUT: return "allocation input out of range or not finite";
    case PAIR_ERR_ALLOC_INFEASIBLE: return "allocation budget below pi_min times the summed cost";
  }
  return "unknown status";
}

int32_t pair_last_launch_count(void) { return g_log.launches; }

void pair_timing_enable(int32_t on) {
  g_log.timing = on != 0;
  g_log.n = 0;
}

int32_t pair_timing_read(int32_t max, float *ms, const char **names) {
  LaunchLog &L = g_log;
  const int n = L.n < max ? L.n : max;
  for (int i = 0; i < n; ++i) {
    float t = -1.f;
    if (cudaEventSynchronize(L.rec[i].stop) == cudaSuccess)
      cudaEventElapsedTime(&t, L.rec[i].start, L.rec[i].stop);
    if (ms) ms[i] = t;
    if (names) names[i] = L.rec[i].name;
  }
  L.n = 0;
  return n;
}

}  // extern "C"
