// pair_selftest_wait_timeout: exercises the failure path of the pipeline
// waits on the GPU without faulting it. One block waits on an mbarrier that
// nothing ever arrives on, through the same bounded-wait helper every
// pipeline kernel uses, with a caller-chosen short limit; the wait gives up,
// raises the block's abort flag and ORs PAIR_DEV_ERR_TIMEOUT into the device
// error word, and the kernel returns normally.
#include "pair_common.cuh"
#include "tc_ptx.cuh"

namespace pairk {
namespace {

using namespace tc;

__global__ void selftest_timeout_kernel(long long limit, int32_t *dev_err, int32_t *seen) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);  // never arrived on
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  volatile int *abort = &abort_flag;
  bool ok = true;
  if (threadIdx.x == 0) ok = wait_limit(&bar, 0, abort, dev_err, limit);
  __syncthreads();
  // A second role sees the raised abort flag and gives up without waiting
  // out its own limit, as the pipeline roles do.
  if (threadIdx.x == 32) ok = wait_limit(&bar, 0, abort, dev_err, 1LL << 62);
  __syncthreads();
  if (threadIdx.x == 0) seen[0] = (ok ? 0 : 1) | (*abort ? 2 : 0);
  if (threadIdx.x == 32) seen[1] = ok ? 0 : 1;
}

}  // namespace
}  // namespace pairk

using namespace pairk;

extern "C" pair_status pair_selftest_wait_timeout(int64_t limit_cycles, int32_t *dev_err,
                                                  int32_t *seen, pair_stream_t stream) {
  reset_launches();
  if (!dev_err || !seen || limit_cycles <= 0 || limit_cycles > (int64_t)4000000000LL)
    return PAIR_ERR_INVALID_ARG;
  const pair_status dv = check_device();
  if (dv != PAIR_OK) return dv;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  PAIR_BEGIN("selftest_timeout", s);
  selftest_timeout_kernel<<<1, 64, 0, s>>>((long long)limit_cycles, dev_err, seen);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}
