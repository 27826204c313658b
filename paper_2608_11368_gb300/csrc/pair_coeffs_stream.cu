// Streaming coefficient kernel: the group coefficient collapse (Sec. 4.5,
// Eq. pair-advantage) with the observed-edge counts of Algorithm 1 and, for
// the weighting variants of the practical estimator (clipped,
// self-normalised), the group's weight diagnostics, for groups of at most 64
// candidates with G a multiple of 4 (the collapse itself is
// pair_coeffs_stream.cuh).
//
// Shape: a persistent grid of kSW-warp blocks, one per SM; every warp owns a
// stream of groups and stages them in its own shared memory (kStages at a
// time). With one stage per warp the SM holds as many warps as its shared
// memory allows, and the rho stream from HBM overlaps the arithmetic across
// warps: while some warps wait for their copies, the others collapse.
#include <algorithm>

#include "pair_coeffs_stream.cuh"

namespace pairk {
namespace {

constexpr int kStages = 1;  // groups staged per warp
constexpr int kSW = kStages == 1 ? 19 : 10;  // warps per block (as many as shared memory holds)

static_assert(kStages == 1 || kStages == 2, "one or two stages per warp");

struct StreamSmem {
  int Qt[kGMax];
  // Per warp: kStages stages, then the packed lists, barriers and abort flag.
  __align__(16) unsigned char warp[kSW][kStages * kStageBytes + kWarpAux];
};

template <int WM, bool DIAG>
__global__ void __launch_bounds__(kSW * 32, 1) coeffs_stream_kernel(
    int B, int G, const float *__restrict__ r, const uint8_t *__restrict__ J,
    const float *__restrict__ rho, float scale, uint32_t flags, float w_max,
    float *__restrict__ a, uint8_t *__restrict__ active, int32_t *__restrict__ edges,
    int32_t *__restrict__ contrast, float *__restrict__ ess, float *__restrict__ max_w,
    int32_t *dev_err, const StreamGeom geom) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  StreamSmem &sm = *reinterpret_cast<StreamSmem *>(smem_raw);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  // Launched as a programmatic dependent of the previous kernel in the
  // stream: a following launch of this kernel may be scheduled as soon as
  // every block got here, and its prologue (which reads no global memory)
  // overlaps this launch's tail.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  stream_qt(geom, sm.Qt);
  __syncthreads();  // the only block-wide barrier: warps are independent after it
  // Groups dealt warp-major (b = warp * blocks + block, stride all warps),
  // so every SM gets the same number of groups to within one per warp row.
  const int nw = gridDim.x * kSW;
  const int b0 = warp * gridDim.x + blockIdx.x;
  if (b0 >= B) return;  // no group for this warp (small batches)

  unsigned char *wbase = sm.warp[warp];
  unsigned char *aux = wbase + kStages * kStageBytes;
  uint64_t *bar = reinterpret_cast<uint64_t *>(aux + 64 * 4 * 3);  // one per stage
  volatile int *abort = reinterpret_cast<volatile int *>(bar + kStages);
  const int2 dg = stream_diag(G, sm.Qt);
  const RowCopies rc = stream_rows(G, sm.Qt, geom.group_bytes);
#pragma unroll
  for (int s = 0; s < kStages; ++s) stream_init_gaps(wbase + s * kStageBytes, G, sm.Qt);
  if (lane == 0) {
    for (int s = 0; s < kStages; ++s) tc::mbar_init(&bar[s], 1);
    *abort = 0;
    tc::fence_mbar_init();
  }
  __syncwarp();
  // Every global read below happens after the previous grid in the stream
  // has completed and its writes are visible.
  asm volatile("griddepcontrol.wait;" ::: "memory");

  uint32_t ph = 0;       // bit s: parity of the next completion of stage s
  uint32_t pending = 0;  // bit s: stage s has copies issued and not yet waited for
#pragma unroll
  for (int s = 0; s < kStages - 1; ++s) {
    const int b = b0 + s * nw;
    if (b < B) {
      issue_group(wbase + s * kStageBytes, &bar[s], rho, r, load_j_word(J, b, B, G), b, G, rc);
      pending |= 1u << s;
    }
  }
  // Completion flags of the next group to issue, loaded one group ahead (the
  // row copies depend on them).
  uint32_t jnext = load_j_word(J, b0 + (kStages - 1) * nw, B, G);

  int it = 0;
  for (int b = b0; b < B; b += nw, ++it) {
    const int s = it % kStages;
    {
      const int sn = (it + kStages - 1) % kStages;
      const int bn = b + (kStages - 1) * nw;
      if (bn < B) {
        issue_group(wbase + sn * kStageBytes, &bar[sn], rho, r, jnext, bn, G, rc);
        pending |= 1u << sn;
      }
      jnext = load_j_word(J, bn + nw, B, G);
    }
    if (!__all_sync(0xffffffffu, tc::wait(&bar[s], (ph >> s) & 1u, abort, dev_err)))
      break;  // timed out (error flagged); warp-uniform
    ph ^= 1u << s;
    pending &= ~(1u << s);
    __syncwarp();
    const WarpCoeffs o = warp_group_coeffs<WM, DIAG>(wbase + s * kStageBytes, sm.Qt, dg, G,
                                                     scale, flags, w_max, aux, dev_err);
    const size_t gb = (size_t)b * G;
    if (lane < G) {
      a[gb + lane] = o.a0;
      if (active) active[gb + lane] = o.act0 ? 1 : 0;
    }
    if (lane + 32 < G) {
      a[gb + lane + 32] = o.a1;
      if (active) active[gb + lane + 32] = o.act1 ? 1 : 0;
    }
    if (lane == 0) {
      if (edges) edges[b] = o.K * (o.K - 1) / 2;
      if (contrast) contrast[b] = o.C;
      if (DIAG) {
        if (ess) ess[b] = o.W2 > 0.f ? __fdiv_rn(o.W * o.W, o.W2) : 0.f;
        if (max_w) max_w[b] = o.Wmax;
      }
    }
    __syncwarp();  // the stage and the packed lists are rewritten next
  }
  // After a timed-out wait, let the copies already issued land (bounded)
  // before the block's shared memory is released.
#pragma unroll
  for (int s = 0; s < kStages; ++s)
    if (pending & (1u << s)) drain_wait(&bar[s], (ph >> s) & 1u);
}

template <int WM, bool DIAG>
pair_status launch_stream(int32_t B, int32_t G, const float *r, const uint8_t *J,
                          const float *rho, float scale, uint32_t flags, float w_max, float *a,
                          uint8_t *active, int32_t *edges, int32_t *contrast, float *ess,
                          float *max_w, int32_t *dev_err, cudaStream_t s) {
  const int smem = (int)sizeof(StreamSmem);
  PAIR_CUDA_TRY(cudaFuncSetAttribute(coeffs_stream_kernel<WM, DIAG>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
  int nsm = 0, dev = 0;
  PAIR_CUDA_TRY(cudaGetDevice(&dev));
  PAIR_CUDA_TRY(cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev));
  // One block per SM (groups are dealt warp-major, so a small batch still
  // spreads over the SMs).
  const int blocks = (int)std::min<int64_t>(B, nsm > 0 ? nsm : 1);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(blocks, 1, 1);
  cfg.blockDim = dim3(kSW * 32, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  PAIR_BEGIN(DIAG ? "coeffs_w" : "coeffs", s);
  PAIR_CUDA_TRY(cudaLaunchKernelEx(&cfg, coeffs_stream_kernel<WM, DIAG>, B, G, r, J, rho, scale,
                                   flags, w_max, a, active, edges, contrast, ess, max_w, dev_err,
                                   make_stream_geom(G)));
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

}  // namespace

bool coeffs_stream_applies(int32_t G, const float *r, const uint8_t *J, const float *rho) {
  return G >= 4 && G <= kGMax && G % 4 == 0 && rho &&
         (reinterpret_cast<uintptr_t>(rho) & 15) == 0 &&
         (reinterpret_cast<uintptr_t>(r) & 15) == 0 && (reinterpret_cast<uintptr_t>(J) & 3) == 0;
}

pair_status launch_coeffs_stream(int32_t B, int32_t G, const float *r, const uint8_t *J,
                                 const float *rho, float scale, uint32_t flags, int wmode,
                                 bool diag, float w_max, float *a, uint8_t *active,
                                 int32_t *edges, int32_t *contrast, float *ess, float *max_w,
                                 int32_t *dev_err, cudaStream_t s) {
  if (wmode == PAIR_W_HT && !diag)
    return launch_stream<PAIR_W_HT, false>(B, G, r, J, rho, scale, flags, w_max, a, active,
                                           edges, contrast, ess, max_w, dev_err, s);
  if (wmode == PAIR_W_HT)
    return launch_stream<PAIR_W_HT, true>(B, G, r, J, rho, scale, flags, w_max, a, active,
                                          edges, contrast, ess, max_w, dev_err, s);
  if (wmode == PAIR_W_CLIPPED)
    return launch_stream<PAIR_W_CLIPPED, true>(B, G, r, J, rho, scale, flags, w_max, a, active,
                                               edges, contrast, ess, max_w, dev_err, s);
  if (wmode == PAIR_W_HAJEK)
    return launch_stream<PAIR_W_HAJEK, true>(B, G, r, J, rho, scale, flags, w_max, a, active,
                                             edges, contrast, ess, max_w, dev_err, s);
  return PAIR_ERR_INVALID_ARG;
}

}  // namespace pairk
