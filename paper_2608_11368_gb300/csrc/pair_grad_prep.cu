// pair_grad bookkeeping kernels: active-token compaction, per-rollout and
// total objective, exact one-hot gradient parts, workspace layout.
//
// The objective of Sec. 4.5 is sum_i a_i log pi(o_i | q) with log pi a sum
// over response tokens; rollouts with a_i == 0 contribute nothing and are
// removed before any head arithmetic. The surviving tokens are packed in
// their original order (rollout by rollout), so every per-rollout sum below
// runs over a contiguous range in a fixed order (bit-reproducible).
#include <cuda_bf16.h>

#include "pair_common.cuh"

namespace pairk {
namespace {

constexpr int kNSplit = 16;  // vocabulary splits of the log-sum-exp pass

__device__ __forceinline__ bool coef_nonzero(float a) {
  return (__float_as_uint(a) & 0x7fffffffu) != 0u;
}

__device__ __forceinline__ int clamp_i(int v, int lo, int hi) {
  return v < lo ? lo : (v > hi ? hi : v);
}

// Counts the active tokens of each rollout; validates every mask=1 target.
__global__ void seg_count_kernel(int R, int T, int V, const int32_t *cu,
                                 const uint8_t *mask, const int32_t *y,
                                 const float *a, int32_t *seg_cnt,
                                 int32_t *dev_err) {
  const int i = blockIdx.x;
  const int beg = clamp_i(cu[i], 0, T), end = clamp_i(cu[i + 1], beg, T);
  const bool on = coef_nonzero(a[i]);
  int n = 0, bad = 0;
  for (int t = beg + threadIdx.x; t < end; t += blockDim.x) {
    if (mask[t]) {
      ++n;
      const int yt = y[t];
      bad |= (yt < 0 || yt >= V);
    }
  }
  for (int o = 16; o > 0; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
  __shared__ int red[32];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = n;
  if (bad) flag_error(dev_err, PAIR_DEV_ERR_TARGET_RANGE);
  __syncthreads();
  if (threadIdx.x == 0) {
    int s = 0;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) s += red[k];
    seg_cnt[i] = on ? s : 0;
  }
}

// Exclusive prefix over rollouts (one block, sequential chunks of 1024).
__global__ void seg_scan_kernel(int R, const int32_t *seg_cnt, int32_t *seg_off,
                                int32_t *counters) {
  __shared__ int buf[1024];
  __shared__ int carry;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int base = 0; base < R; base += 1024) {
    const int i = base + threadIdx.x;
    const int v = i < R ? seg_cnt[i] : 0;
    buf[threadIdx.x] = v;
    __syncthreads();
    for (int o = 1; o < 1024; o <<= 1) {
      const int add = threadIdx.x >= o ? buf[threadIdx.x - o] : 0;
      __syncthreads();
      buf[threadIdx.x] += add;
      __syncthreads();
    }
    if (i < R) seg_off[i] = carry + buf[threadIdx.x] - v;
    __syncthreads();
    if (threadIdx.x == 1023) carry += buf[1023];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    seg_off[R] = carry;
    counters[0] = carry;
  }
}

// In-order compaction of each active rollout's mask=1 tokens.
__global__ void gather_kernel(int R, int T, const int32_t *cu,
                              const uint8_t *mask, const int32_t *y,
                              const float *a, const int32_t *seg_off,
                              int32_t *tok_idx, int32_t *tok_y, float *tok_c) {
  const int i = blockIdx.x;
  if (!coef_nonzero(a[i])) return;
  const int beg = clamp_i(cu[i], 0, T), end = clamp_i(cu[i + 1], beg, T);
  const float c = a[i];
  __shared__ int wsum[32];
  __shared__ int carry;
  if (threadIdx.x == 0) carry = seg_off[i];
  __syncthreads();
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int nw = blockDim.x >> 5;
  for (int base = beg; base < end; base += blockDim.x) {
    const int t = base + threadIdx.x;
    const int f = (t < end && mask[t]) ? 1 : 0;
    const unsigned bal = __ballot_sync(0xffffffffu, f);
    const int rank_w = __popc(bal & ((1u << lane) - 1u));
    if (lane == 0) wsum[w] = __popc(bal);
    __syncthreads();
    int before = 0, total = 0;
    for (int k = 0; k < nw; ++k) {
      before += (k < w) ? wsum[k] : 0;
      total += wsum[k];
    }
    if (f) {
      const int p = carry + before + rank_w;
      tok_idx[p] = t;
      tok_y[p] = y[t];
      tok_c[p] = c;
    }
    __syncthreads();
    if (threadIdx.x == 0) carry += total;
    __syncthreads();
  }
}

// Hc[p] = H[tok_idx[p]] for p < T_eff; zero rows up to the next multiple of
// 128 (the token-tile height), so tail tiles carry finite zeros.
template <typename Tin>
__global__ void copy_rows_kernel(int64_t Tpad, int d, const int32_t *counters,
                                 const int32_t *tok_idx, const Tin *H, Tin *Hc) {
  const int Teff = counters[0];
  const int64_t Tz = ((int64_t)Teff + 127) / 128 * 128;
  const int vec = 16 / (int)sizeof(Tin);
  const int dv = d / vec;
  for (int64_t p = blockIdx.x; p < Tz && p < Tpad; p += gridDim.x) {
    uint4 *dst = reinterpret_cast<uint4 *>(Hc + p * d);
    if (p < Teff) {
      const uint4 *src = reinterpret_cast<const uint4 *>(H + (int64_t)tok_idx[p] * d);
      for (int k = threadIdx.x; k < dv; k += blockDim.x) dst[k] = src[k];
    } else {
      for (int k = threadIdx.x; k < dv; k += blockDim.x) dst[k] = make_uint4(0, 0, 0, 0);
    }
  }
}

// Zero the dH rows of tokens outside the objective (mask = 0 or a = 0).
constexpr int kZeroCuSmem = 8192;  // rollout offsets staged in shared memory, at most

__global__ void zero_inactive_rows_kernel(int64_t T, int d, int R,
                                          const int32_t *cu,
                                          const uint8_t *mask, const float *a,
                                          float *dH) {
  // The rollout offsets are searched once per row by every thread: from
  // shared memory when they fit, so the search costs no global round trips.
  extern __shared__ int32_t cu_s[];
  const bool staged = R + 1 <= kZeroCuSmem;
  if (staged)
    for (int i = threadIdx.x; i <= R; i += blockDim.x) cu_s[i] = cu[i];
  __syncthreads();
  const int32_t *cs = staged ? cu_s : cu;
  for (int64_t t = blockIdx.x; t < T; t += gridDim.x) {
    // rollout of t: last i with cu[i] <= t
    int lo = 0, hi = R - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (cs[mid] <= t) lo = mid; else hi = mid - 1;
    }
    const bool live = mask[t] && coef_nonzero(a[lo]) && cs[lo] <= t && t < cs[lo + 1];
    if (live) continue;
    float4 *row = reinterpret_cast<float4 *>(dH + t * d);
    if ((d & 3) == 0) {
      for (int k = threadIdx.x; k < d / 4; k += blockDim.x)
        row[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    } else {
      for (int k = threadIdx.x; k < d; k += blockDim.x) dH[t * d + k] = 0.f;
    }
  }
}

// Per-rollout sum of logp_t = zy - lse over the rollout's compacted range
// (fp64, fixed tree order).
__global__ void seg_logp_kernel(int R, const int32_t *seg_off, const float *zy,
                                const float *lse, double *seg_logp) {
  const int i = blockIdx.x;
  const int beg = seg_off[i], end = seg_off[i + 1];
  double s = 0.0;
  for (int p = beg + threadIdx.x; p < end; p += blockDim.x)
    s += (double)zy[p] - (double)lse[p];
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  __shared__ double red[32];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) t += red[k];
    seg_logp[i] = t;
  }
}

// Jobj = sum_i a_i * logp_seq_i (fp64, fixed order); logp_seq out.
__global__ void objective_kernel(int R, const float *a, const double *seg_logp,
                                 double *Jobj, float *logp_seq) {
  __shared__ double red[32];
  double s = 0.0;
  for (int i = threadIdx.x; i < R; i += blockDim.x) {
    const bool on = coef_nonzero(a[i]);
    const double lp = on ? seg_logp[i] : 0.0;
    if (logp_seq) logp_seq[i] = (float)lp;
    s += on ? (double)a[i] * lp : 0.0;
  }
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) t += red[k];
    *Jobj = t;
  }
}

// Eight consecutive elements as fp32.
__device__ __forceinline__ void load8(const __nv_bfloat16 *h, float (&x)[8]) {
  const uint4 u = *reinterpret_cast<const uint4 *>(h);
  const __nv_bfloat162 *b = reinterpret_cast<const __nv_bfloat162 *>(&u);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __bfloat1622float2(b[i]);
    x[2 * i] = f.x;
    x[2 * i + 1] = f.y;
  }
}
__device__ __forceinline__ void load8(const float *h, float (&x)[8]) {
  const float4 a = reinterpret_cast<const float4 *>(h)[0];
  const float4 b = reinterpret_cast<const float4 *>(h)[1];
  x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w;
  x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
}

// dH_t += c_t W[y_t]  (the one-hot part of dJ/dh_t, exact in fp32): 8
// columns per thread with vector accesses (d is a multiple of 8 on both
// paths), two tokens in flight per block.
template <typename Tin>
__global__ void onehot_dh_kernel(int d, const int32_t *counters,
                                 const int32_t *tok_idx, const int32_t *tok_y,
                                 const float *tok_c, const Tin *W, float *dH) {
  const int Teff = counters[0];
  const int d8 = d / 8;
  for (int p0 = 2 * blockIdx.x; p0 < Teff; p0 += 2 * gridDim.x) {
    const bool two = p0 + 1 < Teff;
    const float c0 = tok_c[p0], c1 = two ? tok_c[p0 + 1] : 0.f;
    const Tin *w0 = W + (int64_t)tok_y[p0] * d;
    const Tin *w1 = two ? W + (int64_t)tok_y[p0 + 1] * d : w0;
    float *r0 = dH + (int64_t)tok_idx[p0] * d;
    float *r1 = two ? dH + (int64_t)tok_idx[p0 + 1] * d : r0;
    for (int k8 = threadIdx.x; k8 < d8; k8 += blockDim.x) {
      const int k = 8 * k8;
      float x0[8], x1[8];
      load8(w0 + k, x0);
      float4 a0 = reinterpret_cast<float4 *>(r0 + k)[0];
      float4 b0 = reinterpret_cast<float4 *>(r0 + k)[1];
      float4 a1 = a0, b1 = b0;
      if (two) {
        load8(w1 + k, x1);
        a1 = reinterpret_cast<float4 *>(r1 + k)[0];
        b1 = reinterpret_cast<float4 *>(r1 + k)[1];
      }
      reinterpret_cast<float4 *>(r0 + k)[0] =
          make_float4(fmaf(c0, x0[0], a0.x), fmaf(c0, x0[1], a0.y), fmaf(c0, x0[2], a0.z),
                      fmaf(c0, x0[3], a0.w));
      reinterpret_cast<float4 *>(r0 + k)[1] =
          make_float4(fmaf(c0, x0[4], b0.x), fmaf(c0, x0[5], b0.y), fmaf(c0, x0[6], b0.z),
                      fmaf(c0, x0[7], b0.w));
      if (two) {
        reinterpret_cast<float4 *>(r1 + k)[0] =
            make_float4(fmaf(c1, x1[0], a1.x), fmaf(c1, x1[1], a1.y), fmaf(c1, x1[2], a1.z),
                        fmaf(c1, x1[3], a1.w));
        reinterpret_cast<float4 *>(r1 + k)[1] =
            make_float4(fmaf(c1, x1[4], b1.x), fmaf(c1, x1[5], b1.y), fmaf(c1, x1[6], b1.z),
                        fmaf(c1, x1[7], b1.w));
      }
    }
  }
}

// dW_v += sum_{t: y_t = v} c_t h_t (the one-hot part of dJ/dW_v), exact in
// fp32, tokens added in their packed order. The compacted tokens are grouped
// by target bucket (kOneHotBucket vocabulary rows): counts, offsets and a
// fill (in any order); then one warp owns a bucket and puts its tokens in
// packed order: up to 32 by a bitonic sort in registers, up to
// kOneHotRankMax by ranking each against all others into shared memory; a
// heavier bucket instead scans the compacted targets in order for its rows
// (four 32-token chunks per round, so the target loads overlap). A row is
// updated with 16-byte vector accesses when d allows it.
template <typename Tin>
__device__ __forceinline__ void axpy_row(int d, float c, const Tin *__restrict__ h,
                                         float *__restrict__ row, int lane) {
  if ((d & 7) == 0) {
    for (int k0 = lane * 8; k0 < d; k0 += 32 * 8 * 2) {
      // Two independent 8-element groups per iteration.
      const int k1 = k0 + 32 * 8;
      float x0[8], x1[8];
      load8(h + k0, x0);
      float4 r0a = reinterpret_cast<float4 *>(row + k0)[0];
      float4 r0b = reinterpret_cast<float4 *>(row + k0)[1];
      float4 r1a = make_float4(0.f, 0.f, 0.f, 0.f), r1b = r1a;
      const bool has1 = k1 < d;
      if (has1) {
        load8(h + k1, x1);
        r1a = reinterpret_cast<float4 *>(row + k1)[0];
        r1b = reinterpret_cast<float4 *>(row + k1)[1];
      }
      r0a = make_float4(fmaf(c, x0[0], r0a.x), fmaf(c, x0[1], r0a.y), fmaf(c, x0[2], r0a.z),
                        fmaf(c, x0[3], r0a.w));
      r0b = make_float4(fmaf(c, x0[4], r0b.x), fmaf(c, x0[5], r0b.y), fmaf(c, x0[6], r0b.z),
                        fmaf(c, x0[7], r0b.w));
      reinterpret_cast<float4 *>(row + k0)[0] = r0a;
      reinterpret_cast<float4 *>(row + k0)[1] = r0b;
      if (has1) {
        r1a = make_float4(fmaf(c, x1[0], r1a.x), fmaf(c, x1[1], r1a.y), fmaf(c, x1[2], r1a.z),
                          fmaf(c, x1[3], r1a.w));
        r1b = make_float4(fmaf(c, x1[4], r1b.x), fmaf(c, x1[5], r1b.y), fmaf(c, x1[6], r1b.z),
                          fmaf(c, x1[7], r1b.w));
        reinterpret_cast<float4 *>(row + k1)[0] = r1a;
        reinterpret_cast<float4 *>(row + k1)[1] = r1b;
      }
    }
  } else {
    for (int k = lane; k < d; k += 32) row[k] = fmaf(c, (float)h[k], row[k]);
  }
}

__global__ void onehot_count_kernel(const int32_t *counters, const int32_t *tok_y,
                                    int32_t *cnt) {
  const int Teff = counters[0];
  for (int p = blockIdx.x * blockDim.x + threadIdx.x; p < Teff; p += gridDim.x * blockDim.x)
    atomicAdd(&cnt[tok_y[p] / kOneHotBucket], 1);
}

// off[b] = sum of cnt[< b] for b <= nb (one block of 1024 threads).
__global__ void __launch_bounds__(1024) onehot_scan_kernel(int nb, const int32_t *cnt,
                                                           int32_t *off) {
  __shared__ int32_t wsum[32];
  __shared__ int32_t carry;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int base = 0; base <= nb; base += 1024) {
    const int b = base + threadIdx.x;
    const int v = b < nb ? cnt[b] : 0;
    int x = v;  // inclusive warp scan
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) wsum[warp] = x;
    __syncthreads();
    if (warp == 0) {
      int w = wsum[lane];
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += y;
      }
      wsum[lane] = w;
    }
    __syncthreads();
    const int excl = carry + (warp ? wsum[warp - 1] : 0) + x - v;
    if (b <= nb) off[b] = excl;
    __syncthreads();
    if (threadIdx.x == 1023) carry = excl + v;
    __syncthreads();
  }
}

__global__ void onehot_fill_kernel(const int32_t *counters, const int32_t *tok_y,
                                   const int32_t *off, int32_t *fill, int32_t *blist) {
  const int Teff = counters[0];
  for (int p = blockIdx.x * blockDim.x + threadIdx.x; p < Teff; p += gridDim.x * blockDim.x) {
    const int b = tok_y[p] / kOneHotBucket;
    blist[off[b] + atomicAdd(&fill[b], 1)] = p;
  }
}

// row += c h over d elements by 8 lanes (lane8 = lane index within them).
template <typename Tin>
__device__ __forceinline__ void axpy_row8(int d, float c, const Tin *__restrict__ h,
                                          float *__restrict__ row, int lane8) {
  if ((d & 7) == 0) {
    for (int k0 = lane8 * 8; k0 < d; k0 += 64) {
      float x[8];
      load8(h + k0, x);
      float4 ra = reinterpret_cast<float4 *>(row + k0)[0];
      float4 rb = reinterpret_cast<float4 *>(row + k0)[1];
      ra = make_float4(fmaf(c, x[0], ra.x), fmaf(c, x[1], ra.y), fmaf(c, x[2], ra.z),
                       fmaf(c, x[3], ra.w));
      rb = make_float4(fmaf(c, x[4], rb.x), fmaf(c, x[5], rb.y), fmaf(c, x[6], rb.z),
                       fmaf(c, x[7], rb.w));
      reinterpret_cast<float4 *>(row + k0)[0] = ra;
      reinterpret_cast<float4 *>(row + k0)[1] = rb;
    }
  } else {
    for (int k = lane8; k < d; k += 8) row[k] = fmaf(c, (float)h[k], row[k]);
  }
}

// Adds the one-hot terms of tokens q_0 < q_1 < ... (packed positions, given
// by get(i), i < n) in that order per target row: four consecutive tokens at
// a time, 8 lanes each, when their four rows differ; one at a time otherwise.
template <typename Tin, typename Get>
__device__ __forceinline__ void onehot_apply_sorted(int d, int n, Get get, const int32_t *tok_y,
                                                    const float *tok_c, const Tin *Hc,
                                                    float *dW, int lane) {
  int i = 0;
  while (i < n) {
    if (i + 4 <= n) {
      const int q0 = get(i), q1 = get(i + 1), q2 = get(i + 2), q3 = get(i + 3);
      const int y0 = tok_y[q0], y1 = tok_y[q1], y2 = tok_y[q2], y3 = tok_y[q3];
      if (y0 != y1 && y0 != y2 && y0 != y3 && y1 != y2 && y1 != y3 && y2 != y3) {
        const int g = lane >> 3;
        const int q = g == 0 ? q0 : g == 1 ? q1 : g == 2 ? q2 : q3;
        const int y = g == 0 ? y0 : g == 1 ? y1 : g == 2 ? y2 : y3;
        axpy_row8(d, tok_c[q], Hc + (int64_t)q * d, dW + (int64_t)y * d, lane & 7);
        __syncwarp();
        i += 4;
        continue;
      }
    }
    const int q = get(i);
    axpy_row(d, tok_c[q], Hc + (int64_t)q * d, dW + (int64_t)tok_y[q] * d, lane);
    __syncwarp();
    ++i;
  }
}

constexpr int kOneHotRankMax = 512;  // bucket tokens ranked in shared memory, at most

template <typename Tin>
__global__ void __launch_bounds__(256)
    onehot_dw_kernel(int d, int V, int nb, const int32_t *counters, const int32_t *tok_y,
                     const float *tok_c, const int32_t *off, const int32_t *blist,
                     const Tin *Hc, float *dW) {
  __shared__ int32_t sorted[8][kOneHotRankMax];  // per warp of the block
  const int bk = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (bk >= nb) return;
  const int b0 = off[bk], n = off[bk + 1] - b0;
  if (n == 0) return;
  if (n > 32 && n <= kOneHotRankMax) {
    // Rank each token against all others of the bucket (positions are
    // distinct), then add them in rank order.
    int32_t *srt = sorted[threadIdx.x >> 5];
    for (int i = lane; i < n; i += 32) {
      const int p = blist[b0 + i];
      int rank = 0;
      for (int j = 0; j < n; ++j) rank += blist[b0 + j] < p ? 1 : 0;
      srt[rank] = p;
    }
    __syncwarp();
    onehot_apply_sorted(d, n, [&](int i) { return srt[i]; }, tok_y, tok_c, Hc, dW, lane);
    return;
  }
  if (n <= 32) {
    // Bitonic sort of the bucket's packed positions across the warp.
    int p = lane < n ? blist[b0 + lane] : 0x7fffffff;
#pragma unroll
    for (int k = 2; k <= 32; k <<= 1)
#pragma unroll
      for (int j = k >> 1; j > 0; j >>= 1) {
        const int q = __shfl_xor_sync(0xffffffffu, p, j);
        p = (((lane & j) == 0) == ((lane & k) == 0)) ? min(p, q) : max(p, q);
      }
    onehot_apply_sorted(
        d, n, [&](int i) { return __shfl_sync(0xffffffffu, p, i); }, tok_y, tok_c, Hc, dW, lane);
    return;
  }
  const int v0 = bk * kOneHotBucket;
  const int v1 = min(V, v0 + kOneHotBucket);
  const int Teff = counters[0];
  for (int base = 0; base < Teff; base += 128) {
    int yt[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int pp = base + 32 * i + lane;
      yt[i] = pp < Teff ? tok_y[pp] : -1;
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      unsigned hit = __ballot_sync(0xffffffffu, yt[i] >= v0 && yt[i] < v1);
      while (hit) {
        const int src = __ffs(hit) - 1;
        hit &= hit - 1;
        const int q = base + 32 * i + src;
        const int v = __shfl_sync(0xffffffffu, yt[i], src);
        axpy_row(d, tok_c[q], Hc + (int64_t)q * d, dW + (int64_t)v * d, lane);
      }
    }
  }
}

// Clipped trajectory-ratio surrogate of the practical PPO epochs (Sec. 4.5,
// App. "Practical departures"): for rollout i with detached coefficient
// A_i = a_i and ratio rho_i = exp(logp_seq_i - logp_old_i),
//   L_i = min(rho_i A_i, clip(rho_i, 1 - eps, 1 + eps) A_i),
// and the gradient coefficient c_i = A_i rho_i where the unclipped term is the
// minimum (A_i > 0: rho_i <= 1 + eps; A_i < 0: rho_i >= 1 - eps), else 0.
// The ratio is formed in fp64 from the fp64 per-rollout log-probability.
__global__ void ppo_coef_kernel(int R, const float *a, const double *seg_logp,
                                const float *logp_old, float eps, float *c, double *L,
                                float *coef_out) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < R; i += gridDim.x * blockDim.x) {
    const double A = (double)a[i];
    float ci = 0.f;
    double li = 0.0;
    if (coef_nonzero(a[i])) {
      const double ratio = exp(seg_logp[i] - (double)logp_old[i]);
      const double lo = 1.0 - (double)eps, hi = 1.0 + (double)eps;
      const double clipped = ratio < lo ? lo : (ratio > hi ? hi : ratio);
      const double u = ratio * A, v = clipped * A;
      li = u < v ? u : v;
      const bool unclipped = A > 0.0 ? ratio <= hi : ratio >= lo;
      ci = unclipped ? (float)(A * ratio) : 0.f;
    }
    c[i] = ci;
    L[i] = li;
    if (coef_out) coef_out[i] = ci;
  }
}

// tok_c[p] = c_i for every compacted token p of rollout i.
__global__ void retarget_c_kernel(int R, const int32_t *seg_off, const float *c, float *tok_c) {
  const int i = blockIdx.x;
  const int beg = seg_off[i], end = seg_off[i + 1];
  const float ci = c[i];
  for (int p = beg + threadIdx.x; p < end; p += blockDim.x) tok_c[p] = ci;
}

// Jobj = sum_i L_i (fp64, fixed order); logp_seq out as in objective_kernel.
__global__ void ppo_objective_kernel(int R, const float *a, const double *seg_logp,
                                     const double *L, double *Jobj, float *logp_seq) {
  __shared__ double red[32];
  double s = 0.0;
  for (int i = threadIdx.x; i < R; i += blockDim.x) {
    const bool on = coef_nonzero(a[i]);
    if (logp_seq) logp_seq[i] = on ? (float)seg_logp[i] : 0.f;
    s += L[i];
  }
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) t += red[k];
    *Jobj = t;
  }
}

// logp_tok[t] = 0 for every packed token (the scatter below then fills the
// active ones).
__global__ void zero_f32_kernel(int64_t n, float *x) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    x[i] = 0.f;
}

// logp_tok[tok_idx[p]] = zy[p] - lse[p] for every compacted token p.
__global__ void scatter_logp_kernel(const int32_t *counters, const int32_t *tok_idx,
                                    const float *zy, const float *lse, float *logp_tok) {
  const int Teff = counters[0];
  for (int p = blockIdx.x * blockDim.x + threadIdx.x; p < Teff; p += gridDim.x * blockDim.x)
    logp_tok[tok_idx[p]] = zy[p] - lse[p];
}

}  // namespace

size_t grad_workspace_bytes(int64_t T, int32_t d, int32_t V, int32_t R,
                            pair_dtype dt, GradWorkspace *out, void *base, int gimg_rb) {
  const int64_t Tpad = (T + 127) / 128 * 128 + 128;
  const size_t esz = dt == PAIR_BF16 ? 2 : 4;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += (bytes + 255) / 256 * 256;
    return o;
  };
  const size_t o_cnt = take(64 * sizeof(int32_t));
  const size_t o_segc = take((size_t)R * 4);
  const size_t o_sego = take((size_t)(R + 1) * 4);
  const size_t o_idx = take((size_t)Tpad * 4);
  const size_t o_y = take((size_t)Tpad * 4);
  const size_t o_c = take((size_t)Tpad * 4);
  const size_t o_lse = take((size_t)Tpad * 4);
  const size_t o_zy = take((size_t)Tpad * 4);
  const size_t o_part = take((size_t)kNSplit * Tpad * sizeof(float2));
  const size_t o_segl = take((size_t)R * 8);
  const size_t o_ppoc = take((size_t)R * 4);
  const size_t o_ppol = take((size_t)R * 8);
  const size_t o_hc = take((size_t)Tpad * d * esz);
  const size_t nb = (size_t)((V + kOneHotBucket - 1) / kOneHotBucket);
  const size_t o_bkt = take(3 * (nb + 1) * 4);
  const size_t o_blist = take((size_t)Tpad * 4);
  const size_t o_ring = dt == PAIR_BF16 ? take((size_t)kMaxClusters * kRingBytesPerCluster) : off;
  const bool cl = dt == PAIR_BF16 && grad_cluster_path(d);
  // Hidden sizes the image backward takes (grad_gimg_rows): per-token
  // reference and softmax sum of its log-sum-exp pass.
  const bool img = dt == PAIR_BF16 && d >= 512 && d % 512 == 0;
  const size_t o_tail = cl ? take((size_t)kMaxClusters * 2 * 128 * d * sizeof(float)) : off;
  const int n_rbmax = (int)(Tpad / 128);
  const int n_slots = n_rbmax + 2 * kMaxClusters;
  const size_t o_ref = (cl || img) ? take((size_t)Tpad * 4) : off;
  const size_t o_mrow = (cl || img) ? take((size_t)Tpad * 4) : off;
  const size_t o_lsum = img ? take((size_t)Tpad * 4) : off;
  const size_t o_prog = img ? take((size_t)kMaxPairs * 4) : off;
  const size_t o_rbflag = cl ? take((size_t)n_rbmax * 4) : off;
  const size_t o_rblist = cl ? take((size_t)n_rbmax * 4) : off;
  const size_t o_ready = cl ? take((size_t)n_slots * 4) : off;
  const size_t o_lpart = cl ? take((size_t)n_slots * 8 * 256 * 4) : off;
  const size_t o_taill = cl ? take((size_t)kMaxClusters * 2 * 256 * 4) : off;
  // The image comes last, so that a larger workspace only adds token blocks.
  const size_t n_vt = (size_t)((V + 127) / 128);
  const size_t o_gimg = gimg_rb ? take((size_t)gimg_rb * n_vt * kGImgTileBytes) : off;
  const size_t o_hs = gimg_rb ? take((size_t)gimg_rb * 128 * d * 2) : off;
  if (out) {
    char *b = static_cast<char *>(base);
    out->counters = reinterpret_cast<int32_t *>(b + o_cnt);
    out->seg_cnt = reinterpret_cast<int32_t *>(b + o_segc);
    out->seg_off = reinterpret_cast<int32_t *>(b + o_sego);
    out->tok_idx = reinterpret_cast<int32_t *>(b + o_idx);
    out->tok_y = reinterpret_cast<int32_t *>(b + o_y);
    out->tok_c = reinterpret_cast<float *>(b + o_c);
    out->lse = reinterpret_cast<float *>(b + o_lse);
    out->zy = reinterpret_cast<float *>(b + o_zy);
    out->part = reinterpret_cast<float2 *>(b + o_part);
    out->seg_logp = reinterpret_cast<double *>(b + o_segl);
    out->ppo_c = reinterpret_cast<float *>(b + o_ppoc);
    out->ppo_L = reinterpret_cast<double *>(b + o_ppol);
    out->Hc = b + o_hc;
    out->bkt = reinterpret_cast<int32_t *>(b + o_bkt);
    out->blist = reinterpret_cast<int32_t *>(b + o_blist);
    out->gring = b + o_ring;
    out->tailbuf = cl ? reinterpret_cast<float *>(b + o_tail) : nullptr;
    out->ref = (cl || img) ? reinterpret_cast<float *>(b + o_ref) : nullptr;
    out->mrow = (cl || img) ? reinterpret_cast<float *>(b + o_mrow) : nullptr;
    out->lsum = img ? reinterpret_cast<float *>(b + o_lsum) : nullptr;
    out->prog = img ? reinterpret_cast<int32_t *>(b + o_prog) : nullptr;
    out->rbflag = cl ? reinterpret_cast<int32_t *>(b + o_rbflag) : nullptr;
    out->rb_list = cl ? reinterpret_cast<int32_t *>(b + o_rblist) : nullptr;
    out->ready = cl ? reinterpret_cast<int32_t *>(b + o_ready) : nullptr;
    out->lpart = cl ? reinterpret_cast<float *>(b + o_lpart) : nullptr;
    out->tail_l = cl ? reinterpret_cast<float *>(b + o_taill) : nullptr;
    out->n_rbmax = n_rbmax;
    out->n_slots = n_slots;
    out->gimg = gimg_rb ? b + o_gimg : nullptr;
    out->hs = gimg_rb ? b + o_hs : nullptr;
    out->gimg_rb = gimg_rb;
    out->Tpad = Tpad;
    out->nsplit = kNSplit;
  }
  return off;
}

int grad_gimg_rows_fit(int64_t T, int32_t d, int32_t V, int32_t R, pair_dtype dt,
                       size_t ws_bytes) {
  const size_t base = grad_workspace_bytes(T, d, V, R, dt, nullptr, nullptr, 0);
  if (ws_bytes < base) return -1;
  const int pref = grad_gimg_rows(T, d, V, dt);
  if (pref == 0) return 0;
  const size_t fit = (ws_bytes - base) / grad_image_block_bytes(d, V);
  return fit < (size_t)pref ? (int)fit : pref;
}

pair_status grad_prepare(const GradArgs &g, const GradWorkspace &w,
                         cudaStream_t s) {
  PAIR_BEGIN("seg_count", s);
  seg_count_kernel<<<g.R, 256, 0, s>>>(g.R, (int)g.T, g.V, g.cu, g.mask, g.y,
                                       g.a, w.seg_cnt, g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("seg_scan", s);
  seg_scan_kernel<<<1, 1024, 0, s>>>(g.R, w.seg_cnt, w.seg_off, w.counters);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("gather", s);
  gather_kernel<<<g.R, 256, 0, s>>>(g.R, (int)g.T, g.cu, g.mask, g.y, g.a,
                                    w.seg_off, w.tok_idx, w.tok_y, w.tok_c);
  PAIR_LAUNCH_CHECK(s);
  const int rows_grid = 152 * 16;
  PAIR_BEGIN("copy_rows", s);
  if (g.dt == PAIR_BF16)
    copy_rows_kernel<uint16_t><<<rows_grid, 128, 0, s>>>(
        w.Tpad, g.d, w.counters, w.tok_idx,
        static_cast<const uint16_t *>(g.H), static_cast<uint16_t *>(w.Hc));
  else
    copy_rows_kernel<float><<<rows_grid, 128, 0, s>>>(
        w.Tpad, g.d, w.counters, w.tok_idx, static_cast<const float *>(g.H),
        static_cast<float *>(w.Hc));
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("zero_inactive", s);
  const size_t cu_smem = g.R + 1 <= kZeroCuSmem ? (size_t)(g.R + 1) * sizeof(int32_t) : 0;
  zero_inactive_rows_kernel<<<rows_grid, 128, cu_smem, s>>>(g.T, g.d, g.R, g.cu,
                                                            g.mask, g.a, g.dH);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

pair_status grad_finalize(const GradArgs &g, const GradWorkspace &w,
                          cudaStream_t s) {
  PAIR_BEGIN("seg_logp", s);
  seg_logp_kernel<<<g.R, 256, 0, s>>>(g.R, w.seg_off, w.zy, w.lse, w.seg_logp);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("objective", s);
  objective_kernel<<<1, 1024, 0, s>>>(g.R, g.a, w.seg_logp, g.Jobj,
                                      g.logp_seq);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

pair_status grad_token_logp(int64_t T, const GradWorkspace &w, float *logp_tok,
                            cudaStream_t s) {
  PAIR_BEGIN("zero_logp", s);
  zero_f32_kernel<<<152 * 4, 256, 0, s>>>(T, logp_tok);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("scatter_logp", s);
  scatter_logp_kernel<<<152 * 4, 256, 0, s>>>(w.counters, w.tok_idx, w.zy, w.lse, logp_tok);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

pair_status grad_ppo_coefficients(const GradArgs &g, const GradWorkspace &w,
                                  const float *logp_old, float eps, float *coef_out,
                                  cudaStream_t s) {
  PAIR_BEGIN("seg_logp", s);
  seg_logp_kernel<<<g.R, 256, 0, s>>>(g.R, w.seg_off, w.zy, w.lse, w.seg_logp);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("ppo_coef", s);
  ppo_coef_kernel<<<(int)ceil_div(g.R, 256), 256, 0, s>>>(g.R, g.a, w.seg_logp, logp_old, eps,
                                                          w.ppo_c, w.ppo_L, coef_out);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("retarget_c", s);
  retarget_c_kernel<<<g.R, 256, 0, s>>>(g.R, w.seg_off, w.ppo_c, w.tok_c);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

pair_status grad_ppo_finalize(const GradArgs &g, const GradWorkspace &w, cudaStream_t s) {
  PAIR_BEGIN("ppo_objective", s);
  ppo_objective_kernel<<<1, 1024, 0, s>>>(g.R, g.a, w.seg_logp, w.ppo_L, g.Jobj, g.logp_seq);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

pair_status grad_onehot(const GradArgs &g, const GradWorkspace &w,
                        cudaStream_t s) {
  const int nb = (g.V + kOneHotBucket - 1) / kOneHotBucket;
  int32_t *cnt = w.bkt, *off = w.bkt + (nb + 1), *fill = w.bkt + 2 * (nb + 1);
  PAIR_CUDA_TRY(cudaMemsetAsync(cnt, 0, (size_t)(nb + 1) * sizeof(int32_t), s));
  PAIR_CUDA_TRY(cudaMemsetAsync(fill, 0, (size_t)(nb + 1) * sizeof(int32_t), s));
  PAIR_BEGIN("onehot_count", s);
  onehot_count_kernel<<<152 * 4, 256, 0, s>>>(w.counters, w.tok_y, cnt);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("onehot_scan", s);
  onehot_scan_kernel<<<1, 1024, 0, s>>>(nb, cnt, off);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("onehot_fill", s);
  onehot_fill_kernel<<<152 * 4, 256, 0, s>>>(w.counters, w.tok_y, off, fill, w.blist);
  PAIR_LAUNCH_CHECK(s);
  const int blocks = (int)ceil_div(nb, 8);  // 8 warps (buckets) per block
  if (g.dt == PAIR_BF16) {
    const __nv_bfloat16 *W = static_cast<const __nv_bfloat16 *>(g.W);
    PAIR_BEGIN("onehot_dh", s);
    onehot_dh_kernel<__nv_bfloat16><<<152 * 16, 256, 0, s>>>(
        g.d, w.counters, w.tok_idx, w.tok_y, w.tok_c, W, g.dH);
    PAIR_LAUNCH_CHECK(s);
    PAIR_BEGIN("onehot_dw", s);
    onehot_dw_kernel<__nv_bfloat16><<<blocks, 256, 0, s>>>(
        g.d, g.V, nb, w.counters, w.tok_y, w.tok_c, off, w.blist,
        static_cast<const __nv_bfloat16 *>(w.Hc), g.dW);
    PAIR_LAUNCH_CHECK(s);
  } else {
    PAIR_BEGIN("onehot_dh", s);
    onehot_dh_kernel<float><<<152 * 16, 256, 0, s>>>(
        g.d, w.counters, w.tok_idx, w.tok_y, w.tok_c,
        static_cast<const float *>(g.W), g.dH);
    PAIR_LAUNCH_CHECK(s);
    PAIR_BEGIN("onehot_dw", s);
    onehot_dw_kernel<float><<<blocks, 256, 0, s>>>(
        g.d, g.V, nb, w.counters, w.tok_y, w.tok_c, off, w.blist,
        static_cast<const float *>(w.Hc), g.dW);
    PAIR_LAUNCH_CHECK(s);
  }
  return PAIR_OK;
}

}  // namespace pairk
