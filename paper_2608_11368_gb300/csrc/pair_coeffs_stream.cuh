// Warp-level group coefficient collapse on a staged group (Sec. 4.5, Eq.
// pair-advantage), shared by the streaming coefficient kernel
// (pair_coeffs_stream.cu) and the dense estimator (pair_coeffs.cu), so both
// return bit-identical coefficients:
//
//   a_i = scale * 1/2 sum_{j != i} J_i J_j (r_i - r_j) w_ij,   w_ij = 1/rho_ij
//
// for groups of at most 64 candidates with G a multiple of 4.
//
// Staging: the strict upper triangle rows of the group's completed vertices
// (no other row is ever read) are copied by bulk copies (one per row)
// completing on an mbarrier, row i from column (i + 1) rounded down to a
// multiple of 4 up to G - 1; each row is preceded by a gap of at least
// 4 floats, widened so that row bases fall in different shared-memory banks
// (lanes reading one column of many rows then conflict less). Entry (i, j)
// sits at float Qt[i] + j of the stage. Gap cells hold +inf (written once),
// and after each copy the staged diagonal cells are set to +inf too, so a
// read of the diagonal, or of column G of any row (the next gap), gives
// weight 1/inf = 0. Rewards and completion flags follow the triangle.
//
// Collapse: only completed vertices take part in an edge, so the warp packs
// them to the front (K of G, vertex order); slots past K name column G. Lane
// c then sums packed row c: per term one shared-memory load of rho, one
// hardware reciprocal, one subtract, one multiply and one tree addition, with
// no mask (the diagonal and the slots past K read +inf), and a running check
// that rho >= 2^-126 (so a subnormal rho is reported like rho <= 0). Rows
// 32..K-1 (K > 32) are summed by the whole warp. Contrast edges and active
// flags follow from the rewards alone (warp match on equal rewards). Every
// sum has a fixed order (bit-identical reruns): a lane's row is a pairwise
// tree of 8-term blocks, a warp-summed row a butterfly.
#pragma once

#include "pair_coeffs_dev.cuh"
#include "tc_ptx.cuh"

namespace pairk {
namespace {

constexpr int kGMax = 64;                               // largest group of this form
constexpr int kTriFloats = 2620;                        // largest staged triangle (G = 64)
constexpr int kTriBytes = kTriFloats * 4;
constexpr int kStageBytes = kTriBytes + 256 + 64;       // triangle, r[64], J[64]
constexpr int kWarpAux = 64 * 4 * 3 + 32;               // packed r, column, Q; 2 barriers; abort
constexpr float kRhoMin = 1.17549435e-38f;              // 2^-126, smallest normal float

using tc::smem_u32;

// First staged column of upper-triangle row i (i + 1 rounded down to 4).
__host__ __device__ __forceinline__ int row_col0(int i) { return (i + 1) & ~3; }

// Butterfly reductions over the warp (every lane ends with the same value).
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Row geometry of this G (built on the host at each launch, passed by value). Row i
// (i <= G - 2) holds columns row_col0(i) .. G - 1 and starts at float D_i;
// row G - 1 has no entries and 4 gap floats follow it. Between rows there
// are at least 4 gap floats, more where needed so that the bank of Q_i =
// D_i - row_col0(i) (mod 32 words) differs from the previous three rows'.
// Qt[v] = Q_v (v <= G - 2), D_{G-1} - G (v = G - 1), 0 (v >= G): column G
// of every row, and the diagonal of a row whose staging starts at column
// i + 1, then land in a gap.
struct StreamGeom {
  int Qt[kGMax];
  uint32_t group_bytes;  // bulk-copied bytes of one group: triangle rows + rewards
};

inline StreamGeom make_stream_geom(int G) {
  StreamGeom g = {};
  int d = 4, recent[3] = {-1, -1, -1}, nrec = 0;
  uint32_t tri = 0;
  for (int i = 0; i < G; ++i) {
    if (i <= G - 2) {
      auto used = [&](int res) {
        for (int k = 0; k < 3 && k < nrec; ++k)
          if (recent[k] == res) return true;
        return false;
      };
      while (used((d - row_col0(i)) & 31)) d += 4;
      recent[nrec % 3] = (d - row_col0(i)) & 31;
      ++nrec;
      g.Qt[i] = d - row_col0(i);
      tri += (uint32_t)(G - row_col0(i));
      d += G - row_col0(i) + 4;
    } else {
      g.Qt[i] = d - G;
    }
  }
  g.group_bytes = 4u * (tri + (uint32_t)G);
  return g;
}

// Copies Qt into shared memory (threads 0..63 of the block; the caller
// synchronises before use).
__device__ __forceinline__ void stream_qt(const StreamGeom &geom, int *Qt) {
  if (threadIdx.x < kGMax) Qt[threadIdx.x] = geom.Qt[threadIdx.x];
}

// Sets the gap cells of a stage to +inf (once per stage; copies never write
// them): the cells before each row and the 4 after row G - 1. Whole warp
// calls.
__device__ __forceinline__ void stream_init_gaps(unsigned char *stage, int G, const int *Qt) {
  float *tri = reinterpret_cast<float *>(stage);
  const int lane = threadIdx.x & 31;
  const float inf = __int_as_float(0x7f800000);
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int i = lane + 32 * h;
    if (i < G) {
      const int start = (i == 0) ? 0 : Qt[i - 1] + G;  // end of row i - 1
      const int D = (i <= G - 2) ? Qt[i] + row_col0(i) : Qt[i] + G;
      for (int e = start; e < D; ++e) tri[e] = inf;
      if (i == G - 1)
        for (int e = 0; e < 4; ++e) tri[D + e] = inf;
    }
  }
}

// Float index of this lane's staged diagonal cells (rows lane, lane + 32),
// or -1 where the diagonal is not staged (it then lies in a gap).
__device__ __forceinline__ int2 stream_diag(int G, const int *Qt) {
  const int lane = threadIdx.x & 31;
  int2 d;
  d.x = (lane <= G - 2 && row_col0(lane) <= lane) ? Qt[lane] + lane : -1;
  d.y = (lane + 32 <= G - 2 && row_col0(lane + 32) <= lane + 32) ? Qt[lane + 32] + lane + 32 : -1;
  return d;
}

// This lane's share of a group's copies: triangle rows lane and lane + 32
// (one bulk copy each, rows <= G - 2), and for lane 31 the rewards.
struct RowCopies {
  int src0, src1;       // float offset within rho_g, -1 = no row
  int dst0, dst1;       // float offset within the stage
  uint32_t by0, by1;    // bytes
  uint32_t group_bytes; // bytes of all bulk copies of one group (triangle + rewards)
};

__device__ __forceinline__ RowCopies stream_rows(int G, const int *Qt, uint32_t group_bytes) {
  const int lane = threadIdx.x & 31;
  RowCopies rc;
  const int i0 = lane, i1 = lane + 32;
  rc.src0 = (i0 <= G - 2) ? i0 * G + row_col0(i0) : -1;
  rc.src1 = (i1 <= G - 2) ? i1 * G + row_col0(i1) : -1;
  rc.dst0 = (i0 <= G - 2) ? Qt[i0] + row_col0(i0) : 0;
  rc.dst1 = (i1 <= G - 2) ? Qt[i1] + row_col0(i1) : 0;
  rc.by0 = (i0 <= G - 2) ? 4u * (uint32_t)(G - row_col0(i0)) : 0u;
  rc.by1 = (i1 <= G - 2) ? 4u * (uint32_t)(G - row_col0(i1)) : 0u;
  rc.group_bytes = group_bytes;
  return rc;
}

// Bulk copy global -> this CTA's shared memory, completing on `bar`.
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes,
                                         uint64_t *bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes "
      "[%0], [%1], %2, [%3];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Bounded wait that ignores any abort flag: after a timed-out wait, lets
// the copies already issued into a stage land before the stage is released.
__device__ __forceinline__ void drain_wait(uint64_t *bar, uint32_t parity) {
  const long long t0 = clock64();
  while (!tc::mbar_try_wait(bar, parity) && clock64() - t0 < tc::kWaitCycles) {
  }
}

// This lane's 4 completion flags of group b (lanes 0 .. G/4 - 1; 0 elsewhere
// and past the last group). J is 4-byte aligned and G a multiple of 4.
__device__ __forceinline__ uint32_t load_j_word(const uint8_t *J, int b, int B, int G) {
  const int lane = threadIdx.x & 31;
  if (b >= B || lane >= (G >> 2)) return 0u;
  return __ldg(reinterpret_cast<const uint32_t *>(J + (size_t)b * G) + lane);
}

// Issues group b into `stage` (whole warp; jw = this lane's load_j_word of
// group b): the expected bytes on `bar`, a bulk copy of the triangle row of
// every completed vertex (the collapse reads no other row: an edge needs
// both endpoints completed) and of the rewards, and the completion flags
// stored from registers. The warp's earlier reads and writes of the stage
// are ordered before the copies.
__device__ __forceinline__ void issue_group(unsigned char *stage, uint64_t *bar,
                                            const float *rho, const float *r, uint32_t jw,
                                            int b, int G, const RowCopies &rc) {
  const int lane = threadIdx.x & 31;
  // Flags of rows lane and lane + 32 (byte v & 3 of lane v >> 2's word).
  const uint32_t w0 = __shfl_sync(0xffffffffu, jw, lane >> 2);
  const uint32_t w1 = __shfl_sync(0xffffffffu, jw, (lane + 32) >> 2);
  const int sh = 8 * (lane & 3);
  const bool c0 = rc.src0 >= 0 && ((w0 >> sh) & 0xffu) != 0u;
  const bool c1 = rc.src1 >= 0 && ((w1 >> sh) & 0xffu) != 0u;
  uint32_t tx = (c0 ? rc.by0 : 0u) + (c1 ? rc.by1 : 0u);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) tx += __shfl_xor_sync(0xffffffffu, tx, o);
  tx += 4u * (uint32_t)G;
  fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0) tc::mbar_expect_tx(bar, tx);
  __syncwarp();
  const float *rho_g = rho + (size_t)b * G * G;
  float *tri = reinterpret_cast<float *>(stage);
  if (c0) bulk_g2s(tri + rc.dst0, rho_g + rc.src0, rc.by0, bar);
  if (c1) bulk_g2s(tri + rc.dst1, rho_g + rc.src1, rc.by1, bar);
  if (lane == 31) bulk_g2s(stage + kTriBytes, r + (size_t)b * G, 4u * (uint32_t)G, bar);
  if (lane < (G >> 2)) reinterpret_cast<uint32_t *>(stage + kTriBytes + 256)[lane] = jw;
}

// Reciprocal by the hardware approximation (PTX rcp.approx.ftz.f32: at most
// 1 ulp, one instruction; 1/inf = 0; an input below 2^-126 counts as 0,
// which is why a completed edge's rho must be at least kRhoMin). A term (r_i - r_j) *
// rcp(rho_ij) is then within 1.5 ulp of the quotient, is exactly 0 when
// r_i = r_j, and is exactly antisymmetric (both directions use the same
// weight).
__device__ __forceinline__ float rcp_hw(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// One group's result, per lane for vertices v0 = lane and v1 = lane + 32:
// coefficients (scale applied; 0 for vertices that are not completed or
// beyond G), active flags; K, contrast edges and weight sums for the group.
struct WarpCoeffs {
  float a0, a1;
  bool act0, act1;
  int K, C;
  float W, W2, Wmax;
};

// Weight of one staged rho under weighting WM: 1/rho (HT, self-normalised)
// or min(1/rho, w_max) (clipped); +inf cells give 0.
template <int WM>
__device__ __forceinline__ float weight_of(float rho, float w_max) {
  const float w = rcp_hw(rho);
  return WM == PAIR_W_CLIPPED ? fminf(w, w_max) : w;
}

// Collapses the group staged at `stage` (whole warp calls, after the stage's
// copies completed and the warp synchronised; `dg` from stream_diag; `aux` is
// the warp's kWarpAux bytes, 16-byte aligned). WM is the weighting, DIAG
// whether the weight sums are wanted. Flags: PAIR_CENTER, PAIR_STANDARDIZE.
// A device error bit is set for rho < 2^-126 (zero, negative, subnormal) or NaN
// on a completed edge.
template <int WM, bool DIAG>
__device__ WarpCoeffs warp_group_coeffs(unsigned char *stage, const int *Qt, int2 dg, int G,
                                        float scale, uint32_t flags, float w_max,
                                        unsigned char *aux, int32_t *dev_err) {
  const int lane = threadIdx.x & 31;
  float *tri = reinterpret_cast<float *>(stage);
  const float *rs = reinterpret_cast<const float *>(stage + kTriBytes);
  const uint8_t *js = stage + kTriBytes + 256;
  float *cr = reinterpret_cast<float *>(aux);  // packed r (0 past K)
  int *co = reinterpret_cast<int *>(cr + 64);  // packed column (G past K)
  int *cq = co + 64;                           // packed Q (0 past K)
  const float inf = __int_as_float(0x7f800000);

  // Staged diagonal cells read as +inf (weight 0).
  if (dg.x >= 0) tri[dg.x] = inf;
  if (dg.y >= 0) tri[dg.y] = inf;

  // Pack the completed vertices to the front (vertex order); slots past K
  // name column G, whose cell in every row is a gap.
  const int v0 = lane, v1 = lane + 32;
  const bool j0 = v0 < G && js[v0] != 0;
  const bool j1 = v1 < G && js[v1] != 0;
  const unsigned m0 = __ballot_sync(0xffffffffu, j0);
  const unsigned m1 = __ballot_sync(0xffffffffu, j1);
  const unsigned lt = (1u << lane) - 1u;
  const int K0 = __popc(m0), K = K0 + __popc(m1);
  const int below0 = __popc(m0 & lt), below1 = __popc(m1 & lt);
  const int p0 = j0 ? below0 : K + (lane - below0);
  const int p1 = j1 ? K0 + below1 : K + (32 - K0) + (lane - below1);
  cr[p0] = j0 ? rs[v0] : 0.f;
  co[p0] = j0 ? v0 : G;
  cq[p0] = j0 ? Qt[v0] : 0;
  cr[p1] = j1 ? rs[v1] : 0.f;
  co[p1] = j1 ? v1 : G;
  cq[p1] = j1 ? Qt[v1] : 0;
  __syncwarp();

  const int c = lane;
  const bool row0 = c < K, row1 = c + 32 < K;
  const float rc = cr[c];
  const int oc = co[c], Qc = cq[c];

  // Sweep, rows 0..31: lane c sums row c over 8-term blocks (fixed 3-level
  // tree), the 8 block sums combined by a pairwise tree.
  bool ok0 = true;  // every rho read by row c is >= kRhoMin (+inf cells pass)
  float sw0 = 0.f, sq0 = 0.f, mw0 = 0.f, sum0;
  {
    float p[4];
#pragma unroll
    for (int blk = 0; blk < 8; ++blk) {
      float sblk = 0.f;
      if (blk * 8 < K) {
        const float4 ra = reinterpret_cast<const float4 *>(cr)[2 * blk];
        const float4 rb = reinterpret_cast<const float4 *>(cr)[2 * blk + 1];
        const int4 oa = reinterpret_cast<const int4 *>(co)[2 * blk];
        const int4 ob = reinterpret_cast<const int4 *>(co)[2 * blk + 1];
        const int4 qa = reinterpret_cast<const int4 *>(cq)[2 * blk];
        const int4 qb = reinterpret_cast<const int4 *>(cq)[2 * blk + 1];
        const float rv[8] = {ra.x, ra.y, ra.z, ra.w, rb.x, rb.y, rb.z, rb.w};
        const int ov[8] = {oa.x, oa.y, oa.z, oa.w, ob.x, ob.y, ob.z, ob.w};
        const int qv[8] = {qa.x, qa.y, qa.z, qa.w, qb.x, qb.y, qb.z, qb.w};
        float x[8], swb = 0.f, sqb = 0.f;
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int cp = blk * 8 + u;
          const float rho = tri[(cp < c) ? qv[u] + oc : Qc + ov[u]];
          ok0 = ok0 && (rho >= kRhoMin);
          const float w = weight_of<WM>(rho, w_max);
          x[u] = (rc - rv[u]) * w;
          if (DIAG) {
            swb += w;
            sqb = fmaf(w, w, sqb);
            mw0 = fmaxf(mw0, w);
          }
        }
        sblk = ((x[0] + x[1]) + (x[2] + x[3])) + ((x[4] + x[5]) + (x[6] + x[7]));
        if (DIAG) {
          sw0 += swb;
          sq0 += sqb;
        }
      }
      float cy = sblk;
      int m = blk;
#pragma unroll
      for (int l = 0; l < 4; ++l) {
        if (m & 1) {
          cy = p[l] + cy;
          m >>= 1;
        } else {
          p[l] = cy;
          break;
        }
      }
    }
    sum0 = p[3];
  }

  // Rows 32..K-1: each lane takes partners lane and lane + 32, the warp sums
  // them by a butterfly; lane c - 32 keeps row c. Every visit here belongs
  // to a completed row.
  bool okx = true;
  float sum1 = 0.f, swx = 0.f, sqx = 0.f, mwx = 0.f;
  {
    const float ra = cr[lane], rb = cr[lane + 32];
    const int ob = co[lane + 32], qa = cq[lane], qb = cq[lane + 32];
#pragma unroll 2
    for (int cx = 32; cx < K; ++cx) {
      const float rx = cr[cx];
      const int ox = co[cx], Qx = cq[cx];
      const float rho_a = tri[qa + ox];  // lane < 32 <= cx
      const float rho_b = tri[(lane + 32 < cx) ? qb + ox : Qx + ob];
      okx = okx && (rho_a >= kRhoMin) && (rho_b >= kRhoMin);
      const float wa = weight_of<WM>(rho_a, w_max), wb = weight_of<WM>(rho_b, w_max);
      if (DIAG) {
        swx += wa + wb;
        sqx = fmaf(wa, wa, fmaf(wb, wb, sqx));
        mwx = fmaxf(mwx, fmaxf(wa, wb));
      }
      const float s = warp_sum((rx - ra) * wa + (rx - rb) * wb);
      if (lane == cx - 32) sum1 = s;
    }
  }

  const bool bad = (row0 && !ok0) || !okx;
  if (__any_sync(0xffffffffu, bad) && lane == 0)
    flag_error(dev_err, PAIR_DEV_ERR_NONPOSITIVE_INCLUSION);

  // Equal completed rewards per slot (itself included), by warp match on
  // the reward bits (+0 and -0 merged): contrast edges are the pairs with
  // different rewards, and a vertex is active iff some partner differs.
  const float k0 = rc + 0.f, k1 = cr[c + 32] + 0.f;
  int eq0 = 0, eq1 = 0;
  {
    const unsigned lo = (K >= 32) ? 0xffffffffu : ((1u << K) - 1u);
    if (row0) eq0 = __popc(__match_any_sync(lo, __float_as_uint(k0)));
    if (K > 32) {
      const unsigned hi = (K >= 64) ? 0xffffffffu : ((1u << (K - 32)) - 1u);
      if (row1) eq1 = __popc(__match_any_sync(hi, __float_as_uint(k1)));
      for (int x = 32; x < K; ++x) {
        const float kx = cr[x] + 0.f;
        const unsigned same = __ballot_sync(0xffffffffu, k0 == kx);
        eq0 += (k0 == kx) ? 1 : 0;
        if (lane == x - 32) eq1 += __popc(same);
      }
    }
  }

  WarpCoeffs o;
  o.K = K;
  o.C = (K * K - __reduce_add_sync(0xffffffffu, (row0 ? eq0 : 0) + (row1 ? eq1 : 0))) / 2;
  float av0 = row0 ? ((sum0 == 0.f) ? 0.f : 0.5f * sum0) : 0.f;
  float av1 = row1 ? ((sum1 == 0.f) ? 0.f : 0.5f * sum1) : 0.f;
  o.W = o.W2 = o.Wmax = 0.f;
  if (DIAG || WM == PAIR_W_HAJEK) {
    // Each completed edge was visited from both ends.
    o.W = 0.5f * warp_sum((row0 ? sw0 : 0.f) + swx);
    o.W2 = 0.5f * warp_sum((row0 ? sq0 : 0.f) + sqx);
    o.Wmax = warp_max(fmaxf(row0 ? mw0 : 0.f, mwx));
  }
  if (WM == PAIR_W_HAJEK) {
    av0 = o.W > 0.f ? __fdiv_rn(av0, o.W) : 0.f;
    av1 = o.W > 0.f ? __fdiv_rn(av1, o.W) : 0.f;
  }
  if ((flags & PAIR_STANDARDIZE) && K >= 2) {
    // Sample standard deviation (n - 1) of the completed rewards, two-pass.
    const float r0 = row0 ? rc : 0.f, r1 = row1 ? cr[c + 32] : 0.f;
    const float mean = warp_sum(r0 + r1) / (float)K;
    const float d0 = row0 ? r0 - mean : 0.f, d1 = row1 ? r1 - mean : 0.f;
    const float sd = sqrtf(warp_sum(d0 * d0 + d1 * d1) / (float)(K - 1));
    av0 = sd > 0.f ? __fdiv_rn(av0, sd) : 0.f;
    av1 = sd > 0.f ? __fdiv_rn(av1, sd) : 0.f;
  }
  if ((flags & PAIR_CENTER) && K > 0) {
    const float mean = warp_sum(av0 + av1) / (float)K;
    if (row0) av0 -= mean;
    if (row1) av1 -= mean;
  }

  // Back to vertex order: vertex v sits at packed slot p (p < K if completed),
  // held by lane p & 31 (first row if p < 32, second otherwise).
  const bool ac0 = row0 && eq0 < K, ac1 = row1 && eq1 < K;
  const float g0a = __shfl_sync(0xffffffffu, av0, p0 & 31);
  const float g0b = __shfl_sync(0xffffffffu, av1, p0 & 31);
  const float g1a = __shfl_sync(0xffffffffu, av0, p1 & 31);
  const float g1b = __shfl_sync(0xffffffffu, av1, p1 & 31);
  const unsigned A0 = __ballot_sync(0xffffffffu, ac0), A1 = __ballot_sync(0xffffffffu, ac1);
  o.a0 = j0 ? (p0 < 32 ? g0a : g0b) * scale : 0.f;
  o.a1 = j1 ? (p1 < 32 ? g1a : g1b) * scale : 0.f;
  o.act0 = j0 && (((p0 < 32 ? A0 : A1) >> (p0 & 31)) & 1u);
  o.act1 = j1 && (((p1 < 32 ? A0 : A1) >> (p1 & 31)) & 1u);
  return o;
}

}  // namespace
}  // namespace pairk
