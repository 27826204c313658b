// Backward of the bf16 LM-head path without an image of softmax terms (the
// no-alloc path and minimum workspaces): the logits are recomputed. For
// d = 512 A (A <= 6), 8-CTA clusters share each Gs tile through an L2 ring
// (bwd_cluster_kernel); otherwise one CTA per row block and 256-wide d-slice
// (bwd_kernel).
#include "tc_kernels.cuh"

namespace pairk {
namespace {

using namespace tc;
using namespace tck;

// ------------------------------------------------------------- backward
constexpr int kBwdBN = 128;     // S tile columns
constexpr int kSlice = 256;     // output columns held in TMEM per unit
constexpr int kBwdStages = 3;
constexpr uint32_t kBwdStageTx = 2 * kAtom128;
constexpr uint32_t kIdescS = idesc_bf16(128, kBwdBN, 0, 0);

struct BwdSmem {
  uint8_t a[kBwdStages][kAtom128];   // rows-operand atoms (128 x 64)
  uint8_t b[kBwdStages][kAtom128];   // cols-operand atoms (128 x 64)
  uint8_t cs[kSlice / 64][kAtom128]; // cols operand, d-slice (MN-major B)
  uint8_t g[kBwdBN / 64][kAtom128];  // Gs tile, K-major A (2 atoms along K)
  float col_c[kBwdBN], col_l[kBwdBN];
  uint64_t full[kBwdStages], empty[kBwdStages];
  uint64_t s_full[2], s_empty[2];
  uint64_t g_full, g_empty, cs_full, cs_empty, o_full, o_empty, mma_done;
  uint32_t tmem_base;
  int abort;
};

// kTokenRows: rows = tokens (output dH), cols = vocabulary.
// otherwise : rows = vocabulary (output dW), cols = tokens.
template <bool kTokenRows>
__global__ void __launch_bounds__(kThreads, 1)
    bwd_kernel(const __grid_constant__ CUtensorMap tmR,
               const __grid_constant__ CUtensorMap tmC, int d, int V,
               const int32_t *counters, const int32_t *tok_idx,
               const float *tok_c, const float *lse, float *out,
               int32_t *dev_err) {
  extern __shared__ uint8_t smem_raw[];
  BwdSmem &sm = *reinterpret_cast<BwdSmem *>(align1k(smem_raw));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Teff = counters[0];
  const int nsl = (d + kSlice - 1) / kSlice;
  const int n_rb = kTokenRows ? (Teff + 127) / 128 : (V + 127) / 128;
  const int n_ct = kTokenRows ? (V + kBwdBN - 1) / kBwdBN : (Teff + kBwdBN - 1) / kBwdBN;
  const int n_units = n_rb * nsl;
  const int nk = d / 64;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kBwdStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sm.s_full[s], 1);
      mbar_init(&sm.s_empty[s], 128);
    }
    mbar_init(&sm.g_full, 128);
    mbar_init(&sm.g_empty, 1);
    mbar_init(&sm.cs_full, 1);
    mbar_init(&sm.cs_empty, 1);
    mbar_init(&sm.o_full, 1);
    mbar_init(&sm.o_empty, 128);
    mbar_init(&sm.mma_done, 1);
    sm.abort = 0;
    fence_mbar_init();
    prefetch_tmap(&tmR);
    prefetch_tmap(&tmC);
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  const uint32_t tmem_o = tmem + 2 * kBwdBN;  // columns [256, 512)
  volatile int *abort = &sm.abort;

  if (warp == 0) {
    {  // whole warp: uniform loop state; elected lane issues
      int stage = 0;
      uint32_t ph = 0, cs_ph = 0;
      int last_ph[kBwdStages];
      for (int s = 0; s < kBwdStages; ++s) last_ph[s] = -1;
      int cs_last = -1;
      bool ok = true;
      auto load_s = [&](int rb, int ct) {
        for (int k = 0; k < nk && ok; ++k) {
          if (!(ok = wait(&sm.empty[stage], ph ^ 1, abort, dev_err))) break;
          if (elect_one()) {
            mbar_expect_tx(&sm.full[stage], kBwdStageTx);
            tma_load_2d(sm.a[stage], &tmR, &sm.full[stage], k * 64, rb * 128);
            tma_load_2d(sm.b[stage], &tmC, &sm.full[stage], k * 64, ct * kBwdBN);
          }
          __syncwarp();
          last_ph[stage] = (int)ph;
          if (++stage == kBwdStages) { stage = 0; ph ^= 1; }
        }
      };
      auto load_cs = [&](int sl, int w, int ct) {
        if (!ok) return;
        if (!(ok = wait(&sm.cs_empty, cs_ph ^ 1, abort, dev_err))) return;
        if (elect_one()) {
          mbar_expect_tx(&sm.cs_full, (uint32_t)(w / 64) * kAtom128);
          for (int j = 0; j < w / 64; ++j)
            tma_load_2d(sm.cs[j], &tmC, &sm.cs_full, sl * kSlice + j * 64, ct * kBwdBN);
        }
        __syncwarp();
        cs_last = (int)cs_ph;
        cs_ph ^= 1;
      };
      for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
        const int rb = u / nsl, sl = u % nsl;
        const int w = min(kSlice, d - sl * kSlice);
        if (n_ct == 0) continue;
        load_s(rb, 0);
        for (int ct = 1; ct < n_ct && ok; ++ct) {
          load_s(rb, ct);
          load_cs(sl, w, ct - 1);
        }
        load_cs(sl, w, n_ct - 1);
      }
      volatile int never = 0;
      for (int s = 0; s < kBwdStages; ++s)
        if (last_ph[s] >= 0) wait(&sm.full[s], (uint32_t)last_ph[s], &never, dev_err);
      if (cs_last >= 0) wait(&sm.cs_full, (uint32_t)cs_last, &never, dev_err);
    }
  } else if (warp == 1) {
    {  // whole warp: uniform loop state; elected lane issues
      int stage = 0;
      uint32_t ph = 0, s_ph[2] = {0, 0}, g_ph = 0, cs_ph = 0, o_ph = 0;
      bool ok = true;
      auto issue_s = [&](int ct) {
        const int buf = ct & 1;
        if (!(ok = wait(&sm.s_empty[buf], s_ph[buf] ^ 1, abort, dev_err))) return;
        tc_fence_after();
        const uint32_t dt = tmem + buf * kBwdBN;
        for (int k = 0; k < nk; ++k) {
          if (!(ok = wait(&sm.full[stage], ph, abort, dev_err))) return;
          const uint32_t sa = smem_u32(sm.a[stage]), sb = smem_u32(sm.b[stage]);
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              mma_bf16(dt, sdesc_sw128(sa + kk * 32, 16, 1024),
                       sdesc_sw128(sb + kk * 32, 16, 1024), kIdescS,
                       (k | kk) != 0);
            mma_commit(&sm.empty[stage]);
          }
          __syncwarp();
          if (++stage == kBwdStages) { stage = 0; ph ^= 1; }
        }
        if (elect_one()) mma_commit(&sm.s_full[buf]);
        __syncwarp();
        s_ph[buf] ^= 1;
      };
      auto issue_o = [&](int ct, int w) {
        if (!ok) return;
        if (!(ok = wait(&sm.g_full, g_ph, abort, dev_err))) return;
        if (!(ok = wait(&sm.cs_full, cs_ph, abort, dev_err))) return;
        if (ct == 0 && !(ok = wait(&sm.o_empty, o_ph ^ 1, abort, dev_err))) return;
        tc_fence_after();
        const uint32_t idesc = idesc_bf16(128, w, 0, 1);
        const uint32_t sg = smem_u32(sm.g[0]), sc = smem_u32(sm.cs[0]);
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < kBwdBN / 16; ++kk) {
            const uint64_t ad = sdesc_sw128(sg + (kk >> 2) * kAtom128 + (kk & 3) * 32, 16, 1024);
            const uint64_t bd = sdesc_sw128(sc + kk * 2048, kAtom128, 1024);
            mma_bf16(tmem_o, ad, bd, idesc, (ct | kk) != 0);
          }
          mma_commit(&sm.g_empty);
          mma_commit(&sm.cs_empty);
        }
        __syncwarp();
        g_ph ^= 1;
        cs_ph ^= 1;
      };
      for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
        const int sl = u % nsl;
        const int w = min(kSlice, d - sl * kSlice);
        if (n_ct == 0) continue;
        issue_s(0);
        for (int ct = 0; ct < n_ct && ok; ++ct) {
          if (ct + 1 < n_ct) issue_s(ct + 1);
          issue_o(ct, w);
        }
        if (!ok) break;
        if (elect_one()) mma_commit(&sm.o_full);
        __syncwarp();
        o_ph ^= 1;
      }
      if (elect_one()) mma_commit(&sm.mma_done);
      __syncwarp();
      volatile int never = 0;
      wait(&sm.mma_done, 0, &never, dev_err);
    }
  } else {
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    uint32_t s_ph[2] = {0, 0}, g_ph = 0, o_ph = 0;
    bool ok = true;
    for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
      const int rb = u / nsl, sl = u % nsl;
      const int w = min(kSlice, d - sl * kSlice);
      const int rid = rb * 128 + row;  // token position or vocabulary id
      float rc = 0.f, rl = 0.f;
      if (kTokenRows && rid < Teff) {
        rc = tok_c[rid];
        rl = lse[rid] * kLog2e;
      }
      for (int ct = 0; ct < n_ct; ++ct) {
        if (!kTokenRows) {
          epi_sync();
          const int p = ct * kBwdBN + row;
          sm.col_c[row] = p < Teff ? tok_c[p] : 0.f;
          sm.col_l[row] = p < Teff ? lse[p] * kLog2e : 0.f;
          epi_sync();
        }
        const int buf = ct & 1;
        if (!(ok = wait(&sm.s_full[buf], s_ph[buf], abort, dev_err))) break;
        s_ph[buf] ^= 1;
        if (!(ok = wait(&sm.g_empty, g_ph ^ 1, abort, dev_err))) break;
        tc_fence_after();
#pragma unroll 1
        for (int c = 0; c < kBwdBN / 32; ++c) {
          float v[32];
          tmem_ld32(tmem + lane_off + buf * kBwdBN + c * 32, v);
          uint32_t pk[16];
#pragma unroll
          for (int j = 0; j < 32; j += 2) {
            float g2[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int col = c * 32 + j + e;
              float cc, ll;
              bool live;
              if (kTokenRows) {
                cc = rc; ll = rl;
                live = (rc != 0.f) && (ct * kBwdBN + col < V);
              } else {
                cc = sm.col_c[col]; ll = sm.col_l[col];
                live = cc != 0.f;
              }
              g2[e] = live ? -cc * ex2_approx(fmaf(v[j + e], kLog2e, -ll)) : 0.f;
            }
            __nv_bfloat162 b2 = __floats2bfloat162_rn(g2[0], g2[1]);
            pk[j >> 1] = *reinterpret_cast<uint32_t *>(&b2);
          }
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const int k = c * 32 + q * 8;  // first column of this 16-byte piece
            uint8_t *dst = sm.g[k >> 6] + sw128_offset(row, k & 63);
            *reinterpret_cast<uint4 *>(dst) =
                make_uint4(pk[q * 4], pk[q * 4 + 1], pk[q * 4 + 2], pk[q * 4 + 3]);
          }
        }
        tc_fence_before();
        mbar_arrive(&sm.s_empty[buf]);
        fence_async_smem();
        mbar_arrive(&sm.g_full);
        g_ph ^= 1;
      }
      if (!ok) break;
      const bool valid = kTokenRows ? (rid < Teff) : (rid < V);
      float *dst = nullptr;
      if (valid)
        dst = out + (kTokenRows ? (int64_t)tok_idx[rid] : (int64_t)rid) * d + sl * kSlice;
      if (n_ct == 0) {
        if (valid)
          for (int k = 0; k < w; ++k) dst[k] = 0.f;
        continue;
      }
      if (!(ok = wait(&sm.o_full, o_ph, abort, dev_err))) break;
      o_ph ^= 1;
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < w / 32; ++c) {
        float v[32];
        tmem_ld32(tmem_o + lane_off + c * 32, v);
        if (valid) {
#pragma unroll
          for (int q = 0; q < 8; ++q)
            reinterpret_cast<float4 *>(dst + c * 32)[q] =
                make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        }
      }
      tc_fence_before();
      mbar_arrive(&sm.o_empty);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// ------------------------------------------------- backward, cluster form
//
// One 8-CTA cluster owns a row block (128 tokens for dH, 128 vocabulary rows
// for dW); CTA k of the cluster keeps out[rows, k*w : (k+1)*w] (w = d/8) in
// TMEM for the whole unit, so each logit-gradient tile Gs is formed once per
// cluster instead of once per d-slice.
//
// Tile ownership rotates: the owner of column tile g (g mod 8) accumulates
// the full-depth S tile in TMEM, spread evenly over the 8 slots that end
// kClLag slots before the tile is used (d/512 K-atoms per slot), converts it
// to bf16 Gs and publishes the 32 KB tile (already in the swizzled K-major
// layout of the MMA operand) once, to a per-cluster ring in global memory,
// then signals every CTA of the cluster through its pub[owner][m & 1]
// mbarrier (m = g / 8, the owner's tile count). Every CTA pulls Gs(s) into
// shared memory with a bulk copy and updates out += Gs(s) . C[s, slice].
// The ring holds two tiles per owner, and an owner overwrites its slot of
// tile g - 16 only after every CTA is done with that tile; with two pub
// barriers per owner this also keeps any consumer's parity wait unambiguous,
// and it leaves 16 slots (not 8) for the round trip consume -> convert ->
// publish -> load. The exchange goes through L2
// because distributed shared memory sustains far less per-SM egress than a
// broadcast of a 32 KB tile to 7 peers per slot needs. In every slot every
// CTA issues the same tensor work: a share of one S accumulation plus one
// output update. The slot counter runs across units, so the staggered S
// schedule never drains at unit boundaries.
//
// The column tile is BN wide (BN = 128 for d <= 2048, 96 for d = 2560, 64
// for d = 3072): TMEM holds two BN-column S buffers plus the d/8-column
// output slice, 2 BN + d/8 <= 512.
constexpr int kCl = 8;          // cluster size (power of two)
constexpr int kClStages = 4;    // S operand stages
constexpr int kClLag = 3;       // slots between an S tile's completion and its use
constexpr int kClJ = kCl + kClLag;
constexpr int kGSlots = 1;      // Gs tiles staged in shared memory
constexpr int kClThreads = 256; // + warp 6: loads of C[s, slice] and Gs; warp 7: output MMAs

template <int BN>
struct ClTile {
  static constexpr uint32_t kColAtom = BN * 64 * 2;         // BN rows x 64 bf16
  static constexpr int kGsAtoms = (BN + 63) / 64;           // Gs K-major atoms
  static constexpr uint32_t kGsBytes = kGsAtoms * kAtom128; // one Gs tile
  static constexpr int kCsAtoms = (512 - 2 * BN) / 64;      // max output-slice atoms
  static constexpr uint32_t kIdescS = idesc_bf16(128, BN, 0, 0);
};

template <int BN>
struct ClSmem {
  using T = ClTile<BN>;
  uint8_t a[kClStages][kAtom128];                 // rows operand atoms (128 x 64)
  uint8_t b[kClStages][T::kColAtom];              // column operand atoms (BN x 64)
  uint8_t cs[T::kCsAtoms][T::kColAtom];           // C[s, slice]: MN-major B
  uint8_t g[kGSlots][T::kGsAtoms][kAtom128];      // Gs tiles: 128 x BN bf16, K-major A
  float col_c[BN], col_l[BN];
  uint64_t full[kClStages], empty[kClStages];
  uint64_t s_full[2], s_empty[2];
  uint64_t g_full[kGSlots], gs_empty[kGSlots];
  uint64_t cs_full[2], cs_empty[2];  // C[s, slice] in two column parts
  uint64_t pub[kCl][2];              // owner o published its tile m (by m & 1)
  uint64_t gfree[2];                 // (owner) all CTAs done with its tile m (by m & 1)
  uint64_t o_full, o_empty, mma_done;
  uint32_t tmem_base;
  int abort;
};

// The tiles of one cluster, in processing order: first its F = n_rb / ncl
// full row blocks (cid, cid + ncl, ...), each with all n_ct column tiles;
// then an even share [t0, t1) of the row-major tiles of the remaining
// R = n_rb mod ncl row blocks, so that all clusters finish within a tile of
// each other. A unit (run of tiles with one row block) in that tail may cover
// only part of its row block. Since R < ncl, a cluster's share has at most
// n_ct tiles and so at most two tail units; each is stored to the cluster's
// scratch slot (cid, u) and tail_reduce_kernel sums the slots of every tail
// row in cluster order (deterministic, no atomics).
struct TileMap {
  int n_ct, ncl, cid, gT, t0, rbT, N;
  __device__ void setup(int n_rb, int n_ct_, int cid_, int ncl_) {
    n_ct = n_ct_;
    ncl = ncl_;
    cid = cid_;
    const int F = n_ct ? n_rb / ncl : 0;
    const int R = n_ct ? n_rb - F * ncl : 0;
    const int64_t T = (int64_t)R * n_ct;
    gT = F * n_ct;
    rbT = F * ncl;
    t0 = (int)(T * cid / ncl);
    N = gT + (int)(T * (cid + 1) / ncl) - t0;
  }
  __device__ bool tail(int g) const { return g >= gT; }
};

// Walks tile indices g = 0, 1, 2, ... of a TileMap as (row block, column
// tile) pairs without divisions in the loop.
struct TileCursor {
  int ct, rb, g;
  __device__ void init(const TileMap &mp, int g_) {
    g = g_;
    if (mp.n_ct == 0) {
      ct = 0;
      rb = mp.cid;
    } else if (g < mp.gT) {
      ct = g % mp.n_ct;
      rb = mp.cid + (g / mp.n_ct) * mp.ncl;
    } else {
      const int t = mp.t0 + (g - mp.gT);
      ct = t % mp.n_ct;
      rb = mp.rbT + t / mp.n_ct;
    }
  }
  __device__ void next(const TileMap &mp) {
    ++g;
    if (g == mp.gT) {
      ct = mp.t0 % mp.n_ct;
      rb = mp.rbT + mp.t0 / mp.n_ct;
    } else if (++ct == mp.n_ct) {
      ct = 0;
      rb += g < mp.gT ? mp.ncl : 1;
    }
  }
  __device__ bool unit_start(const TileMap &mp) const { return ct == 0 || g == mp.gT; }
  __device__ bool unit_end(const TileMap &mp) const { return ct == mp.n_ct - 1 || g == mp.N - 1; }
};

// Final values of the tail rows (see TileMap) of the chunk of row blocks
// [rb0, rb0 + cap): for each row, the sum in cluster order of the partial
// units the clusters stored to their scratch slots.
template <bool kTokenRows, int BN>
__global__ void tail_reduce_kernel(int d, int V, int ncl, int rb0, int cap,
                                   const int32_t *counters, const int32_t *tok_idx,
                                   const float *tailbuf, float *out) {
  const int Teff = counters[0];
  const int n_rows = kTokenRows ? Teff : V;
  const int n_ct = kTokenRows ? (V + BN - 1) / BN : (Teff + BN - 1) / BN;
  const int n_rb = min(max((n_rows + 127) / 128 - rb0, 0), cap);
  if (n_ct == 0) return;
  const int F = n_rb / ncl, R = n_rb - F * ncl;
  if (R == 0) return;
  const int64_t Tt = (int64_t)R * n_ct;
  const int r0 = (rb0 + F * ncl) * 128;
  const int r1 = min(n_rows, (rb0 + n_rb) * 128);
  const int vec = d / 4;
  const float4 *src = reinterpret_cast<const float4 *>(tailbuf);
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
       i < (int64_t)(r1 - r0) * vec; i += (int64_t)gridDim.x * blockDim.x) {
    const int off = (int)(i / vec);           // row offset from r0
    const int rl = off >> 7, rr = off & 127;  // tail row block, row within it
    const int c4 = (int)(i % vec);
    const int64_t lo = (int64_t)rl * n_ct, hi = lo + n_ct;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int c = 0; c < ncl; ++c) {
      const int64_t a = Tt * c / ncl, b = Tt * (c + 1) / ncl;
      if ((a > lo ? a : lo) < (b < hi ? b : hi)) {
        const int u = rl - (int)(a / n_ct);  // this row block's unit in cluster c
        const float4 p = src[((int64_t)(c * 2 + u) * 128 + rr) * vec + c4];
        acc.x += p.x; acc.y += p.y; acc.z += p.z; acc.w += p.w;
      }
    }
    const int rid = r0 + off;
    const int64_t row = kTokenRows ? (int64_t)tok_idx[rid] : (int64_t)rid;
    reinterpret_cast<float4 *>(out + row * d)[c4] = acc;
  }
}

// State of the fused log-sum-exp + dH pass (kFused; null otherwise).
//
// Every active token t gets a fixed reference R_t (log2 units) before the
// pass: its target logit z_t[y_t] log2 e (target_logit_kernel), or, for the
// row blocks the fix-up pass redoes, the row maximum found by the first pass.
// The owner of a tile converts S to P = 2^(S log2 e - R_t) (bf16 operand of
// the output MMA, which accumulates O_t = sum_v P_tv W_v) and adds the fp32 P
// to its running l_t = sum_v P_tv; at the end of every unit each CTA writes
// its l and row-maximum partials to lpart[slot][k] and counts itself into
// ready[slot]; the drain waits for all kCl partials, sums them in CTA order
// and writes dH_t = -c_t O_t / l_t and lse_t = (R_t + log2 l_t) ln 2. Since
// z_t[y_t] <= max_v z_tv, P never underflows where it matters; a row whose
// maximum exceeds R_t by more than kFixLog2 (P would approach the fp32 range)
// flags its row block, and the fix-up pass redoes those blocks with R_t = the
// row maximum. Tail units keep O, l and the maximum unscaled for
// tail_fused_kernel.
struct FusedArgs {
  const float *ref;      // [Tpad] R_t, log2 units
  float *lse;            // [Tpad] out: log-sum-exp (natural units)
  float *mrow;           // [Tpad] out: row maximum of the logits, log2 units
  int *rbflag;           // [n_rb] out: 1 = the row block needs the fix-up pass
  float *lpart;          // [slots][kCl][2][128] per-CTA partials (l, max)
  int *ready;            // [slots] CTAs that published their partials (zeroed)
  float *tail_l;         // [kMaxClusters][2][2][128] cluster sums of tail units
  const int *rb_list;    // row blocks to process (fix-up pass), or null
  const int *n_list;     // their count (device), with rb_list
};
constexpr float kFixLog2 = 64.f;
constexpr float kLn2 = 0.69314718055994531f;

// Bounded wait until *ctr >= target (acquire at GPU scope).
__device__ __forceinline__ bool wait_count(const int *ctr, int target, volatile int *abort,
                                           int32_t *dev_err) {
  const long long t0 = clock64();
  while (true) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
    if (v >= target) return true;
    if (*abort) return false;
    if (clock64() - t0 > kWaitCycles) {
      *abort = 1;
      flag_error(dev_err, PAIR_DEV_ERR_TIMEOUT);
      return false;
    }
    __nanosleep(64);
  }
}

// z_t[y_t] = <Hc_p, W_{y_p}> for every compacted token p (target_logit_dot)
// and its log2-unit reference R_p = z log2 e for the fused pass; also zeroes
// the fused pass's counters and row-block flags.
__global__ void target_logit_kernel(int d, const int32_t *counters, const int32_t *tok_y,
                                    const __nv_bfloat16 *Hc, const __nv_bfloat16 *W,
                                    float *zy, float *ref, int *ready, int n_ready, int *rbflag,
                                    int n_rbflag) {
  const int tid = blockIdx.x * blockDim.x + threadIdx.x;
  const int nth = gridDim.x * blockDim.x;
  for (int i = tid; i < n_ready; i += nth) ready[i] = 0;
  for (int i = tid; i < n_rbflag; i += nth) rbflag[i] = 0;
  const int Teff = counters[0];
  const int lane = threadIdx.x & 31;
  for (int p = tid >> 5; p < Teff; p += nth >> 5) {
    const float acc =
        target_logit_dot(d, Hc + (int64_t)p * d, W + (int64_t)tok_y[p] * d, lane);
    if (lane == 0) {
      zy[p] = acc;
      ref[p] = acc * kLog2e;
    }
  }
}

// Tail rows of the fused pass (see TileMap and FusedArgs): O, l and the row
// maximum summed (maximum taken) in cluster order over the partial units that
// cover the row, then dH_t = -c_t O_t / l_t, lse_t and the fix-up flag.
template <int BN>
__global__ void tail_fused_kernel(int d, int V, int ncl, const int32_t *counters,
                                  const int32_t *tok_idx, const float *tok_c,
                                  const float *tailbuf, FusedArgs fa, float *out) {
  const int Teff = counters[0];
  const int n_ct = (V + BN - 1) / BN;
  const int n_rb = fa.rb_list ? *fa.n_list : (Teff + 127) / 128;
  const int F = n_rb / ncl, R = n_rb - F * ncl;
  if (R == 0) return;
  const int64_t Tt = (int64_t)R * n_ct;
  const int vec = d / 4;
  const float4 *src = reinterpret_cast<const float4 *>(tailbuf);
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < (int64_t)R * 128 * vec;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int off = (int)(i / vec);
    const int rl = off >> 7, rr = off & 127;
    const int c4 = (int)(i % vec);
    const int prb = fa.rb_list ? fa.rb_list[F * ncl + rl] : F * ncl + rl;
    const int rid = prb * 128 + rr;
    if (rid >= Teff) continue;
    const int64_t lo = (int64_t)rl * n_ct, hi = lo + n_ct;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    float L = 0.f, M = -INFINITY;
    for (int c = 0; c < ncl; ++c) {
      const int64_t a = Tt * c / ncl, b = Tt * (c + 1) / ncl;
      if ((a > lo ? a : lo) < (b < hi ? b : hi)) {
        const int u = rl - (int)(a / n_ct);
        const float4 p = src[((int64_t)(c * 2 + u) * 128 + rr) * vec + c4];
        acc.x += p.x; acc.y += p.y; acc.z += p.z; acc.w += p.w;
        L += fa.tail_l[(c * 2 + u) * 256 + rr];
        M = fmaxf(M, fa.tail_l[(c * 2 + u) * 256 + 128 + rr]);
      }
    }
    const float R2 = fa.ref[rid];
    const float scale = -tok_c[rid] / L;
    reinterpret_cast<float4 *>(out + (int64_t)tok_idx[rid] * d)[c4] =
        make_float4(acc.x * scale, acc.y * scale, acc.z * scale, acc.w * scale);
    if (c4 == 0) {
      const float M2 = M * kLog2e;
      fa.lse[rid] = (R2 + log2f(L)) * kLn2;
      fa.mrow[rid] = M2;
      if (!(L > 0.f) || !(L < INFINITY) || !(M2 - R2 <= kFixLog2)) fa.rbflag[prb] = 1;
    }
  }
}

// Between the fused pass and its fix-up: the flagged row blocks, in order,
// become the fix-up pass's list (count in *n_list), their rows' reference
// becomes the row maximum the first pass found, and the pass counters are
// zeroed again. One block.
__global__ void fixup_prep_kernel(const int32_t *counters, const int *rbflag, int *rb_list,
                                  int *n_list, float *ref, const float *mrow, int *ready,
                                  int n_ready) {
  __shared__ int count;
  const int Teff = counters[0];
  const int n_rb = (Teff + 127) / 128;
  for (int i = threadIdx.x; i < n_ready; i += blockDim.x) ready[i] = 0;
  if (threadIdx.x < 32) {
    int base = 0;
    for (int r0 = 0; r0 < n_rb; r0 += 32) {
      const int r = r0 + (int)threadIdx.x;
      const bool f = r < n_rb && rbflag[r] != 0;
      const unsigned bal = __ballot_sync(0xffffffffu, f);
      if (f) rb_list[base + __popc(bal & ((1u << threadIdx.x) - 1u))] = r;
      base += __popc(bal);
    }
    if (threadIdx.x == 0) {
      count = base;
      *n_list = base;
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < count * 128; i += blockDim.x) {
    const int p = rb_list[i >> 7] * 128 + (i & 127);
    if (p < Teff) ref[p] = mrow[p];
  }
}

template <bool kTokenRows, int BN, bool kFused = false>
__global__ void __cluster_dims__(kCl, 1, 1) __launch_bounds__(kClThreads, 1)
    bwd_cluster_kernel(const __grid_constant__ CUtensorMap tmR,
                       const __grid_constant__ CUtensorMap tmC,
                       const __grid_constant__ CUtensorMap tmC64, int d, int V,
                       const int32_t *counters, const int32_t *tok_idx,
                       const float *tok_c, const float *lse, float *out,
                       uint8_t *gring, float *tailbuf, int rb0, int cap,
                       FusedArgs fa, int32_t *dev_err) {
  extern __shared__ uint8_t smem_raw[];
  ClSmem<BN> &sm = *reinterpret_cast<ClSmem<BN> *>(align1k(smem_raw));
  using Tl = ClTile<BN>;
  constexpr uint32_t kGsBytes = Tl::kGsBytes, kColAtom = Tl::kColAtom;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int k = (int)cluster_rank();
  const int cid = (int)cluster_id_x(), ncl = (int)num_clusters_x();
  const int Teff = counters[0];
  const int A = d / (64 * kCl);            // K-atoms per slot (d / 512)
  const int w = 64 * A;                    // this CTA's d-slice width
  const int nk = d / 64;
  // The output update runs in two parts with their own operand barriers, so
  // part 0's operands of the next slot load while part 1 still computes.
  // With a 128-wide tile and a slice of at most 256 columns (d <= 2048) the
  // parts are the two 64-row K halves of the tile (Gs atom p with rows
  // [64p, 64p + 64) of C[s, slice]; 256-wide MMAs); otherwise they are two
  // column parts of A0 and A - A0 atoms of the slice.
  const bool ksplit = BN == 128 && A <= 4;
  const int A0 = ksplit ? A : (A + 1) >> 1, A1 = ksplit ? A : A - A0;
  // Row blocks [rb0, rb0 + n_rb) of this launch (one chunk); TileMap and
  // TileCursor count them from 0.
  const int n_rb = (kFused && fa.rb_list)
                       ? min(*fa.n_list, cap)
                       : min(max((kTokenRows ? (Teff + 127) / 128 : (V + 127) / 128) - rb0, 0), cap);
  const int n_ct = kTokenRows ? (V + BN - 1) / BN : (Teff + BN - 1) / BN;
  // Row block of the launch's row-block index rb (TileMap counts from 0): the
  // chunk's rb0 + rb, or the fix-up pass's list entry.
  auto phys_rb = [&](int rb) { return (kFused && fa.rb_list) ? fa.rb_list[rb] : rb0 + rb; };
  const int n_my = cid < n_rb ? (n_rb - cid + ncl - 1) / ncl : 0;
  TileMap mp;
  mp.setup(n_rb, n_ct, cid, ncl);
  const int N = mp.N;                      // tiles of this cluster
  // Ring of published Gs tiles: [owner][job parity] for this cluster.
  uint8_t *ring = gring + (size_t)cid * kCl * 2 * kGsBytes;
  // Where tile g is published: its owner's ring slot for the tile's parity.
  auto gs_tile = [&](int g) {
    return ring + ((size_t)(g & (kCl - 1)) * 2 + (size_t)((g >> 3) & 1)) * kGsBytes;
  };
  // The tile whose S this CTA accumulates during slot s (may be < 0 or >= N).
  auto job_of = [&](int s) {
    const int g0 = s + kClLag + 1;
    return g0 + ((k - g0) & (kCl - 1));
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < kClStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sm.s_full[s], 1);
      mbar_init(&sm.s_empty[s], 128);
      mbar_init(&sm.gfree[s], kCl);
    }
    for (int s = 0; s < kGSlots; ++s) {
      mbar_init(&sm.g_full[s], 1);
      mbar_init(&sm.gs_empty[s], 1);
    }
    for (int p = 0; p < 2; ++p) {
      mbar_init(&sm.cs_full[p], 1);
      mbar_init(&sm.cs_empty[p], 1);
    }
    for (int o = 0; o < kCl; ++o) {
      mbar_init(&sm.pub[o][0], 1);
      mbar_init(&sm.pub[o][1], 1);
    }
    mbar_init(&sm.o_full, 1);
    mbar_init(&sm.o_empty, 128);
    mbar_init(&sm.mma_done, 2);  // one final commit per MMA-issuing warp
    sm.abort = 0;
    fence_mbar_init();
    prefetch_tmap(&tmR);
    prefetch_tmap(&tmC);
    prefetch_tmap(&tmC64);
  }
  if (warp == 1) {
    tmem_alloc(&sm.tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // every CTA's barriers exist before anyone signals them
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  const uint32_t tmem_o = tmem + 2 * BN;
  volatile int *abort = &sm.abort;

  if (warp == 0) {
    // Producer of the S operands (this CTA's share of its owned tiles).
    {  // whole warp: uniform loop state; elected lane issues
      int stage = 0;
      uint32_t ph = 0;
      int last_ph[kClStages];
      for (int s = 0; s < kClStages; ++s) last_ph[s] = -1;
      bool ok = true;
      int job_rb = 0, job_ct = 0, job_g = -1;
      for (int s = -kClJ; s < N && ok; ++s) {
        const int gj = job_of(s);
        if (gj < 0 || gj >= N) continue;
        if (gj != job_g) {
          TileCursor c;
          c.init(mp, gj);
          job_rb = c.rb; job_ct = c.ct; job_g = gj;
        }
        const int a0 = (s - (gj - kClJ)) * A;
        for (int a = a0; a < a0 + A; ++a) {
          if (!(ok = wait(&sm.empty[stage], ph ^ 1, abort, dev_err))) break;
          if (elect_one()) {
            mbar_expect_tx(&sm.full[stage], kAtom128 + kColAtom);
            tma_load_2d(sm.a[stage], &tmR, &sm.full[stage], a * 64, phys_rb(job_rb) * 128);
            tma_load_2d(sm.b[stage], &tmC, &sm.full[stage], a * 64, job_ct * BN);
          }
          __syncwarp();
          last_ph[stage] = (int)ph;
          if (++stage == kClStages) { stage = 0; ph ^= 1; }
        }
      }
      volatile int never = 0;
      for (int s = 0; s < kClStages; ++s)
        if (last_ph[s] >= 0) wait(&sm.full[s], (uint32_t)last_ph[s], &never, dev_err);
    }
  } else if (warp == 6) {
    // Producer of the output-update operands: C[s, slice] and Gs(s).
    {  // whole warp: uniform loop state; elected lane issues
      uint32_t cs_ph[2] = {0, 0}, ge_ph[kGSlots] = {};
      int cs_last[2] = {-1, -1}, g_last[kGSlots];
      for (int i = 0; i < kGSlots; ++i) g_last[i] = -1;
      bool ok = true;
      TileCursor cur;
      cur.init(mp, 0);
      // Output operand C[s, slice], column part p (atoms [j0, j0 + na)).
      auto load_cs = [&](int p, int j0, int na, int ct) {
        if (!(ok = wait(&sm.cs_empty[p], cs_ph[p] ^ 1, abort, dev_err))) return;
        if (elect_one()) {
          mbar_expect_tx(&sm.cs_full[p], (uint32_t)na * kColAtom);
          for (int j = j0; j < j0 + na; ++j)
            tma_load_2d(sm.cs[j], &tmC, &sm.cs_full[p], k * w + j * 64, ct * BN);
        }
        __syncwarp();
        cs_last[p] = (int)cs_ph[p];
        cs_ph[p] ^= 1;
      };
      // K-split: part p = Gs atom p and rows [64p, 64p + 64) of every slice
      // atom, on one barrier.
      auto load_khalf = [&](int p, int s, int rb, int ct) {
        if (!(ok = wait(&sm.cs_empty[p], cs_ph[p] ^ 1, abort, dev_err))) return;
        if (p == 0) {
          // pub[o][b] completes once per two tiles of owner o: parity (m >> 1) & 1.
          if (!(ok = wait_cluster(&sm.pub[s & (kCl - 1)][(s >> 3) & 1], (uint32_t)((s >> 4) & 1),
                                  abort, dev_err)))
            return;
          fence_proxy_async_global();
        }
        if (elect_one()) {
          mbar_expect_tx(&sm.cs_full[p], kAtom128 + (uint32_t)A * (kColAtom / 2));
          bulk_load(sm.g[0][p], gs_tile(s) + p * kAtom128, kAtom128, &sm.cs_full[p]);
          for (int j = 0; j < A; ++j)
            tma_load_2d(sm.cs[j] + p * (kColAtom / 2), &tmC64, &sm.cs_full[p], k * w + j * 64,
                        ct * BN + 64 * p);
        }
        __syncwarp();
        cs_last[p] = (int)cs_ph[p];
        cs_ph[p] ^= 1;
      };
      for (int s = 0; s < N && ok && ksplit; ++s, cur.next(mp)) {
        load_khalf(0, s, cur.rb, cur.ct);
        if (!ok) break;
        load_khalf(1, s, cur.rb, cur.ct);
      }
      for (int s = 0; s < N && ok && !ksplit; ++s, cur.next(mp)) {
        load_cs(0, 0, A0, cur.ct);
        if (!ok) break;
        // Gs(s) from its owner's ring slot.
        const int gb = s & (kGSlots - 1);
        // pub[o][b] completes once per two tiles of owner o: parity (m >> 1) & 1.
        if (!(ok = wait_cluster(&sm.pub[s & (kCl - 1)][(s >> 3) & 1], (uint32_t)((s >> 4) & 1), abort,
                                dev_err)))
          break;
        fence_proxy_async_global();
        if (!(ok = wait(&sm.gs_empty[gb], ge_ph[gb] ^ 1, abort, dev_err))) break;
        if (elect_one()) {
          mbar_expect_tx(&sm.g_full[gb], kGsBytes);
          bulk_load(sm.g[gb][0], gs_tile(s), kGsBytes, &sm.g_full[gb]);
        }
        __syncwarp();
        g_last[gb] = (int)ge_ph[gb];
        ge_ph[gb] ^= 1;
        if (A1 > 0) load_cs(1, A0, A1, cur.ct);
      }
      volatile int never = 0;
      for (int p = 0; p < 2; ++p)
        if (cs_last[p] >= 0) wait(&sm.cs_full[p], (uint32_t)cs_last[p], &never, dev_err);
      for (int i = 0; i < kGSlots; ++i)
        if (g_last[i] >= 0) wait(&sm.g_full[i], (uint32_t)g_last[i], &never, dev_err);
    }
  } else if (warp == 1 || warp == 7) {
    // Two MMA issuers with independent instruction streams: warp 1 the S
    // accumulations (TMEM columns [0, 256)), warp 7 the output update
    // (columns [256, 512)). tcgen05.mma issue runs only about one instruction
    // ahead of execution, so the bookkeeping between one warp's MMAs (barrier
    // polls, loop state) would otherwise leave the tensor pipe idle; with two
    // streams the other warp's MMAs fill those gaps. Each warp's commits
    // track its own MMAs only.
    {  // whole warp: uniform loop state; elected lane issues
      // Descriptors of every buffer, built once; K steps add to the start
      // address field (16-byte units). Buffers of one kind are contiguous,
      // so buffer i adds i times its size (in 16-byte units) to the base.
      const uint64_t da0 = sdesc_sw128(smem_u32(sm.a[0]), 16, 1024);
      const uint64_t db0 = sdesc_sw128(smem_u32(sm.b[0]), 16, 1024);
      const uint64_t dg0 = sdesc_sw128(smem_u32(sm.g[0][0]), 16, 1024);
      const uint64_t dc = sdesc_sw128(smem_u32(sm.cs[0]), kColAtom, 1024);
      constexpr uint32_t kAtomU = kAtom128 >> 4, kColU = kColAtom >> 4, kGsU = kGsBytes >> 4;
      bool ok = true;
      if (warp == 1) {
        int stage = 0;
        uint32_t ph = 0, s_ph[2] = {0, 0};
        for (int s = -kClJ; s < N && ok; ++s) {
          const int gj = job_of(s);
          if (gj < 0 || gj >= N) continue;
          const int buf = (gj >> 3) & 1;
          const int a0 = (s - (gj - kClJ)) * A;
          if (a0 == 0) {
            if (!(ok = wait(&sm.s_empty[buf], s_ph[buf] ^ 1, abort, dev_err))) break;
            tc_fence_after();
          }
          const uint32_t dt = tmem + buf * BN;
          for (int a = a0; a < a0 + A; ++a) {
            if (!(ok = wait(&sm.full[stage], ph, abort, dev_err))) break;
            const uint64_t da = da0 + stage * kAtomU, db = db0 + stage * kColU;
            if (elect_one()) {
#pragma unroll
              for (int kk = 0; kk < 4; ++kk)
                mma_bf16(dt, da + 2 * kk, db + 2 * kk, Tl::kIdescS, (a | kk) != 0);
              mma_commit(&sm.empty[stage]);
              if (a + 1 == nk) mma_commit(&sm.s_full[buf]);
            }
            __syncwarp();
            if (++stage == kClStages) { stage = 0; ph ^= 1; }
          }
          if (a0 + A == nk) s_ph[buf] ^= 1;
        }
      } else {
        uint32_t o_ph = 0, cs_ph[2] = {0, 0}, g_ph[kGSlots] = {};
        const uint32_t idesc_o0 = idesc_bf16(128, 64 * A0, 0, 1);
        const uint32_t idesc_o1 = idesc_bf16(128, 64 * (A1 > 0 ? A1 : 1), 0, 1);
        const uint64_t dc1 = dc + (uint64_t)A0 * kColU;
        TileCursor cur;  // tile of slot s
        cur.init(mp, 0);
        const uint32_t idesc_w = idesc_bf16(128, 64 * A, 0, 1);
        for (int s = 0; s < N && ok && ksplit; ++s, cur.next(mp)) {
          const bool unit_start = cur.unit_start(mp);
          const bool unit_end = cur.unit_end(mp);
          if (unit_start && !(ok = wait(&sm.o_empty, o_ph ^ 1, abort, dev_err))) break;
          for (int p = 0; p < 2 && ok; ++p) {
            if (!(ok = wait(&sm.cs_full[p], cs_ph[p], abort, dev_err))) break;
            cs_ph[p] ^= 1;
            tc_fence_after();
            if (elect_one()) {
#pragma unroll
              for (int q = 0; q < 4; ++q)
                mma_bf16(tmem_o, dg0 + p * kAtomU + q * 2,
                         dc + p * (kColU / 2) + q * (2048 >> 4), idesc_w,
                         !(unit_start && p == 0 && q == 0));
              mma_commit(&sm.cs_empty[p]);
              if (p == 1) {
                // Tell the owner of s that this CTA is done with tile s (see below).
                if (s + 2 * kCl < N)
                  mma_commit_multicast(&sm.gfree[(s >> 3) & 1], (uint16_t)(1u << (s & (kCl - 1))));
                if (unit_end) mma_commit(&sm.o_full);
              }
            }
            __syncwarp();
          }
          if (ok && unit_end) o_ph ^= 1;
        }
        for (int s = 0; s < N && ok && !ksplit; ++s, cur.next(mp)) {
          const int gb = s & (kGSlots - 1);
          const bool unit_start = cur.unit_start(mp);
          const bool unit_end = cur.unit_end(mp);
          if (unit_start && !(ok = wait(&sm.o_empty, o_ph ^ 1, abort, dev_err))) break;
          if (!(ok = wait(&sm.g_full[gb], g_ph[gb], abort, dev_err))) break;
          g_ph[gb] ^= 1;
          if (!(ok = wait(&sm.cs_full[0], cs_ph[0], abort, dev_err))) break;
          cs_ph[0] ^= 1;
          tc_fence_after();
          const uint64_t dg = dg0 + gb * kGsU;
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < BN / 16; ++kk)
              mma_bf16(tmem_o, dg + (kk >> 2) * kAtomU + (kk & 3) * 2, dc + kk * (2048 >> 4),
                       idesc_o0, !(unit_start && kk == 0));
            mma_commit(&sm.cs_empty[0]);
          }
          __syncwarp();
          if (A1 > 0) {
            if (!(ok = wait(&sm.cs_full[1], cs_ph[1], abort, dev_err))) break;
            cs_ph[1] ^= 1;
            tc_fence_after();
          }
          // Tell the owner of s that this CTA is done with tile s. The owner
          // publishes tile s + 16 (same ring slot, same pub barrier) only after
          // all 8 CTAs are, so no pub phase can run ahead of a consumer still
          // waiting on an earlier one.
          const bool notify = s + 2 * kCl < N;
          if (elect_one()) {
            if (A1 > 0) {
#pragma unroll
              for (int kk = 0; kk < BN / 16; ++kk)
                mma_bf16(tmem_o + 64 * A0, dg + (kk >> 2) * kAtomU + (kk & 3) * 2,
                         dc1 + kk * (2048 >> 4), idesc_o1, !(unit_start && kk == 0));
              mma_commit(&sm.cs_empty[1]);
            }
            mma_commit(&sm.gs_empty[gb]);
            if (notify)
              mma_commit_multicast(&sm.gfree[(s >> 3) & 1], (uint16_t)(1u << (s & (kCl - 1))));
            if (unit_end) mma_commit(&sm.o_full);
          }
          __syncwarp();
          if (unit_end) o_ph ^= 1;
        }
      }
      if (elect_one()) mma_commit(&sm.mma_done);
      __syncwarp();
      volatile int never = 0;
      wait(&sm.mma_done, 0, &never, dev_err);
    }
  } else {
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    uint32_t sf_ph[2] = {0, 0}, free_ph[2] = {0, 0}, o_ph = 0;
    bool ok = true;
    TileCursor cur;  // tile of slot s (s >= 0), for unit drains
    cur.init(mp, 0);
    // kFused: this thread's row partials (sum of P, maximum logit) over the
    // tiles this CTA owns in the current unit, and the tile of the
    // conversion phase (to find unit ends).
    float lacc = 0.f, macc = -INFINITY;
    TileCursor cg;
    cg.init(mp, 0);
    // Slot of the fused partials of the unit holding a tile: full units by
    // row block, tail units after them by (cluster, tail unit).
    auto fused_slot = [&](const TileCursor &t) {
      return mp.tail(t.g) ? n_rb + 2 * cid + ((t.rb - mp.rbT) - mp.t0 / mp.n_ct) : t.rb;
    };
    for (int s = -kClJ; s < N && ok; ++s) {
      const int g = s + kClLag + 1;  // tile whose S completes in slot s
      if (g >= 0 && g < N && (g & (kCl - 1)) == k) {
        const int m = g >> 3;
        const int buf = m & 1;
        TileCursor gt;
        gt.init(mp, g);
        const int rb = gt.rb, ct = gt.ct;
        float rc = 0.f, rl = 0.f;
        if (kTokenRows) {
          const int p = phys_rb(rb) * 128 + row;
          if (p < Teff) { rc = tok_c[p]; rl = kFused ? fa.ref[p] : lse[p] * kLog2e; }
        } else {
          epi_sync();
          const int p = ct * BN + row;
          if (row < BN) {
            sm.col_c[row] = p < Teff ? tok_c[p] : 0.f;
            sm.col_l[row] = p < Teff ? lse[p] * kLog2e : 0.f;
          }
          epi_sync();
        }
        if (!(ok = wait_sleepy(&sm.s_full[buf], sf_ph[buf], abort, dev_err))) break;
        sf_ph[buf] ^= 1;
        if (m >= 2) {
          // Every CTA has finished with this owner's tile g - 16.
          const int pb = m & 1;
          if (!(ok = wait_cluster(&sm.gfree[pb], free_ph[pb], abort, dev_err))) break;
          free_ph[pb] ^= 1;
        }
        tc_fence_after();
        uint8_t *dst_tile = gs_tile(g);
        float tsum = 0.f, tmax = -INFINITY;
#pragma unroll 1
        for (int c = 0; c < BN / 32; ++c) {
          float v[32];
          tmem_ld32(tmem + lane_off + buf * BN + c * 32, v);
          uint32_t pk[16];
#pragma unroll
          for (int j = 0; j < 32; j += 2) {
            float g2[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int col = c * 32 + j + e;
              float cc, ll;
              bool live;
              if (kTokenRows) {
                cc = rc; ll = rl;
                live = (rc != 0.f) && (ct * BN + col < V);
              } else {
                cc = sm.col_c[col]; ll = sm.col_l[col];
                live = cc != 0.f;
              }
              if (kFused) {
                // P = 2^(z log2 e - R_t); l and the maximum from the fp32 values.
                g2[e] = live ? ex2_approx(fmaf(v[j + e], kLog2e, -ll)) : 0.f;
                tsum += g2[e];
                if (live) tmax = fmaxf(tmax, v[j + e]);
              } else {
                g2[e] = live ? -cc * ex2_approx(fmaf(v[j + e], kLog2e, -ll)) : 0.f;
              }
            }
            __nv_bfloat162 b2 = __floats2bfloat162_rn(g2[0], g2[1]);
            pk[j >> 1] = *reinterpret_cast<uint32_t *>(&b2);
          }
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const int kc = c * 32 + q * 8;
            *reinterpret_cast<uint4 *>(dst_tile + (kc >> 6) * kAtom128 +
                                       sw128_offset(row, kc & 63)) =
                make_uint4(pk[q * 4], pk[q * 4 + 1], pk[q * 4 + 2], pk[q * 4 + 3]);
          }
        }
        if (kFused) {
          lacc += tsum;
          macc = fmaxf(macc, tmax);
        }
        tc_fence_before();
        mbar_arrive(&sm.s_empty[buf]);
        // The CTA barrier orders every epilogue thread's stores before the
        // elected thread's cluster-scope release (cumulativity); readers
        // fence the async proxy after acquiring pub[].
        epi_sync();
        if (warp == 2 && lane < kCl) {
          // One lane per destination CTA, in parallel: fence, then a relaxed
          // arrive (a release pattern per lane).
          fence_acq_rel_cluster();
          mbar_arrive_cluster_relaxed(mapa(smem_u32(&sm.pub[k][m & 1]), (uint32_t)lane));
        }
      }
      if (kFused && g >= 0 && g < N) {
        // Every CTA passes every tile g in order; at the last tile of a unit
        // it has converted all of its own tiles of that unit and publishes
        // its row partials (a CTA owning none of them publishes zeros).
        if (cg.unit_end(mp)) {
          const int slot = fused_slot(cg);
          float *lp = fa.lpart + ((size_t)slot * kCl + k) * 256;
          lp[row] = lacc;
          lp[128 + row] = macc;
          __threadfence();
          epi_sync();
          if (warp == 2 && lane == 0) {
            __threadfence();
            atomicAdd(&fa.ready[slot], 1);
          }
          lacc = 0.f;
          macc = -INFINITY;
        }
        cg.next(mp);
      }
      if (s < 0) continue;
      const bool unit_end = cur.unit_end(mp);
      const bool tail = mp.tail(cur.g);
      const int rb = cur.rb;
      // A tail unit's slot: its row block's place among this cluster's tail units.
      const int tu = tail ? (rb - mp.rbT) - mp.t0 / mp.n_ct : 0;
      const int fslot = kFused ? fused_slot(cur) : 0;
      cur.next(mp);
      if (unit_end) {
        // Drain the finished unit: out[rows, k*w : (k+1)*w].
        if (!(ok = wait_sleepy(&sm.o_full, o_ph, abort, dev_err))) break;
        o_ph ^= 1;
        tc_fence_after();
        const int rid = phys_rb(rb) * 128 + row;
        const bool valid = kTokenRows ? (rid < Teff) : (rid < V);
        float scale = 1.f;
        if (kFused) {
          // The unit's l and maximum: all kCl CTAs' partials, in CTA order.
          if (!(ok = wait_count(&fa.ready[fslot], kCl, abort, dev_err))) break;
          const float *lp = fa.lpart + (size_t)fslot * kCl * 256;
          float L = 0.f, M = -INFINITY;
#pragma unroll 1
          for (int j = 0; j < kCl; ++j) {
            L += __ldcg(lp + j * 256 + row);
            M = fmaxf(M, __ldcg(lp + j * 256 + 128 + row));
          }
          if (tail) {
            if (k == 0) {
              fa.tail_l[(cid * 2 + tu) * 256 + row] = L;
              fa.tail_l[(cid * 2 + tu) * 256 + 128 + row] = M;
            }
          } else if (valid) {
            const float R = fa.ref[rid];
            scale = -tok_c[rid] / L;
            if (k == 0) {
              const float M2 = M * kLog2e;
              fa.lse[rid] = (R + log2f(L)) * kLn2;
              fa.mrow[rid] = M2;
              if (!(L > 0.f) || !(L < INFINITY) || !(M2 - R <= kFixLog2))
                fa.rbflag[phys_rb(rb)] = 1;
            }
          }
        }
        float *dst = nullptr;
        if (tail)
          dst = tailbuf + ((int64_t)(cid * 2 + tu) * 128 + row) * d + k * w;
        else if (valid)
          dst = out + (kTokenRows ? (int64_t)tok_idx[rid] : (int64_t)rid) * d + k * w;
#pragma unroll 1
        for (int c = 0; c < w / 32; ++c) {
          float v[32];
          tmem_ld32(tmem_o + lane_off + c * 32, v);
          if (dst) {
#pragma unroll
            for (int q = 0; q < 8; ++q)
              reinterpret_cast<float4 *>(dst + c * 32)[q] =
                  make_float4(v[4 * q] * scale, v[4 * q + 1] * scale, v[4 * q + 2] * scale,
                              v[4 * q + 3] * scale);
          }
        }
        tc_fence_before();
        mbar_arrive(&sm.o_empty);
      }
    }
    // No column tiles at all (no active token): the slice is zero.
    if (ok && n_ct == 0) {
      for (int j = 0; j < n_my; ++j) {
        const int rid = (rb0 + cid + j * ncl) * 128 + row;
        if (!kTokenRows && rid < V)
          for (int c = 0; c < w; ++c) out[(int64_t)rid * d + k * w + c] = 0.f;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no CTA leaves while a peer may still signal its barriers
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// The cluster backward needs d = 8 * 64 * A with 1 <= A <= 6: each CTA's
// output slice of 64 * A columns stays in TMEM beside two S buffers of the
// column-tile width BN (2 BN + 64 A <= 512).
bool use_cluster_path(int d) { return grad_cluster_path(d); }
int cluster_tile_width(int d) { return d <= 2048 ? 128 : d <= 2560 ? 96 : 64; }

// Clusters that fit at once (persistent grid), from the occupancy API.
template <int BN>
int cluster_grid(const void *kernel, size_t smem) {
  static int cached = 0;
  if (cached) return cached;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kCl * 64, 1, 1);
  cfg.blockDim = dim3(kClThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    n = num_sms() / kCl;
  }
  if (n > kMaxClusters) n = kMaxClusters;
  cached = n > 0 ? n : 1;
  return cached;
}

// dH and dW by the cluster kernels with BN-wide column tiles. Row operands
// use 128-row boxes (mH for dH, mW128 for dW); column operands BN-row boxes.
template <int BN>
pair_status grad_bwd_cluster(const GradArgs &g, const GradWorkspace &w, cudaStream_t s,
                             const CUtensorMap &mH, const CUtensorMap &mW128) {
  CUtensorMap mHc, mWc, mHc64, mWc64;
  if (!make_map(&mHc, w.Hc, w.Tpad, g.d, BN) || !make_map(&mWc, g.W, g.V, g.d, BN) ||
      !make_map(&mHc64, w.Hc, w.Tpad, g.d, 64) || !make_map(&mWc64, g.W, g.V, g.d, 64))
    return PAIR_ERR_CUDA;
  const int nsm = num_sms();
  const size_t cl_smem = sizeof(ClSmem<BN>) + 1024;
  PAIR_CUDA_TRY(cudaFuncSetAttribute(bwd_cluster_kernel<true, BN>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)cl_smem));
  PAIR_CUDA_TRY(cudaFuncSetAttribute(bwd_cluster_kernel<false, BN>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)cl_smem));
  const int ncl = cluster_grid<BN>((const void *)bwd_cluster_kernel<true, BN>, cl_smem);
  uint8_t *gring = static_cast<uint8_t *>(w.gring);
  constexpr int kAll = 0x7fffffff;
  PAIR_BEGIN("bwd_dh_tc", s);
  bwd_cluster_kernel<true, BN><<<ncl * kCl, kClThreads, cl_smem, s>>>(
      mH, mWc, mWc64, g.d, g.V, w.counters, w.tok_idx, w.tok_c, w.lse, g.dH, gring,
      w.tailbuf, 0, kAll, FusedArgs{}, g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("tail_dh", s);
  tail_reduce_kernel<true, BN><<<nsm, 256, 0, s>>>(g.d, g.V, ncl, 0, kAll, w.counters,
                                                   w.tok_idx, w.tailbuf, g.dH);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("bwd_dw_tc", s);
  bwd_cluster_kernel<false, BN><<<ncl * kCl, kClThreads, cl_smem, s>>>(
      mW128, mHc, mHc64, g.d, g.V, w.counters, w.tok_idx, w.tok_c, w.lse, g.dW, gring,
      w.tailbuf, 0, kAll, FusedArgs{}, g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("tail_dw", s);
  tail_reduce_kernel<false, BN><<<nsm, 256, 0, s>>>(g.d, g.V, ncl, 0, kAll, w.counters,
                                                    w.tok_idx, w.tailbuf, g.dW);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

// The whole bf16 head without keeping any logit-sized tensor: target logits,
// the fused log-sum-exp + dH pass (and its fix-up for flagged row blocks),
// then dW by the recomputing cluster kernel. 4 logit-sized GEMMs per call.
template <int BN>
pair_status grad_head_fused(const GradArgs &g, const GradWorkspace &w, cudaStream_t s) {
  CUtensorMap mH, mW128, mHc, mWc, mHc64, mWc64;
  if (!make_map(&mH, w.Hc, w.Tpad, g.d, 128) || !make_map(&mW128, g.W, g.V, g.d, 128) ||
      !make_map(&mHc, w.Hc, w.Tpad, g.d, BN) || !make_map(&mWc, g.W, g.V, g.d, BN) ||
      !make_map(&mHc64, w.Hc, w.Tpad, g.d, 64) || !make_map(&mWc64, g.W, g.V, g.d, 64))
    return PAIR_ERR_CUDA;
  const int nsm = num_sms();
  const size_t cl_smem = sizeof(ClSmem<BN>) + 1024;
  PAIR_CUDA_TRY(cudaFuncSetAttribute(bwd_cluster_kernel<true, BN, true>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)cl_smem));
  PAIR_CUDA_TRY(cudaFuncSetAttribute(bwd_cluster_kernel<false, BN>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)cl_smem));
  const int ncl = cluster_grid<BN>((const void *)bwd_cluster_kernel<false, BN>, cl_smem);
  uint8_t *gring = static_cast<uint8_t *>(w.gring);
  constexpr int kAll = 0x7fffffff;
  const __nv_bfloat16 *Hc = static_cast<const __nv_bfloat16 *>(w.Hc);
  const __nv_bfloat16 *W = static_cast<const __nv_bfloat16 *>(g.W);
  PAIR_BEGIN("target_logit", s);
  target_logit_kernel<<<nsm * 8, 256, 0, s>>>(g.d, w.counters, w.tok_y, Hc, W, w.zy, w.ref,
                                              w.ready, w.n_slots, w.rbflag, w.n_rbmax);
  PAIR_LAUNCH_CHECK(s);
  FusedArgs fa{w.ref, w.lse, w.mrow, w.rbflag, w.lpart, w.ready, w.tail_l, nullptr, nullptr};
  for (int pass = 0; pass < 2; ++pass) {
    if (pass == 1) {
      PAIR_BEGIN("fixup_prep", s);
      fixup_prep_kernel<<<1, 1024, 0, s>>>(w.counters, w.rbflag, w.rb_list, w.counters + 1,
                                           w.ref, w.mrow, w.ready, w.n_slots);
      PAIR_LAUNCH_CHECK(s);
      fa.rb_list = w.rb_list;
      fa.n_list = w.counters + 1;
    }
    PAIR_BEGIN(pass == 0 ? "lse_dh_tc" : "lse_dh_fixup", s);
    bwd_cluster_kernel<true, BN, true><<<ncl * kCl, kClThreads, cl_smem, s>>>(
        mH, mWc, mWc64, g.d, g.V, w.counters, w.tok_idx, w.tok_c, nullptr, g.dH, gring,
        w.tailbuf, 0, kAll, fa, g.dev_err);
    PAIR_LAUNCH_CHECK(s);
    PAIR_BEGIN("tail_lse_dh", s);
    tail_fused_kernel<BN><<<nsm, 256, 0, s>>>(g.d, g.V, ncl, w.counters, w.tok_idx, w.tok_c,
                                               w.tailbuf, fa, g.dH);
    PAIR_LAUNCH_CHECK(s);
  }
  PAIR_BEGIN("bwd_dw_tc", s);
  bwd_cluster_kernel<false, BN><<<ncl * kCl, kClThreads, cl_smem, s>>>(
      mW128, mHc, mHc64, g.d, g.V, w.counters, w.tok_idx, w.tok_c, w.lse, g.dW, gring,
      w.tailbuf, 0, kAll, FusedArgs{}, g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("tail_dw", s);
  tail_reduce_kernel<false, BN><<<nsm, 256, 0, s>>>(g.d, g.V, ncl, 0, kAll, w.counters,
                                                    w.tok_idx, w.tailbuf, g.dW);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}

}  // namespace

namespace tck {

// The bf16 head without an image of softmax terms: the fused log-sum-exp + dH
// pass and the recomputing dW pass (cluster form), for the hidden sizes the
// cluster kernels take; false elsewhere (the caller runs the three passes).
bool onchip_fused_applies(int d) { return use_cluster_path(d); }

pair_status grad_head_onchip(const GradArgs &g, const GradWorkspace &w, cudaStream_t s) {
  switch (cluster_tile_width(g.d)) {
    case 128: return grad_head_fused<128>(g, w, s);
    case 96: return grad_head_fused<96>(g, w, s);
    default: return grad_head_fused<64>(g, w, s);
  }
}

// Softmax parts of dH and dW, recomputing the logits.
pair_status grad_bwd_recompute(const GradArgs &g, const GradWorkspace &w, cudaStream_t s) {
  CUtensorMap mH, mW128;
  if (!make_map(&mH, w.Hc, w.Tpad, g.d, 128) || !make_map(&mW128, g.W, g.V, g.d, 128))
    return PAIR_ERR_CUDA;
  if (use_cluster_path(g.d)) {
    switch (cluster_tile_width(g.d)) {
      case 128: return grad_bwd_cluster<128>(g, w, s, mH, mW128);
      case 96: return grad_bwd_cluster<96>(g, w, s, mH, mW128);
      default: return grad_bwd_cluster<64>(g, w, s, mH, mW128);
    }
  }
  const int nsm = num_sms();
  const size_t bwd_smem = sizeof(BwdSmem) + 1024;
  PAIR_CUDA_TRY(cudaFuncSetAttribute(bwd_kernel<true>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bwd_smem));
  PAIR_CUDA_TRY(cudaFuncSetAttribute(bwd_kernel<false>,
                                     cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bwd_smem));
  PAIR_BEGIN("bwd_dh_tc", s);
  bwd_kernel<true><<<nsm, kThreads, bwd_smem, s>>>(
      mH, mW128, g.d, g.V, w.counters, w.tok_idx, w.tok_c, w.lse, g.dH, g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  PAIR_BEGIN("bwd_dw_tc", s);
  bwd_kernel<false><<<nsm, kThreads, bwd_smem, s>>>(
      mW128, mH, g.d, g.V, w.counters, w.tok_idx, w.tok_c, w.lse, g.dW, g.dev_err);
  PAIR_LAUNCH_CHECK(s);
  return PAIR_OK;
}


}  // namespace tck
}  // namespace pairk
