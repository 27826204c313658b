"""Seeded synthetic workloads for the Pair estimator hot path.

This module only draws random inputs; it contains none of the estimator's
arithmetic. The same arrays feed the CUDA path and the fp64 oracle.

The workloads mirror the RLVR setting of the paper (Sec. 3.3, adaptive suffix
continuation): G candidate rollouts per prompt, binary verifiable rewards
r_i ~ Bernoulli(q) with a per-prompt success rate q, continuation
probabilities p_i, completion indicators J_i ~ Bernoulli(p_i) and the logged
joint inclusion matrix rho (rho_ij = p_i p_j under the independent design).
The LM-head workloads add a packed variable-length token batch shaped like a
Qwen3-1.7B / Qwen3-4B output head: hidden states H ~ N(0, 1), head weight
W ~ N(0, 1/d), uniform target tokens.

Every array comes from its own PCG64 stream spawned from one SeedSequence,
so each array is reproducible on its own and independent of array sizes
drawn before it.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np

# Rollout segments in the packed buffer are padded to this multiple with
# mask = 0 tokens.
SEG_ALIGN = 8

# Stream indices (one PCG64 stream per array).
_S_Q, _S_R, _S_P, _S_J, _S_RHO, _S_LEN, _S_H, _S_W, _S_Y, _S_S = range(10)


@dataclasses.dataclass(frozen=True)
class Workload:
    """A named synthetic workload.

    kind: "head" (pair_coeffs + pair_grad over a packed token batch) or
          "dense" (pair_coeffs + pair_estimate_dense over explicit scores).
    """
    name: str
    kind: str
    B: int
    G: int
    d: int = 0            # hidden size (head) or score dimension D (dense)
    V: int = 0            # vocabulary size (head)
    dtype: str = "f32"    # "f32" or "bf16" storage of H and W
    q_dist: str = "uniform"   # "uniform" -> U(0,1); "beta" -> Beta(1/2, 1/2)
    p_low: float = 0.2        # p_i ~ U(p_low, 1)
    rho_kind: str = "product"  # "product" or "general"
    len_dist: str = "uniform"  # "uniform" or "lognormal"
    len_lo: int = 0
    len_hi: int = 0
    ln_median: float = 0.0
    ln_sigma: float = 0.0
    len_cap: int = 0
    prefix: int = 0           # > 0: non-continued rollouts truncated here


# The five workloads of the benchmark contract, sized as specified there.
WORKLOADS = {
    # fp32 reference: 4 prompts x 8 rollouts, d=256, V=4096.
    "pr1_ref_fp32": Workload("pr1_ref_fp32", "head", B=4, G=8, d=256, V=4096,
                             dtype="f32", p_low=0.2, len_lo=32, len_hi=64),
    # Qwen3-1.7B output head: d=2048, V=151936, 8 prompts x 8 rollouts.
    "qwen3_1p7b_head": Workload("qwen3_1p7b_head", "head", B=8, G=8, d=2048,
                                V=151936, dtype="bf16", p_low=0.2,
                                len_lo=256, len_hi=2048),
    # Qwen3-4B output head: d=2560, 16 prompts x 16 rollouts, q ~ Beta(.5,.5).
    "qwen3_4b_head": Workload("qwen3_4b_head", "head", B=16, G=16, d=2560,
                              V=151936, dtype="bf16", q_dist="beta",
                              p_low=0.1, len_lo=512, len_hi=4096),
    # Coefficient / dense-estimator stress: 4096 groups x 64, D=4096.
    "coeffs_dense_stress": Workload("coeffs_dense_stress", "dense", B=4096,
                                    G=64, d=4096, dtype="f32", p_low=0.05,
                                    rho_kind="general"),
    # Heavy-tailed long-context skew, Qwen3-1.7B head, 32 x 16 rollouts.
    "longctx_skew": Workload("longctx_skew", "head", B=32, G=16, d=2048,
                             V=151936, dtype="bf16", p_low=0.05,
                             len_dist="lognormal", ln_median=1500.0,
                             ln_sigma=0.9, len_cap=16384, prefix=256),
}
WORKLOAD_ORDER = ["pr1_ref_fp32", "qwen3_1p7b_head", "qwen3_4b_head",
                  "coeffs_dense_stress", "longctx_skew"]


def _streams(seed: int, n: int = 10):
    ss = np.random.SeedSequence(seed)
    return [np.random.Generator(np.random.PCG64(s)) for s in ss.spawn(n)]


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (round to nearest even); returns the
    16-bit patterns as uint16. Inputs are finite."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1)))
    return (rounded >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact upcast of bfloat16 bit patterns to float32."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32)
            << np.uint32(16)).view(np.float32)


def draw_group_inputs(wl: Workload, seed: int, B: Optional[int] = None,
                      G: Optional[int] = None):
    """Rewards, continuation probabilities, completion mask and logged
    inclusion matrix for B groups of G candidates.

    Returns dict with r [B,G] f32, p [B,G] f32, J [B,G] u8, rho [B,G,G] f32.
    rho is symmetric with rho_ii = p_i.
    """
    B = wl.B if B is None else B
    G = wl.G if G is None else G
    st = _streams(seed)
    if wl.q_dist == "beta":
        q = st[_S_Q].beta(0.5, 0.5, size=B)
    else:
        q = st[_S_Q].random(size=B)
    r = (st[_S_R].random(size=(B, G)) < q[:, None]).astype(np.float32)
    # p_i ~ U(p_low, 1]: 1 - U[0,1) lies in (0, 1].
    p = (wl.p_low + (1.0 - wl.p_low) * (1.0 - st[_S_P].random(size=(B, G))))
    p = p.astype(np.float32)
    J = (st[_S_J].random(size=(B, G)) < p).astype(np.uint8)
    if wl.rho_kind == "general":
        u = (0.05 + 0.95 * (1.0 - st[_S_RHO].random(size=(B, G, G))))
        u = u.astype(np.float32)
        upper = np.triu(u, 1)
        rho = upper + np.transpose(upper, (0, 2, 1))
        cap = np.minimum(p[:, :, None], p[:, None, :])
        rho = np.minimum(rho, cap).astype(np.float32)
    else:
        rho = (p[:, :, None] * p[:, None, :]).astype(np.float32)
    idx = np.arange(G)
    rho[:, idx, idx] = p
    return {"r": r, "p": p, "J": J, "rho": np.ascontiguousarray(rho)}


def draw_lengths(wl: Workload, seed: int, J: np.ndarray) -> np.ndarray:
    """Per-rollout response lengths [B*G] (int64), group-major order."""
    st = _streams(seed)[_S_LEN]
    n = J.size
    if wl.len_dist == "lognormal":
        L = np.exp(math.log(wl.ln_median) + wl.ln_sigma * st.standard_normal(n))
        L = np.minimum(np.maximum(np.rint(L), 1), wl.len_cap).astype(np.int64)
    else:
        L = st.integers(wl.len_lo, wl.len_hi, size=n, endpoint=True)
        L = L.astype(np.int64)
    if wl.prefix > 0:
        stopped = J.reshape(-1) == 0
        L[stopped] = np.minimum(L[stopped], wl.prefix)
    return L


def pack_lengths(L: np.ndarray):
    """Padded segment layout: cu_seqlens [R+1] int32 over padded segments and
    the token mask [T] uint8 (1 on response tokens, 0 on padding)."""
    padded = (L + SEG_ALIGN - 1) // SEG_ALIGN * SEG_ALIGN
    cu = np.zeros(L.size + 1, dtype=np.int64)
    np.cumsum(padded, out=cu[1:])
    T = int(cu[-1])
    mask = np.zeros(T, dtype=np.uint8)
    for i in range(L.size):
        mask[cu[i]:cu[i] + L[i]] = 1
    return cu.astype(np.int32), mask


def _normal_bits(gen, rows, cols, std, as_bf16, chunk=8192):
    """rows x cols N(0, std^2) draws, as bf16 bits (uint16) or float32."""
    out = np.empty((rows, cols), dtype=np.uint16 if as_bf16 else np.float32)
    for s in range(0, rows, chunk):
        e = min(rows, s + chunk)
        x = gen.standard_normal(size=(e - s, cols), dtype=np.float32)
        if std != 1.0:
            x *= np.float32(std)
        out[s:e] = f32_to_bf16_bits(x) if as_bf16 else x
    return out


def make_head_workload(wl: Workload, seed: int, B: Optional[int] = None,
                       G: Optional[int] = None, len_scale: float = 1.0,
                       V: Optional[int] = None, d: Optional[int] = None,
                       pad_fill: str = "zero", w_std_mult: float = 1.0,
                       draw_hw: bool = True):
    """Complete input set for pair_coeffs + pair_grad.

    Optional overrides shrink a workload (fewer groups, shorter responses,
    smaller V or d) for tests; the draws keep the workload's distributions.
    pad_fill: "zero" or "nan" for the hidden rows of padding tokens.
    w_std_mult scales the head weight std (a peaky-softmax variant for tests).
    draw_hw=False leaves H and W out (None): every other array is the same.
    """
    assert wl.kind == "head"
    B = wl.B if B is None else B
    G = wl.G if G is None else G
    V = wl.V if V is None else V
    d = wl.d if d is None else d
    grp = draw_group_inputs(wl, seed, B, G)
    L = draw_lengths(wl, seed, grp["J"])
    if len_scale != 1.0:
        L = np.maximum(1, np.rint(L * len_scale)).astype(np.int64)
    cu, mask = pack_lengths(L)
    T = int(cu[-1])
    st = _streams(seed)
    bf = wl.dtype == "bf16"
    H = _normal_bits(st[_S_H], T, d, 1.0, bf) if draw_hw else None
    W = _normal_bits(st[_S_W], V, d, w_std_mult / math.sqrt(d), bf) if draw_hw else None
    y = st[_S_Y].integers(0, V, size=T).astype(np.int32)
    pad = mask == 0
    y[pad] = -100
    if H is not None:
        if pad_fill == "nan":
            H[pad] = 0x7FC0 if bf else np.float32(np.nan)
        else:
            H[pad] = 0
    out = dict(grp)
    out.update(name=wl.name, B=B, G=G, R=B * G, T=T, d=d, V=V,
               dtype=wl.dtype, H=H, W=W, y=y, mask=mask, cu_seqlens=cu,
               lengths=L)
    return out


def make_dense_workload(wl: Workload, seed: int, B: Optional[int] = None,
                        G: Optional[int] = None, D: Optional[int] = None):
    """Complete input set for pair_coeffs + pair_estimate_dense: group inputs
    plus explicit per-rollout score vectors S [B, G, D] ~ N(0, 1)."""
    assert wl.kind == "dense"
    B = wl.B if B is None else B
    G = wl.G if G is None else G
    D = wl.d if D is None else D
    grp = draw_group_inputs(wl, seed, B, G)
    st = _streams(seed)
    S = _normal_bits(st[_S_S], B * G, D, 1.0, False).reshape(B, G, D)
    out = dict(grp)
    out.update(name=wl.name, B=B, G=G, D=D, S=S)
    return out


def as_float(x: np.ndarray, dtype: str) -> np.ndarray:
    """float32 view of stored H or W values (exact upcast for bf16)."""
    return bf16_bits_to_f32(x) if dtype == "bf16" else np.asarray(x, np.float32)


def make_alloc_inputs(seed: int, B: int, G: int, budget_frac: float = 0.5,
                      pi_min: float = 0.08, score_norms: bool = False):
    """Inputs of the allocation step (Sec. 4.3-4.4) for B groups of G
    candidates: predicted success probabilities p_hat ~ U(0.02, 0.98),
    predicted suffix costs c_hat ~ lognormal(ln 1, 0.6) (relative units),
    optionally score-norm predictions m_hat ~ U(0.3, 3), and a budget of
    budget_frac of each group's summed cost (the paper's 50 % default);
    float32 like the library's arguments. Returns a dict."""
    g = _streams(seed, 3)
    p_hat = g[0].uniform(0.02, 0.98, (B, G)).astype(np.float32)
    c_hat = g[1].lognormal(0.0, 0.6, (B, G)).astype(np.float32)
    m_hat = g[2].uniform(0.3, 3.0, (B, G)).astype(np.float32) if score_norms else None
    budget = (budget_frac * c_hat.astype(np.float64).sum(1)).astype(np.float32)
    return {"p_hat": p_hat, "c_hat": c_hat, "m_hat": m_hat, "budget": budget,
            "pi_min": np.float32(pi_min)}
