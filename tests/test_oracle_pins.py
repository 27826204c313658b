"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Nothing here compares the oracle with itself: every check is a closed form,
a theorem of the paper verified by exact enumeration, a hand-worked example,
a library routine, or finite differences.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest

import oracle
from paper_2608_11368_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rng(seed):
    return np.random.default_rng(seed)


def _loo(r, S):
    """Eq. (loo): (1/G) sum_i (r_i - mean_{j != i} r_j) s_i."""
    G = r.size
    out = np.zeros(S.shape[1])
    for i in range(G):
        rbar = (r.sum() - r[i]) / (G - 1)
        out += (r[i] - rbar) * S[i]
    return out / G


def _enumerate_J(p):
    """All 2^n inclusion vectors with their independent-design probability."""
    n = p.size
    for bits in itertools.product((0, 1), repeat=n):
        J = np.array(bits, np.uint8)
        prob = float(np.prod(np.where(J == 1, p, 1.0 - p)))
        yield J, prob


# --------------------------------------------------------------- hand example

def test_golden_hand_example():
    ex = json.load(open(os.path.join(GOLDEN, "coeffs_hand_g4.json")))
    r = np.array([ex["r"]]); J = np.array([ex["J"]], np.uint8)
    rho = np.array([ex["rho"]])
    c = oracle.coeffs(r, J, rho)
    np.testing.assert_allclose(c["a"][0], ex["a_scale1"], rtol=0, atol=1e-15)
    assert c["active"][0].tolist() == ex["active"]
    assert int(c["edges"][0]) == ex["edges"]
    assert int(c["contrast"][0]) == ex["contrast_edges"]
    S = np.array([ex["S"]])
    g, st = oracle.estimate_dense(r, J, rho, S)
    assert st == 0
    np.testing.assert_allclose(g[0], ex["g_scale1"], rtol=0, atol=1e-15)
    # scale = 1/M gives the paper's A_i (M = C(G,2) over all candidates).
    M = math.comb(ex["G"], 2)
    c2 = oracle.coeffs(r, J, rho, scale=1.0 / M)
    np.testing.assert_allclose(c2["a"][0], np.array(ex["a_scale1"]) / M,
                               rtol=1e-15, atol=0)


# --------------------------------------------- closed form: all observed, rho=1

@pytest.mark.parametrize("seed", range(6))
def test_closed_form_rho_one(seed):
    rng = _rng(seed)
    G = int(rng.integers(2, 13))
    binary = seed % 2 == 0
    r = (rng.random((3, G)) < 0.5).astype(float) if binary else rng.random((3, G))
    J = np.ones((3, G), np.uint8)
    rho = np.ones((3, G, G))
    c = oracle.coeffs(r, J, rho)
    # sum_{j != i} (r_i - r_j) = G r_i - sum_j r_j.
    expect = 0.5 * (G * r - r.sum(axis=1, keepdims=True))
    np.testing.assert_allclose(c["a"], expect, rtol=1e-13, atol=1e-13)
    assert (c["edges"] == G * (G - 1) // 2).all()


# ------------------------------------------------------------ Theorem 1 (LOO)

@pytest.mark.parametrize("seed", range(5))
def test_thm1_pair_average_is_loo(seed):
    rng = _rng(100 + seed)
    G = int(rng.integers(2, 11)); D = 5
    r = (rng.random(G) < 0.6).astype(float) if seed % 2 else rng.random(G)
    S = rng.standard_normal((1, G, D))
    M = math.comb(G, 2)
    g, st = oracle.estimate_dense(r[None], np.ones((1, G), np.uint8),
                                  np.ones((1, G, G)), S, scale=1.0 / M)
    assert st == 0
    loo = _loo(r, S[0])
    np.testing.assert_allclose(g[0], loo, rtol=1e-12, atol=1e-13)
    # Group-mean baseline = (G-1)/G times the pair average (Thm. 1).
    gm = ((r - r.mean())[:, None] * S[0]).sum(axis=0) / G
    np.testing.assert_allclose(gm, (G - 1) / G * g[0], rtol=1e-12, atol=1e-13)


# ------------------------------------- Theorem 2 / Prop. bias by enumeration

@pytest.mark.parametrize("seed", range(4))
def test_thm2_design_unbiased_and_naive_bias(seed):
    rng = _rng(200 + seed)
    G = int(rng.integers(3, 9)); D = 4
    r = (rng.random(G) < 0.5).astype(float)
    if r.min() == r.max():
        r[0] = 1.0 - r[0]
    S = rng.standard_normal((1, G, D))
    p = rng.uniform(0.15, 0.95, G)
    rho = np.outer(p, p)              # independent design (Sec. 3.3)
    M = math.comb(G, 2)
    target = _loo(r, S[0])            # complete-pair average (Thm. 1)
    E_ht = np.zeros(D); E_naive = np.zeros(D)
    for J, prob in _enumerate_J(p):
        g, st = oracle.estimate_dense(r[None], J[None], rho[None], S, 1.0 / M)
        assert st == 0
        E_ht += prob * g[0]
        g0, _ = oracle.estimate_dense(r[None], J[None], np.ones((1, G, G)), S,
                                      1.0 / M)
        E_naive += prob * g0[0]
    np.testing.assert_allclose(E_ht, target, rtol=1e-11, atol=1e-12)
    # Prop. bias: E[naive] - target = (1/M) sum_{i<j} (rho_ij - 1) h_ij.
    bias = np.zeros(D)
    for i in range(G):
        for j in range(i + 1, G):
            h = 0.5 * (r[i] - r[j]) * (S[0, i] - S[0, j])
            bias += (rho[i, j] - 1.0) * h
    bias /= M
    np.testing.assert_allclose(E_naive - target, bias, rtol=1e-11, atol=1e-12)
    assert np.abs(bias).max() > 1e-3


def test_ratio_estimator_is_biased():
    """App. A.4: dividing by the observed edge count K_E is not unbiased."""
    G = 5; D = 2
    r = np.array([1.0, 0, 0, 1, 0])
    S = np.array([[[3.0, -1], [0, 2], [1, 1], [-2, 0.5], [0.5, 0]]])
    p = np.array([0.9, 0.2, 0.5, 0.3, 0.8])
    rho = np.outer(p, p)
    target = _loo(r, S[0])
    num = np.zeros(D); pk = 0.0
    for J, prob in _enumerate_J(p):
        K = int(J.sum())
        KE = K * (K - 1) // 2
        if KE == 0:
            continue
        g0, _ = oracle.estimate_dense(r[None], J[None], np.ones((1, G, G)), S, 1.0)
        num += prob * g0[0] / KE
        pk += prob
    ratio = num / pk
    assert np.abs(ratio - target).max() > 1e-3


@pytest.mark.parametrize("seed", range(3))
def test_prop_covariance_independent_design(seed):
    """Prop. bias/covariance: exact design covariance for independent
    Bernoulli vertices versus enumeration."""
    rng = _rng(300 + seed)
    G = int(rng.integers(3, 8)); D = 3
    r = rng.random(G)
    S = rng.standard_normal((1, G, D))
    p = rng.uniform(0.2, 0.95, G)
    rho = np.outer(p, p)
    M = math.comb(G, 2)
    mean = np.zeros(D); second = np.zeros((D, D))
    for J, prob in _enumerate_J(p):
        g, _ = oracle.estimate_dense(r[None], J[None], rho[None], S, 1.0 / M)
        mean += prob * g[0]
        second += prob * np.outer(g[0], g[0])
    cov_enum = second - np.outer(mean, mean)

    def h(i, j):
        return 0.5 * (r[i] - r[j]) * (S[0, i] - S[0, j])
    C = np.zeros((D, D))
    for i in range(G):
        for j in range(i + 1, G):
            C += (1.0 / (p[i] * p[j]) - 1.0) * np.outer(h(i, j), h(i, j))
    for i in range(G):
        others = [j for j in range(G) if j != i]
        for j, k in itertools.combinations(others, 2):
            term = np.outer(h(i, j), h(i, k))
            C += (1.0 / p[i] - 1.0) * (term + term.T)   # symmetric completion
    C /= M * M
    np.testing.assert_allclose(cov_enum, C, rtol=1e-9, atol=1e-12)


# ------------------------------------------- edge-sum = coefficient collapse

@pytest.mark.parametrize("seed", range(4))
def test_edge_sum_equals_coefficient_collapse(seed):
    wl = synth.WORKLOADS["coeffs_dense_stress"]
    inp = synth.make_dense_workload(wl, seed, B=24, G=int(5 + 9 * seed), D=7)
    for scale in (1.0, 0.37):
        c = oracle.coeffs(inp["r"], inp["J"], inp["rho"], scale=scale)
        g, st = oracle.estimate_dense(inp["r"], inp["J"], inp["rho"], inp["S"],
                                      scale)
        assert st == 0
        coll = np.einsum("bg,bgd->bd", c["a"], inp["S"].astype(np.float64))
        bound = np.einsum("bg,bgd->bd", c["a_mag"],
                          np.abs(inp["S"].astype(np.float64)))
        assert (np.abs(g - coll) <= 1e-12 * bound + 1e-300).all()


# -------------------------------------------------------------- invariants

@pytest.mark.parametrize("name", ["pr1_ref_fp32", "qwen3_4b_head",
                                  "coeffs_dense_stress", "longctx_skew"])
def test_invariants(name):
    wl = synth.WORKLOADS[name]
    g = synth.draw_group_inputs(wl, 7, B=min(wl.B, 64))
    c = oracle.coeffs(g["r"], g["J"], g["rho"])
    a, J, r = c["a"], g["J"], g["r"]
    K = J.sum(axis=1).astype(int)
    assert (c["edges"] == K * (K - 1) // 2).all()
    # Binary rewards: contrast edges = (#observed with r=1) * (#observed r=0).
    K1 = (J * (r == 1)).sum(axis=1); K0 = (J * (r == 0)).sum(axis=1)
    assert (c["contrast"] == K1 * K0).all()
    # Sum over observed vertices vanishes (antisymmetric edge terms).
    s = (a * J).sum(axis=1)
    assert (np.abs(s) <= 1e-12 * np.abs(c["a_mag"]).sum(axis=1) + 1e-300).all()
    # a_i = 0 exactly off the active set; sign(a_i) = sign(2 r_i - 1) on it.
    act = c["active"] == 1
    assert (a[~act] == 0).all()
    assert (np.sign(a[act]) == np.sign(2 * r[act] - 1)).all()
    assert (act == ((J == 1) & (K1[:, None] > 0) & (K0[:, None] > 0))).all()


def test_center_flag_only_moves_rounding():
    wl = synth.WORKLOADS["coeffs_dense_stress"]
    g = synth.draw_group_inputs(wl, 3, B=32)
    c0 = oracle.coeffs(g["r"], g["J"], g["rho"])
    c1 = oracle.coeffs(g["r"], g["J"], g["rho"], center=True)
    assert (np.abs(c1["a"] - c0["a"]) <= 1e-12 * c0["a_mag"].max()).all()
    assert (c1["a"][g["J"] == 0] == 0).all()


def test_nonpositive_inclusion():
    r = np.array([[1.0, 0.0, 1.0]])
    rho = np.full((1, 3, 3), 0.5)
    rho[0, 0, 1] = 0.0
    # Completed edge with rho <= 0: flagged (the paper requires rho > 0).
    c = oracle.coeffs(r, np.array([[1, 1, 0]], np.uint8), rho)
    assert c["status"] == oracle.ORACLE_ERR_NONPOSITIVE_INCLUSION
    rho[0, 0, 1] = np.nan
    c = oracle.coeffs(r, np.array([[1, 1, 0]], np.uint8), rho)
    assert c["status"] == oracle.ORACLE_ERR_NONPOSITIVE_INCLUSION
    # The same rho on an edge that is not observed is never read.
    c = oracle.coeffs(r, np.array([[1, 0, 1]], np.uint8), rho)
    assert c["status"] == 0


# ----------------------------------------------------------------- LM head

def _tiny_head(seed, B=2, G=3, d=12, V=37, w_mult=1.0):
    wl = synth.WORKLOADS["pr1_ref_fp32"]
    inp = synth.make_head_workload(wl, seed, B=B, G=G, V=V, d=d,
                                   len_scale=0.12, w_std_mult=w_mult)
    return inp


@pytest.mark.parametrize("seed,w_mult", [(0, 1.0), (1, 8.0), (2, 1.0)])
def test_head_matches_torch_autograd(seed, w_mult):
    torch = pytest.importorskip("torch")
    inp = _tiny_head(seed, w_mult=w_mult)
    rng = _rng(seed)
    a = rng.standard_normal(inp["R"])
    a[0] = 0.0
    ref = oracle.pair_grad_ref(inp, a, full=True)
    H = torch.tensor(inp["H"], dtype=torch.float64, requires_grad=True)
    W = torch.tensor(inp["W"], dtype=torch.float64, requires_grad=True)
    seg = oracle.segment_ids(inp["cu_seqlens"])
    c = torch.tensor(a[seg] * inp["mask"], dtype=torch.float64)
    y = torch.tensor(np.where(inp["mask"] == 1, inp["y"], 0), dtype=torch.int64)
    lp = torch.log_softmax(H @ W.T, dim=1).gather(1, y[:, None])[:, 0]
    Jt = (c * lp).sum()
    Jt.backward()
    assert abs(ref["J"] - Jt.item()) <= 1e-12 * max(1.0, ref["J_abs"])
    np.testing.assert_allclose(ref["dH"], H.grad.numpy(), rtol=1e-11, atol=1e-13)
    np.testing.assert_allclose(ref["dW"], W.grad.numpy(), rtol=1e-11, atol=1e-13)
    # Rows outside the objective are exactly zero.
    off = (inp["mask"] == 0) | (a[seg] == 0)
    assert (ref["dH"][off] == 0).all()


def test_head_finite_differences():
    inp = _tiny_head(5, d=6, V=11)
    a = np.linspace(-1.0, 1.5, inp["R"])
    ref = oracle.pair_grad_ref(inp, a, full=True)
    Hf = inp["H"].astype(np.float64); Wf = inp["W"].astype(np.float64)

    def objective(Hm, Wm):
        idx, c, _ = oracle.compact_tokens(inp["cu_seqlens"], inp["mask"], a)
        Z = Hm[idx] @ Wm.T
        m = Z.max(axis=1, keepdims=True)
        logp = Z - m - np.log(np.exp(Z - m).sum(axis=1, keepdims=True))
        return float((c * logp[np.arange(idx.size), inp["y"][idx]]).sum())

    eps = 1e-6
    idx = np.nonzero(inp["mask"])[0]
    for t, k in [(idx[0], 0), (idx[3], 2), (idx[-1], 5)]:
        Hp = Hf.copy(); Hp[t, k] += eps
        Hm = Hf.copy(); Hm[t, k] -= eps
        fd = (objective(Hp, Wf) - objective(Hm, Wf)) / (2 * eps)
        assert abs(fd - ref["dH"][t, k]) < 1e-6
    for v, k in [(0, 1), (int(inp["y"][idx[2]]), 3), (10, 4)]:
        Wp = Wf.copy(); Wp[v, k] += eps
        Wm = Wf.copy(); Wm[v, k] -= eps
        fd = (objective(Hf, Wp) - objective(Hf, Wm)) / (2 * eps)
        assert abs(fd - ref["dW"][v, k]) < 1e-6


def test_head_gradient_is_pair_ht_over_sequence_scores():
    """dW of sum_i A_i log pi equals Eq. (pair-ht) over the materialised
    sequence scores s_i = d log pi(o_i|q) / dW (Sec. 4.5)."""
    inp = _tiny_head(9, B=2, G=4, d=5, V=9)
    c = oracle.coeffs(inp["r"], inp["J"], inp["rho"])
    a = c["a"].reshape(-1)
    R = inp["R"]; V, d = inp["V"], inp["d"]
    scores = np.zeros((R, V * d))
    for i in range(R):
        e = np.zeros(R); e[i] = 1.0
        scores[i] = oracle.pair_grad_ref(inp, e, full=True)["dW"].reshape(-1)
    dW = oracle.pair_grad_ref(inp, a, full=True)["dW"].reshape(-1)
    g, st = oracle.estimate_dense(inp["r"], inp["J"], inp["rho"],
                                  scores.reshape(inp["B"], inp["G"], V * d))
    assert st == 0
    np.testing.assert_allclose(dW, g.sum(axis=0), rtol=1e-10, atol=1e-12)


def test_compaction_definition():
    inp = _tiny_head(3)
    a = np.arange(inp["R"], dtype=float) - 2.0
    idx, c, seg = oracle.compact_tokens(inp["cu_seqlens"], inp["mask"], a)
    cu = inp["cu_seqlens"]
    brute = [t for i in range(inp["R"]) for t in range(cu[i], cu[i + 1])
             if inp["mask"][t] == 1 and a[i] != 0]
    assert idx.tolist() == brute
    assert all(c[k] == a[seg[k]] for k in range(idx.size))
