"""Pins of the oracle's clipped trajectory-ratio surrogate (practical PPO
epochs, Sec. 4.5 and App. "Practical departures"): the on-policy special
case, torch autograd of the surrogate, and finite differences."""
import numpy as np
import pytest

import oracle
from paper_2608_11368_gb300 import synth


def _tiny_head(seed, d=8, V=23):
    wl = synth.WORKLOADS["pr1_ref_fp32"]
    return synth.make_head_workload(wl, seed, B=2, G=3, V=V, d=d, len_scale=0.12)


def _logp_old(inp, a, deltas, eps):
    """Old log-probabilities placing each trajectory ratio exp(delta) clearly
    inside or outside the clip interval."""
    base = oracle.pair_grad_ref(inp, a, full=True)
    return base["logp_seq"] - np.resize(np.asarray(deltas, np.float64), inp["R"])


def test_on_policy_point_is_the_pair_gradient():
    """At theta = theta_old every ratio is 1 and clipping is inactive."""
    inp = _tiny_head(1)
    a = np.linspace(-1.0, 1.0, inp["R"])
    base = oracle.pair_grad_ref(inp, a, full=True)
    out = oracle.pair_grad_clipped_ref(inp, a, base["logp_seq"], 0.2)
    np.testing.assert_array_equal(out["coef"], a)
    np.testing.assert_allclose(out["dH"], base["dH"], rtol=0, atol=0)
    np.testing.assert_allclose(out["dW"], base["dW"], rtol=0, atol=0)
    assert out["J"] == pytest.approx(float(a[a != 0].sum()), rel=1e-15)


@pytest.mark.parametrize("seed", [0, 1])
def test_surrogate_matches_torch_autograd(seed):
    torch = pytest.importorskip("torch")
    inp = _tiny_head(seed)
    rng = np.random.default_rng(seed)
    a = rng.standard_normal(inp["R"])
    a[0] = 0.0
    eps = 0.2
    lo = _logp_old(inp, a, [-0.6, -0.1, 0.0, 0.1, 0.6, 0.35], eps)
    out = oracle.pair_grad_clipped_ref(inp, a, lo, eps)
    H = torch.tensor(inp["H"], dtype=torch.float64, requires_grad=True)
    W = torch.tensor(inp["W"], dtype=torch.float64, requires_grad=True)
    seg = oracle.segment_ids(inp["cu_seqlens"])
    y = torch.tensor(np.where(inp["mask"] == 1, inp["y"], 0), dtype=torch.int64)
    lp = torch.log_softmax(H @ W.T, dim=1).gather(1, y[:, None])[:, 0]
    lp = lp * torch.tensor(inp["mask"], dtype=torch.float64)
    lps = torch.zeros(inp["R"], dtype=torch.float64).index_add(0, torch.tensor(seg), lp)
    A = torch.tensor(a)
    ratio = torch.exp(lps - torch.tensor(lo))
    L = torch.minimum(ratio * A, torch.clamp(ratio, 1 - eps, 1 + eps) * A)
    L = torch.where(A != 0, L, torch.zeros_like(L))
    L.sum().backward()
    assert out["J"] == pytest.approx(L.sum().item(), rel=1e-12)
    np.testing.assert_allclose(out["dH"], H.grad.numpy(), rtol=1e-10, atol=1e-13)
    np.testing.assert_allclose(out["dW"], W.grad.numpy(), rtol=1e-10, atol=1e-13)
    # At least one rollout of each kind: clipped (zero coefficient) and not.
    assert np.any((a != 0) & (out["coef"] == 0)) and np.any(out["coef"] != 0)


def test_surrogate_finite_differences():
    inp = _tiny_head(4, d=6, V=11)
    a = np.linspace(-1.0, 1.5, inp["R"])
    eps = 0.2
    lo = _logp_old(inp, a, [0.5, -0.05, 0.05, -0.5], eps)
    out = oracle.pair_grad_clipped_ref(inp, a, lo, eps)
    Hf = inp["H"].astype(np.float64)
    Wf = inp["W"].astype(np.float64)
    seg = oracle.segment_ids(inp["cu_seqlens"])
    m1 = inp["mask"] == 1

    def objective(Hm, Wm):
        Z = Hm @ Wm.T
        mx = Z.max(axis=1, keepdims=True)
        logp = Z - mx - np.log(np.exp(Z - mx).sum(axis=1, keepdims=True))
        lt = np.where(m1, logp[np.arange(Z.shape[0]), np.where(m1, inp["y"], 0)], 0.0)
        lps = np.zeros(inp["R"])
        np.add.at(lps, seg, lt)
        _, L = oracle.ppo_surrogate(a, lps, lo, eps)
        return float(L.sum())

    h = 1e-6
    idx = np.nonzero(inp["mask"])[0]
    for t, k in [(idx[0], 0), (idx[len(idx) // 2], 3), (idx[-1], 5)]:
        Hp = Hf.copy(); Hp[t, k] += h
        Hm = Hf.copy(); Hm[t, k] -= h
        fd = (objective(Hp, Wf) - objective(Hm, Wf)) / (2 * h)
        assert abs(fd - out["dH"][t, k]) < 1e-6
    for v, k in [(0, 1), (7, 4)]:
        Wp = Wf.copy(); Wp[v, k] += h
        Wm = Wf.copy(); Wm[v, k] -= h
        fd = (objective(Hf, Wp) - objective(Hf, Wm)) / (2 * h)
        assert abs(fd - out["dW"][v, k]) < 1e-6
