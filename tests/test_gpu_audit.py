"""GPU parity of pair_audit (frozen-population audit through the Gram matrix)
against the explicit fp64 oracle."""
import math

import numpy as np
import pytest
import torch

import oracle
from tests.gpu_util import dev, dev_err_word

pytestmark = pytest.mark.gpu

MODES = [oracle.W_HT, oracle.W_UNWEIGHTED, oracle.W_MARGINAL, oracle.W_CLIPPED, oracle.W_HAJEK]
KEYS = ("bias_norm", "mse", "cos", "vertices", "edges", "ess", "target_sq", "weight")


def _binding():
    from paper_2608_11368_gb300 import binding
    return binding


def _population(seed, G, D, N):
    rng = np.random.default_rng(seed)
    r = (rng.random(G) < 0.5).astype(np.float32)
    r[0], r[1] = 1.0, 0.0
    S = rng.standard_normal((G, D)).astype(np.float32)
    p = rng.uniform(0.1, 0.95, G).astype(np.float32)
    rho = np.outer(p, p).astype(np.float32)
    np.fill_diagonal(rho, p)
    Jd = (rng.random((N, G)) < p[None]).astype(np.uint8)
    return r, S, p, rho, Jd


def _check(stats, bias, ref, rtol):
    st = stats.cpu().numpy()
    for k, name in enumerate(KEYS):
        want = ref[name]
        scale = abs(want) if name not in ("bias_norm",) else math.sqrt(ref["target_sq"] + ref["mse"])
        assert abs(st[k] - want) <= rtol * scale + 1e-30, (name, st[k], want)
    bn = math.sqrt(ref["target_sq"] + ref["mse"])
    np.testing.assert_allclose(bias.cpu().numpy(), ref["bias"], rtol=0, atol=rtol * bn)


@pytest.mark.parametrize("G", [3, 8, 33, 64, 100])
@pytest.mark.parametrize("wmode", MODES)
def test_audit_parity(G, wmode):
    B = _binding()
    N, D = 700, 37
    r, S, p, rho, Jd = _population(800 + G, G, D, N)
    M = math.comb(G, 2)
    err = dev_err_word()
    stats, bias = B.pair_audit(dev(r), dev(rho), dev(S), dev(Jd), wmode=wmode, w_max=12.0,
                               scale=1.0 / M, dev_err=err)
    assert B.pair_last_launch_count() == 4
    assert B.pair_status_sync(err) == 0
    ref = oracle.audit(r, rho, S, Jd, scale=1.0 / M, wmode=wmode, w_max=12.0)
    _check(stats, bias, ref, rtol=2e-5)


def test_audit_exact_enumeration_on_gpu():
    """All 2^G draws with their probabilities: HT bias vanishes to fp32
    coefficient accuracy and the moments match the oracle."""
    B = _binding()
    G, D = 10, 16
    r, S, p, rho, _ = _population(850, G, D, 1)
    draws, probs = [], []
    for bits in range(1 << G):
        J = np.array([(bits >> i) & 1 for i in range(G)], np.uint8)
        draws.append(J)
        probs.append(float(np.prod(np.where(J == 1, p.astype(np.float64), 1.0 - p))))
    Jd = np.array(draws, np.uint8)
    w = np.array(probs)
    M = math.comb(G, 2)
    stats, bias = B.pair_audit(dev(r), dev(rho), dev(S), dev(Jd), draw_weight=dev(w),
                               scale=1.0 / M)
    ref = oracle.audit(r, rho, S, Jd, w, scale=1.0 / M)
    _check(stats, bias, ref, rtol=2e-5)
    assert stats[0].item() <= 1e-5 * math.sqrt(ref["target_sq"])


def test_audit_workspace_rules():
    B = _binding()
    L = B.lib()
    assert L.pair_audit_workspace_size(0, 8, 4) == 0
    assert L.pair_audit_workspace_size(10, 1, 4) == 0
    assert L.pair_audit_workspace_size(10, 129, 4) == 0
    assert L.pair_audit_workspace_size(10, 8, 0) == 0
    r, S, p, rho, Jd = _population(860, 6, 5, 20)
    small = torch.empty(64, dtype=torch.uint8, device="cuda")
    with pytest.raises(B.PairError):
        B.pair_audit(dev(r), dev(rho), dev(S), dev(Jd), ws=small)
