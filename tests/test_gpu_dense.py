"""GPU parity of pair_estimate_dense against the oracle's explicit edge
enumeration of Eq. (pair-ht)."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_11368_gb300 import synth
from tests.gpu_util import dev, dev_err_word

pytestmark = pytest.mark.gpu


def _binding():
    from paper_2608_11368_gb300 import binding
    return binding


def _check(inp, g_gpu, scale, tol=1e-5):
    ref, st = oracle.estimate_dense(inp["r"], inp["J"], inp["rho"], inp["S"], scale)
    assert st == 0
    c = oracle.coeffs(inp["r"], inp["J"], inp["rho"], scale=scale)
    S64 = inp["S"].astype(np.float64)
    bound = tol * np.einsum("bg,bg->b", np.abs(c["a"]), np.linalg.norm(S64, axis=2))
    g = g_gpu.cpu().numpy().astype(np.float64)
    err = np.linalg.norm(g - ref, axis=1)
    assert (err <= bound + 1e-30).all(), float((err - bound).max())
    none = ~(c["active"].astype(bool).any(axis=1))
    assert (g[none] == 0).all()


def test_dense_stress_full_size():
    B = _binding()
    wl = synth.WORKLOADS["coeffs_dense_stress"]
    inp = synth.make_dense_workload(wl, 0)
    err = dev_err_word()
    a = torch.empty((wl.B, wl.G), device="cuda")
    S = dev(inp["S"])
    g, _ = B.pair_estimate_dense(dev(inp["r"]), dev(inp["J"]), dev(inp["rho"]),
                                 S, a=a, dev_err=err)
    assert B.pair_status_sync(err) == 0
    assert B.pair_last_launch_count() == 1
    _check(inp, g, 1.0)
    a2 = B.pair_coeffs(dev(inp["r"]), dev(inp["J"]), dev(inp["rho"]))[0]
    assert torch.equal(a, a2)


@pytest.mark.parametrize("G,D", [(2, 1), (8, 3), (16, 4), (33, 7), (64, 1000),
                                 (100, 256), (128, 4096)])
def test_dense_shapes(G, D):
    B = _binding()
    wl = synth.WORKLOADS["coeffs_dense_stress"]
    inp = synth.make_dense_workload(wl, G + D, B=19, G=G, D=D)
    inp["J"][0] = 0                 # a group with no observed edge
    scale = 1.0 / math.comb(G, 2)
    g, _ = B.pair_estimate_dense(dev(inp["r"]), dev(inp["J"]), dev(inp["rho"]),
                                 dev(inp["S"]), scale=scale)
    _check(inp, g, scale)
    g2, _ = B.pair_estimate_dense(dev(inp["r"]), dev(inp["J"]), dev(inp["rho"]),
                                  dev(inp["S"]), scale=scale)
    assert torch.equal(g, g2)
