"""GPU parity of pair_coeffs against the fp64 oracle (Eq. pair-advantage)."""
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


def _check(ref, a, act, edges, contrast, tol=1e-6, center=False):
    a = a.cpu().numpy().astype(np.float64)
    bound = tol * ref["a_mag"]
    if center:
        bound = bound + tol * ref["a_mag"].mean(axis=1, keepdims=True)
    err = np.abs(a - ref["a"])
    assert (err <= bound + 1e-30).all(), float((err - bound).max())
    assert (a[ref["a"] == 0] == 0).all()
    assert np.array_equal(act.cpu().numpy(), ref["active"])
    assert np.array_equal(edges.cpu().numpy(), ref["edges"])
    assert np.array_equal(contrast.cpu().numpy(), ref["contrast"])


@pytest.mark.parametrize("seed", [0, 1, 2])
@pytest.mark.parametrize("name", synth.WORKLOAD_ORDER)
def test_coeffs_parity_workloads(name, seed):
    B = _binding()
    wl = synth.WORKLOADS[name]
    g = synth.draw_group_inputs(wl, seed)
    r, J, rho = dev(g["r"]), dev(g["J"]), dev(g["rho"])
    M = math.comb(wl.G, 2)
    for scale, flags in [(1.0, 0), (1.0 / M, 0), (1.0, B.PAIR_CENTER)]:
        err = dev_err_word()
        out = B.pair_coeffs(r, J, rho, scale=scale, flags=flags, dev_err=err)
        assert B.pair_last_launch_count() == 1
        assert B.pair_status_sync(err) == 0
        ref = oracle.coeffs(g["r"], g["J"], g["rho"], scale=scale,
                            center=bool(flags))
        _check(ref, *out, center=bool(flags))


@pytest.mark.parametrize("G", [2, 3, 5, 31, 32, 33, 63, 64, 65, 100, 127, 128])
def test_coeffs_group_sizes_partial_credit(G):
    B = _binding()
    rng = np.random.default_rng(G)
    nb = 37
    r = rng.random((nb, G)).astype(np.float32)
    r[::3] = (r[::3] < 0.5)
    J = (rng.random((nb, G)) < 0.6).astype(np.uint8)
    J[0] = 0                      # K = 0
    J[1] = 0; J[1, G - 1] = 1     # K = 1
    J[2] = 1; r[2] = 1.0          # all completed, all equal rewards
    u = rng.uniform(0.05, 1.0, (nb, G, G)).astype(np.float32)
    rho = np.triu(u, 1) + np.transpose(np.triu(u, 1), (0, 2, 1))
    err = dev_err_word()
    out = B.pair_coeffs(dev(r), dev(J), dev(rho), scale=0.3, dev_err=err)
    assert B.pair_status_sync(err) == 0
    ref = oracle.coeffs(r, J, rho, scale=0.3)
    _check(ref, *out)
    a = out[0].cpu().numpy()
    assert (a[0] == 0).all() and (a[1] == 0).all() and (a[2] == 0).all()
    # Bit-reproducible.
    again = B.pair_coeffs(dev(r), dev(J), dev(rho), scale=0.3)
    assert torch.equal(again[0], out[0])


def test_coeffs_rho_one_closed_form():
    B = _binding()
    G = 16
    r = (np.random.default_rng(1).random((8, G)) < 0.5).astype(np.float32)
    J = np.ones((8, G), np.uint8)
    rho = np.ones((8, G, G), np.float32)
    a = B.pair_coeffs(dev(r), dev(J), dev(rho))[0].cpu().numpy()
    expect = 0.5 * (G * r - r.sum(axis=1, keepdims=True))
    assert np.array_equal(a, expect.astype(np.float32))


def test_coeffs_nonpositive_inclusion_flagged_only_on_completed_edges():
    B = _binding()
    r = np.array([[1, 0, 1, 0]], np.float32)
    rho = np.full((1, 4, 4), 0.5, np.float32)
    rho[0, 0, 1] = 0.0
    err = dev_err_word()
    B.pair_coeffs(dev(r), dev(np.array([[1, 1, 1, 0]], np.uint8)), dev(rho),
                  dev_err=err)
    assert B.pair_status_sync(err) == 4
    assert int(err.item()) == 0          # reset by pair_status_sync
    rho[0, 0, 1] = np.nan
    B.pair_coeffs(dev(r), dev(np.array([[1, 1, 0, 1]], np.uint8)), dev(rho),
                  dev_err=err)
    assert B.pair_status_sync(err) == 4
    # Same bad value on an edge that is not observed: no error.
    out = B.pair_coeffs(dev(r), dev(np.array([[1, 0, 1, 1]], np.uint8)),
                        dev(rho), dev_err=err)
    assert B.pair_status_sync(err) == 0
    ref = oracle.coeffs(r, np.array([[1, 0, 1, 1]], np.uint8), rho)
    _check(ref, *out)


def test_coeffs_invalid_arguments():
    B = _binding()
    r = torch.zeros((2, 129), device="cuda")
    with pytest.raises(B.PairError) as e:
        B.pair_coeffs(r, torch.zeros((2, 129), dtype=torch.uint8, device="cuda"),
                      torch.zeros((2, 129, 129), device="cuda"))
    assert e.value.status == 1
    r = torch.zeros((2, 1), device="cuda")
    with pytest.raises(B.PairError):
        B.pair_coeffs(r, torch.zeros((2, 1), dtype=torch.uint8, device="cuda"),
                      torch.zeros((2, 1, 1), device="cuda"))
