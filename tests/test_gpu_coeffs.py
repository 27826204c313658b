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


def _boundary_inputs(seed, nb, G):
    """Groups whose completed counts sit at the packing boundaries of the
    streaming kernel (0, 1, 2, 31, 32, 33, 63, 64 completed, capped at G, at
    random positions), the rest with a per-group completion rate; one group
    carries NaN rewards on its incomplete rollouts, one signed-zero rewards,
    one a zero diagonal of rho."""
    rng = np.random.default_rng(seed)
    r = rng.random((nb, G)).astype(np.float32)
    r[::2] = (r[::2] < 0.5)
    J = (rng.random((nb, G)) < rng.uniform(0.05, 1.0, (nb, 1))).astype(np.uint8)
    for row, k in enumerate([0, 1, 2, 31, 32, 33, 63, 64]):
        J[row] = 0
        J[row, rng.permutation(G)[:min(k, G)]] = 1
    r[8] = 1.0                      # equal rewards: no contrast edge
    r[9][J[9] == 0] = np.nan        # rewards of rollouts that were not completed are unused
    J[10] = 1
    r[10, ::3] = -0.0               # -0 and +0 are equal rewards
    r[10, 1::3] = 0.0
    rho = rng.uniform(0.02, 1.0, (nb, G, G)).astype(np.float32)
    rho[11, np.arange(G), np.arange(G)] = 0.0   # the diagonal is never read
    return r, J, rho


@pytest.mark.parametrize("G", [4, 8, 12, 16, 36, 60, 64])
def test_coeffs_streaming_form(G):
    """Groups of at most 64 candidates with G a multiple of 4 run as a
    stream of groups per warp: completed counts at the packing boundaries,
    4000 groups (more than the resident warps, so each warp runs several),
    every flag combination, bit-identical reruns."""
    B = _binding()
    nb = 4000
    r, J, rho = _boundary_inputs(600 + G, nb, G)
    dr, dJ, drho = dev(r), dev(J), dev(rho)
    for scale, flags in [(1.0, 0), (0.3, B.PAIR_CENTER), (1.0, B.PAIR_STANDARDIZE),
                         (2.0, B.PAIR_STANDARDIZE | B.PAIR_CENTER)]:
        err = dev_err_word()
        out = B.pair_coeffs(dr, dJ, drho, scale=scale, flags=flags, dev_err=err)
        assert B.pair_last_launch_count() == 1
        assert B.pair_status_sync(err) == 0
        center, std = bool(flags & B.PAIR_CENTER), bool(flags & B.PAIR_STANDARDIZE)
        ref = oracle.coeffs_w(r, J, rho, scale=scale, center=center, standardize=std)
        _check(ref, *out, tol=3e-6 if std else 1e-6, center=center)
        again = B.pair_coeffs(dr, dJ, drho, scale=scale, flags=flags)
        for x, y in zip(out, again):
            assert torch.equal(x, y)


def test_coeffs_misaligned_inputs_take_the_general_kernel():
    """r four bytes off a 16-byte boundary: the general kernel runs, with
    the same results up to rounding."""
    B = _binding()
    G, nb = 64, 300
    r, J, rho = _boundary_inputs(77, nb, G)
    store = torch.empty(nb * G + 1, dtype=torch.float32, device="cuda")
    r_off = store[1:].view(nb, G)
    r_off.copy_(torch.from_numpy(r).cuda())
    assert r_off.data_ptr() % 16 != 0
    out = B.pair_coeffs(r_off, dev(J), dev(rho))
    _check(oracle.coeffs(r, J, rho), *out)
    aligned = B.pair_coeffs(dev(r), dev(J), dev(rho))
    for x, y in zip(out[1:], aligned[1:]):
        assert torch.equal(x, y)


def test_coeffs_streaming_form_reports_subnormal_rho():
    """The streaming form (G a multiple of 4, at most 64) takes the hardware
    reciprocal, so a completed edge's rho below 2^-126 is reported like
    rho <= 0; on an edge that was not observed it is never read."""
    B = _binding()
    G = 8
    r = np.tile(np.array([1, 0, 1, 0, 1, 0, 1, 0], np.float32), (2, 1))
    rho = np.full((2, G, G), 0.5, np.float32)
    rho[:, 0, 1] = np.float32(1e-39)          # subnormal
    J = np.ones((2, G), np.uint8)
    err = dev_err_word()
    B.pair_coeffs(dev(r), dev(J), dev(rho), dev_err=err)
    assert B.pair_status_sync(err) == 4
    J[:, 1] = 0
    out = B.pair_coeffs(dev(r), dev(J), dev(rho), dev_err=err)
    assert B.pair_status_sync(err) == 0
    _check(oracle.coeffs(r, J, rho), *out)
