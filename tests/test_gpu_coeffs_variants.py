"""GPU parity of pair_coeffs_weighted (every weighting variant, with ESS and
largest weight) and pair_coeffs_product against the fp64 oracle."""
import math

import numpy as np
import pytest

import oracle
from paper_2608_11368_gb300 import synth
from tests.gpu_util import dev, dev_err_word

pytestmark = pytest.mark.gpu

MODES = [oracle.W_HT, oracle.W_UNWEIGHTED, oracle.W_MARGINAL, oracle.W_CLIPPED, oracle.W_HAJEK]


def _binding():
    from paper_2608_11368_gb300 import binding
    return binding


def _check(ref, out, tol=1e-6, center=False):
    a, act, edges, contrast, ess, max_w = [t.cpu().numpy() for t in out]
    a = a.astype(np.float64)
    bound = tol * ref["a_mag"]
    if center:
        bound = bound + tol * ref["a_mag"].mean(axis=1, keepdims=True)
    err = np.abs(a - ref["a"])
    assert (err <= bound + 1e-30).all(), float((err - bound).max())
    assert (a[ref["a"] == 0] == 0).all()
    assert np.array_equal(act, ref["active"])
    assert np.array_equal(edges, ref["edges"])
    assert np.array_equal(contrast, ref["contrast"])
    # Diagnostics: fp32 tree sums of up to C(128, 2) weights.
    np.testing.assert_allclose(ess, ref["ess"], rtol=2e-5, atol=0)
    np.testing.assert_allclose(max_w, ref["max_w"], rtol=4e-7, atol=0)


def _inputs(seed, B, G, pJ=0.6, lo=0.02):
    rng = np.random.default_rng(seed)
    r = rng.random((B, G)).astype(np.float32)
    r[::2] = (r[::2] < 0.5)
    J = (rng.random((B, G)) < pJ).astype(np.uint8)
    J[0] = 0                      # no completed vertex
    J[1] = 0; J[1, G - 1] = 1     # one completed vertex, no edge
    p = rng.uniform(lo, 1.0, (B, G)).astype(np.float32)
    rho = rng.uniform(lo, 1.0, (B, G, G)).astype(np.float32)
    for b in range(B):
        np.fill_diagonal(rho[b], p[b])   # marginals on the diagonal
    return r, J, p, rho


@pytest.mark.parametrize("G", [2, 3, 4, 12, 17, 32, 33, 36, 60, 64, 65, 128])
@pytest.mark.parametrize("wmode", MODES)
def test_weighted_parity(G, wmode):
    B = _binding()
    r, J, p, rho = _inputs(900 + G, 29, G)
    M = math.comb(G, 2)
    w_max = 6.0
    for scale, flags in [(1.0, 0), (1.0 / M, B.PAIR_CENTER)]:
        err = dev_err_word()
        out = B.pair_coeffs_weighted(dev(r), dev(J), dev(rho), wmode=wmode, w_max=w_max,
                                     scale=scale, flags=flags, dev_err=err)
        assert B.pair_last_launch_count() == 1
        assert B.pair_status_sync(err) == 0
        ref = oracle.coeffs_w(r, J, rho, scale=scale, center=bool(flags), wmode=wmode,
                              w_max=w_max)
        assert ref["status"] == 0
        _check(ref, out, center=bool(flags))


def test_weighted_ht_matches_pair_coeffs_bitwise():
    B = _binding()
    g = synth.draw_group_inputs(synth.WORKLOADS["coeffs_dense_stress"], 0)
    r, J, rho = dev(g["r"][:512]), dev(g["J"][:512]), dev(g["rho"][:512])
    a0 = B.pair_coeffs(r, J, rho)[0]
    a1 = B.pair_coeffs_weighted(r, J, rho, wmode=B.PAIR_W_HT)[0]
    assert np.array_equal(a0.cpu().numpy(), a1.cpu().numpy())


@pytest.mark.parametrize("G", [2, 5, 32, 64, 100, 128])
def test_product_parity(G):
    B = _binding()
    r, J, p, _ = _inputs(950 + G, 31, G, lo=0.05)
    M = math.comb(G, 2)
    for scale, flags in [(1.0, 0), (1.0 / M, B.PAIR_CENTER)]:
        err = dev_err_word()
        out = B.pair_coeffs_product(dev(r), dev(J), dev(p), scale=scale, flags=flags, dev_err=err)
        assert B.pair_last_launch_count() == 1
        assert B.pair_status_sync(err) == 0
        ref = oracle.coeffs_product(r, J, p, scale=scale, center=bool(flags))
        _check(ref, out, tol=2e-6, center=bool(flags))


def test_product_on_stress_workload_marginals():
    """The marginals-only path on the stress workload's marginals."""
    B = _binding()
    g = synth.draw_group_inputs(synth.WORKLOADS["coeffs_dense_stress"], 1)
    r, J, p = g["r"][:1024], g["J"][:1024], g["p"][:1024]
    out = B.pair_coeffs_product(dev(r), dev(J), dev(p))
    ref = oracle.coeffs_product(r, J, p)
    _check(ref, out, tol=2e-6)


def test_variant_device_errors():
    B = _binding()
    G = 8
    r, J, p, rho = _inputs(990, 4, G)
    J[2] = 1
    rho2 = rho.copy(); rho2[2, 0, 5] = 0.0        # joint probability 0 on an edge
    err = dev_err_word()
    B.pair_coeffs_weighted(dev(r), dev(J), dev(rho2), wmode=B.PAIR_W_HAJEK, dev_err=err)
    assert B.pair_status_sync(err) == 4             # PAIR_ERR_NONPOSITIVE_INCLUSION
    B.pair_coeffs_weighted(dev(r), dev(J), dev(rho2), wmode=B.PAIR_W_UNWEIGHTED, dev_err=err)
    assert B.pair_status_sync(err) == 0             # rho is not read
    rho3 = rho.copy(); rho3[2, 3, 3] = -1.0       # marginal <= 0
    B.pair_coeffs_weighted(dev(r), dev(J), dev(rho3), wmode=B.PAIR_W_MARGINAL, dev_err=err)
    assert B.pair_status_sync(err) == 4
    p2 = p.copy(); p2[2, 4] = np.nan
    B.pair_coeffs_product(dev(r), dev(J), dev(p2), dev_err=err)
    assert B.pair_status_sync(err) == 4


def test_variant_host_validation():
    B = _binding()
    r, J, p, rho = _inputs(991, 2, 6)
    with pytest.raises(B.PairError):
        B.pair_coeffs_weighted(dev(r), dev(J), dev(rho), wmode=7)
    with pytest.raises(B.PairError):
        B.pair_coeffs_weighted(dev(r), dev(J), dev(rho), wmode=B.PAIR_W_CLIPPED, w_max=0.0)
    with pytest.raises(B.PairError):
        B.pair_coeffs_weighted(dev(r), dev(J), dev(rho), wmode=B.PAIR_W_CLIPPED,
                               w_max=float("inf"))
    # Unweighted needs no rho at all.
    out = B.pair_coeffs_weighted(dev(r), dev(J), None, wmode=B.PAIR_W_UNWEIGHTED)
    ref = oracle.coeffs_w(r, J, rho, wmode=oracle.W_UNWEIGHTED)
    _check(ref, out)


@pytest.mark.parametrize("G", [2, 8, 9, 33, 40, 64, 128])
def test_standardised_parity(G):
    B = _binding()
    r, J, p, rho = _inputs(970 + G, 23, G)
    J[3] = 0; J[3, 0] = 1; J[3, 1] = 1; r[3, 0] = r[3, 1] = 1.0   # saturated pair
    flags = B.PAIR_STANDARDIZE | B.PAIR_CENTER
    for wmode in (oracle.W_HT, oracle.W_CLIPPED, oracle.W_HAJEK):
        out = B.pair_coeffs_weighted(dev(r), dev(J), dev(rho), wmode=wmode, w_max=6.0,
                                     flags=flags)
        ref = oracle.coeffs_w(r, J, rho, center=True, wmode=wmode, w_max=6.0, standardize=True)
        _check(ref, out, tol=3e-6, center=True)
    a, act, edges, contrast = B.pair_coeffs(dev(r), dev(J), dev(rho), flags=B.PAIR_STANDARDIZE)
    ref = oracle.coeffs_w(r, J, rho, standardize=True)
    err = np.abs(a.cpu().numpy().astype(np.float64) - ref["a"])
    assert (err <= 3e-6 * ref["a_mag"] + 1e-30).all()
    out = B.pair_coeffs_product(dev(r), dev(J), dev(p), flags=B.PAIR_STANDARDIZE)
    ref = oracle.coeffs_product(r, J, p, standardize=True)
    _check(ref, out, tol=4e-6)
