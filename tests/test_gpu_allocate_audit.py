"""The allocation step feeding the estimator (Sec. 4.3-4.5), on the GPU:
pair_allocate chooses the continuation probabilities of a group, and
pair_audit evaluates the HT estimator under that independent design over
all 2^G inclusion sets (exact weights).

Properties checked on the GPU's own allocation: design-unbiasedness (Thm 2:
zero bias under exact enumeration) and the appendix's variance bound (with
the edge proxy a_ij = ||h_ij||^2 the estimator's mean squared error is at
most the objective Phi the allocator minimised), and optimality against the
uniform design of the same expected cost. Parity: the audit of the oracle's
allocation against the oracle's audit of it."""
import itertools
import math

import numpy as np
import pytest
import torch

import oracle
from oracle import allocation as al
from tests.gpu_util import dev, dev_err_word

pytestmark = pytest.mark.gpu
pytest.importorskip("scipy")


def _binding():
    from paper_2608_11368_gb300 import binding
    return binding


def _group(seed, G, D):
    rng = np.random.default_rng(seed)
    r = (rng.random(G) < 0.5).astype(np.float32)
    r[0], r[1] = 1.0, 0.0
    S = rng.standard_normal((G, D)).astype(np.float32)
    Sd = S.astype(np.float64)
    rd = r.astype(np.float64)
    # a_ij = ||h_ij||^2 with h_ij = 1/2 (r_i - r_j)(s_i - s_j) (Eq. pair-kernel).
    a = 0.25 * (rd[:, None] - rd[None, :]) ** 2 * ((Sd[:, None, :] - Sd[None, :, :]) ** 2).sum(-1)
    a = a.astype(np.float32)
    c = rng.uniform(0.5, 2.0, G).astype(np.float32)
    budget = np.float32(0.5 * float(c.astype(np.float64).sum()))
    return r, S, a, c, budget


def _design(pi):
    G = pi.size
    Jd = np.array(list(itertools.product((0, 1), repeat=G)), np.uint8)
    w = np.prod(np.where(Jd == 1, pi[None], 1.0 - pi[None]), axis=1)
    rho = np.outer(pi, pi).astype(np.float32)
    np.fill_diagonal(rho, pi.astype(np.float32))
    return Jd, w, rho


def test_allocated_design_is_unbiased_and_within_its_bound():
    B = _binding()
    G, D, pi_min = 10, 24, 0.08
    r, S, a, c, budget = _group(3, G, D)
    err = dev_err_word()
    pi, st = B.pair_allocate(dev(c[None]), dev(np.array([budget])), pi_min, a=dev(a[None]),
                             dev_err=err)
    assert B.pair_status_sync(err) == 0
    st = st.cpu().numpy()[0]
    assert int(st[4]) == B.ALLOC_OK
    pi = pi.cpu().numpy()[0].astype(np.float64)
    Jd, w, rho = _design(pi.astype(np.float32).astype(np.float64))
    stats, bias = B.pair_audit(dev(r), dev(rho), dev(S), dev(Jd), draw_weight=dev(w), scale=1.0,
                               dev_err=err)
    assert B.pair_status_sync(err) == 0
    s = dict(zip(B.AUDIT_STATS, stats.cpu().numpy()))
    assert abs(s["weight"] - 1.0) < 1e-12
    # Thm 2: the HT estimator is design-unbiased (up to fp32 coefficient rounding).
    assert s["bias_norm"] <= 1e-5 * math.sqrt(s["target_sq"] + s["mse"])
    # Appendix bound: E||ghat - g||^2 = tr Cov <= Phi(-log pi) when a = ||h||^2.
    assert s["mse"] <= st[0] * (1 + 1e-6)
    # The allocator's Phi is no larger than the uniform design's of equal cost.
    uni = np.full(G, float(budget) / float(c.astype(np.float64).sum()))
    b = al.shared_vertex_b(a.astype(np.float64))
    assert st[0] <= al.design_objective(-np.log(uni), a.astype(np.float64), b) * (1 + 1e-9)


def test_audit_of_the_oracle_allocation_matches_the_oracle():
    B = _binding()
    G, D, pi_min = 9, 16, 0.08
    r, S, a, c, budget = _group(4, G, D)
    ref_alloc = al.allocate(a[None].astype(np.float64), c[None], [budget], pi_min)
    assert ref_alloc["status"][0] == al.ALLOC_OK
    pi = ref_alloc["pi"][0].astype(np.float32).astype(np.float64)
    Jd, w, rho = _design(pi)
    M = math.comb(G, 2)
    err = dev_err_word()
    stats, bias = B.pair_audit(dev(r), dev(rho), dev(S), dev(Jd), draw_weight=dev(w),
                               scale=1.0 / M, dev_err=err)
    assert B.pair_status_sync(err) == 0
    ref = oracle.audit(r, rho, S, Jd, draw_weight=w, scale=1.0 / M)
    got = stats.cpu().numpy()
    for k, name in enumerate(B.AUDIT_STATS):
        want = ref[name]
        tol = 2e-5 * (abs(want) if name != "bias_norm"
                      else math.sqrt(ref["target_sq"] + ref["mse"]))
        assert abs(got[k] - want) <= tol + 1e-30, (name, got[k], want)
    # Unbiased up to rho's fp32 rounding (relative 2^-24 per entry).
    assert ref["bias_norm"] <= 1e-7 * math.sqrt(ref["target_sq"] + ref["mse"])
