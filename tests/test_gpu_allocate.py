"""GPU parity of pair_allocate (the allocation step of Sec. 4.3-4.4) against
the fp64 oracle (SLSQP refined to a KKT point).

Tolerances. The program has a unique optimum; both sides reach it in fp64
(the GPU to a duality-gap bound of 1e-12 Phi), and pi is returned in fp32.
So: statuses are equal (both sides classify from the same fp64 sum of c in
index order); Phi agrees to 1e-9 relative; pi to 2e-6 relative (fp32
rounding 6e-8 plus the barrier's O(1/t) offset of coordinates at a bound);
the expected cost never exceeds the budget (the barrier keeps the fp64 point
strictly feasible); and the returned pi satisfies the KKT conditions to the
accuracy its fp32 rounding allows (1e-5)."""
import numpy as np
import pytest
import torch

from oracle import allocation as al
from paper_2608_11368_gb300 import synth
from tests.gpu_util import dev_err_word

pytestmark = pytest.mark.gpu
pytest.importorskip("scipy")


def _binding():
    from paper_2608_11368_gb300 import binding
    return binding


def _dev(x):
    return None if x is None else torch.from_numpy(np.ascontiguousarray(x)).cuda()


def _run(inp, explicit_a=None):
    B = _binding()
    err = dev_err_word()
    pi, stats = B.pair_allocate(_dev(inp["c_hat"]), _dev(inp["budget"]), float(inp["pi_min"]),
                                p_hat=None if explicit_a is not None else _dev(inp["p_hat"]),
                                m_hat=None if explicit_a is not None else _dev(inp["m_hat"]),
                                a=_dev(explicit_a), dev_err=err)
    st = B.pair_status_sync(err)
    return st, pi.cpu().numpy(), stats.cpu().numpy()


def _oracle(inp, explicit_a=None):
    if explicit_a is not None:
        a = explicit_a.astype(np.float64)
    else:
        a = al.edge_proxy(inp["p_hat"], inp["m_hat"])
    return a, al.allocate(a, inp["c_hat"], inp["budget"], float(inp["pi_min"]))


def _compare(inp, explicit_a=None, kkt_groups=4):
    st, pi, stats = _run(inp, explicit_a)
    assert st == 0
    a, ref = _oracle(inp, explicit_a)
    status = stats[:, 4].astype(int)
    np.testing.assert_array_equal(status, ref["status"])
    np.testing.assert_allclose(pi, ref["pi"], rtol=2e-6, atol=0)
    np.testing.assert_allclose(stats[:, 0], ref["phi"], rtol=1e-9, atol=0)
    c = inp["c_hat"].astype(np.float64)
    budget = inp["budget"].astype(np.float64)
    ok = status == al.ALLOC_OK
    assert np.all(stats[ok, 1] <= budget[ok])
    assert np.all(pi >= np.float32(inp["pi_min"])) and np.all(pi <= 1.0)
    b = al.shared_vertex_b(a)
    for g in np.nonzero(ok)[0][:kkt_groups]:
        k = al.kkt_residual(pi[g].astype(np.float64), a[g], b[g], c[g], float(budget[g]),
                            float(inp["pi_min"]), bound_tol=1e-6)
        assert k["stat"] <= 1e-5, (g, k)
    return pi, stats, ref


CASES = [
    # G, budget fraction, pi_min, score norms
    (2, 0.5, 0.08, False),
    (3, 0.3, 0.08, True),
    (8, 0.5, 0.08, False),
    (16, 0.5, 0.08, True),
    (16, 0.9, 0.05, False),   # generous: some pi = 1
    (33, 0.13, 0.08, True),   # tight: some pi = pi_min
    (64, 0.5, 0.08, False),
    (100, 0.3, 0.2, True),
    (128, 0.5, 0.08, False),
]


@pytest.mark.parametrize("case", CASES, ids=[f"G{c[0]}_f{c[1]}_m{int(c[3])}" for c in CASES])
def test_allocate_matches_oracle(case):
    G, frac, pi_min, norms = case
    inp = synth.make_alloc_inputs(G, 6, G, budget_frac=frac, pi_min=pi_min, score_norms=norms)
    _compare(inp)


def test_allocate_explicit_edge_proxy():
    inp = synth.make_alloc_inputs(3, 5, 24, score_norms=True)
    a = al.edge_proxy(inp["p_hat"], inp["m_hat"]).astype(np.float32)
    a = 0.5 * (a + np.swapaxes(a, 1, 2))
    _compare(inp, explicit_a=a)


def test_allocate_special_cases():
    """Slack, floor, infeasible and flat groups in one batch with a solved one."""
    G = 8
    c = np.ones((5, G), np.float32)
    p = np.tile(np.linspace(0.1, 0.9, G, dtype=np.float32), (5, 1))
    p[3] = 1.0                      # all predictions equal: no disagreement (flat)
    budget = np.array([8.0, 0.5, 0.25, 4.0, 4.0], np.float32)
    inp = {"p_hat": p, "c_hat": c, "m_hat": None, "budget": budget,
           "pi_min": np.float32(0.0625)}
    st, pi, stats = _run(inp)
    a, ref = _oracle(inp)
    np.testing.assert_array_equal(stats[:, 4].astype(int),
                                  [al.ALLOC_SLACK, al.ALLOC_FLOOR, al.ALLOC_INFEASIBLE,
                                   al.ALLOC_FLAT, al.ALLOC_OK])
    np.testing.assert_array_equal(stats[:, 4].astype(int), ref["status"])
    assert np.all(pi[0] == 1.0)
    assert np.all(pi[1] == np.float32(0.0625)) and np.all(pi[2] == np.float32(0.0625))
    np.testing.assert_allclose(pi[3], 0.5, rtol=1e-7)
    np.testing.assert_allclose(pi[4], ref["pi"][4], rtol=2e-6)
    assert st == 9  # PAIR_ERR_ALLOC_INFEASIBLE from the infeasible group


def test_allocate_invalid_inputs_are_flagged_per_group():
    inp = synth.make_alloc_inputs(5, 4, 16)
    inp["c_hat"][1, 3] = 0.0
    inp["p_hat"][2, 0] = 1.5
    inp["p_hat"][3, 5] = np.nan
    st, pi, stats = _run(inp)
    assert st == 8  # PAIR_ERR_ALLOC_INPUT
    status = stats[:, 4].astype(int)
    assert list(status[1:]) == [_binding().ALLOC_INVALID] * 3
    assert np.isnan(pi[1:]).all()
    good = {k: (v[:1] if isinstance(v, np.ndarray) and v.ndim else v) for k, v in inp.items()}
    _, ref = _oracle(good)
    np.testing.assert_allclose(pi[0], ref["pi"][0], rtol=2e-6)


def test_allocate_host_validation():
    B = _binding()
    inp = synth.make_alloc_inputs(6, 2, 8)
    c, bud = _dev(inp["c_hat"]), _dev(inp["budget"])
    for kw in ({"pi_min": 0.0}, {"pi_min": 1.5}):
        with pytest.raises(B.PairError):
            B.pair_allocate(c, bud, kw["pi_min"], p_hat=_dev(inp["p_hat"]))
    with pytest.raises(B.PairError):
        B.pair_allocate(c, bud, 0.08)          # neither p_hat nor a


def test_allocate_is_deterministic():
    inp = synth.make_alloc_inputs(7, 16, 64, score_norms=True)
    _, p1, s1 = _run(inp)
    _, p2, s2 = _run(inp)
    assert np.array_equal(p1, p2) and np.array_equal(s1, s2)


def test_allocate_full_size_sampled():
    """4096 groups of 64 (the coefficient stress size) in one launch: sampled
    groups against the oracle, KKT on more, budgets on all."""
    inp = synth.make_alloc_inputs(11, 4096, 64, score_norms=True)
    st, pi, stats = _run(inp)
    assert st == 0
    status = stats[:, 4].astype(int)
    assert np.all(status == al.ALLOC_OK)
    assert np.all(stats[:, 1] <= inp["budget"].astype(np.float64))
    rng = np.random.default_rng(0)
    sample = rng.choice(4096, 12, replace=False)
    sub = {k: (v[sample] if isinstance(v, np.ndarray) and v.ndim else v) for k, v in inp.items()}
    a, ref = _oracle(sub)
    np.testing.assert_allclose(pi[sample], ref["pi"], rtol=2e-6)
    np.testing.assert_allclose(stats[sample, 0], ref["phi"], rtol=1e-9)
