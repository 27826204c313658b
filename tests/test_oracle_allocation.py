"""Pins of the allocation oracle (Sec. 4.3-4.4): the contrast graph, the
shared-vertex surrogate, the convex design and its KKT checker, each against
something other than the oracle's own formulas."""
import itertools

import numpy as np
import pytest

from oracle import allocation as al

pytest.importorskip("scipy")


def _group(rng, G, pi_min=0.08, frac=0.5):
    p = rng.uniform(0.05, 0.95, G)
    c = rng.uniform(0.5, 2.0, G).astype(np.float32)
    a = al.edge_proxy(p[None])[0]
    budget = np.float32(frac * float(np.sum(c.astype(np.float64))))
    return p, a, c, budget, pi_min


def test_disagreement_is_the_probability_of_unequal_rewards():
    """Eq. (disagreement) by enumeration of the four reward outcomes of two
    independent Bernoulli rewards."""
    rng = np.random.default_rng(0)
    p = rng.uniform(0, 1, 6)
    d = al.disagreement(p)
    for i, j in itertools.permutations(range(6), 2):
        prob = sum((p[i] if ri else 1 - p[i]) * (p[j] if rj else 1 - p[j])
                   for ri in (0, 1) for rj in (0, 1) if ri != rj)
        assert abs(d[i, j] - prob) < 1e-15
    assert np.all(np.diag(d) == 0) and np.allclose(d, d.T)
    assert al.disagreement(np.array([0.5, 0.5]))[0, 1] == 0.5
    assert al.disagreement(np.array([1.0, 1.0]))[0, 1] == 0.0


def test_edge_proxy_with_score_norms():
    rng = np.random.default_rng(1)
    p = rng.uniform(0, 1, 5)
    m = rng.uniform(0.5, 3, 5)
    a = al.edge_proxy(p, m)
    d = al.disagreement(p)
    for i, j in itertools.permutations(range(5), 2):
        assert abs(a[i, j] - d[i, j] * ((m[i] + m[j]) / 2) ** 2) < 1e-14
    np.testing.assert_array_equal(al.edge_proxy(p, np.ones(5)), d)


def test_shared_vertex_b_is_the_sum_of_incident_cross_terms():
    """(sum sqrt a)^2 - sum a = 2 sum_{j<k, j,k != i} sqrt(a_ij a_ik)."""
    rng = np.random.default_rng(2)
    G = 7
    a = rng.uniform(0, 2, (G, G))
    a = a + a.T
    b = al.shared_vertex_b(a)
    for i in range(G):
        others = [j for j in range(G) if j != i]
        ref = 2 * sum(np.sqrt(a[i, j] * a[i, k]) for j, k in itertools.combinations(others, 2))
        assert abs(b[i] - ref) <= 1e-12 * max(ref, 1.0)


def _pair_kernels(rng, G, D):
    h = np.zeros((G, G, D))
    for i, j in itertools.combinations(range(G), 2):
        h[i, j] = rng.standard_normal(D)
        h[j, i] = h[i, j]
    return h


def test_b_bounds_the_shared_vertex_cross_products():
    """Cauchy-Schwarz (appendix): with a_ij = ||h_ij||^2,
    2 sum_{j<k} |<h_ij, h_ik>| <= b_i."""
    rng = np.random.default_rng(3)
    G, D = 6, 4
    h = _pair_kernels(rng, G, D)
    a = np.einsum("ijd,ijd->ij", h, h)
    b = al.shared_vertex_b(a)
    for i in range(G):
        others = [j for j in range(G) if j != i]
        cross = 2 * sum(abs(h[i, j] @ h[i, k]) for j, k in itertools.combinations(others, 2))
        assert cross <= b[i] * (1 + 1e-12)
    # Equality when the incident kernels are parallel and equally oriented.
    v = rng.standard_normal(D)
    hp = np.zeros((G, G, D))
    for j in range(1, G):
        hp[0, j] = hp[j, 0] = (j + 1.0) * v
    ap = np.einsum("ijd,ijd->ij", hp, hp)
    others = range(1, G)
    cross = 2 * sum(hp[0, j] @ hp[0, k] for j, k in itertools.combinations(others, 2))
    assert abs(al.shared_vertex_b(ap)[0] - cross) <= 1e-10 * cross


def test_objective_bounds_the_exact_design_covariance():
    """The appendix bound: for an independent Bernoulli(pi) design and
    a_ij >= ||h_ij||^2, the trace of the covariance of
    sum_{i<j} J_i J_j h_ij / (pi_i pi_j) is at most Phi(-log pi). Exact
    covariance by enumerating all 2^G inclusion sets."""
    rng = np.random.default_rng(4)
    G, D = 5, 3
    for trial in range(6):
        h = _pair_kernels(rng, G, D)
        a = np.einsum("ijd,ijd->ij", h, h) * (1.0 if trial % 2 == 0 else 1.3)
        b = al.shared_vertex_b(a)
        pi = rng.uniform(0.15, 1.0, G)
        mean = np.zeros(D)
        second = 0.0
        for J in itertools.product((0, 1), repeat=G):
            w = np.prod([pi[i] if J[i] else 1 - pi[i] for i in range(G)])
            g = sum(h[i, j] / (pi[i] * pi[j]) for i, j in itertools.combinations(range(G), 2)
                    if J[i] and J[j])
            g = np.asarray(g, np.float64) if not np.isscalar(g) else np.zeros(D)
            mean += w * g
            second += w * float(g @ g)
        target = sum(h[i, j] for i, j in itertools.combinations(range(G), 2))
        np.testing.assert_allclose(mean, target, atol=1e-9)  # design-unbiased (Thm 2)
        tr_cov = second - float(mean @ mean)
        assert tr_cov <= al.design_objective(-np.log(pi), a, b) * (1 + 1e-12)


def test_allocation_without_edges_is_the_closed_form():
    """a = 0, b > 0: minimising sum b_i / pi_i subject to sum c_i pi_i = B gives
    pi_i = sqrt(b_i / c_i) B / sum_k sqrt(c_k b_k) (Lagrange), when it lies
    inside [pi_min, 1]."""
    rng = np.random.default_rng(5)
    G = 10
    b = rng.uniform(1.0, 2.0, G)
    c = rng.uniform(0.8, 1.2, G).astype(np.float32)
    budget = np.float32(0.5 * float(np.sum(c.astype(np.float64))))
    out = al.allocate(np.zeros((1, G, G)), c[None], [budget], 0.08, b=b[None])
    cd = c.astype(np.float64)
    ref = np.sqrt(b / cd) * float(budget) / np.sum(np.sqrt(cd * b))
    assert np.all((ref > 0.08) & (ref < 1))
    assert out["status"][0] == al.ALLOC_OK
    np.testing.assert_allclose(out["pi"][0], ref, rtol=1e-12)


def test_symmetric_group_allocates_uniformly():
    G = 12
    a = np.full((1, G, G), 0.3)
    c = np.ones((1, G), np.float32)
    out = al.allocate(a, c, [np.float32(4.5)], 0.08)
    np.testing.assert_allclose(out["pi"][0], 4.5 / G, rtol=1e-7)


def test_special_cases_of_the_budget():
    G = 8
    rng = np.random.default_rng(6)
    a = al.edge_proxy(rng.uniform(0.1, 0.9, (1, G)))
    c = np.ones((1, G), np.float32)
    pi_min = 0.0625
    slack = al.allocate(a, c, [np.float32(8.0)], pi_min)
    assert slack["status"][0] == al.ALLOC_SLACK and np.all(slack["pi"] == 1.0)
    floor = al.allocate(a, c, [np.float32(0.5)], pi_min)
    assert floor["status"][0] == al.ALLOC_FLOOR and np.allclose(floor["pi"], pi_min, rtol=1e-15)
    bad = al.allocate(a, c, [np.float32(0.25)], pi_min)
    assert bad["status"][0] == al.ALLOC_INFEASIBLE
    flat = al.allocate(al.edge_proxy(np.ones((1, G))), c, [np.float32(4.0)], pi_min)
    assert flat["status"][0] == al.ALLOC_FLAT and flat["phi"][0] == 0.0
    np.testing.assert_allclose(flat["pi"][0], 0.5)


def test_allocation_g2_against_a_grid():
    """G = 2: the solver's objective is at most the minimum over a fine grid
    of feasible points, and within the grid's resolution of it."""
    rng = np.random.default_rng(7)
    for _ in range(3):
        p, a, c, budget, pi_min = _group(rng, 2)
        a = a + np.diag(np.zeros(2))
        b = al.shared_vertex_b(a)  # zero for G = 2
        b = b + rng.uniform(0.1, 0.5, 2)
        out = al.allocate(a[None], c[None], [budget], pi_min, b=b[None])
        X = -np.log(pi_min)
        xs = np.linspace(0, X, 801)
        x1, x2 = np.meshgrid(xs, xs, indexing="ij")
        cd = c.astype(np.float64)
        feas = cd[0] * np.exp(-x1) + cd[1] * np.exp(-x2) <= float(budget)
        phi = a[0, 1] * np.exp(x1 + x2) + b[0] * np.exp(x1) + b[1] * np.exp(x2)
        grid_min = phi[feas].min()
        assert out["phi"][0] <= grid_min * (1 + 1e-9)
        assert grid_min <= out["phi"][0] * (1 + 2e-2)


@pytest.mark.parametrize("G", [3, 8, 16, 64])
def test_allocation_satisfies_the_kkt_conditions(G):
    """For this convex program a KKT point is a global minimiser."""
    rng = np.random.default_rng(100 + G)
    for _ in range(3):
        p, a, c, budget, pi_min = _group(rng, G)
        out = al.allocate(a[None], c[None], [budget], pi_min)
        assert out["status"][0] == al.ALLOC_OK
        pi = out["pi"][0]
        assert np.all(pi >= pi_min * (1 - 1e-12)) and np.all(pi <= 1 + 1e-12)
        k = al.kkt_residual(pi, a, al.shared_vertex_b(a), c.astype(np.float64),
                            float(budget), pi_min)
        assert k["stat"] <= 1e-9, k
        assert abs(k["budget_excess"]) <= 1e-12 and k["comp"] <= 1e-9


@pytest.mark.parametrize("frac,pi_min", [(0.9, 0.08), (0.13, 0.08), (0.3, 0.2)])
def test_allocation_with_active_bounds(frac, pi_min):
    """Generous budgets push some pi_i to 1 and tight ones hold some at
    pi_min; the answer is still a KKT point with those bounds active."""
    rng = np.random.default_rng(int(frac * 100))
    G = 24
    n_bound = 0
    for _ in range(4):
        p = rng.uniform(0.02, 0.98, G)
        c = rng.uniform(0.2, 5.0, G).astype(np.float32)
        m = rng.uniform(0.3, 3.0, G)
        a = al.edge_proxy(p, m)
        budget = np.float32(frac * float(np.sum(c.astype(np.float64))))
        out = al.allocate(a[None], c[None], [budget], pi_min)
        assert out["status"][0] == al.ALLOC_OK
        pi = out["pi"][0]
        n_bound += int(np.sum((pi >= 1 - 1e-12) | (pi <= pi_min * (1 + 1e-12))))
        k = al.kkt_residual(pi, a, al.shared_vertex_b(a), c.astype(np.float64), float(budget),
                            pi_min)
        assert k["stat"] <= 1e-9 and abs(k["budget_excess"]) <= 1e-12, k
    assert n_bound > 0


def test_kkt_residual_detects_a_suboptimal_point():
    rng = np.random.default_rng(9)
    p, a, c, budget, pi_min = _group(rng, 16)
    out = al.allocate(a[None], c[None], [budget], pi_min)
    pi = out["pi"][0].copy()
    inner = np.nonzero((pi > pi_min * 1.2) & (pi < 0.8))[0]
    assert inner.size >= 2
    pi[inner[0]] *= 1.1
    pi[inner[1]] -= (pi[inner[0]] - out["pi"][0][inner[0]]) * c[inner[0]] / c[inner[1]]
    b = al.shared_vertex_b(a)
    k = al.kkt_residual(pi, a, b, c.astype(np.float64), float(budget), pi_min)
    assert k["stat"] > 1e-3
    assert al.design_objective(-np.log(pi), a, b) > out["phi"][0]


def test_allocation_does_not_depend_on_the_start():
    rng = np.random.default_rng(10)
    p, a, c, budget, pi_min = _group(rng, 16)
    o1 = al.allocate(a[None], c[None], [budget], pi_min)
    x0 = rng.uniform(0.2, 2.0, (1, 16))
    o2 = al.allocate(a[None], c[None], [budget], pi_min, x0=x0)
    np.testing.assert_allclose(o1["pi"], o2["pi"], rtol=1e-12)
