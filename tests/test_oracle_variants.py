"""Pins of the oracle's weighting variants and product-design path against
what the paper and the mathematics fix (App. "Estimated and stabilized
propensities", the ablation table of Sec. 5, Theorem 2, the ESS definition of
App. D): closed forms, exact design enumeration and special cases."""
import itertools
import math

import numpy as np
import pytest

import oracle


def _rng(seed):
    return np.random.default_rng(seed)


def _loo(r, S):
    """Complete-pair average over the full group (Thm. 1): the LOO form."""
    G = r.size
    out = np.zeros(S.shape[1])
    for i in range(G):
        rbar = (r.sum() - r[i]) / (G - 1)
        out += (r[i] - rbar) * S[i]
    return out / G


def _h(r, S, i, j):
    """Eq. (pair-kernel)."""
    return 0.5 * (r[i] - r[j]) * (S[i] - S[j])


def _binary_rewards(rng, G):
    r = (rng.random(G) < 0.5).astype(float)
    if r.min() == r.max():
        r[0] = 1.0 - r[0]
    return r


def _independent_design(p):
    for bits in itertools.product((0, 1), repeat=p.size):
        J = np.array(bits, np.uint8)
        yield J, float(np.prod(np.where(J == 1, p, 1.0 - p)))


def _estimate(o, S):
    """g = sum_i a_i s_i (the coefficient form of Eq. pair-ht)."""
    return o["a"][0] @ S


@pytest.mark.parametrize("seed", range(3))
def test_unweighted_closed_form(seed):
    rng = _rng(600 + seed)
    G = 9
    r = rng.standard_normal(G)
    J = (rng.random(G) < 0.7).astype(np.uint8)
    J[:2] = 1
    rho = rng.uniform(0.1, 1.0, (G, G))
    o = oracle.coeffs_w(r[None], J[None], rho[None], wmode=oracle.W_UNWEIGHTED)
    assert o["status"] == 0
    K = int(J.sum())
    sK = float(r[J == 1].sum())
    want = np.where(J == 1, 0.5 * (K * r - sK), 0.0)  # 1/2 sum_{j in K} (r_i - r_j)
    np.testing.assert_allclose(o["a"][0], want, rtol=1e-13, atol=1e-13)
    assert o["edges"][0] == K * (K - 1) // 2
    assert o["ess"][0] == pytest.approx(K * (K - 1) / 2, rel=1e-14)  # equal weights
    assert o["max_w"][0] == 1.0


@pytest.mark.parametrize("seed", range(3))
def test_product_design_path_is_unbiased(seed):
    """Theorem 2 for the independent design, through the marginals-only path."""
    rng = _rng(610 + seed)
    G = int(rng.integers(3, 8)); D = 3
    r = _binary_rewards(rng, G)
    S = rng.standard_normal((G, D))
    p = rng.uniform(0.15, 0.95, G)
    M = math.comb(G, 2)
    E = np.zeros(D)
    for J, prob in _independent_design(p):
        o = oracle.coeffs_product(r[None], J[None], p[None], scale=1.0 / M)
        assert o["status"] == 0
        E += prob * _estimate(o, S)
    np.testing.assert_allclose(E, _loo(r, S), rtol=1e-11, atol=1e-12)


def test_marginal_weights_equal_ht_on_product_design():
    rng = _rng(620)
    B, G = 4, 11
    r = rng.standard_normal((B, G))
    J = (rng.random((B, G)) < 0.6).astype(np.uint8)
    p = rng.uniform(0.1, 1.0, (B, G))
    rho = p[:, :, None] * p[:, None, :]
    for b in range(B):
        np.fill_diagonal(rho[b], p[b])
    ht = oracle.coeffs_w(r, J, rho, wmode=oracle.W_HT)
    mg = oracle.coeffs_w(r, J, rho, wmode=oracle.W_MARGINAL)
    np.testing.assert_allclose(mg["a"], ht["a"], rtol=1e-13, atol=1e-14)
    np.testing.assert_allclose(mg["ess"], ht["ess"], rtol=1e-13)


def test_marginal_weights_bias_under_fixed_size_design():
    """Simple random sampling of m of n vertices: pi = m/n, rho = m(m-1)/(n(n-1))
    does not factor. HT is unbiased (Thm. 2 needs only rho > 0); marginal-only
    weights have the estimated-propensity bias (1/M) sum_e (rho_e/(pi_i pi_j) - 1) h_e."""
    n, m, D = 6, 3, 2
    rng = _rng(630)
    r = _binary_rewards(rng, n)
    S = rng.standard_normal((n, D))
    pi = m / n
    rho_e = m * (m - 1) / (n * (n - 1))
    rho = np.full((n, n), rho_e)
    np.fill_diagonal(rho, pi)
    M = math.comb(n, 2)
    subsets = list(itertools.combinations(range(n), m))
    E_ht = np.zeros(D); E_mg = np.zeros(D)
    for sub in subsets:
        J = np.zeros(n, np.uint8); J[list(sub)] = 1
        prob = 1.0 / len(subsets)
        E_ht += prob * _estimate(oracle.coeffs_w(r[None], J[None], rho[None], 1.0 / M), S)
        E_mg += prob * _estimate(oracle.coeffs_w(r[None], J[None], rho[None], 1.0 / M,
                                                 wmode=oracle.W_MARGINAL), S)
    target = _loo(r, S)
    np.testing.assert_allclose(E_ht, target, rtol=1e-12, atol=1e-13)
    bias = sum((rho_e / (pi * pi) - 1.0) * _h(r, S, i, j)
               for i in range(n) for j in range(i + 1, n)) / M
    np.testing.assert_allclose(E_mg - target, bias, rtol=1e-12, atol=1e-13)
    assert np.abs(bias).max() > 1e-2


@pytest.mark.parametrize("seed", range(3))
def test_clipped_weights_bias_formula(seed):
    """Clipped weight min(1/rho, w_max): conditional bias
    (1/M) sum_e (min(1, w_max rho_e) - 1) h_e (App. "Estimated and stabilized
    propensities"), by enumeration of the independent design."""
    rng = _rng(640 + seed)
    G = int(rng.integers(4, 8)); D = 3
    r = _binary_rewards(rng, G)
    S = rng.standard_normal((G, D))
    p = rng.uniform(0.1, 0.9, G)
    rho = np.outer(p, p)
    inv = 1.0 / rho[np.triu_indices(G, 1)]
    w_max = float(np.quantile(inv, 0.5))
    M = math.comb(G, 2)
    E = np.zeros(D)
    for J, prob in _independent_design(p):
        o = oracle.coeffs_w(r[None], J[None], rho[None], 1.0 / M, wmode=oracle.W_CLIPPED,
                            w_max=w_max)
        E += prob * _estimate(o, S)
    bias = sum((min(1.0, w_max * rho[i, j]) - 1.0) * _h(r, S, i, j)
               for i in range(G) for j in range(i + 1, G)) / M
    np.testing.assert_allclose(E - _loo(r, S), bias, rtol=1e-11, atol=1e-12)
    assert np.abs(bias).max() > 1e-3


def test_clipped_weights_limits():
    rng = _rng(650)
    B, G = 3, 12
    r = rng.standard_normal((B, G))
    J = (rng.random((B, G)) < 0.8).astype(np.uint8)
    rho = rng.uniform(0.05, 1.0, (B, G, G))
    ht = oracle.coeffs_w(r, J, rho)
    unw = oracle.coeffs_w(r, J, rho, wmode=oracle.W_UNWEIGHTED)
    hi = oracle.coeffs_w(r, J, rho, wmode=oracle.W_CLIPPED, w_max=1e9)
    lo = oracle.coeffs_w(r, J, rho, wmode=oracle.W_CLIPPED, w_max=0.5)  # < min 1/rho = 1
    np.testing.assert_array_equal(hi["a"], ht["a"])
    np.testing.assert_allclose(lo["a"], 0.5 * unw["a"], rtol=1e-14, atol=1e-15)
    assert np.all(lo["max_w"][lo["edges"] > 0] == 0.5)


@pytest.mark.parametrize("seed", range(3))
def test_hajek_is_the_ratio_estimator(seed):
    """Self-normalised weights: the group estimate is the ratio
    (sum_e I_e h_e / rho_e) / (sum_e I_e / rho_e); its numerator comes from the
    explicit edge enumeration of Eq. (pair-ht)."""
    rng = _rng(660 + seed)
    G, D = 10, 3
    r = rng.standard_normal(G)
    J = (rng.random(G) < 0.7).astype(np.uint8)
    J[:3] = 1
    S = rng.standard_normal((1, G, D))
    rho = rng.uniform(0.1, 1.0, (G, G))
    num, st = oracle.estimate_dense(r[None], J[None], rho[None], S, 1.0)
    assert st == 0
    den = sum(1.0 / rho[i, j] for i in range(G) for j in range(i + 1, G) if J[i] and J[j])
    o = oracle.coeffs_w(r[None], J[None], rho[None], wmode=oracle.W_HAJEK)
    np.testing.assert_allclose(_estimate(o, S[0]), num[0] / den, rtol=1e-12, atol=1e-13)


def test_hajek_with_constant_rho_is_selected_pair_average_and_biased():
    """rho = c: the ratio form reduces to the selected-pair average
    (sum_e I_e h_e) / K_E (App. A.4), which is not unbiased."""
    G, D = 5, 2
    r = np.array([1.0, 0, 0, 1, 0])
    S = np.array([[3.0, -1], [0, 2], [1, 1], [-2, 0.5], [0.5, 0]])
    p = np.array([0.9, 0.2, 0.5, 0.3, 0.8])
    c = 0.37
    rho = np.full((G, G), c)
    num = np.zeros(D); pk = 0.0
    for J, prob in _independent_design(p):
        K = int(J.sum())
        if K < 2:
            continue
        o = oracle.coeffs_w(r[None], J[None], rho[None], wmode=oracle.W_HAJEK)
        avg = sum(_h(r, S, i, j) for i in range(G) for j in range(i + 1, G)
                  if J[i] and J[j]) / (K * (K - 1) / 2)
        np.testing.assert_allclose(_estimate(o, S), avg, rtol=1e-12, atol=1e-13)
        num += prob * avg; pk += prob
    assert np.abs(num / pk - _loo(r, S)).max() > 1e-3


def test_ess_bounds_and_special_cases():
    rng = _rng(670)
    B, G = 50, 16
    r = rng.standard_normal((B, G))
    J = (rng.random((B, G)) < 0.5).astype(np.uint8)
    rho = rng.uniform(0.02, 1.0, (B, G, G))
    o = oracle.coeffs_w(r, J, rho)
    KE = o["edges"]
    has = KE > 0
    # 1 <= ESS <= K_E (Cauchy-Schwarz), equality at K_E = 1; 0 without edges.
    assert np.all(o["ess"][has] >= 1.0 - 1e-12)
    assert np.all(o["ess"][has] <= KE[has] + 1e-9)
    assert np.all(o["ess"][~has] == 0.0) and np.all(o["max_w"][~has] == 0.0)
    one = KE == 1
    np.testing.assert_allclose(o["ess"][one], 1.0, rtol=1e-14)
    # A planted tiny rho on a completed edge is the largest weight.
    J1 = np.ones((1, G), np.uint8)
    rho1 = np.full((1, G, G), 0.5)
    rho1[0, 3, 7] = 1e-3
    o1 = oracle.coeffs_w(r[:1], J1, rho1)
    assert o1["max_w"][0] == pytest.approx(1e3, rel=1e-14)


@pytest.mark.parametrize("wmode", [oracle.W_HT, oracle.W_UNWEIGHTED, oracle.W_MARGINAL,
                                   oracle.W_CLIPPED, oracle.W_HAJEK])
def test_variants_sum_to_zero(wmode):
    """Every variant is an antisymmetric edge sum: sum over J=1 of a_i is 0."""
    rng = _rng(680)
    B, G = 20, 24
    r = (rng.random((B, G)) < 0.5).astype(float)
    J = (rng.random((B, G)) < 0.6).astype(np.uint8)
    rho = rng.uniform(0.05, 1.0, (B, G, G))
    o = oracle.coeffs_w(r, J, rho, wmode=wmode, w_max=8.0)
    s = (o["a"] * J).sum(axis=1)
    assert np.all(np.abs(s) <= 1e-12 * (o["a_mag"].sum(axis=1) + 1e-300))


def test_marginal_rejects_nonpositive_marginal():
    G = 4
    r = np.array([[1.0, 0, 1, 0]])
    J = np.ones((1, G), np.uint8)
    rho = np.full((1, G, G), 0.5)
    rho[0, 2, 2] = 0.0
    assert oracle.coeffs_w(r, J, rho, wmode=oracle.W_MARGINAL)["status"] == 1
    assert oracle.coeffs_w(r, J, rho, wmode=oracle.W_HT)["status"] == 0


# ------------------------------------------------ frozen-population audit

def _exhaustive_draws(p):
    draws, probs = [], []
    for J, prob in _independent_design(p):
        draws.append(J); probs.append(prob)
    return np.array(draws, np.uint8), np.array(probs)


@pytest.mark.parametrize("seed", range(3))
def test_audit_exact_design_moments(seed):
    """Over all 2^G inclusion sets weighted by their probability: HT has zero
    bias (Thm. 2) and MSE equal to the trace of Prop. bias's covariance; the
    vertex and edge counts have means sum p_i and sum_{i<j} p_i p_j."""
    rng = _rng(700 + seed)
    G = int(rng.integers(3, 8)); D = 4
    r = rng.random(G)
    S = rng.standard_normal((G, D))
    p = rng.uniform(0.2, 0.95, G)
    rho = np.outer(p, p)
    M = math.comb(G, 2)
    Jd, w = _exhaustive_draws(p)
    o = oracle.audit(r, rho, S, Jd, w, scale=1.0 / M)
    assert o["status"] == 0
    assert o["bias_norm"] <= 1e-12 * math.sqrt(o["target_sq"])
    tr = 0.0
    for i in range(G):
        for j in range(i + 1, G):
            tr += (1.0 / (p[i] * p[j]) - 1.0) * float(_h(r, S, i, j) @ _h(r, S, i, j))
    for i in range(G):
        others = [j for j in range(G) if j != i]
        for j, k in itertools.combinations(others, 2):
            tr += 2.0 * (1.0 / p[i] - 1.0) * float(_h(r, S, i, j) @ _h(r, S, i, k))
    tr /= M * M
    assert o["mse"] == pytest.approx(tr, rel=1e-10)
    assert o["vertices"] == pytest.approx(p.sum(), rel=1e-13)
    pp = sum(p[i] * p[j] for i in range(G) for j in range(i + 1, G))
    assert o["edges"] == pytest.approx(pp, rel=1e-13)
    assert o["weight"] == pytest.approx(1.0, rel=1e-13)


def test_audit_unweighted_bias_vector():
    """Unweighted selection: bias (1/M) sum_e (rho_e - 1) h_e (Prop. bias)."""
    rng = _rng(710)
    G, D = 6, 3
    r = _binary_rewards(rng, G)
    S = rng.standard_normal((G, D))
    p = rng.uniform(0.2, 0.9, G)
    rho = np.outer(p, p)
    M = math.comb(G, 2)
    Jd, w = _exhaustive_draws(p)
    o = oracle.audit(r, rho, S, Jd, w, scale=1.0 / M, wmode=oracle.W_UNWEIGHTED)
    want = sum((rho[i, j] - 1.0) * _h(r, S, i, j) for i in range(G) for j in range(i + 1, G)) / M
    np.testing.assert_allclose(o["bias"], want, rtol=1e-11, atol=1e-13)
    assert o["bias_norm"] == pytest.approx(float(np.sqrt(want @ want)), rel=1e-11)


def test_audit_full_inclusion_is_exact():
    """Every draw completes the whole group with rho = 1: each estimate is the
    target itself (zero bias, zero MSE, cosine 1)."""
    rng = _rng(720)
    G, D = 7, 5
    r = rng.random(G)
    S = rng.standard_normal((G, D))
    Jd = np.ones((4, G), np.uint8)
    o = oracle.audit(r, np.ones((G, G)), S, Jd)
    assert o["bias_norm"] <= 1e-13 * math.sqrt(o["target_sq"])
    assert o["mse"] <= 1e-26 * o["target_sq"]
    assert o["cos"] == pytest.approx(1.0, abs=1e-14)
    assert o["edges"] == G * (G - 1) / 2


# --------------------------------------------------- reward standardisation

@pytest.mark.parametrize("seed", range(3))
def test_standardised_coefficients_are_grpo_scaled(seed):
    """rho = 1, every vertex completed: a_i = (G/2)(r_i - rbar) (Thm. 1), so the
    standardised coefficients are G/2 times GRPO's (r_i - rbar) / std(r, ddof=1)."""
    rng = _rng(730 + seed)
    G = 9
    r = rng.random(G)
    J = np.ones(G, np.uint8)
    o = oracle.coeffs_w(r[None], J[None], np.ones((1, G, G)), standardize=True)
    want = 0.5 * G * (r - r.mean()) / np.std(r, ddof=1)
    np.testing.assert_allclose(o["a"][0], want, rtol=1e-13, atol=1e-14)
    p = rng.uniform(0.2, 1.0, G)
    o2 = oracle.coeffs_product(r[None], J[None], p[None], standardize=True)
    o3 = oracle.coeffs_product(r[None], J[None], p[None])
    np.testing.assert_allclose(o2["a"][0], o3["a"][0] / np.std(r, ddof=1), rtol=1e-13)


def test_standardisation_uses_completed_rewards_only():
    r = np.array([[1.0, 0.0, 5.0, 1.0, 0.0]])
    J = np.array([[1, 1, 0, 1, 1]], np.uint8)
    rho = np.full((1, 5, 5), 0.5)
    o = oracle.coeffs_w(r, J, rho, standardize=True)
    o0 = oracle.coeffs_w(r, J, rho)
    sd = np.std(r[0][J[0] == 1], ddof=1)
    np.testing.assert_allclose(o["a"], o0["a"] / sd, rtol=1e-14)
    # Saturated group (equal completed rewards): coefficients stay 0.
    r2 = np.array([[1.0, 1.0, 0.0, 1.0]])
    J2 = np.array([[1, 1, 0, 1]], np.uint8)
    o2 = oracle.coeffs_w(r2, J2, np.full((1, 4, 4), 0.5), standardize=True)
    assert np.all(o2["a"] == 0.0) and o2["status"] == 0
