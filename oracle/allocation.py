"""Allocation step before the path (Sec. 4.3-4.4): the contrast graph and the
convex continuation design. TEST INFRASTRUCTURE ONLY, under the same rules as
the rest of ``oracle`` (only tests/, ``__graft_entry__.smoke()`` and the CPU
legs of ``bench.py`` may use it; it shares no code with the CUDA library).

Definitions, each written out from the paper in fp64:

* ``disagreement``: Eq. (disagreement), the probability that two completed
  suffixes with success probabilities p_i, p_j disagree,
  d_ij = p_i (1 - p_j) + (1 - p_i) p_j (pairs i != j; the diagonal is 0).
* ``edge_proxy``: Eq. (edge-proxy), the parameter-free default a_ij = d_ij,
  or d_ij (m_i + m_j)^2 / 4 with a score-norm predictor m.
* ``shared_vertex_b``: Sec. 4.4, b_i = (sum_{j != i} sqrt(a_ij))^2 -
  sum_{j != i} a_ij, the surrogate for the cross-products of edges sharing
  vertex i.
* ``design_objective``: Eq. (convex-objective),
  Phi(x) = sum_{i<j} a_ij e^(x_i + x_j) + sum_i b_i e^(x_i), x_i = -log pi_i.
* ``allocate``: the program of Eqs. (convex-objective)-(budget): minimise
  Phi subject to sum_i c_i e^(-x_i) <= budget and 0 <= x_i <= -log pi_min,
  solved per group with SLSQP in fp64 (the solver App. C names), then
  refined by Newton steps on the KKT equations of the active set SLSQP
  identifies, and accepted only as a KKT point (residual <= 1e-9); the
  paper's fallback to uniform probabilities of the same expected cost
  otherwise.
* ``kkt_residual``: the Karush-Kuhn-Tucker conditions of that program at a
  given pi (stationarity with the best nonnegative multipliers, primal
  feasibility, complementarity); for this convex program a point with zero
  residual is a global minimiser (Prop. convex).

Pinned in tests/test_oracle_allocation.py by: the disagreement probability
by enumeration of the four outcomes; the expansion of b_i and its
Cauchy-Schwarz bound on explicit pair kernels; the variance upper bound of the
appendix against the exact design covariance (2^G enumeration); the
closed-form allocation when a = 0; the symmetric, slack-budget and
floor-budget special cases; brute force over a grid for G = 2; and the KKT
certificate at the solver's answer.
"""
from __future__ import annotations

import numpy as np

# Per-group status of an allocation (shared meaning with the CUDA path).
ALLOC_OK = 0          # interior budget, solved
ALLOC_SLACK = 1       # budget >= sum c: every pi_i = 1 (x = 0 minimises Phi)
ALLOC_FLOOR = 2       # budget == pi_min sum c: the only feasible point, pi = pi_min
ALLOC_INFEASIBLE = 3  # budget < pi_min sum c: pi = pi_min returned, constraint violated
ALLOC_FALLBACK = 4    # solver failed: uniform pi = budget / sum c
ALLOC_FLAT = 5        # a = 0 and b = 0: Phi is identically 0, uniform pi returned


def disagreement(p_hat):
    """Eq. (disagreement) for every pair of a group: p_hat [..., G] ->
    d [..., G, G] with a zero diagonal."""
    p = np.asarray(p_hat, np.float64)
    pi, pj = p[..., :, None], p[..., None, :]
    d = pi * (1.0 - pj) + (1.0 - pi) * pj
    G = p.shape[-1]
    d[..., np.arange(G), np.arange(G)] = 0.0
    return d


def edge_proxy(p_hat, m_hat=None):
    """Eq. (edge-proxy): a = d (default) or d (m_i + m_j)^2 / 4."""
    d = disagreement(p_hat)
    if m_hat is None:
        return d
    m = np.asarray(m_hat, np.float64)
    return d * (m[..., :, None] + m[..., None, :]) ** 2 / 4.0


def shared_vertex_b(a):
    """Sec. 4.4: b_i = (sum_{j != i} sqrt(a_ij))^2 - sum_{j != i} a_ij.
    a [..., G, G] symmetric, nonnegative; the diagonal is ignored."""
    a = np.array(a, np.float64)
    G = a.shape[-1]
    a[..., np.arange(G), np.arange(G)] = 0.0
    return np.sqrt(a).sum(-1) ** 2 - a.sum(-1)


def design_objective(x, a, b):
    """Eq. (convex-objective) for one group: x [G], a [G, G], b [G]."""
    x = np.asarray(x, np.float64)
    a = np.array(a, np.float64)
    G = x.size
    a[np.arange(G), np.arange(G)] = 0.0
    u = np.exp(x)
    return 0.5 * float(u @ a @ u) + float(np.asarray(b, np.float64) @ u)


def _sum_seq(v):
    """fp64 sum in index order (the CUDA path sums the same way, so budget
    classifications agree bit for bit)."""
    s = 0.0
    for t in np.asarray(v, np.float64).ravel():
        s += float(t)
    return s


def classify(c, budget, pi_min):
    """Which case of the program a group is in: ALLOC_OK (interior budget),
    SLACK, FLOOR or INFEASIBLE, from s = sum c in fp64 (index order)."""
    s = _sum_seq(c)
    budget = float(np.float32(budget))
    lo = float(np.float32(pi_min)) * s
    if budget >= s:
        return ALLOC_SLACK
    if budget == lo:
        return ALLOC_FLOOR
    if budget < lo:
        return ALLOC_INFEASIBLE
    return ALLOC_OK


def _polish(x, a, b, c, budget, X, bound_tol=1e-8):
    """Newton iterations on the KKT equations of the active set at x
    (interior case: the budget constraint is active, because Phi increases in
    every x_i): free coordinates F and the multiplier lam solve
        u_i (sum_j a_ij u_j + b_i) - lam c_i e^(-x_i) = 0   (i in F)
        sum_i c_i e^(-x_i) = budget,
    coordinates at a bound stay there. A free coordinate that leaves the box
    is fixed at the bound, a bound coordinate whose multiplier has the wrong
    sign is freed, and the solve repeats. Returns x, or None."""
    G = x.size
    x = np.clip(x.copy(), 0.0, X)
    at = np.where(x <= bound_tol, -1, np.where(x >= X - bound_tol, 1, 0))
    x[at == -1] = 0.0
    x[at == 1] = X
    for _ in range(2 * G + 2):
        F = np.nonzero(at == 0)[0]
        if F.size == 0:
            return None
        lam = 0.0
        for _ in range(60):
            u = np.exp(x)
            e = c * np.exp(-x)
            S = a @ u + b
            grad = u * S
            if lam == 0.0:
                lam = float(grad[F] @ e[F] / (e[F] @ e[F]))
            R = np.concatenate([grad[F] - lam * e[F], [float(e.sum()) - budget]])
            H = a * np.outer(u, u)
            H[np.arange(G), np.arange(G)] = grad
            Jm = np.zeros((F.size + 1, F.size + 1))
            Jm[:-1, :-1] = H[np.ix_(F, F)] + np.diag(lam * e[F])
            Jm[:-1, -1] = -e[F]
            Jm[-1, :-1] = -e[F]
            step = np.linalg.solve(Jm, -R)
            x[F] += step[:-1]
            lam += step[-1]
            if np.max(np.abs(step[:-1])) <= 1e-15 * max(1.0, X):
                break
        u = np.exp(x)
        r = u * (a @ u + b) - lam * c * np.exp(-x)
        out = (x < 0.0) | (x > X)
        if np.any(out[F]):
            i = F[np.argmax(np.where(out[F], np.abs(np.clip(x[F], 0.0, X) - x[F]), -1.0))]
            at[i] = -1 if x[i] < 0.0 else 1
            x = np.clip(x, 0.0, X)
            continue
        wrong = ((at == -1) & (r < 0)) | ((at == 1) & (r > 0))
        if np.any(wrong):
            at[np.argmax(np.where(wrong, np.abs(r), -1.0))] = 0
            continue
        return x
    return None


def _solve_group(a, b, c, budget, pi_min, x0=None):
    """SLSQP on one group of the interior case, then the KKT polish; returns
    (x, ok) with ok when a KKT point (residual <= 1e-9) was found."""
    from scipy.optimize import minimize

    G = c.size
    X = -np.log(pi_min)
    s = _sum_seq(c)
    if x0 is None:
        x0 = np.full(G, -np.log(0.5 * (budget / s + pi_min)))
    u0 = np.exp(x0)
    scale = 0.5 * float(u0 @ a @ u0) + float(b @ u0)

    def fun(x):
        u = np.exp(x)
        return (0.5 * float(u @ a @ u) + float(b @ u)) / scale

    def jac(x):
        u = np.exp(x)
        return u * (a @ u + b) / scale

    cons = [{"type": "ineq",
             "fun": lambda x: (budget - float(c @ np.exp(-x))) / s,
             "jac": lambda x: c * np.exp(-x) / s}]
    res = minimize(fun, x0, jac=jac, method="SLSQP", bounds=[(0.0, X)] * G,
                   constraints=cons, options={"ftol": 1e-12, "maxiter": 2000})
    x = np.clip(res.x, 0.0, X)
    if not np.all(np.isfinite(x)):
        return x, False
    xp = _polish(x, a, b, c, budget, X)
    pi_min_f = float(np.exp(-X))
    for cand in ([xp] if xp is not None else []) + [x]:
        k = kkt_residual(np.exp(-cand), a, b, c, budget, pi_min_f)
        if k["stat"] <= 1e-9 and k["budget_excess"] <= 1e-12:
            return cand, True
    return x, False


def allocate(a, c, budget, pi_min, b=None, x0=None):
    """The continuation design of Eqs. (convex-objective)-(budget) for a batch
    of groups. a [B, G, G] edge proxies (symmetric, >= 0), c [B, G] predicted
    costs (> 0), budget [B], pi_min scalar in (0, 1]; b [B, G] defaults to
    shared_vertex_b(a). c, budget and pi_min are taken at fp32 precision (the CUDA path's
    argument type) and solved in fp64; a is taken as given (fp64 from
    edge_proxy, or an fp32 array). Returns dict(pi [B, G], x, phi [B],
    status [B] int)."""
    a = np.asarray(a, np.float64)
    c = np.asarray(c, np.float32).astype(np.float64)
    budget = np.asarray(budget, np.float32).astype(np.float64).reshape(-1)
    pi_min = float(np.float32(pi_min))
    Bn, G = c.shape
    if b is None:
        b = shared_vertex_b(a)
    b = np.asarray(b, np.float64)
    X = -np.log(pi_min)
    pi = np.empty((Bn, G))
    phi = np.empty(Bn)
    status = np.empty(Bn, np.int32)
    for g in range(Bn):
        ag = a[g].copy()
        ag[np.arange(G), np.arange(G)] = 0.0
        st = classify(c[g], budget[g], pi_min)
        if st == ALLOC_SLACK:
            x = np.zeros(G)
        elif st in (ALLOC_FLOOR, ALLOC_INFEASIBLE):
            x = np.full(G, X)
        elif not (ag.any() or b[g].any()):
            st = ALLOC_FLAT
            x = np.full(G, -np.log(_sum_seq([budget[g]]) / _sum_seq(c[g])))
        else:
            x, ok = _solve_group(ag, b[g], c[g], budget[g], pi_min,
                                 None if x0 is None else x0[g])
            if not ok:
                st = ALLOC_FALLBACK
                x = np.full(G, -np.log(budget[g] / _sum_seq(c[g])))
        pi[g] = np.exp(-x)
        phi[g] = design_objective(x, ag, b[g])
        status[g] = st
    return {"pi": pi, "x": -np.log(pi), "phi": phi, "status": status}


def kkt_residual(pi, a, b, c, budget, pi_min, bound_tol=1e-7):
    """KKT conditions of the program at pi for one group, in x = -log pi.

    With r_i(lam) = dPhi/dx_i - lam c_i e^(-x_i) (the Lagrangian's gradient
    without the box multipliers), coordinate i contributes |r_i| in the
    interior, max(-r_i, 0) at x_i = 0 (pi_i = 1, multiplier r_i >= 0) and
    max(r_i, 0) at x_i = -log pi_min; lam >= 0 is chosen to minimise the
    largest contribution, and is 0 unless the budget is active. Returns
    dict(stat = max contribution / max |dPhi/dx|, lam, budget_excess =
    (sum c pi - budget) / budget, comp = lam * slack / budget)."""
    pi = np.asarray(pi, np.float64)
    a = np.array(a, np.float64)
    c = np.asarray(c, np.float64)
    b = np.asarray(b, np.float64)
    G = pi.size
    a[np.arange(G), np.arange(G)] = 0.0
    x = -np.log(pi)
    X = -np.log(pi_min)
    u = np.exp(x)
    grad = u * (a @ u + b)
    e = c * np.exp(-x)
    at_lo = x <= bound_tol
    at_hi = x >= X - bound_tol
    inner = ~(at_lo | at_hi)
    spent = float(c @ pi)
    slack = budget - spent
    active = slack <= 1e-6 * budget

    def worst(lam):
        r = grad - lam * e
        v = np.where(inner, np.abs(r), np.where(at_lo, np.maximum(-r, 0.0),
                                                 np.maximum(r, 0.0)))
        return float(v.max()) if G else 0.0

    if not active:
        lam = 0.0
    else:
        # The largest contribution is convex piecewise linear in lam: scan
        # the candidate breakpoints and refine by golden section.
        cand = [0.0] + [float(grad[i] / e[i]) for i in range(G) if e[i] > 0]
        lo = 0.0
        hi = max(cand) * 2.0 + 1e-300
        for _ in range(200):
            m1 = lo + (hi - lo) * 0.381966
            m2 = lo + (hi - lo) * 0.618034
            if worst(m1) <= worst(m2):
                hi = m2
            else:
                lo = m1
        lam = 0.5 * (lo + hi)
        best = min(cand, key=worst)
        if worst(best) < worst(lam):
            lam = best
    scale = max(float(np.abs(grad).max()), 1e-300)
    return {"stat": worst(lam) / scale, "lam": lam,
            "budget_excess": (spent - budget) / budget,
            "comp": lam * max(slack, 0.0) / max(budget, 1e-300)}
