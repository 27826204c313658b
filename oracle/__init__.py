"""fp64 CPU oracle for the Pair estimator hot path: TEST INFRASTRUCTURE ONLY.

Only tests/, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package. The CUDA
library shares no code with it, and it imports nothing from the library
package except the seeded input generator's bf16 upcast helper (which holds
none of the estimator's arithmetic).

Contents, each following the paper's definitions literally:

* ``coeffs``: per-rollout coefficients of Eq. (pair-advantage), observed and
  contrast edge counts, active mask. Plain C in fp64 (``pair_oracle.c``),
  computed twice (edge-sum form of Algorithm 1 and the direct row form) and
  cross-checked.
* ``estimate_dense``: Eq. (pair-ht) by explicit enumeration of every observed
  edge with the pair kernel h_ij of Eq. (pair-kernel) formed per coordinate.
* ``head_*`` / ``pair_grad_ref``: the policy objective sum_i A_i log pi(o_i|q)
  of Sec. 4.5 realised on an LM output head: logits z = W h, log-softmax,
  target gather, and the exact gradients of the objective w.r.t. the hidden
  states and the head weight, in fp64 numpy (matmul as a library step).

* ``allocation`` (submodule): the contrast graph, the shared-vertex
  surrogate and the convex continuation design of Sec. 4.3-4.4, solved with
  SLSQP in fp64 and certified by its KKT conditions.

Parity status: the coefficient, dense and head functions are pinned by the
paper's identities (Thm. 1, Thm. 2, Prop. bias/covariance, the edge-sum /
coefficient-collapse identity) and by library/brute-force checks in
tests/test_oracle_pins.py.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "liboracle.so")
_SRC = os.path.join(_HERE, "pair_oracle.c")

ORACLE_OK = 0
ORACLE_ERR_NONPOSITIVE_INCLUSION = 1
ORACLE_ERR_FORMS_DISAGREE = 2


class OracleError(RuntimeError):
    pass


def build_oracle(force: bool = False) -> str:
    """Compile the C oracle with gcc (no fast-math, no FMA contraction)."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_SO)
            and os.path.getmtime(_SO) >= os.path.getmtime(_SRC)):
        return _SO
    tmp = _SO + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
           "-shared", "-pthread", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _SO)
    return _SO


_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build_oracle())
        P = ctypes.c_void_p
        lib.oracle_pair_coeffs.argtypes = [
            ctypes.c_int, ctypes.c_int, P, P, P, ctypes.c_double, ctypes.c_int,
            P, P, P, P, P, ctypes.c_int]
        lib.oracle_pair_coeffs.restype = ctypes.c_int
        lib.oracle_pair_estimate_dense.argtypes = [
            ctypes.c_int, ctypes.c_int, ctypes.c_int, P, P, P, P, P,
            ctypes.c_double, P, ctypes.c_int]
        lib.oracle_pair_estimate_dense.restype = ctypes.c_int
        lib.oracle_pair_coeffs_w.argtypes = [
            ctypes.c_int, ctypes.c_int, P, P, P, ctypes.c_double, ctypes.c_int,
            ctypes.c_int, ctypes.c_double, P, P, P, P, P, P, P, ctypes.c_int]
        lib.oracle_pair_coeffs_w.restype = ctypes.c_int
        lib.oracle_pair_coeffs_product.argtypes = [
            ctypes.c_int, ctypes.c_int, P, P, P, ctypes.c_double, ctypes.c_int,
            P, P, P, P, P, P, P, ctypes.c_int]
        lib.oracle_pair_coeffs_product.restype = ctypes.c_int
        _lib = lib
    return _lib


def n_threads() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p)


def coeffs(r, J, rho, scale=1.0, center=False, threads=None, check=True):
    """Eq. (pair-advantage) without the 1/(2M) -> scale * 1/2 factor.

    r [B,G], J [B,G] (0/1), rho [B,G,G] (only i<j read). Returns dict with
    a, a_mag (scale * 1/2 sum |terms|), active, edges, contrast, status.
    """
    r = np.ascontiguousarray(r, dtype=np.float64)
    J = np.ascontiguousarray(J, dtype=np.uint8)
    rho = np.ascontiguousarray(rho, dtype=np.float64)
    B, G = r.shape
    assert J.shape == (B, G) and rho.shape == (B, G, G)
    a = np.zeros((B, G), np.float64)
    a_mag = np.zeros((B, G), np.float64)
    active = np.zeros((B, G), np.uint8)
    edges = np.zeros(B, np.int32)
    contrast = np.zeros(B, np.int32)
    st = _load().oracle_pair_coeffs(
        B, G, _ptr(r), _ptr(J), _ptr(rho), float(scale), int(bool(center)),
        _ptr(a), _ptr(a_mag), _ptr(active), _ptr(edges), _ptr(contrast),
        threads or n_threads())
    if check and st == ORACLE_ERR_FORMS_DISAGREE:
        raise OracleError("edge-sum and row forms disagree")
    return dict(a=a, a_mag=a_mag, active=active, edges=edges,
                contrast=contrast, status=st)


# Weighting variants (App. "Estimated and stabilized propensities"; ablation
# table): edge weight 1/rho, 1, 1/(pi_i pi_j) with pi = diag(rho),
# min(1/rho, w_max), and 1/rho self-normalised by the group's weight sum.
W_HT, W_UNWEIGHTED, W_MARGINAL, W_CLIPPED, W_HAJEK = 0, 1, 2, 3, 4


def _coeffs_out(B, G):
    return dict(a=np.zeros((B, G), np.float64), a_mag=np.zeros((B, G), np.float64),
                active=np.zeros((B, G), np.uint8), edges=np.zeros(B, np.int32),
                contrast=np.zeros(B, np.int32), ess=np.zeros(B, np.float64),
                max_w=np.zeros(B, np.float64))


def coeffs_w(r, J, rho, scale=1.0, center=False, wmode=W_HT, w_max=0.0, threads=None,
             standardize=False):
    """Coefficients under weighting variant `wmode`, with the per-group ESS
    (sum w)^2 / sum w^2 and largest weight over the completed edges.
    rho [B,G,G]: strict upper triangle read for the joint probabilities, its
    diagonal for the marginals (W_MARGINAL)."""
    r = np.ascontiguousarray(r, dtype=np.float64)
    J = np.ascontiguousarray(J, dtype=np.uint8)
    rho = np.ascontiguousarray(rho, dtype=np.float64)
    B, G = r.shape
    o = _coeffs_out(B, G)
    st = _load().oracle_pair_coeffs_w(
        B, G, _ptr(r), _ptr(J), _ptr(rho), float(scale),
        int(bool(center)) | (2 if standardize else 0), int(wmode),
        float(w_max), _ptr(o["a"]), _ptr(o["a_mag"]), _ptr(o["active"]), _ptr(o["edges"]),
        _ptr(o["contrast"]), _ptr(o["ess"]), _ptr(o["max_w"]), threads or n_threads())
    o["status"] = st
    return o


def coeffs_product(r, J, p, scale=1.0, center=False, threads=None, standardize=False):
    """Inverse-probability coefficients of the independent design, rho_ij =
    p_i p_j, from the marginals p [B,G]; plus ESS and largest weight."""
    r = np.ascontiguousarray(r, dtype=np.float64)
    J = np.ascontiguousarray(J, dtype=np.uint8)
    p = np.ascontiguousarray(p, dtype=np.float64)
    B, G = r.shape
    o = _coeffs_out(B, G)
    st = _load().oracle_pair_coeffs_product(
        B, G, _ptr(r), _ptr(J), _ptr(p), float(scale),
        int(bool(center)) | (2 if standardize else 0),
        _ptr(o["a"]), _ptr(o["a_mag"]), _ptr(o["active"]), _ptr(o["edges"]),
        _ptr(o["contrast"]), _ptr(o["ess"]), _ptr(o["max_w"]), threads or n_threads())
    o["status"] = st
    return o


def audit(r, rho, S, Jdraws, draw_weight=None, scale=1.0, center=False, wmode=W_HT,
          w_max=0.0):
    """Frozen-population audit (Sec. 5; App. D metrics) of one group over
    design draws, formed explicitly in fp64: every draw's estimate
    ghat_b = sum_i a_bi s_i from the oracle's coefficients (coefficient form of
    Eq. pair-ht), the target g = scale * sum_{i<j} h_ij from explicit pair
    kernels (Eq. pair-kernel). Returns dict of weighted means (see pair.h)."""
    r = np.asarray(r, np.float64)
    S = np.asarray(S, np.float64)
    Jdraws = np.asarray(Jdraws, np.uint8)
    N, G = Jdraws.shape
    w = np.full(N, 1.0 / N) if draw_weight is None else np.asarray(draw_weight, np.float64)
    rho = np.ones((G, G)) if rho is None else np.asarray(rho, np.float64)
    g = np.zeros(S.shape[1])
    for i in range(G):
        for j in range(i + 1, G):
            g += 0.5 * (r[i] - r[j]) * (S[i] - S[j])
    g *= scale
    o = coeffs_w(np.repeat(r[None], N, 0), Jdraws, np.repeat(rho[None], N, 0), scale=scale,
                 center=center, wmode=wmode, w_max=w_max)
    ghat = o["a"] @ S
    W = w.sum()
    err2 = ((ghat - g) ** 2).sum(axis=1)
    nrm = np.sqrt((ghat ** 2).sum(axis=1)) * np.sqrt((g ** 2).sum())
    cos = np.where(nrm > 0, (ghat @ g) / np.where(nrm > 0, nrm, 1.0), 0.0)
    K = Jdraws.astype(np.int64).sum(axis=1)
    bias = (w @ ghat) / W - g
    return dict(bias_norm=float(np.sqrt((bias ** 2).sum())), mse=float(w @ err2 / W),
                cos=float(w @ cos / W), vertices=float(w @ K / W),
                edges=float(w @ (K * (K - 1) // 2) / W), ess=float(w @ o["ess"] / W),
                target_sq=float((g ** 2).sum()), weight=float(W), bias=bias, status=o["status"])


def ppo_surrogate(a, logp_seq, logp_old, eps):
    """Clipped trajectory-ratio surrogate of the practical PPO epochs (Sec. 4.5
    and App. "Practical departures"): with detached coefficients A_i and
    trajectory ratios rho_i = exp(logp_seq_i - logp_old_i), rollout i
    contributes L_i = min(rho_i A_i, clip(rho_i, 1 - eps, 1 + eps) A_i). Its
    gradient is c_i * d logp_seq_i with c_i = A_i rho_i where the unclipped term
    is the minimum (A_i > 0: rho_i <= 1 + eps; A_i < 0: rho_i >= 1 - eps) and 0
    where the clip binds. Returns (c, L) in fp64; rollouts with A_i = 0 give 0."""
    a = np.asarray(a, np.float64)
    ratio = np.exp(np.asarray(logp_seq, np.float64) - np.asarray(logp_old, np.float64))
    clipped = np.clip(ratio, 1.0 - eps, 1.0 + eps)
    L = np.where(a != 0, np.minimum(ratio * a, clipped * a), 0.0)
    unclipped = np.where(a > 0, ratio <= 1.0 + eps, ratio >= 1.0 - eps)
    c = np.where((a != 0) & unclipped, a * ratio, 0.0)
    return c, L


def pair_grad_clipped_ref(inp, a, logp_old, eps):
    """Reference outputs of pair_grad_clipped: the forward of pair_grad gives
    every rollout's summed log-probability, the surrogate gives (c, L), and the
    gradients are those of sum_i c_i logp_seq_i with c detached."""
    base = pair_grad_ref(inp, a, full=True)
    c, L = ppo_surrogate(a, base["logp_seq"], logp_old, eps)
    out = pair_grad_ref(inp, c, full=True)
    out["J"] = float(L.sum())
    out["J_abs"] = float(np.abs(L).sum())
    out["logp_seq"] = base["logp_seq"]
    out["coef"] = c
    return out


def estimate_dense(r, J, rho, S, scale=1.0, threads=None):
    """Eq. (pair-ht) times M*scale: scale * sum_{i<j} J_iJ_j h_ij/rho_ij with
    h_ij = 1/2 (r_i - r_j)(s_i - s_j) formed explicitly. S [B,G,D]."""
    r = np.ascontiguousarray(r, dtype=np.float64)
    J = np.ascontiguousarray(J, dtype=np.uint8)
    rho = np.ascontiguousarray(rho, dtype=np.float64)
    B, G = r.shape
    D = S.shape[2]
    g = np.zeros((B, D), np.float64)
    if S.dtype == np.float32:
        S32 = np.ascontiguousarray(S)
        p32, p64 = _ptr(S32), None
    else:
        S64 = np.ascontiguousarray(S, dtype=np.float64)
        p32, p64 = None, _ptr(S64)
    st = _load().oracle_pair_estimate_dense(
        B, G, D, _ptr(r), _ptr(J), _ptr(rho), p32, p64, float(scale),
        _ptr(g), threads or n_threads())
    return g, st


# ----------------------------------------------------------------------------
# LM-head objective: sum_i A_i log pi(o_i | q)   (Sec. 4.5)
# log pi(o_i | q) = sum over the response tokens t of rollout i of
# log softmax(W h_t)[y_t]  (the sequence-level score of Sec. 3.1 is its
# gradient). Ascent convention: the returned gradients are of the objective.
# ----------------------------------------------------------------------------

def segment_ids(cu_seqlens):
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    return np.repeat(np.arange(cu.size - 1), np.diff(cu))


def compact_tokens(cu_seqlens, mask, a):
    """Tokens that enter the objective: mask_t = 1 inside a rollout whose
    coefficient is nonzero. Returns (token index, c_t = a_seg(t), seg(t))."""
    seg = segment_ids(cu_seqlens)
    a = np.asarray(a)
    keep = (np.asarray(mask) == 1) & (a[seg] != 0)
    idx = np.nonzero(keep)[0]
    return idx, np.asarray(a, np.float64)[seg[idx]], seg[idx]


def head_logits(Hrows, W):
    """z_tv = <h_t, W_v> in fp64."""
    return np.asarray(Hrows, np.float64) @ np.asarray(W, np.float64).T


def head_lse(Hrows, W, y, chunk=256, threads=1):
    """Per token: log-sum-exp over the vocabulary (max-shifted) and the
    target logit. Returns (lse, z_target), fp64.

    threads > 1 splits each chunk's rows over that many threads for the
    per-row steps (max, shift, exp, sum, log); every row's arithmetic and its
    order are the same as with one thread. The logit matmul stays one library
    call per chunk."""
    W64 = np.asarray(W, np.float64)
    n = Hrows.shape[0]
    lse = np.empty(n, np.float64)
    zy = np.empty(n, np.float64)

    def rows(Z, s, a, b):
        m = Z[a:b].max(axis=1)
        lse[s + a:s + b] = m + np.log(np.exp(Z[a:b] - m[:, None]).sum(axis=1))
        zy[s + a:s + b] = Z[np.arange(a, b), y[s + a:s + b]]

    pool = None
    if threads > 1:
        import concurrent.futures as cf
        pool = cf.ThreadPoolExecutor(threads)
    try:
        for s in range(0, n, chunk):
            e = min(n, s + chunk)
            Z = np.asarray(Hrows[s:e], np.float64) @ W64.T
            if pool is None:
                rows(Z, s, 0, e - s)
            else:
                step = -(-(e - s) // threads)
                futs = [pool.submit(rows, Z, s, a, min(e - s, a + step))
                        for a in range(0, e - s, step)]
                for f in futs:
                    f.result()
    finally:
        if pool is not None:
            pool.shutdown()
    return lse, zy


def head_dh_rows(Hrows, W, y, c, lse, chunk=256):
    """dJ/dh_t = c_t (W_{y_t} - sum_v softmax(z_t)_v W_v) for the given rows."""
    W64 = np.asarray(W, np.float64)
    n = Hrows.shape[0]
    out = np.empty((n, W64.shape[1]), np.float64)
    c = np.asarray(c, np.float64)
    for s in range(0, n, chunk):
        e = min(n, s + chunk)
        Z = np.asarray(Hrows[s:e], np.float64) @ W64.T
        P = np.exp(Z - lse[s:e, None])
        out[s:e] = c[s:e, None] * (W64[y[s:e]] - P @ W64)
    return out


def head_dw_rows(Hact, W, yact, cact, lse_act, vrows, chunk=4096):
    """dJ/dW_v = sum_t c_t (1[y_t = v] - softmax(z_t)_v) h_t for v in vrows,
    summed over every active token t (rows Hact with targets yact)."""
    H64 = np.asarray(Hact, np.float64)
    W64 = np.asarray(W, np.float64)
    vrows = np.asarray(vrows, np.int64)
    out = np.empty((vrows.size, H64.shape[1]), np.float64)
    for s in range(0, vrows.size, chunk):
        vs = vrows[s:s + chunk]
        Z = H64 @ W64[vs].T
        P = np.exp(Z - lse_act[:, None])
        onehot = (np.asarray(yact)[:, None] == vs[None, :]).astype(np.float64)
        Gt = np.asarray(cact, np.float64)[:, None] * (onehot - P)
        out[s:s + chunk] = Gt.T @ H64
    return out


def pair_grad_ref(inp, a, dh_rows=None, dw_rows=None, lse_tokens=None,
                  full=False, logp_rollouts=None):
    """Reference outputs of pair_grad for inputs from synth.make_head_workload.

    a: per-rollout coefficients [R]. With full=True every output is computed
    (J, logp_seq, dH over all T rows, dW over all V rows). Otherwise only the
    requested pieces: dh_rows / dw_rows select dH / dW rows, lse_tokens
    selects tokens whose lse / logp are returned, logp_rollouts selects
    rollouts whose summed logp is returned. Only the hidden rows that a
    requested output depends on are read.
    """
    from paper_2608_11368_gb300.synth import as_float  # exact upcast only
    dtype = inp["dtype"]

    def hrows(t):
        return as_float(inp["H"][np.asarray(t, np.int64)], dtype)

    Wf = as_float(inp["W"], dtype).astype(np.float64)
    y = inp["y"]
    idx, c, seg = compact_tokens(inp["cu_seqlens"], inp["mask"], a)
    out = {"active_tokens": idx, "c": c}
    R = inp["R"]
    if full:
        Ha = hrows(idx)
        lse, zy = head_lse(Ha, Wf, y[idx])
        logp = zy - lse
        out["lse"], out["logp"] = lse, logp
        out["J"] = float(np.sum(c * logp))
        out["J_abs"] = float(np.sum(np.abs(c * logp)))
        lps = np.zeros(R, np.float64)
        np.add.at(lps, seg, logp)
        out["logp_seq"] = lps
        dH = np.zeros((inp["T"], inp["d"]), np.float64)
        if idx.size:
            dH[idx] = head_dh_rows(Ha, Wf, y[idx], c, lse)
        out["dH"] = dH
        out["dW"] = head_dw_rows(Ha, Wf, y[idx], c, lse, np.arange(inp["V"]))
        return out
    if lse_tokens is not None:
        t = np.asarray(lse_tokens, np.int64)
        lse_t, zy_t = head_lse(hrows(t), Wf, y[t])
        out["lse_sel"], out["logp_sel"] = lse_t, zy_t - lse_t
    if logp_rollouts is not None:
        cu = inp["cu_seqlens"]
        vals = []
        for i in logp_rollouts:
            t = np.arange(cu[i], cu[i + 1])
            t = t[inp["mask"][t] == 1]
            if a[i] == 0 or t.size == 0:
                vals.append(0.0)
                continue
            lse_t, zy_t = head_lse(hrows(t), Wf, y[t])
            vals.append(float(np.sum(zy_t - lse_t)))
        out["logp_seq_sel"] = np.array(vals)
    if dh_rows is not None:
        t = np.asarray(dh_rows, np.int64)
        seg_all = segment_ids(inp["cu_seqlens"])
        ct = np.asarray(a, np.float64)[seg_all[t]] * (inp["mask"][t] == 1)
        rows = np.zeros((t.size, inp["d"]), np.float64)
        nz = ct != 0
        if nz.any():
            Ht = hrows(t[nz])
            lse_t, _ = head_lse(Ht, Wf, y[t[nz]])
            rows[nz] = head_dh_rows(Ht, Wf, y[t[nz]], ct[nz], lse_t)
        out["dH_rows"] = rows
    if dw_rows is not None:
        Ha = hrows(idx)
        lse_a, _ = head_lse(Ha, Wf, y[idx])
        out["dW_rows"] = head_dw_rows(Ha, Wf, y[idx], c, lse_a, dw_rows)
    return out
