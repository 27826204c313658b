"""GPU parity of pair_grad (the LM-head realisation of sum_i a_i log pi of
Sec. 4.5) against the fp64 oracle.

Tolerances: J, dH, dW within a relative Frobenius error of 2e-3 (bf16 inputs,
fp32 accumulation); for J the denominator is sum_t |c_t logp_t| because the
coefficients sum to zero within a group. The softmax parts alone (dH minus
its exact one-hot part, dW on non-target rows) are held to 1e-2: their only
approximation is the bf16 rounding of the on-chip logit gradient
(relative 2^-9 per element, about 1.1e-3 RMS).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_11368_gb300 import synth
from tests.gpu_util import dev_err_word, head_inputs, rel_fro

pytestmark = pytest.mark.gpu

TOL = 2e-3
TOL_SOFT = 1e-2


def _binding():
    from paper_2608_11368_gb300 import binding
    return binding


def _coeffs(inp, scale=1.0):
    c = oracle.coeffs(inp["r"], inp["J"], inp["rho"], scale=scale)
    return c["a"].reshape(-1).astype(np.float32)


def _run(inp, a, image_blocks=None, **kw):
    """image_blocks: size the workspace to hold that many token blocks of
    the image of softmax terms and scaled rows (0 = none: the recomputing
    backward); None = the default pair_grad_workspace_size."""
    B = _binding()
    t = head_inputs(inp, a)
    if image_blocks is not None:
        T, d = t["H"].shape
        V, R = t["W"].shape[0], inp["R"]
        dt = B.PAIR_BF16 if t["H"].dtype == torch.bfloat16 else B.PAIR_F32
        # One token block's kept terms and image: the size difference at T = 128.
        block = (B.pair_grad_workspace_size(128, d, V, R, dt)
                 - B.pair_grad_workspace_min_size(128, d, V, R, dt))
        nbytes = B.pair_grad_workspace_min_size(T, d, V, R, dt) + image_blocks * block
        assert nbytes <= B.pair_grad_workspace_size(T, d, V, R, dt)
        kw["ws"] = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    err = dev_err_word()
    Jo, dH, dW, lps = B.pair_grad(t["H"], t["W"], t["y"], t["mask"],
                                  t["cu_seqlens"], t["a"], dev_err=err, **kw)
    st = B.pair_status_sync(err)
    return st, Jo.item(), dH, dW, lps, t


def _full_check(inp, a, image_blocks=None):
    st, J, dH, dW, lps, t = _run(inp, a, image_blocks)
    assert st == 0
    ref = oracle.pair_grad_ref(inp, a.astype(np.float64), full=True)
    dHn, dWn = dH.cpu().numpy(), dW.cpu().numpy()
    assert abs(J - ref["J"]) <= TOL * max(ref["J_abs"], 1e-30)
    assert rel_fro(dHn, ref["dH"]) <= TOL
    assert rel_fro(dWn, ref["dW"]) <= TOL
    np.testing.assert_allclose(lps.cpu().numpy(), ref["logp_seq"], rtol=1e-4,
                               atol=1e-3)
    # Rows outside the objective are exact zeros.
    seg = oracle.segment_ids(inp["cu_seqlens"])
    off = (inp["mask"] == 0) | (a[seg] == 0)
    assert (dHn[off] == 0).all()
    # Softmax parts on their own.
    Wf = synth.as_float(inp["W"], inp["dtype"]).astype(np.float64)
    idx, c, _ = oracle.compact_tokens(inp["cu_seqlens"], inp["mask"], a)
    if idx.size:
        one = c[:, None] * Wf[inp["y"][idx]]
        assert rel_fro(dHn[idx] - one, ref["dH"][idx] - one) <= TOL_SOFT
        untargeted = np.setdiff1d(np.arange(inp["V"]), inp["y"][idx])
        assert rel_fro(dWn[untargeted], ref["dW"][untargeted]) <= TOL_SOFT
    return J, dH, dW


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_grad_fp32_reference_workload(seed):
    inp = synth.make_head_workload(synth.WORKLOADS["pr1_ref_fp32"], seed)
    _full_check(inp, _coeffs(inp))


CASES = [
    # name, d, V, B, G, len_scale, w_mult
    ("qwen3_1p7b_head", 2048, 151936, 2, 4, 0.06, 1.0),  # full head, tail tile
    ("qwen3_1p7b_head", 192, 1000, 3, 5, 0.05, 8.0),     # ragged V, N=192 slice
    ("qwen3_4b_head", 320, 777, 2, 6, 0.03, 8.0),        # two slices (256 + 64)
    ("longctx_skew", 64, 300, 4, 4, 0.02, 1.0),          # minimal d
    # d = 512 A: the image form (default workspace), with one, two, three
    # 512-column units per token pair, ragged vocabulary tails, and fewer
    # units than clusters (every unit split into vocabulary parts).
    ("qwen3_1p7b_head", 512, 1000, 3, 8, 0.3, 4.0),
    ("longctx_skew", 1024, 5003, 2, 8, 0.15, 2.0),
    ("qwen3_4b_head", 1536, 777, 2, 6, 0.08, 8.0),
    # Wider hidden sizes, ragged in both directions: d = 2560 and 3072
    # (the widest the cluster form's scratch covers), and d = 4096, where the
    # image form runs without that scratch (no split last rounds).
    ("qwen3_4b_head", 2560, 4099, 2, 3, 0.05, 3.0),
    ("longctx_skew", 3072, 2011, 2, 4, 0.04, 3.0),
    ("qwen3_4b_head", 4096, 1500, 2, 8, 0.1, 2.0),
]


@pytest.mark.parametrize("case", CASES, ids=[f"d{c[1]}_V{c[2]}" for c in CASES])
def test_grad_bf16_full_parity(case):
    name, d, V, B, G, ls, wm = case
    inp = synth.make_head_workload(synth.WORKLOADS[name], 5, B=B, G=G, d=d, V=V,
                                   len_scale=ls, w_std_mult=wm)
    a = _coeffs(inp)
    if not (a != 0).any():
        a[0] = 0.75
    _full_check(inp, a)


CHUNKED = [
    # name, d, V, B, G, len_scale, w_mult, image token blocks per chunk
    ("qwen3_1p7b_head", 512, 1000, 3, 8, 0.3, 4.0, 0),      # no image: dW recomputes
    ("qwen3_1p7b_head", 512, 1000, 3, 8, 0.3, 4.0, 1),      # 128-token chunks
    ("longctx_skew", 1024, 5003, 2, 8, 0.15, 2.0, 3),       # ragged V, 3-block chunks
    ("qwen3_1p7b_head", 2048, 20000, 2, 8, 0.15, 1.0, 2),   # d = 2048, 2-block chunks
    ("qwen3_4b_head", 1536, 777, 2, 6, 0.08, 8.0, 1),
    # No image: the cluster backward with its narrower column tiles (96 wide
    # for d = 2560, 64 wide for d = 3072).
    ("qwen3_4b_head", 2560, 4099, 2, 3, 0.05, 3.0, 0),
    ("longctx_skew", 3072, 2011, 2, 4, 0.04, 3.0, 0),
    # No image at d = 2048: the 8-CTA cluster form with a ragged vocabulary
    # and tail row blocks split across clusters.
    ("qwen3_1p7b_head", 2048, 20000, 2, 8, 0.15, 1.0, 0),
    ("longctx_skew", 2048, 5003, 4, 8, 0.12, 2.0, 0),
    # d = 4096: beyond the cluster form, so no image means the per-slice
    # backward; one-block chunks of the image form.
    ("qwen3_4b_head", 4096, 1500, 2, 8, 0.1, 2.0, 0),
    ("qwen3_4b_head", 4096, 1500, 2, 8, 0.1, 2.0, 1),
]


@pytest.mark.parametrize("case", CHUNKED,
                         ids=[f"d{c[1]}_V{c[2]}_blocks{c[7]}" for c in CHUNKED])
def test_grad_bf16_backward_chunks(case):
    """Workspaces below pair_grad_workspace_size: the backward runs in token
    chunks (dW stored by the first, added by later ones), or with no image at
    all; each against the oracle."""
    name, d, V, B, G, ls, wm, blocks = case
    inp = synth.make_head_workload(synth.WORKLOADS[name], 5, B=B, G=G, d=d, V=V,
                                   len_scale=ls, w_std_mult=wm)
    a = _coeffs(inp)
    if not (a != 0).any():
        a[0] = 0.75
    idx, _, _ = oracle.compact_tokens(inp["cu_seqlens"], inp["mask"], a)
    if blocks:
        assert idx.size > 128 * blocks   # several chunks
    _full_check(inp, a, image_blocks=blocks)


def test_grad_no_active_rollout():
    inp = synth.make_head_workload(synth.WORKLOADS["qwen3_1p7b_head"], 1, B=2,
                                   G=2, d=512, V=520, len_scale=0.05)
    a = np.zeros(inp["R"], np.float32)
    a[1] = -0.0
    for blocks in (None, 0, 1):
        st, J, dH, dW, lps, _ = _run(inp, a, blocks)
        assert st == 0 and J == 0.0
        assert (dH == 0).all() and (dW == 0).all() and (lps == 0).all()


def test_grad_nan_padding_is_ignored_and_deterministic():
    wl = synth.WORKLOADS["longctx_skew"]
    kw = dict(B=3, G=4, d=256, V=2000, len_scale=0.05, w_std_mult=2.0)
    inp = synth.make_head_workload(wl, 4, **kw)
    inp_nan = synth.make_head_workload(wl, 4, pad_fill="nan", **kw)
    a = _coeffs(inp)
    r0 = _run(inp, a)
    r1 = _run(inp_nan, a)
    r2 = _run(inp, a)
    for x, y in ((r0, r1), (r0, r2)):
        assert x[1] == y[1]
        assert torch.equal(x[2], y[2]) and torch.equal(x[3], y[3])


@pytest.mark.parametrize("blocks,d", [(None, 512), (0, 512), (2, 512), (0, 2048)])
def test_grad_cluster_path_deterministic(blocks, d):
    """Cluster backward with tail row blocks split across clusters (and, for
    blocks = 2, several token chunks; at d = 2048 in the cluster form): reruns
    are bit-identical."""
    inp = synth.make_head_workload(synth.WORKLOADS["qwen3_1p7b_head"], 5, B=3, G=8, d=d,
                                   V=1000, len_scale=0.3, w_std_mult=4.0)
    a = _coeffs(inp)
    r0 = _run(inp, a, blocks)
    r1 = _run(inp, a, blocks)
    assert r0[0] == 0 and r1[0] == 0 and r0[1] == r1[1]
    assert torch.equal(r0[2], r1[2]) and torch.equal(r0[3], r1[3])


def test_grad_target_out_of_range_flagged():
    inp = synth.make_head_workload(synth.WORKLOADS["pr1_ref_fp32"], 0, V=64,
                                   d=32)
    a = _coeffs(inp)
    t = np.nonzero(inp["mask"])[0][3]
    inp["y"][t] = 64
    st = _run(inp, a)[0]
    assert st == 5
    # -100 on padding tokens is fine (the generator's default).
    inp["y"][t] = 5
    assert _run(inp, a)[0] == 0


FULL = ["qwen3_1p7b_head", "qwen3_4b_head", "longctx_skew"]


def _logp_close(got, ref):
    """Per-token log-probabilities: each within the loss tolerance relative
    to its own magnitude."""
    got = np.asarray(got, np.float64)
    bad = np.abs(got - ref) > TOL * np.abs(ref)
    assert not bad.any(), (int(bad.sum()), float(np.abs(got - ref).max()))


@pytest.mark.parametrize("name", FULL)
def test_grad_full_size_against_oracle(name):
    """Full-size workload in the benchmark's launch configuration (default
    workspace) against the fp64 oracle.
    1.7B head (the benchmark workload): the oracle's lse and logp for every
    active token, so J and every per-token log-probability are compared in
    full, every rollout's logp_seq, dH on 1,024 sampled rows plus two whole
    rollouts, and dW on 256 sampled vocabulary rows (half of them targeted).
    4B and long-context heads: per-token logp on 4,096 sampled active tokens
    and on 8 whole active rollouts (with their logp_seq), dH on 1,024 of those
    rows. Identities that hold at any size cover the rest."""
    B = _binding()
    wl = synth.WORKLOADS[name]
    inp = synth.make_head_workload(wl, 0)
    a = _coeffs(inp)
    t = head_inputs(inp, a)
    T, d, V, R = inp["T"], inp["d"], inp["V"], inp["R"]
    ws = torch.empty(B.pair_grad_workspace_size(T, d, V, R, B.PAIR_BF16), dtype=torch.uint8,
                     device="cuda")
    err = dev_err_word()
    Jo, dH, dW, lps = B.pair_grad(t["H"], t["W"], t["y"], t["mask"], t["cu_seqlens"], t["a"],
                                  ws=ws, dev_err=err)
    assert B.pair_status_sync(err) == 0
    lpt = B.pair_grad_token_logp(T, d, V, R, B.PAIR_BF16, ws).cpu().numpy()
    J = Jo.item()
    lps_n = lps.cpu().numpy()
    del ws
    rng = np.random.default_rng(11)
    idx, c, seg = oracle.compact_tokens(inp["cu_seqlens"], inp["mask"], a)
    assert idx.size > 0
    cu = inp["cu_seqlens"]
    y = inp["y"]
    Wf = synth.as_float(inp["W"], inp["dtype"]).astype(np.float64)
    nthr = oracle.n_threads()
    # Tokens outside the objective have logp 0.
    keep = np.zeros(T, bool)
    keep[idx] = True
    assert (lpt[~keep] == 0).all()
    act_r = np.nonzero(a)[0]

    def hrows(tok):
        return synth.as_float(inp["H"][tok], inp["dtype"]).astype(np.float64)

    if name == "qwen3_1p7b_head":
        Ha = hrows(idx)
        lse, zy = oracle.head_lse(Ha, Wf, y[idx], threads=nthr)
        logp = zy - lse
        J_ref = float(np.sum(c * logp))
        assert abs(J - J_ref) <= TOL * float(np.sum(np.abs(c * logp)))
        _logp_close(lpt[idx], logp)
        lps_ref = np.zeros(R, np.float64)
        np.add.at(lps_ref, seg, logp)
        np.testing.assert_allclose(lps_n, lps_ref, rtol=1e-4, atol=1e-3)
        targeted = np.unique(y[idx])
        vrows = np.unique(np.concatenate([
            rng.choice(targeted, 128, replace=False),
            rng.choice(V, 128, replace=False), [V - 1]]))
        dW_ref = oracle.head_dw_rows(Ha, Wf, y[idx], c, lse, vrows)
        assert rel_fro(dW.cpu().numpy()[vrows], dW_ref) <= TOL
        # dH rows: 1,024 sampled active tokens plus the two shortest active
        # rollouts, from the same lse.
        L = np.diff(cu)[act_r]
        two = act_r[np.argsort(L)[:2]]
        pos = np.nonzero(np.isin(seg, two))[0]
        pos = np.unique(np.concatenate([rng.choice(idx.size, 1024, replace=False), pos]))
        dH_ref = oracle.head_dh_rows(Ha[pos], Wf, y[idx[pos]], c[pos], lse[pos])
        assert rel_fro(dH.cpu().numpy()[idx[pos]], dH_ref) <= TOL
    else:
        eight = rng.choice(act_r, 8, replace=False)
        whole = np.nonzero(np.isin(seg, eight))[0]
        pos = np.unique(np.concatenate([rng.choice(idx.size, 4096, replace=False), whole]))
        Hs = hrows(idx[pos])
        lse, zy = oracle.head_lse(Hs, Wf, y[idx[pos]], threads=nthr)
        logp = zy - lse
        _logp_close(lpt[idx[pos]], logp)
        for i in eight:
            sel = seg[pos] == i
            assert sel.sum() == (seg == i).sum()
            ref_i = float(logp[sel].sum())
            assert abs(lps_n[i] - ref_i) <= 1e-4 * abs(ref_i) + 1e-3
        sub = rng.choice(pos.size, 1024, replace=False)
        dH_ref = oracle.head_dh_rows(Hs[sub], Wf, y[idx[pos[sub]]], c[pos[sub]], lse[sub])
        assert rel_fro(dH.cpu().numpy()[idx[pos[sub]]], dH_ref) <= TOL
    # J is the coefficient-weighted sum of the per-rollout log-probabilities.
    assert abs(J - float(np.dot(a.astype(np.float64), lps_n.astype(np.float64)))) \
        <= 1e-4 * float(np.abs(a).dot(np.abs(lps_n)))
    # Inactive rows exactly zero.
    seg_all = oracle.segment_ids(cu)
    off = (inp["mask"] == 0) | (a[seg_all] == 0)
    assert not dH[torch.from_numpy(off).cuda()].any()
    # Identities that hold at any size: sum_v dJ/dW_v = 0 (softmax rows sum
    # to one), and <dW, W> = <dH, H> = sum_tv G_tv z_tv.
    colsum = dW.double().sum(dim=0)
    assert colsum.abs().max().item() <= 1e-3 * dW.double().abs().sum(dim=0).max().item()
    ip_w = (dW.double() * t["W"].double()).sum().item()
    ip_h = (dH.double() * t["H"].double()).sum().item()
    assert abs(ip_w - ip_h) <= 1e-3 * max(abs(ip_h), 1e-30)
    del dH, dW
    torch.cuda.empty_cache()


@pytest.mark.parametrize("name", FULL)
def test_grad_full_head_single_rollout_dw(name):
    """dW rows at the full head size against the oracle, with one active
    rollout (the oracle's dW costs one pass per active token)."""
    wl = synth.WORKLOADS[name]
    inp = synth.make_head_workload(wl, 1, B=2, G=wl.G, len_scale=0.25)
    a = np.zeros(inp["R"], np.float32)
    a[int(np.argmax(np.diff(inp["cu_seqlens"]) > 0))] = 0.625
    st, J, dH, dW, lps, _ = _run(inp, a)
    assert st == 0
    rng = np.random.default_rng(3)
    idx, _, _ = oracle.compact_tokens(inp["cu_seqlens"], inp["mask"], a)
    targeted = np.unique(inp["y"][idx])
    vrows = np.unique(np.concatenate([
        rng.choice(inp["V"], 192, replace=False),
        rng.choice(targeted, min(64, targeted.size), replace=False),
        [inp["V"] - 1]]))
    ref = oracle.pair_grad_ref(inp, a.astype(np.float64), dw_rows=vrows)
    assert rel_fro(dW.cpu().numpy()[vrows], ref["dW_rows"]) <= TOL


@pytest.mark.parametrize("case", [("pr1_ref_fp32", None, None, None, None), 
                                  ("qwen3_1p7b_head", 512, 1000, "default", 4.0),
                                  ("qwen3_1p7b_head", 512, 1000, "min", 4.0),
                                  ("longctx_skew", 256, 3000, "default", 2.0)],
                         ids=["fp32", "bf16_image", "bf16_min_ws", "bf16_d256"])
def test_token_logp_matches_oracle(case):
    """pair_grad_token_logp returns every active token's logp (0 elsewhere),
    for each head path, and sums to logp_seq per rollout."""
    B = _binding()
    name, d, V, ws_kind, wm = case
    kw = {} if d is None else dict(B=3, G=8, d=d, V=V, len_scale=0.2, w_std_mult=wm)
    inp = synth.make_head_workload(synth.WORKLOADS[name], 2, **kw)
    a = _coeffs(inp)
    if not (a != 0).any():
        a[0] = 0.5
    t = head_inputs(inp, a)
    T, dd, VV, R = inp["T"], inp["d"], inp["V"], inp["R"]
    dt = B.PAIR_BF16 if inp["dtype"] == "bf16" else B.PAIR_F32
    size = (B.pair_grad_workspace_min_size if ws_kind == "min"
            else B.pair_grad_workspace_size)(T, dd, VV, R, dt)
    ws = torch.empty(size, dtype=torch.uint8, device="cuda")
    err = dev_err_word()
    _, _, _, lps = B.pair_grad(t["H"], t["W"], t["y"], t["mask"], t["cu_seqlens"], t["a"],
                               ws=ws, dev_err=err)
    assert B.pair_status_sync(err) == 0
    lpt = B.pair_grad_token_logp(T, dd, VV, R, dt, ws).cpu().numpy()
    ref = oracle.pair_grad_ref(inp, a.astype(np.float64), full=True)
    idx = ref["active_tokens"]
    _logp_close(lpt[idx], ref["logp"])
    keep = np.zeros(T, bool)
    keep[idx] = True
    assert (lpt[~keep] == 0).all()
    seg = oracle.segment_ids(inp["cu_seqlens"])
    sums = np.zeros(R, np.float64)
    np.add.at(sums, seg, lpt.astype(np.float64))
    np.testing.assert_allclose(lps.cpu().numpy(), sums, rtol=1e-5, atol=1e-4)


@pytest.mark.parametrize("blocks", [0, None, 1], ids=["onchip", "image", "image_chunked"])
@pytest.mark.parametrize("case", [(512, 1000, 0.3, 3), (1024, 3001, 0.2, 8),
                                  (2048, 2000, 0.15, 5)],
                         ids=["d512_V1000", "d1024_V3001", "d2048_V2000"])
def test_grad_fixup_rows(case, blocks):
    """Both bf16 head forms take each token's softmax terms relative to its
    target logit (the on-chip form with the minimum workspace, the image form
    with the default one or with one token block per chunk); a row whose
    maximum logit exceeds the target's by more than 2^64 (in log2 units) is
    redone relative to its maximum. Peaky logits (std 24) with some targets
    set to the least likely token of their row force such rows, in full and
    in tail row blocks; the result must still match the oracle."""
    d, V, ls, stride = case
    inp = synth.make_head_workload(synth.WORKLOADS["qwen3_1p7b_head"], 7, B=3, G=8, d=d, V=V,
                                   len_scale=ls, w_std_mult=24.0)
    a = _coeffs(inp)
    if not (a != 0).any():
        a[0] = 0.75
    idx, _, _ = oracle.compact_tokens(inp["cu_seqlens"], inp["mask"], a)
    Hf = synth.as_float(inp["H"][idx[::stride]], "bf16").astype(np.float64)
    Wf = synth.as_float(inp["W"], "bf16").astype(np.float64)
    Z = Hf @ Wf.T
    inp["y"][idx[::stride]] = np.argmin(Z, axis=1).astype(np.int32)
    gap = (Z.max(axis=1) - Z.min(axis=1)) * np.log2(np.e)
    assert (gap > 80).mean() > 0.9    # far beyond the 2^64 threshold
    _full_check(inp, a, image_blocks=blocks)
    # Reruns are bit-identical (the fix-up pass included).
    r0 = _run(inp, a, blocks)
    r1 = _run(inp, a, blocks)
    assert r0[0] == 0 and r0[1] == r1[1]
    assert torch.equal(r0[2], r1[2]) and torch.equal(r0[3], r1[3])
