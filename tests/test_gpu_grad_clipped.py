"""GPU parity of pair_grad_clipped (the clipped trajectory-ratio surrogate of
the practical PPO epochs) against the fp64 oracle.

Tolerances. The trajectory ratio rho_i = exp(logp_seq_i - logp_old_i) turns
the absolute error Delta_i of the summed log-probability (a sum of hundreds of
fp32 per-token terms on the GPU) into a relative error exp(Delta_i) - 1 of
rho_i, and so of the unclipped coefficient c_i = A_i rho_i; clipped
coefficients are exact zeros. So:

* clip decisions are exact: old log-probabilities sit at ratios exp(delta)
  whose log-distance to log(1 -+ eps) is checked to exceed 10 |Delta_i|;
* Delta_i itself is held to pair_grad's logp_seq bound (rtol 1e-4);
* c_i is within |c_i| (e_i + 1e-6) of the oracle, e_i = |exp(Delta_i) - 1|
  plus 2^-24 |logp_seq_i| (the coefficient is formed from the fp64 sum, the
  logp_seq output is its fp32 rounding, from which Delta_i is measured);
* J, dH, dW are within pair_grad's 2e-3 (relative Frobenius; J against
  sum_i |L_i|) plus max_i e_i over the rollouts that contribute.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_11368_gb300 import synth
from tests.gpu_util import dev_err_word, head_inputs, rel_fro

pytestmark = pytest.mark.gpu

TOL = 2e-3
EPS = 0.2
DELTAS = [-0.6, -0.1, 0.0, 0.1, 0.6, 0.35, -0.35]


def _binding():
    from paper_2608_11368_gb300 import binding
    return binding


def _case(inp, deltas=DELTAS):
    c = oracle.coeffs(inp["r"], inp["J"], inp["rho"])
    a = c["a"].reshape(-1).astype(np.float32)
    base = oracle.pair_grad_ref(inp, a.astype(np.float64), full=True)
    lo = (base["logp_seq"] - np.resize(np.asarray(deltas), inp["R"])).astype(np.float32)
    return a, lo


def _check(inp, a, lo, image_blocks=None):
    """image_blocks: size the workspace for that many token blocks of the
    image of softmax terms (several backward chunks, later ones recomputing
    their terms); None = pair_grad_workspace_size."""
    B = _binding()
    t = head_inputs(inp, a)
    err = dev_err_word()
    kw = {}
    if image_blocks is not None:
        T, d = t["H"].shape
        V, R = t["W"].shape[0], inp["R"]
        block = (B.pair_grad_workspace_size(128, d, V, R, B.PAIR_BF16)
                 - B.pair_grad_workspace_min_size(128, d, V, R, B.PAIR_BF16))
        kw["ws"] = torch.empty(B.pair_grad_workspace_min_size(T, d, V, R, B.PAIR_BF16)
                               + image_blocks * block, dtype=torch.uint8, device="cuda")
    J, dH, dW, lps, coef = B.pair_grad_clipped(t["H"], t["W"], t["y"], t["mask"],
                                               t["cu_seqlens"], t["a"],
                                               torch.from_numpy(lo).cuda(), clip_eps=EPS,
                                               dev_err=err, **kw)
    assert B.pair_status_sync(err) == 0
    ref = oracle.pair_grad_clipped_ref(inp, a.astype(np.float64), lo.astype(np.float64), EPS)
    lps_n = lps.cpu().numpy().astype(np.float64)
    np.testing.assert_allclose(lps_n, ref["logp_seq"], rtol=1e-4, atol=1e-3)
    active = a != 0
    delta = np.where(active, lps_n - ref["logp_seq"], 0.0)
    e = np.abs(np.expm1(delta)) + np.abs(lps_n) * 2.0 ** -24
    # Every clip decision is far from its boundary relative to Delta_i.
    log_ratio = ref["logp_seq"] - lo.astype(np.float64)
    margin = np.minimum(np.abs(log_ratio - np.log1p(EPS)), np.abs(log_ratio - np.log1p(-EPS)))
    assert (margin[active] > 10 * np.abs(delta[active]) + 1e-6).all()
    cg = coef.cpu().numpy().astype(np.float64)
    assert np.array_equal(cg == 0, ref["coef"] == 0)        # same clip decisions
    assert (np.abs(cg - ref["coef"]) <= np.abs(ref["coef"]) * (e + 1e-6)).all()
    on = ref["coef"] != 0
    e_max = float(e[on].max()) if on.any() else 0.0
    L = np.abs(np.minimum(np.exp(log_ratio) * a, np.clip(np.exp(log_ratio), 1 - EPS, 1 + EPS) * a))
    assert abs(J.item() - ref["J"]) <= TOL * max(ref["J_abs"], 1e-30) + float((L * e).sum())
    assert rel_fro(dH.cpu().numpy(), ref["dH"]) <= TOL + e_max
    assert rel_fro(dW.cpu().numpy(), ref["dW"]) <= TOL + e_max
    seg = oracle.segment_ids(inp["cu_seqlens"])
    off = (inp["mask"] == 0) | (ref["coef"][seg] == 0)
    assert (dH.cpu().numpy()[off] == 0).all()
    return ref


def test_clipped_fp32_reference_workload():
    inp = synth.make_head_workload(synth.WORKLOADS["pr1_ref_fp32"], 3)
    a, lo = _case(inp)
    ref = _check(inp, a, lo)
    assert np.any((a != 0) & (ref["coef"] == 0))   # some rollout clipped


CASES = [
    ("qwen3_1p7b_head", 2048, 151936, 2, 4, 0.05, 1.0),  # image form, full head
    ("qwen3_1p7b_head", 512, 1000, 3, 8, 0.3, 4.0),      # image form, long rollouts
    ("qwen3_1p7b_head", 192, 1000, 3, 5, 0.05, 8.0),     # per-slice fallback (d % 512 != 0)
]


@pytest.mark.parametrize("case", CASES, ids=[f"d{c[1]}_V{c[2]}" for c in CASES])
def test_clipped_bf16_parity(case):
    name, d, V, B_, G, ls, wm = case
    inp = synth.make_head_workload(synth.WORKLOADS[name], 7, B=B_, G=G, d=d, V=V,
                                   len_scale=ls, w_std_mult=wm)
    a, lo = _case(inp)
    _check(inp, a, lo)


@pytest.mark.parametrize("blocks", [1, 2])
def test_clipped_backward_chunks(blocks):
    """Several backward chunks: the first uses the softmax terms the full
    log-sum-exp pass kept, later chunks recompute theirs."""
    inp = synth.make_head_workload(synth.WORKLOADS["qwen3_1p7b_head"], 7, B=3, G=8, d=512,
                                   V=1000, len_scale=0.3, w_std_mult=4.0)
    a, lo = _case(inp)
    _check(inp, a, lo, image_blocks=blocks)


def test_clipped_on_policy_equals_pair_grad():
    """logp_old = this call's logp_seq: ratio 1, clipping inactive; the result
    is pair_grad's gradient (both against the oracle)."""
    inp = synth.make_head_workload(synth.WORKLOADS["qwen3_1p7b_head"], 9, B=2, G=4, d=512,
                                   V=1000, len_scale=0.2)
    a, lo = _case(inp, deltas=[0.0])
    ref = _check(inp, a, lo)
    np.testing.assert_allclose(ref["coef"], a, rtol=1e-5)


@pytest.mark.parametrize("blocks", [None, 1], ids=["image", "image_chunked"])
def test_clipped_fixup_rows(blocks):
    """pair_grad_clipped runs the whole log-sum-exp first and the backward
    after it (in chunks of one token block for blocks = 1, each recomputing
    its softmax terms). Rows whose maximum logit lies more than 2^64 (log2
    units) above the target logit are redone in that first pass with the row
    maximum as reference, and the later chunks must use the settled
    references. Peaky logits (std 24) with every 16th active token's target
    set to the least likely token of its row force such rows; the ratio
    offsets stay far from the clip boundaries."""
    inp = synth.make_head_workload(synth.WORKLOADS["qwen3_1p7b_head"], 7, B=3, G=8, d=512,
                                   V=1000, len_scale=0.2, w_std_mult=24.0)
    a0 = oracle.coeffs(inp["r"], inp["J"], inp["rho"])["a"].reshape(-1)
    assert (a0 != 0).any()
    idx, _, _ = oracle.compact_tokens(inp["cu_seqlens"], inp["mask"], a0)
    pick = idx[::16]
    Hf = synth.as_float(inp["H"][pick], "bf16").astype(np.float64)
    Wf = synth.as_float(inp["W"], "bf16").astype(np.float64)
    Z = Hf @ Wf.T
    inp["y"][pick] = np.argmin(Z, axis=1).astype(np.int32)
    assert ((Z.max(axis=1) - Z.min(axis=1)) * np.log2(np.e) > 80).mean() > 0.9
    a, lo = _case(inp, deltas=[-0.6, 0.0, 0.6])
    _check(inp, a, lo, image_blocks=blocks)
