"""pair_grad_noalloc: the workspace-free variant of pair_grad for callers
that cannot allocate device memory (a plug-in inside a host program that owns
all device allocations, or code that must avoid cudaMalloc's device-wide
synchronisation). It must give pair_grad's results, call after call, on the
library's fixed device array. Collected last so that a stop-at-first-failure
run has already run every other test."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_11368_gb300 import synth
from tests.gpu_util import dev_err_word, head_inputs, rel_fro

pytestmark = pytest.mark.gpu

TOL = 2e-3


def _case(seed, **kw):
    inp = synth.make_head_workload(synth.WORKLOADS["qwen3_1p7b_head"], seed, **kw)
    c = oracle.coeffs(inp["r"], inp["J"], inp["rho"])
    a = c["a"].reshape(-1).astype(np.float32)
    if not (a != 0).any():
        a[0] = 0.5
    return inp, a


def test_noalloc_matches_pair_grad_twice():
    from paper_2608_11368_gb300 import binding as B
    inp, a = _case(3, B=2, G=8, d=512, V=32000, len_scale=0.2, w_std_mult=4.0)
    t = head_inputs(inp, a)
    need = B.pair_grad_workspace_min_size(inp["T"], inp["d"], inp["V"], inp["R"],
                                          B.PAIR_BF16)
    assert 0 < need <= B.NOALLOC_MAX_WORKSPACE
    err = dev_err_word()
    # pair_grad with the default workspace (dH and dW from the kept image of
    # softmax terms) agrees to rounding; with the minimum workspace it runs the same
    # kernels as the fixed array and agrees bit for bit.
    Jr, dHr, dWr, lpr = B.pair_grad(t["H"], t["W"], t["y"], t["mask"],
                                    t["cu_seqlens"], t["a"], dev_err=err)
    assert B.pair_status_sync(err) == 0
    ws_min = torch.empty(need, dtype=torch.uint8, device="cuda")
    Jm, dHm, dWm, lpm = B.pair_grad(t["H"], t["W"], t["y"], t["mask"],
                                    t["cu_seqlens"], t["a"], ws=ws_min, dev_err=err)
    assert B.pair_status_sync(err) == 0
    for _ in range(2):
        dH = torch.full_like(dHr, float("nan"))
        dW = torch.full_like(dWr, float("nan"))
        Jo = torch.empty_like(Jr)
        lp = torch.empty_like(lpr)
        B.pair_grad_noalloc(t["H"], t["W"], t["y"], t["mask"], t["cu_seqlens"],
                            t["a"], dH=dH, dW=dW, Jobj=Jo, logp_seq=lp,
                            dev_err=err)
        assert B.pair_status_sync(err) == 0
        assert B.pair_last_launch_count() > 0
        assert abs(Jo.item() - Jr.item()) <= TOL * max(abs(Jr.item()), 1e-30)
        assert rel_fro(dH.cpu().numpy(), dHr.cpu().numpy()) <= TOL
        assert rel_fro(dW.cpu().numpy(), dWr.cpu().numpy()) <= TOL
        assert rel_fro(lp.cpu().numpy(), lpr.cpu().numpy()) <= TOL
        assert Jo.item() == Jm.item()
        assert torch.equal(dH, dHm) and torch.equal(dW, dWm) and torch.equal(lp, lpm)


def test_noalloc_rejects_oversized_problem():
    from paper_2608_11368_gb300 import binding as B
    inp, a = _case(1, B=8, G=8, d=2048, V=4096, len_scale=1.0)
    need = B.pair_grad_workspace_min_size(inp["T"], inp["d"], inp["V"], inp["R"],
                                          B.PAIR_BF16)
    assert need > B.NOALLOC_MAX_WORKSPACE
    t = head_inputs(inp, a)
    with pytest.raises(B.PairError) as e:
        B.pair_grad_noalloc(t["H"], t["W"], t["y"], t["mask"], t["cu_seqlens"],
                            t["a"])
    assert e.value.status == 3


def _run_noalloc(B, t, like):
    """pair_grad_noalloc into NaN-filled caller outputs shaped like `like`."""
    dHr, dWr, Jr, lpr = like
    dH = torch.full_like(dHr, float("nan"))
    dW = torch.full_like(dWr, float("nan"))
    Jo = torch.empty_like(Jr)
    lp = torch.empty_like(lpr)
    err = dev_err_word()
    B.pair_grad_noalloc(t["H"], t["W"], t["y"], t["mask"], t["cu_seqlens"], t["a"],
                        dH=dH, dW=dW, Jobj=Jo, logp_seq=lp, dev_err=err)
    assert B.pair_status_sync(err) == 0
    return Jo, dH, dW, lp


def _pair_grad_min_ws(B, t, inp, dt):
    need = B.pair_grad_workspace_min_size(inp["T"], inp["d"], inp["V"], inp["R"], dt)
    assert 0 < need <= B.NOALLOC_MAX_WORKSPACE
    ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    err = dev_err_word()
    out = B.pair_grad(t["H"], t["W"], t["y"], t["mask"], t["cu_seqlens"], t["a"], ws=ws,
                      dev_err=err)
    assert B.pair_status_sync(err) == 0
    return out


def test_noalloc_fp32_head_matches_pair_grad_bitwise():
    """The fp32 CUDA-core head (the 4 x 8, d = 256, V = 4096 workload) on the
    fixed array gives pair_grad's minimum-workspace outputs bit for bit, and
    the oracle's within the tolerance."""
    from paper_2608_11368_gb300 import binding as B
    inp = synth.make_head_workload(synth.WORKLOADS["pr1_ref_fp32"], 0)
    c = oracle.coeffs(inp["r"], inp["J"], inp["rho"])
    a = c["a"].reshape(-1).astype(np.float32)
    t = head_inputs(inp, a)
    Jm, dHm, dWm, lpm = _pair_grad_min_ws(B, t, inp, B.PAIR_F32)
    for _ in range(2):
        Jo, dH, dW, lp = _run_noalloc(B, t, (dHm, dWm, Jm, lpm))
        assert Jo.item() == Jm.item()
        assert torch.equal(dH, dHm) and torch.equal(dW, dWm) and torch.equal(lp, lpm)
    ref = oracle.pair_grad_ref(inp, a.astype(np.float64), full=True)
    assert abs(Jo.item() - ref["J"]) <= TOL * max(ref["J_abs"], 1e-30)
    assert rel_fro(dH.cpu().numpy(), ref["dH"]) <= TOL
    assert rel_fro(dW.cpu().numpy(), ref["dW"]) <= TOL


def test_noalloc_smaller_call_after_larger_is_unaffected():
    """A call with fewer tokens and rollouts after a larger one: whatever the
    larger call left in the shared array must not reach the smaller call's
    results (compared bit for bit with pair_grad on a fresh minimum
    workspace)."""
    from paper_2608_11368_gb300 import binding as B
    big, a_big = _case(5, B=2, G=8, d=512, V=8192, len_scale=0.25, w_std_mult=4.0)
    small, a_small = _case(6, B=1, G=4, d=512, V=8192, len_scale=0.05, w_std_mult=4.0)
    assert small["T"] < big["T"] and small["R"] < big["R"]
    tb = head_inputs(big, a_big)
    ts = head_inputs(small, a_small)
    ref_b = _pair_grad_min_ws(B, tb, big, B.PAIR_BF16)
    ref_s = _pair_grad_min_ws(B, ts, small, B.PAIR_BF16)
    Jb, dHb, dWb, lpb = _run_noalloc(B, tb, (ref_b[1], ref_b[2], ref_b[0], ref_b[3]))
    assert torch.equal(dHb, ref_b[1]) and torch.equal(dWb, ref_b[2])
    Js, dHs, dWs, lps = _run_noalloc(B, ts, (ref_s[1], ref_s[2], ref_s[0], ref_s[3]))
    assert Js.item() == ref_s[0].item()
    assert torch.equal(dHs, ref_s[1]) and torch.equal(dWs, ref_s[2])
    assert torch.equal(lps, ref_s[3])
    ref = oracle.pair_grad_ref(small, a_small.astype(np.float64), full=True)
    assert rel_fro(dHs.cpu().numpy(), ref["dH"]) <= TOL
    assert rel_fro(dWs.cpu().numpy(), ref["dW"]) <= TOL


def test_noalloc_rejects_wrong_shaped_output_before_launch():
    """The binding checks every caller-passed output (shape, dtype, device)
    before the C call, so a wrong-shaped dH never reaches a kernel."""
    from paper_2608_11368_gb300 import binding as B
    inp, a = _case(2, B=1, G=4, d=512, V=1024, len_scale=0.05)
    t = head_inputs(inp, a)
    bad = torch.empty((inp["T"] - 1, inp["d"]), dtype=torch.float32, device="cuda")
    with pytest.raises(ValueError):
        B.pair_grad_noalloc(t["H"], t["W"], t["y"], t["mask"], t["cu_seqlens"], t["a"], dH=bad)
    with pytest.raises(TypeError):
        B.pair_grad_noalloc(t["H"], t["W"], t["y"], t["mask"], t["cu_seqlens"], t["a"],
                            Jobj=torch.empty(1, dtype=torch.float32, device="cuda"))
