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
    # pair_grad with the default workspace (dW from the kept logit-gradient
    # tiles) agrees to rounding; with the minimum workspace it runs the same
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
