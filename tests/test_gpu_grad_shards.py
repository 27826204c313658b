"""The data-parallel decomposition of pair_grad on the GPU path. Whole prompt
groups are split over shards, as ranks would hold them. Each shard runs as its
own pair_grad call on one GPU, one after another, and the dW and J
contributions are summed on the host (the all-reduce a data-parallel trainer
would do). The sum must match the single call over all groups and the fp64
oracle within pair_grad's tolerance. Each shard's dH rows must match the
single call's rows for the same tokens (dH needs no exchange)."""
import numpy as np
import pytest

import oracle
from paper_2608_11368_gb300 import synth
from tests.gpu_util import dev_err_word, head_inputs, rel_fro
from tests.test_multirank import _shard

pytestmark = pytest.mark.gpu

TOL = 2e-3


def _grad(inp, a):
    from paper_2608_11368_gb300 import binding as B
    t = head_inputs(inp, a)
    err = dev_err_word()
    Jo, dH, dW, _ = B.pair_grad(t["H"], t["W"], t["y"], t["mask"], t["cu_seqlens"], t["a"],
                                dev_err=err)
    assert B.pair_status_sync(err) == 0
    return (Jo.item(), dH.cpu().numpy().astype(np.float64),
            dW.cpu().numpy().astype(np.float64))


@pytest.mark.parametrize("nshards", [2, 3])
def test_group_shards_sum_to_the_single_call(nshards):
    inp = synth.make_head_workload(synth.WORKLOADS["qwen3_1p7b_head"], 11, B=6, G=4, d=512,
                                   V=3001, len_scale=0.08)
    c = oracle.coeffs(inp["r"], inp["J"], inp["rho"])
    a = c["a"].reshape(-1).astype(np.float32)
    J1, dH1, dW1 = _grad(inp, a)
    ref = oracle.pair_grad_ref(inp, a.astype(np.float64), full=True)
    cu, G = inp["cu_seqlens"], inp["G"]
    Js, dWs = 0.0, np.zeros_like(dW1)
    for k in range(nshards):
        groups = [b for b in range(inp["B"]) if b % nshards == k]
        rolls = [b * G + i for b in groups for i in range(G)]
        Jk, dHk, dWk = _grad(_shard(inp, groups), a[rolls])
        Js += Jk
        dWs += dWk
        tok = np.concatenate([np.arange(cu[r], cu[r + 1]) for r in rolls])
        assert rel_fro(dHk, dH1[tok]) <= TOL
        assert rel_fro(dHk, ref["dH"][tok]) <= TOL
    assert rel_fro(dWs, dW1) <= TOL
    assert rel_fro(dWs, ref["dW"]) <= TOL
    assert abs(Js - J1) <= TOL * max(ref["J_abs"], 1e-30)
    assert abs(Js - ref["J"]) <= TOL * max(ref["J_abs"], 1e-30)
