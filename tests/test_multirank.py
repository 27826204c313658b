"""The N > 1 path on CPU: two gloo ranks, each owning a disjoint set of whole
prompt groups (groups are independent: no data-path exchange). Each rank
computes its groups' coefficients and head gradients with the fp64 oracle;
the dW contributions are summed with an all-reduce, as a data-parallel
trainer would, and must equal the single-process result over all groups
(the library itself is single-GPU; this exchange belongs to a trainer)."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2608_11368_gb300 import synth


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _inputs():
    wl = synth.WORKLOADS["pr1_ref_fp32"]
    return synth.make_head_workload(wl, 3, B=4, G=4, d=16, V=40, len_scale=0.15)


def _shard(inp, groups):
    """Sub-batch holding only the given groups (rollouts b*G .. b*G+G-1)."""
    G = inp["G"]
    cu = inp["cu_seqlens"]
    rolls = [b * G + i for b in groups for i in range(G)]
    spans = [(cu[r], cu[r + 1]) for r in rolls]
    tok = np.concatenate([np.arange(a, b) for a, b in spans])
    lens = np.array([b - a for a, b in spans])
    out = dict(inp)
    out.update(B=len(groups), R=len(rolls), T=int(tok.size), H=inp["H"][tok],
               y=inp["y"][tok], mask=inp["mask"][tok],
               cu_seqlens=np.concatenate([[0], np.cumsum(lens)]).astype(np.int32),
               r=inp["r"][groups], J=inp["J"][groups], rho=inp["rho"][groups])
    return out


def _worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    inp = _inputs()
    mine = [b for b in range(inp["B"]) if b % world == rank]
    sh = _shard(inp, mine)
    c = oracle.coeffs(sh["r"], sh["J"], sh["rho"])
    ref = oracle.pair_grad_ref(sh, c["a"].reshape(-1), full=True)
    dW = torch.from_numpy(ref["dW"].copy())
    Jt = torch.tensor([ref["J"]], dtype=torch.float64)
    dist.all_reduce(dW)
    dist.all_reduce(Jt)
    t = torch.tensor([float(rank + 1)], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    if rank == 0:
        q.put((dW.numpy(), float(Jt.item()), float(t.item())))
    dist.destroy_process_group()


def test_two_rank_group_sharding_matches_single_process():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    dW, J, tmax = q.get(timeout=120)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    inp = _inputs()
    c = oracle.coeffs(inp["r"], inp["J"], inp["rho"])
    ref = oracle.pair_grad_ref(inp, c["a"].reshape(-1), full=True)
    np.testing.assert_allclose(dW, ref["dW"], rtol=1e-12, atol=1e-14)
    assert abs(J - ref["J"]) <= 1e-12 * max(1.0, ref["J_abs"])
    assert tmax == 2.0
