"""Failure path of the pipeline waits, on the GPU, without faulting it: a wait
on an mbarrier nothing arrives on gives up after a short limit through the
kernels' own bounded-wait code, reports PAIR_ERR_DEVICE_TIMEOUT through the
device error word, and leaves the context usable."""
import numpy as np
import pytest
import torch

from paper_2608_11368_gb300 import binding as B, synth

from .gpu_util import dev

CUDA = "cuda"

pytestmark = pytest.mark.gpu


def test_wait_timeout_reports_and_context_survives():
    err = torch.zeros(1, dtype=torch.int32, device=CUDA)
    seen = torch.zeros(2, dtype=torch.int32, device=CUDA)
    B.pair_selftest_wait_timeout(2_000_000, err, seen)  # about 1 ms of SM clocks
    assert B.pair_status_sync(err) == 7  # PAIR_ERR_DEVICE_TIMEOUT
    assert seen.tolist() == [3, 1]       # gave up, raised abort; the peer role saw it
    assert int(err.item()) == 0           # pair_status_sync clears the word
    # The context is still usable: a normal call runs and reports success.
    inp = synth.make_dense_workload(synth.WORKLOADS["coeffs_dense_stress"], 0, B=4, G=16, D=64)
    r, J, rho = dev(inp["r"]), dev(inp["J"]), dev(inp["rho"])
    a, active, edges, contrast = B.pair_coeffs(r, J, rho, dev_err=err)
    assert B.pair_status_sync(err) == 0
    assert np.all(edges.cpu().numpy() >= 0)


def test_wait_timeout_rejects_bad_limits():
    err = torch.zeros(1, dtype=torch.int32, device=CUDA)
    seen = torch.zeros(2, dtype=torch.int32, device=CUDA)
    for bad in (0, -5, 5_000_000_000):
        with pytest.raises(B.PairError):
            B.pair_selftest_wait_timeout(bad, err, seen)
