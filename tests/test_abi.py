"""The C-ABI library builds for sm_103a, loads, exports every function that
include/pair.h declares, and validates arguments on the host (no GPU needed:
invalid arguments are rejected before any device call)."""
import ctypes
import os
import subprocess
import sys

import pytest

from paper_2608_11368_gb300 import build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    build.build()
    from paper_2608_11368_gb300 import binding
    return binding


def test_exports_every_header_function(L):
    names = L.header_functions()
    assert {"pair_coeffs", "pair_grad", "pair_estimate_dense",
            "pair_grad_workspace_size", "pair_grad_workspace_min_size", "pair_status_sync",
            "pair_status_string", "pair_last_launch_count"} <= set(names)
    lib = L.lib()
    for n in names:
        assert hasattr(lib, n), n


def test_status_strings(L):
    for st in range(8):
        s = L.pair_status_string(st)
        assert s and s != "unknown status"
    assert L.pair_status_string(99) == "unknown status"


def test_workspace_size_rules(L):
    ws = L.pair_grad_workspace_size
    assert ws(1000, 2048, 151936, 64, L.PAIR_BF16) > 1000 * 2048 * 2
    wmin = L.pair_grad_workspace_min_size
    # The fp32 path stages 4-byte hidden rows; bf16 stages 2-byte rows plus a
    # fixed ring of logit-gradient tiles, the clusters' tail scratch
    # (24 x 2 x 128 x d fp32) and the per-token arrays of the log-sum-exp
    # passes (reference, row maximum and softmax sum, 3 x 4 bytes per padded
    # token; one 8 x 256 fp32 partial block per 128-token slot, ceil(T/128) +
    # 48 slots), so fp32 needs more once T is large.
    tpad = (100000 + 127) // 128 * 128
    fused = 3 * 4 * tpad + (tpad // 128 + 48) * 8 * 256 * 4 + (1 << 20)
    fixed = (12 << 20) + 24 * 2 * 128 * 2048 * 4 + (1 << 20) + fused
    assert (wmin(100000, 2048, 151936, 64, L.PAIR_F32)
            - wmin(100000, 2048, 151936, 64, L.PAIR_BF16) > 100000 * 2048 * 2 - fixed)
    # For d a multiple of 512, bf16 also keeps the bf16 image of softmax
    # terms and the scaled hidden rows of min(ceil(T/128), max(32, 24 GiB //
    # per_block)) token blocks, per_block = ceil(V/128) tiles of 32 KB plus
    # 128 rows of d bf16; other widths and fp32 keep none.
    for T, d, V in [(100000, 2048, 151936), (1000, 512, 1000), (10 ** 6, 1024, 10 ** 6),
                    (5000, 1536, 300), (70000, 2560, 151936), (3000, 3072, 4099)]:
        per_block = (V + 127) // 128 * 32768 + 128 * d * 2
        blocks = min((T + 127) // 128, max(32, (24 << 30) // per_block))
        assert ws(T, d, V, 64, L.PAIR_BF16) - wmin(T, d, V, 64, L.PAIR_BF16) == blocks * per_block
    for d, dt in [(640, L.PAIR_BF16), (256, L.PAIR_BF16), (2048, L.PAIR_F32)]:
        assert ws(5000, d, 1000, 8, dt) == wmin(5000, d, 1000, 8, dt)
    assert ws(1000, 96, 100, 4, L.PAIR_BF16) == 0      # bf16 needs d % 64 == 0
    assert ws(1000, 96, 100, 4, L.PAIR_F32) > 0
    assert ws(1000, 20, 100, 4, L.PAIR_F32) == 0       # d % 16 != 0
    assert ws(0, 64, 100, 4, L.PAIR_F32) == 0
    assert ws(10, 64, 100, 0, L.PAIR_F32) == 0
    assert ws(10, 64, 0, 1, L.PAIR_F32) == 0
    assert wmin(1000, 96, 100, 4, L.PAIR_BF16) == 0


def test_host_validation_without_device():
    """Host-side argument checks, run in a child process with no visible
    device: the placeholder pointers below must never reach a kernel, even if
    a check were to let a call through."""
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    code = ("import sys; sys.path.insert(0, %r); import tests.test_abi as t; "
            "from paper_2608_11368_gb300 import binding; t._host_validation_checks(binding)"
            % ROOT)
    res = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True,
                         text=True, timeout=300)
    assert res.returncode == 0, res.stdout[-2000:] + res.stderr[-2000:]


def _host_validation_checks(L):
    lib = L.lib()
    P = ctypes.c_void_p
    one = P(16)  # never dereferenced: validation fails first
    # G < 2, G > PAIR_MAX_G, B < 1, null pointers, bad flags.
    for B, G in [(1, 1), (1, 129), (0, 8)]:
        assert lib.pair_coeffs(B, G, one, one, one, 1.0, 0, one, None, None,
                               None, None, None) == 1
    assert lib.pair_coeffs(1, 8, None, one, one, 1.0, 0, one, None, None, None,
                           None, None) == 1
    assert lib.pair_coeffs(1, 8, one, one, one, 1.0, 4, one, None, None, None,
                           None, None) == 1
    assert lib.pair_estimate_dense(1, 8, 0, one, one, one, one, 1.0, one, None,
                                   None, None) == 1
    # pair_grad: nulls, misalignment, bad shapes, workspace too small.
    args = [100, 128, 256, L.PAIR_BF16, one, one, one, one, one, 2, one, one,
            one, one, None, one, 1 << 30, None, None]
    assert lib.pair_grad(*args) != 0
    bad = list(args); bad[4] = None
    assert lib.pair_grad(*bad) == 1
    bad = list(args); bad[4] = P(8)
    assert lib.pair_grad(*bad) == 1
    bad = list(args); bad[1] = 96
    assert lib.pair_grad(*bad) == 2          # bf16 with d % 64 != 0
    bad = list(args); bad[16] = 1024
    assert lib.pair_grad(*bad) == 3          # workspace too small
    bad = list(args); bad[15] = P(16 + 128)
    assert lib.pair_grad(*bad) == 3          # workspace not 256-aligned
    # pair_grad_token_logp: null output, bad shapes, workspace missing or small.
    need = L.pair_grad_workspace_min_size(100, 128, 256, 2, L.PAIR_BF16)
    ws_ok = P(1 << 20)
    assert lib.pair_grad_token_logp(100, 128, 256, 2, L.PAIR_BF16, ws_ok, need, None,
                                    None) == 1
    assert lib.pair_grad_token_logp(100, 96, 256, 2, L.PAIR_BF16, ws_ok, need, one, None) == 1
    assert lib.pair_grad_token_logp(100, 128, 256, 2, L.PAIR_BF16, None, need, one, None) == 3
    assert lib.pair_grad_token_logp(100, 128, 256, 2, L.PAIR_BF16, ws_ok, need - 1, one,
                                    None) == 3
