"""Seeded input generator: determinism, shapes and the stated distributions."""
import numpy as np
import pytest

from paper_2608_11368_gb300 import synth


def test_bf16_rounding_matches_torch():
    torch = pytest.importorskip("torch")
    x = np.random.default_rng(0).standard_normal(100000).astype(np.float32)
    x[:4] = [1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -1.0 - 2 ** -8, 0.0]  # ties
    bits = synth.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy()
    assert (bits.view(np.int16) == ref).all()
    back = synth.bf16_bits_to_f32(bits)
    assert (back == torch.from_numpy(x).to(torch.bfloat16).float().numpy()).all()


def test_deterministic_and_independent_streams():
    wl = synth.WORKLOADS["pr1_ref_fp32"]
    a = synth.make_head_workload(wl, 11)
    b = synth.make_head_workload(wl, 11)
    for k in ("H", "W", "y", "r", "J", "rho", "mask", "cu_seqlens"):
        assert np.array_equal(a[k], b[k])
    c = synth.make_head_workload(wl, 12)
    assert not np.array_equal(a["H"], c["H"])
    # Group inputs do not depend on the head sizes drawn with them.
    d = synth.make_head_workload(wl, 11, V=64, d=16)
    assert np.array_equal(a["r"], d["r"]) and np.array_equal(a["J"], d["J"])


@pytest.mark.parametrize("name", synth.WORKLOAD_ORDER)
def test_group_inputs(name):
    wl = synth.WORKLOADS[name]
    g = synth.draw_group_inputs(wl, 0, B=min(wl.B, 256))
    B, G = g["r"].shape
    assert G == wl.G
    assert set(np.unique(g["r"])) <= {0.0, 1.0}
    assert (g["p"] > wl.p_low - 1e-7).all() and (g["p"] <= 1.0).all()
    rho = g["rho"]
    assert np.array_equal(rho, np.transpose(rho, (0, 2, 1)))
    assert np.array_equal(rho[:, np.arange(G), np.arange(G)], g["p"])
    assert (rho > 0).all()
    if wl.rho_kind == "general":
        cap = np.minimum(g["p"][:, :, None], g["p"][:, None, :])
        assert (rho <= cap).all() and (rho >= 0.05 - 1e-7).all()
    else:
        off = ~np.eye(G, dtype=bool)
        prod = (g["p"][:, :, None] * g["p"][:, None, :]).astype(np.float32)
        assert np.array_equal(rho[:, off], prod[:, off])


def test_packing_layout():
    wl = synth.WORKLOADS["longctx_skew"]
    inp = synth.make_head_workload(wl, 2, B=4, V=64, d=16)
    cu, mask, L = inp["cu_seqlens"], inp["mask"], inp["lengths"]
    assert cu[0] == 0 and cu[-1] == inp["T"]
    assert ((np.diff(cu) % synth.SEG_ALIGN) == 0).all()
    for i in range(inp["R"]):
        seg = mask[cu[i]:cu[i + 1]]
        assert seg[:L[i]].all() and not seg[L[i]:].any()
    stopped = inp["J"].reshape(-1) == 0
    assert (L[stopped] <= wl.prefix).all() and (L <= wl.len_cap).all()
    assert (inp["y"][mask == 0] == -100).all()
    assert ((inp["y"][mask == 1] >= 0) & (inp["y"][mask == 1] < 64)).all()
