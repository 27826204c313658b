"""Helpers for GPU tests: move generator arrays to the device, norms."""
import numpy as np
import torch


def dev(x, device="cuda"):
    return torch.from_numpy(np.ascontiguousarray(x)).to(device)


def head_inputs(inp, a, device="cuda"):
    """Device tensors for pair_grad from a synth head workload and float32
    coefficients a [R]."""
    if inp["dtype"] == "bf16":
        H = torch.from_numpy(inp["H"].view(np.int16)).to(device).view(torch.bfloat16)
        W = torch.from_numpy(inp["W"].view(np.int16)).to(device).view(torch.bfloat16)
    else:
        H, W = dev(inp["H"], device), dev(inp["W"], device)
    return dict(H=H, W=W, y=dev(inp["y"], device), mask=dev(inp["mask"], device),
                cu_seqlens=dev(inp["cu_seqlens"], device),
                a=dev(np.asarray(a, np.float32), device))


def rel_fro(x, ref):
    x = np.asarray(x, np.float64)
    ref = np.asarray(ref, np.float64)
    den = np.linalg.norm(ref)
    return float(np.linalg.norm(x - ref) / (den if den > 0 else 1.0))


def dev_err_word():
    return torch.zeros(1, dtype=torch.int32, device="cuda")
