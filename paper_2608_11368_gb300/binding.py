"""ctypes binding of libpair.so for torch tensors: argument marshalling only.

The functions carry the C-ABI names (include/pair.h). Every step of the
estimator runs in the library's CUDA kernels; this module only checks
tensor placement/dtypes, allocates outputs with torch when the caller does
not pass them, and forwards raw device pointers plus the current CUDA stream.
There is no CPU fallback: if libpair.so is missing, importing the binding's
library raises.
"""
from __future__ import annotations

import ctypes
import os
import re

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libpair.so")
HEADER = os.path.join(os.path.dirname(_PKG), "include", "pair.h")

PAIR_OK = 0
PAIR_F32, PAIR_BF16 = 0, 1
PAIR_CENTER = 1
PAIR_STANDARDIZE = 2
STATUS_NAMES = {0: "PAIR_OK", 1: "PAIR_ERR_INVALID_ARG", 2: "PAIR_ERR_UNSUPPORTED",
                3: "PAIR_ERR_WORKSPACE", 4: "PAIR_ERR_NONPOSITIVE_INCLUSION",
                5: "PAIR_ERR_TARGET_RANGE", 6: "PAIR_ERR_CUDA",
                7: "PAIR_ERR_DEVICE_TIMEOUT"}


class PairError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__("%s: %s (%s)" % (where, STATUS_NAMES.get(status, status),
                                          pair_status_string(status)))


_lib = None


def lib() -> ctypes.CDLL:
    """Load libpair.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError("libpair.so is not built (run __graft_entry__.build())")
    L = ctypes.CDLL(LIB_PATH)
    P, I32, I64, F32, U32, SZ = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64,
                                 ctypes.c_float, ctypes.c_uint32, ctypes.c_size_t)
    L.pair_coeffs.argtypes = [I32, I32, P, P, P, F32, U32, P, P, P, P, P, P]
    L.pair_coeffs.restype = ctypes.c_int
    L.pair_estimate_dense.argtypes = [I32, I32, I32, P, P, P, P, F32, P, P, P, P]
    L.pair_estimate_dense.restype = ctypes.c_int
    L.pair_grad_workspace_size.argtypes = [I64, I32, I32, I32, ctypes.c_int]
    L.pair_grad_workspace_size.restype = SZ
    L.pair_grad_workspace_min_size.argtypes = [I64, I32, I32, I32, ctypes.c_int]
    L.pair_grad_workspace_min_size.restype = SZ
    L.pair_grad.argtypes = [I64, I32, I32, ctypes.c_int, P, P, P, P, P, I32, P,
                            P, P, P, P, P, SZ, P, P]
    L.pair_grad.restype = ctypes.c_int
    L.pair_status_sync.argtypes = [P, P]
    L.pair_status_sync.restype = ctypes.c_int
    L.pair_status_string.argtypes = [ctypes.c_int]
    L.pair_status_string.restype = ctypes.c_char_p
    L.pair_last_launch_count.argtypes = []
    L.pair_last_launch_count.restype = I32
    L.pair_grad_clipped.argtypes = [I64, I32, I32, ctypes.c_int, P, P, P, P, P, I32, P, P, F32,
                                    P, P, P, P, P, P, SZ, P, P]
    L.pair_grad_clipped.restype = ctypes.c_int
    L.pair_grad_noalloc.argtypes = [I64, I32, I32, ctypes.c_int, P, P, P, P, P,
                                    I32, P, P, P, P, P, P, P]
    L.pair_grad_noalloc.restype = ctypes.c_int
    L.pair_timing_enable.argtypes = [I32]
    L.pair_timing_enable.restype = None
    L.pair_timing_read.argtypes = [I32, P, P]
    L.pair_timing_read.restype = I32
    L.pair_coeffs_weighted.argtypes = [I32, I32, P, P, P, F32, U32, ctypes.c_int, F32,
                                       P, P, P, P, P, P, P, P]
    L.pair_coeffs_weighted.restype = ctypes.c_int
    L.pair_coeffs_product.argtypes = [I32, I32, P, P, P, F32, U32, P, P, P, P, P, P, P, P]
    L.pair_coeffs_product.restype = ctypes.c_int
    L.pair_audit_workspace_size.argtypes = [I32, I32, I32]
    L.pair_audit_workspace_size.restype = SZ
    L.pair_audit.argtypes = [I32, I32, I32, P, P, P, P, P, F32, U32, ctypes.c_int, F32, P, P,
                             P, SZ, P, P]
    L.pair_audit.restype = ctypes.c_int
    L.pair_allocate.argtypes = [I32, I32, P, P, P, P, P, F32, P, P, P, P]
    L.pair_allocate.restype = ctypes.c_int
    L.pair_grad_token_logp.argtypes = [I64, I32, I32, I32, ctypes.c_int, P, SZ, P, P]
    L.pair_grad_token_logp.restype = ctypes.c_int
    L.pair_selftest_wait_timeout.argtypes = [I64, P, P, P]
    L.pair_selftest_wait_timeout.restype = ctypes.c_int
    _lib = L
    return L


def header_functions():
    """Names of the functions declared in include/pair.h."""
    txt = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:[\w\s\*]+?)\b(pair_\w+)\s*\(", txt,
                                 flags=re.M)))


def pair_status_string(status: int) -> str:
    return lib().pair_status_string(int(status)).decode()


def pair_last_launch_count() -> int:
    return int(lib().pair_last_launch_count())


def pair_timing_enable(on: bool) -> None:
    """Start (or stop) recording per-kernel CUDA events for this thread."""
    lib().pair_timing_enable(1 if on else 0)


def pair_timing_read(max_launches: int = 4096):
    """[(kernel name, milliseconds)] of the launches recorded since the last
    enable/read (waits for their events)."""
    ms = (ctypes.c_float * max_launches)()
    names = (ctypes.c_char_p * max_launches)()
    n = lib().pair_timing_read(max_launches, ms, names)
    return [(names[i].decode(), float(ms[i])) for i in range(n)]


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _need(t, name, dtype, shape=None):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError("%s must be a CUDA tensor" % name)
    if t.dtype != dtype:
        raise TypeError("%s must be %s, got %s" % (name, dtype, t.dtype))
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError("%s must have shape %s, got %s" % (name, tuple(shape),
                                                            tuple(t.shape)))


def _check(st, where):
    if st != PAIR_OK:
        raise PairError(st, where)


def _on_device(t):
    """Context manager making t's device current for the call: the library
    launches on the current device and takes its stream from there."""
    return torch.cuda.device(t.device)


def _out(t, name, shape, dtype, dev):
    """Caller-passed output (checked) or a fresh torch allocation."""
    if t is None:
        return torch.empty(shape, dtype=dtype, device=dev)
    _need(t, name, dtype, shape)
    if t.device != dev:
        raise ValueError("%s must be on %s, got %s" % (name, dev, t.device))
    return t


def pair_coeffs(r, J, rho, scale=1.0, flags=0, a=None, active=None, edges=None,
                contrast_edges=None, dev_err=None, stream=None):
    """Coefficients of Eq. (pair-advantage) (times `scale`, see pair.h), on
    r's device. Returns (a, active, edges, contrast_edges)."""
    B, G = r.shape
    dev = r.device
    _need(r, "r", torch.float32)
    _need(J, "J", torch.uint8, (B, G))
    _need(rho, "rho", torch.float32, (B, G, G))
    a = _out(a, "a", (B, G), torch.float32, dev)
    active = _out(active, "active", (B, G), torch.uint8, dev)
    edges = _out(edges, "edges", (B,), torch.int32, dev)
    contrast_edges = _out(contrast_edges, "contrast_edges", (B,), torch.int32, dev)
    with _on_device(r):
        st = lib().pair_coeffs(B, G, _p(r), _p(J), _p(rho), float(scale), int(flags),
                               _p(a), _p(active), _p(edges), _p(contrast_edges),
                               _p(dev_err), _stream(stream))
    _check(st, "pair_coeffs")
    return a, active, edges, contrast_edges


PAIR_W_HT, PAIR_W_UNWEIGHTED, PAIR_W_MARGINAL, PAIR_W_CLIPPED, PAIR_W_HAJEK = 0, 1, 2, 3, 4


def _coeffs_outputs(B, G, dev, a, active, edges, contrast_edges, ess, max_w):
    return (_out(a, "a", (B, G), torch.float32, dev),
            _out(active, "active", (B, G), torch.uint8, dev),
            _out(edges, "edges", (B,), torch.int32, dev),
            _out(contrast_edges, "contrast_edges", (B,), torch.int32, dev),
            _out(ess, "ess", (B,), torch.float32, dev),
            _out(max_w, "max_w", (B,), torch.float32, dev))


def pair_coeffs_weighted(r, J, rho, wmode=PAIR_W_HT, w_max=0.0, scale=1.0, flags=0, a=None,
                         active=None, edges=None, contrast_edges=None, ess=None, max_w=None,
                         dev_err=None, stream=None):
    """pair_coeffs under a weighting variant (see pair.h), with per-group ESS
    and largest weight. Returns (a, active, edges, contrast_edges, ess, max_w)."""
    B, G = r.shape
    _need(r, "r", torch.float32)
    _need(J, "J", torch.uint8, (B, G))
    if rho is not None:
        _need(rho, "rho", torch.float32, (B, G, G))
    outs = _coeffs_outputs(B, G, r.device, a, active, edges, contrast_edges, ess, max_w)
    with _on_device(r):
        st = lib().pair_coeffs_weighted(B, G, _p(r), _p(J), _p(rho), float(scale), int(flags),
                                        int(wmode), float(w_max), *[_p(t) for t in outs],
                                        _p(dev_err), _stream(stream))
    _check(st, "pair_coeffs_weighted")
    return outs


def pair_coeffs_product(r, J, p, scale=1.0, flags=0, a=None, active=None, edges=None,
                        contrast_edges=None, ess=None, max_w=None, dev_err=None, stream=None):
    """Coefficients of the independent design rho_ij = p_i p_j from the
    marginals p [B, G]. Returns (a, active, edges, contrast_edges, ess, max_w)."""
    B, G = r.shape
    _need(r, "r", torch.float32)
    _need(J, "J", torch.uint8, (B, G))
    _need(p, "p", torch.float32, (B, G))
    outs = _coeffs_outputs(B, G, r.device, a, active, edges, contrast_edges, ess, max_w)
    with _on_device(r):
        st = lib().pair_coeffs_product(B, G, _p(r), _p(J), _p(p), float(scale), int(flags),
                                       *[_p(t) for t in outs], _p(dev_err), _stream(stream))
    _check(st, "pair_coeffs_product")
    return outs


AUDIT_STATS = ("bias_norm", "mse", "cos", "vertices", "edges", "ess", "target_sq", "weight")


def pair_audit(r, rho, S, Jdraws, draw_weight=None, wmode=PAIR_W_HT, w_max=0.0, scale=1.0,
               flags=0, stats=None, bias=None, ws=None, dev_err=None, stream=None):
    """Frozen-population audit of one group over design draws (see pair.h).
    r [G], rho [G, G] (None for PAIR_W_UNWEIGHTED), S [G, D], Jdraws [N, G]
    uint8, draw_weight [N] float64 or None. Returns (stats [8] f64, bias [D] f64)."""
    N, G = Jdraws.shape
    D = S.shape[1]
    _need(r, "r", torch.float32, (G,))
    if rho is not None:
        _need(rho, "rho", torch.float32, (G, G))
    _need(S, "S", torch.float32, (G, D))
    _need(Jdraws, "Jdraws", torch.uint8, (N, G))
    if draw_weight is not None:
        _need(draw_weight, "draw_weight", torch.float64, (N,))
    dev = r.device
    stats = _out(stats, "stats", (8,), torch.float64, dev)
    bias = _out(bias, "bias", (D,), torch.float64, dev)
    need = int(lib().pair_audit_workspace_size(N, G, D))
    with _on_device(r):
        if ws is None:
            ws = torch.empty(max(need, 256), dtype=torch.uint8, device=dev)
        _need(ws, "ws", torch.uint8)
        st = lib().pair_audit(N, G, D, _p(r), _p(rho), _p(S), _p(Jdraws), _p(draw_weight),
                              float(scale), int(flags), int(wmode), float(w_max), _p(stats),
                              _p(bias), _p(ws), ws.numel(), _p(dev_err), _stream(stream))
    _check(st, "pair_audit")
    return stats, bias


ALLOC_OK, ALLOC_SLACK, ALLOC_FLOOR, ALLOC_INFEASIBLE, ALLOC_FALLBACK, ALLOC_FLAT, \
    ALLOC_INVALID = range(7)
ALLOC_STATS = ("phi", "spent", "gap", "newton", "status")


def pair_allocate(c_hat, budget, pi_min, p_hat=None, m_hat=None, a=None, pi=None, stats=None,
                  dev_err=None, stream=None):
    """Continuation probabilities of the convex design (see pair.h).
    c_hat [B, G], budget [B], p_hat [B, G] (or a [B, G, G]), m_hat [B, G] or
    None. Returns (pi [B, G] f32, stats [B, 5] f64: phi, spent, gap, newton,
    status)."""
    B, G = c_hat.shape
    _need(c_hat, "c_hat", torch.float32, (B, G))
    _need(budget, "budget", torch.float32, (B,))
    if p_hat is not None:
        _need(p_hat, "p_hat", torch.float32, (B, G))
    if m_hat is not None:
        _need(m_hat, "m_hat", torch.float32, (B, G))
    if a is not None:
        _need(a, "a", torch.float32, (B, G, G))
    dev = c_hat.device
    pi = _out(pi, "pi", (B, G), torch.float32, dev)
    stats = _out(stats, "stats", (B, 5), torch.float64, dev)
    if dev_err is None:
        dev_err = torch.zeros(1, dtype=torch.int32, device=dev)
    with _on_device(c_hat):
        st = lib().pair_allocate(B, G, _p(p_hat), _p(m_hat), _p(a), _p(c_hat), _p(budget),
                                 float(pi_min), _p(pi), _p(stats), _p(dev_err),
                                 _stream(stream))
    _check(st, "pair_allocate")
    return pi, stats


def pair_estimate_dense(r, J, rho, S, scale=1.0, g=None, a=None, dev_err=None,
                        stream=None):
    """Eq. (pair-ht) for explicit scores S [B,G,D], on S's device. Returns (g, a)."""
    B, G, D = S.shape
    _need(r, "r", torch.float32, (B, G))
    _need(J, "J", torch.uint8, (B, G))
    _need(rho, "rho", torch.float32, (B, G, G))
    _need(S, "S", torch.float32)
    g = _out(g, "g", (B, D), torch.float32, S.device)
    if a is not None:
        a = _out(a, "a", (B, G), torch.float32, S.device)
    with _on_device(S):
        st = lib().pair_estimate_dense(B, G, D, _p(r), _p(J), _p(rho), _p(S),
                                       float(scale), _p(g), _p(a), _p(dev_err),
                                       _stream(stream))
    _check(st, "pair_estimate_dense")
    return g, a


def pair_grad_workspace_size(T, d, V, R, dtype) -> int:
    return int(lib().pair_grad_workspace_size(int(T), int(d), int(V), int(R),
                                              int(dtype)))


def pair_grad_workspace_min_size(T, d, V, R, dtype) -> int:
    return int(lib().pair_grad_workspace_min_size(int(T), int(d), int(V), int(R),
                                                  int(dtype)))


def _pair_dtype(t):
    if t.dtype == torch.bfloat16:
        return PAIR_BF16
    if t.dtype == torch.float32:
        return PAIR_F32
    raise TypeError("H/W must be bfloat16 or float32")


def _grad_inputs(H, W, y, mask, cu_seqlens, a):
    T, d = H.shape
    V = W.shape[0]
    R = cu_seqlens.numel() - 1
    dt = _pair_dtype(H)
    _need(H, "H", H.dtype, (T, d))
    _need(W, "W", H.dtype, (V, d))
    _need(y, "y", torch.int32, (T,))
    _need(mask, "mask", torch.uint8, (T,))
    _need(cu_seqlens, "cu_seqlens", torch.int32, (R + 1,))
    _need(a, "a", torch.float32, (R,))
    for t, nm in ((W, "W"), (y, "y"), (mask, "mask"), (cu_seqlens, "cu_seqlens"), (a, "a")):
        if t.device != H.device:
            raise ValueError("%s must be on %s like H, got %s" % (nm, H.device, t.device))
    return T, d, V, R, dt


def _grad_outputs(T, d, V, R, dev, dH, dW, Jobj, logp_seq):
    return (_out(dH, "dH", (T, d), torch.float32, dev), _out(dW, "dW", (V, d), torch.float32, dev),
            _out(Jobj, "Jobj", (1,), torch.float64, dev),
            _out(logp_seq, "logp_seq", (R,), torch.float32, dev))


def pair_grad(H, W, y, mask, cu_seqlens, a, dH=None, dW=None, Jobj=None,
              logp_seq=None, ws=None, dev_err=None, stream=None):
    """LM-head realisation of sum_i a_i log pi(o_i|q) and its gradients.
    Runs on H's device. Returns (Jobj [1] f64, dH [T,d] f32, dW [V,d] f32,
    logp_seq [R] f32)."""
    T, d, V, R, dt = _grad_inputs(H, W, y, mask, cu_seqlens, a)
    dev = H.device
    dH, dW, Jobj, logp_seq = _grad_outputs(T, d, V, R, dev, dH, dW, Jobj, logp_seq)
    with _on_device(H):
        if ws is None:
            need = pair_grad_workspace_size(T, d, V, R, dt)
            ws = torch.empty(max(need, 256), dtype=torch.uint8, device=dev)
        _need(ws, "ws", torch.uint8)
        st = lib().pair_grad(T, d, V, dt, _p(H), _p(W), _p(y), _p(mask),
                             _p(cu_seqlens), R, _p(a), _p(dH), _p(dW), _p(Jobj),
                             _p(logp_seq), _p(ws), ws.numel(), _p(dev_err),
                             _stream(stream))
    _check(st, "pair_grad")
    return Jobj, dH, dW, logp_seq


def pair_grad_token_logp(T, d, V, R, dtype, ws, logp_tok=None, stream=None):
    """Per-token log-probabilities [T] left in `ws` by the last pair_grad (or
    pair_grad_clipped) call with these shapes (see pair.h): logp_t for active
    tokens, 0 elsewhere."""
    _need(ws, "ws", torch.uint8)
    logp_tok = _out(logp_tok, "logp_tok", (int(T),), torch.float32, ws.device)
    with _on_device(ws):
        st = lib().pair_grad_token_logp(int(T), int(d), int(V), int(R), int(dtype), _p(ws),
                                        ws.numel(), _p(logp_tok), _stream(stream))
    _check(st, "pair_grad_token_logp")
    return logp_tok


def pair_grad_clipped(H, W, y, mask, cu_seqlens, a, logp_old, clip_eps=0.2, dH=None, dW=None,
                      Jobj=None, logp_seq=None, coef=None, ws=None, dev_err=None, stream=None):
    """Clipped trajectory-ratio surrogate (see pair.h). Runs on H's device.
    Returns (Jobj [1] f64, dH [T,d] f32, dW [V,d] f32, logp_seq [R] f32, coef [R] f32)."""
    T, d, V, R, dt = _grad_inputs(H, W, y, mask, cu_seqlens, a)
    _need(logp_old, "logp_old", torch.float32, (R,))
    dev = H.device
    dH, dW, Jobj, logp_seq = _grad_outputs(T, d, V, R, dev, dH, dW, Jobj, logp_seq)
    coef = _out(coef, "coef", (R,), torch.float32, dev)
    with _on_device(H):
        if ws is None:
            need = pair_grad_workspace_size(T, d, V, R, dt)
            ws = torch.empty(max(need, 256), dtype=torch.uint8, device=dev)
        _need(ws, "ws", torch.uint8)
        st = lib().pair_grad_clipped(T, d, V, dt, _p(H), _p(W), _p(y), _p(mask), _p(cu_seqlens),
                                     R, _p(a), _p(logp_old), float(clip_eps), _p(dH), _p(dW),
                                     _p(Jobj), _p(logp_seq), _p(coef), _p(ws), ws.numel(),
                                     _p(dev_err), _stream(stream))
    _check(st, "pair_grad_clipped")
    return Jobj, dH, dW, logp_seq, coef


NOALLOC_MAX_WORKSPACE = 32 << 20


def pair_grad_noalloc(H, W, y, mask, cu_seqlens, a, dH=None, dW=None,
                      Jobj=None, logp_seq=None, dev_err=None, stream=None):
    """pair_grad on the library's fixed device workspace (no workspace
    argument; see pair.h for the size limit and the sharing rules). Runs on
    H's device. Output tensors not passed in are allocated here by torch, as
    in pair_grad; pass all four (checked for shape, dtype and device) to keep
    the call allocation-free. Returns (Jobj, dH, dW, logp_seq)."""
    T, d, V, R, dt = _grad_inputs(H, W, y, mask, cu_seqlens, a)
    dev = H.device
    dH, dW, Jobj, logp_seq = _grad_outputs(T, d, V, R, dev, dH, dW, Jobj, logp_seq)
    with _on_device(H):
        st = lib().pair_grad_noalloc(T, d, V, dt, _p(H), _p(W), _p(y), _p(mask),
                                     _p(cu_seqlens), R, _p(a), _p(dH), _p(dW),
                                     _p(Jobj), _p(logp_seq), _p(dev_err),
                                     _stream(stream))
    _check(st, "pair_grad_noalloc")
    return Jobj, dH, dW, logp_seq


def pair_selftest_wait_timeout(limit_cycles, dev_err, seen, stream=None):
    """Launch the bounded-wait failure-path check (see pair.h)."""
    _need(dev_err, "dev_err", torch.int32)
    _need(seen, "seen", torch.int32, (2,))
    st = lib().pair_selftest_wait_timeout(int(limit_cycles), _p(dev_err), _p(seen),
                                          _stream(stream))
    _check(st, "pair_selftest_wait_timeout")


def pair_status_sync(dev_err=None, stream=None) -> int:
    """Synchronise the stream and decode/reset the device error word (on
    dev_err's device when it is given)."""
    if dev_err is None:
        return int(lib().pair_status_sync(_stream(stream), None))
    with _on_device(dev_err):
        return int(lib().pair_status_sync(_stream(stream), _p(dev_err)))
