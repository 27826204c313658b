#!/usr/bin/env python
"""Benchmark of the Pair estimator hot path on GB300.

One step = one pass of the whole hot path over one batch of the Qwen3-1.7B
head workload (8 prompts x 8 rollouts, d = 2048, V = 151936, response
lengths U[256, 2048], packed): pair_coeffs (per-rollout coefficients of
Eq. pair-advantage from rewards, completion mask and the logged inclusion
matrix) followed by pair_grad (LM-head GEMM, vocabulary log-softmax, target
gather, scaling by a_i and the backward to dHidden and dW). The metric is
pair_grad tokens/s (packed tokens per second, forward + backward); the JSON
line also carries pair_coeffs / pair_estimate_dense GB/s on the
4096 x 64 coefficient stress workload.

Usage: python bench.py [--steps K] [--warmup W] [--impl gb300|reference]
The library is single-GPU: every call runs on the current device alone, its
tensor-core kernels pairing CTAs within thread-block clusters of that GPU.
--gpus N with N > 1 (or a torchrun launch with WORLD_SIZE > 1) exits
with an error for the GPU arm; the reference arm (the fp64 CPU oracle) runs
on rank 0 only.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2608_11368_gb300 import synth  # noqa: E402

WORKLOAD = "qwen3_1p7b_head"
STRESS = "coeffs_dense_stress"
METRIC = "pair_grad tokens/s (fwd+bwd) and % dense-BF16 peak; pair_coeffs GB/s vs HBM"
FLUSH_BYTES = 256 << 20          # > 129 MB L2
ORACLE_SAMPLE_TOKENS = 256       # active tokens of the oracle sample (both CPU legs)
EXTRA_WORKLOADS = ("qwen3_4b_head", "longctx_skew")
EXTRA_STEPS, EXTRA_WARMUP = 3, 3
ROT = 8                          # rotating input copies for the coefficient kernels
# Tensor-core kernels of one pair_grad call and the logit-sized GEMMs
# (2 T_eff V d FLOP each) of algorithmic work each is charged per call,
# whatever the number of token chunks it is launched for.
TC_KERNELS = {"lse_tc": 1, "bwd_dh_tc": 1, "bwd_dw_tc": 1, "dh_gemm_tc": 1, "dw_gemm_tc": 1,
              "lse_dh_tc": 2}


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=80)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["gb300", "reference"], default="gb300")
    p.add_argument("--seed", type=int, default=0)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-stress", action="store_true")
    p.add_argument("--no-onchip", action="store_true")
    p.add_argument("--no-extra", action="store_true")
    # Smaller variants of the workload, for profiling captures only.
    p.add_argument("--workload", default=WORKLOAD,
                   choices=["qwen3_1p7b_head", "qwen3_4b_head", "longctx_skew"])
    p.add_argument("--len-scale", type=float, default=1.0)
    p.add_argument("--vocab", type=int, default=0,
                   help="override the head's vocabulary size (0 = the workload's)")
    p.add_argument("--ws-exact", action="store_true",
                   help="size the pair_grad workspace for the active tokens (image of "
                        "softmax terms and scaled rows for ceil(T_eff/128) token blocks) instead "
                        "of pair_grad_workspace_size, which sizes it for the packed length")
    return p.parse_args()


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        pk = json.load(open(path))
        return dict(hbm=float(pk["hbm_gbs"]), bf16=float(pk["bf16_tflops"]),
                    bf16_sus=float(pk["bf16_tflops_sustained"]), src="measured")
    except Exception:
        return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, src="fallback")


def code_hash(path):
    """sha256[:16] of a source file's code: every line with its // comment
    removed and trailing space stripped, blank lines dropped (comment edits
    leave it unchanged, any code change alters it)."""
    import hashlib
    lines = []
    for line in open(path, encoding="utf-8"):
        code = line.split("//", 1)[0].rstrip()
        if code:
            lines.append(code)
    return hashlib.sha256("\n".join(lines).encode()).hexdigest()[:16]


def sources_hash(src):
    """code_hash of one file, or for a comma-separated list of files the
    sha256[:16] of their code_hash values joined by commas (a kernel whose
    code spans several files)."""
    files = src.split(",")
    if len(files) == 1:
        return code_hash(os.path.join(ROOT, files[0]))
    import hashlib
    joined = ",".join(code_hash(os.path.join(ROOT, f)) for f in files)
    return hashlib.sha256(joined.encode()).hexdigest()[:16]


def load_traffic():
    """Per-call DRAM bytes from the committed ncu summary, keyed by kernel,
    valid only while the kernel source code is unchanged (hash recorded
    there, see code_hash)."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.txt")
    out = {}
    if not os.path.exists(path):
        return out
    for line in open(path):
        parts = line.split()
        if len(parts) < 5 or line.startswith("#"):
            continue
        name, wl, bytes_, src, sha = parts[:5]
        try:
            cur = sources_hash(src)
        except OSError:
            continue
        if cur == sha:
            out[(name, wl)] = float(bytes_)
    return out


class ClockSampler:
    """nvidia-smi samples (200 ms) during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,utilization.gpu,"
         "clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.rows = []
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.Q,
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.rows.append([x.strip() for x in line.split(",")])

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=5)
        sm, mx, reasons, power = [], [], set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in self.rows:
            if len(r) < 10:
                continue
            try:
                sm.append(float(r[1])); mx.append(float(r[2])); power.append(float(r[3]))
            except ValueError:
                continue
            for k, nm in enumerate(names):
                if r[6 + k].lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm),
                "power_w_max": max(power) if power else None}


def count_active_tokens(inp, a):
    cu = inp["cu_seqlens"]
    seg = np.repeat(np.arange(cu.size - 1), np.diff(cu))
    return int(((inp["mask"] == 1) & (a[seg] != 0)).sum())


def cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


# ------------------------------------------------------------- CPU oracle leg

class OracleSample:
    """The fp64 oracle (as it stands) on a bounded sample of one step: the
    coefficients of every group plus the complete head work (lse, logp, dH
    rows, dW contribution over all V rows) of the first n_tok active tokens.
    Both CPU legs (cpu_baseline and --impl reference) time this same sample;
    the full step is extrapolated by T_eff / n_tok."""

    def __init__(self, inp, n_tok):
        import oracle
        self.oracle = oracle
        self.inp = inp
        c = oracle.coeffs(inp["r"], inp["J"], inp["rho"])
        idx, cc, _ = oracle.compact_tokens(inp["cu_seqlens"], inp["mask"], c["a"].reshape(-1))
        self.T_eff = int(idx.size)
        sub = idx[:n_tok]
        self.n = int(sub.size)
        # Upcasts (untimed): the oracle works on fp64 copies of the bf16 inputs.
        self.W64 = synth.as_float(inp["W"], inp["dtype"]).astype(np.float64)
        self.Hs = synth.as_float(inp["H"][sub], inp["dtype"]).astype(np.float64)
        self.ys = inp["y"][sub]
        self.cs = cc[:sub.size]

    def run(self):
        """Seconds of (coefficients, head sample)."""
        o, inp = self.oracle, self.inp
        t0 = time.perf_counter()
        o.coeffs(inp["r"], inp["J"], inp["rho"])
        t_coef = time.perf_counter() - t0
        t0 = time.perf_counter()
        lse, _ = o.head_lse(self.Hs, self.W64, self.ys)
        o.head_dh_rows(self.Hs, self.W64, self.ys, self.cs, lse)
        o.head_dw_rows(self.Hs, self.W64, self.ys, self.cs, lse, np.arange(inp["V"]))
        return t_coef, time.perf_counter() - t0

    def full_step_s(self, t_coef, t_head):
        return t_coef + t_head * self.T_eff / max(self.n, 1)

    def describe(self, measured_s):
        return ("fp64 oracle: coefficients of all %d groups + full head work (lse, dH rows, "
                "dW over all V) of %d of %d active tokens; measured %.2f s per sample, step "
                "time extrapolated by T_eff/%d" % (self.inp["B"], self.n, self.T_eff, measured_s,
                                                   self.n))


def cpu_baseline(inp):
    smp = OracleSample(inp, ORACLE_SAMPLE_TOKENS)
    t_coef, t_head = smp.run()
    est = smp.full_step_s(t_coef, t_head)
    return {"value": inp["T"] / est, "unit": "tokens/s", "cores": cores(), "kind": "oracle",
            "measured_sample_s": t_coef + t_head, "extrapolated_step_s": est,
            "sample": smp.describe(t_coef + t_head)}


def bench_config(args, wl, inp, T_eff):
    """The `config` object of both arms' JSON lines."""
    return {"workload": args.workload, "len_scale": args.len_scale, "d": inp["d"],
            "V": inp["V"], "global_batch": wl.B * wl.G, "prompts": wl.B,
            "rollouts_per_prompt": wl.G, "tokens_packed": inp["T"], "tokens_active": T_eff,
            "l2": "flushed between timed steps (256 MiB write); inputs exceed L2",
            "parallelism": "single GPU"}


def run_reference(args, rank):
    """The reference arm: the fp64 oracle as it stands on the host cores, one
    bounded sample per step (the same sample as the GPU arm's cpu_baseline);
    ms_per_step is the measured time of that sample, value the packed tokens
    of the full step over its extrapolated time."""
    if rank != 0:
        return 0
    wl = synth.WORKLOADS[args.workload]
    kw = {"V": args.vocab} if args.vocab else {}
    inp = synth.make_head_workload(wl, args.seed, len_scale=args.len_scale, **kw)
    smp = OracleSample(inp, ORACLE_SAMPLE_TOKENS)
    measured, full = [], []
    for k in range(args.warmup + args.steps):
        t_coef, t_head = smp.run()
        if k >= args.warmup:
            measured.append(t_coef + t_head)
            full.append(smp.full_step_s(t_coef, t_head))
    meas_s = statistics.mean(measured)
    step_s = statistics.mean(full)
    value = inp["T"] / step_s
    line = {"impl": "reference", "metric": METRIC, "value": value,
            "unit": "tokens/s", "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": meas_s * 1e3,
            "extrapolated_full_step_ms": step_s * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f64", "data": "synthetic (seeded; Qwen3-1.7B head shapes, random-init weights)",
            "config": bench_config(args, wl, inp, smp.T_eff),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores(),
                             "kind": "oracle", "measured_sample_s": meas_s,
                             "extrapolated_step_s": step_s,
                             "sample": "per step: " + smp.describe(meas_s)},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------- GPU leg

def timed_steps(B, torch, step, steps, flush):
    """Per-step device times (CUDA events on the current stream, L2 flushed
    before each step) and the library's per-kernel event timings."""
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)]
    torch.cuda.synchronize()
    B.pair_timing_enable(True)
    for k in range(steps):
        flush.zero_()
        ev[k][0].record()
        step()
        ev[k][1].record()
    torch.cuda.synchronize()
    kern = B.pair_timing_read()
    B.pair_timing_enable(False)
    return [s.elapsed_time(e) for s, e in ev], kern


def kernel_report(kern, steps, T_eff, V, d, peaks, traffic, workload):
    """Roofline of the dominant kernel and the per-kernel breakdown of one
    pair_grad call. Each tensor-core kernel is charged its algorithmic share of
    the head's three logit-sized GEMMs (2 T_eff V d FLOP each): one, or two for
    the fused log-sum-exp + dH pass. One "launch" is the kernel's whole share of
    one call (the sum over its token-chunk launches)."""
    agg = {}
    for name, ms in kern:
        n, tot = agg.get(name, (0, 0.0))
        agg[name] = (n + 1, tot + ms)
    flops_gemm = 2.0 * T_eff * V * d
    dominant = max(agg.items(), key=lambda kv: kv[1][1])[0]
    dn, dt_ms = agg[dominant]
    dom_avg = dt_ms / steps
    dom_flops = flops_gemm * TC_KERNELS[dominant] if dominant in TC_KERNELS else None
    achieved = dom_flops / (dom_avg / 1e3) / 1e12 if dom_flops else None
    roofline = {"kernel": dominant, "bound": "tensor",
                "achieved": achieved, "peak": peaks["bf16_sus"], "unit": "TFLOP/s",
                "frac": (achieved / peaks["bf16_sus"]) if achieved else None,
                "traffic": traffic.get((dominant, workload)),
                "peak_source": peaks["src"] + " sustained bf16 (kernel timed inside a long step)",
                "algorithmic_flops_per_launch": dom_flops,
                "avg_launch_ms": dom_avg, "launches_per_call": dn / steps}
    tc_ms = sum(agg[k][1] for k in TC_KERNELS if k in agg) / steps
    grad_ms = sum(t for nm, (n, t) in agg.items() if nm not in ("coeffs",)) / steps
    total = sum(x[1] for x in agg.values())
    info = {
        "algorithmic_tflops": 3 * flops_gemm / (grad_ms / 1e3) / 1e12,
        "frac_of_sustained_bf16": 3 * flops_gemm / (grad_ms / 1e3) / 1e12 / peaks["bf16_sus"],
        "ms_per_call": grad_ms, "tensor_kernels_ms": tc_ms,
        "tokens_active_per_s": T_eff / (grad_ms / 1e3),
        "kernels": {k: {"launches": n, "total_ms": t, "share": t / total}
                    for k, (n, t) in sorted(agg.items(), key=lambda kv: -kv[1][1])}}
    return roofline, info


def device_head_workload(torch, wl, seed):
    """A head workload for a throughput line: rewards, masks, lengths and
    targets from the seeded generator, H ~ N(0, 1) and W ~ N(0, 1/d) drawn on
    the device by torch's seeded generator and rounded to bf16 (the same
    distributions; the timing does not depend on the values)."""
    inp = synth.make_head_workload(wl, seed, draw_hw=False)
    g = torch.Generator(device="cuda")
    g.manual_seed(1000003 * (seed + 1))
    T, d, V = inp["T"], inp["d"], inp["V"]
    H = torch.empty((T, d), dtype=torch.bfloat16, device="cuda")
    for s in range(0, T, 65536):
        e = min(T, s + 65536)
        H[s:e] = torch.randn((e - s, d), generator=g, device="cuda").to(torch.bfloat16)
    H[torch.from_numpy(inp["mask"] == 0).cuda()] = 0
    W = (torch.randn((V, d), generator=g, device="cuda") / math.sqrt(d)).to(torch.bfloat16)
    return inp, H, W


def main():
    args = parse_args()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        return run_reference(args, rank)
    if args.gpus != 1 or world != 1:
        print("bench.py: single-GPU library (every call runs on the current device); "
              "run it with --gpus 1", file=sys.stderr)
        return 2

    import torch
    from paper_2608_11368_gb300 import binding as B

    torch.cuda.set_device(0)
    peaks = load_peaks()
    # The committed DRAM figures are for the workloads as specified; a
    # resized profiling variant has none.
    traffic = load_traffic() if not (args.vocab or args.len_scale != 1.0) else {}
    wl = synth.WORKLOADS[args.workload]
    kw = {"V": args.vocab} if args.vocab else {}
    inp = synth.make_head_workload(wl, args.seed, len_scale=args.len_scale, **kw)
    T, d, V, R = inp["T"], inp["d"], inp["V"], inp["R"]

    def pinned(x):
        t = torch.from_numpy(np.ascontiguousarray(x))
        return t.pin_memory()

    host = {
        "H": pinned(inp["H"].view(np.int16)), "W": pinned(inp["W"].view(np.int16)),
        "y": pinned(inp["y"]), "mask": pinned(inp["mask"]),
        "cu": pinned(inp["cu_seqlens"]), "r": pinned(inp["r"]),
        "J": pinned(inp["J"]), "rho": pinned(inp["rho"]),
    }
    devb = {k: v.to("cuda", non_blocking=False) for k, v in host.items()}
    a = torch.empty((wl.B, wl.G), dtype=torch.float32, device="cuda")
    active = torch.empty((wl.B, wl.G), dtype=torch.uint8, device="cuda")
    edges = torch.empty(wl.B, dtype=torch.int32, device="cuda")
    contrast = torch.empty(wl.B, dtype=torch.int32, device="cuda")
    dH = torch.empty((T, d), dtype=torch.float32, device="cuda")
    dW = torch.empty((V, d), dtype=torch.float32, device="cuda")
    Jobj = torch.empty(1, dtype=torch.float64, device="cuda")
    lps = torch.empty(R, dtype=torch.float32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    if args.ws_exact:
        # The coefficients fix which rollouts are active; image and scaled
        # rows for exactly their token blocks (one block's bytes: the size
        # difference at T = 128).
        B.pair_coeffs(devb["r"], devb["J"], devb["rho"], a=a, active=active, edges=edges,
                      contrast_edges=contrast, dev_err=err)
        blocks = (count_active_tokens(inp, a.view(-1).cpu().numpy()) + 127) // 128
        block = (B.pair_grad_workspace_size(128, d, V, R, B.PAIR_BF16)
                 - B.pair_grad_workspace_min_size(128, d, V, R, B.PAIR_BF16))
        ws_bytes = min(B.pair_grad_workspace_min_size(T, d, V, R, B.PAIR_BF16) + blocks * block,
                       B.pair_grad_workspace_size(T, d, V, R, B.PAIR_BF16))
    else:
        ws_bytes = B.pair_grad_workspace_size(T, d, V, R, B.PAIR_BF16)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    launches = [0]

    def step(bufs=None, wsp=None):
        bufs = devb if bufs is None else bufs
        B.pair_coeffs(bufs["r"], bufs["J"], bufs["rho"], a=a, active=active,
                      edges=edges, contrast_edges=contrast, dev_err=err)
        n = B.pair_last_launch_count()
        B.pair_grad(bufs["H"].view(torch.bfloat16), bufs["W"].view(torch.bfloat16), bufs["y"],
                    bufs["mask"], bufs["cu"], a.view(-1),
                    dH=dH, dW=dW, Jobj=Jobj, logp_seq=lps, ws=ws if wsp is None else wsp,
                    dev_err=err)
        launches[0] += n + B.pair_last_launch_count()

    for _ in range(args.warmup):
        step()
    st = B.pair_status_sync(err)
    if st != 0:
        raise SystemExit("warm-up step failed: %s" % B.pair_status_string(st))
    T_eff = count_active_tokens(inp, a.view(-1).cpu().numpy())

    # ---- timed region: inputs resident in HBM, L2 flushed between steps.
    sampler = ClockSampler(0)
    sampler.start()
    launches[0] = 0
    step_ms, kern = timed_steps(B, torch, step, args.steps, flush)
    clocks = sampler.stop()
    gpu_launches = launches[0]
    total_ms = sum(step_ms)
    if B.pair_status_sync(err) != 0:
        raise SystemExit("timed steps reported a device error")
    value = T * args.steps / (total_ms / 1e3)
    roofline, pair_grad_info = kernel_report(kern, args.steps, T_eff, V, d, peaks, traffic,
                                             args.workload)

    # ---- end-to-end through the C-ABI with host buffers, right after the
    # device-resident steps (same GPU state as `value`): every step copies
    # all of its inputs from pinned host memory and reads J and logp back.
    # Inputs are double-buffered on a copy stream, so step k + 1's copy runs
    # while step k computes (the way a trainer feeds the stream-ordered API);
    # every copy lies inside the timed region.
    out_h = torch.empty(1 + R, dtype=torch.float64).pin_memory()
    names_in = ["H", "W", "y", "mask", "cu", "r", "J", "rho"]
    h2d = sum(host[k].numel() * host[k].element_size() for k in names_in)
    d2h = Jobj.numel() * 8 + lps.numel() * 4
    lps_h = torch.empty(R, dtype=torch.float32).pin_memory()
    sets = [devb, {k: torch.empty_like(v) for k, v in devb.items()}]
    copy_s = torch.cuda.Stream()
    main_s = torch.cuda.current_stream()
    copied = [torch.cuda.Event(), torch.cuda.Event()]
    consumed = [torch.cuda.Event(), torch.cuda.Event()]
    e2e_ev = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))

    def load(j):
        with torch.cuda.stream(copy_s):
            copy_s.wait_event(consumed[j])
            for k in names_in:
                sets[j][k].copy_(host[k], non_blocking=True)
            copied[j].record(copy_s)

    for j in range(2):
        consumed[j].record(main_s)
    torch.cuda.synchronize()
    e2e_ev[0].record(main_s)
    copy_s.wait_event(e2e_ev[0])
    load(0)
    for k in range(args.steps):
        cur = k & 1
        if k + 1 < args.steps:
            load(cur ^ 1)
        main_s.wait_event(copied[cur])
        step(sets[cur])
        consumed[cur].record(main_s)
        out_h[:1].copy_(Jobj, non_blocking=True)
        lps_h.copy_(lps, non_blocking=True)
    e2e_ev[1].record(main_s)
    torch.cuda.synchronize()
    e2e_ms = e2e_ev[0].elapsed_time(e2e_ev[1])
    e2e = {"value": T * args.steps / (e2e_ms / 1e3), "unit": "tokens/s",
           "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}
    del sets

    # ---- the on-chip form: the same step with pair_grad_workspace_min_size,
    # so no logit-sized tensor (no image of softmax terms) is kept
    # in HBM; the backward recomputes the logits in clusters.
    onchip = None
    if not args.no_onchip:
        ws_min = torch.empty(B.pair_grad_workspace_min_size(T, d, V, R, B.PAIR_BF16),
                             dtype=torch.uint8, device="cuda")
        oc_step = lambda: step(wsp=ws_min)
        for _ in range(args.warmup):
            oc_step()
        if B.pair_status_sync(err) != 0:
            raise SystemExit("on-chip warm-up step failed")
        oc_steps = max(3, min(args.steps, 20))
        sampler_oc = ClockSampler(0)
        sampler_oc.start()
        oc_ms, oc_kern = timed_steps(B, torch, oc_step, oc_steps, flush)
        oc_clocks = sampler_oc.stop()
        if B.pair_status_sync(err) != 0:
            raise SystemExit("on-chip steps reported a device error")
        oc_roof, oc_info = kernel_report(oc_kern, oc_steps, T_eff, V, d, peaks, traffic,
                                         args.workload + ":onchip")
        onchip = {"ms_per_step": sum(oc_ms) / oc_steps, "steps": oc_steps,
                  "warmup": args.warmup,
                  "value": T * oc_steps / (sum(oc_ms) / 1e3), "unit": "tokens/s",
                  "workspace_bytes": ws_min.numel(), "roofline": oc_roof, "pair_grad": oc_info,
                  "clocks": oc_clocks}
        del ws_min

    # ---- the other head workloads (Qwen3-4B head; heavy-tailed long context).
    extra = None
    if not args.no_extra:
        extra = {}
        del dH, dW, ws
        torch.cuda.empty_cache()
        for name in EXTRA_WORKLOADS:
            extra[name] = bench_extra(B, torch, name, args.seed, peaks, traffic, flush)
            torch.cuda.empty_cache()

    # ---- pair_coeffs / pair_estimate_dense on the 4096 x 64 stress workload.
    stress = None
    if not args.no_stress:
        stress = bench_stress(B, torch, peaks, flush, args.steps, traffic)

    cpu = None
    if not args.no_cpu_baseline:
        cpu = cpu_baseline(inp)

    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": total_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded; Qwen3-1.7B head shapes, random-init weights)",
        "config": bench_config(args, wl, inp, T_eff),
        "roofline": roofline, "pair_grad": pair_grad_info, "pair_grad_onchip": onchip,
        "configs": extra, "stress": stress, "cpu_baseline": cpu, "e2e": e2e,
        "clocks": clocks, "gpu_launches": gpu_launches,
    }
    print(json.dumps(line), flush=True)
    return 0


def bench_extra(B, torch, name, seed, peaks, traffic, flush):
    """Throughput of the default pair_coeffs + pair_grad step on another head
    workload (inputs resident in HBM, L2 flushed between steps)."""
    wl = synth.WORKLOADS[name]
    inp, H, W = device_head_workload(torch, wl, seed)
    T, d, V, R = inp["T"], inp["d"], inp["V"], inp["R"]
    dv = lambda x: torch.from_numpy(np.ascontiguousarray(x)).cuda()
    r, J, rho = dv(inp["r"]), dv(inp["J"]), dv(inp["rho"])
    y, mask, cu = dv(inp["y"]), dv(inp["mask"]), dv(inp["cu_seqlens"])
    a = torch.empty((wl.B, wl.G), dtype=torch.float32, device="cuda")
    dH = torch.empty((T, d), dtype=torch.float32, device="cuda")
    dW = torch.empty((V, d), dtype=torch.float32, device="cuda")
    Jobj = torch.empty(1, dtype=torch.float64, device="cuda")
    lps = torch.empty(R, dtype=torch.float32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = torch.empty(B.pair_grad_workspace_size(T, d, V, R, B.PAIR_BF16), dtype=torch.uint8,
                     device="cuda")

    def step():
        B.pair_coeffs(r, J, rho, a=a, dev_err=err)
        B.pair_grad(H, W, y, mask, cu, a.view(-1), dH=dH, dW=dW, Jobj=Jobj, logp_seq=lps,
                    ws=ws, dev_err=err)

    for _ in range(EXTRA_WARMUP):
        step()
    if B.pair_status_sync(err) != 0:
        raise SystemExit("%s warm-up step failed" % name)
    T_eff = count_active_tokens(inp, a.view(-1).cpu().numpy())
    sampler = ClockSampler(0)
    sampler.start()
    ms, kern = timed_steps(B, torch, step, EXTRA_STEPS, flush)
    clocks = sampler.stop()
    if B.pair_status_sync(err) != 0:
        raise SystemExit("%s timed steps reported a device error" % name)
    roof, info = kernel_report(kern, EXTRA_STEPS, T_eff, V, d, peaks, traffic, name)
    step_ms = sum(ms) / EXTRA_STEPS
    out = {"ms_per_step": step_ms, "steps": EXTRA_STEPS, "warmup": EXTRA_WARMUP,
           "tokens_packed": T, "tokens_active": T_eff, "d": d, "V": V,
           "prompts": wl.B, "rollouts_per_prompt": wl.G,
           "value": T / (step_ms / 1e3), "unit": "tokens/s",
           "tokens_active_per_s": T_eff / (step_ms / 1e3),
           "roofline": roof, "pair_grad": info, "clocks": clocks,
           "data": "group inputs, lengths and targets from the seeded generator; H, W drawn "
                   "on the device (same distributions)"}
    del H, W, dH, dW, ws
    return out


def bench_stress(B, torch, peaks, flush, steps, traffic):
    wl = synth.WORKLOADS[STRESS]
    inp = synth.make_dense_workload(wl, 100)
    dv = lambda x: torch.from_numpy(np.ascontiguousarray(x)).cuda()
    r, J, rho, S = dv(inp["r"]), dv(inp["J"]), dv(inp["rho"]), dv(inp["S"])
    Bn, G, D = wl.B, wl.G, wl.d
    a = torch.empty((Bn, G), dtype=torch.float32, device="cuda")
    g = torch.empty((Bn, D), dtype=torch.float32, device="cuda")
    act = torch.empty((Bn, G), dtype=torch.uint8, device="cuda")
    e1 = torch.empty(Bn, dtype=torch.int32, device="cuda")
    e2 = torch.empty(Bn, dtype=torch.int32, device="cuda")

    def timed(fn, n):
        """Median device time of fn's kernel, from the events the library
        records right around its own launch (no host overhead inside)."""
        fn()
        torch.cuda.synchronize()
        ts = []
        for _ in range(n):
            flush.zero_()
            B.pair_timing_enable(True)
            fn()
            rec = B.pair_timing_read()
            B.pair_timing_enable(False)
            ts.append(sum(ms for _, ms in rec))
        return statistics.median(ts)

    reps = max(20, steps)
    # Coefficient kernels: CUDA-graph replays of back-to-back calls over
    # rotating copies of the inputs (ROT copies of rho, 8 x 67 MB > 4 x L2),
    # so every launch reads its rho from HBM and no host launch overhead sits
    # between launches; the time per launch is the replay time / ROT.
    rots = [(r.clone(), J.clone(), rho.clone()) for _ in range(ROT)]
    ess = torch.empty(Bn, dtype=torch.float32, device="cuda")
    mw = torch.empty(Bn, dtype=torch.float32, device="cuda")
    p = dv(inp["p"])
    p_rot = [p.clone() for _ in range(ROT)]

    def graph_timed(call):
        """ms per launch of call(k) over the rotating copies (median of 10
        replays of a captured sequence of ROT calls)."""
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            for k in range(ROT):
                call(k)
        torch.cuda.current_stream().wait_stream(side)
        torch.cuda.synchronize()
        g_ = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_, capture_error_mode="relaxed"):
            for k in range(ROT):
                call(k)
        for _ in range(3):
            g_.replay()
        torch.cuda.synchronize()
        ts = []
        for _ in range(10):
            e0 = torch.cuda.Event(enable_timing=True)
            e1_ = torch.cuda.Event(enable_timing=True)
            e0.record()
            g_.replay()
            e1_.record()
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1_) / ROT)
        del g_
        return statistics.median(ts)

    t_c = graph_timed(lambda k: B.pair_coeffs(rots[k][0], rots[k][1], rots[k][2], a=a,
                                              active=act, edges=e1, contrast_edges=e2))
    t_c_single = timed(lambda: B.pair_coeffs(r, J, rho, a=a, active=act, edges=e1,
                                             contrast_edges=e2), reps)
    t_d = timed(lambda: B.pair_estimate_dense(r, J, rho, S, g=g, a=a), reps)
    B.pair_coeffs(r, J, rho, a=a, active=act, edges=e1, contrast_edges=e2)
    n_act = int((a != 0).sum().item())
    Jn = inp["J"].astype(bool)
    # Bytes the method reads (SURVEY's count: the whole strict upper triangle)
    # and the rho bytes it needs (upper-triangle rows of completed vertices:
    # a vertex that is not completed has no edge).
    bytes_c = Bn * (4 * G * (G - 1) // 2 + 4 * G + G + 4 * G + G + 8)
    row_len = np.array([G - 1 - i for i in range(G)])
    needed_c = int(4 * (Jn * row_len[None, :]).sum()) + Bn * (4 * G + G + 4 * G + G + 8)
    # Weighting variants (same rho traffic plus the two diagnostics words)
    # and the product-design path (marginals only: r, J, p in; a, active,
    # counts and diagnostics out).
    variants = {}
    for name, mode in (("clipped", B.PAIR_W_CLIPPED), ("self_normalised", B.PAIR_W_HAJEK)):
        t_w = graph_timed(lambda k: B.pair_coeffs_weighted(
            rots[k][0], rots[k][1], rots[k][2], wmode=mode, w_max=20.0, a=a, active=act,
            edges=e1, contrast_edges=e2, ess=ess, max_w=mw))
        bw = bytes_c + 8 * Bn
        variants[name] = {"bound": "hbm", "achieved": bw / (t_w / 1e3) / 1e9,
                          "peak": peaks["hbm"], "unit": "GB/s",
                          "frac": bw / (t_w / 1e3) / 1e9 / peaks["hbm"], "traffic": None,
                          "ms": t_w, "algorithmic_bytes": bw}
    t_p = graph_timed(lambda k: B.pair_coeffs_product(rots[k][0], rots[k][1], p_rot[k], a=a,
                                                      active=act, edges=e1, contrast_edges=e2,
                                                      ess=ess, max_w=mw))
    del rots, p_rot
    # Frozen-population audit at the paper's audit scale: one 16-candidate
    # group, 50,000 independent-design draws, scores of dimension 4096.
    rng = np.random.default_rng(1234)
    Ga, Da, Na = 16, 4096, 50000
    pa = rng.uniform(0.1, 0.95, Ga)
    ra = dv((rng.random(Ga) < 0.5).astype(np.float32))
    rhoa_np = np.outer(pa, pa).astype(np.float32)
    np.fill_diagonal(rhoa_np, pa.astype(np.float32))
    rhoa = dv(rhoa_np)
    Sa = dv(rng.standard_normal((Ga, Da)).astype(np.float32))
    Jda = dv((rng.random((Na, Ga)) < pa[None]).astype(np.uint8))
    st_a = torch.empty(8, dtype=torch.float64, device="cuda")
    bias_a = torch.empty(Da, dtype=torch.float64, device="cuda")
    ws_a = torch.empty(int(B.lib().pair_audit_workspace_size(Na, Ga, Da)), dtype=torch.uint8,
                       device="cuda")
    Ma = Ga * (Ga - 1) // 2
    t_a = timed(lambda: B.pair_audit(ra, rhoa, Sa, Jda, scale=1.0 / Ma, stats=st_a, bias=bias_a,
                                     ws=ws_a), max(5, min(reps, 10)))
    # Allocation step (Sec. 4.3-4.4): the paper's group size (G = 16) for 64
    # prompts of one RL step, and the 4096 x 64 stress size. Latency bound
    # (a fixed number of small fp64 Newton systems per group).
    alloc = {}
    for nb, ga in ((64, 16), (4096, 64)):
        ai = synth.make_alloc_inputs(77, nb, ga)
        c_al, b_al, p_al = dv(ai["c_hat"]), dv(ai["budget"]), dv(ai["p_hat"])
        pi_al = torch.empty((nb, ga), dtype=torch.float32, device="cuda")
        st_al = torch.empty((nb, 5), dtype=torch.float64, device="cuda")
        t_al = timed(lambda: B.pair_allocate(c_al, b_al, float(ai["pi_min"]), p_hat=p_al,
                                             pi=pi_al, stats=st_al), 3)
        s_al = st_al.cpu().numpy()
        alloc["%dx%d" % (nb, ga)] = {
            "ms": t_al, "groups_per_s": nb / (t_al / 1e3),
            "newton_mean": float(s_al[:, 3].mean()), "newton_max": int(s_al[:, 3].max()),
            "solved": int((s_al[:, 4] == 0).sum()),
            "bound": "latency (fp64 log-barrier Newton, one CTA per group)"}
    bytes_p = Bn * (4 * G + G + 4 * G + 4 * G + G + 16)
    bytes_d = 4 * D * n_act + Bn * (4 * G * (G - 1) // 2 + 4 * G + G) + 4 * Bn * D + 4 * Bn * G
    gbs_c = bytes_c / (t_c / 1e3) / 1e9
    gbs_d = bytes_d / (t_d / 1e3) / 1e9
    return {
        "workload": STRESS,
        "pair_coeffs": {"bound": "hbm", "achieved": gbs_c, "peak": peaks["hbm"],
                        "unit": "GB/s", "frac": gbs_c / peaks["hbm"],
                        "traffic": traffic.get(("coeffs", STRESS)),
                        "ms": t_c, "algorithmic_bytes": bytes_c,
                        "needed_bytes": needed_c,
                        "needed_gbs": needed_c / (t_c / 1e3) / 1e9,
                        "ms_single_launch": t_c_single,
                        "timing": ("CUDA-graph replays of %d back-to-back launches over rotating "
                                   "input copies (%d x 67 MB of rho > 4 x L2), median of 10; "
                                   "ms_single_launch: one launch between CUDA events, L2 flushed"
                                   % (ROT, ROT))},
        "pair_estimate_dense": {"bound": "hbm", "achieved": gbs_d, "peak": peaks["hbm"],
                                "unit": "GB/s", "frac": gbs_d / peaks["hbm"],
                                "traffic": traffic.get(("dense", STRESS)),
                                "ms": t_d, "algorithmic_bytes": bytes_d},
        "pair_coeffs_weighted": variants,
        "pair_audit": {"draws": Na, "G": Ga, "D": Da, "ms": t_a,
                       "draws_per_s": Na / (t_a / 1e3),
                       "stats": dict(zip(B.AUDIT_STATS, st_a.cpu().tolist())),
                       "bound": "latency (per-draw coefficient collapse and quadratic forms)"},
        "pair_allocate": alloc,
        "pair_coeffs_product": {"bound": "hbm", "achieved": bytes_p / (t_p / 1e3) / 1e9,
                                "peak": peaks["hbm"], "unit": "GB/s",
                                "frac": bytes_p / (t_p / 1e3) / 1e9 / peaks["hbm"],
                                "traffic": None, "ms": t_p, "algorithmic_bytes": bytes_p,
                                "speedup_vs_joint_rho": t_c / t_p},
        "timing": ("pair_coeffs, weighted and product paths: CUDA-graph replays over rotating "
                   "input copies (see pair_coeffs.timing); dense estimator, audit and "
                   "allocation: median of single launches, CUDA events recorded by the "
                   "library around its own launch, L2 flushed before each"),
    }


if __name__ == "__main__":
    sys.exit(main())
