"""Benchmark of the fused GEMM + tail path on GB300.

Default workload (the headline line): bf16 Y = GELU_tanh(X W^T + b) * 2 + R,
X[1024x4096], W[4096x4096] -- one kf_fused_gemm call per step.  The JSON line
also carries the other workloads of the path (row log-sum-exp, GroupNorm +
Swish, MoE expert FFN at T=64 and T=4096) under "workloads", each next to its
unfused torch-eager baseline.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl kf|reference] [--main-only]

Timing: CUDA events on the launching stream around each step; a 256 MiB
buffer is written between steps so every step starts with a cold L2 (the
inputs, 59 MB, would otherwise stay resident in the 129 MB L2).  Under
torchrun each rank runs its own replica (weak scaling; no data-path
collective) and the max time over ranks is reported.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import subprocess
import sys
import tempfile
import time

import torch
import torch.nn.functional as F

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import kf_workloads  # noqa: E402

MAIN = "bf16_gelu_scale_residual"
FLUSH_BYTES = 256 << 20


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"], bf16_sus=d["bf16_tflops_sustained"],
                    src="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, src="fallback")


def kernel_source_hash() -> str:
    """Hash of the library's sources (every file under csrc/ and the C header); a
    stored ncu traffic figure is used only while they are unchanged since it was
    captured."""
    h = hashlib.sha256()
    d = os.path.join(ROOT, "paper_2606_02963_gb300", "csrc")
    files = sorted(os.path.join(d, fn) for fn in os.listdir(d) if fn.endswith((".cu", ".cuh", ".h")))
    files.append(os.path.join(ROOT, "include", "kf.h"))
    for fp in files:
        h.update(os.path.basename(fp).encode())
        h.update(open(fp, "rb").read())
    return h.hexdigest()[:16]


def stored_traffic(kernel_tag: str):
    """Per-step DRAM bytes (read + write, all of the path's kernels of one step)
    from profiles/ncu_traffic.txt (lines: '<tag> <source-hash> <bytes>'), or None
    if absent or stale."""
    p = os.path.join(ROOT, "profiles", "ncu_traffic.txt")
    if not os.path.exists(p):
        return None
    cur = kernel_source_hash()
    for line in open(p):
        f = line.split()
        if len(f) >= 3 and f[0] == kernel_tag and f[1] == cur:
            return float(f[2])
    return None


class Clocks:
    """nvidia-smi sampling during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                                          "-i", str(self.index), "-lms", "100"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if not self.path or not os.path.exists(self.path):
            return None
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = max(mx, float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return None
        sm.sort()
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


def reduce_max_over_ranks(values, device, world):
    """Max of each timing over all ranks (the job is as slow as its slowest rank)."""
    if world <= 1:
        return list(values)
    t = torch.tensor(list(values), dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return t.tolist()


def whole_job_tflops(flops_per_rank_step, ms_per_step, world):
    """Whole-job throughput: every rank runs its own replica of the step (weak
    scaling), so the job does world x flops per (max over ranks) step time."""
    return world * flops_per_rank_step / (ms_per_step * 1e-3) / 1e12


SETTLE_S = 0.3


def time_steps(fn, steps, warmup, flush, stream, host_slack=True):
    """Mean device time (ms) of fn() over `steps` calls; L2 flushed before each,
    after `warmup` untimed calls and at least SETTLE_S seconds of untimed calls.
    With host_slack, a ~100 us device-side sleep follows the flush so that the
    host has enqueued the step before its start event fires (host-side argument
    marshalling is then outside the device-timed window)."""
    for _ in range(warmup):
        flush.zero_()
        fn()
    torch.cuda.synchronize()
    # then at least SETTLE_S of back-to-back steps (untimed), so that clocks and
    # caches are in their steady state whatever ran before on this GPU
    t_end = time.perf_counter() + SETTLE_S
    n = 0
    while time.perf_counter() < t_end and n < 2000:
        flush.zero_()
        fn()
        n += 1
        if n % 16 == 0:
            torch.cuda.synchronize()
    torch.cuda.synchronize()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for a, b in evs:
        flush.zero_()
        if host_slack:
            torch.cuda._sleep(200_000)
        a.record(stream)
        fn()
        b.record(stream)
    torch.cuda.synchronize()
    return sum(a.elapsed_time(b) for a, b in evs) / steps


def time_steps_rotating(fns, steps, warmup, stream):
    """Mean device time (ms) per step of `steps` steps run back to back between
    one pair of events; step i calls fns[i % len(fns)], each on its own copy of
    the inputs (the copies together are larger than L2, so no step finds its
    inputs there).  A device-side sleep before the start event gives the host a
    head start: it must finish enqueueing every step before the sleep ends, so
    the device never waits for it (checked; the sleep doubles until it holds).
    Returns (ms, {"sleep_ms", "host_enqueue_ms"})."""
    n = len(fns)
    for i in range(warmup):
        fns[i % n]()
    torch.cuda.synchronize()
    t_end = time.perf_counter() + SETTLE_S
    i = 0
    while time.perf_counter() < t_end and i < 4000:
        fns[i % n]()
        i += 1
        if i % 16 == 0:
            torch.cuda.synchronize()
    torch.cuda.synchronize()
    cycles = 4_000_000
    for _ in range(4):
        s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s0.record(stream)
        torch.cuda._sleep(cycles)
        s1.record(stream)
        a.record(stream)
        h0 = time.perf_counter()
        for j in range(steps):
            fns[j % n]()
        host_ms = (time.perf_counter() - h0) * 1e3
        b.record(stream)
        torch.cuda.synchronize()
        sleep_ms = s0.elapsed_time(s1)
        if host_ms < 0.9 * sleep_ms:
            break
        cycles *= 2
    return a.elapsed_time(b) / steps, {"sleep_ms": round(sleep_ms, 3), "host_enqueue_ms": round(host_ms, 3)}


HEADLINE_COPIES = 6  # x 58.7 MB of inputs and output per step: 352 MB, L2 is 129 MB


# --------------------------------------------------------------- workloads
def dense_chain(wl, d):
    chain = []
    for kind, prm in kf_workloads.chain_spec(wl):
        chain.append((kind, {k: (d[v] if k in ("p0", "p1") else v) for k, v in prm.items()}))
    return chain


def dense_setup(name, dev):
    inp = kf_workloads.generate(name, seed=0)
    d = {k: v.to(dev) for k, v in inp.items()}
    wl = kf_workloads.WORKLOADS[name]
    return wl, inp, d, dense_chain(wl, d)


def dense_bytes(name, wl):
    """Algorithmic bytes of one call: every input read once, the output written once."""
    M, N, K = wl.M, wl.N, wl.K
    e = 4 if wl.dtype == "f32" else 2
    b = e * (M * K + N * K)
    if name == MAIN:
        b += e * (N + M * N + M * N)                # bias, R, Y
    elif name == "bf16_scale_rowlse":
        b += 4 * M                                  # fp32 [M]
    elif name == "bf16_groupnorm_swish":
        b += e * (3 * N + M * N)                    # bias, gamma, beta, Y
    elif name == "fp32_relu_linear":
        b += e * (N + M * N)                        # bias, Y
    return b


def eager_dense(name, d):
    X, W = d["X"], d["W"]
    if name == MAIN:
        return lambda: F.gelu(F.linear(X, W, d["b"]), approximate="tanh") * 2.0 + d["R"]
    if name == "bf16_scale_rowlse":
        return lambda: torch.logsumexp((X @ W.t()).float() * 0.125, dim=1)
    if name == "bf16_groupnorm_swish":
        def f():
            z = F.group_norm(F.linear(X, W, d["b"]), 16, d["gamma"], d["beta"], 1e-5)
            return z * torch.sigmoid(z)
        return f
    raise KeyError(name)


def moe_eager(X, logits, Wgu, Wd, k):
    T, H = X.shape
    E, I2, _ = Wgu.shape
    I = I2 // 2
    v, ids = torch.topk(logits, k, dim=1)
    w = torch.softmax(v, dim=1)
    Y = torch.zeros(T, H, dtype=torch.float32, device=X.device)
    flat = ids.reshape(-1)
    order = torch.argsort(flat, stable=True)
    counts = torch.bincount(flat, minlength=E).tolist()
    tok = order // k
    wf = w.reshape(-1)[order]
    s = 0
    for e in range(E):
        c = counts[e]
        if c == 0:
            continue
        t = tok[s:s + c]
        xe = X[t]
        gu = xe @ Wgu[e].t()
        h = F.silu(gu[:, :I]) * gu[:, I:]
        y = h @ Wd[e].t()
        Y.index_add_(0, t, y.float() * wf[s:s + c, None])
        s += c
    return Y.to(torch.bfloat16)


def run_kf(args, rank, world, dev):
    import paper_2606_02963_gb300 as kf
    kf.lib()
    peaks = _peaks()
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.float32, device=dev)

    # ------------------------------------------------------- headline workload
    wl, inp, d, chain = dense_setup(MAIN, dev)
    flops = 2.0 * wl.M * wl.N * wl.K
    out = torch.empty(wl.M, wl.N, dtype=torch.bfloat16, device=dev)
    step = lambda: kf.fused_gemm(d["X"], d["W"], chain, out=out)

    # e2e: pinned host inputs -> device, kernel, device -> pinned host output
    hin = {k: v.pin_memory() for k, v in inp.items()}
    hout = torch.empty(wl.M, wl.N, dtype=torch.bfloat16).pin_memory()
    h2d = sum(v.numel() * v.element_size() for v in hin.values())
    d2h = hout.numel() * hout.element_size()

    def e2e_step():
        for k2 in hin:
            d[k2].copy_(hin[k2], non_blocking=True)
        kf.fused_gemm(d["X"], d["W"], chain, out=out)
        hout.copy_(out, non_blocking=True)

    # copies of the inputs and the output for back-to-back steps
    copies = [d] + [{k2: v.clone() for k2, v in d.items()} for _ in range(HEADLINE_COPIES - 1)]
    outs = [out] + [torch.empty_like(out) for _ in range(HEADLINE_COPIES - 1)]
    chains = [chain] + [dense_chain(wl, c) for c in copies[1:]]
    rot = [(lambda c=c, ch=ch, o=o: kf.fused_gemm(c["X"], c["W"], ch, out=o)) for c, ch, o in zip(copies, chains, outs)]

    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with Clocks(dev.index if dev.index is not None else 0) as clk:
        ms, rot_info = time_steps_rotating(rot, args.steps, args.warmup, stream)
    clocks = clk.summary()
    ms_iso = time_steps(step, args.steps, args.warmup, flush, stream)
    ms_e2e = time_steps(e2e_step, max(3, args.steps // 2), args.warmup, flush, stream, host_slack=False)
    ms, ms_iso, ms_e2e = reduce_max_over_ranks([ms, ms_iso, ms_e2e], dev, world)
    value = whole_job_tflops(flops, ms, world)
    e2e_value = whole_job_tflops(flops, ms_e2e, world)
    ms_eager, _ = time_steps_rotating([eager_dense(MAIN, c) for c in copies], args.steps, args.warmup, stream)
    ms_cublas, _ = time_steps_rotating([(lambda c=c: torch.matmul(c["X"], c["W"].t())) for c in copies],
                                       args.steps, args.warmup, stream)
    del copies, outs, chains, rot
    traffic = stored_traffic(MAIN)
    achieved = flops / (ms * 1e-3) / 1e12
    line = {
        "metric": "fused GEMM+tail TFLOP/s & % of GB300 roofline; speedup vs unfused torch eager",
        "value": round(value, 2), "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms, 5), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16 operands, fp32 accumulate", "data": "synthetic (seeded)",
        "config": {"workload": MAIN, "M": wl.M, "N": wl.N, "K": wl.K,
                   "chain": "bias -> gelu_tanh -> x2.0 -> +R",
                   "l2": (f"inputs larger than L2: steps rotate over {HEADLINE_COPIES} copies of the inputs and "
                          f"output ({HEADLINE_COPIES} x 58.7 MB), run back to back between one pair of events"),
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU"},
        "roofline": {"bound": "tensor", "achieved": round(achieved, 2), "peak": peaks["bf16"],
                     "peak_src": f"{peaks['src']} bf16 burst", "unit": "TFLOP/s",
                     "frac": round(achieved / peaks["bf16"], 4), "traffic": traffic,
                     "algorithmic_bytes": dense_bytes(MAIN, wl)},
        "e2e": {"value": round(e2e_value, 3), "unit": "TFLOP/s", "ms_per_step": round(ms_e2e, 4),
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "eager": {"ms_per_step": round(ms_eager, 5), "speedup": round(ms_eager / ms, 3),
                  "cublas_gemm_only_ms": round(ms_cublas, 5)},
        "isolated": {"ms_per_step": round(ms_iso, 5),
                     "how": "one step at a time after a 256 MiB L2 flush and a 100 us device sleep"},
        "timing": rot_info,
        "gpu_launches": args.steps,
        "clocks": clocks,
    }
    # -------------------------------------------------- CPU baseline (oracle)
    if rank == 0 and world == 1 and not args.no_cpu:
        line["cpu_baseline"] = cpu_baseline(inp, wl, chain_cpu(MAIN, inp), target_s=args.cpu_seconds)
    # ------------------------------------------------------ other workloads
    if not args.main_only:
        line["workloads"] = other_workloads(args, kf, dev, flush, stream, peaks)
    return line


def chain_cpu(name, inp):
    wl = kf_workloads.WORKLOADS[name]
    return [(kind, {k: (inp[v] if k in ("p0", "p1") else v) for k, v in prm.items()})
            for kind, prm in kf_workloads.chain_spec(wl)]


def cpu_baseline(inp, wl, chain, target_s=8.0):
    """The oracle as it stands, on all host cores, over a bounded sample of rows."""
    import oracle
    oracle.build()
    cores = os.cpu_count() or 1
    rows = 8
    while True:
        t0 = time.perf_counter()
        oracle.fused_gemm(inp["X"], inp["W"], chain, rows=list(range(rows)), nthreads=cores)
        dt = time.perf_counter() - t0
        if dt >= target_s / 4 or rows >= wl.M:
            break
        rows = min(wl.M, max(rows * 2, int(rows * target_s / max(dt, 1e-3) / 2)))
    flops = 2.0 * rows * wl.N * wl.K
    return {"value": round(flops / dt / 1e12, 6), "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
            "sample": f"{rows} of {wl.M} rows of {wl.name} (fp64 C, {dt:.2f} s)"}


def dense_eager_fns(name, d):
    """Unfused torch eager (separate launches per op) and the bare GEMM (cuBLAS),
    fp32 with TF32 off."""
    X, W = d["X"], d["W"]
    if name == "fp32_relu_linear":
        return (lambda: F.relu(F.linear(X, W, d["b"]))), (lambda: torch.matmul(X, W.t()))
    return eager_dense(name, d), (lambda: torch.matmul(X, W.t()))


def cpu_oracle_moe(m_cpu, logits_cpu, T, k, target_s):
    """The oracle's MoE FFN as it stands on all host cores, on a bounded sample of
    tokens; TFLOP/s counted over the sampled tokens' routed rows."""
    import oracle
    oracle.build()
    cores = os.cpu_count() or 1
    r = oracle.moe_route(logits_cpu, k)
    H = m_cpu["W_down"].shape[1]
    I = m_cpu["W_gu"].shape[1] // 2
    n = min(T, cores)
    while True:
        t0 = time.perf_counter()
        oracle.moe_ffn(m_cpu["X"], m_cpu["W_gu"], m_cpu["W_down"], r["topk_ids"], r["topk_w"],
                       tokens=list(range(n)), nthreads=cores)
        dt = time.perf_counter() - t0
        if dt >= target_s / 4 or n >= T:
            break
        n = min(T, max(n * 2, int(n * target_s / max(dt, 1e-3) / 2)))
    flops = 2.0 * n * k * (2 * I * H + H * I)
    return {"value": round(flops / dt / 1e12, 6), "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
            "sample": f"{n} of {T} tokens (fp64 C, {dt:.2f} s)"}


def roofline_block(flops, byts, ms, peaks, traffic=None):
    """Roofline of one step: tensor-bound (FLOP / bf16 peak) or HBM-bound (bytes /
    copy peak), whichever takes longer at the peaks."""
    t_flop = flops / (peaks["bf16"] * 1e12)
    t_mem = byts / (peaks["hbm"] * 1e9)
    if t_flop >= t_mem:
        ach = flops / (ms * 1e-3) / 1e12
        return {"bound": "tensor", "achieved": round(ach, 2), "peak": peaks["bf16"],
                "peak_src": f"{peaks['src']} bf16 burst", "unit": "TFLOP/s", "frac": round(ach / peaks["bf16"], 4),
                "traffic": traffic, "algorithmic_bytes": byts}
    ach = byts / (ms * 1e-3) / 1e9
    return {"bound": "hbm", "achieved": round(ach, 1), "peak": peaks["hbm"], "peak_src": f"{peaks['src']} copy",
            "unit": "GB/s", "frac": round(ach / peaks["hbm"], 4), "traffic": traffic, "algorithmic_bytes": byts}


def dense_config_block(name, args, kf, dev, flush, stream, peaks, steps):
    """One dense configuration with its full record: isolated device time, the
    roofline of its kernel, unfused eager and bare-GEMM baselines, the end-to-end
    time through the public API from pinned host buffers, and the oracle on the
    host cores over a bounded row sample."""
    import ctypes
    wl, inp, d, chain = dense_setup(name, dev)
    M, N, K = wl.M, wl.N, wl.K
    flops = 2.0 * M * N * K
    keep = []
    need = kf.lib().kf_fused_gemm_workspace(M, N, K, ctypes.byref(kf.make_epilogue(chain, keep)))
    ws = kf.new_workspace(need, dev) if need else None
    red = any(kk in kf.ROW_REDUCTIONS for kk, _ in chain)
    out_dt = torch.float32 if (red or wl.dtype == "f32") else torch.bfloat16
    out = torch.empty((M,) if red else (M, N), dtype=out_dt, device=dev)
    fn = lambda: kf.fused_gemm(d["X"], d["W"], chain, out=out, workspace=ws)
    prev = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    try:
        ms = time_steps(fn, steps, args.warmup, flush, stream)
        eager, gemm = dense_eager_fns(name, d)
        ms_e = time_steps(eager, steps, args.warmup, flush, stream)
        ms_c = time_steps(gemm, steps, args.warmup, flush, stream)
    finally:
        torch.backends.cuda.matmul.allow_tf32 = prev
    hin = {k2: v.pin_memory() for k2, v in inp.items()}
    hout = torch.empty(out.shape, dtype=out.dtype).pin_memory()

    def e2e():
        for k2 in hin:
            d[k2].copy_(hin[k2], non_blocking=True)
        kf.fused_gemm(d["X"], d["W"], chain, out=out, workspace=ws)
        hout.copy_(out, non_blocking=True)

    ms_e2e = time_steps(e2e, max(3, steps // 2), args.warmup, flush, stream, host_slack=False)
    h2d = sum(v.numel() * v.element_size() for v in hin.values())
    d2h = hout.numel() * hout.element_size()
    byts = dense_bytes(name, wl)
    rec = {"workload": name, "M": M, "N": N, "K": K, "ms": round(ms, 5),
           "tflops": round(flops / ms / 1e9, 3),
           "roofline": roofline_block(flops, byts, ms, peaks, stored_traffic(name)),
           "eager_ms": round(ms_e, 5), "speedup_vs_eager": round(ms_e / ms, 3),
           "gemm_only_ms": round(ms_c, 5),
           "e2e": {"value": round(flops / ms_e2e / 1e9, 3), "unit": "TFLOP/s", "ms_per_step": round(ms_e2e, 4),
                   "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
           "l2": "256 MiB written between steps (cold L2 for every step)",
           "launches_per_step": 2 if red else 1}
    if name == "fp32_relu_linear":
        rec["us"] = round(ms * 1e3, 2)
        rec["eager_us"] = round(ms_e * 1e3, 2)
        rec["note"] = "fp32 FFMA path (exact fp32); eager and the bare GEMM with TF32 off"
    if not args.no_cpu:
        rec["cpu_baseline"] = cpu_baseline(inp, wl, chain_cpu(name, inp), target_s=args.cpu_seconds / 2)
    del d, inp, hin
    return rec


def moe_config_block(T, m, args, kf, dev, flush, stream, peaks, steps, m_cpu):
    """The routed MoE FFN at T tokens (32 experts, top-4, H = I = 2880): device
    time, roofline (HBM-bound weight streaming at decode, tensor-bound at
    prefill), unfused eager, end to end (tokens and logits in, output out; the
    weights stay resident as in serving) and the oracle on a token sample."""
    E, k, H, I = 32, 4, 2880, 2880
    g = torch.Generator("cpu").manual_seed(0)
    Xc = torch.randn(T, H, generator=g).to(torch.bfloat16)
    lc = torch.randn(T, E, generator=g)
    X, logits = Xc.to(dev), lc.to(dev)
    ws = kf.new_workspace(kf.moe_ffn_workspace_bytes(T, H, I, E, k), dev)
    out = torch.empty(T, H, dtype=torch.bfloat16, device=dev)
    fn = lambda: kf.moe_ffn(X, logits, m["W_gu"], m["W_down"], k, out=out, workspace=ws)
    ms = time_steps(fn, steps, args.warmup, flush, stream)
    ms_e = time_steps(lambda: moe_eager(X, logits, m["W_gu"], m["W_down"], k), max(3, steps // 2),
                      args.warmup, flush, stream)
    hX, hl = Xc.pin_memory(), lc.pin_memory()
    hout = torch.empty(T, H, dtype=torch.bfloat16).pin_memory()

    def e2e():
        X.copy_(hX, non_blocking=True)
        logits.copy_(hl, non_blocking=True)
        kf.moe_ffn(X, logits, m["W_gu"], m["W_down"], k, out=out, workspace=ws)
        hout.copy_(out, non_blocking=True)

    ms_e2e = time_steps(e2e, max(3, steps // 2), args.warmup, flush, stream, host_slack=False)
    ids = torch.topk(logits, k, dim=1).indices
    touched = int(torch.unique(ids).numel())
    wbytes = touched * (2 * I * H + H * I) * 2
    byts = wbytes + 2 * T * H * 2 + 4 * T * E
    flops = 2.0 * T * k * (2 * I * H + H * I)
    rec = {"workload": f"moe_ffn_T{T}", "T": T, "H": H, "I": I, "E": E, "k": k, "ms": round(ms, 5),
           "tflops": round(flops / ms / 1e9, 2), "gbs": round(byts / ms / 1e6, 1),
           "roofline": roofline_block(flops, byts, ms, peaks, stored_traffic(f"moe_T{T}")),
           "experts_touched": touched, "eager_ms": round(ms_e, 5), "speedup_vs_eager": round(ms_e / ms, 3),
           "e2e": {"value": round(flops / ms_e2e / 1e9, 3), "unit": "TFLOP/s", "ms_per_step": round(ms_e2e, 4),
                   "h2d_bytes_per_step": hX.numel() * 2 + hl.numel() * 4, "d2h_bytes_per_step": hout.numel() * 2},
           "l2": "256 MiB written between steps; the 1.59 GB of expert weights exceed L2 anyway",
           "launches_per_step": 6}
    if not args.no_cpu:
        mc = dict(X=Xc, W_gu=m_cpu["W_gu"], W_down=m_cpu["W_down"])
        rec["cpu_baseline"] = cpu_oracle_moe(mc, lc, T, k, args.cpu_seconds / 2)
    return rec


def other_workloads(args, kf, dev, flush, stream, peaks):
    res = {}
    steps = max(3, min(args.steps, 20))
    for name in ("fp32_relu_linear", "bf16_scale_rowlse", "bf16_groupnorm_swish"):
        res[name] = dense_config_block(name, args, kf, dev, flush, stream, peaks, steps)
    E, k, H, I = 32, 4, 2880, 2880
    gd = torch.Generator(dev).manual_seed(1)
    m = dict(W_gu=(torch.randn(E, 2 * I, H, generator=gd, device=dev) * 0.02).to(torch.bfloat16),
             W_down=(torch.randn(E, H, I, generator=gd, device=dev) * 0.02).to(torch.bfloat16))
    m_cpu = None if args.no_cpu else {kk: v.cpu() for kk, v in m.items()}
    for T in (64, 4096):
        res[f"moe_T{T}"] = moe_config_block(T, m, args, kf, dev, flush, stream, peaks, steps, m_cpu)
    del m_cpu
    # MoE block tail at decode: residual add + RMSNorm fused into the MoE finalize,
    # against the same MoE FFN followed by torch's add and rms_norm
    T = 64
    g = torch.Generator("cpu").manual_seed(0)
    X = torch.randn(T, H, generator=g).to(torch.bfloat16).to(dev)
    logits = torch.randn(T, E, generator=g).to(dev)
    R = torch.randn(T, H, generator=g).to(torch.bfloat16).to(dev)
    gamma = (torch.rand(H, generator=g) + 0.5).to(torch.bfloat16).to(dev)
    ws = kf.new_workspace(kf.moe_ffn_workspace_bytes(T, H, I, E, k), dev)
    y_out = torch.empty(T, H, dtype=torch.bfloat16, device=dev)
    r_out = torch.empty(T, H, dtype=torch.bfloat16, device=dev)
    fused = lambda: kf.moe_ffn_add_rmsnorm(X, logits, m["W_gu"], m["W_down"], k, R, gamma, 1e-5, out=y_out,
                                           r_out=r_out, workspace=ws)
    def unfused():
        y = kf.moe_ffn(X, logits, m["W_gu"], m["W_down"], k, workspace=ws)
        h = R + y
        return F.rms_norm(h, (H,), weight=gamma, eps=1e-5), h
    ms = time_steps(fused, steps, args.warmup, flush, stream)
    ms_u = time_steps(unfused, steps, args.warmup, flush, stream)
    touched = int(torch.unique(torch.topk(logits, k, dim=1).indices).numel())
    byts = touched * (2 * I * H + H * I) * 2 + T * H * 2 * 4 + 4 * T * E
    res["moe_T64_add_rmsnorm"] = {"ms": round(ms, 5), "gbs": round(byts / ms / 1e6, 1), "bound": "hbm",
                                  "roofline_frac": round(byts / (peaks["hbm"] * 1e9) * 1e3 / ms, 4),
                                  "unfused_ms": round(ms_u, 5), "speedup_vs_unfused": round(ms_u / ms, 3),
                                  "launches_per_step": 6}
    # the gpt-oss expert activation (per-expert biases, clamped gated SwiGLU) at
    # decode, against the plain SwiGLU path on the same inputs
    b = kf_workloads.moe_bias_generate(E, H, I, seed=0)
    act = dict(kf_workloads.GPT_OSS_ACT, b_gu=b["b_gu"].to(dev), b_down=b["b_down"].to(dev))
    g = torch.Generator("cpu").manual_seed(0)
    X = torch.randn(T, H, generator=g).to(torch.bfloat16).to(dev)
    logits = torch.randn(T, E, generator=g).to(dev)
    gated = lambda: kf.moe_ffn(X, logits, m["W_gu"], m["W_down"], k, out=y_out, workspace=ws, act=act)
    plain = lambda: kf.moe_ffn(X, logits, m["W_gu"], m["W_down"], k, out=y_out, workspace=ws)
    ms = time_steps(gated, steps, args.warmup, flush, stream)
    ms_p = time_steps(plain, steps, args.warmup, flush, stream)
    touched = int(torch.unique(torch.topk(logits, k, dim=1).indices).numel())
    byts = touched * ((2 * I * H + H * I) * 2 + (2 * I + H) * 2) + 2 * T * H * 2 + 4 * T * E
    res["moe_T64_gptoss_act"] = {"ms": round(ms, 5), "gbs": round(byts / ms / 1e6, 1), "bound": "hbm",
                                 "roofline_frac": round(byts / (peaks["hbm"] * 1e9) * 1e3 / ms, 4),
                                 "plain_swiglu_ms": round(ms_p, 5), "launches_per_step": 6}
    # fp32 operands on the tensor cores (3xTF32) against cuBLAS's fp32 GEMM and
    # our exact FFMA path; roofline: the tf32 rate (half the bf16 peak) over 3
    Mf = Nf = Kf = 4096
    g = torch.Generator("cpu").manual_seed(0)
    Xf = torch.randn(Mf, Kf, generator=g).to(dev)
    Wf = (torch.randn(Nf, Kf, generator=g) / Kf ** 0.5).to(dev)
    bf = torch.randn(Nf, generator=g).to(dev)
    yf = torch.empty(Mf, Nf, device=dev)
    chf = [("bias", {"p0": bf}), ("relu", {})]
    ms = time_steps(lambda: kf.fused_gemm(Xf, Wf, chf, out=yf, f32_mode="tf32x3"), steps, args.warmup, flush, stream)
    ms_ffma = time_steps(lambda: kf.fused_gemm(Xf, Wf, chf, out=yf, f32_mode="ffma"), 3, 1, flush, stream)
    prev = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    ms_c = time_steps(lambda: torch.matmul(Xf, Wf.t()), steps, args.warmup, flush, stream)
    torch.backends.cuda.matmul.allow_tf32 = prev
    flops = 2.0 * Mf * Nf * Kf
    peak3 = peaks["bf16"] / 2 / 3
    res["fp32_bias_relu_4096_3xtf32"] = {"tflops": round(flops / ms / 1e9, 2), "ms": round(ms, 5), "bound": "tensor",
                                         "roofline_frac": round(flops / ms / 1e9 / peak3, 4),
                                         "roofline_peak_tflops": round(peak3, 1), "ffma_path_ms": round(ms_ffma, 5),
                                         "cublas_fp32_gemm_only_ms": round(ms_c, 5), "launches_per_step": 1}
    del Xf, Wf, yf
    # attention input projection with bias + rotary embedding + KV-cache write in
    # its epilogue (gpt-oss-20b shape), against our GEMM + bias followed by torch's
    # rotation and cache copies, and cuBLAS's GEMM alone
    sh = kf_workloads.QKV_SHAPE
    nq, nkv, dh, Hq = sh["nq"], sh["nkv"], sh["d"], sh["H"]
    Nq = (nq + 2 * nkv) * dh
    for T in (1, 64, 4096):
        inp = kf_workloads.qkv_generate(T, seed=0, prefill=T > 128, cache_rows=max(8192, T))
        g = {k2: v.to(dev) for k2, v in inp.items() if k2 != "rows"}
        rows = int(inp["rows"])
        kc = torch.zeros(rows, nkv * dh, dtype=torch.bfloat16, device=dev)
        vc = torch.zeros_like(kc)
        q = torch.empty(T, nq * dh, dtype=torch.bfloat16, device=dev)
        y = torch.empty(T, Nq, dtype=torch.bfloat16, device=dev)
        byts = Nq * Hq * 2 + T * Hq * 2 + Nq * 2 + T * Nq * 2 + 2 * T * (dh // 2) * 4
        flops = 2.0 * T * Nq * Hq
        # steps rotate over copies of the inputs, together more than twice L2
        ncop = max(2, -(-300_000_000 // byts))
        gs = [g] + [{k2: v.clone() for k2, v in g.items()} for _ in range(ncop - 1)]

        def make_fused(gc):
            return lambda: kf.qkv_rope_kv(gc["X"], gc["W"], gc["b"], gc["positions"], gc["cache_rows"], gc["cos"],
                                          gc["sin"], nq, nkv, dh, kc, vc, q_out=q)

        def make_unfused(gc):
            pos, crow = gc["positions"].long(), gc["cache_rows"].long()

            def unfused():
                kf.fused_gemm(gc["X"], gc["W"], [("bias", {"p0": gc["b"]})], out=y)
                hd = y.view(T, nq + 2 * nkv, dh)
                c, sn = gc["cos"][pos][:, None, :], gc["sin"][pos][:, None, :]
                x = hd[:, :nq + nkv].float()
                a, b = x[..., :dh // 2], x[..., dh // 2:]
                r = torch.cat([a * c - b * sn, b * c + a * sn], -1).to(torch.bfloat16)
                q.copy_(r[:, :nq].reshape(T, -1))
                kc.index_copy_(0, crow, r[:, nq:].reshape(T, -1))
                vc.index_copy_(0, crow, hd[:, nq + nkv:].reshape(T, -1))
            return unfused

        ms, _ = time_steps_rotating([make_fused(gc) for gc in gs], steps, args.warmup, stream)
        ms_u, _ = time_steps_rotating([make_unfused(gc) for gc in gs], steps, args.warmup, stream)
        ms_c, _ = time_steps_rotating([(lambda gc=gc: torch.matmul(gc["X"], gc["W"].t())) for gc in gs], steps,
                                      args.warmup, stream)
        ms_iso = time_steps(make_fused(g), steps, args.warmup, flush, stream)
        t_roof = max(flops / (peaks["bf16"] * 1e12), byts / (peaks["hbm"] * 1e9)) * 1e3
        bound = "hbm" if byts / (peaks["hbm"] * 1e9) > flops / (peaks["bf16"] * 1e12) else "tensor"
        res[f"qkv_rope_kv_T{T}"] = {"tflops": round(flops / ms / 1e9, 2), "gbs": round(byts / ms / 1e6, 1),
                                   "ms": round(ms, 5), "bound": bound, "roofline_frac": round(t_roof / ms, 4),
                                   "path": "clusters splitting K" if T <= 64 else "tcgen05 tiles",
                                   "unfused_ms": round(ms_u, 5),
                                   "speedup_vs_unfused": round(ms_u / ms, 3), "cublas_gemm_only_ms": round(ms_c, 5),
                                   "isolated_ms": round(ms_iso, 5),
                                   "l2": f"steps rotate over {ncop} copies of the inputs, back to back",
                                   "launches_per_step": 1}
        del gs
        del g, inp, kc, vc
    return res


def profile_workload(name, dev, reps):
    """Run one workload through the public API `reps` times (no timing): the
    command that ncu launch lists and captures of that workload are taken on."""
    import paper_2606_02963_gb300 as kf
    if name.startswith("fp32_tf32x3_"):
        n = int(name[len("fp32_tf32x3_"):])
        g = torch.Generator("cpu").manual_seed(0)
        X = torch.randn(n, n, generator=g).to(dev)
        W = (torch.randn(n, n, generator=g) / n ** 0.5).to(dev)
        b = torch.randn(n, generator=g).to(dev)
        for _ in range(reps):
            kf.fused_gemm(X, W, [("bias", {"p0": b}), ("relu", {})], f32_mode="tf32x3")
    elif name.startswith("qkv_T"):
        T = int(name[5:])
        sh = kf_workloads.QKV_SHAPE
        inp = kf_workloads.qkv_generate(T, seed=0, prefill=T > 128, cache_rows=max(8192, T))
        g = {k: v.to(dev) for k, v in inp.items() if k != "rows"}
        kc = torch.zeros(int(inp["rows"]), sh["nkv"] * sh["d"], dtype=torch.bfloat16, device=dev)
        vc = torch.zeros_like(kc)
        for _ in range(reps):
            kf.qkv_rope_kv(g["X"], g["W"], g["b"], g["positions"], g["cache_rows"], g["cos"], g["sin"], sh["nq"],
                           sh["nkv"], sh["d"], kc, vc)
    elif name.startswith("moe_T"):
        T, E, k, H, I = int(name[5:]), 32, 4, 2880, 2880
        g = torch.Generator("cpu").manual_seed(0)
        X = torch.randn(T, H, generator=g).to(torch.bfloat16).to(dev)
        logits = torch.randn(T, E, generator=g).to(dev)
        gd = torch.Generator(dev).manual_seed(1)
        Wgu = (torch.randn(E, 2 * I, H, generator=gd, device=dev) * 0.02).to(torch.bfloat16)
        Wd = (torch.randn(E, H, I, generator=gd, device=dev) * 0.02).to(torch.bfloat16)
        for _ in range(reps):
            kf.moe_ffn(X, logits, Wgu, Wd, k)
    else:
        wl, inp, d, chain = dense_setup(name, dev)
        for _ in range(reps):
            kf.fused_gemm(d["X"], d["W"], chain)
    torch.cuda.synchronize()
    print(f"profiled {name} x{reps}")


def run_reference(args, rank, world):
    """The oracle as it stands on the host cores, on bounded row samples of the
    headline workload (one sample per step)."""
    import oracle
    oracle.build()
    wl = kf_workloads.WORKLOADS[MAIN]
    inp = kf_workloads.generate(MAIN, seed=0)
    chain = chain_cpu(MAIN, inp)
    cores = os.cpu_count() or 1
    rows = args.ref_rows
    sample = lambda i: [(i * rows + r) % wl.M for r in range(rows)]
    for i in range(args.warmup):
        oracle.fused_gemm(inp["X"], inp["W"], chain, rows=sample(i), nthreads=cores)
    t0 = time.perf_counter()
    for i in range(args.steps):
        oracle.fused_gemm(inp["X"], inp["W"], chain, rows=sample(args.warmup + i), nthreads=cores)
    dt = (time.perf_counter() - t0) / args.steps
    flops = 2.0 * rows * wl.N * wl.K
    v = flops / dt / 1e12
    return {"metric": "fused GEMM+tail TFLOP/s & % of GB300 roofline; speedup vs unfused torch eager",
            "impl": "reference", "value": round(v, 6), "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(dt * 1e3, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded)",
            "config": {"workload": MAIN, "M": wl.M, "N": wl.N, "K": wl.K,
                       "chain": "bias -> gelu_tanh -> x2.0 -> +R"},
            "cpu_baseline": {"value": round(v, 6), "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
                             "sample": f"{rows} rows of {wl.M} per step (fp64 C oracle)"},
            "e2e": {"value": round(v, 6), "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="kf", choices=["kf", "reference"])
    ap.add_argument("--main-only", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=8.0)
    ap.add_argument("--ref-rows", type=int, default=16)
    ap.add_argument("--profile-workload", default=None,
                    help="run one workload's calls --steps times, untimed (the command ncu captures of it use): "
                         "bf16_gelu_scale_residual, bf16_scale_rowlse, bf16_groupnorm_swish, moe_T64, moe_T4096, "
                         "qkv_T<tokens> or fp32_tf32x3_<n>")
    args = ap.parse_args()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args, rank, world)), flush=True)
        return
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    if args.profile_workload:
        profile_workload(args.profile_workload, dev, args.steps)
        return
    if world > 1:
        torch.distributed.init_process_group("nccl", device_id=dev)
    line = run_kf(args, rank, world, dev)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
