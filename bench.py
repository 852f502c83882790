#!/usr/bin/env python
"""Benchmark of the Ember optimizer step on GB300 (one JSON line on stdout).

A step is one dense Ember step (row/column reduction, state update, apply)
over one V x D table: by default the large LM head, V = 128256, D = 8192,
bf16 weights, fp32 gradient and state.  Inputs are resident in HBM when the
timed region starts; L2 is flushed between timed steps, outside the per-step
CUDA events: a 512 MiB write, then a 512 MiB read of another buffer, so that
the step starts with a cold L2 that holds no dirty line of the flush.
`value` is algorithmic bytes per step over the mean step time, summed over
ranks (independent replicas: the step has no cross-GPU exchange on one table
held whole by each GPU).  The same line
carries one sub-object per workload of the method (`configs`: the 1024 x 64
fp32 table, the 32000 x 4096 and 151936 x 896 bf16 tables, the sparse
262144 x 2048 step with 32768 ids, and the LM head), each with its step
time, its GB/s and the roofline of its dominant kernel, the fused LM-head
step, the row-only variant and the CPU oracle on one core and on all cores.

  python bench.py [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

--impl reference times the CPU oracle (plain C; its OpenMP build on all host
cores, which gives the same bits) on a bounded row sample of the same
workload: the paper ships no implementation to compare with, so that is the
reference arm.
"""
import argparse
import json
import os
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

DEFAULT_WORKLOAD = "dense_lmhead_v128256_d8192_bf16"
METRIC = "Ember step GB/s and % of GB300 HBM roofline (dense and sparse), params/sec"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
L2_FLUSH_BYTES = 512 << 20
L2_NOTE = "flushed between steps (512 MiB write, then 512 MiB read; outside the events)"


class L2Flush:
    """Evicts L2 between timed steps: writes one buffer four times the size of
    L2, then reads another of the same size, so that the write's dirty lines
    are written back here and not inside the next step."""

    def __init__(self, dev):
        import torch
        self.w = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
        self.r = torch.ones(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
        self.out = torch.empty((), dtype=torch.float32, device=dev)

    def __call__(self):
        import torch
        self.w.zero_()
        torch.amax(self.r, dim=0, out=self.out)

# DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) per launch of a
# dominant kernel, from an ncu capture of the kernel as it is now, with where
# it came from.  A kernel that changes gets None here until it is captured
# again.
TRAFFIC = {
    # the 32768 x 8192 quarter table measured 2.1156 GB per launch (mean of
    # two launches); every row of G and W is read once and W written once,
    # so the traffic is scaled by rows
    ("k_apply_dense", "dense_lmhead_v128256_d8192_bf16"): (
        int(2.1156e9 * 128256 / 32768),
        "ncu dram__bytes_read.sum + dram__bytes_write.sum of k_apply_dense on the 32768 x 8192 table, "
        "2.1156 GB per launch, scaled by rows (2026-12-02, reciprocal-multiply division)"),
    ("k_sp_segsum", "sparse_v262144_d2048_bf16_n32768"): (
        274328064, "ncu dram__bytes_read.sum + dram__bytes_write.sum of k_sp_segsum on this workload "
                   "(2026-12-02, full-batch loop)"),
    # k_lmhead_grad: the re-reads of its operands do not grow in proportion
    # to the rows (3.2 x the algorithmic reads at 32768 rows), so no
    # full-size figure is derived from the quarter-size capture
    ("k_lmhead_grad", "lmhead_grad_v128256_d8192_t4096_bf16"): None,
}

def wbytes(wl):
    return 2 if wl.wdtype == "bf16" else 4


def step_bytes(wl):
    """Algorithmic bytes of one dense step: G read twice (every update needs
    the column statistics of all rows), W read and written once, the V + D
    state read and written once."""
    V, D, w = wl.V, wl.D, wbytes(wl)
    return (8 + 2 * w) * V * D + 8 * (V + D)


def kernel_bytes(wl):
    """Algorithmic bytes per launch of each kernel of the dense step."""
    V, D, w = wl.V, wl.D, wbytes(wl)
    return {"reduce": 4 * V * D + 8 * V, "state": 8 * D, "apply": (4 + 2 * w) * V * D + 4 * (V + D)}


def sparse_bytes(wl, U):
    """Algorithmic bytes of one sparse step with U distinct ids: the grad
    rows read once, the ids read once, the summed rows visited a second time
    (written and read back, or the rows re-read, whichever is less), the
    touched W rows read and written, r read and written for all V rows."""
    N, D, V, w = wl.N, wl.D, wl.V, wbytes(wl)
    return 4 * N * D + 8 * N + min(8 * U * D, 4 * N * D) + 2 * w * U * D + 8 * V + 8 * D


SPARSE_KERNELS = ("tile_sort", "rank", "scatter", "segments", "segsum", "carry",
                  "rows_and_state", "apply")
TRACE_EVERY = 4  # every 4th timed step records kernel-boundary events


def traced_steps(steps):
    """Timed steps that record kernel boundaries: every TRACE_EVERY-th one,
    and never all of them (at least one untraced step times the whole step)."""
    if steps < 2:
        raise SystemExit("--steps must be at least 2")
    t = [k for k in range(steps) if k % TRACE_EVERY == TRACE_EVERY - 1]
    return t or [steps - 1]


def traffic_of(kernel, name):
    """{"traffic": bytes or None, "traffic_source": where they came from}."""
    t = TRAFFIC.get((kernel, name))
    if t is None:
        return {"traffic": None, "traffic_source": "not captured for this kernel version"}
    return {"traffic": t[0], "traffic_source": t[1]}


def hbm_roofline(kernel, bytes_per_launch, ms_per_launch, wl_name):
    peak, peak_kind = measured_hbm_peak()
    ach = bytes_per_launch / (ms_per_launch * 1e-3) / 1e9
    return {"bound": "hbm", "kernel": kernel, "achieved": ach, "peak": peak, "unit": "GB/s",
            "frac": ach / peak, "peak_kind": peak_kind, "algorithmic_bytes_per_launch": bytes_per_launch,
            **traffic_of(kernel, wl_name)}


def run_dense(wl, dev, steps, warmup, flush, seed=0, clocks_for=None):
    """Times ember_step_dense on one workload (L2 flushed between steps).
    Untraced steps time the whole step; for a table that runs as three
    launches, every TRACE_EVERY-th step records events at the kernel
    boundaries for the per-kernel times (a small table runs as one cluster
    launch, whose time is the step's)."""
    import torch
    from paper_2607_01455_gb300 import synth
    from paper_2607_01455_gb300.ember import Ember
    W = synth.init_weights(wl, seed, dev)
    G = synth.dense_grad(wl, seed, 1, dev)
    emb = Ember(wl.V, wl.D, wdtype=wl.wdtype, device=dev)
    vec = wl.D % 4 == 0
    launches = emb.dense_step_launches(vec)
    npan = emb.column_panels(vec)
    three = launches == 2 * npan + 1
    t = 0
    warm_ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    for i in range(warmup):
        t += 1
        flush()
        emb.trace(warm_ev if (three and i % 2) else [])
        emb.step_dense(W, G, wl.lr, t)
    torch.cuda.synchronize()
    step_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    traced = traced_steps(steps) if three else []
    kern_ev = {k: [torch.cuda.Event(enable_timing=True) for _ in range(4)] for k in traced}
    stream = torch.cuda.current_stream(dev)
    torch.cuda.synchronize()
    wall0 = time.perf_counter()
    sampler = clocks_for if clocks_for is not None else _NullClocks()
    with sampler:
        for k in range(steps):
            t += 1
            flush()
            emb.trace(kern_ev.get(k, []))
            step_ev[k][0].record(stream)
            emb.step_dense(W, G, wl.lr, t)
            step_ev[k][1].record(stream)
        torch.cuda.synchronize()
    wall = time.perf_counter() - wall0
    emb.trace([])
    if emb.device_status() != 0:
        raise SystemExit(f"device status after the {wl.name} steps")
    plain = [k for k in range(steps) if k not in kern_ev]
    ms = sum(step_ev[k][0].elapsed_time(step_ev[k][1]) for k in plain) / len(plain)
    B = step_bytes(wl)
    peak, _ = measured_hbm_peak()
    out = {"workload": wl.name, "V": wl.V, "D": wl.D, "w_dtype": wl.wdtype, "steps": steps,
           "ms_per_step": ms, "value": B / (ms * 1e-3) / 1e9, "unit": "GB/s", "algorithmic_bytes": B,
           "frac_of_measured_hbm": B / (ms * 1e-3) / 1e9 / peak,
           "frac_of_nominal_8TBs": B / (ms * 1e-3) / 1e9 / NOMINAL_HBM_GBS,
           "params_per_s": wl.V * wl.D / (ms * 1e-3), "launches_per_step": launches,
           "gpu_launches": launches * steps, "wall_s_timed_region": wall}
    if three:
        kb = kernel_bytes(wl)
        per = {"reduce": [], "state": [], "apply": [], "traced_step": []}
        for ev in kern_ev.values():
            per["reduce"].append(ev[0].elapsed_time(ev[1]))
            per["state"].append(ev[1].elapsed_time(ev[2]))
            per["apply"].append(ev[2].elapsed_time(ev[3]))
            per["traced_step"].append(ev[0].elapsed_time(ev[3]))
        mean = {k: sum(v) / len(v) for k, v in per.items()}
        out["kernels"] = {k: {"ms": mean[k], "gbs": kb[k] / (mean[k] * 1e-3) / 1e9}
                          for k in ("reduce", "state", "apply")}
        out["ms_per_step_traced"] = mean["traced_step"]
        # the apply pass is the dominant kernel (2/3 of the bytes); with
        # column panels its launches are per panel and the figures per pass
        out["roofline"] = hbm_roofline("k_apply_dense", kb["apply"], mean["apply"], wl.name)
        if npan > 1:
            out["roofline"]["launches_per_pass"] = npan
        out["timing"] = (f"step time: CUDA events around each untraced step; kernel times: every "
                         f"{TRACE_EVERY}th step records events at kernel boundaries")
    else:
        # one cluster launch: G read from HBM once, W read and written, the
        # state read and written once
        w = wbytes(wl)
        kbytes = (4 + 2 * w) * wl.V * wl.D + 8 * (wl.V + wl.D)
        out["kernels"] = {"cluster": {"ms": ms, "gbs": kbytes / (ms * 1e-3) / 1e9}}
        out["roofline"] = hbm_roofline("k_dense_cluster", kbytes, ms, wl.name)
        out["timing"] = "CUDA events around each step (one kernel launch per step)"
    return out


class _NullClocks:
    def __enter__(self):
        return self

    def __exit__(self, *exc):
        return False


def run_sparse(wl, dev, steps, warmup, flush, seed=0):
    """Times the sparse step on one fixed batch (L2 flushed between steps)."""
    import torch
    from paper_2607_01455_gb300 import synth
    from paper_2607_01455_gb300.ember import Ember
    W = synth.init_weights(wl, seed, dev)
    ids, rows = synth.sparse_batch(wl, seed, 1, dev)
    U = int(torch.unique(ids).numel())
    emb = Ember(wl.V, wl.D, wdtype=wl.wdtype, max_sparse_N=wl.N, device=dev)
    names = SPARSE_KERNELS
    nk = len(names)
    t = 0
    warm = [torch.cuda.Event(enable_timing=True) for _ in range(nk + 1)]
    for i in range(warmup):
        t += 1
        flush()
        emb.trace(warm if i % 2 else [])
        emb.step_sparse(W, ids, rows, wl.lr, t)
    torch.cuda.synchronize()
    # untraced steps time the whole step (kernels overlap their launches);
    # every TRACE_EVERY-th step records kernel boundaries instead
    step_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(steps)]
    traced = traced_steps(steps)
    kern_ev = {k: [torch.cuda.Event(enable_timing=True) for _ in range(nk + 1)] for k in traced}
    for k in range(steps):
        t += 1
        flush()
        emb.trace(kern_ev.get(k, []))
        step_ev[k][0].record()
        emb.step_sparse(W, ids, rows, wl.lr, t)
        step_ev[k][1].record()
    torch.cuda.synchronize()
    emb.trace([])
    if emb.device_status() != 0:
        raise SystemExit("device status after the sparse steps")
    plain = [k for k in range(steps) if k not in kern_ev]
    per = {name: sum(kern_ev[k][i].elapsed_time(kern_ev[k][i + 1]) for k in traced) / len(traced)
           for i, name in enumerate(names)}
    ms = sum(step_ev[k][0].elapsed_time(step_ev[k][1]) for k in plain) / len(plain)
    ms_traced = sum(step_ev[k][0].elapsed_time(step_ev[k][1]) for k in traced) / len(traced)
    # the same step replayed from a CUDA graph (how a training loop would run it)
    side = torch.cuda.Stream(dev)
    side.wait_stream(torch.cuda.current_stream(dev))
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=side):
        emb.step_sparse(W, ids, rows, wl.lr, t + 1, stream=side)
    gev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for k in range(steps):
        flush()
        gev[k][0].record()
        graph.replay()
        gev[k][1].record()
    torch.cuda.synchronize()
    ms_graph = sum(a.elapsed_time(b) for a, b in gev) / steps
    B = sparse_bytes(wl, U)
    kb = sparse_kernel_bytes(wl, U)
    peak, _ = measured_hbm_peak()
    return {"workload": wl.name, "ms_per_step_graph": ms_graph, "V": wl.V, "D": wl.D, "N": wl.N, "unique_ids": U,
            "roofline": hbm_roofline("k_sp_segsum", kb["segsum"], per["segsum"], wl.name),
            "frac_of_measured_hbm": B / (ms * 1e-3) / 1e9 / peak,
            "frac_of_nominal_8TBs": B / (ms * 1e-3) / 1e9 / NOMINAL_HBM_GBS,
            "ms_per_step": ms, "value": B / (ms * 1e-3) / 1e9, "unit": "GB/s",
            "algorithmic_bytes": B, "touched_params_per_s": U * wl.D / (ms * 1e-3),
            "occurrence_params_per_s": wl.N * wl.D / (ms * 1e-3),
            "kernels_ms": per, "ms_per_step_traced": ms_traced, "gpu_launches": nk * steps}


def run_row_only(wl, dev, steps, warmup, flush, W, G):
    """The row-only variant (vtil = rhat, one fused pass over G and W) on the
    same table: 4VD + 2wVD + 8(V + D) algorithmic bytes per step."""
    import torch
    from paper_2607_01455_gb300.ember import Ember
    emb = Ember(wl.V, wl.D, wdtype=wl.wdtype, variant="row", device=dev)
    t = 0
    for _ in range(warmup):
        t += 1
        flush()
        emb.step_dense(W, G, wl.lr, t)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for k in range(steps):
        t += 1
        flush()
        ev[k][0].record()
        emb.step_dense(W, G, wl.lr, t)
        ev[k][1].record()
    torch.cuda.synchronize()
    if emb.device_status() != 0:
        raise SystemExit("device status after the row-only steps")
    ms = sum(a.elapsed_time(b) for a, b in ev) / steps
    B = (4 + 2 * wbytes(wl)) * wl.V * wl.D + 8 * (wl.V + wl.D)
    npan = emb.column_panels(wl.D % 4 == 0)
    # a table in column panels has no one-pass kernel: reduce, state and
    # apply passes per step, G read twice
    launches = 2 if npan == 1 else 2 * npan + 1
    return {"variant": "row", "ms_per_step": ms, "value": B / (ms * 1e-3) / 1e9, "unit": "GB/s",
            "algorithmic_bytes": B, "params_per_s": wl.V * wl.D / (ms * 1e-3), "gpu_launches": launches * steps,
            "one_pass": npan == 1}


LMHEAD_KERNELS = ["lmhead_grad", "state", "apply"]


def run_lmhead(wl, dev, steps, warmup, flush, seed=0):
    """The LM-head step fused with the producer of its gradient
    (ember_step_lmhead: G = dlogits^T H on the tensor cores with the sums of
    g^2 in the epilogue, then the state and apply passes), against the same
    step built from cuBLAS (torch.mm, fp32 output) and ember_step_dense."""
    import torch
    from paper_2607_01455_gb300 import synth
    from paper_2607_01455_gb300.ember import Ember
    V, D, T = wl.V, wl.D, wl.T
    emb = Ember(V, D, wdtype=wl.wdtype, device=dev)
    W = synth.init_weights(wl, seed, dev)
    G = torch.empty(V, D, device=dev)
    dl, h = synth.lmhead_inputs(V, D, T, seed, 1, dev)
    nk = len(LMHEAD_KERNELS)
    t = 0
    for _ in range(warmup):
        t += 1
        flush()
        emb.step_lmhead(W, dl, h, G, wl.lr, t)
    torch.cuda.synchronize()
    step_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(steps)]
    traced = traced_steps(steps)
    kern_ev = {k: [torch.cuda.Event(enable_timing=True) for _ in range(nk + 1)] for k in traced}
    for k in range(steps):
        t += 1
        flush()
        emb.trace(kern_ev.get(k, []))
        step_ev[k][0].record()
        emb.step_lmhead(W, dl, h, G, wl.lr, t)
        step_ev[k][1].record()
    torch.cuda.synchronize()
    emb.trace([])
    if emb.device_status() != 0:
        raise SystemExit("device status after the LM-head steps")
    plain = [k for k in range(steps) if k not in kern_ev]
    per = {name: sum(kern_ev[k][i].elapsed_time(kern_ev[k][i + 1]) for k in traced) / len(traced)
           for i, name in enumerate(LMHEAD_KERNELS)}
    ms = sum(step_ev[k][0].elapsed_time(step_ev[k][1]) for k in plain) / len(plain)

    # the unfused step: cuBLAS forms G, then the two-pass dense step
    emb2 = Ember(V, D, wdtype=wl.wdtype, device=dev)
    dlT = dl.t()
    try:
        torch.mm(dlT, h, out_dtype=torch.float32)
        gemm = lambda: torch.mm(dlT, h, out_dtype=torch.float32)  # noqa: E731
        cublas_out = "fp32"
    except (TypeError, RuntimeError):
        gemm = lambda: torch.mm(dlT, h).float()  # noqa: E731
        cublas_out = "bf16 then converted"
    for _ in range(warmup):
        t += 1
        flush()
        emb2.step_dense(W, gemm(), wl.lr, t)
    torch.cuda.synchronize()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    for k in range(steps):
        t += 1
        flush()
        ev[k][0].record()
        Gc = gemm()
        ev[k][1].record()
        emb2.step_dense(W, Gc, wl.lr, t)
        ev[k][2].record()
    torch.cuda.synchronize()
    ms_unfused = sum(e[0].elapsed_time(e[2]) for e in ev) / steps
    ms_cublas = sum(e[0].elapsed_time(e[1]) for e in ev) / steps

    flops = 2.0 * V * D * T
    tf = flops / (per["lmhead_grad"] * 1e-3) / 1e12
    tf_cublas = flops / (ms_cublas * 1e-3) / 1e12
    peaks = {}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        peaks = {"burst": float(pk["bf16_tflops"]), "sustained": float(pk["bf16_tflops_sustained"])}
        peak_kind = "measured"
    except Exception:
        peaks = {"burst": 1900.0, "sustained": 1700.0}
        peak_kind = "fallback"
    B_fused = (4 + 4 + 2 * wbytes(wl)) * V * D + 2 * T * (V + D)
    return {"workload": wl.name, "V": V, "D": D, "T": T, "ms_per_step": ms,
            "kernels_ms": per, "gpu_launches": nk * steps,
            "roofline": {"bound": "tensor", "kernel": "k_lmhead_grad", "achieved": tf, "peak": peaks["burst"],
                         "unit": "TFLOP/s", "frac": tf / peaks["burst"],
                         "frac_of_sustained": tf / peaks["sustained"], "peak_kind": peak_kind,
                         "flops_per_launch": flops,
                         **traffic_of("k_lmhead_grad", wl.name),
                         "algorithmic_dram_bytes_per_launch": 2 * T * (V + D) + 4 * V * D},
            "unfused": {"ms_per_step": ms_unfused, "cublas_gemm_ms": ms_cublas, "cublas_tflops": tf_cublas,
                        "cublas_output": cublas_out,
                        "what": "torch.mm(dlogits^T, H) then ember_step_dense (reduce, state, apply)"},
            "speedup_vs_unfused": ms_unfused / ms,
            "hbm_bytes_fused_step": B_fused,
            "what": "ember_step_lmhead: G = dlogits^T H (tcgen05, fp32 G written) with per-tile sums of g^2 "
                    "in the epilogue, state pass, apply pass (G read once)"}


def measured_hbm_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons, sampled every 20 ms."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    # where the raw samples go (EMBER_CLOCK_LOG_DIR, default: the temp dir)
    LOG_DIR = os.environ.get("EMBER_CLOCK_LOG_DIR") or tempfile.gettempdir()

    def __init__(self, gpu_index):
        self.gpu_index = gpu_index
        self.proc = None
        self.path = os.path.join(self.LOG_DIR, f"ember_clocks_gpu{gpu_index}.csv")

    def __enter__(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu_index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=self.out, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.out.close()

    def summary(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        with open(self.path) as f:
            for line in f:
                p = [x.strip() for x in line.split(",")]
                if len(p) >= 9 and p[1].replace(".", "").isdigit():
                    rows.append(p)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        sm = sorted(float(p[1]) for p in rows)
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for p in rows for n, v in zip(names, p[5:9]) if v.lower() == "active"})
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": float(rows[0][2]), "reasons": reasons,
                "samples": len(rows), "power_w_max": max(float(p[3]) for p in rows)}


class OracleSample:
    """The oracle's dense step on the first `rows` rows of the workload (a
    rows x D table drawn with the workload's generator), stepped repeatedly."""

    def __init__(self, wl, rows, seed=0):
        import numpy as np
        import torch
        from paper_2607_01455_gb300 import synth
        sub = synth.Workload(wl.name + "_sample", rows, wl.D, wl.wdtype, 1,
                             zero_frac=wl.zero_frac, heavy_frac=wl.heavy_frac)
        W = synth.init_weights(sub, seed, "cpu")
        self.W = (W.view(torch.int16).numpy().view(np.uint16).copy() if wl.wdtype == "bf16"
                  else W.numpy().copy())
        self.G = synth.dense_grad(sub, seed, 1, "cpu").numpy()
        self.r = np.zeros(rows, np.float32)
        self.c = np.zeros(wl.D, np.float32)
        self.lr, self.t, self.rows = wl.lr, 0, rows
        self.bytes = step_bytes(sub)

    def step(self, all_cores=False):
        """One oracle step; returns its seconds.  all_cores: the OpenMP build
        of the same source on every host core (the same bits)."""
        import oracle
        self.t += 1
        t0 = time.perf_counter()
        oracle.step_dense(self.W, self.G, self.r, self.c, self.lr, self.t, all_cores=all_cores)
        return time.perf_counter() - t0


def host_cores():
    """Threads the all-cores oracle uses: every core this process may run on."""
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def sample_rows_for(wl, seconds, all_cores=False):
    """Rows of a sample whose oracle step takes about `seconds`."""
    probe = 64 if not all_cores else 1024
    smp = OracleSample(wl, min(probe, wl.V))
    smp.step(all_cores)  # the first call loads the library and starts the threads
    dt = smp.step(all_cores)
    return int(max(16, min(wl.V, smp.rows * seconds / max(dt, 1e-6))))


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("gloo")
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def allreduce_max(world, x):
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def run_reference(args, world, rank):
    import oracle
    from paper_2607_01455_gb300 import synth
    wl = synth.WORKLOADS[args.workload]
    if rank != 0:
        return 0
    cores = oracle.threads(host_cores())
    budget = 90.0  # seconds of oracle work for the whole warm-up + timed run
    rows = sample_rows_for(wl, budget / (args.steps + args.warmup), all_cores=True)
    smp = OracleSample(wl, rows)
    for _ in range(args.warmup):
        smp.step(all_cores=True)
    times = [smp.step(all_cores=True) for _ in range(args.steps)]
    sec = sum(times) / len(times)
    gbs = smp.bytes / sec / 1e9
    sample = (f"oracle dense step on the first {rows} of {wl.V} rows (D={wl.D}, {wl.wdtype} W), "
              f"OpenMP build on {cores} threads")
    line = {
        "impl": "reference", "metric": METRIC, "value": gbs, "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": wl.name, "V": wl.V, "D": wl.D,
                                        "w_dtype": wl.wdtype, "sample_rows": rows},
        "cpu_baseline": {"value": gbs, "unit": "GB/s", "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": gbs, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def sparse_kernel_bytes(wl, U):
    """Algorithmic bytes per launch of the segment-sum kernel (grad rows read,
    summed rows written, sorted order read) and of the apply kernel."""
    N, D, w = wl.N, wl.D, wbytes(wl)
    return {"segsum": 4 * N * D + 4 * U * D + 8 * N, "apply": 4 * U * D + 2 * w * U * D + 8 * U}


def run_sparse_line(args, wl, world, rank, dev):
    import torch
    flush = L2Flush(dev)
    barrier(world)
    with ClockSampler(dev.index or 0) as clocks:
        sp = run_sparse(wl, dev, args.steps, args.warmup, flush, seed=rank)
        barrier(world)
    ms = allreduce_max(world, sp["ms_per_step"])
    line = {
        "metric": METRIC, "value": world * sp["algorithmic_bytes"] / (ms * 1e-3) / 1e9, "unit": "GB/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic",
        "config": {"workload": wl.name, "V": wl.V, "D": wl.D, "N": wl.N, "w_dtype": wl.wdtype,
                   "ids": "int64", "l2": L2_NOTE,
                   "parallelism": f"replicas x{world}"},
        "roofline": sp["roofline"],
        "cpu_baseline": None, "e2e": None, "gpu_launches": sp["gpu_launches"],
        "clocks": clocks.summary(), "sparse": sp,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


def run_lmhead_line(args, wl, world, rank, dev):
    """Stand-alone line for an LM-head gradient workload: the fused step
    (ember_step_lmhead) is the step; value = its HBM bytes per second (G
    written and read once, W read and written, dlogits and H read)."""
    import torch
    flush = L2Flush(dev)
    barrier(world)
    with ClockSampler(dev.index or 0) as clocks:
        lm = run_lmhead(wl, dev, args.steps, args.warmup, flush, seed=rank)
        barrier(world)
    ms = allreduce_max(world, lm["ms_per_step"])
    line = {
        "metric": METRIC, "value": world * lm["hbm_bytes_fused_step"] / (ms * 1e-3) / 1e9, "unit": "GB/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16 x bf16 -> f32",
        "data": "synthetic",
        "config": {"workload": wl.name, "V": wl.V, "D": wl.D, "T": wl.T, "w_dtype": wl.wdtype,
                   "l2": "inputs larger than L2, and " + L2_NOTE,
                   "parallelism": f"replicas x{world}"},
        "roofline": lm["roofline"], "cpu_baseline": None, "e2e": None, "gpu_launches": lm["gpu_launches"],
        "clocks": clocks.summary(), "lmhead_fused": lm,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


CONFIGS = (  # the method's workloads, reported in every default run
    ("c1", "dense_v1024_d64_f32", 400),
    ("c2", "dense_v32000_d4096_bf16", 100),
    ("c3", "dense_tied_v151936_d896_bf16", 100),
    ("c4", "sparse_v262144_d2048_bf16_n32768", 100),
)


def run_ours(args, world, rank, local):
    import torch
    from paper_2607_01455_gb300 import synth
    from paper_2607_01455_gb300.ember import Ember

    wl = synth.WORKLOADS[args.workload]
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    if wl.kind == "lmhead":
        return run_lmhead_line(args, wl, world, rank, dev)
    if wl.kind == "sparse":
        return run_sparse_line(args, wl, world, rank, dev)

    flush = L2Flush(dev)
    peak, peak_kind = measured_hbm_peak()
    # clocks sampled over every timed region of the run (the main step first)
    with ClockSampler(local) as clocks:
        barrier(world)
        main = run_dense(wl, dev, args.steps, args.warmup, flush, seed=rank)
        barrier(world)
        ms = allreduce_max(world, main["ms_per_step"])
        B = step_bytes(wl)
        value = world * B / (ms * 1e-3) / 1e9

        configs = {}
        if not args.no_configs:
            for tag, name, steps in CONFIGS:
                cwl = synth.WORKLOADS[name]
                if cwl.kind == "sparse":
                    if args.no_sparse:
                        continue
                    configs[tag] = run_sparse(cwl, dev, max(2 * TRACE_EVERY, min(steps, 5 * args.steps)), args.warmup,
                                              flush, seed=rank)
                else:
                    configs[tag] = run_dense(cwl, dev, max(2 * TRACE_EVERY, min(steps, 5 * args.steps)), args.warmup,
                                             flush, seed=rank)
            configs["c5"] = {k: main[k] for k in ("workload", "ms_per_step", "value", "unit", "frac_of_measured_hbm",
                                                 "launches_per_step", "roofline")}

        # end to end through the C ABI: the gradient comes in from pinned host
        # memory, the step runs, and its result -- the optimizer state r, c
        # (V + D floats) -- goes back to pinned host memory.  W stays on the
        # device, as model weights do in training.
        e2e = None
        if not args.no_e2e:
            W = synth.init_weights(wl, rank, dev)
            G = synth.dense_grad(wl, rank, 1, dev)
            emb = Ember(wl.V, wl.D, wdtype=wl.wdtype, device=dev)
            n_e2e = max(1, min(args.steps, 10))
            Gh = G.cpu().pin_memory()
            Sh = torch.empty(emb.state.shape, dtype=emb.state.dtype, pin_memory=True)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            G2 = torch.empty_like(G)
            t = 0
            ts = []
            for _ in range(n_e2e):
                t += 1
                flush()
                e0.record(stream)
                G2.copy_(Gh, non_blocking=True)
                emb.step_dense(W, G2, wl.lr, t)
                Sh.copy_(emb.state, non_blocking=True)
                e1.record(stream)
                e1.synchronize()
                ts.append(e0.elapsed_time(e1))
            ms_copy = allreduce_max(world, sum(ts) / len(ts))
            # the same, with the reduce pass reading G over the chip-to-chip
            # link and staging it in HBM (ember_step_dense_from_host)
            ts = []
            for _ in range(n_e2e):
                t += 1
                flush()
                e0.record(stream)
                emb.step_dense_from_host(W, Gh, G2, wl.lr, t)
                Sh.copy_(emb.state, non_blocking=True)
                e1.record(stream)
                e1.synchronize()
                ts.append(e0.elapsed_time(e1))
            ms_e2e = allreduce_max(world, sum(ts) / len(ts))
            if emb.device_status() != 0:
                raise SystemExit("device status after the end-to-end steps")
            e2e = {"value": world * B / (ms_e2e * 1e-3) / 1e9, "unit": "GB/s",
                   "h2d_bytes_per_step": G.numel() * 4, "d2h_bytes_per_step": emb.state.numel() * 4,
                   "ms_per_step": ms_e2e, "steps": n_e2e,
                   "what": "pinned-host G read by the reduce pass over the chip-to-chip link and staged in "
                           "HBM (ember_step_dense_from_host), state r,c -> pinned host",
                   "copy_engine": {"ms_per_step": ms_copy, "value": world * B / (ms_copy * 1e-3) / 1e9,
                                   "what": "cudaMemcpyAsync of G to HBM, ember_step_dense, state back"}}
            del W, G, G2, emb, Gh

        row_only = None
        if not args.no_row_only:
            Wr = synth.init_weights(wl, rank, dev)
            Gr = synth.dense_grad(wl, rank, 1, dev)
            row_only = run_row_only(wl, dev, max(2 * TRACE_EVERY, min(args.steps, 100)), args.warmup, flush, Wr, Gr)
            row_only["frac_of_measured_hbm"] = row_only["value"] / peak
            del Wr, Gr

        lmhead = None
        if not args.no_lmhead:
            lwl = synth.WORKLOADS["lmhead_grad_v128256_d8192_t4096_bf16"]
            lmhead = run_lmhead(lwl, dev, max(2 * TRACE_EVERY, min(args.steps, 20)), args.warmup, flush,
                                seed=rank)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        rows = sample_rows_for(wl, 5.0)
        smp = OracleSample(wl, rows)
        secs = [smp.step() for _ in range(3)]
        sec = sum(secs) / len(secs)
        cores = oracle.threads(host_cores())
        rows_mc = sample_rows_for(wl, 5.0, all_cores=True)
        smp_mc = OracleSample(wl, rows_mc)
        smp_mc.step(all_cores=True)
        secs_mc = [smp_mc.step(all_cores=True) for _ in range(3)]
        sec_mc = sum(secs_mc) / len(secs_mc)
        cpu = {"value": smp.bytes / sec / 1e9, "unit": "GB/s", "cores": 1, "kind": "oracle",
               "sample": f"3 oracle dense steps on the first {rows} of {wl.V} rows (D={wl.D}), one thread",
               "ms_per_step": sec * 1e3,
               "all_cores": {"value": smp_mc.bytes / sec_mc / 1e9, "unit": "GB/s", "cores": cores,
                             "kind": "oracle (OpenMP build of the same source: the same bits)",
                             "sample": f"3 oracle dense steps on the first {rows_mc} of {wl.V} rows "
                                       f"(D={wl.D}), {cores} threads",
                             "ms_per_step": sec_mc * 1e3}}

    npan = main.get("roofline", {}).get("launches_per_pass", 1)
    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": wl.name, "V": wl.V, "D": wl.D, "w_dtype": wl.wdtype, "g_dtype": "f32",
                   "state_dtype": "f32", "l2": L2_NOTE,
                   "parallelism": f"replicas x{world}"},
        "roofline": main["roofline"],
        "cpu_baseline": cpu,
        "e2e": e2e,
        "gpu_launches": main["gpu_launches"],
        "clocks": clocks.summary(),
        "params_per_s": world * wl.V * wl.D / (ms * 1e-3),
        "frac_of_nominal_8TBs": value / world / NOMINAL_HBM_GBS,
        "frac_of_measured_hbm": value / world / peak,
        "peak_kind": peak_kind,
        "kernels": main.get("kernels"),
        "ms_per_step_traced": main.get("ms_per_step_traced"),
        "timing": main["timing"],
        "wall_s_timed_region": main["wall_s_timed_region"],
        "column_panels": npan,
        "configs": configs,
        "sparse": configs.get("c4"),
        "row_only": row_only,
        "lmhead_fused": lmhead,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-sparse", action="store_true")
    ap.add_argument("--no-row-only", action="store_true")
    ap.add_argument("--no-lmhead", action="store_true")
    ap.add_argument("--no-configs", action="store_true")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3
    world, rank, local = dist_setup()
    if args.impl == "reference":
        rc = run_reference(args, world, rank)
    else:
        rc = run_ours(args, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return rc


if __name__ == "__main__":
    sys.exit(main())
