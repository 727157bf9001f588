#!/usr/bin/env python3
"""Throughput of the AViTS resolution transition on GB300.

One step = one pass of the whole hot path over one FLUX-1024-shaped transition
(batch 1): spatial score (Eq. 3-5) -> temporal score -> fuse + top-k
(Eq. 8-9) -> selective upsample (Stage 2) -> final merge (Stage 3), all on the
device through the C ABI.  Inputs are resident in HBM; the step rotates over
NSETS copies of the inputs (> L2) so that no step reads inputs left in L2 by
the previous ones.  The timed region replays CUDA graphs of those steps.

Prints one JSON line.  --impl reference times the CPU oracle instead.
Multi-GPU (torchrun): every rank runs an independent replica ("replicas
only": the path has no exchange step); value = all ranks' transitions / max
rank time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "transitions/s at FLUX-1024 shape"
UNIT = "transitions/s"
WORKLOAD = "flux1024"
WORKLOAD_STR = ("FLUX-1024-shaped transition: 32x32 -> 64x64 tokens, 512 text keys, H=24, "
                "d=128, D=3072, C=16 p=2, bf16, alpha=0.5, k=307, batch 1, seed 1 "
                "(%s upsample)")
L2_BYTES = 129 * 1024 * 1024


def _args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--mode", default="nearest", choices=["nearest", "bilinear"])
    ap.add_argument("--sets", type=int, default=10, help="input copies rotated per step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--quick", action="store_true", help="skip the secondary measurements")
    return ap.parse_args()


# ----------------------------------------------------------------- dist ----
def dist_setup(n_gpus):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    pg = None
    if world > 1:
        import torch.distributed as dist
        backend = os.environ.get("AVITS_BENCH_BACKEND", "nccl")
        dist.init_process_group(backend=backend)
        pg = dist
    return world, rank, local, pg


def barrier(pg):
    if pg is not None:
        pg.barrier()


def max_over_ranks(pg, value: float, device=None) -> float:
    """Largest `value` over all ranks (the slowest rank sets the job time)."""
    if pg is None:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def aggregate(units_per_rank: int, world: int, max_seconds: float):
    """Whole-job throughput: every rank's units over the slowest rank's time."""
    return units_per_rank * world / max_seconds


# --------------------------------------------------------------- clocks ----
class ClockSampler:
    """nvidia-smi samples taken while the GPU runs the measured work."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def mark(self):
        return time.time()

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self, t0: float, t1: float):
        rows = [l for (t, l) in self.lines if t0 <= t <= t1] or [l for (_, l) in self.lines]
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for l in rows:
            f = [x.strip() for x in l.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------- roofline inputs ----
def algorithmic_work(tr, mode):
    """Per-launch algorithmic FLOPs / bytes of each kernel (one transition)."""
    elt = 2 if tr.dtype == "bf16" else 4
    B, H, M, Nk, d, D, T = tr.B, tr.H, tr.M, tr.Nk, tr.d, tr.D, tr.C * 4
    NO = M + 3 * tr.k
    F = 4 * tr.frame_h * tr.frame_w
    return {
        "spatial": {"flops": 2.0 * B * H * M * Nk * d, "exps": float(B * H * M * Nk),
                    "bytes": float(B * H * (M + Nk) * d * elt + 4 * B * M)},
        "temporal": {"bytes": float(2 * B * M * D * elt + 4 * B * M)},
        "select": {"bytes": float(8 * B * M + 4 * B * M + 4 * B * tr.k + B * M + 4 * B * M)},
        "upsample": {"bytes": float(B * M * T * elt + B * M * 5 + B * NO * (T * elt + 17))},
        "select_upsample": {"bytes": float(8 * B * M + 4 * B * M + 4 * B * tr.k + B * M
                                           + 4 * B * M + B * M * T * elt
                                           + B * NO * (T * elt + 17))},
        "merge": {"bytes": float(B * NO * (T * elt + 12) + B * F * T * elt)},
    }


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16_tflops": float(p["bf16_tflops"]),
                "bf16_tflops_sustained": float(p["bf16_tflops_sustained"]), "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "source": "fallback"}


def profiled_traffic(kernel_src: str, summary: str):
    """DRAM bytes per launch recorded by an ncu capture (profiles/), or None
    when the kernel source changed since that capture."""
    path = os.path.join(ROOT, "profiles", summary)
    try:
        text = open(path).read()
        with open(kernel_src, "rb") as f:
            sha = hashlib.sha1(f.read()).hexdigest()[:12]
    except OSError:
        return None
    m = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", text)
    s = re.search(r"kernel_source_sha1:\s*([0-9a-f]+)", text)
    if not m or not s or s.group(1) != sha:
        return None
    return float(m.group(1))


def _smi_id(torch, dev, local):
    """nvidia-smi -i argument of this rank's GPU (UUID when torch exposes it)."""
    try:
        u = str(torch.cuda.get_device_properties(dev).uuid)
        if u:
            return u if u.startswith("GPU-") else "GPU-" + u
    except (AttributeError, RuntimeError):
        pass
    vis = os.environ.get("CUDA_VISIBLE_DEVICES", "")
    ids = [x for x in vis.split(",") if x.strip()]
    return ids[local] if local < len(ids) else str(local)


# ------------------------------------------------------------------ ours ----
def run_ours(args, world, rank, local, pg):
    import torch
    import paper_2608_17995_gb300 as av
    from paper_2608_17995_gb300.pipeline import TransitionBuffers, to_device
    from paper_2608_17995_gb300.workloads import make_transition

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    av.build()
    av.lib()
    tr = make_transition(WORKLOAD, seed=1 + 1000 * rank if rank else None)
    mode = args.mode
    buf = TransitionBuffers(tr, device=dev, mode=mode, inputs=True)
    stream = torch.cuda.Stream(device=dev)

    # NSETS resident copies of the inputs, rotated per step (> L2 in total)
    base = (buf.q, buf.k, buf.h_t, buf.h_prev, buf.latent)
    set_bytes = sum(t.numel() * t.element_size() for t in base)
    nsets = max(args.sets, int(math.ceil(2.0 * L2_BYTES / set_bytes)) + 1)
    sets = [base] + [tuple(t.clone() for t in base) for _ in range(nsets - 1)]
    torch.cuda.synchronize()

    # our kernels per step: spatial + temporal (beside it), the fused
    # selection + upsample, the merge (bilinear: map + gather)
    kernels_per_step = 4 if buf.mode == av.NEAREST else 5
    names = ["spatial", "temporal", "select", "upsample", "merge", "select_upsample"]

    def step(s, st):
        buf.set_inputs(*sets[s % nsets])
        buf.run(st)

    # eager warm-up (also builds the spatial workspace), then graphs
    with torch.cuda.stream(stream):
        for s in range(max(args.warmup, 3)):
            step(s, stream)
    stream.synchronize()
    if av.avits_device_status(stream) != 0:
        raise RuntimeError("device status error during warm-up")

    # the timed region is ONE graph of exactly K steps (the input copies
    # rotated step by step), so the number of graph launches in it does not
    # depend on K; the warm-up is one graph of W steps
    K, W = args.steps, args.warmup

    def graph_of(n, first=0):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for s in range(first, first + n):
                step(s, stream)
        return g

    g_warm = graph_of(max(W, 3))
    g_timed = graph_of(K, first=max(W, 3))
    g_soak = graph_of(nsets)
    with torch.cuda.stream(stream):
        g_warm.replay()
    stream.synchronize()

    clocks = ClockSampler(_smi_id(torch, dev, local))
    clocks.start()
    time.sleep(0.4)
    soak_t0 = clocks.mark()
    # keep the GPU under the same load while the sampler settles (untimed)
    with torch.cuda.stream(stream):
        t_end = time.time() + 0.6
        while time.time() < t_end:
            g_soak.replay()
            stream.synchronize()
        g_warm.replay()
    stream.synchronize()

    # ---------------- timed region: exactly K steps ----------------
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    barrier(pg)
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        ev0.record(stream)
        g_timed.replay()
        ev1.record(stream)
    stream.synchronize()
    torch.cuda.synchronize()
    barrier(pg)
    t_ms = ev0.elapsed_time(ev1)
    clock_t1 = clocks.mark()
    time.sleep(0.25)
    clocks.stop()
    clk = clocks.summary(soak_t0, clock_t1)
    status = av.avits_device_status(stream)
    if status != 0:
        raise RuntimeError("device status %d after the timed region" % status)
    max_ms = max_over_ranks(pg, t_ms, dev)
    value = aggregate(K, world, max_ms / 1e3)

    # ---------------- per-kernel durations (events between kernels) ----------
    per_kernel = per_kernel_times(torch, av, buf, sets, nsets, stream, names, args)
    work = algorithmic_work(tr, mode)
    peaks = measured_peaks()
    kt = {}
    for n in names:
        ms = per_kernel.get(n)
        if ms is None:
            continue
        e = {"us": round(ms * 1e3, 3)}
        w = work[n]
        if "flops" in w:
            e["tflops"] = round(w["flops"] / (ms * 1e-3) / 1e12, 2)
            e["frac_tensor"] = round(e["tflops"] / peaks["bf16_tflops"], 4)
            e["gexp_per_s"] = round(w["exps"] / (ms * 1e-3) / 1e9, 1)
        e["gbs"] = round(w["bytes"] / (ms * 1e-3) / 1e9, 1)
        e["frac_hbm"] = round(e["gbs"] / peaks["hbm_gbs"], 4)
        kt[n] = e
    sp_ms = per_kernel.get("spatial")
    traffic = profiled_traffic(os.path.join(ROOT, "paper_2608_17995_gb300", "csrc", "spatial_tc.cu"),
                               "spatial_tc_flux1024.md")
    roofline = None
    if sp_ms:
        achieved = work["spatial"]["flops"] / (sp_ms * 1e-3) / 1e12
        roofline = {"kernel": "spatial_tc_kernel + its merge (one avits_score_spatial call)",
                    "bound": "tensor",
                    "achieved": round(achieved, 2), "peak": peaks["bf16_tflops"],
                    "unit": "TFLOP/s", "frac": round(achieved / peaks["bf16_tflops"], 4),
                    "peak_source": peaks["source"] + " bf16 burst (MEASURED_PEAKS.json)",
                    "traffic": traffic}

    result = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
        "steps": K, "warmup": W, "ms_per_step": round(max_ms / K, 6),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": WORKLOAD_STR % mode,
                   "global_batch": world, "parallelism": "replicas x%d" % world,
                   "l2": "inputs rotated over %d resident copies (%.0f MB > 129 MB L2)"
                         % (nsets, nsets * set_bytes / 1e6),
                   "timing": "one CUDA graph of exactly K steps replayed once between CUDA "
                             "events on the launching stream (W warm-up steps before)"},
        "gpu_launches": K * kernels_per_step,
        "clocks": clk,
        "kernels": kt,
        "kernels_timing": per_kernel["_how"],
        "roofline": roofline,
    }
    if not args.no_e2e and not args.quick:
        result["e2e"] = e2e_measure(torch, av, buf, tr, stream, K, W, world, pg, dev)
    if mode == "nearest" and not args.quick:
        result["bilinear"] = mode_measure(torch, av, tr, dev, stream, sets, nsets, K)
    if not args.quick:
        result["warm_l2"] = warm_measure(torch, buf, sets, stream, K)
        result["batched_schedule"] = batched_schedule_measure(torch, av, dev, stream, K)
        result["temporal_var"] = temporal_var_measure(torch, av, tr, dev, stream, peaks)
        result["spatial_keymask"] = keymask_measure(torch, av, buf, tr, sets, nsets, stream, peaks)
        result["spatial_from_lse"] = lse_measure(torch, av, buf, tr, sets, nsets, stream, peaks)
        result["flux2048"] = config_measure(torch, av, dev, stream, peaks, "flux2048")
        result["edit"] = config_measure(torch, av, dev, stream, peaks, "edit")
        result["tiny"] = config_measure(torch, av, dev, stream, peaks, "tiny")
        result["batch_sweep"] = batch_sweep_measure(torch, av, dev, stream, peaks)
        result["attention_forward"] = {
            n: attention_measure(torch, av, dev, stream, peaks, n) for n in ("flux1024", "flux2048")}
    return result, tr


def per_kernel_times(torch, av, buf, sets, nsets, stream, names, args):
    """Average device time per call of each entry point: a CUDA graph of
    `n` back-to-back calls of that one entry point (rotating over the input
    copies) is replayed between CUDA events on the launching stream.  A call's
    time includes its in-graph launch gap; avits_score_spatial is two kernels
    (scores + merge)."""
    calls = {"spatial": buf.spatial, "temporal": buf.temporal, "select": buf.select,
             "upsample": buf.upsample, "merge": buf.merge,
             "select_upsample": buf.select_upsample}
    n, reps = max(nsets * 4, 48), 10
    out = {"_how": "graph of %d back-to-back calls per entry point, %d replays" % (n, reps)}
    for name in names:
        fn = calls[name]
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for s in range(n):
                buf.set_inputs(*sets[s % nsets])
                fn(stream)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            g.replay()
            e0.record(stream)
            for _ in range(reps):
                g.replay()
            e1.record(stream)
        stream.synchronize()
        out[name] = e0.elapsed_time(e1) / (n * reps)
    return out


def mode_measure(torch, av, tr, dev, stream, sets, nsets, K):
    """Step time with bilinear upsampling / merge (same inputs, graph replay)."""
    from paper_2608_17995_gb300.pipeline import TransitionBuffers
    b2 = TransitionBuffers(tr, device=dev, mode="bilinear", inputs=False)

    def step(s):
        b2.set_inputs(*sets[s % nsets])
        b2.run(stream)

    with torch.cuda.stream(stream):
        for s in range(3):
            step(s)
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for s in range(nsets):
            step(s)
    reps = max(1, K // nsets)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        g.replay()
        e0.record(stream)
        for _ in range(reps):
            g.replay()
        e1.record(stream)
    stream.synchronize()
    ms = e0.elapsed_time(e1) / (reps * nsets)
    st = av.avits_device_status(stream)
    return {"ms_per_step": round(ms, 6), "value": round(1e3 / ms, 1), "unit": UNIT,
            "status": st}


def _graph_time_ms(torch, stream, fn, reps):
    """Average device time of fn() replayed from one CUDA graph."""
    with torch.cuda.stream(stream):
        for _ in range(3):
            fn()
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        fn()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        g.replay()
        e0.record(stream)
        for _ in range(reps):
            g.replay()
        e1.record(stream)
    stream.synchronize()
    return e0.elapsed_time(e1) / reps


def warm_measure(torch, buf, sets, stream, K, per_graph=10):
    """The same steps on ONE input set (inputs left in L2 by the previous
    step): the warm-L2 figure reported beside the flushed one.  One graph
    holds per_graph steps, as the flushed measurement's does."""
    def fn():
        for _ in range(per_graph):
            buf.set_inputs(*sets[0])
            buf.run(stream)
    ms = _graph_time_ms(torch, stream, fn, max(10, min(K // per_graph, 200))) / per_graph
    return {"ms_per_step": round(ms, 6), "value": round(1e3 / ms, 1), "unit": UNIT,
            "l2": "one input set, resident in L2"}


def batch_sweep_measure(torch, av, dev, stream, peaks, batches=(1, 8, 32, 64)):
    """Bytes-scaled sweep at the FLUX-1024 shape (H=24, M=1024, L=512, d=128,
    D=3072, C=16, k=307): B transitions per call.  Per entry point, the
    average device time per call in a graph of back-to-back calls rotating
    over input copies (> 2x L2 in total), and the achieved rate against the
    algorithmic work: TFLOP/s for the spatial score, GB/s for the others.
    Inputs are drawn on the device (Q, K ~ N(0, 3) per element, logits of
    std ~3; h, latent ~ N(0, 1); A, V uniform): these calls measure time, not
    parity, which the tests establish."""
    from types import SimpleNamespace
    from paper_2608_17995_gb300 import SpatialWorkspace
    H, M, L, d, D, C, k, G = 24, 1024, 512, 128, 3072, 16, 307, 32
    Nk = L + M
    NO = M + 3 * k
    out = {}
    g = torch.Generator(device=dev)
    g.manual_seed(5)
    for B in batches:
        bf = torch.bfloat16

        def one_set():
            q = (torch.randn(B, H, M, d, device=dev, generator=g) * math.sqrt(3.0)).to(bf)
            kk = (torch.randn(B, H, Nk, d, device=dev, generator=g) * math.sqrt(3.0)).to(bf)
            ht = torch.randn(B, M, D, device=dev, generator=g).to(bf)
            hp = torch.randn(B, M, D, device=dev, generator=g).to(bf)
            lat = torch.randn(B, M, C * 4, device=dev, generator=g).to(bf)
            A = torch.rand(B, M, device=dev, generator=g)
            V = torch.rand(B, M, device=dev, generator=g)
            return q, kk, ht, hp, lat, A, V

        first = one_set()
        set_bytes = sum(t.numel() * t.element_size() for t in first)
        nsets = min(11, max(2, int(math.ceil(2.0 * L2_BYTES / set_bytes)) + 1))
        sets = [first] + [one_set() for _ in range(nsets - 1)]
        A_out = torch.empty(B, M, device=dev)
        V_out = torch.empty(B, M, device=dev)
        ws = SpatialWorkspace(dev)
        sel = [torch.empty(B, k, dtype=torch.int32, device=dev) for _ in range(nsets)]
        off = [torch.empty(B, M, dtype=torch.int32, device=dev) for _ in range(nsets)]
        msk = [torch.empty(B, M, dtype=torch.uint8, device=dev) for _ in range(nsets)]
        mixed = [torch.empty(B, NO, C * 4, dtype=bf, device=dev) for _ in range(nsets)]
        pos = [torch.empty(B, NO, 2, dtype=torch.int32, device=dev) for _ in range(nsets)]
        span = [torch.empty(B, NO, dtype=torch.int32, device=dev) for _ in range(nsets)]
        stok = [torch.empty(B, NO, dtype=torch.int32, device=dev) for _ in range(nsets)]
        ssub = [torch.empty(B, NO, dtype=torch.int8, device=dev) for _ in range(nsets)]
        full = torch.empty(B, 4 * G * G, C * 4, dtype=bf, device=dev)
        mws = torch.zeros(av.avits_merge_final_workspace(av.NEAREST, B, 2 * G, 2 * G),
                          dtype=torch.uint8, device=dev)

        def spatial(i):
            av.avits_score_spatial(sets[i][0], sets[i][1], L, 1.0 / math.sqrt(d), A_out,
                                   workspace=ws, stream=stream)

        def temporal(i):
            av.avits_score_temporal(sets[i][2], sets[i][3], V_out, stream=stream)

        def select_upsample(i):
            av.avits_select_upsample(sets[i][5], sets[i][6], 0.5, k, sel[i], off[i], msk[i],
                                     sets[i][4], G, G, mixed[i], pos[i], span[i], stok[i],
                                     ssub[i], stream=stream)

        def merge(i):
            av.avits_merge_final(mixed[i], pos[i], span[i], 2 * G, 2 * G, full,
                                 mode=av.NEAREST, workspace=mws, stream=stream)

        with torch.cuda.stream(stream):
            for i in range(nsets):
                select_upsample(i)   # valid mixed sequences for the merge
        stream.synchronize()
        tr = SimpleNamespace(dtype="bf16", B=B, H=H, M=M, Nk=Nk, d=d, D=D, C=C, k=k,
                             frame_h=G, frame_w=G)
        work = algorithmic_work(tr, "nearest")
        e = {}
        for name, fn in (("spatial", spatial), ("temporal", temporal),
                         ("select_upsample", select_upsample), ("merge", merge)):
            n = max(2 * nsets, 16 if B >= 32 else 48)

            def calls():
                for j in range(n):
                    fn(j % nsets)

            ms = _graph_time_ms(torch, stream, calls, 10) / n
            r = {"us": round(ms * 1e3, 3)}
            w = work[name]
            if "flops" in w:
                tf = w["flops"] / (ms * 1e-3) / 1e12
                r["tflops"] = round(tf, 2)
                r["frac_tensor"] = round(tf / peaks["bf16_tflops"], 4)
            gbs = w["bytes"] / (ms * 1e-3) / 1e9
            r["gbs"] = round(gbs, 1)
            r["frac_hbm"] = round(gbs / peaks["hbm_gbs"], 4)
            r["bytes"] = int(w["bytes"])
            e[name] = r
        e["status"] = av.avits_device_status(stream)
        out["B%d" % B] = e
        del sets, first
        torch.cuda.empty_cache()
    out["how"] = ("graph of back-to-back calls per entry point rotating over input copies "
                  "(> 2x L2), device-drawn inputs at the FLUX-1024 shape, B transitions per call")
    return out


CONFIG_NOTES = {
    "tiny": "B=1, H=2, 16x16 -> 32x32 tokens, M=256, L=32, Nk=288, d=64, D=128, fp32 "
            "(CUDA-core path), k=64, nearest",
    "flux2048": "B=1, H=24, 64x64 -> 128x128 tokens, M=4096, L=512, Nk=4608, k=1024, nearest",
    "edit": "B=1, H=24, 32x32 -> 64x64 tokens, M=1024, L=512, 4096 reference keys, Nk=5632, "
            "k=205, nearest",
}


def config_measure(torch, av, dev, stream, peaks, name, nsets=3):
    """Another configuration's transition: the whole step and the spatial
    call, inputs rotated over nsets copies (> L2).  FLUX-2048 (M = 4096,
    Nk = 4608, 116 GFLOP in the spatial score): every CTA of the spatial
    kernel runs ~90 items, so start-up and the merge are a small share of
    its time.  Editing (M = 1024 with 4096 reference keys, Nk = 5632)."""
    from paper_2608_17995_gb300.pipeline import TransitionBuffers
    from paper_2608_17995_gb300.workloads import make_transition
    t2 = make_transition(name)
    b2 = TransitionBuffers(t2, device=dev)
    base = (b2.q, b2.k, b2.h_t, b2.h_prev, b2.latent)
    sets2 = [base] + [tuple(x.clone() for x in base) for _ in range(nsets - 1)]

    def step():
        for s_ in range(nsets):
            b2.set_inputs(*sets2[s_])
            b2.run(stream)

    def spatial():
        for s_ in range(nsets):
            b2.set_inputs(*sets2[s_])
            b2.spatial(stream)

    def temporal():
        for s_ in range(nsets):
            b2.set_inputs(*sets2[s_])
            b2.temporal(stream)

    ms_step = _graph_time_ms(torch, stream, step, 20) / nsets
    ms_sp = _graph_time_ms(torch, stream, spatial, 20) / nsets
    ms_tp = _graph_time_ms(torch, stream, temporal, 20) / nsets
    flops = 2.0 * t2.B * t2.H * t2.M * t2.Nk * t2.d
    tf = flops / (ms_sp * 1e-3) / 1e12
    tbytes = 2.0 * t2.B * t2.M * t2.D * b2.h_t.element_size() + 4.0 * t2.B * t2.M
    tgbs = tbytes / (ms_tp * 1e-3) / 1e9
    return {"ms_per_step": round(ms_step, 6), "value": round(1e3 / ms_step, 1), "unit": UNIT,
            "spatial_us": round(ms_sp * 1e3, 3), "spatial_tflops": round(tf, 2),
            "spatial_frac_tensor": round(tf / peaks["bf16_tflops"], 4),
            "temporal_us": round(ms_tp * 1e3, 3), "temporal_gbs": round(tgbs, 1),
            "temporal_frac_hbm": round(tgbs / peaks["hbm_gbs"], 4),
            "status": av.avits_device_status(stream), "config": CONFIG_NOTES[name]}


def batched_schedule_measure(torch, av, dev, stream, K):
    """The batched multi-stage schedule at FLUX shape: 8 elements, 16x16 ->
    32x32 (k = 128) -> 64x64 (every mixed token re-scored, k = 192), then the
    final merge to 64x64.  Its inputs (about 230 MB) exceed L2."""
    from paper_2608_17995_gb300.pipeline import TransitionBuffers, to_numpy
    from paper_2608_17995_gb300.workloads import make_batched_stage2, make_transition
    t1 = make_transition("batched")
    b1 = TransitionBuffers(t1, device=dev)
    with torch.cuda.stream(stream):
        b1.run(stream, merge=False)
    stream.synchronize()
    t2 = make_batched_stage2(to_numpy(b1.pos), to_numpy(b1.span), frame=32,
                             latent=to_numpy(b1.mixed))
    b2 = TransitionBuffers(t2, device=dev)
    # the second transition reads the first one's device outputs
    b2.set_inputs(b2.q, b2.k, b2.h_t, b2.h_prev, b1.mixed, b1.pos, b1.span)

    def fn():
        b1.run(stream, merge=False)
        b2.run(stream)

    ms = _graph_time_ms(torch, stream, fn, max(20, min(K // 10, 200)))
    st = av.avits_device_status(stream)
    return {"ms_per_schedule": round(ms, 6), "schedules_per_s": round(1e3 / ms, 1),
            "transitions_per_s": round(2 * t1.B * 1e3 / ms, 1), "status": st,
            "config": "B=8, FLUX heads/width, 16x16 -> 32x32 (k=128) -> 64x64 (k=192, 640 "
                      "mixed tokens re-scored), final merge; nearest"}


def keymask_measure(torch, av, buf, tr, sets, nsets, stream, peaks):
    """avits_score_spatial_keymask at the FLUX-1024 shape (interleaved text
    and image keys): text blocks between image blocks (a unified MLLM-style
    sequence; most key halves all text or all image) and a random 30 % mask
    (every key half mixed, the slow path)."""
    Nk = tr.Nk
    g = torch.Generator(device="cpu")
    g.manual_seed(3)
    blocks = torch.zeros(tr.B, Nk, dtype=torch.uint8)
    blocks[:, 0:200] = 1
    blocks[:, 700:900] = 1
    blocks[:, 1400:1512] = 1
    rand = (torch.rand(tr.B, Nk, generator=g) < 0.3).to(torch.uint8)
    A = torch.empty(tr.B, tr.M, dtype=torch.float32, device=buf.A.device)
    out = {}
    flops = 2.0 * tr.B * tr.H * tr.M * Nk * tr.d
    for name, m in (("blocks", blocks), ("random", rand)):
        md = m.to(buf.A.device)

        def fn():
            for s_ in range(nsets):
                av.avits_score_spatial(sets[s_][0], sets[s_][1], 0, tr.softmax_scale, A,
                                       workspace=buf.ws, stream=stream, text_mask=md)

        ms = _graph_time_ms(torch, stream, fn, 20) / nsets
        tf = flops / (ms * 1e-3) / 1e12
        out[name] = {"us": round(ms * 1e3, 3), "tflops": round(tf, 2),
                     "frac_tensor": round(tf / peaks["bf16_tflops"], 4),
                     "text_keys": int(m.sum())}
    out["status"] = av.avits_device_status(stream)
    return out


def lse_measure(torch, av, buf, tr, sets, nsets, stream, peaks):
    """avits_score_spatial_lse at the FLUX-1024 shape: the text mass from the
    caller's logsumexp over all keys (as a model's attention forward returns
    it) and the L = 512 text keys only, rotated over the same input copies."""
    A = torch.empty(tr.B, tr.M, dtype=torch.float32, device=buf.A.device)
    lse = torch.empty(tr.B, tr.H, tr.M, 2, dtype=torch.float32, device=buf.A.device)
    av.avits_score_spatial(sets[0][0], sets[0][1], tr.L, tr.softmax_scale, A, lse=lse,
                           workspace=buf.ws, stream=stream)
    lse_all = lse[..., 0].contiguous()

    def fn():
        for s_ in range(nsets):
            av.avits_score_spatial_lse(sets[s_][0], sets[s_][1][:, :, :tr.L], lse_all,
                                       tr.softmax_scale, A, workspace=buf.ws, stream=stream)

    ms = _graph_time_ms(torch, stream, fn, 20) / nsets
    flops = 2.0 * tr.B * tr.H * tr.M * tr.L * tr.d
    tf = flops / (ms * 1e-3) / 1e12
    return {"us": round(ms * 1e3, 3), "tflops": round(tf, 2),
            "frac_tensor": round(tf / peaks["bf16_tflops"], 4), "text_keys": tr.L,
            "status": av.avits_device_status(stream)}


def attention_measure(torch, av, dev, stream, peaks, name, nsets=5):
    """The joint-attention forward with the spatial score (avits_attention_forward)
    on the joint sequence of a configuration (queries = keys = text + image
    tokens; Q, K, V bf16 rotated over nsets copies, more than L2), three ways:
    with A and lse, with O only (the cost of the score is the difference), and
    the separate spatial-score pass over the image rows that the forward makes
    unnecessary."""
    from paper_2608_17995_gb300.pipeline import to_device
    from paper_2608_17995_gb300.workloads import make_transition, make_joint_attention
    tr = make_transition(name)
    q, v = make_joint_attention(tr)
    B, H, Mq, d = q.shape
    Nk = tr.Nk
    sets = []
    for i in range(nsets):
        qd, kd, vd = (to_device(a, "bf16", dev) for a in (q, tr.k_all, v))
        sets.append((qd, kd, vd, torch.empty_like(qd)))
    A = torch.zeros(B, Mq, dtype=torch.float32, device=dev)
    lse = torch.empty(B, H, Mq, 2, dtype=torch.float32, device=dev)
    A_sp = torch.zeros(B, tr.M, dtype=torch.float32, device=dev)
    ws = av.SpatialWorkspace(dev)

    def fwd(with_score):
        def fn():
            for (qd, kd, vd, od) in sets:
                av.avits_attention_forward(qd, kd, vd, tr.L, tr.softmax_scale, od,
                                           lse=lse if with_score else None,
                                           A=A if with_score else None, workspace=ws,
                                           stream=stream)
        return fn

    def spatial():
        for (qd, kd, _, _) in sets:
            av.avits_score_spatial(qd[:, :, tr.L:tr.L + tr.M], kd, tr.L, tr.softmax_scale, A_sp,
                                   workspace=ws, stream=stream)

    reps = 20 if Mq <= 2048 else 5
    ms_a = _graph_time_ms(torch, stream, fwd(True), reps) / nsets
    ms_o = _graph_time_ms(torch, stream, fwd(False), reps) / nsets
    ms_s = _graph_time_ms(torch, stream, spatial, reps) / nsets
    flops = 4.0 * B * H * Mq * Nk * d
    tf = flops / (ms_a * 1e-3) / 1e12
    return {"shape": {"B": B, "H": H, "Mq": Mq, "Nk": Nk, "L": tr.L, "d": d},
            "us": round(ms_a * 1e3, 3), "tflops": round(tf, 2),
            "frac_tensor": round(tf / peaks["bf16_tflops"], 4),
            "us_o_only": round(ms_o * 1e3, 3),
            "tflops_o_only": round(flops / (ms_o * 1e-3) / 1e12, 2),
            "score_cost_us": round((ms_a - ms_o) * 1e3, 3),
            "separate_spatial_pass_us": round(ms_s * 1e3, 3),
            "flops_per_call": flops,
            "status": av.avits_device_status(stream)}


def temporal_var_measure(torch, av, tr, dev, stream, peaks, n_t=4, n_sets=6):
    """Eq. 6-7 step variance over n_t snapshots of the FLUX-1024 hidden
    states (bf16 [1, 1024, 3072] each), rotated over n_sets snapshot sets
    (151 MB > L2) so that every call reads from HBM."""
    g = torch.Generator(device=dev)
    g.manual_seed(7)
    sets = [[torch.randn(tr.B, tr.M, tr.D, device=dev, generator=g).to(torch.bfloat16)
             for _ in range(n_t)] for _ in range(n_sets)]
    V = torch.empty(tr.B, tr.M, device=dev, dtype=torch.float32)

    def fn():
        for snaps in sets:
            av.avits_score_temporal_var(snaps, V, stream=stream)

    ms = _graph_time_ms(torch, stream, fn, 50) / n_sets
    nbytes = n_t * tr.B * tr.M * tr.D * 2 + 4 * tr.B * tr.M
    gbs = nbytes / (ms * 1e-3) / 1e9
    return {"us": round(ms * 1e3, 3), "snapshots": n_t, "gbs": round(gbs, 1),
            "frac_hbm": round(gbs / peaks["hbm_gbs"], 4),
            "l2": "%d snapshot sets rotated (%.0f MB)" % (n_sets, n_sets * nbytes / 1e6)}


def e2e_measure(torch, av, buf, tr, stream, K, W, world, pg, dev):
    """Same metric through the public API from pinned HOST buffers.  Every step
    copies its inputs host->device, runs the five calls and reads the merged
    latent and the selected indices back.  The copies are pipelined the way a
    serving loop would: while step i computes on one device copy of the
    inputs, the inputs of step i+1 stream into the other on a copy stream (two
    graphs, replayed alternately); every step still has its own H2D copy and
    D2H read inside the timed region.  CUDA events on the compute stream."""
    inputs = (buf.q, buf.k, buf.h_t, buf.h_prev, buf.latent)
    host_in = [t.cpu().pin_memory() for t in inputs]
    dev_in = [[torch.empty_like(t) for t in inputs] for _ in range(2)]
    host_full = torch.empty(buf.full.shape, dtype=buf.full.dtype).pin_memory()
    host_sel = torch.empty(buf.sel_idx.shape, dtype=buf.sel_idx.dtype).pin_memory()
    h2d = sum(t.numel() * t.element_size() for t in host_in)
    d2h = host_full.numel() * host_full.element_size() + host_sel.numel() * host_sel.element_size()
    copy_stream = torch.cuda.Stream(device=dev)

    def step(cur):
        # inputs of the next step -> the other buffer, beside this step's compute
        fork = torch.cuda.Event()
        fork.record(stream)
        copy_stream.wait_event(fork)
        with torch.cuda.stream(copy_stream):
            for d, h in zip(dev_in[1 - cur], host_in):
                d.copy_(h, non_blocking=True)
        join = torch.cuda.Event()
        join.record(copy_stream)
        buf.set_inputs(*dev_in[cur])
        buf.run(stream)
        host_full.copy_(buf.full, non_blocking=True)
        host_sel.copy_(buf.sel_idx, non_blocking=True)
        stream.wait_event(join)

    with torch.cuda.stream(stream):
        for d, h in zip(dev_in[0], host_in):
            d.copy_(h, non_blocking=True)
        for i in range(4):
            step(i % 2)
    stream.synchronize()
    graphs = []
    for cur in range(2):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            step(cur)
        graphs.append(g)
    n = max(10, min(K, 500))
    n += n % 2
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        # the graph for buffer 0 computes on inputs the previous replay (or the
        # prologue) copied into buffer 0
        for i in range(4):
            graphs[i % 2].replay()
        barrier(pg)
        e0.record(stream)
        for i in range(n):
            graphs[i % 2].replay()
        e1.record(stream)
    stream.synchronize()
    barrier(pg)
    ms = max_over_ranks(pg, e0.elapsed_time(e1), dev)
    return {"value": round(aggregate(n, world, ms / 1e3), 1), "unit": UNIT,
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h), "steps": n,
            "ms_per_step": round(ms / n, 6),
            "pipelining": "H2D of step i+1 on a copy stream beside the compute of step i"}


# ---------------------------------------------------------- CPU oracle ----
def oracle_stage_times(tr, orc, mode=None, min_sample_s=0.05):
    """Seconds of each stage of one oracle transition of `tr` on the oracle's
    current thread count.  The spatial score is timed on an evenly spaced
    sample of the B*M image rows (all heads, all keys; grown x4 from 8 rows
    until it takes min_sample_s) and scaled to all rows; the temporal score,
    fuse + top-k, selective upsample and merge run in full."""
    import numpy as np
    n_all = tr.B * tr.M
    nr = 8
    while True:
        rows = np.unique(np.linspace(0, n_all - 1, min(nr, n_all)).astype(np.int32))
        t0 = time.perf_counter()
        A, _, _ = orc.score_spatial(tr.q_img, tr.k_all, tr.L, tr.softmax_scale, rows=rows)
        dt = time.perf_counter() - t0
        if dt >= min_sample_s or len(rows) >= n_all:
            break
        nr *= 4
    out = {"spatial": dt * n_all / len(rows), "spatial_rows_timed": int(len(rows))}
    t0 = time.perf_counter()
    V = orc.score_temporal(tr.h_t, tr.h_prev)
    out["temporal"] = time.perf_counter() - t0
    t0 = time.perf_counter()
    S = orc.fuse(A, V, tr.alpha)
    _, mask, _ = orc.topk(S, tr.k)
    out["fuse_topk"] = time.perf_counter() - t0
    mname = mode or tr.mode
    t0 = time.perf_counter()
    mixed, pos, span, _, _ = orc.selective_upsample(tr.latent, tr.grid_h, tr.grid_w, mask,
                                                    pos_in=tr.pos_in, span_in=tr.span_in,
                                                    mode=mname)
    out["upsample"] = time.perf_counter() - t0
    t0 = time.perf_counter()
    orc.merge_final(mixed, pos, span, 2 * tr.frame_h, 2 * tr.frame_w, mode=mname)
    out["merge"] = time.perf_counter() - t0
    out["total"] = sum(out[k] for k in ("spatial", "temporal", "fuse_topk", "upsample", "merge"))
    out["_mixed"] = (mixed, pos, span)
    return out


def _rounded(d):
    return {k: (round(v, 6) if isinstance(v, float) else v) for k, v in d.items()
            if not k.startswith("_")}


def cpu_baseline_detail(orc, cores):
    """The oracle per stage and per configuration, at one thread and at all
    host cores: seconds per stage of one transition and transitions/s.  The
    batched multi-stage schedule (B = 8) is its two transitions plus the
    final merge, reported per schedule and per transition."""
    from paper_2608_17995_gb300.workloads import make_batched_stage2, make_transition
    cfgs = [("tiny", "tiny", None), ("flux1024", "flux1024", "nearest"),
            ("flux1024_bilinear", "flux1024", "bilinear"), ("flux2048", "flux2048", None),
            ("edit", "edit", None)]
    trs = {name: make_transition(name) for name in ("tiny", "flux1024", "flux2048", "edit",
                                                    "batched")}
    out = {}
    for nthreads in (1, cores):
        orc.set_threads(nthreads)
        key = "threads_%d" % nthreads
        for label, name, mode in cfgs:
            st = oracle_stage_times(trs[name], orc, mode=mode)
            e = _rounded(st)
            e["transitions_per_s"] = round(1.0 / st["total"], 4)
            out.setdefault(label, {})[key] = e
        # batched schedule: transition 1, transition 2 on its mixed output, merge
        t1 = trs["batched"]
        st1 = oracle_stage_times(t1, orc)
        mixed, pos, span = st1["_mixed"]
        t2 = make_batched_stage2(pos, span, frame=2 * t1.frame_h, latent=mixed)
        st2 = oracle_stage_times(t2, orc)
        sched = st1["total"] - st1["merge"] + st2["total"]
        out.setdefault("batched", {})[key] = {
            "transition1": _rounded(st1), "transition2": _rounded(st2),
            "schedule_s": round(sched, 6), "schedules_per_s": round(1.0 / sched, 4),
            "transitions_per_s": round(2 * t1.B / sched, 4)}
    orc.set_threads(cores)
    return out


def cpu_baseline(tr, orc, cores):
    """The bench line's cpu_baseline: the oracle's FLUX-1024 transition at all
    host cores (and at one thread), per stage timed as oracle_stage_times
    does, averaged over repeats until ~budget seconds."""
    def run(nthreads, budget_s):
        orc.set_threads(nthreads)
        tot, n, t_start = 0.0, 0, time.perf_counter()
        while True:
            tot += oracle_stage_times(tr, orc)["total"]
            n += 1
            if time.perf_counter() - t_start > budget_s or n >= 20:
                break
        return tot / n, n
    per_all, n_all = run(cores, 6.0)
    per_one, n_one = run(1, 4.0)
    orc.set_threads(cores)
    return {"value": round(1.0 / per_all, 4), "unit": UNIT, "cores": cores, "kind": "oracle",
            "value_1thread": round(1.0 / per_one, 4),
            "sample": "%d (all cores) and %d (one thread) oracle runs of the FLUX-1024 "
                      "transition: temporal score, fuse + top-k, upsample and merge in full, "
                      "the spatial score timed on an evenly spaced sample of the 1024 image "
                      "rows (all 24 heads, all 1536 keys) and scaled to all rows"
                      % (n_all, n_one)}


def run_reference(args, world, rank, pg):
    """The oracle timed as it stands (bench's reference arm): every timed step
    is one oracle transition of the FLUX-1024 workload on all host cores, and
    ms_per_step is the measured wall time per step.  When K + W full
    transitions would not fit in ~150 s, each step scores only an evenly
    spaced 1/f of the image rows (f a power of two), the value then being the
    transition rate with the spatial time scaled by f (stated in `sample`)."""
    from paper_2608_17995_gb300.workloads import make_transition
    import numpy as np
    import oracle as orc
    orc.build()
    if rank != 0:
        return None
    cores = orc.threads()
    orc.set_threads(cores)
    tr = make_transition(WORKLOAD)
    K, W = args.steps, args.warmup
    rows_all = np.arange(tr.B * tr.M, dtype=np.int32)

    def one(rows):
        t0 = time.perf_counter()
        A, _, _ = orc.score_spatial(tr.q_img, tr.k_all, tr.L, tr.softmax_scale, rows=rows)
        t1 = time.perf_counter()
        V = orc.score_temporal(tr.h_t, tr.h_prev)
        S = orc.fuse(A, V, tr.alpha)
        _, mask, _ = orc.topk(S, tr.k)
        mixed, pos, span, _, _ = orc.selective_upsample(tr.latent, tr.grid_h, tr.grid_w, mask)
        orc.merge_final(mixed, pos, span, 2 * tr.grid_h, 2 * tr.grid_w)
        t2 = time.perf_counter()
        return t1 - t0, t2 - t1

    sp, rest = one(rows_all)          # calibration (untimed)
    frac = 1
    while (K + W) * (sp / frac + rest) > 150.0 and frac < 64:
        frac *= 2
    rows = rows_all[::frac]
    for _ in range(W):
        one(rows)
    tsp, trest = 0.0, 0.0
    t0 = time.perf_counter()
    for _ in range(K):
        a, b = one(rows)
        tsp += a
        trest += b
    wall = time.perf_counter() - t0
    per = (frac * tsp + trest) / K        # seconds per whole transition
    value = 1.0 / per
    sample = ("each step: the oracle FLUX-1024 transition on %d threads (%s); ms_per_step is "
              "the measured wall time per step" %
              (cores, "all image rows" if frac == 1 else
               "the spatial score on 1/%d of the image rows, the rest in full; value = "
               "transitions/s with the spatial time x %d" % (frac, frac)))
    cfg = {"workload": WORKLOAD_STR % "nearest", "global_batch": 1,
           "parallelism": "host cores x%d" % cores}
    return {"impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": UNIT,
            "n_gpus": world, "steps": K, "warmup": W,
            "ms_per_step": round(wall / K * 1e3, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": cfg,
            "cpu_baseline": {"value": round(value, 4), "unit": UNIT, "cores": cores,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 4), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0},
            "wall_s": round(wall, 3), "rows_fraction": 1.0 / frac}


def main():
    args = _args()
    world, rank, local, pg = dist_setup(args.gpus)
    if args.impl == "reference":
        res = run_reference(args, world, rank, pg)
        if res is not None:
            print(json.dumps(res), flush=True)
        if pg is not None:
            pg.destroy_process_group()
        return 0
    res, tr = run_ours(args, world, rank, local, pg)
    if rank == 0:
        if world == 1 and not args.no_cpu_baseline:
            import oracle as orc
            orc.build()
            cores = orc.threads()
            res["cpu_baseline"] = cpu_baseline(tr, orc, cores)
            if not args.quick:
                res["cpu_baseline_detail"] = cpu_baseline_detail(orc, cores)
        print(json.dumps(res), flush=True)
    if pg is not None:
        pg.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
