"""Benchmark of the KQ hot path on GB300: kernel x codeword distance evals/s.

One step = one pass of the whole hot path over the 2048x2048 stress layer
(n = 4,194,304 kernels, K = 65,536 codewords, 10 Lloyd iterations) through the
entry points a user calls: kq_init_codebook (codebook from seeded kernels),
kq_fit_codebook (10 x (assignment + centroid update), the final assignment and
its cluster sizes), kq_quantize_codebook_6bit, kq_reconstruct (K+C). The metric
counts (iters + 1) * n * K distance evaluations per step.

Default (impl "kq"): the CUDA path through the C ABI, inputs resident in HBM
(the 151 MB weight matrix is larger than the 129 MB L2, so no flush is needed),
timed with CUDA events on the launching stream; a kernel trace (kq_trace_*)
times every kernel of the timed steps on its stream, from which the rooflines
come. "e2e" re-times the same calls with the weights coming from pinned host
memory and every output copied back. --impl reference times the CPU oracle on a
bounded row sample of the same workload on the host cores.

Multi-GPU (torchrun): the path does not shard here, so every rank runs an
independent replica; value = all ranks' evals / max-over-ranks time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "kernel x codeword distance evals/s per Lloyd iteration"
UNIT = "evals/s"
SM_COUNT_NOMINAL = 152
FP32_LANES_PER_SM = 128
DIRECT_OPS_PER_PAIR = 18  # the fp32 direct form: 9 FSUB + 9 FFMA
METHOD_FLOPS_PER_PAIR = 18  # the contraction of Eq. 1's distance: the 9-term dot product x . c
# What the tensor-core assign executes per pair: an (n x 32) . (32 x K) split-fp16 GEMM, 2 * 32 flops.
GEMM_FLOPS_PER_PAIR = 64
WORKLOAD_CFG = 5


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f)
    except OSError:
        return {}


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu = gpu_id
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            p = [x.strip() for x in ln.split(",")]
            if len(p) < 7:
                continue
            try:
                sm.append(float(p[0]))
                mx = float(p[1])
            except ValueError:
                continue
            for nm, v in zip(names, p[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


def replica_throughput(local_ms: float, units_per_step: float, steps: int, world: int, device):
    """Weak scaling of independent replicas: (all ranks' units / max-over-ranks
    seconds, max-over-ranks ms). Needs an initialised process group when world > 1
    (NCCL with a CUDA device, or gloo with the CPU)."""
    import torch
    import torch.distributed as dist

    t = torch.tensor([local_ms], dtype=torch.float64, device=device)
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    ms_max = float(t.item())
    return world * steps * units_per_step / (ms_max / 1e3), ms_max


def _ncu_traffic():
    """Per-launch DRAM bytes (read + write) from the committed ncu summary, or {}."""
    out = {}
    try:
        with open(os.path.join(ROOT, "profiles", "ncu_traffic.txt")) as f:
            for line in f:
                p = line.split()
                if len(p) >= 2 and not line.startswith("#"):
                    out[p[0]] = int(p[1])
    except (OSError, ValueError):
        return {}
    return out


def _smi_id(dev) -> str:
    """nvidia-smi -i argument for a torch device (its UUID when torch exposes it)."""
    import torch

    props = torch.cuda.get_device_properties(dev)
    uuid = getattr(props, "uuid", None)
    if uuid is not None:
        u = str(uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        return vis.split(",")[dev.index or 0]
    return str(dev.index or 0)


def _cpu_sample(W, C, seconds: float, threads: int):
    """Time the oracle's assignment on a seeded row sample sized for ~`seconds`."""
    import oracle

    rows_all = synth.below(synth.stream_key(4242, 9), 1 << 20, W.shape[0])
    probe = 64
    t0 = time.perf_counter()
    oracle.assign(W[rows_all[:probe]], C, threads=threads)
    dt = max(time.perf_counter() - t0, 1e-3)
    rows = int(min(len(rows_all), max(probe, probe * seconds / dt)))
    rows = max(threads, rows - rows % threads)
    t0 = time.perf_counter()
    oracle.assign(W[rows_all[:rows]], C, threads=threads)
    dt = time.perf_counter() - t0
    return rows, dt


def _cpu_lloyd_iteration(wl, seconds: float):
    """The oracle's ms per Lloyd iteration of a whole workload on the host cores: per
    layer, its assignment timed on a seeded row sample (rows are independent) and
    scaled to every row, plus its update over every row."""
    import oracle

    threads = oracle.default_threads()
    per_layer = max(0.05, seconds / len(wl.layers))
    total_ms, sampled, rows_all = 0.0, 0, 0
    for lay in wl.layers:
        W, sel = synth.layer_inputs(lay)
        C0 = oracle.gather_rows(W, sel)
        n = W.shape[0]
        rows, dt = _cpu_sample(W, C0, per_layer, threads) if n * lay.K > 2e8 else (n, None)
        if dt is None:
            t0 = time.perf_counter()
            idx, _ = oracle.assign(W, C0, threads=threads)
            dt = time.perf_counter() - t0
        else:
            idx = synth.below(synth.stream_key(lay.seed, 17), n, lay.K).astype(np.int32)
        t0 = time.perf_counter()
        oracle.update(W, idx, C0)
        du = time.perf_counter() - t0
        total_ms += 1e3 * (dt * n / rows + du)
        sampled += rows
        rows_all += n
    return {"ms_per_lloyd_iter": total_ms, "cores": threads, "kind": "oracle",
            "sample": f"assignment timed on {sampled} of {rows_all} rows and scaled to all; update over every row "
                      f"(indices: the oracle's own where every row was assigned, else seeded)"}


def run_reference(args, rank, world):
    """CPU oracle on the host cores (rank 0 only)."""
    if rank != 0:
        return
    import oracle

    lay = synth.workload(WORKLOAD_CFG).layers[0]
    W, sel = synth.layer_inputs(lay)
    C0 = oracle.gather_rows(W, sel)
    threads = oracle.default_threads()
    per_step = []
    rows = None
    for s in range(args.warmup + args.steps):
        rows, dt = _cpu_sample(W, C0, args.ref_seconds, threads)
        if s >= args.warmup:
            per_step.append((rows, dt))
    pairs = sum(r for r, _ in per_step) * lay.K
    secs = sum(d for _, d in per_step)
    value = pairs / secs
    sample = (f"assign step of the oracle (the step holding ~all of the work) on {rows} seeded rows of the "
              f"{lay.n}-kernel layer against all K={lay.K} codewords, per step")
    out = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * secs / len(per_step), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": "stress_2048x2048_K65536_T10", "n": lay.n, "K": lay.K, "iters": 10},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(out), flush=True)


def _trace_summary(trace, steps):
    """Per kernel: launches, total device ms and share of the traced time."""
    tot = sum(ms for _, ms in trace) or 1.0
    out = {}
    for name, ms in trace:
        d = out.setdefault(name, {"launches": 0, "ms_total": 0.0})
        d["launches"] += 1
        d["ms_total"] += ms
    for d in out.values():
        d["share"] = round(d["ms_total"] / tot, 5)
        d["ms_per_step"] = round(d["ms_total"] / steps, 4)
        d["ms_total"] = round(d["ms_total"], 4)
    return dict(sorted(out.items(), key=lambda kv: -kv[1]["ms_total"]))


def run_kq(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist

    from paper_2003_05148_gb300 import build, kq

    build.build()
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    lay = synth.workload(WORKLOAD_CFG).layers[0]
    T = synth.workload(WORKLOAD_CFG).iters
    n, K = lay.n, lay.K
    W_h, sel_h = synth.layer_inputs(lay)
    stream = torch.cuda.current_stream()

    W = torch.from_numpy(W_h).to(dev)
    sel = torch.from_numpy(sel_h).to(dev)
    ws = kq.workspace(n, K, dev)
    C0 = torch.empty(K, 9, dtype=torch.float32, device=dev)
    C = torch.empty_like(C0)
    idx = torch.empty(n, dtype=torch.int32, device=dev)
    counts = torch.empty(K, dtype=torch.int32, device=dev)
    obj = torch.empty(T + 1, dtype=torch.float64, device=dev)
    levels = torch.empty(64, dtype=torch.float32, device=dev)
    codes = torch.empty(K, 9, dtype=torch.uint8, device=dev)
    Wr = torch.empty_like(W)

    def pair():
        return (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))

    def step(rec=None):
        """One pass of the hot path through the entry points a user calls: codebook
        init, the k-means fit (T updates and the final assignment), 6-bit codebook
        quantisation, K+C recovery. `rec` brackets the recovery call."""
        kq.kq_init_codebook(W, sel, C0, ws)
        kq.kq_fit_codebook(W, C0, T, C, idx, counts, obj, ws)
        kq.kq_quantize_codebook_6bit(C, counts, 100, levels, codes, None, ws)
        if rec:
            rec[0].record(stream)
        kq.kq_reconstruct(idx, None, codes, levels, Wr, ws, K=K)
        if rec:
            rec[1].record(stream)

    l0 = kq.kq_kernel_launches()
    for _ in range(args.warmup):
        step()
    per_step_launches = (kq.kq_kernel_launches() - l0) // max(1, args.warmup)
    st, flags = kq.kq_device_status(ws)
    if st != 0:
        raise RuntimeError(f"device status {st} flags {flags:#x} after warm-up")

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    recs = [pair() for _ in range(args.steps)]
    # every kernel of the timed steps gets a pair of events on its launch stream
    kq.kq_trace_start(per_step_launches * args.steps + 64)
    launches0 = kq.kq_kernel_launches()
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(_smi_id(dev)) as clocks:
        e0.record(stream)
        for s in range(args.steps):
            step(recs[s])
        e1.record(stream)
        barrier()
    kq.kq_trace_stop()
    launches = kq.kq_kernel_launches() - launches0
    ms_total = e0.elapsed_time(e1)
    trace = kq.kq_trace_read()
    rec_ms = [a.elapsed_time(b) for a, b in recs]
    pairs_per_step = (T + 1) * n * K
    value, ms_max = replica_throughput(ms_total, pairs_per_step, args.steps, world, dev)

    st, flags = kq.kq_device_status(ws)
    if st != 0:
        raise RuntimeError(f"device status {st} flags {flags:#x} after the timed steps")

    # the standalone update call (every row accumulated: the step of Eq. 1 as defined),
    # on the fit's final assignment, for its HBM roofline
    Cn = torch.empty_like(C)
    cnt2 = torch.empty_like(counts)
    upd = [pair() for _ in range(args.update_reps)]
    kq.kq_trace_start(8 * args.update_reps + 8)
    for a, b in upd:
        a.record(stream)
        kq.kq_update_centroids(W, idx, C, Cn, cnt2, ws)
        b.record(stream)
    torch.cuda.synchronize()
    kq.kq_trace_stop()
    upd_trace = kq.kq_trace_read()
    upd_ms = [a.elapsed_time(b) for a, b in upd]

    # ---- end to end through the same calls: pinned host in, every output back ----
    W_pin = torch.from_numpy(W_h).pin_memory()
    sel_pin = torch.from_numpy(sel_h).pin_memory()
    outs = {"C": torch.empty(K, 9, dtype=torch.float32).pin_memory(),
            "idx": torch.empty(n, dtype=torch.int32).pin_memory(),
            "counts": torch.empty(K, dtype=torch.int32).pin_memory(),
            "levels": torch.empty(64, dtype=torch.float32).pin_memory(),
            "codes": torch.empty(K, 9, dtype=torch.uint8).pin_memory(),
            "Wr": torch.empty(n, 9, dtype=torch.float32).pin_memory(),
            "objective": torch.empty(T + 1, dtype=torch.float64).pin_memory()}
    # Steps are pipelined over two buffer sets: step s computes on the default stream
    # while a copy stream brings in step s + 1's inputs and reads out step s - 1's
    # outputs (events order each copy against the compute that produces or consumes
    # its buffers). Every step's inputs still cross from pinned host memory and all
    # its outputs come back inside the timed region.
    main = torch.cuda.current_stream(dev)
    cs = torch.cuda.Stream(dev)
    bufs = [{"W": torch.empty_like(W), "sel": torch.empty_like(sel),
             "C0": torch.empty(K, 9, dtype=torch.float32, device=dev),
             "C": torch.empty(K, 9, dtype=torch.float32, device=dev),
             "idx": torch.empty(n, dtype=torch.int32, device=dev),
             "counts": torch.empty(K, dtype=torch.int32, device=dev),
             "levels": torch.empty(64, dtype=torch.float32, device=dev),
             "codes": torch.empty(K, 9, dtype=torch.uint8, device=dev),
             "Wr": torch.empty_like(W),
             "objective": torch.empty(T + 1, dtype=torch.float64, device=dev)} for _ in range(2)]
    ev = {k: [torch.cuda.Event() for _ in range(2)] for k in ("in", "used", "out")}

    def e2e_run(steps):
        def fetch(s):
            b = bufs[s % 2]
            with torch.cuda.stream(cs):
                if s >= 2:
                    cs.wait_event(ev["used"][s % 2])  # step s - 2 is done with these inputs
                b["W"].copy_(W_pin, non_blocking=True)
                b["sel"].copy_(sel_pin, non_blocking=True)
                ev["in"][s % 2].record(cs)

        fetch(0)
        for s in range(steps):
            b = bufs[s % 2]
            if s + 1 < steps:
                fetch(s + 1)
            main.wait_event(ev["in"][s % 2])
            if s >= 2:
                main.wait_event(ev["out"][s % 2])  # step s - 2's outputs have been read out
            kq.kq_init_codebook(b["W"], b["sel"], b["C0"], ws)
            kq.kq_fit_codebook(b["W"], b["C0"], T, b["C"], b["idx"], b["counts"], b["objective"], ws)
            kq.kq_quantize_codebook_6bit(b["C"], b["counts"], 100, b["levels"], b["codes"], None, ws)
            kq.kq_reconstruct(b["idx"], None, b["codes"], b["levels"], b["Wr"], ws, K=K)
            ev["used"][s % 2].record(main)
            with torch.cuda.stream(cs):
                cs.wait_event(ev["used"][s % 2])
                for name in outs:
                    outs[name].copy_(b[name], non_blocking=True)
                ev["out"][s % 2].record(cs)

    e2e_steps = args.e2e_steps if args.e2e_steps > 0 else args.steps
    e2e_run(1)
    torch.cuda.synchronize()
    barrier()
    t0 = time.perf_counter()
    e2e_run(e2e_steps)
    torch.cuda.synchronize()
    e2e_s = time.perf_counter() - t0
    e2e_value, _ = replica_throughput(1e3 * e2e_s, pairs_per_step, e2e_steps, world, dev)
    h2d = W_pin.numel() * 4 + sel_pin.numel() * 8
    d2h = sum(t.numel() * t.element_size() for t in outs.values())
    # the e2e fit must give what the device-timed one gave (same inputs, deterministic)
    if not (torch.equal(outs["idx"], idx.cpu()) and torch.equal(outs["Wr"], Wr.cpu())):
        raise RuntimeError("end-to-end outputs differ from the device-timed step's")

    if rank != 0:
        return
    peaks = _peaks()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    clk = clocks.summary()
    max_mhz = float(peaks.get("sm_max_mhz", 2070.0))
    fp32_peak = sms * FP32_LANES_PER_SM * max_mhz * 1e6 / 1e12
    traffic = _ncu_traffic()
    kernels = _trace_summary(trace, args.steps)
    tc_ms = [ms for name, ms in trace if name == "assign_tc_kernel"]
    cc_ms = [ms for name, ms in trace if name == "assign_kernel"]
    if tc_ms:
        # kernel timed inside a long step: the sustained bf16 figure (fp16 runs at the bf16 rate)
        bf16 = float(peaks.get("bf16_tflops_sustained", peaks.get("bf16_tflops", 1700.0)))
        per_step = len(tc_ms) // args.steps
        pilots = per_step - (T + 1)  # the cold first assignment's pilot pass (K / 16 codewords)
        full = [ms for i, ms in enumerate(tc_ms) if i % per_step >= pilots]
        t_step = sum(tc_ms) / args.steps / 1e3  # s of tensor-core assign per step, pilot included
        achieved = METHOD_FLOPS_PER_PAIR * pairs_per_step / t_step / 1e12
        gemm_pairs = n * (K * (T + 1) + pilots * (K // 16))
        gemm = GEMM_FLOPS_PER_PAIR * gemm_pairs / t_step / 1e12
        roofline = {
            "bound": "tensor", "achieved": achieved, "peak": bf16, "unit": "TFLOP/s", "frac": achieved / bf16,
            "traffic": traffic.get("assign_tc_kernel"), "kernel": "assign_tc_kernel",
            "work": f"{METHOD_FLOPS_PER_PAIR} flops per kernel x codeword pair (the 9-term dot product x . c of "
                    f"Eq. 1's distance), (T + 1) n K = {pairs_per_step:.4g} pairs per step, over the device time "
                    f"of every assign_tc_kernel launch of the step (the cold pass's pilot included)",
            "peak_basis": f"measured cuBLAS bf16 sustained {bf16:.1f} TFLOP/s (of measured; dense fp16 and bf16 "
                          f"share one rate); the kernel is timed inside the long step",
            "launches": len(tc_ms), "ms_mean": statistics.mean(tc_ms),
            "ms_mean_full_pass": statistics.mean(full),
            # the first full pass of a step starts from k-d leaf hints (cold), the later T from the
            # previous assignment (warm)
            "ms_first_pass": statistics.mean(full[0::T + 1]),
            "ms_warm_pass": statistics.mean([ms for i, ms in enumerate(full) if i % (T + 1)]) if T else None,
            "ms_mean_pilot": statistics.mean(
                [ms for i, ms in enumerate(tc_ms) if i % per_step < pilots]) if pilots > 0 else None,
            "frac_of_burst": achieved / float(peaks.get("bf16_tflops", bf16)),
            "gemm": {"flops_per_pair": GEMM_FLOPS_PER_PAIR, "achieved": gemm, "frac_of_peak": gemm / bf16,
                     "overhead_vs_method": GEMM_FLOPS_PER_PAIR / METHOD_FLOPS_PER_PAIR,
                     "note": "what the tensor core executes: the split-fp16 test GEMM, K = 32 fp16 per row "
                             "(three cross terms of the hi/lo split plus the threshold slots; 27 of 32 used), "
                             "pilot pairs included; the exact fp32 re-evaluations of candidate pairs run on the "
                             "CUDA cores and are not counted"},
        }
    else:
        t_step = sum(cc_ms) / args.steps / 1e3
        achieved = DIRECT_OPS_PER_PAIR * pairs_per_step / t_step / 1e12
        roofline = {"bound": "alu", "achieved": achieved, "peak": fp32_peak, "unit": "Tops/s",
                    "frac": achieved / fp32_peak, "traffic": traffic.get("assign_kernel"), "kernel": "assign_kernel",
                    "peak_basis": f"{sms} SMs x {FP32_LANES_PER_SM} FP32 lanes x {max_mhz:.0f} MHz",
                    "launches": len(cc_ms)}
    roofline["direct_form_equivalent"] = {
        "achieved_tops": DIRECT_OPS_PER_PAIR * pairs_per_step / t_step / 1e12,
        "frac_of_fp32_peak": DIRECT_OPS_PER_PAIR * pairs_per_step / t_step / 1e12 / fp32_peak,
        "note": "18 FP32 lane ops per pair (9 FSUB + 9 FFMA): the rate a direct-form CUDA-core kernel would "
                f"need for the same time, against {sms} x {FP32_LANES_PER_SM} lanes x {max_mhz:.0f} MHz"}
    hbm = float(peaks.get("hbm_gbs", 6776.3))

    def hbm_roofline(kernel, bytes_per_launch, ms_list, note, call_bytes, call_ms, call_note):
        # the dominant kernel's launches (CUDA events on its stream), and the whole call beside it
        t = statistics.mean(ms_list) / 1e3
        a = bytes_per_launch / t / 1e9
        tc = statistics.mean(call_ms) / 1e3
        ac = call_bytes / tc / 1e9
        return {"bound": "hbm", "achieved": a, "peak": hbm, "unit": "GB/s", "frac": a / hbm, "target_frac": 0.6,
                "target_met": a / hbm >= 0.6,
                "traffic": traffic.get(kernel), "kernel": kernel, "launches": len(ms_list), "us_mean": 1e6 * t,
                "algorithmic_bytes": int(bytes_per_launch), "note": note,
                "whole_call": {"us_mean": 1e6 * tc, "calls": len(call_ms), "algorithmic_bytes": int(call_bytes),
                               "achieved": ac, "frac": ac / hbm, "note": call_note}}

    acc_ms = [ms for name, ms in upd_trace if name == "accumulate_kernel"]
    gat_ms = [ms for name, ms in trace if name == "gather_codes_kernel"]
    roofline_update = hbm_roofline(
        "accumulate_kernel", n * (36 + 4) + K * 80, acc_ms,
        "accumulate_kernel of standalone kq_update_centroids calls on the fit's final assignment, after the timed "
        "steps: reads W and idx once (40 B per kernel), every codeword's ten 64-bit sums written once (80 B)",
        n * (36 + 4) + K * (36 + 36 + 4), upd_ms,
        "the whole call (prepare + accumulate + fallback check + finalize); inside the fit the update moves only "
        "the rows whose codeword changed (see kernels)")
    roofline_reconstruct = hbm_roofline(
        "gather_codes_kernel", n * (4 + 36) + 8 * K + 256, gat_ms,
        "gather_codes_kernel of every timed step (K+C recovery): 4 B index read and 36 B written per kernel, the "
        "8 B packed code word per codeword and the 256 B level table read once",
        n * (4 + 36) + 9 * K + 256, rec_ms, "the whole kq_reconstruct call (decode codes + gather)")
    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms_max / args.steps, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32", "data": "synthetic",
        "config": {"workload": "stress_2048x2048_K65536_T10", "n": n, "K": K, "iters": T,
                   "step": "kq_init_codebook + kq_fit_codebook (10 updates, final assignment, counts) + "
                           "kq_quantize_codebook_6bit + kq_reconstruct (K+C)",
                   "l2": "inputs larger than L2 (W is 151 MB, L2 129 MB): no flush",
                   "parallelism": f"replicas x{world}"},
        "roofline": roofline,
        "roofline_update": roofline_update,
        "roofline_reconstruct": roofline_reconstruct,
        "kernels": kernels,
        "gpu_launches": int(launches),
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
                "steps": e2e_steps, "api": "kq_init_codebook + kq_fit_codebook + kq_quantize_codebook_6bit + "
                                           "kq_reconstruct, pinned host buffers, all outputs copied back; "
                                           "copies on a second stream, overlapped with the neighbouring "
                                           "steps' compute (two buffer sets); host clock"},
    }
    if clk:
        out["clocks"] = clk
    if world == 1 and not args.no_cpu_baseline:
        import oracle

        threads = oracle.default_threads()
        C0_h = oracle.gather_rows(W_h, sel_h)
        rows, dt = _cpu_sample(W_h, C0_h, args.ref_seconds, threads)
        rows1, dt1 = _cpu_sample(W_h, C0_h, min(args.ref_seconds, 3.0), 1)  # and on one core
        out["cpu_baseline"] = {"value": rows * K / dt, "unit": UNIT, "cores": threads, "kind": "oracle",
                               "sample": f"oracle assign (the step holding ~all of the work) of {rows} seeded rows "
                                         f"against all K={K} codewords ({rows * K:.3g} evals, {dt:.1f} s)",
                               "value_1core": rows1 * K / dt1,
                               "sample_1core": f"{rows1} rows on one thread ({dt1:.1f} s)"}
    print(json.dumps(out), flush=True)


def run_only(args):
    """One hot-path step on its own, for profiler captures: synthetic stress-layer
    inputs with n / K overridden, `reps` launches of the chosen entry point."""
    import torch

    from paper_2003_05148_gb300 import build, kq

    build.build()
    dev = torch.device("cuda", 0)
    base = synth.workload(WORKLOAD_CFG).layers[0]
    p = base.p if args.n % base.p == 0 else 1
    lay = synth.Layer("profile", p, args.n // p, args.K, min(4 * args.K, args.n), base.seed)
    W_h, sel_h = synth.layer_inputs(lay)
    n, K = W_h.shape[0], args.K
    W = torch.from_numpy(W_h).to(dev)
    sel = torch.from_numpy(sel_h).to(dev)
    ws = kq.workspace(n, K, dev)
    C = torch.empty(K, 9, dtype=torch.float32, device=dev)
    C2 = torch.empty_like(C)
    kq.kq_init_codebook(W, sel, C, ws)
    idx = torch.empty(n, dtype=torch.int32, device=dev)
    counts = torch.empty(K, dtype=torch.int32, device=dev)
    kq.kq_assign(W, C, idx, None, ws)
    kq.kq_update_centroids(W, idx, C, C2, counts, ws)
    levels = torch.empty(64, dtype=torch.float32, device=dev)
    codes = torch.empty(K, 9, dtype=torch.uint8, device=dev)
    kq.kq_quantize_codebook_6bit(C2, counts, 100, levels, codes, None, ws)
    Wr = torch.empty_like(W)
    idx2 = torch.empty_like(idx)
    calls = {
        # --hint: one Lloyd step later, warm-started from the previous assignment (as in a fit)
        "assign": (lambda: kq.kq_assign(W, C2, idx2, None, ws, hint=idx)) if args.hint
        else (lambda: kq.kq_assign(W, C, idx, None, ws)),
        "update": lambda: kq.kq_update_centroids(W, idx, C, C2, counts, ws),
        "quantize": lambda: kq.kq_quantize_codebook_6bit(C2, counts, 100, levels, codes, None, ws),
        "reconstruct": lambda: kq.kq_reconstruct(idx, None, codes, levels, Wr, ws, K=K),
        "fusedrecon": lambda: kq.kq_quantize_reconstruct(idx, C2, levels, codes, Wr, ws),
    }
    # retraining steps (Eq. 2; Sec. 3.2): the kernels themselves stand in for the
    # gradients (the timing depends on sizes and the code distribution only)
    lv_next = torch.empty(64, dtype=torch.float32, device=dev)
    lv_counts = torch.empty(64, dtype=torch.int64, device=dev)
    calls["gradstep"] = lambda: kq.kq_codebook_grad_step(W, idx, 0.01, C2, C, counts, ws)
    calls["levelgrad"] = lambda: kq.kq_levels_grad_step(W, idx, codes, 0.01, levels, lv_next, lv_counts, ws)
    alg_bytes = {"update": 40 * n + 76 * K, "gradstep": 40 * n + 76 * K, "levelgrad": 40 * n + 9 * K,
                 "reconstruct": 40 * n + 9 * K + 256, "fusedrecon": 40 * n + 45 * K + 256}
    if args.only == "search":
        # Algorithm 1 on the VGG-16 conv3_2 layer (workload 2): alpha = 0.25, r = 0.5,
        # 8 bisection steps, 20 Lloyd updates per trial (the workload's own count)
        lay2 = synth.workload(2).layers[0]
        W2_h, _ = synth.layer_inputs(lay2)
        n2 = W2_h.shape[0]
        n_init = int(np.floor(0.25 * n2))
        sel2 = torch.from_numpy(synth.init_selection(n2, n_init, lay2.seed + 1)).to(dev)
        W2 = torch.from_numpy(W2_h).to(dev)
        C_s = torch.empty(n_init, 9, dtype=torch.float32, device=dev)
        idx_s = torch.empty(n2, dtype=torch.int32, device=dev)
        cnt_s = torch.empty(n_init, dtype=torch.int32, device=dev)
        ws2 = kq.workspace(n2, n_init, dev)
        search_out = {}

        def run_search():
            search_out["r"] = kq.kq_search_codebook_size(W2, sel2, 0.25, 0.5, 8, 20, C_s, idx_s, cnt_s, ws2)

        calls["search"] = run_search
        n, K = n2, n_init
    if args.only == "fcquant":
        # 6-bit quantisation of a fully-connected weight of m scalars (He-scaled
        # Gaussian, seeded), 100 iterations at most
        gen = torch.Generator(device=dev)
        gen.manual_seed(WORKLOAD_CFG * 1000 + 7)
        v = torch.randn(args.m, generator=gen, device=dev) * float(np.sqrt(2.0 / 4096))
        fc_codes = torch.empty(args.m, dtype=torch.uint8, device=dev)
        fc_it = torch.zeros(1, dtype=torch.int32, device=dev)
        calls["fcquant"] = lambda: kq.kq_quantize_scalars_6bit(v, 100, levels, fc_codes, fc_it, ws)
        n, K = args.m, 64
    if args.only in ("fit", "prunefit"):
        # the fit as a user calls it (the workload's iteration count, from the seeded
        # initial codebook), without or with the tile pruning that stands for Yinyang
        T_fit = synth.workload(WORKLOAD_CFG).iters
        C_fit = torch.empty_like(C)
        obj_fit = torch.empty(T_fit + 1, dtype=torch.float64, device=dev)
        fit_flags = kq.FIT_PRUNE if args.only == "prunefit" else 0
        calls[args.only] = lambda: kq.kq_fit_codebook(W, C, T_fit, C_fit, idx2, counts, obj_fit, ws, flags=fit_flags)
    f = calls[args.only]
    # --l2-drain: after every call, outside its events, read a 512 MB buffer (larger
    # than L2), so that the call's dirty L2 lines go to DRAM before the next call
    # starts; a profiler capture of that read then shows the rest of the call's writes
    drain = torch.ones(128 << 20, dtype=torch.float32, device=dev) if args.l2_drain else None
    for _ in range(2):
        f()
        if drain is not None:
            drain.sum()
    torch.cuda.synchronize()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.reps)]
    stream = torch.cuda.current_stream()
    for a, b in evs:
        a.record(stream)
        f()
        b.record(stream)
        if drain is not None:
            drain.sum()
    torch.cuda.synchronize()
    # the work of the last pruned fit (nothing else has run on ws since)
    tiles = kq.kq_fit_prune_stats(ws) if args.only == "prunefit" else None
    st, flags = kq.kq_device_status(ws)
    ms = [a.elapsed_time(b) for a, b in evs]
    out = {"only": args.only, "n": n, "K": K, "reps": args.reps, "ms_mean": statistics.mean(ms),
           "ms_min": min(ms), "status": st, "flags": flags, "l2_drain": bool(args.l2_drain)}
    if args.only in alg_bytes:
        out["alg_bytes"] = alg_bytes[args.only]
        out["GB_s_at_min"] = alg_bytes[args.only] / (min(ms) * 1e-3) / 1e9
    if args.only == "search":
        k_s, e_s, tr_s = search_out["r"]
        out["K_chosen"], out["error"], out["trials"] = k_s, e_s, len(tr_s)
        out["trace"] = [[a, round(b, 6)] for a, b in tr_s]
    if args.only in ("fit", "prunefit"):
        evals = (T_fit + 1) * n * K  # kernel x codeword distances the fit's assignments decide
        out["iters"] = T_fit
        out["effective_evals_per_s"] = evals / (statistics.mean(ms) * 1e-3)
        if tiles is not None:
            tiles_run, tiles_all = tiles
            out["tiles_run"], out["tiles_all"] = tiles_run, tiles_all
            frac = tiles_run / tiles_all if tiles_all else 1.0
            out["executed_fraction"] = frac
            # (256-kernel block, 256-codeword tile) pairs the tensor core processed
            out["executed_evals_per_s"] = frac * out["effective_evals_per_s"]
    if args.only == "fcquant":
        it = int(fc_it.item())
        out["iters_run"] = it
        out["ms_per_iter"] = min(ms) / max(it, 1)
    print(json.dumps(out), flush=True)
    if st != 0:
        sys.exit(1)


def run_configs(args):
    """Every configuration (the five seeded workloads) through the public API on one
    GPU: per layer kq_init_codebook + kq_fit_codebook (the workload's iteration
    count) + kq_quantize_codebook_6bit + K+C kq_reconstruct, inputs resident in HBM,
    CUDA events around `reps` runs of the whole workload after one untimed run.
    Prints one JSON line per configuration (a report, not the bench line)."""
    import torch

    from paper_2003_05148_gb300 import build, kq

    build.build()
    dev = torch.device("cuda", 0)
    for cfg in [int(c) for c in args.configs.split(",")]:
        wl = synth.workload(cfg)
        T = wl.iters
        layers = []
        for lay in wl.layers:
            W_h, sel_h = synth.layer_inputs(lay)
            n, K = W_h.shape[0], lay.K
            layers.append({
                "n": n, "K": K,
                "W": torch.from_numpy(W_h).to(dev), "sel": torch.from_numpy(sel_h).to(dev),
                "ws": kq.workspace(n, K, dev),
                "Ca": torch.empty(K, 9, dtype=torch.float32, device=dev),
                "Cb": torch.empty(K, 9, dtype=torch.float32, device=dev),
                "idx": torch.empty(n, dtype=torch.int32, device=dev),
                "counts": torch.empty(K, dtype=torch.int32, device=dev),
                "obj": torch.empty(T + 1, dtype=torch.float64, device=dev),
                "levels": torch.empty(64, dtype=torch.float32, device=dev),
                "codes": torch.empty(K, 9, dtype=torch.uint8, device=dev),
                "Wr": torch.empty(n, 9, dtype=torch.float32, device=dev)})

        # The layers are independent problems: with --streams S > 1 layer i runs on
        # stream i % S (each layer has its own workspace and buffers), so one layer's
        # latency-bound phases overlap another's work.
        stream = torch.cuda.current_stream()
        side = [torch.cuda.Stream(device=dev) for _ in range(args.streams)] if args.streams > 1 else [stream]

        jobs = [{"W": L["W"], "sel": L["sel"], "C": L["Ca"], "idx": L["idx"], "counts": L["counts"],
                 "objective": L["obj"], "levels": L["levels"], "codes": L["codes"], "W_out": L["Wr"], "ws": L["ws"]}
                for L in layers]

        def run_all():
            if args.grouped:  # one kq_fit_layers call: the library spreads the layers over its streams
                kq.kq_fit_layers(jobs, T, 100, 0, stream=stream)
                return
            for s in side:
                s.wait_stream(stream)
            for i, L in enumerate(layers):
                with torch.cuda.stream(side[i % len(side)]):
                    kq.kq_init_codebook(L["W"], L["sel"], L["Ca"], L["ws"])
                    kq.kq_fit_codebook(L["W"], L["Ca"], T, L["Cb"], L["idx"], L["counts"], L["obj"], L["ws"])
                    kq.kq_quantize_codebook_6bit(L["Cb"], L["counts"], 100, L["levels"], L["codes"], None, L["ws"])
                    kq.kq_reconstruct(L["idx"], None, L["codes"], L["levels"], L["Wr"], L["ws"], K=L["K"])
            for s in side:
                stream.wait_stream(s)

        run_all()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        launches0 = kq.kq_kernel_launches()
        e0.record(stream)
        for _ in range(args.reps):
            run_all()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / args.reps
        statuses = [kq.kq_device_status(L["ws"]) for L in layers]
        evals = sum((T + 1) * L["n"] * L["K"] for L in layers)
        rate = evals / (ms / 1e3)
        sms = torch.cuda.get_device_properties(dev).multi_processor_count
        peaks = _peaks()
        bf16 = float(peaks.get("bf16_tflops_sustained", peaks.get("bf16_tflops", 1700.0)))
        max_mhz = float(peaks.get("sm_max_mhz", 2070.0))
        line = {
            "config": wl.name, "layers": len(layers), "kernels": sum(L["n"] for L in layers),
            "codewords": sum(L["K"] for L in layers), "iters": T, "evals": evals, "ms_per_run": ms,
            "ms_per_lloyd_iter": ms / (T + 1), "evals_per_s": rate,
            # whole-run figures (init, fit, 6-bit quantisation and recovery all in the time),
            # so lower bounds for the assignment kernels alone; method work = 18 flops per pair
            "frac_of_tensor_peak": rate * METHOD_FLOPS_PER_PAIR / 1e12 / bf16,
            "direct_form_frac_of_fp32_peak": rate * DIRECT_OPS_PER_PAIR / (sms * FP32_LANES_PER_SM * max_mhz * 1e6),
            "gpu_launches_per_run": (kq.kq_kernel_launches() - launches0) // args.reps,
            "status": max(st for st, _ in statuses), "reps": args.reps,
            "mode": "kq_fit_layers (one call)" if args.grouped else f"per-layer calls on {len(side)} stream(s)"}
        if not args.no_cpu_baseline:
            line["cpu_baseline"] = _cpu_lloyd_iteration(wl, args.ref_seconds)
            line["cpu_baseline"]["speedup_per_lloyd_iter"] = line["cpu_baseline"]["ms_per_lloyd_iter"] / line[
                "ms_per_lloyd_iter"]
        print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["kq", "reference"], default="kq")
    ap.add_argument("--e2e-steps", type=int, default=0, help="end-to-end steps (default: --steps)")
    ap.add_argument("--update-reps", type=int, default=10, help="standalone update calls for its roofline")
    ap.add_argument("--ref-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--only", choices=["assign", "update", "quantize", "reconstruct", "gradstep", "levelgrad",
                                       "fcquant", "search", "fusedrecon", "fit", "prunefit"],
                    help="profiling aid: time one entry point on its own (no bench line)")
    ap.add_argument("--n", type=int, default=4194304)
    ap.add_argument("--K", type=int, default=65536)
    ap.add_argument("--m", type=int, default=25088 * 4096, help="with --only fcquant: scalars (VGG-16 fc6)")
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--hint", action="store_true", help="with --only assign: warm start as in a fit")
    ap.add_argument("--l2-drain", action="store_true",
                    help="with --only: read a 512 MB buffer after every call, outside the timed events")
    ap.add_argument("--streams", type=int, default=1,
                    help="with --configs: independent layers round-robin over this many streams")
    ap.add_argument("--grouped", action="store_true",
                    help="with --configs: all layers of a workload through one kq_fit_layers call")
    ap.add_argument("--configs", default=None,
                    help="report aid: fit the listed workloads (e.g. 1,2,3,4,5) end to end, one line each")
    args = ap.parse_args()
    if args.only:
        run_only(args)
        return
    if args.configs:
        run_configs(args)
        return
    if args.warmup < 3:
        print("warning: fewer than 3 warm-up steps", file=sys.stderr)
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if world > 1:
        import torch
        import torch.distributed as dist

        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    try:
        run_kq(args, rank, world, local_rank)
    finally:
        if world > 1:
            import torch.distributed as dist

            dist.destroy_process_group()


if __name__ == "__main__":
    main()
