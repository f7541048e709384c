"""Attention-forward benchmark on GB300: TFLOP/s, ms per call, roofline fraction.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

One step = one attention forward (one vdx_attn_fwd / vdx_attn_fwd_varlen /
vdx_attn_fwd_segments / vdx_attn_fwd_win3d / vdx_attn_fwd_rope3d call) over
the whole workload, inputs
resident in HBM.  The default workload is the largest single-GPU
configuration, the large-DiT 720p self-attention (B=1, H=40, D=128,
S = 21*45*80 = 75600 tokens).  FLOPs = 4*B*H*Sq*Skv*D
(effective key counts for the padded-text workload; the (query, key) pairs
of equal segment id for the joint text-video workload; the (query, key)
pairs inside the windows for the windowed workload).

Timing: W untimed warm-up steps, then K steps bracketed by a barrier and a
device synchronisation, timed with CUDA events on the launching stream; the
max over ranks is reported.  Inputs (large720's Q, K, V and O: 3.1 GB)
exceed the 129 MB L2, so no flush is inserted.  SM clocks are sampled with nvidia-smi during
the timed region.  A second timed pass ("e2e") starts from pinned host
buffers: every step copies Q, K, V host->device, runs the kernel and copies
O and LSE back.  Each step is one host-buffer call (vdx_attn_fwd_host, or its
segment, window or RoPE variant): the library cuts the (b, h) rows into
chunks and overlaps the copies with the kernels.

--impl reference times the fp64 CPU oracle (the only reference this
method has) on a bounded row sample of the same workload.  Under torchrun
(N > 1) each rank runs its own copy of the workload (independent problems:
weak scaling, no collective on the data path).  --gpus N > 1 outside torchrun
relaunches this script under torch.distributed.run with N processes; inside
torchrun it must equal WORLD_SIZE.
"""
from __future__ import annotations

import argparse
import csv
import io
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "attention fwd TFLOP/s and ms/call at 1 GB300; fraction of dense bf16 peak"
UNIT = "TFLOP/s"
FALLBACK_PEAKS = {"bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "hbm_gbs": 6800.0}


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def dist_env():
    return int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")), \
        int(os.environ.get("LOCAL_RANK", "0"))


def max_over_ranks(x, world, device=None):
    """Max of a host float over all ranks (identity for one rank); any backend."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


class ClockSampler:
    """nvidia-smi clock / throttle-reason sampling around the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int, log_path: str | None = None):
        self.index = index
        self.proc = None
        self.log_path = log_path

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        self.text = ""
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.text, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.text, _ = self.proc.communicate()
        if self.log_path:
            with open(self.log_path, "w") as f:
                f.write(self.text)
        return False

    def summary(self, max_mhz_hint=None):
        rows = [r for r in csv.reader(io.StringIO(self.text)) if len(r) >= 9]
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
            except ValueError:
                continue
            for name, val in zip(names, r[5:9]):
                if val.strip().lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": max_mhz_hint, "reasons": [], "samples": 0}
        # samples under load: the timed region dominates the window
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx) if mx else max_mhz_hint,
                "reasons": sorted(reasons), "samples": len(sm)}


def make_inputs(name):
    from paper_2609_18077_gb300 import workloads
    w = workloads.generate(name)
    flops = w["workload"].flops(w["kv_lens"], w["q_seg"], w["kv_seg"])
    return w, flops


def run_ours(args):
    import torch
    import torch.distributed as dist
    from paper_2609_18077_gb300 import binding

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)

    w, flops = make_inputs(args.workload)
    wl = w["workload"]
    q, k, v = (t.to(dev) for t in (w["q"], w["k"], w["v"]))
    lens = None if w["kv_lens"] is None else torch.from_numpy(w["kv_lens"]).to(dev)
    segs = None if w["q_seg"] is None else tuple(torch.from_numpy(w[n]).to(dev) for n in ("q_seg", "kv_seg"))
    out = torch.empty_like(q)
    lse = torch.empty(q.shape[:3], dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    # kernels of ours per step: the segment path builds its key-tile lists first
    launches_per_step = 3 if segs is not None else 1
    mode = "seg" if segs is not None else ("varlen" if lens is not None else "dense")
    if wl.window is not None:
        mode = "win"
        launches_per_step = 1     # the attention (key boxes follow from each unit's index: no lists)
    rope = wl.rope
    if rope is not None:
        # the step turns Q and K (two RoPE launches), then attends
        q_r = torch.empty_like(q)   # the standalone RoPE timing's output
        launches_per_step = 3

    def step():
        if wl.window is not None:
            binding.attn_fwd_win3d(q, k, v, wl.latent, wl.window[0], wl.window[1], scale=wl.scale, out=out, lse=lse)
        elif rope is not None:
            # one call: Q and K turned into the library's buffers, then the attention
            grid, s0, dims, theta, inter = rope
            binding.attn_fwd_rope3d(q, k, v, grid, s0, dims, theta, inter, scale=wl.scale, out=out, lse=lse)
        elif segs is not None:
            binding.attn_fwd_segments(q, k, v, segs[0], segs[1], scale=wl.scale, out=out, lse=lse)
        elif lens is None:
            binding.attn_fwd(q, k, v, scale=wl.scale, out=out, lse=lse)
        else:
            binding.attn_fwd_varlen(q, k, v, lens, scale=wl.scale, out=out, lse=lse)

    def barrier():
        if world > 1:
            dist.barrier(device_ids=[local])
        torch.cuda.synchronize(dev)

    for _ in range(args.warmup):
        step()
    st = binding.check_device_error(dev)
    if st != binding.VDX_OK:
        raise RuntimeError(binding.status_string(st))

    # ---- device-resident timed region
    peaks, peak_kind = load_peaks()
    clocks_log = os.environ.get("VDX_BENCH_CLOCKS_CSV") or None   # optional raw nvidia-smi samples
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local, clocks_log) as clk:
        barrier()
        # one event between consecutive calls (recording an event launches
        # no work): the per-call times below; the total spans them all
        marks = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
        start.record(stream)
        marks[0].record(stream)
        for i in range(args.steps):
            step()
            marks[i + 1].record(stream)
        end.record(stream)
        barrier()
    ms_total = max_over_ranks(start.elapsed_time(end), world, dev)
    per_call = [marks[i].elapsed_time(marks[i + 1]) for i in range(args.steps)]
    st = binding.check_device_error(dev)
    if st != binding.VDX_OK:
        raise RuntimeError(binding.status_string(st))
    ms_step = ms_total / args.steps
    tflops = flops * world / (ms_step * 1e-3) / 1e12
    per_launch_tflops = flops / (ms_step * 1e-3) / 1e12

    # ---- the rotary kernel alone against the HBM roofline
    rope_rec = None
    if rope is not None:
        grid, s0, dims, theta, inter = rope
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        for _ in range(3):
            binding.rope3d(q, grid, s0, dims, theta, inter, out=q_r)
        barrier()
        n_rope = 50
        a.record(stream)
        for _ in range(n_rope):
            binding.rope3d(q, grid, s0, dims, theta, inter, out=q_r)
        b.record(stream)
        barrier()
        rope_ms = a.elapsed_time(b) / n_rope
        rope_bytes = 2 * q.numel() * q.element_size()     # one read and one write of the tensor
        hbm = float(load_peaks()[0].get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
        rope_rec = {"kernel": "vdx::rope3d_vec_kernel" if inter and wl.D % 8 == 0 else
                    "vdx::rope3d_kernel<%s>" % ("true" if inter else "false"),
                    "ms_per_call": round(rope_ms, 4), "bytes_per_call": rope_bytes,
                    "achieved_gbs": round(rope_bytes / (rope_ms * 1e-3) / 1e9, 1), "peak_gbs": hbm,
                    "frac_of_hbm": round(rope_bytes / (rope_ms * 1e-3) / 1e9 / hbm, 4),
                    "note": "Q alone, back to back; the tensor (100.6 MB read + written) exceeds L2"}

    # ---- end to end through the C ABI with pinned host buffers
    qh, kh, vh = (t.pin_memory() for t in (w["q"], w["k"], w["v"]))
    lh = None if w["kv_lens"] is None else torch.from_numpy(w["kv_lens"]).pin_memory()
    sh = None if segs is None else tuple(torch.from_numpy(w[n]).pin_memory() for n in ("q_seg", "kv_seg"))
    oh = torch.empty(out.shape, dtype=out.dtype).pin_memory()
    lseh = torch.empty(lse.shape, dtype=lse.dtype).pin_memory()
    h2d = sum(t.numel() * t.element_size() for t in (qh, kh, vh)) + (0 if lh is None else lh.numel() * 4) + \
        (0 if sh is None else sum(t.numel() * 4 for t in sh))
    d2h = oh.numel() * oh.element_size() + lseh.numel() * lseh.element_size()

    def e2e_step():
        # one host-buffer call: chunks of (b, h) rows, copies overlapped with the kernels
        if rope is not None:
            grid, s0, dims, theta, inter = rope
            binding.attn_fwd_rope3d_host(qh, kh, vh, grid, s0, dims, theta, inter, scale=wl.scale, out=oh,
                                         lse=lseh, device=dev, synchronize=False)
        elif wl.window is not None:
            binding.attn_fwd_win3d_host(qh, kh, vh, wl.latent, wl.window[0], wl.window[1], scale=wl.scale,
                                        out=oh, lse=lseh, device=dev, synchronize=False)
        elif sh is not None:
            binding.attn_fwd_segments_host(qh, kh, vh, sh[0], sh[1], scale=wl.scale, out=oh, lse=lseh,
                                           device=dev, synchronize=False)
        else:
            binding.attn_fwd_host(qh, kh, vh, kv_lens=lh, scale=wl.scale, out=oh, lse=lseh, device=dev,
                                  synchronize=False)

    e2e_steps = max(3, min(args.steps, 50))
    for _ in range(2):
        e2e_step()
    barrier()
    s2, e2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s2.record(stream)
    for _ in range(e2e_steps):
        e2e_step()
    e2.record(stream)
    barrier()
    e2e_ms = max_over_ranks(s2.elapsed_time(e2), world, dev) / e2e_steps
    e2e_tflops = flops * world / (e2e_ms * 1e-3) / 1e12

    # ---- oracle on the host cores (rank 0, N = 1 only)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = time_oracle(w, target_s=args.cpu_seconds, gpu=(out, lse))

    if world > 1:
        dist.destroy_process_group()
    if rank != 0:
        return

    clocks = clk.summary(peaks.get("sm_max_mhz"))
    peak = float(peaks["bf16_tflops"])
    traffic = load_traffic(args.workload)
    line = {
        "metric": METRIC, "value": round(tflops, 2), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 4),
        "ms_per_call": {"median": round(statistics.median(per_call), 4), "min": round(min(per_call), 4),
                        "max": round(max(per_call), 4), "note": "rank 0, events between consecutive calls"},
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) bf16 tensors shaped like the workload; no dataset)",
        "config": {"workload": wl.name, "description": wl.description, "B": wl.B, "H": wl.H,
                   "Sq": wl.Sq, "Skv": wl.Skv, "D": wl.D, "scale": wl.scale,
                   "flops_per_call": flops,
                   "l2": "inputs larger than L2 (no flush): Q+K+V+O = %.0f MB" % (
                       4 * q.numel() * 2 / 1e6 if lens is None else (2 * q.numel() + 2 * k.numel()) * 2 / 1e6),
                   "parallelism": f"replicas x{world} (independent problems per GPU)"},
        "clocks": clocks,
        "e2e": {"value": round(e2e_tflops, 2), "unit": UNIT, "ms_per_step": round(e2e_ms, 4),
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "path": "host-buffer entry point (vdx_attn_fwd%s_host): pinned host buffers, chunks of (b, h) "
                        "rows, copies in and out overlapped with the kernels" % (
                            "_rope3d" if rope is not None else
                            ("_win3d" if wl.window is not None else ("_segments" if sh is not None else "")))},
        "gpu_launches": args.steps * launches_per_step,
        "roofline": {"bound": "tensor", "achieved": round(per_launch_tflops, 2), "peak": peak,
                     "unit": "TFLOP/s", "frac": round(per_launch_tflops / peak, 4),
                     "peak_kind": f"{peak_kind} bf16 dense burst",
                     "frac_of_sustained": round(per_launch_tflops / float(peaks["bf16_tflops_sustained"]), 4),
                     "traffic": traffic,
                     "kernel": "vdx::attn_fwd_kernel<%d,%s,%s>" % (wl.D, mode, "1,2" if wl.D == 128 else "2,4")},
        "cpu_baseline": cpu,
    }
    if rope_rec is not None:
        line["rope"] = rope_rec
    print(json.dumps(line), flush=True)


def kernel_source_hash():
    """sha256 over the code (comments and whitespace removed) of the CUDA
    sources that build and launch the attention kernel, to tell whether a
    stored ncu capture of it still applies.  The 3D RoPE kernel's own header
    is left out: the captures are of the attention kernel, whose code does not
    depend on it."""
    import hashlib
    import re
    csrc = os.path.join(ROOT, "paper_2609_18077_gb300", "csrc")
    h = hashlib.sha256()
    for name in sorted(os.listdir(csrc)):
        if name.endswith((".cu", ".cuh", ".h")) and name != "rope3d.cuh":
            with open(os.path.join(csrc, name)) as f:
                code = f.read()
            code = re.sub(r"/\*.*?\*/", " ", code, flags=re.S)   # block comments
            code = re.sub(r"//[^\n]*", " ", code)                  # line comments
            code = "".join(code.split())                            # whitespace
            h.update(name.encode() + b"\0" + code.encode())
    return h.hexdigest()[:16]


def load_traffic(workload):
    """DRAM bytes per launch from the committed ncu summary, or None when the
    kernel sources changed since that capture (or no capture covers the workload)."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        d = json.load(f)
    entry = d.get(workload)
    if not entry or entry.get("kernel_source_sha") != kernel_source_hash():
        return None
    return entry.get("dram_bytes_per_launch")


class OracleTimer:
    """Times the fp64 oracle on seeded query-row samples of a workload.

    calibrate() picks the rows per (b, h) that take about target_s seconds;
    run() times one such sample and returns the cpu_baseline record.
    """

    def __init__(self, w, threads=0):
        import oracle
        from paper_2609_18077_gb300 import workloads
        self.orc = oracle.default()
        self.cores = self.orc.set_threads(threads)
        self.w = w
        wl = w["workload"]
        self.wl = wl
        self.bits = tuple(workloads.bf16_bits(w[n]) for n in ("q", "k", "v"))
        self.rng = np.random.default_rng(wl.seed)
        lens = w["kv_lens"]
        keys = wl.Skv if lens is None else float(np.mean(np.clip(lens, 0, wl.Skv)))
        if w["q_seg"] is not None:   # mean keys per query row
            keys = workloads.segment_pairs(w["q_seg"], w["kv_seg"]) / float(wl.B * wl.Sq)
        if wl.window is not None:
            keys = workloads.window_pairs(wl.latent, *wl.window) / float(wl.Sq)
        self.flops_per_row = 4.0 * keys * wl.D
        self.bh = wl.B * wl.H
        self.n = 1

    def _time(self, n):
        rows = np.stack([np.sort(self.rng.choice(self.wl.Sq, size=n, replace=False))
                         for _ in range(self.bh)]).astype(np.int32)
        t0 = time.perf_counter()
        if self.wl.window is not None:
            res = self.orc.attn_fwd_win3d(*self.bits, self.wl.scale, self.wl.latent, self.wl.window[0],
                                          self.wl.window[1], rows=rows)
        else:
            res = self.orc.attn_fwd(*self.bits, self.wl.scale, kv_lens=self.w["kv_lens"], rows=rows,
                                    q_seg=self.w["q_seg"], kv_seg=self.w["kv_seg"])
        dt = time.perf_counter() - t0
        self.last = (rows, res)
        return dt

    def calibrate(self, target_s):
        n, dt = 1, self._time(1)
        while dt < 0.25 and n < self.wl.Sq:
            n = min(self.wl.Sq, n * 4)
            dt = self._time(n)
        self.n = int(min(self.wl.Sq, max(1, math.ceil(n * target_s / max(dt, 1e-6)))))
        return self.n

    def run(self):
        dt = self._time(self.n)
        flops = self.flops_per_row * self.n * self.bh
        full = self.flops_per_row * self.wl.Sq * self.bh   # the whole call's FLOP
        return {"value": round(flops / dt / 1e12, 6), "unit": UNIT, "cores": self.cores, "kind": "oracle",
                "seconds": round(dt, 3),
                "full_call_seconds_extrapolated": round(dt * full / flops, 1),
                "sample": f"{self.n} seeded query rows per (b,h) x {self.bh} (b,h) pairs of workload "
                          f"{self.wl.name} ({flops:.3e} FLOP in fp64, OpenMP)"}


def sample_parity(rows, ref, out, lse):
    """The timed oracle sample against the GPU's output of the same call at
    the same rows: max and mean |O| error, max relative LSE error (the
    tolerances of the parity tests are 2e-2, 2e-3 and 1e-3)."""
    import torch
    o_ref, lse_ref = ref
    B, H, Sq, D = out.shape
    idx = torch.from_numpy(rows.astype(np.int64)).to(out.device).view(B, H, -1)
    o = torch.gather(out, 2, idx.unsqueeze(-1).expand(-1, -1, -1, D)).float().double().cpu().numpy()
    ls = torch.gather(lse, 2, idx).double().cpu().numpy()
    err = np.abs(o - o_ref)
    fin = np.isfinite(lse_ref)
    rel = np.abs(ls[fin] - lse_ref[fin]) / np.maximum(1.0, np.abs(lse_ref[fin]))
    return {"o_max_abs": float(f"{err.max():.3e}"), "o_mean_abs": float(f"{err.mean():.3e}"),
            "lse_max_rel": float(f"{rel.max():.3e}") if rel.size else 0.0,
            "lse_neg_inf_pattern_equal": bool(np.array_equal(np.isneginf(ls), ~fin)),
            "rows": f"the timed sample's {rows.shape[1]} rows per (b,h)"}


def time_oracle(w, target_s=15.0, gpu=None):
    """The cpu_baseline record; with gpu = (out, lse) of the timed calls, the
    sample's rows also serve as a parity spot check of that output."""
    t = OracleTimer(w)
    t.calibrate(target_s)
    rec = t.run()
    if gpu is not None:
        if w["workload"].rope is not None:
            rec["parity_on_sample"] = "not compared: this sample times the attention without the rotation"
        else:
            rec["parity_on_sample"] = sample_parity(*t.last, *gpu)
    return rec


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    w, flops = make_inputs(args.workload)
    wl = w["workload"]
    timer = OracleTimer(w)
    per_step = min(5.0, max(0.2, args.cpu_seconds * 4 / max(1, args.steps + args.warmup)))
    timer.calibrate(per_step)
    for _ in range(args.warmup):
        timer.run()
    recs = [timer.run() for _ in range(args.steps)]
    value = statistics.median(r["value"] for r in recs)
    # ms_per_step: the wall time of one timed step (one sample), as run; the
    # full call at the sampled rate is reported beside it
    ms_per_step = statistics.median(r["seconds"] for r in recs) * 1e3
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded N(0,1) bf16 tensors shaped like the workload; no dataset)",
        "config": {"workload": wl.name, "description": wl.description, "B": wl.B, "H": wl.H, "Sq": wl.Sq,
                   "Skv": wl.Skv, "D": wl.D, "scale": wl.scale, "flops_per_call": flops,
                   "parallelism": f"replicas x{world} (rank 0 times the oracle)",
                   "note": "each step times the oracle on a bounded seeded row sample of the workload; "
                           "ms_per_step is one such step; ms_full_call_extrapolated is the whole call at "
                           "the sampled rate",
                   "ms_full_call_extrapolated": round(flops / (value * 1e12) * 1e3, 1)},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": recs[-1]["cores"], "kind": "oracle",
                         "sample": recs[-1]["sample"] + " per step"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
    }
    print(json.dumps(line), flush=True)


def main():
    from paper_2609_18077_gb300 import workloads
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=None, help="GPUs (default: WORLD_SIZE under torchrun, else 1)")
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--workload", default=workloads.DEFAULT_WORKLOAD, choices=sorted(workloads.WORKLOADS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    args = ap.parse_args()
    if "WORLD_SIZE" not in os.environ and (args.gpus or 1) > 1:
        # one process per GPU: relaunch under torchrun on this node
        import socket
        with socket.socket() as sock:
            sock.bind(("127.0.0.1", 0))
            port = sock.getsockname()[1]
        cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={args.gpus}",
               "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.abspath(__file__)] + sys.argv[1:]
        sys.exit(subprocess.call(cmd))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if args.gpus is not None and args.gpus != world:
        ap.error(f"--gpus {args.gpus} but WORLD_SIZE is {world}")
    if args.warmup < 3 and args.impl == "ours":
        print("note: fewer than 3 warm-up steps", file=sys.stderr)
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
