"""Benchmark of the WaveFilter hot path on GB300.

One step = one denoising-step layer of the method after the cache exists:
wf_step, i.e. the skim + multi-scale scan filter (Eq. 7-11) and the sparse
attention (final step of Algorithm 1) over every (batch, head) of the
workload, with the Haar pyramid of the prompt keys already built (the paper
computes it at the initial step; the 32-layer workload "c5" instead
refreshes it every 8 steps inside the timed loop).  For bf16 / head_dim 128
that is one fused kernel launch per layer.

value = algorithmic HBM bytes of the step / device time (GB/s): the bytes
that must move are the query block, the candidate coefficient rows of every
scale, the level-0 trim rows, K[mu0] and V[mu0], the generation rows, the
output block and the index list.  L2 is flushed (256 MiB write) before every
timed step; each step is timed with CUDA events on the launching stream.
value and ms_per_step use the mean step time over the K timed steps (the
whole-job rate); step_us_median is the median of the same steps.  On one
GPU the default run also measures the 128K-token workload (c4) in the same
process (10 warm-up steps, median of 50) under the key "c4".

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--workload c3]
                       [--impl reference]
Under torchrun every rank runs its own replica of the workload (the path
shards by (batch, head) with no exchange: weak scaling); rank 0 prints one
JSON line with the max time over ranks.
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

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2606_00724_gb300 import synth  # noqa: E402

METRIC = "fused filter+sparse-attn step latency (us) & achieved HBM GB/s vs roofline, 1 GB300"
DEFAULT_WORKLOAD = "c3"
WAVELET = None  # None: the Haar pyramid path (wf_step); "haar" / "db2": the literal path (wf_step_wavelet)


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


# ---------------------------------------------------------------------------
# Algorithmic bytes (per (batch, head) unit).
# ---------------------------------------------------------------------------
def unit_bytes(w: synth.Workload) -> dict:
    e = 4 if w.dtype == "f32" else 2
    row = w.head_dim * e
    L, keep = w.levels, [int(x) for x in w.keep]
    cands = [w.n >> L] + [2 * keep[b + 1] for b in range(L - 1, 0, -1)]
    trim = 2 * keep[1] if keep[0] < 2 * keep[1] else 0
    k = keep[0]
    q = w.q * w.group * row  # the query rows (and output rows) of every query head of the unit's group
    coeff = sum(cands) * row
    filt = q + coeff + trim * row + 4 * k
    attn = q + 4 * k + 2 * k * row + 2 * w.ng * row + q
    step = q + coeff + trim * row + 2 * k * row + 2 * w.ng * row + q + 4 * k
    dwt = w.n * row + (w.n - (w.n >> L)) * row
    if WAVELET:
        step = wavelet_unit_bytes(w)
        dwt = w.n * row + (w.n >> L) * row  # the scale-L rows of the whole prompt
    return {"filter": filt, "attn": attn, "step": step, "dwt": dwt}


def wavelet_unit_bytes(w: synth.Workload) -> int:
    """Algorithmic bytes of one unit's step on the literal path (Eq. 11 for a
    generic basis): the cached scale-L rows, the keys of every finer scale's
    gathered candidate blocks (2 keep[b+1] blocks of 2^b tokens, read once),
    the level-0 trim rows, the sparse K/V rows, Q, O and the indices."""
    e = 4 if w.dtype == "f32" else 2
    row = w.head_dim * e
    L, keep = w.levels, [int(x) for x in w.keep]
    gathered = sum(2 * keep[b + 1] << b for b in range(L - 1, 0, -1))
    trim = 2 * keep[1] if keep[0] < 2 * keep[1] else 0
    k = keep[0]
    q = w.q * w.group * row
    return q + ((w.n >> L) + gathered + trim + 2 * k + 2 * w.ng) * row + q + 4 * k


def fused_eligible(w: synth.Workload) -> bool:
    """wf_step runs its single fused kernel for bf16, head_dim 128, <= 32 query
    rows and one query head per key head (the Haar pyramid path)."""
    return WAVELET is None and fused_shape(w)


def fused_shape(w: synth.Workload) -> bool:
    """Shapes the fused kernel serves: bf16, head_dim 128, <= 32 query rows,
    one query head per key head."""
    return w.dtype == "bf16" and w.head_dim == 128 and w.q <= 32 and w.group == 1


def grouped_fused(w: synth.Workload) -> bool:
    """Grouped query heads that wf_step filters with the grouped filter kernel
    (bf16, head_dim 128, <= 32 rows a query head, <= 256 stacked rows), then
    attends with the per-stage tensor-core attention (split + combine)."""
    return (WAVELET is None and w.dtype == "bf16" and w.head_dim == 128 and w.q <= 32 and w.group > 1
            and w.group * w.q <= 256)


def recorded_traffic(w: synth.Workload):
    """DRAM bytes per launch of the fused kernel from the committed ncu record,
    if it was taken on this workload with the current kernel source."""
    import hashlib
    rec = os.path.join(ROOT, "profiles", "wf_fused_kernel_traffic.md")
    src = os.path.join(ROOT, "paper_2606_00724_gb300", "csrc", "wf_fused.cu")
    if not (os.path.exists(rec) and os.path.exists(src)):
        return None
    h = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    for ln in open(rec):
        cells = [c.strip() for c in ln.strip().strip("|").split("|")]
        if len(cells) == 6 and cells[0] == w.name and cells[5] == h:
            try:
                return int(cells[3])
            except ValueError:
                return None
    return None


def launches_per_step(w: synth.Workload) -> int:
    if fused_eligible(w):
        return 1
    if grouped_fused(w):  # the grouped filter kernel, the attention split and its combine
        return 3
    trim = int(w.keep[0]) < 2 * int(w.keep[1])
    if WAVELET and fused_shape(w):  # one fused launch per scale, a transform before each below the top
        return w.levels + (w.levels - 1)
    if WAVELET:  # one transform kernel per scale below the top
        return 3 * w.levels + (w.levels - 1) + 3 * trim + 2
    return 3 * w.levels + 3 * trim + 2


# ---------------------------------------------------------------------------
# Clock sampling during the timed region.
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.lines = []
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.dev}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except (OSError, FileNotFoundError):
            self.proc = None

    def _read(self):
        for ln in self.proc.stdout:
            self.lines.append(ln.strip())

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
            except ValueError:
                continue
            for name, val in zip(names, parts[4:8]):
                if val.lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# CPU oracle timing (baseline / reference arm).
# ---------------------------------------------------------------------------
def oracle_units_seconds(w: synth.Workload, cfg: str, budget_s: float, max_units: int | None = None,
                         start_unit: int = 0):
    """Time the oracle's filter + sparse attention on consecutive units until
    the time budget is spent.  Returns (units, seconds)."""
    import oracle
    oracle.build()
    done, spent, u = 0, 0.0, start_unit
    while True:
        b, h = divmod(u % w.units, w.heads)
        unit = synth.make_unit(w, b, h, planted=False, device="cpu", cfg=cfg)
        dt = synth.storage_dtype(w)
        Q, K, V, Kg, Vg = (t.to(dt).double().numpy() for t in (unit.Q, unit.K, unit.V, unit.Kg, unit.Vg))
        pyr = oracle.haar_pyramid_spec32(K.astype(np.float32), w.levels, w.dtype == "bf16").astype(np.float64)
        t0 = time.perf_counter()
        if WAVELET:
            basis = oracle.DB2 if WAVELET == "db2" else oracle.HAAR
            mu0 = oracle.filter_wavelet(Q, K, w.levels, np.array(w.keep), basis, spec32=False)
            oracle.sparse_attn(Q, K, V, mu0, Kg, Vg)
        elif w.group > 1:
            Qh = Q.reshape(w.group, w.q, w.head_dim)
            mu0 = oracle.filter_gqa(Qh, pyr, K, w.n, w.levels, np.array(w.keep))
            oracle.sparse_attn_gqa(Qh, K, V, mu0, Kg, Vg)
        else:
            mu0 = oracle.filter(Q, pyr, K, w.n, w.levels, np.array(w.keep))
            oracle.sparse_attn(Q, K, V, mu0, Kg, Vg)
        spent += time.perf_counter() - t0
        done += 1
        u += 1
        if spent >= budget_s or (max_units is not None and done >= max_units):
            return done, spent


# ---------------------------------------------------------------------------
# Multi-rank aggregation (one replica per rank, weak scaling).
# ---------------------------------------------------------------------------
def max_over_ranks(values, device):
    """Each value's MAX over the ranks of the default process group (the
    values themselves on a single rank)."""
    dist = torch.distributed
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return [float(v) for v in values]
    t = torch.tensor([float(v) for v in values], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t]


def aggregate(world: int, step_bytes: float, total_ms: float, steps: int):
    """(ms per step, whole-job GB/s): every rank moves step_bytes per step and
    the slowest rank's time counts."""
    ms_per_step = total_ms / steps
    return ms_per_step, world * step_bytes / (ms_per_step * 1e-3) / 1e9


# ---------------------------------------------------------------------------
# GPU arm.
# ---------------------------------------------------------------------------
def make_inputs(w, cfg, device, rank):
    if cfg == "c5":
        return [synth.make_batch_fast(w, layer=l, device=device, seed_salt=rank) for l in range(w.layers)]
    return [synth.make_batch(w, layer=rank, planted=False, device=device, cfg=cfg)]


def measure_cache_update(args, w, cfg, device, hbm_peak, peak_kind):
    """wf_cache_update of R new rows per unit (written into the K/V caches with
    the touched pyramid blocks refreshed) against a full wf_dwt_build, on one
    layer of the workload; the window moves by R rows every call."""
    from paper_2606_00724_gb300 import wf
    R = args.update_rows
    lay = (synth.make_batch_fast(w, layer=0, device=device) if cfg == "c5" else
           synth.make_batch(w, layer=0, planted=False, device=device, cfg=cfg))
    K, V = lay.K, lay.V
    dt = K.dtype
    coeffs = torch.empty(wf.wf_coeffs_bytes(K, w.levels), dtype=torch.uint8, device=device)
    wf.wf_dwt_build(K, w.levels, coeffs)
    g = torch.Generator(device=device).manual_seed(7)
    Kn = torch.randn(w.batch, w.heads, R, w.head_dim, generator=g, device=device).to(dt)
    Vn = torch.randn(w.batch, w.heads, R, w.head_dim, generator=g, device=device).to(dt)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=device)
    row = w.head_dim * K.element_size()
    blk = 1 << w.levels

    def timed(fn, steps):
        t = 0.0
        for i in range(args.warmup + steps):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            fn(i)
            b.record()
            torch.cuda.synchronize()
            if i >= args.warmup:
                t += a.elapsed_time(b)
        return t / steps * 1e3  # us

    assert w.n % R == 0, "--update-rows must divide the context"
    pos_of = lambda i: (i * R) % w.n  # windows aligned to R
    upd_us = timed(lambda i: wf.wf_cache_update(Kn, Vn, K, V, pos_of(i), w.levels, coeffs), args.steps)
    full_us = timed(lambda i: wf.wf_dwt_build(K, w.levels, coeffs), max(3, args.steps // 10))
    nblk = ((R - 1) >> w.levels) + 1  # 2^L-token blocks an aligned window of R rows touches
    upd_bytes = w.units * (4 * R * row + (nblk * blk - R) * row + nblk * (blk - 1) * row)
    full_bytes = w.units * (w.n * row + (w.n - (w.n >> w.levels)) * row)
    return {"metric": "cache update + incremental pyramid refresh latency (us)", "value": upd_us, "unit": "us",
            "higher_is_better": False, "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
            "dtype": "bf16" if dt == torch.bfloat16 else "f32", "data": "synthetic",
            "config": {"workload": w.name, "batch": w.batch, "heads": w.heads, "context": w.n, "levels": w.levels,
                       "update_rows": R, "l2": "flushed before every timed call (256 MiB write)"},
            "bytes_per_call": upd_bytes, "achieved_gbs": upd_bytes / upd_us / 1e3,
            "full_rebuild": {"us": full_us, "bytes": full_bytes, "achieved_gbs": full_bytes / full_us / 1e3,
                             "peak_gbs": hbm_peak, "peak_kind": peak_kind}}


def run_gpu(args, cfg, rank, world, device):
    from paper_2606_00724_gb300 import wf

    w = synth.WORKLOADS[cfg]
    keep = [int(x) for x in w.keep]
    layers = make_inputs(w, cfg, device, rank)
    bufs = []
    basis = {"haar": wf.WF_WAVELET_HAAR, "db2": wf.WF_WAVELET_DB2}.get(WAVELET)
    for lay in layers:
        if WAVELET:
            # The literal path: the scale-L rows of the whole prompt once (like
            # the pyramid), the finer scales' transforms inside every step.
            coeffs = torch.empty(w.batch, w.heads, w.n >> w.levels, w.head_dim, dtype=lay.K.dtype, device=device)
            wf.wf_wavelet_approx(lay.K, w.levels, basis, coeffs)
            ws = torch.zeros(wf.wf_step_wavelet_workspace_bytes(lay.Q, lay.K, w.levels, keep, basis, w.ng),
                             dtype=torch.uint8, device=device)
        else:
            coeffs = torch.empty(wf.wf_coeffs_bytes(lay.K, w.levels), dtype=torch.uint8, device=device)
            wf.wf_dwt_build(lay.K, w.levels, coeffs)
            ws = torch.zeros(wf.wf_step_workspace_bytes(lay.Q, lay.K, w.levels, keep, w.ng), dtype=torch.uint8,
                             device=device)
        bufs.append(dict(coeffs=coeffs, ws=ws, idx=torch.empty(w.units, w.k, dtype=torch.int32, device=device),
                         O=torch.empty_like(lay.Q)))

    def one(lay, bf, Q, Kg, Vg, refresh):
        st = torch.cuda.current_stream()  # the capture stream while a graph is recorded
        if WAVELET:
            if refresh:
                wf.wf_wavelet_approx(lay.K, w.levels, basis, bf["coeffs"], stream=st)
            wf.wf_step_wavelet(Q, bf["coeffs"], lay.K, lay.V, Kg, Vg, w.levels, keep, basis, bf["idx"], bf["O"],
                               bf["ws"], stream=st)
        else:
            wf.wf_step(Q, lay.K, lay.V, Kg, Vg, bf["coeffs"], refresh, w.levels, keep, bf["idx"], bf["O"], bf["ws"],
                       st)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=device)
    stream = torch.cuda.current_stream()
    refresh_every = w.refresh_every

    def step(i):
        for lay, bf in zip(layers, bufs):
            refresh = bool(refresh_every) and (i % refresh_every == 0)
            one(lay, bf, lay.Q, lay.Kg, lay.Vg, refresh)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    if args.graph:
        # One step's launches recorded once and replayed: the same kernels,
        # without the host launch gaps between them.
        if refresh_every:
            raise SystemExit("bench.py: --graph takes workloads without a periodic refresh")
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            step(0)
        torch.cuda.synchronize()
        step = lambda i: graph.replay()  # noqa: E731

    # Pre-roll of the same steps so that the clock samples see the GPU under load.
    sampler = ClockSampler(device.index if device.index is not None else 0)
    sampler.start()
    t_end = time.time() + args.preroll
    i = 0
    while time.time() < t_end:
        flush.zero_()
        step(i)
        i += 1
        if i % 32 == 0:
            torch.cuda.synchronize()
    torch.cuda.synchronize()

    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    for i in range(args.steps):
        flush.zero_()
        evs[i][0].record(stream)
        step(i)
        evs[i][1].record(stream)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    clocks = sampler.stop()
    step_ms = [a.elapsed_time(b) for a, b in evs]
    total_ms = sum(step_ms)

    lay, bf = layers[0], bufs[0]
    # End to end through the public API with host buffers: copy the step's
    # query block and generation rows in from pinned memory, run the step,
    # copy O and the indices out.  The inputs sit back to back in one pinned
    # staging buffer and the outputs in another, so each direction is one
    # copy; the step reads and writes views of the device buffers.
    def packed(shapes_dtypes, device_or_pin):
        offs, off = [], 0
        for shape, dt in shapes_dtypes:
            offs.append(off)
            off += (math.prod(shape) * torch.tensor([], dtype=dt).element_size() + 255) // 256 * 256
        if device_or_pin == "pin":
            buf = torch.empty(off, dtype=torch.uint8, pin_memory=True)
        else:
            buf = torch.empty(off, dtype=torch.uint8, device=device_or_pin)
        views = [buf[o:o + math.prod(sh) * torch.tensor([], dtype=dt).element_size()].view(dt).view(sh)
                 for o, (sh, dt) in zip(offs, shapes_dtypes)]
        return buf, views
    ins = [(tuple(lay.Q.shape), lay.Q.dtype), (tuple(lay.Kg.shape), lay.Kg.dtype), (tuple(lay.Vg.shape), lay.Vg.dtype)]
    outs = [(tuple(lay.Q.shape), lay.Q.dtype), ((w.units, w.k), torch.int32)]
    hin, (hQ, hKg, hVg) = packed(ins, "pin")
    din, (dQ, dKg, dVg) = packed(ins, device)
    hout, _ = packed(outs, "pin")
    dout, (dO, didx) = packed(outs, device)
    hQ.copy_(lay.Q.cpu())
    hKg.copy_(lay.Kg.cpu())
    hVg.copy_(lay.Vg.cpu())
    bf_e2e = dict(bf, O=dO, idx=didx)
    e2e_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(max(args.steps, 20))]
    for a, b in e2e_ev:
        flush.zero_()
        a.record(stream)
        din.copy_(hin, non_blocking=True)
        one(lay, bf_e2e, dQ, dKg, dVg, False)
        hout.copy_(dout, non_blocking=True)
        b.record(stream)
    torch.cuda.synchronize()
    e2e_ms = statistics.mean(a.elapsed_time(b) for a, b in e2e_ev)
    h2d = hin.numel()
    d2h = hout.numel()
    return dict(w=w, total_ms=total_ms, step_ms=step_ms, clocks=clocks, e2e_ms=e2e_ms, h2d=h2d, d2h=d2h,
                layers=len(layers))


def kernel_name(w):
    """The kernels a step of workload w runs (the roofline's "kernel")."""
    if fused_eligible(w):
        return "wf_fused_kernel"
    if WAVELET:
        return ("approx_kernel + wf_fused_kernel (one launch per scale)" if fused_shape(w) else
                "per-stage kernels (approx/score/weights/select/attn)")
    if grouped_fused(w):
        return "wf_gqa_filter_kernel + tc_attn_rows_kernel + attn_combine_kernel"
    return "per-stage kernels (score/weights/select/attn)"


def measure_extra(args, cfg, device, hbm_peak, peak_kind):
    """A second workload measured in the same process: 10 warm-up steps, 50
    timed steps (L2 flushed before each), median and mean step time, the
    fused kernel's roofline and the clock record of its own timed region."""
    import types
    w = synth.WORKLOADS[cfg]
    a = types.SimpleNamespace(**vars(args))
    a.steps, a.warmup = 50, 10
    r = run_gpu(a, cfg, 0, 1, device)
    ub = unit_bytes(w)
    mean_us = r["total_ms"] / a.steps * 1e3
    med_us = statistics.median(r["step_ms"]) * 1e3
    bytes_launch = ub["step"] * w.units
    return {"workload": w.name, "steps": a.steps, "warmup": a.warmup, "step_us_median": med_us,
            "step_us_mean": mean_us,
            "roofline": {"bound": "hbm", "achieved": bytes_launch / (med_us * 1e-6) / 1e9, "peak": hbm_peak,
                         "unit": "GB/s", "frac": bytes_launch / (med_us * 1e-6) / 1e9 / hbm_peak,
                         "frac_of_mean": bytes_launch / (mean_us * 1e-6) / 1e9 / hbm_peak,
                         "traffic": recorded_traffic(w) if fused_eligible(w) else None,
                         "kernel": kernel_name(w),
                         "peak_kind": peak_kind, "bytes_per_launch": bytes_launch},
            "clocks": r["clocks"]}


def main():
    global WAVELET
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=list(synth.WORKLOADS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--preroll", type=float, default=1.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--batch", type=int, default=None, help="override the workload's batch (small profiling cases)")
    ap.add_argument("--heads", type=int, default=None, help="override the workload's head count")
    ap.add_argument("--graph", action="store_true",
                    help="replay each step from a CUDA graph recorded after the warm-up")
    ap.add_argument("--wavelet", default=None, choices=["haar", "db2"],
                    help="time the literal path for a generic basis (wf_step_wavelet): the transform of the "
                         "gathered candidate blocks at every scale")
    ap.add_argument("--schedule", default="default", choices=["default", "level0"],
                    help="kept counts: the default schedule, or the token level as its own selection step")
    ap.add_argument("--measure", default="step", choices=["step", "cache-update"],
                    help="step: the filter + sparse-attention step (the metric); cache-update: wf_cache_update of "
                         "--update-rows rows per unit against a full pyramid rebuild")
    ap.add_argument("--update-rows", type=int, default=32)
    ap.add_argument("--no-extra", action="store_true",
                    help="skip the other workloads (c4, g1) that the default single-GPU run also measures")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    cfg = args.workload
    w = synth.WORKLOADS[cfg]
    if args.batch or args.heads:
        import dataclasses
        w = dataclasses.replace(w, batch=args.batch or w.batch, heads=args.heads or w.heads,
                                name=f"{w.name}_B{args.batch or w.batch}_H{args.heads or w.heads}")
        synth.WORKLOADS[cfg] = w
    if args.wavelet:
        import dataclasses
        WAVELET = args.wavelet
        w = dataclasses.replace(w, name=f"{w.name}_{args.wavelet}_literal")
        synth.WORKLOADS[cfg] = w
    if args.schedule == "level0":
        # The token level as its own selection step (one proportion over L+1 scans).
        import dataclasses
        from paper_2606_00724_gb300 import wf
        keep = tuple(wf.wf_level0_schedule(w.n, w.levels, w.k))
        w = dataclasses.replace(w, keep=keep, name=f"{w.name}_level0")
        synth.WORKLOADS[cfg] = w
    ub = unit_bytes(w)
    hbm_peak, peak_kind = peaks()

    config = {"workload": w.name, "batch": w.batch, "heads": w.heads, "query_heads": w.q_heads,
              "head_dim": w.head_dim,
              "context": w.n, "query_block": w.q, "generation_rows": w.ng, "levels": w.levels, "k": w.k,
              "keep": list(w.keep), "layers": w.layers, "storage": w.dtype,
              "step": ("wf_step (one fused filter + sparse-attention kernel) per layer" if fused_eligible(w) else
                       f"wf_step_wavelet ({WAVELET}, periodized; the gathered candidate blocks transformed at every "
                       "scale" + ("; one fused filter launch per scale, the last with the sparse attention)"
                                  if fused_shape(w) else "; per-stage kernels)") + " per layer" if WAVELET else
                       ("wf_step (grouped filter kernel, then the per-stage sparse-attention kernels) per layer"
                        if grouped_fused(w) else
                        "wf_step (per-stage filter and sparse-attention kernels) per layer")) + (
                  f"; wf_dwt_build refresh every {w.refresh_every} steps" if w.refresh_every else
                  ("; scale-L rows built once before timing" if WAVELET else "; pyramid built once before timing")),
              "l2": "flushed before every timed step (256 MiB write)", "parallelism": f"replicas{args.gpus}",
              "cuda_graph": bool(args.graph)}
    step_bytes = ub["step"] * w.units * w.layers
    if w.refresh_every:
        step_bytes += ub["dwt"] * w.units * w.layers / w.refresh_every

    if args.impl == "reference":
        if rank != 0:
            return
        units, secs = oracle_units_seconds(w, cfg, budget_s=0.0, max_units=1)  # warm-up / build
        tot_units, tot_s = 0, 0.0
        for i in range(args.warmup):
            oracle_units_seconds(w, cfg, budget_s=0.0, max_units=1, start_unit=i)
        for i in range(args.steps):
            u, s = oracle_units_seconds(w, cfg, budget_s=0.0, max_units=1, start_unit=args.warmup + i)
            tot_units += u
            tot_s += s
        gbs = tot_units * ub["step"] / tot_s / 1e9
        line = {"metric": METRIC, "value": gbs, "unit": "GB/s", "impl": "reference", "n_gpus": args.gpus,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": tot_s / args.steps * 1e3,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                "data": "synthetic", "config": config,
                "cpu_baseline": {"value": gbs, "unit": "GB/s", "cores": 1, "kind": "oracle",
                                 "sample": f"one (batch, head) unit per step ({tot_units} units), "
                                           "filter + sparse attention, pyramid precomputed"},
                "e2e": {"value": gbs, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return

    if not torch.cuda.is_available():
        raise SystemExit("bench.py: no CUDA device (the GPU arm has no CPU fallback)")
    if world > 1:
        torch.distributed.init_process_group("nccl")
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    from paper_2606_00724_gb300 import build as wf_build
    wf_build.build()

    if args.measure == "cache-update":
        if rank == 0:
            print(json.dumps(measure_cache_update(args, w, cfg, device, hbm_peak, peak_kind)))
        return

    r = run_gpu(args, cfg, rank, world, device)
    step_us_median = statistics.median(r["step_ms"]) * 1e3
    total_ms = r["total_ms"]
    e2e_ms = r["e2e_ms"]
    total_ms, e2e_ms = max_over_ranks([total_ms, e2e_ms], device)
    ms_per_step, value = aggregate(world, step_bytes, total_ms, args.steps)

    # Roofline of the dominant kernel: the fused step kernel is the only kernel
    # of a step (one launch per layer), so its algorithmic bytes per launch are
    # the step's bytes of one layer and its launch time is the step time per
    # layer (a 4-byte status reset rides along on the same stream).
    per_layer_ms = ms_per_step / w.layers
    achieved = ub["step"] * w.units / (per_layer_ms * 1e-3) / 1e9
    if w.refresh_every:
        achieved = step_bytes / w.layers / (per_layer_ms * 1e-3) / 1e9
    kname = kernel_name(w)
    roofline = {"bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s", "frac": achieved / hbm_peak,
                "frac_of_nominal_7900": achieved / 7900.0,
                "traffic": recorded_traffic(w) if fused_eligible(w) else None, "kernel": kname,
                "peak_kind": peak_kind,
                "bytes_per_launch": ub["step"] * w.units, "launch_us": per_layer_ms * 1e3,
                "frac_median": (ub["step"] * w.units / (step_us_median / w.layers * 1e-6) / 1e9 / hbm_peak
                                if not w.refresh_every else None)}
    e2e_bytes_per_step = ub["step"] * w.units
    line = {"metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "step_us": ms_per_step * 1e3,
            "step_us_median": step_us_median,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16" if (w.dtype == "bf16" and w.head_dim == 128) else "f32",
            "data": "synthetic", "config": config, "roofline": roofline, "clocks": r["clocks"],
            "e2e": {"value": world * e2e_bytes_per_step / (e2e_ms * 1e-3) / 1e9, "unit": "GB/s",
                    "h2d_bytes_per_step": r["h2d"], "d2h_bytes_per_step": r["d2h"], "ms_per_step": e2e_ms,
                    "layers": 1},
            "gpu_launches": launches_per_step(w) * w.layers * args.steps + (
                w.layers * math.ceil(args.steps / w.refresh_every) if w.refresh_every else 0)}
    if world == 1 and cfg == DEFAULT_WORKLOAD and not args.no_extra and not (args.batch or args.heads) and \
            not args.wavelet and args.schedule == "default" and not args.graph:
        line["c4"] = measure_extra(args, "c4", device, hbm_peak, peak_kind)
        line["g1"] = measure_extra(args, "g1", device, hbm_peak, peak_kind)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        units, secs = oracle_units_seconds(w, cfg, args.cpu_seconds)
        line["cpu_baseline"] = {"value": units * ub["step"] / secs / 1e9, "unit": "GB/s", "cores": 1,
                                "kind": "oracle",
                                "sample": f"{units} (batch, head) units of the same workload, filter + sparse "
                                          f"attention ({secs:.1f} s single-threaded fp64, pyramid precomputed)"}
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
