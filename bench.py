"""Benchmark of the PnP-Nystra window-attention hot path on GB300.

One step = one ``nystra_attention`` call over the whole batch of the workload
(default: the 1280x720 super-resolution map -- 6 heads, d_h = 30, 32x32
windows edge-padded to 736 rows (920 windows), m = 16 landmarks, 6
pseudo-inverse iterations, bf16 I/O; the 16x16-window map and SwinIR-like
denoising at 256x256 are timed beside it under "extra_workloads").
Prints ONE JSON line (rank 0).  Metric: tokens*heads per second.  A "-qkv"
workload times the fused Q/K/V projection front end instead (one
``nystra_attention_qkv`` call; tensor roofline, unfused path as comparator).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the float64 CPU oracle, host cores

Under torchrun every rank runs its own full batch (units are independent, no
collective on the data path): weak scaling, value = all ranks' units / max time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2506_08520_gb300 import binding, shard, workloads  # noqa: E402

METRIC = "Nystrom attention tokens*heads/s"

# DRAM bytes (read + write) per launch from one ncu capture (profiles/), valid only
# for the sources of the kernel they were taken with: reported as null once any
# of those files changes.
MEASURED_TRAFFIC = {
    "sr720p-w16-m16-bf16": {"files": ["common.cuh", "nystra_team.cuh", "nystra_tc.cuh", "nystra_tc_n256.cu",
                                      "ptx.cuh"],
        "src_hash": "1b521d4f6ce92163", "bytes": 995_407_360 + 273_398_784},
    "sr720p-w32-m16-bf16": {"files": ["common.cuh", "nystra_stream.cuh", "nystra_tc.cuh", "nystra_tc_n1024.cu",
                                      "ptx.cuh"],
        "src_hash": "e847d1950a7301d2", "bytes": 1_030_822_656 + 284_172_544},
    "large-w16-m64": {"files": ["common.cuh", "nystra_tc.cuh", "nystra_tc_n256.cu", "nystra_team.cuh", "ptx.cuh"],
        "src_hash": "8e80904b0aac3611", "bytes": 245_142_272},
    "sr720p-w32-m16-bf16-qkv": {"files": ["common.cuh", "nystra_pool.cuh", "nystra_qkv.cuh", "nystra_qkv_stream.cuh",
                                          "nystra_qkvs_bf16.cu", "nystra_tc.cuh", "ptx.cuh"],
        "src_hash": "0ecb2b5c71d59518", "bytes": 640_227_072},
}


def _kernel_src_hash(files) -> str:
    import hashlib
    h = hashlib.sha256()
    for name in sorted(files):
        h.update(name.encode())
        with open(os.path.join(ROOT, "paper_2506_08520_gb300", "csrc", name), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]
UNIT = "tokens*heads/s"
# The largest memory-bound configuration: the 1280x720 map with 32x32 windows
# and m = 16 landmarks (1357 MB of Q, K, V, O per call).
DEFAULT_WORKLOAD = "sr720p-w32-m16-bf16"
# Reported beside a headline workload, each with its own roofline and comparator.
EXTRA_WORKLOADS = {
    "sr720p-w32-m16-bf16": ["sr720p-w32-m16-bf16-s16", "sr720p-w16-m16-bf16", "swinir256-bf16"],
    "sr720p-w16-m16-bf16": ["sr720p-w16-m16-bf16-s16", "sr720p-w32-m16-bf16", "swinir256-bf16"],
}


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


class ClockSampler:
    """nvidia-smi SM clock / throttle sampling while the timed region runs."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.idx = device_index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            import tempfile
            fd, self.path = tempfile.mkstemp(prefix=f"nystra_clocks_{self.idx}_", suffix=".csv")
            self.f = os.fdopen(fd, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
            if self.path:
                os.remove(self.path)
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        with open(self.path) as fh:
            lines = fh.readlines()
        os.remove(self.path)
        for line in lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i, x in enumerate(r) if x.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


def _oracle_bias(wl, lo: int, hi: int):
    """The score bias of units lo .. hi - 1 for the oracle (unit u uses head u % heads), or None."""
    bias = workloads.make_bias(wl)
    if bias is None:
        return None
    return bias.double().numpy()[np.arange(lo, hi) % wl.heads]


def _oracle_inputs(wl):
    """Host float64 (q, k, v) ``[units, N, d]`` the oracle times; for a fused
    front end the oracle's own projections of the workload's tokens."""
    import oracle  # CPU baseline only
    if wl.front == "qkv":
        x, w = workloads.make_x_wqkv(wl)
        q, k, v = oracle.project_qkv(x, w, None, wl.heads)
        return tuple(a.reshape(-1, wl.N, wl.d) for a in (q, k, v))
    return tuple(x.reshape(-1, wl.N, wl.d).double().numpy() for x in workloads.make_qkv(wl))


def _time_oracle(wl, q, k, v, budget_s: float, max_units: int | None = None):
    """Time the float64 oracle on a bounded sample of the workload's units
    (q, k, v: float64 ``[units, N, d]``; a fused front end's projections are
    made outside the timed region)."""
    import oracle  # CPU baseline only
    qd, kd, vd = q, k, v
    # calibrate on a few units, then size the sample to the budget
    n0 = min(64, qd.shape[0])
    t0 = time.perf_counter()
    oracle.nystra_attention(qd[:n0], kd[:n0], vd[:n0], wl.m, wl.iters, wl.landmarks, _oracle_bias(wl, 0, n0))
    per_unit = max((time.perf_counter() - t0) / n0, 1e-9)
    n = int(min(qd.shape[0], max(1, budget_s / per_unit)))
    if max_units:
        n = min(n, max_units)
    # repeat passes over the sample until the budget is used (at least one pass)
    passes, t0 = 0, time.perf_counter()
    while True:
        oracle.nystra_attention(qd[:n], kd[:n], vd[:n], wl.m, wl.iters, wl.landmarks, _oracle_bias(wl, 0, n))
        passes += 1
        dt = time.perf_counter() - t0
        if dt >= budget_s:
            break
    return passes * n * wl.N / dt, n, passes, dt, oracle.threads()


def _l2_bytes() -> int:
    if torch.cuda.is_available():
        return int(torch.cuda.get_device_properties(0).L2_cache_size)
    return 126 * 2**20  # GB300 (only when no GPU is visible)


def _config(wl, ws: int):
    """The `config` object both arms report: the workload and how the timed
    launches avoid L2 residency (rotating input/output sets > 3x L2)."""
    io_bytes = wl.io_bytes
    nsets = max(2, -(-3 * _l2_bytes() // io_bytes))
    cfg = {
        "workload": wl.name, "n_windows": wl.n_windows, "heads": wl.heads, "N": wl.N, "d_h": wl.d, "m": wl.m,
        "iters": wl.iters, "io_dtype": wl.dtype, "landmarks": wl.landmarks, "bias": wl.bias or "none",
        "factors": "hi+lo 16-bit pairs" if wl.factors == "pairs" else "16-bit (NYSTRA_FACTORS_16)",
        "l2": f"rotating {nsets} input/output sets ({nsets * io_bytes / 1e6:.0f} MB > 3x L2)",
        "parallelism": f"replica x{ws} (independent windows)"}
    if wl.front == "qkv":
        cfg["front"] = "fused Q/K/V projection (tokens and W_QKV in)"
    return nsets, io_bytes, cfg


def unit_flops(wl) -> int:
    """Algorithmic flops of one (window, head) unit: the products of the
    method (S_L, S_U, S_A, W = G_U^n [V | 1], the iteration's four m x m
    products per step, Y = Z W, O = G_L^n Y), the landmark sums and, for a
    fused front end, the unit's share of the projection (2 N C 3 d_h)."""
    N, d, m = wl.N, wl.d, wl.m
    f = (2 * N * m * d + 2 * m * N * d + 2 * m * m * d + 2 * m * N * (d + 1) + 8 * wl.iters * m ** 3
         + 2 * m * m * (d + 1) + 2 * N * m * (d + 1) + 2 * N * d)
    if wl.front == "qkv":
        f += 2 * N * wl.C * 3 * d
    return f


def _tensor_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]), "measured"
    except Exception:
        return 1900.0, "fallback"


def run_reference(args, wl):
    ws, rank, _ = _dist()
    if rank != 0:
        return
    import oracle
    # per-step sample sized so that warmup+steps fit in about a minute
    per_step_budget = max(0.002, 60.0 / max(1, args.steps + args.warmup))
    qd, kd, vd = _oracle_inputs(wl)
    n0 = min(32, qd.shape[0])
    t0 = time.perf_counter()
    oracle.nystra_attention(qd[:n0], kd[:n0], vd[:n0], wl.m, wl.iters, wl.landmarks, _oracle_bias(wl, 0, n0))
    per_unit = max((time.perf_counter() - t0) / n0, 1e-9)
    n = int(min(qd.shape[0], max(1, per_step_budget / per_unit)))
    for _ in range(args.warmup):
        oracle.nystra_attention(qd[:n], kd[:n], vd[:n], wl.m, wl.iters, wl.landmarks, _oracle_bias(wl, 0, n))
    t0 = time.perf_counter()
    for s in range(args.steps):
        off = (s * n) % max(1, qd.shape[0] - n + 1)
        oracle.nystra_attention(qd[off:off + n], kd[off:off + n], vd[off:off + n], wl.m, wl.iters,
                                wl.landmarks, _oracle_bias(wl, off, off + n))
    dt = time.perf_counter() - t0
    value = args.steps * n * wl.N / dt
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": _config(wl, ws)[2],
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle.threads(), "kind": "oracle",
                         "sample": f"{n} of {qd.shape[0]} units per step (float64 C oracle, OpenMP"
                                   + ("; projections made beforehand)" if wl.front == "qkv" else ")")},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def _time_kernel(wl, dev, steps: int, warmup: int, ws: int, sampler=None):
    """Device-resident timing of one workload: `steps` launches of
    ``nystra_attention`` (bracketed by barriers, CUDA events on the launching
    stream, rotating input/output sets > 3x L2), then the exact window
    attention kernel on the same inputs.  Returns the timing record, the
    host inputs (for the end-to-end loop) and the device sets."""
    q, k, v = workloads.make_qkv(wl)
    esize = q.element_size()
    nsets, io_bytes, config = _config(wl, ws)
    assert io_bytes == 4 * q.numel() * esize
    sets = [tuple(x.to(dev) for x in (q, k, v)) + (torch.empty_like(q, device=dev),) for _ in range(nsets)]
    stream = torch.cuda.current_stream(dev)
    sptr = stream.cuda_stream
    bias = workloads.make_bias(wl)  # a model constant: pooled once, outside the timed region
    pooled = None if bias is None else binding.pool_bias(bias.to(dev), wl.m, wl.landmarks)
    shape = (wl.n_windows, wl.heads, wl.N, wl.d)
    dcode = {"f32": 0, "bf16": 1, "f16": 2}[wl.dtype]

    def step(i, exact=False):
        qd, kd, vd, od = sets[i % nsets]
        if exact:
            rc = binding.exact_window_attention(qd.data_ptr(), kd.data_ptr(), vd.data_ptr(), od.data_ptr(),
                                                *shape, dcode, sptr)
        elif pooled is not None:
            rc = binding.nystra_attention_bias(qd.data_ptr(), kd.data_ptr(), vd.data_ptr(), od.data_ptr(), *shape,
                                               wl.m, wl.iters, binding._lm(wl.landmarks, wl.factors),
                                               *(x.data_ptr() for x in pooled), 1, dcode, sptr)
        elif wl.landmarks == "patches" or wl.factors != "pairs":
            rc = binding.nystra_attention_ex(qd.data_ptr(), kd.data_ptr(), vd.data_ptr(), od.data_ptr(), *shape,
                                             wl.m, wl.iters, binding._lm(wl.landmarks, wl.factors), dcode, sptr)
        else:
            rc = binding.nystra_attention(qd.data_ptr(), kd.data_ptr(), vd.data_ptr(), od.data_ptr(), *shape,
                                          wl.m, wl.iters, dcode, sptr)
        if rc != 0:
            raise binding.NystraError(rc, "bench step")

    def barrier():
        torch.cuda.synchronize(dev)
        if ws > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize(dev)

    w0 = time.perf_counter()
    for i in range(warmup):
        step(i)
    barrier()
    per_launch = (time.perf_counter() - w0) / max(1, warmup)
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    if sampler is not None:
        sampler.__enter__()
    try:
        # Untimed launches of the same kernel while the clock sampler runs, so
        # that its samples see the GPU under this load even when the timed
        # region itself is shorter than the sampling interval.
        if sampler is not None:
            for i in range(min(20000, int(0.6 / max(per_launch, 1e-6)))):
                step(i)
        barrier()
        for i in range(steps):
            starts[i].record(stream)
            step(i)
            ends[i].record(stream)
        barrier()
    finally:
        if sampler is not None:
            sampler.__exit__()
    total_ms = starts[0].elapsed_time(ends[-1])
    kern_ms = statistics.mean(s.elapsed_time(e) for s, e in zip(starts, ends))
    total_ms = shard.max_over_ranks(total_ms, dev)

    # exact window attention on the same inputs (the computation replaced)
    esteps = max(3, min(steps, 200))
    for i in range(3):
        step(i, exact=True)
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(esteps):
        step(i, exact=True)
    e1.record(stream)
    barrier()
    exact_ms = e0.elapsed_time(e1) / esteps

    peak, peak_kind = _peaks()
    achieved = io_bytes / (kern_ms * 1e-3) / 1e9
    mt = MEASURED_TRAFFIC.get(wl.name)
    traffic = mt["bytes"] if mt and mt["src_hash"] == _kernel_src_hash(mt["files"]) else None
    units_tokens = wl.n_windows * wl.heads * wl.N
    rec = {
        "total_ms": total_ms, "kern_ms": kern_ms, "config": config, "pooled": pooled,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic, "peak_kind": peak_kind,
                     "bytes_per_launch": io_bytes, "kernel_ms": kern_ms},
        "comparator": {"kernel": "exact_window_attention", "ms_per_step": exact_ms,
                       "value": units_tokens / (exact_ms * 1e-3), "speedup": exact_ms / (total_ms / steps)},
    }
    return rec, (q, k, v), sets


def run_cuda(args, wl):
    ws, rank, local = _dist()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    binding.lib()  # fail loudly if the library is missing

    clk = ClockSampler(local)
    rec, (q, k, v), sets = _time_kernel(wl, dev, args.steps, args.warmup, ws, sampler=clk)
    total_ms, pooled = rec["total_ms"], rec["pooled"]
    esize = q.element_size()
    units_tokens = wl.n_windows * wl.heads * wl.N
    value = shard.aggregate_rate(units_tokens, args.steps, total_ms, ws)

    def barrier():
        torch.cuda.synchronize(dev)
        if ws > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize(dev)

    # End to end through the public API: every step copies its inputs from
    # pinned host memory, makes the call and reads the output back.  Two
    # streams with their own device buffers let step i+1's copies overlap step
    # i's kernel and read-back (separate copy engines for each direction).
    hq, hk, hv = (x.pin_memory() for x in (q, k, v))
    hos = [torch.empty_like(q).pin_memory() for _ in range(2)]
    streams = [torch.cuda.Stream(dev) for _ in range(2)]

    def e2e_step(i):
        dq, dk, dv, do = sets[i % 2]
        with torch.cuda.stream(streams[i % 2]):
            dq.copy_(hq, non_blocking=True); dk.copy_(hk, non_blocking=True); dv.copy_(hv, non_blocking=True)
            if pooled is None:
                binding.nystra(dq, dk, dv, wl.m, wl.iters, out=do, landmarks=wl.landmarks, factors=wl.factors)
            else:
                binding.nystra_biased(dq, dk, dv, pooled, wl.m, wl.iters, out=do, landmarks=wl.landmarks,
                                      factors=wl.factors)
            hos[i % 2].copy_(do, non_blocking=True)

    e2e_steps = max(4, min(args.steps, 50))
    for i in range(2):
        e2e_step(i)
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(streams[0])
    streams[1].wait_event(e0)
    for i in range(e2e_steps):
        e2e_step(i)
    done1 = torch.cuda.Event()
    done1.record(streams[1])
    streams[0].wait_event(done1)
    e1.record(streams[0])
    barrier()
    e2e_ms = shard.max_over_ranks(e0.elapsed_time(e1) / e2e_steps, dev)
    e2e_value = shard.aggregate_rate(units_tokens, 1, e2e_ms, ws)
    del sets, hq, hk, hv, hos

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype, "data": "synthetic",
        "config": rec["config"], "roofline": rec["roofline"], "comparator": rec["comparator"],
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": 3 * q.numel() * esize,
                "d2h_bytes_per_step": q.numel() * esize, "streams": 2},
        "gpu_launches": args.steps,
        "clocks": clk.summary(),
    }
    # The other workloads the headline sits beside, each with its own roofline
    # and comparator (same timing rules; not part of `value`).
    extra = []
    for name in ([] if args.no_extra else EXTRA_WORKLOADS.get(wl.name, [])):
        xwl = workloads.WORKLOADS[name]
        xrec, _, xsets = _time_kernel(xwl, dev, max(args.steps, 20), args.warmup, ws)
        del xsets
        extra.append({"workload": name, "value": shard.aggregate_rate(xwl.units * xwl.N, max(args.steps, 20),
                                                                      xrec["total_ms"], ws),
                      "ms_per_step": xrec["total_ms"] / max(args.steps, 20), "config": xrec["config"],
                      "roofline": xrec["roofline"], "comparator": xrec["comparator"]})
    if extra:
        line["extra_workloads"] = extra
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        val, n, passes, dt, cores = _time_oracle(wl, *_oracle_inputs(wl), budget_s=args.cpu_budget)
        line["cpu_baseline"] = {"value": val, "unit": UNIT, "cores": cores, "kind": "oracle",
                                "sample": f"{n} of {wl.units} units x {passes} passes, {dt:.1f} s "
                                          "(float64 C oracle, OpenMP)"}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


def run_cuda_qkv(args, wl):
    """One step = one nystra_attention_qkv call: the window tokens and W_QKV in,
    the projections of Eq. (1) and PnP-Nystra fused.  Its comparator is the
    unfused path it replaces (cuBLAS projection, head split, nystra_attention)."""
    ws, rank, local = _dist()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    binding.lib()  # fail loudly if the library is missing

    x, w = workloads.make_x_wqkv(wl)
    esize = x.element_size()
    nsets, io_bytes, config = _config(wl, ws)
    assert io_bytes == (2 * x.numel() + w.numel()) * esize
    wd = w.to(dev)  # a model constant: resident
    sets = [(x.to(dev), torch.empty(wl.shape, dtype=x.dtype, device=dev)) for _ in range(nsets)]
    stream = torch.cuda.current_stream(dev)
    sptr = stream.cuda_stream
    bias = workloads.make_bias(wl)
    pooled = None if bias is None else binding.pool_bias(bias.to(dev), wl.m, wl.landmarks)
    bp = (0, 0, 0) if pooled is None else tuple(t.data_ptr() for t in pooled)
    dcode = {"bf16": 1, "f16": 2}[wl.dtype]

    def step(i):
        xd, od = sets[i % nsets]
        rc = binding.nystra_attention_qkv(xd.data_ptr(), wd.data_ptr(), 0, od.data_ptr(), wl.n_windows, wl.heads,
                                          wl.N, wl.d, wl.m, wl.iters, binding._lm(wl.landmarks, wl.factors), *bp,
                                          1 if pooled is not None else 0, dcode, sptr)
        if rc != 0:
            raise binding.NystraError(rc, "bench step")

    def unfused_step(i):
        xd, od = sets[i % nsets]
        y = xd.reshape(-1, wl.C) @ wd.T
        q, k, v = (y.view(wl.n_windows, wl.N, 3, wl.heads, wl.d)[:, :, j].transpose(1, 2).contiguous()
                   for j in range(3))
        if pooled is None:
            binding.nystra(q, k, v, wl.m, wl.iters, out=od, landmarks=wl.landmarks)
        else:
            binding.nystra_biased(q, k, v, pooled, wl.m, wl.iters, out=od, landmarks=wl.landmarks)

    def barrier():
        torch.cuda.synchronize(dev)
        if ws > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize(dev)

    for i in range(args.warmup):
        step(i)
    barrier()
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    with ClockSampler(local) as clk:
        barrier()
        for i in range(args.steps):
            starts[i].record(stream)
            step(i)
            ends[i].record(stream)
        barrier()
    total_ms = starts[0].elapsed_time(ends[-1])
    kern_ms = statistics.mean(s.elapsed_time(e) for s, e in zip(starts, ends))
    total_ms = shard.max_over_ranks(total_ms, dev)
    units_tokens = wl.units * wl.N
    value = shard.aggregate_rate(units_tokens, args.steps, total_ms, ws)

    # the library's two-pass path: nystra_project_qkv (the projection with the
    # head split on the tcgen05 tensor cores) into resident Q, K, V, then
    # nystra_attention; and the projection alone
    qkv = tuple(torch.empty(wl.shape, dtype=x.dtype, device=dev) for _ in range(3))

    def project_step(i):
        binding.project_qkv(sets[i % nsets][0], wd, wl.heads, out=qkv, stream=stream)

    def two_pass_step(i):
        xd, od = sets[i % nsets]
        q, k, v = binding.project_qkv(xd, wd, wl.heads, out=qkv, stream=stream)
        if pooled is None:
            binding.nystra(q, k, v, wl.m, wl.iters, out=od, landmarks=wl.landmarks, factors=wl.factors)
        else:
            binding.nystra_biased(q, k, v, pooled, wl.m, wl.iters, out=od, landmarks=wl.landmarks,
                                  factors=wl.factors)

    usteps = max(3, min(args.steps, 100))

    def time_steps(fn):
        for i in range(3):
            fn(i)
        barrier()
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        for i in range(usteps):
            fn(i)
        a1.record(stream)
        barrier()
        return a0.elapsed_time(a1) / usteps

    unfused_ms = time_steps(unfused_step)
    project_ms = time_steps(project_step)
    two_pass_ms = time_steps(two_pass_step)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    # End to end: every step copies its tokens from pinned host memory and
    # reads the output back (the weights are a resident model constant).
    hx = x.pin_memory()
    hos = [torch.empty(wl.shape, dtype=x.dtype).pin_memory() for _ in range(2)]
    streams = [torch.cuda.Stream(dev) for _ in range(2)]

    def e2e_step(i):
        xd, od = sets[i % 2]
        with torch.cuda.stream(streams[i % 2]):
            xd.copy_(hx, non_blocking=True)
            binding.nystra_qkv(xd, wd, wl.heads, wl.m, wl.iters, pooled=pooled, out=od, landmarks=wl.landmarks,
                               factors=wl.factors)
            hos[i % 2].copy_(od, non_blocking=True)

    e2e_steps = max(4, min(args.steps, 50))
    for i in range(2):
        e2e_step(i)
    barrier()
    e0.record(streams[0])
    streams[1].wait_event(e0)
    for i in range(e2e_steps):
        e2e_step(i)
    done1 = torch.cuda.Event()
    done1.record(streams[1])
    streams[0].wait_event(done1)
    e1.record(streams[0])
    barrier()
    e2e_ms = shard.max_over_ranks(e0.elapsed_time(e1) / e2e_steps, dev)
    e2e_value = shard.aggregate_rate(units_tokens, 1, e2e_ms, ws)

    peak, peak_kind = _tensor_peak()
    flops = unit_flops(wl) * wl.units
    achieved = flops / (kern_ms * 1e-3) / 1e12
    mt = MEASURED_TRAFFIC.get(wl.name)
    traffic = mt["bytes"] if mt and mt["src_hash"] == _kernel_src_hash(mt["files"]) else None
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype, "data": "synthetic",
        "config": config,
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "traffic": traffic, "peak_kind": peak_kind,
                     "flops_per_launch": flops, "bytes_per_launch": io_bytes, "kernel_ms": kern_ms,
                     "hbm_GBps": io_bytes / (kern_ms * 1e-3) / 1e9},
        "comparator": {"kernel": "cuBLAS projection + head split + nystra_attention", "ms_per_step": unfused_ms,
                       "value": units_tokens / (unfused_ms * 1e-3), "speedup": unfused_ms / (total_ms / args.steps)},
        "two_pass": {"kernels": "nystra_project_qkv (tcgen05) + nystra_attention", "ms_per_step": two_pass_ms,
                     "value": units_tokens / (two_pass_ms * 1e-3),
                     "speedup_vs_fused": (total_ms / args.steps) / two_pass_ms,
                     "project_ms": project_ms,
                     "project_hbm_GBps": (4 * x.numel() * esize + w.numel() * esize) / (project_ms * 1e-3) / 1e9,
                     "project_TFLOPs": 2.0 * x.numel() * 3 * wl.C / (project_ms * 1e-3) / 1e12},
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": x.numel() * esize,
                "d2h_bytes_per_step": x.numel() * esize, "streams": 2},
        "gpu_launches": args.steps,
        "clocks": clk.summary(),
    }
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        val, n, passes, dt, cores = _time_oracle(wl, *_oracle_inputs(wl), budget_s=args.cpu_budget)
        line["cpu_baseline"] = {"value": val, "unit": UNIT, "cores": cores, "kind": "oracle",
                                "sample": f"{n} of {wl.units} units x {passes} passes, {dt:.1f} s "
                                          "(float64 C oracle, OpenMP; projections made beforehand)"}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="cuda", choices=["cuda", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(workloads.WORKLOADS))
    ap.add_argument("--cpu-budget", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extra", action="store_true", help="time the headline workload only")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    wl = workloads.WORKLOADS[args.workload]
    if args.impl == "reference":
        run_reference(args, wl)
    elif wl.front == "qkv":
        run_cuda_qkv(args, wl)
    else:
        run_cuda(args, wl)


if __name__ == "__main__":
    main()
