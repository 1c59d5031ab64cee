"""Throughput sweep over the synthetic workloads: PnP-Nystra and the exact
window attention it replaces, on the same device inputs.

    python -m paper_2506_08520_gb300.sweep [--list] [name ...]

One JSON line per workload: the median CUDA-event time of each kernel over
rotating input/output sets (together more than 3x the L2 size, so every launch
reads its inputs from HBM), the algorithmic bytes (Q, K, V read once, O written
once), the achieved GB/s and its fraction of the measured HBM copy bandwidth,
tokens*heads/s (for edge-padded maps also counting only the real tokens), and
the speedup over exact attention (which runs without the bias).  A mix
("uformer-mix": Uformer stages 1 and 4) launches its workloads back to back on
one stream and is timed as one.  A workload with a relative-position bias
pools it once (a model constant) and times the biased call.  A fused-projection
workload ("-qkv": tokens X and W_QKV in, algorithmic bytes X + W + O) is timed
against the unfused path it replaces: one cuBLAS projection X W_QKV^T (torch),
the copy that splits heads, and nystra_attention; and against the library's
own two-pass path: nystra_project_qkv (the projection with the head split on
the tcgen05 tensor cores, timed alone too) followed by nystra_attention.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import sys

import torch

from . import binding, workloads

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# Workloads launched back to back and timed as one step.
MIXES = {"uformer-mix": ("uformer-s1", "uformer-s4")}

DEFAULT = (["tiny", "swinir256-f32", "swinir256-bf16", "uformer-s1", "uformer-s4", "uformer-mix"]
           + [f"large-w{w}-m{m}" for w in (16, 32) for m in (32, 64)]
           + [f"sr720p-w{w}-m{m}-{dt}" for w in (8, 16, 32) for m in (8, 16, 32, 64) for dt in ("bf16", "f16")]
           + [f"{n}-{x}" for x in ("patches", "relpos")
              for n in ("swinir256-bf16", "sr720p-w16-m16-bf16", "sr720p-w32-m16-bf16")]
           + [n for n in workloads.WORKLOADS if n.endswith("-qkv")]
           + [n for n in workloads.WORKLOADS if n.endswith("-s16")])


def hbm_peak_gbs() -> tuple[float, str]:
    """Measured HBM copy bandwidth of this GPU pool, else the fallback figure."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


def _real_tokens(wl: workloads.Workload) -> int:
    if wl.recipe == "map":
        H, W, _ = wl.map_hw
        return H * W * wl.heads
    return wl.units * wl.N


def _median_ms(launch, n_sets: int, reps: int) -> float:
    stream = torch.cuda.current_stream()
    for i in range(min(5, reps)):
        launch(i % n_sets)
    torch.cuda.synchronize()
    evs = []
    for i in range(reps):
        s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s.record(stream)
        launch(i % n_sets)
        e.record(stream)
        evs.append((s, e))
    torch.cuda.synchronize()
    return statistics.median(s.elapsed_time(e) for s, e in evs)


def run_qkv(wl: workloads.Workload, l2_bytes: int, peak: float, reps: int = 50) -> dict:
    """The fused projection against projecting first (cuBLAS + head split + nystra_attention)."""
    io = wl.io_bytes
    n_sets = max(2, -(-3 * l2_bytes // io))
    dev = torch.device("cuda")
    x, w = workloads.make_x_wqkv(wl)
    w = w.to(dev)
    bias = workloads.make_bias(wl)
    pooled = None if bias is None else binding.pool_bias(bias.to(dev), wl.m, wl.landmarks)
    sets = [(x.to(dev), torch.empty(wl.shape, dtype=x.dtype, device=dev)) for _ in range(n_sets)]

    def fused(i):
        xs, o = sets[i]
        binding.nystra_qkv(xs, w, wl.heads, wl.m, wl.iters, pooled=pooled, out=o, landmarks=wl.landmarks,
                           factors=wl.factors)

    def unfused(i):
        xs, o = sets[i]
        y = xs.reshape(-1, wl.C) @ w.T
        q, k, v = (y.view(wl.n_windows, wl.N, 3, wl.heads, wl.d)[:, :, j].transpose(1, 2).contiguous()
                   for j in range(3))
        if pooled is None:
            binding.nystra(q, k, v, wl.m, wl.iters, out=o, landmarks=wl.landmarks, factors=wl.factors)
        else:
            binding.nystra_biased(q, k, v, pooled, wl.m, wl.iters, out=o, landmarks=wl.landmarks,
                                  factors=wl.factors)

    qkv = tuple(torch.empty(wl.shape, dtype=x.dtype, device=dev) for _ in range(3))

    def project(i):
        binding.project_qkv(sets[i][0], w, wl.heads, out=qkv)

    def two_pass(i):
        xs, o = sets[i]
        q, k, v = binding.project_qkv(xs, w, wl.heads, out=qkv)
        if pooled is None:
            binding.nystra(q, k, v, wl.m, wl.iters, out=o, landmarks=wl.landmarks, factors=wl.factors)
        else:
            binding.nystra_biased(q, k, v, pooled, wl.m, wl.iters, out=o, landmarks=wl.landmarks,
                                  factors=wl.factors)

    t_f = _median_ms(fused, n_sets, reps)
    t_u = _median_ms(unfused, n_sets, max(10, reps // 5))
    t_p = _median_ms(project, n_sets, reps)
    t_2 = _median_ms(two_pass, n_sets, reps)
    tokens = wl.units * wl.N
    gbs = io / (t_f * 1e-3) / 1e9
    proj_bytes = x.numel() * x.element_size() * 4 + w.numel() * w.element_size()  # X in, Q K V out, W
    res = {"name": wl.name, "units": wl.units, "io_MB": io / 1e6, "nystra_ms": t_f, "unfused_ms": t_u,
           "GBps": gbs, "frac_of_hbm": gbs / peak, "tokens_heads_per_s": tokens / (t_f * 1e-3),
           "speedup_vs_unfused": t_u / t_f, "project_ms": t_p,
           "project_frac_of_hbm": proj_bytes / (t_p * 1e-3) / 1e9 / peak,
           "project_TFLOPs": 2.0 * x.numel() * 3 * wl.C / (t_p * 1e-3) / 1e12,
           "two_pass_ms": t_2, "speedup_vs_two_pass": t_2 / t_f}
    real = _real_tokens(wl)
    if real != tokens:
        res["real_tokens_heads_per_s"] = real / (t_f * 1e-3)
    del sets
    torch.cuda.empty_cache()
    return res


def run(name: str, l2_bytes: int, peak: float, reps: int = 50, exact_reps: int = 10) -> dict:
    if name in workloads.WORKLOADS and workloads.WORKLOADS[name].front == "qkv":
        return run_qkv(workloads.WORKLOADS[name], l2_bytes, peak, reps)
    parts = [workloads.WORKLOADS[n] for n in MIXES.get(name, (name,))]
    io = sum(wl.io_bytes for wl in parts)
    n_sets = max(2, -(-3 * l2_bytes // io))
    dev = torch.device("cuda")
    sets, pooled = [], []
    for wl in parts:
        q, k, v = workloads.make_qkv(wl)
        sets.append([tuple(x.to(dev) for x in (q, k, v)) + (torch.empty_like(q, device=dev),)
                     for _ in range(n_sets)])
        bias = workloads.make_bias(wl)  # pooled once: a model constant
        pooled.append(None if bias is None else binding.pool_bias(bias.to(dev), wl.m, wl.landmarks))

    def nystra(i):
        for wl, ss, pb in zip(parts, sets, pooled):
            a, b, c, o = ss[i]
            if pb is None:
                binding.nystra(a, b, c, wl.m, wl.iters, out=o, landmarks=wl.landmarks, factors=wl.factors)
            else:
                binding.nystra_biased(a, b, c, pb, wl.m, wl.iters, out=o, landmarks=wl.landmarks,
                                      factors=wl.factors)

    def exact(i):
        for ss in sets:
            a, b, c, o = ss[i]
            binding.exact(a, b, c, out=o)

    t_n = _median_ms(nystra, n_sets, reps)
    t_e = _median_ms(exact, n_sets, exact_reps)
    tokens = sum(wl.units * wl.N for wl in parts)
    gbs = io / (t_n * 1e-3) / 1e9
    res = {"name": name, "units": sum(wl.units for wl in parts), "io_MB": io / 1e6, "nystra_ms": t_n,
           "exact_ms": t_e, "GBps": gbs, "frac_of_hbm": gbs / peak,
           "tokens_heads_per_s": tokens / (t_n * 1e-3), "speedup_vs_exact": t_e / t_n}
    real = sum(_real_tokens(wl) for wl in parts)
    if real != tokens:
        res["real_tokens_heads_per_s"] = real / (t_n * 1e-3)
    del sets, pooled
    torch.cuda.empty_cache()
    return res


def main(argv=None) -> int:
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("names", nargs="*", help="workloads or mixes (default: all)")
    ap.add_argument("--list", action="store_true", help="print the workload names and exit")
    ap.add_argument("--reps", type=int, default=50)
    args = ap.parse_args(argv)
    names = args.names or DEFAULT
    unknown = [n for n in names if n not in workloads.WORKLOADS and n not in MIXES]
    if unknown:
        ap.error(f"unknown workloads: {unknown}")
    if args.list:
        print("\n".join(names))
        return 0
    binding.lib()  # fail loudly without the library
    l2 = int(torch.cuda.get_device_properties(0).L2_cache_size)
    peak, kind = hbm_peak_gbs()
    for n in names:
        r = run(n, l2, peak, reps=args.reps)
        r["peak_gbs"], r["peak_kind"] = peak, kind
        print(json.dumps(r), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())
