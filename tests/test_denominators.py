"""Step 7 divides by G_L^n Z G_U^n 1_N with no guard (Algorithm 1 as written).
Record, on each workload family's inputs (reduced in size, same recipe and
seed), how far the oracle's denominators stay from zero: min |den| / max |den|
per unit must not come within 1e-6, so that no parity case rests on a
near-singular division."""
import numpy as np
import pytest

import oracle
from paper_2506_08520_gb300 import workloads

W = workloads.WORKLOADS
CASES = [
    W["tiny"],
    W["swinir256-bf16"].with_(n_windows=16),
    W["uformer-s1"].with_(n_windows=32),
    W["uformer-s4"],
    W["large-w16-m32"].with_(n_windows=4),
    W["large-w16-m64"].with_(n_windows=4),
    W["large-w32-m32"].with_(n_windows=2),
    W["sr720p-w8-m8-bf16"].with_(map_hw=(32, 32, 8), n_windows=16),
    W["sr720p-w16-m16-f16"].with_(map_hw=(32, 32, 16), n_windows=4),
    W["sr720p-w32-m16-bf16"].with_(map_hw=(48, 64, 32), n_windows=4),  # edge-padded rows
]


@pytest.mark.parametrize("wl", CASES, ids=[c.name for c in CASES])
def test_denominators_stay_away_from_zero(wl):
    q, k, v = workloads.make_qkv(wl)
    qu, ku, vu = (x.reshape(-1, wl.N, wl.d) for x in (q, k, v))
    ratios = []
    for u in range(min(8, qu.shape[0])):
        den = oracle.nystra_stages(qu[u], ku[u], vu[u], wl.m, wl.iters)["den"]
        ratios.append(np.abs(den).min() / np.abs(den).max())
    print(f"{wl.name}: min|den|/max|den| over {len(ratios)} units = {min(ratios):.3e}")
    assert min(ratios) > 1e-6
