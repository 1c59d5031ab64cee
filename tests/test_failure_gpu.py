"""Failure detection on the GPU without a fault: a wait that can only time
out (nothing ever arrives on its mbarrier) must end at its limit, be reported
as NYSTRA_ETIMEOUT by the status call, and leave the context usable."""
import time

import pytest
import torch

from paper_2506_08520_gb300 import binding, workloads
from tests.parity import TOL, check_nystra

pytestmark = pytest.mark.gpu


def test_bounded_wait_reports_timeout_and_context_survives():
    torch.cuda.synchronize()
    assert binding.status() == binding.NYSTRA_OK
    t0 = time.perf_counter()
    assert binding.debug_wait_timeout(20_000_000) == binding.NYSTRA_OK  # 20 ms limit
    assert binding.status() == binding.NYSTRA_ETIMEOUT
    elapsed = time.perf_counter() - t0
    assert 0.015 <= elapsed < 5.0, f"wait ended after {elapsed:.3f} s"
    assert binding.check() == binding.NYSTRA_OK  # the record was cleared
    # the context still computes correctly
    q, k, v = workloads.random_qkv(8, 64, 30, "bf16", seed=11)
    err, worst = check_nystra(q, k, v, 16, 6)
    assert err <= TOL["bf16"], f"max rel err {err:.3e} at unit {worst}"
    assert binding.status() == binding.NYSTRA_OK
