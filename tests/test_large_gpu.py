"""Maximum sizes: more than 2^32 elements per tensor (about 9 GB each in bf16),
so any 32-bit element offset would wrap.  Inputs are drawn on the device from
a seeded generator; the oracle checks a sample that includes the last unit."""
import numpy as np
import pytest
import torch

import oracle
from paper_2506_08520_gb300 import binding
from tests.parity import TOL, per_unit_rel, sample_units

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2506_08520_gb300 import build
    build.build()


@pytest.mark.parametrize("N,d,m", [(64, 32, 16), (256, 32, 16), (1024, 32, 16)])
def test_more_than_2_to_the_32_elements(N, d, m):
    units = (1 << 32) // (N * d) + 3  # the last units start beyond element 2^32
    g = torch.Generator(device="cuda").manual_seed(N)
    q, k, v = (torch.randn(units, N, d, device="cuda", dtype=torch.bfloat16, generator=g) for _ in range(3))
    out = binding.nystra(q, k, v, m, 6)
    torch.cuda.synchronize()
    assert binding.status() == binding.NYSTRA_OK
    idx = sample_units(units, 48)
    assert idx[-1] == units - 1
    sel = torch.as_tensor(idx, device="cuda")
    qs, ks, vs, os_ = (x.index_select(0, sel).cpu() for x in (q, k, v, out))
    del q, k, v, out
    torch.cuda.empty_cache()
    err = per_unit_rel(os_.double().numpy(), oracle.nystra_attention(qs, ks, vs, m, 6))
    assert err.max() <= TOL["bf16"], f"max rel err {err.max():.3e} at sampled unit {int(idx[err.argmax()])}"
