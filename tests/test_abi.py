"""C-ABI checks that need no GPU: the library loads, exports every symbol the
public header declares, and rejects invalid arguments before launching."""
import ctypes
import os
import re

import pytest

from paper_2506_08520_gb300 import build as nbuild
from paper_2506_08520_gb300 import binding as nb

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "nystra.h")


@pytest.fixture(scope="module")
def lib():
    nbuild.build()
    return nb.lib()


def declared_symbols():
    text = open(HEADER).read()
    return re.findall(r"NYSTRA_API\s+[\w\s\*]+?\b(\w+)\s*\(", text)


def test_header_declares_the_boundary():
    names = declared_symbols()
    for required in ("nystra_attention", "exact_window_attention", "nystra_strerror",
                     "nystra_version", "nystra_status", "nystra_check", "nystra_last_cuda_error",
                     "nystra_debug_wait_timeout", "nystra_debug_stages", "nystra_debug_stages_size",
                     "nystra_attention_ex", "nystra_pool_bias", "nystra_attention_bias", "nystra_attention_qkv",
                     "nystra_project_qkv"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    raw = ctypes.CDLL(nb.LIB_PATH)
    for name in declared_symbols():
        assert hasattr(raw, name), f"{name} declared in nystra.h but not exported"


def test_strerror_and_version(lib):
    for code in (0, -1, -2, -3, -4, -5, 7):
        assert isinstance(nb.strerror(code), str) and nb.strerror(code)
    assert nb.version() >= 100


# Pointers that are never dereferenced: every call below must fail validation
# (or be an empty no-op) before any CUDA call is made.
P = 1 << 20


@pytest.mark.parametrize("args,code", [
    (dict(N=64, d=30, m=16, iters=6, dtype=5), nb.NYSTRA_EDTYPE),
    (dict(N=64, d=30, m=15, iters=6), nb.NYSTRA_EINVAL),        # m does not divide N
    (dict(N=64, d=30, m=0, iters=6), nb.NYSTRA_EINVAL),
    (dict(N=64, d=30, m=128, iters=6), nb.NYSTRA_EINVAL),       # m > N
    (dict(N=2048, d=30, m=16, iters=6), nb.NYSTRA_EINVAL),      # N > 1024
    (dict(N=128, d=30, m=128, iters=6), nb.NYSTRA_EINVAL),      # m > 64
    (dict(N=64, d=65, m=16, iters=6), nb.NYSTRA_EINVAL),        # d_h > 64
    (dict(N=64, d=0, m=16, iters=6), nb.NYSTRA_EINVAL),
    (dict(N=64, d=30, m=16, iters=-1), nb.NYSTRA_EINVAL),
    (dict(N=64, d=30, m=16, iters=101), nb.NYSTRA_EINVAL),
    (dict(N=64, d=30, m=16, iters=6, q=0), nb.NYSTRA_EINVAL),   # null pointer
    (dict(N=64, d=30, m=16, iters=6, q=P + 8), nb.NYSTRA_EINVAL),  # misaligned
    (dict(N=64, d=30, m=16, iters=6, out=P), nb.NYSTRA_EINVAL),    # out aliases q
    (dict(N=64, d=30, m=16, iters=6, nw=-1), nb.NYSTRA_EINVAL),
    (dict(N=64, d=30, m=16, iters=6, nw=0), nb.NYSTRA_OK),         # empty: no-op
    (dict(N=64, d=30, m=16, iters=6, heads=0), nb.NYSTRA_OK),
])
def test_nystra_argument_validation(lib, args, code):
    q = args.get("q", P)
    out = args.get("out", 64 * P)
    rc = nb.nystra_attention(q, 2 * P, 3 * P, out, args.get("nw", 4), args.get("heads", 2),
                             args["N"], args["d"], args["m"], args["iters"], args.get("dtype", 1), None)
    assert rc == code


@pytest.mark.parametrize("args,code", [
    (dict(N=64, d=30, dtype=3), nb.NYSTRA_EDTYPE),
    (dict(N=0, d=30), nb.NYSTRA_EINVAL),
    (dict(N=1025, d=30), nb.NYSTRA_EINVAL),
    (dict(N=64, d=30, out=3 * P + 64), nb.NYSTRA_EINVAL),     # out overlaps v
    (dict(N=64, d=30, nw=0), nb.NYSTRA_OK),
])
def test_exact_argument_validation(lib, args, code):
    rc = nb.exact_window_attention(P, 2 * P, 3 * P, args.get("out", 64 * P), args.get("nw", 4), 2,
                                   args["N"], args["d"], args.get("dtype", 0), None)
    assert rc == code


def test_torch_wrappers_refuse_cpu_tensors(lib):
    import torch
    x = torch.zeros(1, 1, 64, 30)
    with pytest.raises(ValueError):
        nb.nystra(x, x, x)
    with pytest.raises(ValueError):
        nb.exact(x, x, x)


@pytest.mark.parametrize("limit_ns", [0, 999, 1_000_000_001, 1 << 62])
def test_debug_wait_limit_validation(lib, limit_ns):
    # out-of-range limits are refused on the host, before any launch
    assert nb.lib().nystra_debug_wait_timeout(limit_ns, None) == nb.NYSTRA_EINVAL


@pytest.mark.parametrize("N,d,m", [(64, 30, 16), (64, 32, 8), (64, 2, 16)])
def test_debug_stages_size(lib, N, d, m):
    # Qbar, Kbar, G_L^n, m_U, W, G_A^n, Z, Y, O
    want = 2 * m * d + N * m + m + 2 * m * (d + 1) + 2 * m * m + N * d
    assert nb.nystra_debug_stages_size(N, d, m) == want


@pytest.mark.parametrize("N,d,m", [(256, 30, 16), (64, 31, 16), (64, 34, 16), (64, 30, 32), (64, 30, 4)])
def test_debug_stages_size_rejects_other_shapes(lib, N, d, m):
    assert nb.nystra_debug_stages_size(N, d, m) == nb.NYSTRA_EINVAL


@pytest.mark.parametrize("args,code", [
    (dict(dtype=3), nb.NYSTRA_EDTYPE),
    (dict(N=256), nb.NYSTRA_EINVAL),          # only the 8x8-window path
    (dict(m=32), nb.NYSTRA_EINVAL),
    (dict(d=31), nb.NYSTRA_EINVAL),
    (dict(iters=-1), nb.NYSTRA_EINVAL),
    (dict(dtype=0, iters=7), nb.NYSTRA_EINVAL),  # fp32 runs this path up to 6 steps
    (dict(iters=13), nb.NYSTRA_EINVAL),          # 16-bit up to 12
    (dict(unit=8), nb.NYSTRA_EINVAL),         # units are 0..7
    (dict(unit=-1), nb.NYSTRA_EINVAL),
    (dict(dump=0), nb.NYSTRA_EINVAL),
    (dict(dump=5 * P + 4), nb.NYSTRA_EINVAL),  # misaligned
    (dict(lm=2), nb.NYSTRA_EINVAL),           # no such pooling
    (dict(lm=1, m=8), nb.NYSTRA_EINVAL),      # 8 landmarks are no square grid
    (dict(lm=1, dtype=0), nb.NYSTRA_EINVAL),  # patches: 16-bit I/O only here
])
def test_debug_stages_argument_validation(lib, args, code):
    a = dict(N=64, d=30, m=16, iters=6, dtype=1, unit=0, dump=5 * P)
    a.update(args)
    rc = nb.nystra_debug_stages(P, 2 * P, 3 * P, 4, 2, a["N"], a["d"], a["m"], a["iters"], a.get("lm", 0),
                                a["dtype"], a["unit"], a["dump"], None)
    assert rc == code


@pytest.mark.parametrize("args,code", [
    (dict(N=64, m=16, lm=2), nb.NYSTRA_EINVAL),     # no such pooling
    (dict(N=64, m=8, lm=1), nb.NYSTRA_EINVAL),      # m not a square
    (dict(N=128, m=16, lm=1), nb.NYSTRA_EINVAL),    # N not a square
    (dict(N=256, m=36, lm=1), nb.NYSTRA_EINVAL),    # 6 patches do not tile 16 columns (36 does not divide 256 either)
    (dict(N=64, m=16, lm=1, nw=0), nb.NYSTRA_OK),   # empty: no-op
    (dict(N=64, m=16, lm=0, nw=0), nb.NYSTRA_OK),
])
def test_nystra_ex_argument_validation(lib, args, code):
    rc = nb.nystra_attention_ex(P, 2 * P, 3 * P, 64 * P, args.get("nw", 4), 2, args["N"], 30, args["m"], 6,
                                args["lm"], 1, None)
    assert rc == code


@pytest.mark.parametrize("args,code", [
    (dict(N=64, m=15), nb.NYSTRA_EINVAL),          # m does not divide N
    (dict(N=64, m=8, lm=1), nb.NYSTRA_EINVAL),     # no square grid
    (dict(N=64, m=16, lm=2), nb.NYSTRA_EINVAL),
    (dict(nb=-1), nb.NYSTRA_EINVAL),
    (dict(nb=0), nb.NYSTRA_OK),                    # nothing to pool
    (dict(bias=0), nb.NYSTRA_EINVAL),
    (dict(bL=5 * P + 4), nb.NYSTRA_EINVAL),        # misaligned
    (dict(bU=P), nb.NYSTRA_EINVAL),                # output overlaps the bias
])
def test_pool_bias_argument_validation(lib, args, code):
    a = dict(N=64, m=16, lm=0, nb=6, bias=P, bL=8 * P, bU=9 * P, bA=10 * P)
    a.update(args)
    rc = nb.nystra_pool_bias(a["bias"], a["nb"], a["N"], a["m"], a["lm"], a["bL"], a["bU"], a["bA"], None)
    assert rc == code


@pytest.mark.parametrize("args,code", [
    (dict(bw=3), nb.NYSTRA_EINVAL),               # neither 1 nor n_windows
    (dict(bL=0), nb.NYSTRA_EINVAL),
    (dict(bA=10 * P + 8), nb.NYSTRA_EINVAL),      # misaligned
    (dict(bL=64 * P), nb.NYSTRA_EINVAL),          # overlaps out
    (dict(m=15), nb.NYSTRA_EINVAL),
    (dict(nw=0), nb.NYSTRA_OK),                   # empty: no-op
])
def test_attention_bias_argument_validation(lib, args, code):
    a = dict(nw=4, m=16, bL=8 * P, bU=9 * P, bA=10 * P, bw=1)
    a.update(args)
    rc = nb.nystra_attention_bias(P, 2 * P, 3 * P, 64 * P, a["nw"], 2, 64, 30, a["m"], 6, 0, a["bL"], a["bU"],
                                  a["bA"], a["bw"], 1, None)
    assert rc == code


@pytest.mark.parametrize("args,code", [
    (dict(dtype=0), nb.NYSTRA_EDTYPE),            # fp32: 16-bit I/O only
    (dict(dtype=7), nb.NYSTRA_EDTYPE),
    (dict(N=128), nb.NYSTRA_EINVAL),              # windows of 64, 256 or 1024 tokens
    (dict(m=32), nb.NYSTRA_EINVAL),               # m = 32 only with 32x32 windows
    (dict(N=256, m=32), nb.NYSTRA_EINVAL),
    (dict(N=1024, m=32, bL=8 * P), nb.NYSTRA_EINVAL),  # a score bias needs m <= 16
    (dict(N=256, m=64), nb.NYSTRA_EINVAL),
    (dict(d=31), nb.NYSTRA_EINVAL),               # odd d_h
    (dict(d=34), nb.NYSTRA_EINVAL),               # d_h > 32
    (dict(heads=12, d=32), nb.NYSTRA_EINVAL),     # C = 384 > NYSTRA_QKV_MAX_C
    (dict(iters=13), nb.NYSTRA_EINVAL),
    (dict(lm=1, m=8), nb.NYSTRA_EINVAL),          # square patches need m = 16
    (dict(lm=2), nb.NYSTRA_EINVAL),
    (dict(x=0), nb.NYSTRA_EINVAL),
    (dict(w=2 * P + 4), nb.NYSTRA_EINVAL),        # misaligned
    (dict(b=3 * P + 8), nb.NYSTRA_EINVAL),
    (dict(out=P + 64), nb.NYSTRA_EINVAL),         # overlaps x
    (dict(out=3 * P), nb.NYSTRA_EINVAL),          # overlaps the projection bias
    (dict(bL=8 * P, bw=3), nb.NYSTRA_EINVAL),     # bias windows neither 1 nor n_windows
    (dict(bL=8 * P, bA=0), nb.NYSTRA_EINVAL),
    (dict(bL=64 * P), nb.NYSTRA_EINVAL),          # score bias overlaps out
    (dict(nw=0), nb.NYSTRA_OK),                   # empty: no-op
    (dict(heads=0), nb.NYSTRA_OK),
])
def test_attention_qkv_argument_validation(lib, args, code):
    a = dict(x=P, w=2 * P, b=3 * P, out=64 * P, nw=4, heads=6, N=64, d=30, m=16, iters=6, lm=0,
             bL=0, bU=9 * P, bA=10 * P, bw=1, dtype=1)
    a.update(args)
    rc = nb.nystra_attention_qkv(a["x"], a["w"], a["b"], a["out"], a["nw"], a["heads"], a["N"], a["d"], a["m"],
                                 a["iters"], a["lm"], a["bL"], a["bU"], a["bA"], a["bw"], a["dtype"], None)
    assert rc == code


def test_qkv_max_width_matches_the_header():
    text = open(HEADER).read()
    assert f"#define NYSTRA_QKV_MAX_C {nb.QKV_MAX_C}" in text
    assert f"#define NYSTRA_PROJ_MAX_C {nb.PROJ_MAX_C}" in text
    assert f"#define NYSTRA_PROJ_MAX_N {nb.PROJ_MAX_N}" in text


@pytest.mark.parametrize("args,code", [
    (dict(dtype=0), nb.NYSTRA_EDTYPE),            # fp32: 16-bit I/O only
    (dict(dtype=7), nb.NYSTRA_EDTYPE),
    (dict(N=48), nb.NYSTRA_EINVAL),               # not a multiple of 32
    (dict(N=0), nb.NYSTRA_EINVAL),
    (dict(N=65536 + 32), nb.NYSTRA_EINVAL),
    (dict(d=31), nb.NYSTRA_EINVAL),               # odd d_h
    (dict(d=34), nb.NYSTRA_EINVAL),               # d_h > 32
    (dict(heads=13, d=30), nb.NYSTRA_EINVAL),     # C = 390 > NYSTRA_PROJ_MAX_C
    (dict(nw=-1), nb.NYSTRA_EINVAL),
    (dict(x=0), nb.NYSTRA_EINVAL),
    (dict(vv=0), nb.NYSTRA_EINVAL),
    (dict(w=2 * P + 4), nb.NYSTRA_EINVAL),        # misaligned
    (dict(b=3 * P + 8), nb.NYSTRA_EINVAL),
    (dict(q=P + 64), nb.NYSTRA_EINVAL),           # q overlaps x
    (dict(k=64 * P + 4096), nb.NYSTRA_EINVAL),    # k overlaps q
    (dict(v=3 * P), nb.NYSTRA_EINVAL),            # v overlaps the bias
    (dict(nw=0), nb.NYSTRA_OK),                   # empty: no-op
    (dict(heads=0), nb.NYSTRA_OK),
])
def test_project_qkv_argument_validation(lib, args, code):
    a = dict(x=P, w=2 * P, b=3 * P, q=64 * P, k=96 * P, vv=128 * P, nw=4, heads=6, N=64, d=30, dtype=1)
    if "v" in args:
        args = dict(args, vv=args.pop("v"))
    a.update(args)
    rc = nb.nystra_project_qkv(a["x"], a["w"], a["b"], a["q"], a["k"], a["vv"], a["nw"], a["heads"], a["N"], a["d"],
                               a["dtype"], None)
    assert rc == code


@pytest.mark.parametrize("lm,m,nw,code", [
    (nb.NYSTRA_FACTORS_16, 16, 0, nb.NYSTRA_OK),                               # segments, 16-bit factors: valid
    (nb.NYSTRA_FACTORS_16 | nb.NYSTRA_LANDMARKS_PATCHES, 16, 0, nb.NYSTRA_OK),  # square patches too
    (nb.NYSTRA_FACTORS_16 | nb.NYSTRA_LANDMARKS_PATCHES, 8, 4, nb.NYSTRA_EINVAL),  # 8 is no square
    (32, 16, 4, nb.NYSTRA_EINVAL),                                            # no such flag
    (nb.NYSTRA_FACTORS_16 | 2, 16, 4, nb.NYSTRA_EINVAL),                      # no such pooling
])
def test_factor_flag_validation(lib, lm, m, nw, code):
    assert nb.nystra_attention_ex(P, 2 * P, 3 * P, 64 * P, nw, 2, 64, 30, m, 6, lm, 1, None) == code


def test_factor_flag_is_refused_where_it_has_no_meaning(lib):
    # pooling a bias and the stage dump take a pooling only
    assert nb.nystra_pool_bias(P, 1, 64, 16, nb.NYSTRA_FACTORS_16, 2 * P, 3 * P, 4 * P, None) == nb.NYSTRA_EINVAL
    assert nb.nystra_debug_stages(P, 2 * P, 3 * P, 1, 1, 64, 30, 16, 6, nb.NYSTRA_FACTORS_16, 1, 0, 4 * P,
                                  None) == nb.NYSTRA_EINVAL


def _has_gpu():
    import torch
    return torch.cuda.is_available()


@pytest.mark.skipif(_has_gpu(), reason="checks the answer of a host without a usable sm_103 device")
def test_valid_calls_without_an_sm103_device_return_edevice(lib):
    # every argument is valid, so the calls reach the device check, which
    # finds no sm_103 GPU and refuses before any launch
    assert nb.nystra_attention(P, 2 * P, 3 * P, 64 * P, 4, 2, 64, 30, 16, 6, 1, None) == nb.NYSTRA_EDEVICE
    assert nb.nystra_attention_ex(P, 2 * P, 3 * P, 64 * P, 4, 2, 64, 30, 16, 6, nb.NYSTRA_FACTORS_16, 1,
                                  None) == nb.NYSTRA_EDEVICE
    assert nb.exact_window_attention(P, 2 * P, 3 * P, 64 * P, 4, 2, 64, 30, 1, None) == nb.NYSTRA_EDEVICE
    assert nb.nystra_pool_bias(P, 1, 64, 16, 0, 2 * P, 3 * P, 4 * P, None) == nb.NYSTRA_EDEVICE
    assert nb.nystra_attention_qkv(P, 2 * P, 0, 64 * P, 4, 2, 64, 30, 16, 6, 0, 0, 0, 0, 0, 1,
                                   None) == nb.NYSTRA_EDEVICE
    assert nb.nystra_project_qkv(P, 2 * P, 0, 64 * P, 96 * P, 128 * P, 4, 2, 64, 30, 1, None) == nb.NYSTRA_EDEVICE
    assert nb.nystra_debug_stages(P, 2 * P, 3 * P, 4, 2, 64, 30, 16, 6, 0, 1, 0, 4 * P, None) == nb.NYSTRA_EDEVICE
    assert nb.lib().nystra_debug_wait_timeout(10_000, None) == nb.NYSTRA_EDEVICE
    assert nb.strerror(nb.NYSTRA_EDEVICE) == "unsupported device (sm_103 required)"
