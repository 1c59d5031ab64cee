"""Seeded synthetic window-attention inputs shaped like the paper's workloads.

This module only draws random numbers and lays them out; it contains none of
the attention method's arithmetic.  It is the one piece shared by the CUDA
path's tests/benchmark and the float64 oracle's tests.

The paper evaluates PnP-Nystra inside pretrained SwinIR, Uformer-B and
Dehazeformer (Sec. 3, Table 2); neither the weights nor the datasets are
available, so each workload below is a synthetic stand-in with the same
window geometry (8x8 / 16x16 / 32x32 windows), head count and head width.

All tensors use the layout ``[n_windows, heads, N, d_h]`` (row-major,
contiguous), tokens of a window in row-major spatial order; the tokens of the
fused-projection workloads are ``[n_windows, N, heads*d_h]``.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import torch

DTYPES = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16}


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    n_windows: int
    heads: int
    N: int
    d: int
    m: int
    iters: int
    dtype: str
    seed: int
    recipe: str          # "iid" | "proj" | "lowrank" | "map"
    map_hw: tuple = ()   # (H, W, window) for recipe == "map"
    landmarks: str = "segments"  # landmark pooling: "segments" | "patches"
    bias: str = ""               # score bias: "" (none) | "relpos" (per-head relative-position bias)
    front: str = ""              # "" (inputs are Q, K, V) | "qkv" (inputs are the tokens X and W_QKV)
    factors: str = "pairs"       # derived factors: "pairs" (hi + lo, default) | "16" (NYSTRA_FACTORS_16)

    @property
    def units(self) -> int:
        return self.n_windows * self.heads

    @property
    def shape(self) -> tuple:
        return (self.n_windows, self.heads, self.N, self.d)

    @property
    def C(self) -> int:
        """Token width heads * d_h (the projections' input width)."""
        return self.heads * self.d

    @property
    def io_bytes(self) -> int:
        """Q, K, V read once and O written once; with the fused projection, X
        and the weights read once and O written once."""
        es = torch.tensor([], dtype=DTYPES[self.dtype]).element_size()
        if self.front == "qkv":
            return (2 * self.units * self.N * self.d + 3 * self.C * self.C) * es
        return 4 * self.units * self.N * self.d * es

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


def _sr_map(window: int, m: int, dtype: str) -> Workload:
    H, W = 720, 1280
    Hp = -(-H // window) * window
    nw = (Hp // window) * (W // window)
    return Workload(f"sr720p-w{window}-m{m}-{dtype}", nw, 6, window * window, 30, m, 6, dtype, 4,
                    "map", (H, W, window))


# Five workload families, sized like the paper's models (SwinIR, Uformer, Dehazeformer windows).
WORKLOADS = {
    # SwinIR-like 64x64 feature map, 8x8 windows: 64 windows, 6 heads, d_h = 30.
    "tiny": Workload("tiny", 64, 6, 64, 30, 16, 6, "f32", 0, "iid"),
    # SwinIR-like denoising at 256x256: 1024 windows of 8x8, Q/K/V = X W.
    "swinir256-f32": Workload("swinir256-f32", 1024, 6, 64, 30, 16, 6, "f32", 1, "proj"),
    "swinir256-bf16": Workload("swinir256-bf16", 1024, 6, 64, 30, 16, 6, "bf16", 1, "proj"),
    # Uformer-like 512x512: stage 1 (4096 windows, 1 head) and stage 4 (64 windows, 8 heads).
    "uformer-s1": Workload("uformer-s1", 4096, 1, 64, 32, 16, 6, "bf16", 2, "iid"),
    "uformer-s4": Workload("uformer-s4", 64, 8, 64, 32, 16, 6, "bf16", 2, "iid"),
    # Large windows with low-rank Q/K: 16x16 and 32x32 windows.
    "large-w16-m32": Workload("large-w16-m32", 1024, 4, 256, 32, 32, 6, "bf16", 3, "lowrank"),
    "large-w16-m64": Workload("large-w16-m64", 1024, 4, 256, 32, 64, 6, "bf16", 3, "lowrank"),
    "large-w32-m32": Workload("large-w32-m32", 256, 4, 1024, 32, 32, 6, "bf16", 3, "lowrank"),
    "large-w32-m64": Workload("large-w32-m64", 256, 4, 1024, 32, 64, 6, "bf16", 3, "lowrank"),
}
for _w in (8, 16, 32):
    for _m in (8, 16, 32, 64):
        for _dt in ("bf16", "f16"):
            _wl = _sr_map(_w, _m, _dt)
            WORKLOADS[_wl.name] = _wl
# The same inputs with square-patch landmarks (4 x 4 patches), and with a
# relative-position score bias.
for _name in ("swinir256-bf16", "sr720p-w16-m16-bf16", "sr720p-w32-m16-bf16"):
    WORKLOADS[_name + "-patches"] = WORKLOADS[_name].with_(name=_name + "-patches", landmarks="patches")
    WORKLOADS[_name + "-relpos"] = WORKLOADS[_name].with_(name=_name + "-relpos", bias="relpos")
# The same inputs with the derived factors rounded to 16 bits (NYSTRA_FACTORS_16).
for _name in ("swinir256-bf16", "sr720p-w8-m16-bf16", "sr720p-w16-m16-bf16", "sr720p-w32-m16-bf16",
              "sr720p-w32-m32-bf16", "large-w16-m64", "large-w32-m32", "uformer-s1"):
    WORKLOADS[_name + "-s16"] = WORKLOADS[_name].with_(name=_name + "-s16", factors="16")
# The same windows given as tokens X and projection weights (fused Q/K/V projection).
for _name in ("swinir256-bf16", "uformer-s1", "uformer-s4", "sr720p-w8-m16-bf16", "sr720p-w8-m16-f16",
              "swinir256-bf16-relpos", "sr720p-w16-m16-bf16", "sr720p-w32-m16-bf16", "sr720p-w32-m32-bf16",
              "sr720p-w16-m16-bf16-relpos"):
    WORKLOADS[_name + "-qkv"] = WORKLOADS[_name].with_(name=_name + "-qkv", front="qkv")


def _cast(x: np.ndarray, dtype: str) -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(x))
    if t.dtype == torch.float64 and dtype != "f32":
        t = t.float()
    return t.to(DTYPES[dtype]).contiguous()


def _iid(wl: Workload):
    rng = np.random.default_rng(wl.seed)
    return [rng.standard_normal(wl.shape) for _ in range(3)]


def _proj(wl: Workload):
    # X ~ N(0,1) [tokens, heads*d]; W_{Q,K,V} ~ N(0, 1/(heads*d)); tokens window-major.
    rng = np.random.default_rng(wl.seed)
    dm = wl.heads * wl.d
    X = rng.standard_normal((wl.n_windows * wl.N, dm))
    out = []
    for _ in range(3):
        Wt = rng.standard_normal((dm, dm)) / np.sqrt(dm)
        Y = (X @ Wt).reshape(wl.n_windows, wl.N, wl.heads, wl.d).transpose(0, 2, 1, 3)
        out.append(Y)
    return out


def _lowrank(wl: Workload, rank: int = 8, noise: float = 0.1):
    # Q, K = C B + noise * eps per head (B shared by all windows of a head); V ~ N(0,1).
    rng = np.random.default_rng(wl.seed)
    T = wl.n_windows * wl.N
    out = []
    for _ in range(2):
        B = rng.standard_normal((wl.heads, rank, wl.d)) / np.sqrt(rank)
        C = rng.standard_normal((wl.heads, T, rank))
        eps = rng.standard_normal((wl.heads, T, wl.d))
        X = np.einsum("htr,hrd->htd", C, B) + noise * eps
        out.append(X.reshape(wl.heads, wl.n_windows, wl.N, wl.d).transpose(1, 0, 2, 3))
    out.append(rng.standard_normal(wl.shape))
    return out


def _partition(fmap: np.ndarray, window: int) -> np.ndarray:
    """[heads, H, W, d] -> [n_windows, heads, window*window, d], edge-padding H."""
    h, H, W, d = fmap.shape
    Hp = -(-H // window) * window
    if Hp != H:
        fmap = np.concatenate([fmap, np.repeat(fmap[:, H - 1:H], Hp - H, axis=1)], axis=1)
    x = fmap.reshape(h, Hp // window, window, W // window, window, d)
    x = x.transpose(1, 3, 0, 2, 4, 5)
    return x.reshape(-1, h, window * window, d)


def _map(wl: Workload):
    H, W, window = wl.map_hw
    rng = np.random.default_rng(wl.seed)
    return [_partition(rng.standard_normal((wl.heads, H, W, wl.d), dtype=np.float32), window)
            for _ in range(3)]


_RECIPES = {"iid": _iid, "proj": _proj, "lowrank": _lowrank, "map": _map}


def make_qkv(wl: Workload | str):
    """Seeded host tensors (q, k, v) in the workload's I/O dtype, ``[n_windows, heads, N, d]``."""
    if isinstance(wl, str):
        wl = WORKLOADS[wl]
    return tuple(_cast(x, wl.dtype) for x in _RECIPES[wl.recipe](wl))


def _tokens_and_weights(wl: Workload):
    """Float64 tokens X ``[n_windows, N, C]`` and weights ``[3C, C]`` (row o is
    output feature o: the Q, K, V weights transposed and stacked).  The "proj"
    recipe returns the very draws ``_proj`` multiplies; the others draw X (an
    edge-padded feature map for "map") and W ~ N(0, 1/C)."""
    C = wl.C
    rng = np.random.default_rng(wl.seed)
    if wl.recipe == "map":
        H, W, window = wl.map_hw
        X = _partition(rng.standard_normal((1, H, W, C), dtype=np.float32), window)[:, 0]
    else:
        X = rng.standard_normal((wl.n_windows * wl.N, C)).reshape(wl.n_windows, wl.N, C)
    Ws = [rng.standard_normal((C, C)) / np.sqrt(C) for _ in range(3)]
    return X, np.concatenate([Wt.T for Wt in Ws], axis=0)


def make_x_wqkv(wl: Workload | str):
    """Seeded host tensors (x ``[n_windows, N, C]``, w_qkv ``[3C, C]``) in the
    workload's I/O dtype, for the fused projection."""
    if isinstance(wl, str):
        wl = WORKLOADS[wl]
    return tuple(_cast(a, wl.dtype) for a in _tokens_and_weights(wl))


def random_x_wqkv(n_windows: int, N: int, heads: int, d: int, dtype: str = "bf16", seed: int = 0,
                  with_bias: bool = True):
    """i.i.d. tokens N(0, 1), weights N(0, 1/C) and (optionally) an fp32 bias
    N(0, 0.1^2) for small parity and edge cases of the fused projection."""
    rng = np.random.default_rng(seed)
    C = heads * d
    x = _cast(rng.standard_normal((n_windows, N, C)), dtype)
    w = _cast(rng.standard_normal((3 * C, C)) / np.sqrt(C), dtype)
    b = torch.from_numpy(0.1 * rng.standard_normal(3 * C)).float() if with_bias else None
    return x, w, b


def random_qkv(n_units: int, N: int, d: int, dtype: str = "f32", seed: int = 0, scale: float = 1.0):
    """i.i.d. N(0, scale^2) inputs ``[n_units, N, d]`` for small parity and edge cases."""
    rng = np.random.default_rng(seed)
    return tuple(_cast(scale * rng.standard_normal((n_units, N, d)), dtype) for _ in range(3))


def relpos_bias(window: int, heads: int, seed: int, scale: float = 0.5) -> np.ndarray:
    """A relative-position score bias of a window x window window, as Swin-style
    layers add it: a seeded table of (2 window - 1)^2 offsets per head, indexed
    by the row and column offset of each token pair.  fp32 ``[heads, N, N]``."""
    rng = np.random.default_rng(seed)
    table = scale * rng.standard_normal(((2 * window - 1) ** 2, heads))
    r, c = np.divmod(np.arange(window * window), window)
    idx = (r[:, None] - r[None, :] + window - 1) * (2 * window - 1) + (c[:, None] - c[None, :] + window - 1)
    return np.ascontiguousarray(table[idx].transpose(2, 0, 1)).astype(np.float32)


def make_bias(wl: Workload | str):
    """The workload's score bias ``[heads, N, N]`` (fp32 host tensor), or None."""
    if isinstance(wl, str):
        wl = WORKLOADS[wl]
    if not wl.bias:
        return None
    return torch.from_numpy(relpos_bias(int(round(wl.N ** 0.5)), wl.heads, wl.seed + 100))
