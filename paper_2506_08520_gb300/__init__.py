"""GB300-native (sm_103a) PnP-Nystra window attention.

Device tensors ``[n_windows, heads, N, d_h]`` (fp32, bf16 or fp16); for the
fused projection, tokens ``x`` ``[n_windows, N, heads*d_h]`` and a linear
layer's weight ``w_qkv`` ``[3 heads d_h, heads d_h]`` (16-bit)::

    import paper_2506_08520_gb300 as pn
    o = pn.nystra(q, k, v, m=16, iters=6)                      # segment landmarks
    o = pn.nystra(q, k, v, m=16, iters=6, landmarks="patches") # square patches
    pooled = pn.pool_bias(bias, m=16)                          # bias [heads, N, N] fp32, once
    o = pn.nystra_biased(q, k, v, pooled, m=16, iters=6)       # with a score bias
    e = pn.exact(q, k, v)                                      # exact window attention
    o = pn.nystra_qkv(x, w_qkv, heads=6, b_qkv=b)              # fused Q/K/V projection
    q, k, v = pn.project_qkv(x, w_qkv, heads=6, b_qkv=b)       # the projection alone (tcgen05)

Every call goes through the C ABI of ``libnystra.so`` (``include/nystra.h``),
loaded on first use; it fails loudly if the library is missing: the GPU
binding has no CPU path.  The separate multi-core CPU library is
``paper_2506_08520_gb300.host`` (fp32 host tensors).  ``workloads`` holds the
seeded synthetic inputs; ``sweep`` times them
(``python -m paper_2506_08520_gb300.sweep``).
"""
from .binding import (NystraError, check, debug_stages, debug_wait_timeout, exact, exact_window_attention,
                      nystra, nystra_attention, nystra_attention_bias, nystra_attention_ex, nystra_biased,
                      nystra_attention_qkv, nystra_pool_bias, nystra_project_qkv, nystra_qkv, pool_bias, project_qkv,
                      status, strerror, version)

__all__ = ["nystra", "exact", "nystra_attention", "nystra_attention_ex", "nystra_attention_bias", "nystra_pool_bias",
           "pool_bias", "nystra_biased", "nystra_attention_qkv", "nystra_qkv", "nystra_project_qkv", "project_qkv",
           "exact_window_attention", "status", "check",
           "debug_wait_timeout", "debug_stages", "strerror", "version", "NystraError"]
