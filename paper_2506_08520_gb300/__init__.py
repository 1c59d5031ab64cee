"""GB300-native (sm_103a) PnP-Nystra window attention.

``nystra(q, k, v, m, iters)`` and ``exact(q, k, v)`` call the C-ABI CUDA
library ``libnystra.so`` (see ``include/nystra.h``); ``workloads`` holds the
seeded synthetic inputs.  The library is loaded on first use and every call
fails loudly if it is missing: there is no CPU path.
"""
from .binding import (NystraError, check, debug_stages, debug_wait_timeout, exact, exact_window_attention,
                      nystra, nystra_attention, nystra_attention_bias, nystra_attention_ex, nystra_biased,
                      nystra_pool_bias, pool_bias, status, strerror, version)

__all__ = ["nystra", "exact", "nystra_attention", "nystra_attention_ex", "nystra_attention_bias", "nystra_pool_bias",
           "pool_bias", "nystra_biased", "exact_window_attention", "status", "check",
           "debug_wait_timeout", "debug_stages", "strerror", "version", "NystraError"]
