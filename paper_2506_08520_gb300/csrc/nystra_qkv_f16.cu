// Fused Q/K/V projection + PnP-Nystra for 8x8 windows, f16 I/O (nystra_qkv.cuh).
#include "nystra_qkv.cuh"

NYSTRA_QKV_DEFINE(f16, __half)
