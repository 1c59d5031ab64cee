// Fused Q/K/V projection + PnP-Nystra for 8x8 windows, bf16 I/O (nystra_qkv.cuh).
#include "nystra_qkv.cuh"

NYSTRA_QKV_DEFINE(bf16, __nv_bfloat16)
