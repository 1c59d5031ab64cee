// Fused Q/K/V projection + PnP-Nystra for 8x8 windows, fp16 I/O, derived
// factors rounded to fp16 (NYSTRA_FACTORS_16; nystra_qkv.cuh).
#include "nystra_qkv.cuh"

NYSTRA_QKV_DEFINE(f16_s16, nystra::Single16<__half>)
