// C ABI of the PnP-Nystra library: argument validation and kernel dispatch.
// Declarations and the full contract are in include/nystra.h.
#include <stdint.h>

#include <atomic>

#include "common.cuh"
#include "nystra.h"

namespace {

thread_local int g_last_cuda_error = 0;

int fail_cuda(cudaError_t e) {
    g_last_cuda_error = (int)e;
    return NYSTRA_ELAUNCH;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

bool overlaps(const void* a, const void* b, size_t bytes) {
    const uintptr_t x = (uintptr_t)a, y = (uintptr_t)b;
    return x < y + bytes && y < x + bytes;
}

// [a, a + na) and [b, b + nb) intersect.
bool overlaps2(const void* a, size_t na, const void* b, size_t nb) {
    const uintptr_t x = (uintptr_t)a, y = (uintptr_t)b;
    return x < y + nb && y < x + na;
}

size_t elem_size(int dtype) { return dtype == NYSTRA_F32 ? 4 : 2; }

// Shared checks of both entry points.  Returns NYSTRA_OK or an error code.
int check_common(const void* q, const void* k, const void* v, void* out, int n_windows, int heads,
                 int N, int d_h, int dtype) {
    if (dtype != NYSTRA_F32 && dtype != NYSTRA_BF16 && dtype != NYSTRA_F16) return NYSTRA_EDTYPE;
    if (n_windows < 0 || heads < 0) return NYSTRA_EINVAL;
    if (N < 1 || N > NYSTRA_MAX_N || d_h < 1 || d_h > NYSTRA_MAX_DH) return NYSTRA_EINVAL;
    if ((long long)n_windows * heads == 0) return NYSTRA_OK;
    if (!q || !k || !v || !out) return NYSTRA_EINVAL;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out)) return NYSTRA_EINVAL;
    const size_t bytes = (size_t)n_windows * heads * N * d_h * elem_size(dtype);
    if (overlaps(out, q, bytes) || overlaps(out, k, bytes) || overlaps(out, v, bytes)) return NYSTRA_EINVAL;
    return NYSTRA_OK;
}

// Whether the current device is an sm_103 GPU (the kernels' only target);
// false when there is no usable device.  Cached per device ordinal.
bool device_ok() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= nystra::kMaxDevices) {
        (void)cudaGetLastError();
        return false;
    }
    static std::atomic<int> cache[nystra::kMaxDevices];  // 0 unknown, 1 sm_103, 2 other
    int c = cache[dev].load(std::memory_order_relaxed);
    if (c == 0) {
        int major = 0, minor = 0;
        const bool ok = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) == cudaSuccess &&
                        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) == cudaSuccess &&
                        major == 10 && minor == 3;
        if (!ok) (void)cudaGetLastError();
        c = ok ? 1 : 2;
        cache[dev].store(c, std::memory_order_relaxed);
    }
    return c == 1;
}

// Landmark pooling and option flags of the `landmarks` argument.
constexpr int kPoolMask = 15;
bool flags_ok(int landmarks) {
    const int pool = landmarks & kPoolMask, rest = landmarks & ~kPoolMask;
    return (pool == NYSTRA_LANDMARKS_SEGMENTS || pool == NYSTRA_LANDMARKS_PATCHES) &&
           (rest == 0 || rest == NYSTRA_FACTORS_16);
}

// Integer square root of n, or -1 if n is not a perfect square.
int exact_sqrt(int n) {
    int r = 0;
    while ((r + 1) * (r + 1) <= n) ++r;
    return r * r == n ? r : -1;
}

}  // namespace

namespace {

// The body of every PnP-Nystra entry point; bias.L == nullptr: no bias.
int nystra_call(const void* q, const void* k, const void* v, void* out, int n_windows, int heads, int N,
                int d_h, int m, int iters, int landmarks, int dtype, void* stream, const nystra::NystraBias& bias) {
    int rc = check_common(q, k, v, out, n_windows, heads, N, d_h, dtype);
    if (rc != NYSTRA_OK) return rc;
    if (m < 1 || m > N || m > NYSTRA_MAX_M || N % m != 0) return NYSTRA_EINVAL;
    if (iters < 0 || iters > NYSTRA_MAX_ITERS) return NYSTRA_EINVAL;
    if (!flags_ok(landmarks)) return NYSTRA_EINVAL;
    const bool patches = (landmarks & kPoolMask) == NYSTRA_LANDMARKS_PATCHES;
    const bool f16 = (landmarks & NYSTRA_FACTORS_16) != 0;  // derived factors rounded to 16 bits
    if (patches) {  // a square grid of square patches must tile the square window
        const int w = exact_sqrt(N), p = exact_sqrt(m);
        if (w < 0 || p < 0 || w % p != 0) return NYSTRA_EINVAL;
    }
    const long long units = (long long)n_windows * heads;
    if (units == 0) return NYSTRA_OK;
    if (!device_ok()) return NYSTRA_EDEVICE;
    const cudaStream_t s = (cudaStream_t)stream;
    // fp32 I/O on the tensor cores: 8x8 windows, m <= 16, at most the paper's 6
    // iterations (beyond them the fp16-split iteration's round-off, amplified
    // by ||G_A^n|| ||Z||, exceeds what fp32 I/O asks; the SIMT path iterates in fp32).
    // Square patches on the tensor cores: 16-bit I/O with m = 16.
    // 16-bit I/O on the tensor cores up to 12 iterations: their iteration
    // carries X = A Z beside Z (one product per step fewer), and over many
    // steps X drifts from A Z until the polynomial leaves its basin; the SIMT
    // path forms X = A Z afresh every step.
    const bool io16 = dtype == NYSTRA_BF16 || dtype == NYSTRA_F16;
    const bool tc16 = io16 && iters <= 12 && (patches ? m == 16 : (m == 8 || m == 16 || m == 32 || m == 64));
    const bool tc32 = !patches && dtype == NYSTRA_F32 && N == 64 && (m == 8 || m == 16) && iters <= 6;
    // A score bias on the tensor cores: the one-warp core, m <= 16.
    const bool biased = bias.L != nullptr;
    const bool tc = (tc16 || tc32) && d_h % 2 == 0 && d_h <= 32 && (!biased || m <= 16);
    const nystra::NystraBias* bp = biased ? &bias : nullptr;
    const int pool = patches ? 1 : 0;
    cudaError_t e;
    // NYSTRA_FACTORS_16 selects the kernels whose derived factors are 16-bit
    // (16-bit I/O on the tensor cores; the SIMT path is fp32 throughout).
    const bool s16 = f16 && io16;
    if (tc && N == 64)
        e = s16 ? nystra_host::launch_nystra_tc_n64_s16(q, k, v, out, units, d_h, m, iters, pool, dtype, s, bp)
                : nystra_host::launch_nystra_tc_n64(q, k, v, out, units, d_h, m, iters, pool, dtype, s, bp);
    else if (tc && N == 256)
        e = s16 ? nystra_host::launch_nystra_tc_n256_s16(q, k, v, out, units, d_h, m, iters, pool, dtype, s, bp)
                : nystra_host::launch_nystra_tc_n256(q, k, v, out, units, d_h, m, iters, pool, dtype, s, bp);
    else if (tc && N == 1024)
        e = s16 ? nystra_host::launch_nystra_tc_n1024_s16(q, k, v, out, units, d_h, m, iters, pool, dtype, s, bp)
                : nystra_host::launch_nystra_tc_n1024(q, k, v, out, units, d_h, m, iters, pool, dtype, s, bp);
    else
        e = nystra_host::launch_nystra_generic(q, k, v, out, units, N, d_h, m, iters, pool, dtype, s, bias);
    return e == cudaSuccess ? NYSTRA_OK : fail_cuda(e);
}

}  // namespace

extern "C" {

int nystra_attention_ex(const void* q, const void* k, const void* v, void* out, int n_windows, int heads,
                        int N, int d_h, int m, int iters, int landmarks, int dtype, void* stream) {
    return nystra_call(q, k, v, out, n_windows, heads, N, d_h, m, iters, landmarks, dtype, stream, {});
}

int nystra_pool_bias(const float* bias, int n_bias, int N, int m, int landmarks, float* bias_L, float* bias_U,
                     float* bias_A, void* stream) {
    if (n_bias < 0 || N < 1 || N > NYSTRA_MAX_N || m < 1 || m > N || m > NYSTRA_MAX_M || N % m != 0)
        return NYSTRA_EINVAL;
    if (landmarks != NYSTRA_LANDMARKS_SEGMENTS && landmarks != NYSTRA_LANDMARKS_PATCHES) return NYSTRA_EINVAL;
    if (landmarks == NYSTRA_LANDMARKS_PATCHES) {
        const int w = exact_sqrt(N), p = exact_sqrt(m);
        if (w < 0 || p < 0 || w % p != 0) return NYSTRA_EINVAL;
    }
    if (n_bias == 0) return NYSTRA_OK;
    if (!bias || !bias_L || !bias_U || !bias_A) return NYSTRA_EINVAL;
    if (!aligned16(bias) || !aligned16(bias_L) || !aligned16(bias_U) || !aligned16(bias_A)) return NYSTRA_EINVAL;
    const size_t in = (size_t)n_bias * N * N * 4, nm = (size_t)n_bias * N * m * 4, mm = (size_t)n_bias * m * m * 4;
    if (overlaps2(bias, in, bias_L, nm) || overlaps2(bias, in, bias_U, nm) || overlaps2(bias, in, bias_A, mm) ||
        overlaps2(bias_L, nm, bias_U, nm) || overlaps2(bias_L, nm, bias_A, mm) || overlaps2(bias_U, nm, bias_A, mm))
        return NYSTRA_EINVAL;
    if (!device_ok()) return NYSTRA_EDEVICE;
    const cudaError_t e = nystra_host::launch_pool_bias(bias, n_bias, N, m, landmarks, bias_L, bias_U, bias_A,
                                                        (cudaStream_t)stream);
    return e == cudaSuccess ? NYSTRA_OK : fail_cuda(e);
}

int nystra_attention_bias(const void* q, const void* k, const void* v, void* out, int n_windows, int heads,
                          int N, int d_h, int m, int iters, int landmarks, const float* bias_L, const float* bias_U,
                          const float* bias_A, int bias_windows, int dtype, void* stream) {
    if (n_windows > 0 && heads > 0) {
        if (bias_windows != 1 && bias_windows != n_windows) return NYSTRA_EINVAL;
        if (!bias_L || !bias_U || !bias_A) return NYSTRA_EINVAL;
        if (!aligned16(bias_L) || !aligned16(bias_U) || !aligned16(bias_A)) return NYSTRA_EINVAL;
        if (N >= 1 && m >= 1) {
            const size_t es = dtype == NYSTRA_F32 ? 4 : 2;
            const size_t ob = (size_t)n_windows * heads * N * d_h * es;
            const size_t nm = (size_t)bias_windows * heads * N * m * 4, mm = (size_t)bias_windows * heads * m * m * 4;
            if (overlaps2(out, ob, bias_L, nm) || overlaps2(out, ob, bias_U, nm) || overlaps2(out, ob, bias_A, mm))
                return NYSTRA_EINVAL;
        }
    }
    nystra::NystraBias b;
    b.L = bias_L;
    b.U = bias_U;
    b.A = bias_A;
    b.heads = heads > 0 ? heads : 1;
    b.per_window = bias_windows != 1 ? 1 : 0;
    return nystra_call(q, k, v, out, n_windows, heads, N, d_h, m, iters, landmarks, dtype, stream, b);
}

int nystra_attention(const void* q, const void* k, const void* v, void* out, int n_windows, int heads,
                     int N, int d_h, int m, int iters, int dtype, void* stream) {
    return nystra_attention_ex(q, k, v, out, n_windows, heads, N, d_h, m, iters, NYSTRA_LANDMARKS_SEGMENTS,
                               dtype, stream);
}

int nystra_attention_qkv(const void* x, const void* w_qkv, const float* b_qkv, void* out, int n_windows, int heads,
                         int N, int d_h, int m, int iters, int landmarks, const float* bias_L, const float* bias_U,
                         const float* bias_A, int bias_windows, int dtype, void* stream) {
    if (dtype != NYSTRA_BF16 && dtype != NYSTRA_F16) return NYSTRA_EDTYPE;  // 16-bit I/O only
    if (n_windows < 0 || heads < 0) return NYSTRA_EINVAL;
    if (N != 64 && N != 256 && N != 1024) return NYSTRA_EINVAL;
    if (d_h < 2 || d_h > 32 || d_h % 2 != 0) return NYSTRA_EINVAL;
    if (m != 8 && m != 16 && !(N == 1024 && m == 32)) return NYSTRA_EINVAL;
    if (iters < 0 || iters > 12) return NYSTRA_EINVAL;
    if (!flags_ok(landmarks)) return NYSTRA_EINVAL;
    const bool patches = (landmarks & kPoolMask) == NYSTRA_LANDMARKS_PATCHES;
    const bool s16 = (landmarks & NYSTRA_FACTORS_16) != 0;
    if (patches && m != 16) return NYSTRA_EINVAL;
    if ((long long)heads * d_h > NYSTRA_QKV_MAX_C) return NYSTRA_EINVAL;
    if (bias_L && m > 16) return NYSTRA_EINVAL;  // a score bias runs with the one-warp core
    if ((long long)n_windows * heads == 0) return NYSTRA_OK;
    const size_t C = (size_t)heads * d_h;
    const size_t xb = (size_t)n_windows * N * C * 2, wb = 3 * C * C * 2, ob = xb;
    if (!x || !w_qkv || !out) return NYSTRA_EINVAL;
    if (!aligned16(x) || !aligned16(w_qkv) || !aligned16(out) || (b_qkv && !aligned16(b_qkv))) return NYSTRA_EINVAL;
    if (overlaps2(out, ob, x, xb) || overlaps2(out, ob, w_qkv, wb) || (b_qkv && overlaps2(out, ob, b_qkv, 3 * C * 4)))
        return NYSTRA_EINVAL;
    nystra::NystraBias b;
    if (bias_L) {
        if (bias_windows != 1 && bias_windows != n_windows) return NYSTRA_EINVAL;
        if (!bias_U || !bias_A) return NYSTRA_EINVAL;
        if (!aligned16(bias_L) || !aligned16(bias_U) || !aligned16(bias_A)) return NYSTRA_EINVAL;
        const size_t nm = (size_t)bias_windows * heads * N * m * 4, mm = (size_t)bias_windows * heads * m * m * 4;
        if (overlaps2(out, ob, bias_L, nm) || overlaps2(out, ob, bias_U, nm) || overlaps2(out, ob, bias_A, mm))
            return NYSTRA_EINVAL;
        b.L = bias_L;
        b.U = bias_U;
        b.A = bias_A;
        b.heads = heads;
        b.per_window = bias_windows != 1 ? 1 : 0;
    }
    const nystra::NystraBias* bp = bias_L ? &b : nullptr;
    const int pool = patches ? 1 : 0;
    if (!device_ok()) return NYSTRA_EDEVICE;
    const cudaStream_t st = (cudaStream_t)stream;
    cudaError_t e;
    if (N == 64) {
        if (dtype == NYSTRA_BF16)
            e = s16 ? nystra_host::launch_nystra_qkv_bf16_s16(x, w_qkv, b_qkv, out, n_windows, heads, d_h, m, iters,
                                                              pool, st, bp)
                    : nystra_host::launch_nystra_qkv_bf16(x, w_qkv, b_qkv, out, n_windows, heads, d_h, m, iters,
                                                          pool, st, bp);
        else
            e = s16 ? nystra_host::launch_nystra_qkv_f16_s16(x, w_qkv, b_qkv, out, n_windows, heads, d_h, m, iters,
                                                             pool, st, bp)
                    : nystra_host::launch_nystra_qkv_f16(x, w_qkv, b_qkv, out, n_windows, heads, d_h, m, iters,
                                                         pool, st, bp);
    } else {  // 16x16 and 32x32 windows: the streaming kernel's structure
        if (dtype == NYSTRA_BF16)
            e = s16 ? nystra_host::launch_nystra_qkvs_bf16_s16(x, w_qkv, b_qkv, out, n_windows, heads, N, d_h, m,
                                                               iters, pool, st, bp)
                    : nystra_host::launch_nystra_qkvs_bf16(x, w_qkv, b_qkv, out, n_windows, heads, N, d_h, m, iters,
                                                           pool, st, bp);
        else
            e = s16 ? nystra_host::launch_nystra_qkvs_f16_s16(x, w_qkv, b_qkv, out, n_windows, heads, N, d_h, m,
                                                              iters, pool, st, bp)
                    : nystra_host::launch_nystra_qkvs_f16(x, w_qkv, b_qkv, out, n_windows, heads, N, d_h, m, iters,
                                                          pool, st, bp);
    }
    return e == cudaSuccess ? NYSTRA_OK : fail_cuda(e);
}

int nystra_project_qkv(const void* x, const void* w_qkv, const float* b_qkv, void* q, void* k, void* v,
                       int n_windows, int heads, int N, int d_h, int dtype, void* stream) {
    if (dtype != NYSTRA_BF16 && dtype != NYSTRA_F16) return NYSTRA_EDTYPE;  // 16-bit I/O only
    if (n_windows < 0 || heads < 0) return NYSTRA_EINVAL;
    if (N < 32 || N > NYSTRA_PROJ_MAX_N || N % 32 != 0) return NYSTRA_EINVAL;
    if (d_h < 2 || d_h > 32 || d_h % 2 != 0) return NYSTRA_EINVAL;
    if ((long long)heads * d_h > NYSTRA_PROJ_MAX_C) return NYSTRA_EINVAL;
    if ((long long)n_windows * heads == 0) return NYSTRA_OK;
    if (!x || !w_qkv || !q || !k || !v) return NYSTRA_EINVAL;
    if (!aligned16(x) || !aligned16(w_qkv) || !aligned16(q) || !aligned16(k) || !aligned16(v) ||
        (b_qkv && !aligned16(b_qkv)))
        return NYSTRA_EINVAL;
    const size_t C = (size_t)heads * d_h;
    const size_t xb = (size_t)n_windows * N * C * 2, wb = 3 * C * C * 2, bb = 3 * C * 4, ob = xb;
    const void* outs[3] = {q, k, v};
    for (int i = 0; i < 3; ++i) {
        if (overlaps2(outs[i], ob, x, xb) || overlaps2(outs[i], ob, w_qkv, wb) ||
            (b_qkv && overlaps2(outs[i], ob, b_qkv, bb)))
            return NYSTRA_EINVAL;
        for (int j = i + 1; j < 3; ++j)
            if (overlaps2(outs[i], ob, outs[j], ob)) return NYSTRA_EINVAL;
    }
    if (!device_ok()) return NYSTRA_EDEVICE;
    const cudaError_t e = nystra_host::launch_project_qkv(x, w_qkv, b_qkv, q, k, v, n_windows, heads, N, d_h, dtype,
                                                          (cudaStream_t)stream);
    return e == cudaSuccess ? NYSTRA_OK : fail_cuda(e);
}

int exact_window_attention(const void* q, const void* k, const void* v, void* out, int n_windows,
                           int heads, int N, int d_h, int dtype, void* stream) {
    int rc = check_common(q, k, v, out, n_windows, heads, N, d_h, dtype);
    if (rc != NYSTRA_OK) return rc;
    const long long units = (long long)n_windows * heads;
    if (units == 0) return NYSTRA_OK;
    if (!device_ok()) return NYSTRA_EDEVICE;
    cudaError_t e = nystra_host::exact_tc_supports(N, d_h, dtype)
                        ? nystra_host::launch_exact_tc(q, k, v, out, units, N, d_h, dtype, (cudaStream_t)stream)
                        : nystra_host::launch_exact_generic(q, k, v, out, units, N, d_h, dtype,
                                                            (cudaStream_t)stream);
    return e == cudaSuccess ? NYSTRA_OK : fail_cuda(e);
}

const char* nystra_strerror(int status) {
    switch (status) {
        case NYSTRA_OK: return "success";
        case NYSTRA_EINVAL: return "invalid argument (size, pointer, alignment or aliasing)";
        case NYSTRA_EDTYPE: return "unsupported dtype";
        case NYSTRA_ELAUNCH: return "CUDA launch or runtime error";
        case NYSTRA_ETIMEOUT: return "a bounded device-side wait timed out";
        case NYSTRA_EDEVICE: return "unsupported device (sm_103 required)";
        default: return "unknown status";
    }
}

int nystra_version(void) { return 100; }

int nystra_last_cuda_error(void) { return g_last_cuda_error; }

int nystra_status(void* stream) {
    cudaError_t e = cudaSuccess;
    const unsigned int words = nystra_host::take_fault_words((cudaStream_t)stream, &e);
    if (e != cudaSuccess) return fail_cuda(e);
    return (words & 1u) ? NYSTRA_ETIMEOUT : NYSTRA_OK;
}

int nystra_check(void* stream) { return nystra_status(stream); }

long long nystra_debug_stages_size(int N, int d_h, int m) {
    if (N != 64 || (m != 8 && m != 16) || d_h < 2 || d_h > 32 || d_h % 2 != 0) return NYSTRA_EINVAL;
    return nystra_host::debug_stages_size(N, d_h, m);
}

int nystra_debug_stages(const void* q, const void* k, const void* v, int n_windows, int heads, int N, int d_h,
                        int m, int iters, int landmarks, int dtype, long long unit, float* dump, void* stream) {
    if (dtype != NYSTRA_F32 && dtype != NYSTRA_BF16 && dtype != NYSTRA_F16) return NYSTRA_EDTYPE;
    if (nystra_debug_stages_size(N, d_h, m) < 0) return NYSTRA_EINVAL;
    if (iters < 0 || iters > 12 || (dtype == NYSTRA_F32 && iters > 6)) return NYSTRA_EINVAL;
    // square patches: the 16-bit I/O path with m = 16 (2x2 patches)
    if (landmarks != NYSTRA_LANDMARKS_SEGMENTS && landmarks != NYSTRA_LANDMARKS_PATCHES) return NYSTRA_EINVAL;
    if (landmarks == NYSTRA_LANDMARKS_PATCHES && (m != 16 || dtype == NYSTRA_F32)) return NYSTRA_EINVAL;
    if (n_windows < 0 || heads < 0 || unit < 0 || unit >= (long long)n_windows * heads) return NYSTRA_EINVAL;
    if (!q || !k || !v || !dump) return NYSTRA_EINVAL;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(dump)) return NYSTRA_EINVAL;
    if (!device_ok()) return NYSTRA_EDEVICE;
    const cudaError_t e = nystra_host::launch_debug_stages(q, k, v, unit, d_h, m, iters, landmarks, dtype, dump,
                                                           (cudaStream_t)stream);
    return e == cudaSuccess ? NYSTRA_OK : fail_cuda(e);
}

int nystra_debug_wait_timeout(unsigned long long limit_ns, void* stream) {
    if (limit_ns < 1000ull || limit_ns > 1000000000ull) return NYSTRA_EINVAL;
    if (!device_ok()) return NYSTRA_EDEVICE;
    const cudaError_t e = nystra_host::launch_debug_wait(limit_ns, (cudaStream_t)stream);
    return e == cudaSuccess ? NYSTRA_OK : fail_cuda(e);
}

}  // extern "C"

namespace nystra_host {
unsigned int take_fault_words(cudaStream_t stream, cudaError_t* err) {
    *err = cudaStreamSynchronize(stream);
    if (*err != cudaSuccess) return 0u;
    unsigned int w = 0;
    unsigned int (*const take[17])(cudaError_t*) = {
        take_fault_word_tc_n64,       take_fault_word_tc_n256,       take_fault_word_tc_n1024,
        take_fault_word_tc_n64_s16,   take_fault_word_tc_n256_s16,   take_fault_word_tc_n1024_s16,
        take_fault_word_exact_tc,     take_fault_word_debug,         take_fault_word_qkv_bf16,
        take_fault_word_qkv_f16,      take_fault_word_qkv_bf16_s16,  take_fault_word_qkv_f16_s16,
        take_fault_word_qkvs_bf16,    take_fault_word_qkvs_f16,      take_fault_word_qkvs_bf16_s16,
        take_fault_word_qkvs_f16_s16, take_fault_word_proj};
    for (auto f : take) {
        w |= f(err);
        if (*err != cudaSuccess) return w;
    }
    return w;
}
}  // namespace nystra_host
