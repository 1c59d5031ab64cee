/*
 * nystra.h -- C ABI of the GB300 (sm_103a) PnP-Nystra window-attention library.
 *
 * PnP-Nystra ("Plug-and-Play Linear Attention with Provable Guarantees for
 * Training-Free Image Restoration", arXiv 2506.08520) replaces the exact
 * softmax attention of one (window, head) pair,
 *     O = softmax(Q K^T / sqrt(d_h)) V                              (Eq. 1)
 * by the Nystrom approximation of the kernel matrix G = exp(Q K^T/sqrt(d_h)),
 *     G^ = G_L G_A^+ G_U,  O^ = (G^ V) ./ (G^ 1_N)     (Eq. 6-7, Algorithm 1)
 * evaluated in the row-max-stabilised form of Sec. 2.2 (Eq. 8).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  Layout   q, k, v and out are contiguous row-major tensors of shape
 *           [n_windows, heads, N, d_h]; one "unit" = one (window, head) pair,
 *           whose N x d_h block starts at element (w*heads + h) * N * d_h.
 *           (nystra_attention_qkv takes the tokens x [n_windows, N, heads*d_h]
 *           and the projection weights instead of q, k, v; see there.)
 *  Memory   every pointer is DEVICE memory owned by the caller, 16-byte
 *           aligned, and stays valid until the work on `stream` completes.
 *           q, k and v may alias one another; out must not overlap any input.
 *           The library allocates no device memory per call.
 *  dtype    element type of q, k, v and out (nystra_dtype).
 *  Precision products run on the tensor cores with fp32 accumulation: 16-bit
 *           inputs enter them as they are; the factors computed from them
 *           (landmarks, G_L^n, G_U^n, Y) are carried as hi + lo pairs of the
 *           I/O type (16 significant bits in bf16; NYSTRA_FACTORS_16 rounds
 *           them to a single 16-bit value instead); the pseudo-inverse
 *           iteration uses fp16 two-term splits (about 22 bits) of matrices
 *           scaled by powers of two so that none underflows; fp32 I/O splits
 *           every operand into bf16 hi + lo (three products each).  Shapes
 *           outside the tensor-core paths (odd d_h or d_h > 32, N not
 *           64/256/1024, m not 8/16/32/64, fp32 I/O with N != 64 or more than
 *           6 iterations, 16-bit I/O with more than 12) run in fp32 SIMT
 *           arithmetic.  The output is rounded to nearest-even.  Against a
 *           float64 evaluation the max relative Frobenius error per unit is
 *           <= 1e-4 (fp32 I/O) and <= 2e-2 (16-bit I/O) at the paper's
 *           iteration counts for logits q.k/sqrt(d_h) of standard deviation
 *           up to about 1.5.  Sharper attention makes G_A^n ill-conditioned
 *           and the method amplifies any rounding: a unit whose float64
 *           output moves by more than the bar when its landmarks are rounded
 *           once to 16 significant bits cannot be held to the bar by any
 *           evaluation at that precision.  Results stay finite wherever the
 *           float64 evaluation is.
 *  Stream   `stream` is a cudaStream_t (NULL = legacy default stream).  Calls
 *           are asynchronous: a return of NYSTRA_OK means the kernels were
 *           enqueued; results are ready when the stream is synchronised.
 *  Errors   invalid arguments are rejected before anything is launched and
 *           leave `out` untouched.  No call aborts, traps or prints.
 *  Device   the kernels are built for sm_103a (GB300) only.
 */
#ifndef NYSTRA_H
#define NYSTRA_H

#if defined(__GNUC__)
#define NYSTRA_API __attribute__((visibility("default")))
#else
#define NYSTRA_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Element type of q, k, v and out. */
typedef enum { NYSTRA_F32 = 0, NYSTRA_BF16 = 1, NYSTRA_F16 = 2 } nystra_dtype;

/* Landmark pooling (Algorithm 1 step 1; Sec. 2.2 pools landmarks by averaging
 * over non-overlapping windows, which reads two ways):
 *  SEGMENTS  m contiguous runs of N/m tokens in the window's token order;
 *  PATCHES   the window as a w x w grid (N = w^2, tokens row-major) cut into
 *            a p x p grid of square b x b patches (m = p^2, b = w/p), landmark
 *            j = patch (j / p, j % p). */
typedef enum { NYSTRA_LANDMARKS_SEGMENTS = 0, NYSTRA_LANDMARKS_PATCHES = 1 } nystra_landmarks;

/* Option flag, OR-ed into the `landmarks` argument of nystra_attention_ex,
 * nystra_attention_bias and nystra_attention_qkv (not nystra_pool_bias or
 * nystra_debug_stages, which reject it with NYSTRA_EINVAL):
 *  FACTORS_16  16-bit I/O on the tensor cores rounds the derived factors
 *              (landmarks, G_L^n, G_U^n, Y) to the I/O type instead of
 *              carrying each as a hi + lo pair of that type.  One MMA per
 *              product instead of two or three: faster (about 1.2x on 32x32
 *              windows), and within the 2e-2 bar only while attention stays
 *              soft (logits q.k/sqrt(d_h) of standard deviation up to about
 *              1.5); sharper attention makes G_A^n ill-conditioned and the
 *              method amplifies that rounding.  No effect on fp32 I/O or the
 *              SIMT path.  Not a step of the paper: a speed/accuracy choice of
 *              this implementation. */
#define NYSTRA_FACTORS_16 16

/* Status codes returned by every entry point (0 = success, negative = error). */
enum {
    NYSTRA_OK = 0,
    NYSTRA_EINVAL = -1,   /* a size, pointer, alignment or aliasing rule is violated  */
    NYSTRA_EDTYPE = -2,   /* dtype is not one of nystra_dtype                          */
    NYSTRA_ELAUNCH = -3,  /* a CUDA call failed; nystra_last_cuda_error() has the code */
    NYSTRA_ETIMEOUT = -4, /* a bounded device-side wait gave up (see nystra_status)    */
    NYSTRA_EDEVICE = -5   /* the current device is not an sm_103 GPU                   */
};

/* Size limits of the kernels (checked on every call). */
#define NYSTRA_MAX_N 1024     /* tokens per window                     */
#define NYSTRA_MAX_DH 64      /* head dimension d_h                    */
#define NYSTRA_MAX_M 64       /* landmarks per window                  */
#define NYSTRA_MAX_ITERS 100  /* pseudo-inverse iterations             */

/*
 * nystra_attention -- PnP-Nystra attention for every (window, head) unit.
 *
 * Per unit, following Algorithm 1 in the stabilised form of Sec. 2.2:
 *  1. landmarks Qbar, Kbar (m x d_h): means of m contiguous, non-overlapping
 *     segments of N/m tokens ("average pooling over non-overlapping windows");
 *  2-3. S_L = Q Kbar^T s, S_U = Qbar K^T s, S_A = Qbar Kbar^T s with
 *     s = 1/sqrt(d_h); row maxima m_L (over m landmarks) and m_U (over all N
 *     keys); G_L^n = exp(S_L - m_L), G_U^n = exp(S_U - m_U),
 *     G_A^n = exp(S_A - m_U);
 *  4. Z ~ (G_A^n)^+ by `iters` steps of the third-order iteration of
 *     Razavi et al. (2014): Z_0 = A^T/(||A||_1 ||A||_inf),
 *     Z <- Z (13I - AZ(15I - AZ(7I - AZ)))/4 with A = G_A^n;
 *  5-7. O = (G_L^n Z G_U^n V) ./ (G_L^n Z G_U^n 1_N), evaluated as
 *     G_L^n (Z (G_U^n [V | 1_N])) (an exact re-association of steps 5-6).
 *
 * Arguments
 *  q, k, v   [n_windows, heads, N, d_h] inputs (device, caller-owned).
 *  out       [n_windows, heads, N, d_h] output (device, caller-owned).
 *  n_windows, heads   >= 0; n_windows*heads == 0 is a no-op returning OK.
 *  N         tokens per window, 1..NYSTRA_MAX_N.
 *  d_h       head dimension, 1..NYSTRA_MAX_DH.
 *  m         landmarks, 1..min(N, NYSTRA_MAX_M), and m must divide N.
 *  iters     pseudo-inverse iterations, 0..NYSTRA_MAX_ITERS (paper: 4-6).
 *  dtype     nystra_dtype of q, k, v and out.
 *  stream    cudaStream_t to enqueue on.
 * Returns NYSTRA_OK, NYSTRA_EINVAL, NYSTRA_EDTYPE, NYSTRA_ELAUNCH or
 * NYSTRA_EDEVICE.  The denominator is not guarded (Algorithm 1 step 7
 * divides as written); a zero denominator yields inf/nan in that row.
 */
NYSTRA_API int nystra_attention(const void* q, const void* k, const void* v, void* out,
                     int n_windows, int heads, int N, int d_h, int m, int iters,
                     int dtype, void* stream);

/*
 * nystra_attention_ex -- nystra_attention with a choice of landmark pooling.
 * `landmarks` is a nystra_landmarks value, optionally OR-ed with
 * NYSTRA_FACTORS_16; NYSTRA_LANDMARKS_PATCHES needs N and m perfect squares
 * with sqrt(m) dividing sqrt(N) (else NYSTRA_EINVAL).
 * nystra_attention(...) is nystra_attention_ex(..., NYSTRA_LANDMARKS_SEGMENTS,
 * ...).  Square patches run on the tensor cores for 16-bit I/O with m = 16
 * and N in {64, 256, 1024} (even d_h <= 32), on the fp32 SIMT path otherwise.
 * Other arguments, layout and return codes as nystra_attention.
 */
NYSTRA_API int nystra_attention_ex(const void* q, const void* k, const void* v, void* out,
                                   int n_windows, int heads, int N, int d_h, int m, int iters,
                                   int landmarks, int dtype, void* stream);

/*
 * Additive score bias (window attention's relative-position bias and masks).
 * Eq. (1) has none; a window-attention layer adds B (N x N per head, or per
 * window and head) to Q K^T / sqrt(d_h) before the softmax.  Here a landmark
 * stands for the mean of its tokens, so it also carries the mean of their
 * biases: the blocks of Sec. 2.2 become
 *   S_L[i][j] += mean_{t in j} B[i][t],   S_U[j][t] += mean_{s in j} B[s][t],
 *   S_A[i][j] += mean_{s in i, t in j} B[s][t]
 * (with m = N and a converged inverse this is exact biased attention).  Use
 * finite mask values (e.g. -100): an infinite one poisons every landmark whose
 * tokens it touches.
 *
 * nystra_pool_bias -- the three landmark blocks of n_bias biases:
 *   bias    [n_bias, N, N] fp32 (device, caller-owned);
 *   bias_L  [n_bias, N, m], bias_U [n_bias, m, N], bias_A [n_bias, m, m] fp32
 *           outputs (device, caller-owned, no overlap with each other or bias).
 * `landmarks` as for nystra_attention_ex.  All pointers 16-byte aligned.  Meant
 * to run once per model constant.  Returns NYSTRA_OK, NYSTRA_EINVAL (shape,
 * pointer, alignment, overlap, or a `landmarks` value with option flags),
 * NYSTRA_ELAUNCH or NYSTRA_EDEVICE.
 */
NYSTRA_API int nystra_pool_bias(const float* bias, int n_bias, int N, int m, int landmarks, float* bias_L,
                                float* bias_U, float* bias_A, void* stream);

/*
 * nystra_attention_bias -- nystra_attention_ex with a pooled score bias.
 * bias_L/U/A as written by nystra_pool_bias for bias_windows * heads slices:
 * bias_windows = 1 (one bias per head, shared by every window: the
 * relative-position bias) or n_windows (per window and head: masks of
 * shifted windows).  Unit (w, h) uses slice h, or w * heads + h.  The blocks
 * must not overlap out.  m in {8, 16} runs on the tensor-core kernels of
 * nystra_attention (with the bias added to the scaled scores before each row
 * maximum), other shapes on the fp32 SIMT path.  Other arguments and return
 * codes as nystra_attention_ex.
 */
NYSTRA_API int nystra_attention_bias(const void* q, const void* k, const void* v, void* out, int n_windows,
                                     int heads, int N, int d_h, int m, int iters, int landmarks,
                                     const float* bias_L, const float* bias_U, const float* bias_A,
                                     int bias_windows, int dtype, void* stream);

/*
 * nystra_attention_qkv -- the projections of Eq. (1) fused with PnP-Nystra:
 * per window, Q = X W_Q, K = X W_K, V = X W_V (+ an optional projection
 * bias, which the restoration models' layers add and Eq. (1) omits), split
 * into heads of d_h features, then nystra_attention_ex on every (window,
 * head) unit.  Q, K and V stay on chip: the call reads the tokens and the
 * weights instead of Q, K and V.
 *
 * Arguments
 *  x       [n_windows, N, C] tokens, C = heads * d_h, each window's tokens in
 *          the order nystra_attention_ex pools them (device, caller-owned).
 *  w_qkv   [3C, C]: row o holds the weights of output feature o, rows 0..C-1
 *          for Q, C..2C-1 for K, 2C..3C-1 for V (the transposes of W_Q, W_K,
 *          W_V stacked: the layout of a linear layer's weight); head h owns
 *          features h*d_h .. h*d_h + d_h - 1 of each.  Same dtype as x.
 *  b_qkv   [3C] fp32 projection bias, or NULL for none.
 *  out     [n_windows, heads, N, d_h] output, as nystra_attention writes it.
 *  bias_L, bias_U, bias_A, bias_windows   an optional pooled score bias as for
 *          nystra_attention_bias; bias_L == NULL for none.
 *  Other arguments as nystra_attention_ex.
 * The projected Q, K, V are rounded to the I/O type before the attention, as
 * an unfused projection would store them.  Supported: 16-bit I/O (fp32 returns
 * NYSTRA_EDTYPE), N in {64, 256, 1024} (8x8, 16x16, 32x32 windows), m in
 * {8, 16} (also 32 with N = 1024, without a score bias; square patches:
 * m = 16), even d_h <= 32, C <= NYSTRA_QKV_MAX_C, iters <= 12; anything else
 * returns NYSTRA_EINVAL, as do null (other than b_qkv and the bias) or not
 * 16-byte aligned pointers and an out that overlaps an input.  `landmarks`
 * may carry NYSTRA_FACTORS_16.  Returns NYSTRA_OK, NYSTRA_EINVAL,
 * NYSTRA_EDTYPE, NYSTRA_ELAUNCH or NYSTRA_EDEVICE.
 */
#define NYSTRA_QKV_MAX_C 352
NYSTRA_API int nystra_attention_qkv(const void* x, const void* w_qkv, const float* b_qkv, void* out,
                                    int n_windows, int heads, int N, int d_h, int m, int iters, int landmarks,
                                    const float* bias_L, const float* bias_U, const float* bias_A,
                                    int bias_windows, int dtype, void* stream);

/*
 * nystra_project_qkv -- the projections of Eq. (1) on their own: per window,
 * Q = X W_Q, K = X W_K, V = X W_V (+ an optional projection bias), split into
 * heads of d_h features and written in the [n_windows, heads, N, d_h] layout
 * nystra_attention and exact_window_attention read.  One GEMM of the
 * n_windows * N token rows against the stacked weights on the fifth-
 * generation tensor cores (tcgen05: operands in shared memory, fp32
 * accumulators in tensor memory), the head split done as the accumulators
 * are stored.  Followed by nystra_attention_ex it computes what
 * nystra_attention_qkv computes, with Q, K and V passing through HBM (the
 * caller provides their memory).  On a GB300 that two-pass form is the
 * faster one for wide tokens over many windows (C = 180 over a 1280x720
 * map: 1.8x with 8x8 windows to 2.9x with 32x32), the fused entry point for
 * narrow tokens or few windows (C = 32, or 64 windows of C = 256).
 *
 * Arguments
 *  x, w_qkv, b_qkv   as nystra_attention_qkv (tokens [n_windows, N, C],
 *          C = heads * d_h; weights [3C, C]; fp32 bias [3C] or NULL).
 *  q, k, v [n_windows, heads, N, d_h] outputs (device, caller-owned), each
 *          element the fp32-accumulated dot product plus bias, rounded to
 *          the I/O type (nearest-even).
 * Supported: 16-bit I/O (fp32 returns NYSTRA_EDTYPE), N a multiple of 32 in
 * [32, NYSTRA_PROJ_MAX_N], even d_h <= 32, C <= NYSTRA_PROJ_MAX_C; anything
 * else returns NYSTRA_EINVAL, as do null (other than b_qkv) or not 16-byte
 * aligned pointers, and outputs that overlap an input or one another.  The
 * library allocates nothing; asynchronous on `stream`.  Returns NYSTRA_OK,
 * NYSTRA_EINVAL, NYSTRA_EDTYPE, NYSTRA_ELAUNCH or NYSTRA_EDEVICE.
 */
#define NYSTRA_PROJ_MAX_C 384
#define NYSTRA_PROJ_MAX_N 65536
NYSTRA_API int nystra_project_qkv(const void* x, const void* w_qkv, const float* b_qkv, void* q, void* k, void* v,
                                  int n_windows, int heads, int N, int d_h, int dtype, void* stream);

/*
 * exact_window_attention -- exact softmax attention per unit, Eq. (1):
 * O = softmax(Q K^T / sqrt(d_h)) V with row-max-shifted exponentials
 * (Eq. 2).  This is the computation PnP-Nystra replaces; it serves as the
 * in-library comparator.  Arguments and return codes as nystra_attention
 * (no m, no iters).
 */
NYSTRA_API int exact_window_attention(const void* q, const void* k, const void* v, void* out,
                           int n_windows, int heads, int N, int d_h,
                           int dtype, void* stream);

/* Human-readable text for a status code (static storage, never NULL). */
NYSTRA_API const char* nystra_strerror(int status);

/* Library version as major*10000 + minor*100 + patch. */
NYSTRA_API int nystra_version(void);

/* cudaError_t of the most recent NYSTRA_ELAUNCH on the calling thread (0 if none). */
NYSTRA_API int nystra_last_cuda_error(void);

/*
 * nystra_status -- synchronise `stream` and report device-side faults
 * recorded by kernels on the current device since the previous call:
 * NYSTRA_ETIMEOUT if a bounded wait gave up, else NYSTRA_OK (or
 * NYSTRA_ELAUNCH if the synchronisation itself failed).  Clears the record.
 * The record is per device, not per stream: a timeout in a kernel still
 * running on another stream is reported by whichever call reads the record
 * after it is set (synchronise those streams first to attribute it).
 */
NYSTRA_API int nystra_status(void* stream);

/*
 * nystra_check -- the same as nystra_status (the name the method's
 * integration notes use for the synchronising status helper).
 */
NYSTRA_API int nystra_check(void* stream);

/*
 * nystra_debug_wait_timeout -- test-only (the paper has no counterpart):
 * launches one warp on `stream` that waits, through the same bounded
 * mbarrier wait the kernels use, on an mbarrier nothing ever arrives on.
 * After limit_ns nanoseconds of %globaltimer it gives up and records the
 * timeout exactly as a kernel would, so the next nystra_status(stream)
 * returns NYSTRA_ETIMEOUT and the context stays usable.  limit_ns must lie in
 * [1000, 1000000000] (1 us to 1 s), else NYSTRA_EINVAL; NYSTRA_EDEVICE without
 * an sm_103 device; nothing is allocated.
 */
NYSTRA_API int nystra_debug_wait_timeout(unsigned long long limit_ns, void* stream);

/*
 * nystra_debug_stages -- test-only (the paper has no counterpart): every
 * intermediate of Algorithm 1 for ONE unit, as the tensor-core path for 8x8
 * windows computes it.  One warp runs, for unit `unit` (window*heads + head)
 * of the [n_windows, heads, N, d_h] tensors q, k, v, the same device functions
 * the N = 64 kernel runs, and writes fp32 values, row-major, to `dump`
 * (device memory, caller-owned, 16-byte aligned, nystra_debug_stages_size()
 * floats), regions in this order:
 *   Qbar  m x d_h      landmarks (step 1), as the kernel carries them (hi + lo)
 *   Kbar  m x d_h
 *   G_L^n N x m        exp(S_L - m_L) (steps 2-3), as carried (hi + lo)
 *   m_U   m            row maxima of S_U over all N keys (natural-log domain)
 *   W     m x (d_h+1)  G_U^n [V | 1_N] (step 5); column d_h is G_U^n 1_N
 *   G_A^n m x m        exp(S_A - m_U) (step 3)
 *   Z     m x m        the pseudo-inverse after `iters` steps (step 4)
 *   Y     m x (d_h+1)  Z W (the re-associated step 6)
 *   O     N x d_h      the output (step 7), as rounded to the I/O type
 * `landmarks` is a nystra_landmarks value (square patches: 16-bit I/O, m = 16).
 * Supported: N = 64, m in {8, 16}, even d_h <= 32 (the shapes nystra_attention
 * runs on this path: iters <= 12, and <= 6 for fp32 I/O); anything else returns
 * NYSTRA_EINVAL, as do unit outside [0, n_windows*heads), null or misaligned
 * pointers (and a `landmarks` value with option flags).  Asynchronous on
 * `stream`; allocates nothing.  Returns NYSTRA_OK, NYSTRA_EINVAL,
 * NYSTRA_EDTYPE, NYSTRA_ELAUNCH or NYSTRA_EDEVICE.
 */
NYSTRA_API int nystra_debug_stages(const void* q, const void* k, const void* v, int n_windows, int heads,
                                   int N, int d_h, int m, int iters, int landmarks, int dtype, long long unit,
                                   float* dump, void* stream);

/* Floats nystra_debug_stages writes for (N, d_h, m):
 * 2 m d_h + N m + m + 2 m (d_h+1) + 2 m^2 + N d_h; NYSTRA_EINVAL (negative)
 * for a shape it does not support.  Touches no device. */
NYSTRA_API long long nystra_debug_stages_size(int N, int d_h, int m);

#ifdef __cplusplus
}
#endif
#endif /* NYSTRA_H */
