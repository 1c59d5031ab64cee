// Inline-PTX helpers for sm_103a: bulk async copies with mbarriers (bounded
// waits), warp-level tensor-core MMA, tf32 conversion and ex2.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include "common.cuh"

namespace nystra {

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// ---------------------------------------------------------------- mbarrier
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}
// Plain arrival (release semantics at CTA scope: the arriving thread's prior
// shared-memory writes are visible to threads that observe the phase change).
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}
// Makes mbarrier initialisation visible to the async (bulk-copy) proxy.
__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
// Orders this thread's prior generic-proxy shared-memory accesses before
// subsequent async-proxy (bulk copy) accesses.
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Wait for phase `parity` of `bar` to complete, for at most `limit_ns`
// nanoseconds of wall time.  Returns false if the wait gave up.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (global_ns() - t0 > limit_ns) return false;
    }
    return true;
}
// 1-D bulk copy global -> shared, completing `bytes` of transaction on `bar`.
// dst and src 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}

// Named barrier over `nthreads` threads (a multiple of 32); id 0 is the one
// __syncthreads uses, so groups of warps take ids 1..15.
__device__ __forceinline__ void named_barrier(int id, int nthreads) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}
// Named barrier that also ORs `pred` over the participating threads: every
// thread gets the same result, so a decision taken on it (leave the loop) is
// the same in every warp.
__device__ __forceinline__ bool named_barrier_or(int id, int nthreads, bool pred) {
    uint32_t r;
    asm volatile(
        "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.or.pred q, %2, %3, p;\n selp.u32 %0, 1, 0, q;\n}\n"
        : "=r"(r)
        : "r"((uint32_t)pred), "r"(id), "r"(nthreads)
        : "memory");
    return r != 0u;
}

// L2 eviction-priority policies for bulk copies (fraction 1.0 of the bytes).
__device__ __forceinline__ uint64_t l2_evict_last() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint64_t l2_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}
// bulk_g2s with an L2 cache policy.
__device__ __forceinline__ void bulk_g2s_hint(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                              uint64_t policy) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], "
        "%4;" ::"r"(smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(policy)
        : "memory");
}

// 1-D bulk copy shared -> global (bulk-group completion).  Same alignment
// rules as bulk_g2s.  Generic-proxy writes to `src` must be ordered before it
// with fence_proxy_async_smem().
__device__ __forceinline__ void bulk_s2g(void* dst, const void* src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(smem_addr(src)),
                 "r"(bytes)
                 : "memory");
}
// bulk_s2g with an L2 cache policy.
__device__ __forceinline__ void bulk_s2g_hint(void* dst, const void* src, uint32_t bytes, uint64_t policy) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group.L2::cache_hint [%0], [%1], %2, %3;" ::"l"(dst),
                 "r"(smem_addr(src)), "r"(bytes), "l"(policy)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// Wait until every committed bulk store has finished reading its source.
__device__ __forceinline__ void bulk_wait_read_all() {
    asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// Wait until every committed bulk store has completed.
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// ------------------------------------------------------------------ math
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
// Transpose of an 8x8 matrix of 16-bit elements held one row pair per lane
// (lane 4r + c holds row r, columns 2c and 2c+1).
__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t x) {
    uint32_t y;
    asm("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
    return y;
}
// Byte permute: result byte k is byte sel.nibble[k] of the pair {b, a}
// (bytes 0-3 from a, 4-7 from b).
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}
// ldmatrix: four 8x8 b16 blocks; lanes 8i..8i+7 give the row addresses of
// block i (16-byte aligned); register i returns block i in fragment layout
// (lane (g, t) holds row g, columns 2t and 2t+1), or its transpose (_t).
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void* p) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(smem_addr(p))
                 : "memory");
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(smem_addr(p))
                 : "memory");
}
// Max over the warp of non-negative floats: their bit patterns order like
// unsigned integers, so one redux.sync does it.
__device__ __forceinline__ float warp_max_nonneg(float x) {
    return __uint_as_float(__reduce_max_sync(0xffffffffu, __float_as_uint(x)));
}
__device__ __forceinline__ float quad_max(float x) {
    x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, 1));
    return fmaxf(x, __shfl_xor_sync(0xffffffffu, x, 2));
}

// Split of an fp32 value into two tf32 parts: hi = x with its low 13 mantissa
// bits cleared (the tensor core ignores those bits of a .tf32 operand, so x
// itself is passed as hi) and lo = x - hi, exact in fp32 and again truncated
// to tf32 by the hardware.  hi + lo equals x to within 2^-20 |x|; the three
// products lo*hi, hi*lo and hi*hi give a product accurate to about 2^-19.
__device__ __forceinline__ uint32_t tf32_lo(float x) {
    return __float_as_uint(x - __uint_as_float(__float_as_uint(x) & 0xffffe000u));
}

// m16n8k8 tf32 MMA, fp32 accumulate: c += a (16x8, row) * b (8x8, col).
__device__ __forceinline__ void mma_tf32(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// fp16 two-term split of a pair of fp32 values: hi = rn(x), lo = rn(x - hi)
// (x - hi is exact in fp32).  hi + lo carries 22 significant bits for values
// in fp16's normal range; callers keep operands there by power-of-two scaling.
struct H2Pair {
    uint32_t hi, lo;
};
__device__ __forceinline__ H2Pair split_h2(float x0, float x1) {
    __half2 h = __floats2half2_rn(x0, x1);
    const float2 hf = __half22float2(h);
    __half2 l = __floats2half2_rn(x0 - hf.x, x1 - hf.y);
    return {*reinterpret_cast<uint32_t*>(&h), *reinterpret_cast<uint32_t*>(&l)};
}

// 16-bit MMAs (both operands of the same 16-bit type), fp32 accumulate.
template <typename T> struct Mma16;

template <> struct Mma16<__nv_bfloat16> {
    static __device__ __forceinline__ void k16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
        asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
            "{%0,%1,%2,%3};"
            : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
            : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
    }
    static __device__ __forceinline__ void k8(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t b0) {
        asm("mma.sync.aligned.m16n8k8.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5}, {%6}, {%0,%1,%2,%3};"
            : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
            : "r"(a0), "r"(a1), "r"(b0));
    }
    static __device__ __forceinline__ uint32_t pack(float lo, float hi) {
        __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
        return *reinterpret_cast<uint32_t*>(&h);
    }
    static __device__ __forceinline__ float2 unpack(uint32_t w) {
        return __bfloat1622float2(*reinterpret_cast<__nv_bfloat162*>(&w));
    }
    static constexpr uint32_t kOne = 0x3F80u;  // 1.0
    static constexpr bool kNarrowRange = false;
};

template <> struct Mma16<__half> {
    static __device__ __forceinline__ void k16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
        asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
            "{%0,%1,%2,%3};"
            : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
            : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
    }
    static __device__ __forceinline__ void k8(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t b0) {
        asm("mma.sync.aligned.m16n8k8.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5}, {%6}, {%0,%1,%2,%3};"
            : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
            : "r"(a0), "r"(a1), "r"(b0));
    }
    static __device__ __forceinline__ uint32_t pack(float lo, float hi) {
        __half2 h = __floats2half2_rn(lo, hi);
        return *reinterpret_cast<uint32_t*>(&h);
    }
    static __device__ __forceinline__ float2 unpack(uint32_t w) {
        return __half22float2(*reinterpret_cast<__half2*>(&w));
    }
    static constexpr uint32_t kOne = 0x3C00u;  // 1.0
    static constexpr bool kNarrowRange = true;  // values above 65504 overflow
};

// Operand policy for the products with token or d_h extents: how I/O-type
// values become m16n8k16 operands.  16-bit I/O: one register holds two
// elements.  fp32 I/O: each element is split into bf16 hi + lo (16
// significant bits each, fp32's range) and a product takes three MMAs
// (lo*hi + hi*lo + hi*hi), about 2^-16 relative error per product.
//
// Derived operands (DReg: the landmarks, G_L^n, G_U^n and Y, which the
// kernels compute in fp32) are always such hi + lo pairs in the MMA type, so
// that they keep 16 (bf16) or 22 (fp16) significant bits: rounding them to a
// single 16-bit value perturbs the Nystrom output by the method's own
// amplification of the landmark-block conditioning, which grows quickly as
// attention sharpens.  A product of a raw I/O operand with a derived one
// takes two MMAs (lo first), of two derived operands three.
struct RegPair {
    uint32_t hi, lo;
};
template <typename T>
struct Opnd {
    using Op = Mma16<T>;
    using Reg = uint32_t;
    using DReg = RegPair;
    static constexpr bool kNarrowRange = Op::kNarrowRange;
    static __device__ __forceinline__ Reg ld(const T* p) { return *reinterpret_cast<const uint32_t*>(p); }
    static __device__ __forceinline__ Reg pk(float a, float b) { return Op::pack(a, b); }
    static __device__ __forceinline__ Reg tr(Reg r) { return movmatrix_trans(r); }
    static __device__ __forceinline__ Reg zero() { return 0u; }
    static __device__ __forceinline__ Reg one() { return Op::kOne; }  // the pair (1, 0)
    static __device__ __forceinline__ void mma(float (&c)[4], const Reg (&a)[4], Reg b0, Reg b1) {
        Op::k16(c, a, b0, b1);
    }
    static __device__ __forceinline__ void mma8(float (&c)[4], Reg a0, Reg a1, Reg b0) { Op::k8(c, a0, a1, b0); }
    static __device__ __forceinline__ void st2(T* p, float a, float b) {
        *reinterpret_cast<uint32_t*>(p) = Op::pack(a, b);
    }
    // ---- derived operands ----
    static __device__ __forceinline__ DReg dpk(float a, float b) {
        const uint32_t h = Op::pack(a, b);
        const float2 hf = Op::unpack(h);
        return {h, Op::pack(a - hf.x, b - hf.y)};
    }
    static __device__ __forceinline__ DReg dzero() { return {0u, 0u}; }
    static __device__ __forceinline__ DReg dtr(DReg r) { return {movmatrix_trans(r.hi), movmatrix_trans(r.lo)}; }
    // raw x derived
    static __device__ __forceinline__ void mma(float (&c)[4], const Reg (&a)[4], DReg b0, DReg b1) {
        Op::k16(c, a, b0.lo, b1.lo);
        Op::k16(c, a, b0.hi, b1.hi);
    }
    // derived x raw
    static __device__ __forceinline__ void mma(float (&c)[4], const DReg (&a)[4], Reg b0, Reg b1) {
        const uint32_t ah[4] = {a[0].hi, a[1].hi, a[2].hi, a[3].hi};
        const uint32_t al[4] = {a[0].lo, a[1].lo, a[2].lo, a[3].lo};
        Op::k16(c, al, b0, b1);
        Op::k16(c, ah, b0, b1);
    }
    // derived x derived (the lo*lo term is below the pair's precision)
    static __device__ __forceinline__ void mma(float (&c)[4], const DReg (&a)[4], DReg b0, DReg b1) {
        const uint32_t ah[4] = {a[0].hi, a[1].hi, a[2].hi, a[3].hi};
        const uint32_t al[4] = {a[0].lo, a[1].lo, a[2].lo, a[3].lo};
        Op::k16(c, al, b0.hi, b1.hi);
        Op::k16(c, ah, b0.lo, b1.lo);
        Op::k16(c, ah, b0.hi, b1.hi);
    }
    static __device__ __forceinline__ void mma8(float (&c)[4], DReg a0, DReg a1, DReg b0) {
        Op::k8(c, a0.lo, a1.lo, b0.hi);
        Op::k8(c, a0.hi, a1.hi, b0.lo);
        Op::k8(c, a0.hi, a1.hi, b0.hi);
    }
};
template <>
struct Opnd<float> {
    using Op = Mma16<__nv_bfloat16>;
    using Reg = RegPair;
    using DReg = RegPair;
    static constexpr bool kNarrowRange = false;
    static __device__ __forceinline__ Reg pk(float a, float b) {
        const uint32_t h = Op::pack(a, b);
        const float2 hf = Op::unpack(h);
        return {h, Op::pack(a - hf.x, b - hf.y)};
    }
    static __device__ __forceinline__ Reg ld(const float* p) {
        const float2 v = *reinterpret_cast<const float2*>(p);
        return pk(v.x, v.y);
    }
    static __device__ __forceinline__ Reg tr(Reg r) { return {movmatrix_trans(r.hi), movmatrix_trans(r.lo)}; }
    static __device__ __forceinline__ Reg zero() { return {0u, 0u}; }
    static __device__ __forceinline__ Reg one() { return {Op::kOne, 0u}; }
    static __device__ __forceinline__ void mma(float (&c)[4], const Reg (&a)[4], Reg b0, Reg b1) {
        const uint32_t ah[4] = {a[0].hi, a[1].hi, a[2].hi, a[3].hi};
        const uint32_t al[4] = {a[0].lo, a[1].lo, a[2].lo, a[3].lo};
        Op::k16(c, al, b0.hi, b1.hi);
        Op::k16(c, ah, b0.lo, b1.lo);
        Op::k16(c, ah, b0.hi, b1.hi);
    }
    static __device__ __forceinline__ void mma8(float (&c)[4], Reg a0, Reg a1, Reg b0) {
        Op::k8(c, a0.lo, a1.lo, b0.hi);
        Op::k8(c, a0.hi, a1.hi, b0.lo);
        Op::k8(c, a0.hi, a1.hi, b0.hi);
    }
    static __device__ __forceinline__ void st2(float* p, float a, float b) {
        *reinterpret_cast<float2*>(p) = make_float2(a, b);
    }
    static __device__ __forceinline__ DReg dpk(float a, float b) { return pk(a, b); }
    static __device__ __forceinline__ DReg dzero() { return zero(); }
    static __device__ __forceinline__ DReg dtr(DReg r) { return tr(r); }
};

// Single16<T>: derived operands rounded to the 16-bit I/O type (one register,
// one MMA per product), as a caller selecting NYSTRA_FACTORS_16 asks for.
template <typename T>
struct Mma16<Single16<T>> : Mma16<T> {};
template <typename T>
struct Opnd<Single16<T>> {
    using Op = Mma16<T>;
    using Reg = uint32_t;
    using DReg = uint32_t;
    static constexpr bool kNarrowRange = Op::kNarrowRange;
    static __device__ __forceinline__ Reg ld(const Single16<T>* p) { return *reinterpret_cast<const uint32_t*>(p); }
    static __device__ __forceinline__ Reg pk(float a, float b) { return Op::pack(a, b); }
    static __device__ __forceinline__ Reg tr(Reg r) { return movmatrix_trans(r); }
    static __device__ __forceinline__ Reg zero() { return 0u; }
    static __device__ __forceinline__ Reg one() { return Op::kOne; }
    static __device__ __forceinline__ void mma(float (&c)[4], const Reg (&a)[4], Reg b0, Reg b1) {
        Op::k16(c, a, b0, b1);
    }
    static __device__ __forceinline__ void mma8(float (&c)[4], Reg a0, Reg a1, Reg b0) { Op::k8(c, a0, a1, b0); }
    static __device__ __forceinline__ void st2(Single16<T>* p, float a, float b) {
        *reinterpret_cast<uint32_t*>(p) = Op::pack(a, b);
    }
    static __device__ __forceinline__ DReg dpk(float a, float b) { return pk(a, b); }
    static __device__ __forceinline__ DReg dzero() { return 0u; }
    static __device__ __forceinline__ DReg dtr(DReg r) { return tr(r); }
};

// Storage of derived operands in shared memory.  16-bit I/O: the hi and lo
// parts of a row live in one row of the T-typed array, lo at element offset
// `lo` (LmS: landmark rows of 32 features, hi in columns 0..31 and lo in
// 32..63, row stride 72 = 36 words, so the 8 rows of a fragment load fall in
// distinct banks); fp32 I/O: one fp32 value, split when loaded.
template <typename T>
struct DSt {
    static __device__ __forceinline__ void put(T* p, int lo, float x) {
        const T h = from_f32<T>(x);
        p[0] = h;
        p[lo] = from_f32<T>(x - to_f32(h));
    }
    static __device__ __forceinline__ void zero(T* p, int lo) {
        p[0] = from_f32<T>(0.f);
        p[lo] = from_f32<T>(0.f);
    }
    // the pair register of elements p[0], p[1]
    static __device__ __forceinline__ RegPair ld(const T* p, int lo) {
        return {*reinterpret_cast<const uint32_t*>(p), *reinterpret_cast<const uint32_t*>(p + lo)};
    }
};
template <>
struct DSt<float> {
    static __device__ __forceinline__ void put(float* p, int, float x) { p[0] = x; }
    static __device__ __forceinline__ void zero(float* p, int) { p[0] = 0.f; }
    static __device__ __forceinline__ RegPair ld(const float* p, int) { return Opnd<float>::ld(p); }
};
template <typename T>
struct DSt<Single16<T>> {
    static __device__ __forceinline__ void put(Single16<T>* p, int, float x) { p[0] = from_f32<Single16<T>>(x); }
    static __device__ __forceinline__ void zero(Single16<T>* p, int) { p[0] = from_f32<Single16<T>>(0.f); }
    static __device__ __forceinline__ uint32_t ld(const Single16<T>* p, int) {
        return *reinterpret_cast<const uint32_t*>(p);
    }
};
// Landmark rows (Qbar, Kbar): row stride and lo offset in elements of T.
template <typename T>
struct LmS {
    static constexpr int LS = sizeof(T) == 2 ? 72 : 40;
    static constexpr int LO = sizeof(T) == 2 ? 32 : 0;
    static constexpr size_t bytes(int rows) { return (size_t)rows * LS * sizeof(T); }
};
template <typename T>
struct LmS<Single16<T>> {  // one 16-bit value per element, row stride 40 (20 words: conflict-free)
    static constexpr int LS = 40;
    static constexpr int LO = 0;
    static constexpr size_t bytes(int rows) { return (size_t)rows * LS * 2; }
};
// Y^T rows (features and the ones column) over MY = max(16, m) landmarks:
// 16-bit I/O hi in columns 0..MY-1, lo in MY..2MY-1, row stride 2 MY + 8
// (fragment loads conflict-free); fp32 I/O stride MY + 8.
template <typename T, int M>
struct YtS {
    static constexpr int MY = M < 16 ? 16 : M;
    static constexpr int YS = sizeof(T) == 2 ? 2 * MY + 8 : MY + 8;
    static constexpr int LO = sizeof(T) == 2 ? MY : 0;
    static constexpr size_t bytes(int ncol) { return (((size_t)ncol * YS * sizeof(T)) + 15) / 16 * 16; }
};
template <typename T, int M>
struct YtS<Single16<T>, M> {
    static constexpr int MY = M < 16 ? 16 : M;
    static constexpr int YS = MY + 8;
    static constexpr int LO = 0;
    static constexpr size_t bytes(int ncol) { return (((size_t)ncol * YS * 2) + 15) / 16 * 16; }
};

}  // namespace nystra
