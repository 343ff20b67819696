// common.cuh -- device primitives shared by the sm_103a kernels of the
// verifier-skipping SDD logits path: inline-PTX wrappers (packed f32x2
// arithmetic, MUFU ex2, mbarrier and 1D bulk-copy TMA), the Philox4x32-10
// generator, and the records the kernels exchange through the workspace.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/sdd.h"

namespace sdd {

// ---------------------------------------------------------------------------
// Constants
// ---------------------------------------------------------------------------
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr double kLn2d = 0.6931471805599453094;
constexpr double kLog2ed = 1.4426950408889634074;
// Every logit is clamped from below to -2^23 (exact in bf16 and fp32).  A
// masked (-inf) logit then contributes 2^(-huge) = 0 to every sum and 0 * y = 0
// to the entropy accumulator without ever forming inf - inf or 0 * inf, and
// every scaling reference (an integer in log2 units, see SoftState) stays an
// exactly representable fp32 integer.  Finite logits below -2^23 act as masked.
constexpr uint32_t kClampBits = 0xCB000000u;      // -2^23 as fp32 bits
constexpr uint32_t kClampPairBf16 = 0xCB00CB00u;  // the same value in both bf16 halves
constexpr uint32_t kNegInfPairBf16 = 0xFF80FF80u;

__device__ __forceinline__ float clamp_floor() { return __uint_as_float(kClampBits); }
// ceil(-2^23 * log2(e)) in fp32: the reference of an empty / fully masked state.
__device__ __forceinline__ float clamp_ref() { return ceilf(clamp_floor() * kLog2e); }

// Exact powers of two 2^k for integer-valued k <= 0 (0 below the normal range).
__device__ __forceinline__ float pow2f_int(float k) {
    return (k < -126.f) ? 0.f : __int_as_float((127 + static_cast<int>(k)) << 23);
}
__device__ __forceinline__ double pow2d_int(float k) {
    return (k < -1022.f) ? 0.0 : __longlong_as_double(static_cast<long long>(1023 + static_cast<int>(k)) << 52);
}

// ---------------------------------------------------------------------------
// Records exchanged through the workspace
// ---------------------------------------------------------------------------
// Partial softmax state of one warp's piece of one row.  Sums are taken
// relative to an integer reference r in log2 units:
//   s = sum 2^(z log2(e) - r),  t2 = sum 2^(z log2(e) - r) (z log2(e) - r).
struct __align__(32) Partial {
    float m;        // max of the clamped logits of the piece
    float r;        // integer reference (log2 units), >= m log2(e) up to rounding
    float t2;       // entropy accumulator (drafter rows)
    int32_t amax;   // lowest index attaining m (INT32_MAX if none)
    int32_t rank;   // saturated count of entries ranked before the drafted token
    int32_t pad;
    double s;
};

// Final statistics of one row, written by the warp that merges its partials.
struct __align__(32) RowRec {
    double lse;     // log sum_v exp(z(v)) in fp64
    float M;        // max of the clamped logits
    float g;        // clamped logit of the drafted token (NaN if the row has none)
    float q;        // exp(g - lse)
    float logq;     // g - lse
    int32_t argmax; // lowest index attaining M, -1 if the row is invalid
    int32_t rank;   // target rows: saturated rank of the drafted token
};

// ---------------------------------------------------------------------------
// Packed fp32 pair arithmetic (sm_100-family f32x2 instructions)
// ---------------------------------------------------------------------------
typedef unsigned long long f2_t;

__device__ __forceinline__ f2_t f2_pack(float lo, float hi) {
    f2_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void f2_unpack(f2_t v, float &lo, float &hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ f2_t f2_add(f2_t a, f2_t b) {
    f2_t d;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ f2_t f2_sub(f2_t a, f2_t b) {
    f2_t d;
    asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ f2_t f2_mul(f2_t a, f2_t b) {
    f2_t d;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ f2_t f2_fma(f2_t a, f2_t b, f2_t c) {
    f2_t d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}

// 2^x on the MUFU pipe (PTX ex2.approx.ftz.f32).
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// NaN-propagating maxima: a NaN logit must poison its row, never vanish.
__device__ __forceinline__ uint32_t bf16x2_max_nan(uint32_t a, uint32_t b) {
    uint32_t d;
    asm("max.NaN.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}
__device__ __forceinline__ float fmax_nan(float a, float b) {
    float d;
    asm("max.NaN.f32 %0, %1, %2;" : "=f"(d) : "f"(a), "f"(b));
    return d;
}
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// ---------------------------------------------------------------------------
// mbarrier + 1D bulk copy (TMA) helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait: gives up after max_iter polls (each poll may suspend the warp
// for a hardware-chosen interval) and returns false.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity, uint32_t max_iter) {
    for (uint32_t i = 0; i < max_iter; ++i)
        if (mbar_try_wait(bar, parity)) return true;
    return false;
}
// Global -> shared bulk copy of `bytes` (multiple of 16, both ends 16-byte
// aligned); completion is signalled as transaction bytes on `bar`.
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11) and the uniform mapping
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 k) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        if (r) {
            k.x += 0x9E3779B9u;
            k.y += 0xBB67AE85u;
        }
        const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
        const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
        c = make_uint4(hi1 ^ c.y ^ k.x, lo1, hi0 ^ c.w ^ k.y, lo0);
    }
    return c;
}

// u = ((word0 >> 8) | 1) * 2^-24 for key (seed) and counter
// (j, b, round_lo, purpose | round_hi << 8): exact in fp32, inside (0, 1).
__device__ __forceinline__ float philox_uniform(uint64_t seed, uint32_t j, uint32_t b, uint64_t round,
                                                uint32_t purpose) {
    const uint4 c = make_uint4(j, b, static_cast<uint32_t>(round),
                               (purpose & 0xFFu) | (static_cast<uint32_t>(round >> 32) << 8));
    const uint2 k = make_uint2(static_cast<uint32_t>(seed), static_cast<uint32_t>(seed >> 32));
    const uint4 o = philox4x32_10(c, k);
    return static_cast<float>((o.x >> 8) | 1u) * 5.9604644775390625e-08f;  // 2^-24
}

enum : uint32_t { kPurposeAccept = 0, kPurposeResid = 1, kPurposeBonus = 2 };

// ---------------------------------------------------------------------------
// Online-softmax state and its merge.  All rescaling is by exact powers of
// two (the references are integers), so merging never rounds the scale.
// ---------------------------------------------------------------------------
struct SoftState {
    float m, r, t2;
    double s;
    int32_t amax, rank;
};

__device__ __forceinline__ SoftState soft_identity() {
    SoftState z;
    z.m = clamp_floor();
    z.r = clamp_ref();
    z.t2 = 0.f;
    z.s = 0.0;
    z.amax = INT32_MAX;
    z.rank = 0;
    return z;
}

__device__ __forceinline__ SoftState soft_merge(SoftState a, SoftState b) {
    SoftState o;
    o.m = fmax_nan(a.m, b.m);
    o.r = fmaxf(a.r, b.r);
    const float ka = a.r - o.r, kb = b.r - o.r;  // integers <= 0
    // t2 relative to R: 2^k (t2 + k s)
    o.t2 = pow2f_int(ka) * (a.t2 + ka * static_cast<float>(a.s)) + pow2f_int(kb) * (b.t2 + kb * static_cast<float>(b.s));
    o.s = a.s * pow2d_int(ka) + b.s * pow2d_int(kb);
    if (b.m > a.m)
        o.amax = b.amax;
    else if (b.m < a.m)
        o.amax = a.amax;
    else
        o.amax = min(a.amax, b.amax);
    o.rank = a.rank + b.rank;
    return o;
}

__device__ __forceinline__ SoftState soft_warp_reduce(SoftState v) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        SoftState o;
        o.m = __shfl_xor_sync(0xFFFFFFFFu, v.m, off);
        o.r = __shfl_xor_sync(0xFFFFFFFFu, v.r, off);
        o.t2 = __shfl_xor_sync(0xFFFFFFFFu, v.t2, off);
        o.s = __shfl_xor_sync(0xFFFFFFFFu, v.s, off);
        o.amax = __shfl_xor_sync(0xFFFFFFFFu, v.amax, off);
        o.rank = __shfl_xor_sync(0xFFFFFFFFu, v.rank, off);
        // merge in a fixed order (lower lane first) so every lane agrees bitwise
        const bool lower = (threadIdx.x & off) == 0;
        v = lower ? soft_merge(v, o) : soft_merge(o, v);
    }
    return v;
}

__device__ __forceinline__ void status_or(int32_t *status, uint32_t bits) {
    if (status) atomicOr(reinterpret_cast<unsigned int *>(status), bits);
}

}  // namespace sdd
