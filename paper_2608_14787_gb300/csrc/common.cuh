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
//   s = sum 2^(z log2(e) - r)  (kept as an unevaluated fp32 pair sh + sl),
//   t2 = sum 2^(z log2(e) - r) (z - m) log2(e), against the piece's maximum m
//   (each term <= 0; the maximum's own term is 0, so on a peaked row t2 stays
//   small and the entropy ln S' - ln 2 t2 / S involves no cancellation).
struct __align__(32) Partial {
    float m;        // max of the clamped logits of the piece
    float r;        // integer reference (log2 units), >= m log2(e) up to rounding
    float t2;       // entropy accumulator (drafter rows)
    float sh, sl;   // exp-sum as a double-float
    int32_t amax;   // lowest index attaining m (INT32_MAX if none)
    int32_t rank;   // saturated count of entries ranked before the drafted token; -1: token out of range
    float g;        // clamped logit of the row's drafted token (NaN if the row has none)
};

// ---------------------------------------------------------------------------
// Double-float arithmetic: a value is an unevaluated pair hi + lo of fp32
// numbers with |lo| <= ulp(hi) / 2.  Built on the error-free transformations
// TwoSum (Knuth) and FastTwoSum (Dekker) and on the FMA residual of a product;
// used wherever the path needs more than fp32 precision, because fp64
// instructions issue at a small fraction of the fp32 rate on this part.
// ---------------------------------------------------------------------------
constexpr float kLn2Hi = 0.693147182464599609375f;    // fp32 nearest ln 2
constexpr float kLn2Lo = -1.9046542121259336e-09f;    // ln 2 - kLn2Hi

__device__ __forceinline__ void two_sum(float a, float b, float &s, float &err) {
    s = a + b;
    const float bb = s - a;
    err = (a - (s - bb)) + (b - bb);
}
// Requires |a| >= |b| (or a == 0).
__device__ __forceinline__ void fast_two_sum(float a, float b, float &s, float &err) {
    s = a + b;
    err = b - (s - a);
}

struct df {
    float hi, lo;
};

// A non-finite hi carries lo = 0, so infinities and NaN propagate through hi
// alone and never form inf - inf in lo.
__device__ __forceinline__ df df_make(float h, float l) {
    df r;
    if (!isfinite(h)) return df{h, 0.f};
    two_sum(h, l, r.hi, r.lo);   // no ordering precondition: the lo part may exceed a cancelled hi
    if (!isfinite(r.hi)) r.lo = 0.f;
    return r;
}
__device__ __forceinline__ df df_add(df a, df b) {
    float s, e;
    two_sum(a.hi, b.hi, s, e);
    if (!isfinite(s)) return df{s, 0.f};
    return df_make(s, e + (a.lo + b.lo));
}
__device__ __forceinline__ df df_sub(df a, df b) { return df_add(a, df{-b.hi, -b.lo}); }
// a - b for two fp32 numbers, exactly.
__device__ __forceinline__ df df_diff(float a, float b) {
    df r;
    two_sum(a, -b, r.hi, r.lo);
    if (!isfinite(r.hi)) r.lo = 0.f;
    return r;
}
// a * b for an fp32 b (relative error ~2^-46).
__device__ __forceinline__ df df_mul_f(df a, float b) {
    const float p = a.hi * b;
    if (!isfinite(p)) return df{p, 0.f};
    const float e = fmaf(a.hi, b, -p);
    return df_make(p, fmaf(a.lo, b, e));
}
// a >= b; infinities compare by their hi parts.
__device__ __forceinline__ bool df_ge(df a, df b) {
    if (!isfinite(a.hi) || !isfinite(b.hi)) return a.hi >= b.hi;
    return a.hi > b.hi || (a.hi == b.hi && a.lo >= b.lo);
}
// Host-side split of a double into a double-float (exact to ~2^-48 relative).
__host__ __device__ inline df df_from_double(double x) {
    df r;
    r.hi = static_cast<float>(x);
    r.lo = 0.f;
    if (r.hi - r.hi == 0.f) r.lo = static_cast<float>(x - static_cast<double>(r.hi));   // hi finite
    return r;
}

// Natural logarithm of a positive double-float x = xh + xl with xh normal and
// 2^-126 < x < 2^126, to about 1e-9 absolute, in fp32 arithmetic only:
// x = 2^k m (1 + xl / xh) with m in [sqrt(1/2), sqrt(2)), and
// ln x = k ln 2 + 2 atanh(u),  u = (m - 1 + l) / (m + 1 + l),  l = xl 2^-k,
// where |u| <= 0.1716 and the series 2 (u + u^3/3 + ... + u^13/13) is exact to
// 5e-13; its leading term 2u is carried as a double-float (the quotient
// corrected by its FMA residual), the rest in fp32.
__device__ __forceinline__ df ln_df(float xh, float xl) {
    const uint32_t bits = __float_as_uint(xh);
    int k = static_cast<int>((bits >> 23) & 0xFFu) - 127;
    float m = __uint_as_float((bits & 0x007FFFFFu) | 0x3F800000u);   // [1, 2)
    if (m > 1.41421354f) {
        m *= 0.5f;
        k += 1;
    }
    const float l = xl * __uint_as_float(static_cast<uint32_t>(127 - k) << 23);   // xl 2^-k
    float fh, fl, dh, dl;
    two_sum(m - 1.f, l, fh, fl);            // m - 1 is exact
    two_sum(m, 1.f, dh, dl);
    dl += l;
    const float uh = __fdividef(fh, dh);
    const float res = fmaf(-uh, dh, fh) + (fl - uh * dl);
    const float ul = __fdividef(res, dh);
    const float v = uh * uh;
    float poly = 1.f / 13.f;
    poly = fmaf(poly, v, 1.f / 11.f);
    poly = fmaf(poly, v, 1.f / 9.f);
    poly = fmaf(poly, v, 1.f / 7.f);
    poly = fmaf(poly, v, 1.f / 5.f);
    poly = fmaf(poly, v, 1.f / 3.f);
    const float tail = 2.f * uh * v * poly;
    const float kf = static_cast<float>(k);
    const float a = kf * kLn2Hi;
    const float ae = fmaf(kf, kLn2Hi, -a);
    float s, e;
    two_sum(a, 2.f * uh, s, e);
    return df_make(s, e + ((ae + kf * kLn2Lo) + (2.f * ul + tail)));
}

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

__device__ __forceinline__ float qnan() { return __int_as_float(0x7FC00000); }

// One logit of a row (bf16 widened exactly to fp32).
template <int DT>
__device__ __forceinline__ float logit_at(const char *rowp, int v) {
    if (DT == SDD_BF16) {
        const uint16_t h = __ldg(reinterpret_cast<const unsigned short *>(rowp) + v);
        return __uint_as_float(static_cast<uint32_t>(h) << 16);
    } else {
        return __ldg(reinterpret_cast<const float *>(rowp) + v);
    }
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
// Per-half comparisons of bf16 pairs: each 16-bit half of the result is
// all ones where the comparison holds, zero elsewhere.
__device__ __forceinline__ uint32_t bf16x2_gt(uint32_t a, uint32_t b) {
    uint32_t d;
    asm("set.gt.u32.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}
__device__ __forceinline__ uint32_t bf16x2_eq(uint32_t a, uint32_t b) {
    uint32_t d;
    asm("set.eq.u32.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
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
// An L2 policy that evicts the lines it is attached to first: for data read
// exactly once (the logits stream), so that it does not push out what later
// kernels reuse (their code, the partials, the next round's small arrays).
__device__ __forceinline__ uint64_t l2_evict_first_policy() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

// Global -> shared bulk copy of `bytes` (multiple of 16, both ends 16-byte
// aligned) under L2 policy `pol`; completion is signalled as transaction
// bytes on `bar`.
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar, uint64_t pol) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
            smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(pol)
        : "memory");
}

// 16-byte global -> shared copy through L2 (cp.async.cg), completed by
// cp_async_wait_all().
__device__ __forceinline__ void cp_async16(void *smem_dst, const void *gsrc) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(smem_dst)), "l"(gsrc) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }

// Atomic add with acquire-release semantics at GPU scope (returns the old value).
__device__ __forceinline__ uint32_t atom_add_acq_rel_gpu(uint32_t *addr, uint32_t v) {
    uint32_t old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(addr), "r"(v) : "memory");
    return old;
}

// ---------------------------------------------------------------------------
// Programmatic dependent launch: a grid launched with the programmatic
// stream-serialization attribute may be scheduled before the grid ahead of it
// in the stream completes; griddep_wait() blocks until that grid has completed
// and its memory operations are visible (a no-op for an ordinary launch).
// ---------------------------------------------------------------------------
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
// Lets the grid launched behind this one be scheduled once every CTA of this
// grid has called it or exited (its griddep_wait still waits for completion).
__device__ __forceinline__ void griddep_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Launch `kernel` behind the previous work of `stream` as a programmatic
// dependent grid (host side).
template <class Params>
inline cudaError_t launch_dependent(void (*kernel)(Params), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                                    const Params &p) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, p);
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
// two (the references are integers), so merging never rounds the scale; the
// exp-sum stays a double-float throughout.
// ---------------------------------------------------------------------------
// The five largest (clamped) logits of a drafter row piece, descending, with
// multiplicity (-inf where the piece holds fewer): the extended features.
struct FeatPartial {
    float top[5];
    float pad[3];
};

struct SoftState {
    float m, r, t2;
    float sh, sl;
    int32_t amax, rank;
};

__device__ __forceinline__ SoftState soft_identity() {
    SoftState z;
    z.m = clamp_floor();
    z.r = clamp_ref();
    z.t2 = 0.f;
    z.sh = 0.f;
    z.sl = 0.f;
    z.amax = INT32_MAX;
    z.rank = 0;
    return z;
}

__device__ __forceinline__ SoftState soft_merge(const SoftState &a, const SoftState &b) {
    SoftState o;
    o.m = fmax_nan(a.m, b.m);
    o.r = fmaxf(a.r, b.r);
    const float ka = a.r - o.r, kb = b.r - o.r;  // integers <= 0
    const float pa = pow2f_int(ka), pb = pow2f_int(kb);
    // t2 against the merged maximum, relative to the new reference:
    // 2^k (t2 + (m - m') log2(e) s)
    o.t2 = pa * fmaf((a.m - o.m) * kLog2e, a.sh + a.sl, a.t2) + pb * fmaf((b.m - o.m) * kLog2e, b.sh + b.sl, b.t2);
    float h, e;
    two_sum(a.sh * pa, b.sh * pb, h, e);
    fast_two_sum(h, fmaf(a.sl, pa, fmaf(b.sl, pb, e)), o.sh, o.sl);
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
        o.sh = __shfl_xor_sync(0xFFFFFFFFu, v.sh, off);
        o.sl = __shfl_xor_sync(0xFFFFFFFFu, v.sl, off);
        o.amax = __shfl_xor_sync(0xFFFFFFFFu, v.amax, off);
        o.rank = __shfl_xor_sync(0xFFFFFFFFu, v.rank, off);
        // merge in a fixed order (lower lane first) so every lane agrees bitwise
        const bool lower = (threadIdx.x & off) == 0;
        v = lower ? soft_merge(v, o) : soft_merge(o, v);
    }
    return v;
}

// ---------------------------------------------------------------------------
// 16-byte vectors of logits (8 bf16 or 4 fp32 entries)
// ---------------------------------------------------------------------------
// Entries of one 16-byte vector past the end of the row become -inf.
template <int DT>
__device__ __forceinline__ void mask_tail(uint4 &w, int valid) {
    uint32_t *u = reinterpret_cast<uint32_t *>(&w);
    if (DT == SDD_BF16) {
#pragma unroll
        for (int e = 0; e < 8; ++e)
            if (e >= valid) {
                const uint32_t sh = (e & 1) ? 16u : 0u;
                u[e >> 1] = (u[e >> 1] & ~(0xFFFFu << sh)) | (0xFF80u << sh);
            }
    } else {
#pragma unroll
        for (int e = 0; e < 4; ++e)
            if (e >= valid) u[e] = 0xFF800000u;
    }
}

// Entry e of a vector for a run-time e: the word is picked by selects, so the
// vector never has to live in memory to be indexed.
template <int DT>
__device__ __forceinline__ float vec_elem_sel(const uint4 &w, int e) {
    const int k = (DT == SDD_BF16) ? (e >> 1) : e;
    const uint32_t u = (k < 2) ? ((k == 0) ? w.x : w.y) : ((k == 2) ? w.z : w.w);
    if (DT == SDD_BF16) return (e & 1) ? bf16_hi(u) : bf16_lo(u);
    return __uint_as_float(u);
}

template <int DT>
__device__ __forceinline__ float vec_elem(const uint4 &w, int e) {
    const uint32_t *u = reinterpret_cast<const uint32_t *>(&w);
    if (DT == SDD_BF16) return (e & 1) ? bf16_hi(u[e >> 1]) : bf16_lo(u[e >> 1]);
    return __uint_as_float(u[e]);
}

// Clamp one vector from below (NaN-propagating).
template <int DT>
__device__ __forceinline__ uint4 clamp_vec(uint4 w) {
    uint32_t *u = reinterpret_cast<uint32_t *>(&w);
    if (DT == SDD_BF16) {
#pragma unroll
        for (int q = 0; q < 4; ++q) u[q] = bf16x2_max_nan(u[q], kClampPairBf16);
    } else {
#pragma unroll
        for (int q = 0; q < 4; ++q) u[q] = __float_as_uint(fmax_nan(__uint_as_float(u[q]), clamp_floor()));
    }
    return w;
}

__device__ __forceinline__ void status_or(int32_t *status, uint32_t bits) {
    if (status) atomicOr(reinterpret_cast<unsigned int *>(status), bits);
}

}  // namespace sdd
