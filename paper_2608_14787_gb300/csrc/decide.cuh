// decide.cuh -- the per-block work after the streaming pass (decide_cta) and
// its helpers; included by decide.cu (decide_kernel, shard_draw_kernel) and
// pipe.cu (the pipelined round).
//
// One team of NT threads (kDecThreads in decide_kernel) per (listed block,
// draw segment).
// Phase 1: every team finalises all rows of its block, one row per thread,
// into shared memory (rules.cuh).  Phase 2 (sampling rule): every team takes
// the strict accepted length L.  Phase 3: the inverse-CDF draw of the
// speculative-sampling rule cited by Sec. 3.1 -- at the first rejected
// position the residual norm(max(0, p_t - p_d)), or, when the whole block is
// accepted, p_t of the bonus row: each team sums its segment of the draw row
// and publishes its per-thread prefix sums; the last to finish (atomic
// arrival, no waiting) locates the segment, then the thread, from those sums,
// and searches that thread's run with one warp.  Last, every other rule
// (lenience, top-k; greedy strict), the skip schedule and the agreement
// counters, one warp per rule or threshold pair, shared round robin by the
// block's segment teams under the sampling rule; the segment-0 team writes
// the commits.
#pragma once

#include "rules.cuh"

namespace sdd {

namespace {

// The decide's barrier: named barrier 1 over the NT threads that run it (the
// whole CTA of decide_kernel and shard_draw_kernel; the first warps of a CTA
// of the pipelined round, whose other warps never wait on it).
template <int NT = kDecThreads>
__device__ __forceinline__ void dec_sync() { asm volatile("bar.sync 1, %0;" ::"n"(NT) : "memory"); }

// Draw-row context: integer references and the hi/lo LSE difference.
struct DrawCtx {
    const char *zt_row, *zd_row;
    float nrt, nrd, d_hi, d_lo;
    f2_t nrt2, nrd2, d_hi2, d_lo2;   // the same constants in both halves of a pair
};

__device__ __forceinline__ DrawCtx draw_ctx(const char *zt_row, const char *zd_row, df lse_t, df lse_d) {
    DrawCtx c;
    c.zt_row = zt_row;
    c.zd_row = zd_row;
    c.nrt = -ceilf(lse_t.hi * kLog2e);
    c.nrd = 0.f;
    c.d_hi = 0.f;
    c.d_lo = 0.f;
    if (zd_row) {
        c.nrd = -ceilf(lse_d.hi * kLog2e);
        const df D = df_sub(lse_t, lse_d);
        c.d_hi = D.hi;
        c.d_lo = D.lo;
    }
    c.nrt2 = f2_pack(c.nrt, c.nrt);
    c.nrd2 = f2_pack(c.nrd, c.nrd);
    c.d_hi2 = f2_pack(c.d_hi, c.d_hi);
    c.d_lo2 = f2_pack(c.d_lo, c.d_lo);
    return c;
}

// e^x - 1 for x > 0.  Below 0.35 the Taylor polynomial of degree 7 in Horner
// form (truncation error x^8/8! < 2e-8 relative there); above it 2^(x log2 e)
// - 1, where the subtraction loses less than a factor 3.4 of relative accuracy.
__device__ __forceinline__ float expm1_pos(float x) {
    if (x < 0.35f) {
        float p = 1.f / 5040.f;
        p = fmaf(p, x, 1.f / 720.f);
        p = fmaf(p, x, 1.f / 120.f);
        p = fmaf(p, x, 1.f / 24.f);
        p = fmaf(p, x, 1.f / 6.f);
        p = fmaf(p, x, 0.5f);
        p = fmaf(p, x, 1.f);
        return p * x;
    }
    return ex2(x * kLog2e) - 1.f;
}

// Weight of one entry of the draw row (fp32; the product is rounded, never
// fused into a following sum, so every pass sees the same weight):
//   residual: p_t - p_d = p_d (exp(D(v)) - 1) with the log-ratio
//             D(v) = (z_t(v) - z_d(v)) - (LSE_t - LSE_d); the LSE difference is
//             applied as two fp32 terms (hi + lo) and the difference by expm1, so
//             no cancellation between near-equal p_t and p_d loses precision;
//             p_d(v) = 2^(z_d(v) log2(e) - r_d) up to the common factor of the row;
//   bonus (zd_row == nullptr): 2^(z_t(v) log2(e) - r_t).
// Entries past V weigh 0.
__device__ __forceinline__ float entry_weight(const DrawCtx &c, float zt, float zd, int v, int V) {
    zt = fmax_nan(zt, clamp_floor());
    zd = fmax_nan(zd, clamp_floor());
    float w;
    if (c.zd_row) {
        const float dv = ((zt - zd) - c.d_hi) - c.d_lo;
        w = (dv > 0.f) ? __fmul_rn(ex2(fmaf(zd, kLog2e, c.nrd)), expm1_pos(dv)) : 0.f;
    } else {
        w = ex2(fmaf(zt, kLog2e, c.nrt));
    }
    return (v < V) ? w : 0.f;
}

__device__ __forceinline__ f2_t f2_splat(float v) { return f2_pack(v, v); }

// expm1_pos on both halves of a pair, without branches: the same Taylor
// polynomial and the same 2^(x log2 e) - 1, each rounded as the scalar form
// rounds it, the half's range picking the result.
__device__ __forceinline__ f2_t expm1_pos2(f2_t x) {
    f2_t p = f2_splat(1.f / 5040.f);
    p = f2_fma(p, x, f2_splat(1.f / 720.f));
    p = f2_fma(p, x, f2_splat(1.f / 120.f));
    p = f2_fma(p, x, f2_splat(1.f / 24.f));
    p = f2_fma(p, x, f2_splat(1.f / 6.f));
    p = f2_fma(p, x, f2_splat(0.5f));
    p = f2_fma(p, x, f2_splat(1.f));
    p = f2_mul(p, x);
    float y0, y1, x0, x1, p0, p1;
    f2_unpack(f2_mul(x, f2_splat(kLog2e)), y0, y1);
    f2_unpack(x, x0, x1);
    f2_unpack(p, p0, p1);
    const f2_t e = f2_sub(f2_pack(ex2(y0), ex2(y1)), f2_splat(1.f));
    float e0, e1;
    f2_unpack(e, e0, e1);
    return f2_pack(x0 < 0.35f ? p0 : e0, x1 < 0.35f ? p1 : e1);
}

// entry_weight of two entries at once (both below V), through the packed
// f32x2 pipe: every half is rounded exactly as the scalar form rounds it, so
// both give the same weights bit for bit.  zt0..zd1 are clamped logits.
__device__ __forceinline__ void pair_weights(const DrawCtx &c, float zt0, float zt1, float zd0, float zd1, float &w0,
                                             float &w1) {
    if (c.zd_row) {
        const f2_t zd = f2_pack(zd0, zd1);
        const f2_t dv = f2_sub(f2_sub(f2_sub(f2_pack(zt0, zt1), zd), c.d_hi2), c.d_lo2);
        float a0, a1, q0, q1, d0, d1;
        f2_unpack(f2_fma(zd, f2_splat(kLog2e), c.nrd2), a0, a1);
        f2_unpack(f2_mul(f2_pack(ex2(a0), ex2(a1)), expm1_pos2(dv)), q0, q1);
        f2_unpack(dv, d0, d1);
        w0 = (d0 > 0.f) ? q0 : 0.f;
        w1 = (d1 > 0.f) ? q1 : 0.f;
    } else {
        float a0, a1;
        f2_unpack(f2_fma(f2_pack(zt0, zt1), f2_splat(kLog2e), c.nrt2), a0, a1);
        w0 = ex2(a0);
        w1 = ex2(a1);
    }
}

// Entry e of a 16-byte vector of logits, widened to fp32.
// (Word picked by selects: a run-time e never indexes a local array.)
template <int DT>
__device__ __forceinline__ float vec_entry(const uint4 &a, int e) {
    const int k = (DT == SDD_BF16) ? (e >> 1) : e;
    const uint32_t u = (k < 2) ? ((k == 0) ? a.x : a.y) : ((k == 2) ? a.z : a.w);
    if (DT == SDD_BF16) return (e & 1) ? bf16_hi(u) : bf16_lo(u);
    return __uint_as_float(u);
}

// Weights of the draw for the EPV entries of one 16-byte vector (the values
// of entry_weight; entries past V weigh 0).
template <int DT>
__device__ __forceinline__ void vec_weights(const DrawCtx &c, uint4 a, uint4 d, int vec, int V, float (&w)[8]) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    const uint32_t *au = reinterpret_cast<const uint32_t *>(&a);
    const uint32_t *du = reinterpret_cast<const uint32_t *>(&d);
    if (DT == SDD_BF16) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const uint32_t t2 = bf16x2_max_nan(au[k], kClampPairBf16), d2 = bf16x2_max_nan(du[k], kClampPairBf16);
            pair_weights(c, bf16_lo(t2), bf16_hi(t2), bf16_lo(d2), bf16_hi(d2), w[2 * k], w[2 * k + 1]);
        }
    } else {
#pragma unroll
        for (int k = 0; k < 2; ++k)
            pair_weights(c, fmax_nan(__uint_as_float(au[2 * k]), clamp_floor()),
                         fmax_nan(__uint_as_float(au[2 * k + 1]), clamp_floor()),
                         fmax_nan(__uint_as_float(du[2 * k]), clamp_floor()),
                         fmax_nan(__uint_as_float(du[2 * k + 1]), clamp_floor()), w[2 * k], w[2 * k + 1]);
    }
    if (static_cast<int64_t>(vec + 1) * EPV > V) {
#pragma unroll
        for (int e = 0; e < EPV; ++e)
            if (vec * EPV + e >= V) w[e] = 0.f;
    }
}

// The first entry of vectors [vb, ve) at which the running weight sum exceeds
// rem (a double-float), by one warp: 32 entries at a time, one per lane, a
// warp prefix sum and a ballot.  If rounding leaves no such entry, the last
// entry of positive weight; -1 if there is none.
template <int DT>
__device__ __forceinline__ int warp_search(const DrawCtx &c, int vb, int ve, int V, df rem, int lane) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    const int n = (ve - vb) * EPV;
    float carry = 0.f;
    int lastp = -1;
    for (int k0 = 0; k0 < n; k0 += 32) {
        const int k = k0 + lane;
        float w = 0.f;
        if (k < n) {
            const int vec = vb + k / EPV, e = k % EPV;
            const uint4 a = __ldg(reinterpret_cast<const uint4 *>(c.zt_row) + vec);
            const uint4 d = c.zd_row ? __ldg(reinterpret_cast<const uint4 *>(c.zd_row) + vec) : make_uint4(0, 0, 0, 0);
            w = entry_weight(c, vec_entry<DT>(a, e), vec_entry<DT>(d, e), vec * EPV + e, V);
        }
        float run = w;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const float t = __shfl_up_sync(0xFFFFFFFFu, run, off);
            if (lane >= off) run += t;
        }
        run += carry;
        const unsigned hit = __ballot_sync(0xFFFFFFFFu, w > 0.f && !df_ge(rem, df{run, 0.f}));
        if (hit) return vb * EPV + k0 + __ffs(hit) - 1;
        const unsigned pos = __ballot_sync(0xFFFFFFFFu, w > 0.f);
        if (pos) lastp = vb * EPV + k0 + 31 - __clz(pos);
        carry = __shfl_sync(0xFFFFFFFFu, run, 31);
    }
    return lastp;
}

// Inclusive scan of one fp32 value per thread over a team of NT threads.
// Returns the thread's inclusive value; *total receives the CTA total.
template <int NT = kDecThreads>
__device__ __forceinline__ float cta_incl_scan(float v, float *warp_tot, float *total) {
    constexpr int NW = NT / 32;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const float t = __shfl_up_sync(0xFFFFFFFFu, v, off);
        if (lane >= off) v += t;
    }
    if (lane == 31) warp_tot[warp] = v;
    dec_sync<NT>();
    if (threadIdx.x < 32) {
        float t = (lane < NW) ? warp_tot[lane] : 0.f;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const float s = __shfl_up_sync(0xFFFFFFFFu, t, off);
            if (lane >= off) t += s;
        }
        if (lane < NW) warp_tot[NW + lane] = t;   // inclusive prefix of the warp totals
    }
    dec_sync<NT>();
    const float r = ((warp > 0) ? warp_tot[NW + warp - 1] : 0.f) + v;
    *total = warp_tot[2 * NW - 1];
    dec_sync<NT>();
    return r;
}

// Sum (fp32, ascending order) of the draw weights of vectors [vb, ve).
template <int DT>
__device__ __forceinline__ float run_sum(const DrawCtx &c, int vb, int ve, int V) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    float sum = 0.f;
    for (int v = vb; v < ve; v += 4) {
        uint4 a[4], d[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int vec = v + k;
            a[k] = d[k] = make_uint4(0, 0, 0, 0);
            if (vec < ve) {
                a[k] = __ldg(reinterpret_cast<const uint4 *>(c.zt_row) + vec);
                if (c.zd_row) d[k] = __ldg(reinterpret_cast<const uint4 *>(c.zd_row) + vec);
            }
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int vec = v + k;
            if (vec < ve) {
                float w[8];
                vec_weights<DT>(c, a[k], d[k], vec, V, w);
#pragma unroll
                for (int e = 0; e < EPV; ++e) sum += w[e];
            }
        }
    }
    return sum;
}

// run_sum over a chunk staged in shared memory, added to sum: st / sd hold
// the draw rows' vectors [v0, v0 + n) (sd unused for the bonus row); vectors
// [lb, le) of the chunk (none when lb >= le), the same order and arithmetic
// as run_sum.
template <int DT>
__device__ __forceinline__ float stage_sum(const DrawCtx &c, const uint4 *st, const uint4 *sd, int lb, int le,
                                           int v0, int V, float sum) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    for (int v = lb; v < le; ++v) {
        const uint4 a = st[v];
        const uint4 d = c.zd_row ? sd[v] : make_uint4(0, 0, 0, 0);
        float w[8];
        vec_weights<DT>(c, a, d, v0 + v, V, w);
#pragma unroll
        for (int e = 0; e < EPV; ++e) sum += w[e];
    }
    return sum;
}

// The first entry of vectors [vb, ve) whose running sum (same order and
// arithmetic as run_sum) exceeds rem, a double-float; -1 if none.
template <int DT>
__device__ __forceinline__ int run_find(const DrawCtx &c, int vb, int ve, int V, df rem, int &last_pos) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    float sum = 0.f;
    for (int vec = vb; vec < ve; ++vec) {
        const uint4 a = __ldg(reinterpret_cast<const uint4 *>(c.zt_row) + vec);
        const uint4 d = c.zd_row ? __ldg(reinterpret_cast<const uint4 *>(c.zd_row) + vec) : make_uint4(0, 0, 0, 0);
        float w[8];
        vec_weights<DT>(c, a, d, vec, V, w);
#pragma unroll
        for (int e = 0; e < EPV; ++e) {
            sum += w[e];
            if (w[e] > 0.f) {
                last_pos = vec * EPV + e;
                if (!df_ge(rem, df{sum, 0.f})) return vec * EPV + e;
            }
        }
    }
    return -1;
}

// Inverse CDF over vectors [v0, v1) of the draw row, one contiguous run of
// `vpt` vectors per thread: the first entry at which the running sum exceeds
// rem (a double-float), or the last positive entry if rounding leaves none;
// identical in every thread.
template <int DT, int NT = kDecThreads>
__device__ int cta_find(const DrawCtx &c, int v0, int v1, int vpt, int V, df rem, float *s_warp, int *s_thr,
                        int *s_tok) {
    const int vb = min(v1, v0 + static_cast<int>(threadIdx.x) * vpt), ve = min(v1, vb + vpt);
    const float ts = run_sum<DT>(c, vb, ve, V);
    float tot;
    const float incl = cta_incl_scan<NT>(ts, s_warp, &tot);
    if (threadIdx.x == 0) *s_thr = INT32_MAX;
    dec_sync<NT>();
    const bool mine = (ve > vb) && !df_ge(rem, df{incl, 0.f});
    const unsigned bal = __ballot_sync(0xFFFFFFFFu, mine);
    if ((threadIdx.x & 31) == 0 && bal) atomicMin(s_thr, static_cast<int>(threadIdx.x) + __ffs(bal) - 1);
    dec_sync<NT>();
    const int thr = *s_thr;
    if (thr == INT32_MAX) return -1;
    if (static_cast<int>(threadIdx.x) == thr) {
        int lp = -1;
        const int pick = run_find<DT>(c, vb, ve, V, df_sub(rem, df{incl - ts, 0.f}), lp);
        *s_tok = (pick >= 0) ? pick : lp;
    }
    dec_sync<NT>();
    return *s_tok;
}

// Vocabulary-sharded draw: the weight sum of thread tid's run of a draw row of
// RV vectors cut into one run of ceil(RV / kDecThreads) vectors per thread --
// the same runs in the decide kernel's slice mass and in the draw, so that
// both see the same sums bit for bit.
template <int DT>
__device__ __forceinline__ float slice_thread_sum(const DrawCtx &c, int RV, int V) {
    const int vpt = (RV + kDecThreads - 1) / kDecThreads;
    const int vb = min(RV, static_cast<int>(threadIdx.x) * vpt), ve = min(RV, vb + vpt);
    return run_sum<DT>(c, vb, ve, V);
}

// Inverse CDF over a whole draw row of RV vectors by one CTA (the runs of
// slice_thread_sum): the first entry at which the running sum exceeds rem, or
// -- when rounding leaves none, or rem is infinite -- the row's last entry of
// positive weight; -1 if the row has no weight.  Identical in every thread.
template <int DT>
__device__ int slice_find(const DrawCtx &c, int RV, int V, df rem, float *s_warp, int *s_thr, int *s_last,
                          int *s_tok) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int vpt = (RV + kDecThreads - 1) / kDecThreads;
    const int vb = min(RV, static_cast<int>(threadIdx.x) * vpt), ve = min(RV, vb + vpt);
    const float ts = run_sum<DT>(c, vb, ve, V);
    float tot;
    const float incl = cta_incl_scan(ts, s_warp, &tot);
    if (threadIdx.x == 0) {
        *s_thr = INT32_MAX;
        *s_last = -1;
        *s_tok = -1;
    }
    dec_sync();
    const unsigned bal = __ballot_sync(0xFFFFFFFFu, (ve > vb) && !df_ge(rem, df{incl, 0.f}));
    if (lane == 0 && bal) atomicMin(s_thr, warp * 32 + __ffs(bal) - 1);
    const unsigned pos = __ballot_sync(0xFFFFFFFFu, ts > 0.f);
    if (lane == 0 && pos) atomicMax(s_last, warp * 32 + 31 - __clz(pos));
    dec_sync();
    int thr = *s_thr;
    df r2 = df_sub(rem, df{incl - ts, 0.f});
    if (thr == INT32_MAX) {
        thr = *s_last;
        r2 = df{__int_as_float(0x7F800000), 0.f};
    }
    if (static_cast<int>(threadIdx.x) == thr) {
        int lp = -1;
        const int pick = run_find<DT>(c, vb, ve, V, r2, lp);
        *s_tok = (pick >= 0) ? pick : lp;
    }
    dec_sync();
    return *s_tok;
}

// Skip schedule of threshold pair t for a block (Sec. 4.1), by one warp, from
// the drafter facts: prefix sums of ln q as double-floats, then sched_step
// chunk by chunk and sched_final.
__device__ __forceinline__ void sched_pair(const DecideParams &d, const BlockFacts &F, int t, bool force, int D,
                                           int lane, int &Kh, int &K, int &Do) {
    Kh = K = Do = 0;
    if (force || d.tau_off[t]) return;
    const int gamma = d.gamma;
    if (d.signal == SDD_SIG_PERIODIC) {
        Kh = periodic_khat(gamma, d.period[t], d.K_skip, d.round, [&](int j) { return F.guard[j] != 0; }, lane);
        sched_final(Kh, D, d.K_min, d.S_max, K, Do);
        return;
    }
    int kb = gamma, best = 0;
    df carry = df{0.f, 0.f};
    for (int c = 0; c < gamma && kb >= c; c += 32) {
        const int j = c + lane;
        const bool in = j < gamma;
        const df S = df_add(carry, warp_prefix_df(in ? df{F.d_lq[j], 0.f} : df{0.f, 0.f}, lane));
        carry.hi = __shfl_sync(0xFFFFFFFFu, S.hi, 31);
        carry.lo = __shfl_sync(0xFFFFFFFFu, S.lo, 31);
        sched_step(c, lane, gamma, in, in ? F.d_q[j] : 0.f, in && F.guard[j] != 0, S, d.eta_loc[t], d.log_eta_c[t],
                   d.signal, kb, best);
    }
    Kh = (d.signal == SDD_SIG_MARGINAL) ? kb : best;
    sched_final(Kh, D, d.K_min, d.S_max, K, Do);
}

// The draw's last step over staged segment prefixes: s_pref_all holds nseg
// segments' per-thread inclusive prefix sums ([nseg][NT]; a
// segment's total is its last prefix).
//
// segment_cum (warp 0): the segments' cumulative totals as double-floats
// into s_cum; returns the total, and in last_seg the last segment of
// positive mass (-1: none).
template <int NT = kDecThreads>
__device__ __forceinline__ df segment_cum(const float *s_pref_all, int nseg, df *s_cum, int lane, int &last_seg) {
    df carry = df{0.f, 0.f};
    last_seg = -1;
    for (int s0 = 0; s0 < nseg; s0 += 32) {
        const int sg = s0 + lane;
        const float t = (sg < nseg) ? s_pref_all[sg * NT + NT - 1] : 0.f;
        const df cum = df_add(carry, warp_prefix_df(df{t, 0.f}, lane));
        if (sg < nseg) s_cum[sg] = cum;
        if (t > 0.f) last_seg = sg;
        carry.hi = __shfl_sync(0xFFFFFFFFu, cum.hi, 31);
        carry.lo = __shfl_sync(0xFFFFFFFFu, cum.lo, 31);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) last_seg = max(last_seg, __shfl_xor_sync(0xFFFFFFFFu, last_seg, off));
    return carry;
}

// segment_pick (warp 0, after segment_cum and a __syncwarp): the first
// segment of positive mass whose cumulative total exceeds target; -1 if
// rounding leaves none.
template <int NT = kDecThreads>
__device__ __forceinline__ int segment_pick(const float *s_pref_all, int nseg, const df *s_cum, df target, int lane) {
    for (int s0 = 0; s0 < nseg; s0 += 32) {
        const int sg = s0 + lane;
        const bool hit = (sg < nseg) && s_pref_all[sg * NT + NT - 1] > 0.f &&
                         !df_ge(target, s_cum[sg]);
        const unsigned bal = __ballot_sync(0xFFFFFFFFu, hit);
        if (bal) return s0 + __ffs(bal) - 1;
    }
    return -1;
}

// segment_find (every thread of the CTA): the entry of segment sel (vectors
// [sel seg_vec, ...) of a row of RV vectors, NT runs of seg_vec / NT
// vectors) at which the running sum exceeds rem, a
// double-float measured from the segment's start: the thread from the
// segment's prefixes, the entry by warp 0 (warp_search).  When rounding
// leaves no thread, the last thread whose run has positive weight, searched
// to its end.  *s_thr must be INT32_MAX and *s_thr_last -1 on entry.
template <int DT, int NT = kDecThreads>
__device__ int segment_find(const DrawCtx &c, const float *s_pref_all, int sel, df rem, int seg_vec, int RV, int V,
                            int *s_thr, int *s_thr_last, int *s_tok) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int vpt = seg_vec / NT;
    const float *s_pref = s_pref_all + sel * NT;
    const float pv = s_pref[tid];
    const unsigned bal = __ballot_sync(0xFFFFFFFFu, !df_ge(rem, df{pv, 0.f}));
    if (lane == 0 && bal) atomicMin(s_thr, warp * 32 + __ffs(bal) - 1);
    dec_sync<NT>();
    int thr = *s_thr;
    df rem2 = rem;
    if (thr == INT32_MAX) {
        const bool rose = pv > ((tid > 0) ? s_pref[tid - 1] : 0.f);
        const unsigned up = __ballot_sync(0xFFFFFFFFu, rose);
        if (lane == 0 && up) atomicMax(s_thr_last, warp * 32 + 31 - __clz(up));
        dec_sync<NT>();
        thr = *s_thr_last;
        rem2 = df{__int_as_float(0x7F800000), 0.f};
    } else if (thr > 0) {
        rem2 = df_sub(rem, df{s_pref[thr - 1], 0.f});
    }
    if (warp == 0) {
        int pick = -1;
        if (thr >= 0) {
            const int sv0 = sel * seg_vec, sv1 = min(RV, sv0 + seg_vec);
            const int vb = min(sv1, sv0 + thr * vpt), ve = min(sv1, vb + vpt);
            pick = warp_search<DT>(c, vb, ve, V, rem2, lane);
        }
        if (lane == 0) *s_tok = pick;
    }
    dec_sync<NT>();
    return *s_tok;
}

// Draw geometry of one CTA: its listed block i, its segment of the draw row,
// the block's segment count and vectors per segment.  From the host's
// (blocks x segments) grid, or -- when the block count lives on the device
// and the call draws -- from a one-dimensional grid of max(resident CTAs, B)
// CTAs cut on the device into (listed block, segment) pairs the way the host
// cuts its grid (init_dec), so that few listed blocks get more segments.
struct DecGeom {
    int i, seg, nseg, seg_vec;
};
__device__ __forceinline__ DecGeom dec_geom(const ScanParams &p, const PartView &pv, bool draw) {
    DecGeom g;
    if (p.nb_dev == nullptr || !draw) {
        g.i = blockIdx.x;
        g.seg = blockIdx.y;
        g.nseg = p.dec.nseg;
        g.seg_vec = p.dec.seg_vec;
        return g;
    }
    const int nb = static_cast<int>(max(pv.nb, static_cast<int64_t>(1)));
    const int want = max(1, min(kDrawMaxSeg, min(p.dec.dec_ctas, static_cast<int>(gridDim.x)) / nb));
    const int per_thread = max(2, (p.RV + kDecThreads * want - 1) / (kDecThreads * want));
    g.seg_vec = per_thread * kDecThreads;
    g.nseg = (p.RV + g.seg_vec - 1) / g.seg_vec;
    g.i = static_cast<int>(blockIdx.x) / g.nseg;
    g.seg = static_cast<int>(blockIdx.x) % g.nseg;
    return g;
}

// The decide work of one team of NT threads (the whole CTA of decide_kernel,
// NT = kDecThreads; the first NT / 32 warps of a CTA of the pipelined round) for the
// (listed block, draw segment) pair geo, after the streaming pass over p's
// rows has completed.  s_pref_all: nseg * NT floats of shared memory
// (the last segment to arrive stages every segment's prefixes there);
// s_stage: 2 * stage_vec vectors of shared memory through which the team
// reads its segment of both draw rows, or null (read from global memory).  Every
// return is taken by the whole team.  FEAT: also the extended features of the
// drafter rows; SHARD: the vocabulary-sharded round (records of S slices
// instead of warp partials, the draw left to shard_draw_kernel).
template <int DT, bool FEAT, bool SHARD, int NT = kDecThreads>
__device__ __forceinline__ void decide_cta(const ScanParams &p, const PartView &pv, const DecGeom &geo,
                                           float *s_pref_all, uint4 *s_stage = nullptr, int stage_vec = 0) {
    static_assert(!SHARD || NT == kDecThreads, "the sharded round's layouts assume kDecThreads");
    static_assert(NT % 32 == 0 && 2 * NT >= SDD_MAX_GAMMA, "at most two drafted positions per thread");
    const DecideParams &d = p.dec;
    const int i = geo.i;            // listed block
    const int seg = geo.seg;        // segment of the draw row
    const int nseg = geo.nseg, seg_vec = geo.seg_vec;
    const bool leader = seg == 0;   // writes the block's outputs
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    constexpr int NW = NT / 32;
    const int gamma = p.gamma;

    __shared__ BlockFacts F;
    __shared__ int s_L[kMaxRules], s_corr[kMaxRules];
    __shared__ int s_K0, s_force, s_D;

    int gd = -1, gt = -1;
    for (int gi = 0; gi < p.n_groups; ++gi) {
        if (p.grp[gi].kind == 0)
            gd = gi;
        else
            gt = gi;
    }
    if (i >= pv.nb) return;   // (a device block count below the grid's)
    const int32_t *bidx = p.grp[0].bidx;
    const int b = bidx ? __ldg(bidx + i) : i;
    if (b < 0 || b >= p.B) {
        if (leader && tid == 0) status_or(p.status, SDD_DEV_BAD_TOKEN);
        return;
    }
    const bool dec = d.enabled != 0;
    const bool sampling = dec && d.do_strict && !d.greedy;
    const bool has_d = gd >= 0;
    const bool alone_d = !has_d && sampling;   // drafter facts from the caller's LSE
    const int nd = (has_d || alone_d) ? gamma : 0;
    const int nt = (gt >= 0) ? gamma + 1 : 0;
    const int64_t ob = static_cast<int64_t>(b) * gamma;
    const int64_t bo = static_cast<int64_t>(b) * (gamma + 1);

    // ---- phase 1: facts of every row of the block, one row per thread ----
    // the drafted tokens, guard flags and the block's schedule inputs (gamma <=
    // 2 NT: at most two positions per thread) are loaded in the same batch as
    // the rows' partials below and stored after them: one round trip
    int32_t xj[2] = {0, 0}, force_b = 0, D_b = 0;
    uint8_t gj[2] = {0, 0};
    if (dec) {
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            const int j = tid + k * NT;
            if (j < gamma) {
                xj[k] = __ldg(d.tokens + ob + j);
                gj[k] = d.guard ? d.guard[ob + j] : 0;
            }
        }
        if (tid == 0) {
            force_b = d.force_strict ? d.force_strict[b] : 0;
            D_b = d.D_in ? d.D_in[b] : 0;
        }
    }
    for (int s = tid; s < nd + nt; s += NT) {
        if (s < nd) {
            const int j = s;
            RowFacts f;
            if (has_d) {
                const ScanGroup &G = p.grp[gd];
                SoftState acc;
                float g;
                bool bad;
                const int64_t r = (gd ? pv.rows0 : 0) + static_cast<int64_t>(i) * G.npos + j;
                if (SHARD) {
                    merge_row_shards(p, r, -1, false, acc, g, bad);
                    f = row_final(p, G, j, b, acc, g, bad, leader);
                } else if (FEAT && leader) {
                    float top[5];
                    merge_row_t<true>(p, pv, r, acc, g, bad, top);
                    f = row_final(p, G, j, b, acc, g, bad, leader);
                    feat_final(G, static_cast<int64_t>(b) * p.gamma + j, top, f.lse);
                } else {
                    merge_row(p, pv, r, acc, g, bad);
                    f = row_final(p, G, j, b, acc, g, bad, leader);
                }
            } else {
                // stand-alone acceptance: the caller's drafter LSE and the token's drafter logit
                f = facts_invalid();
                f.lse = df_from_double(__ldg(d.d_lse + ob + j));
                const int xj = __ldg(d.tokens + ob + j);
                f.g = (xj >= 0 && xj < p.V)
                          ? fmax_nan(logit_at<DT>(d.zd + (ob + j) * d.stride_bytes, xj), clamp_floor())
                          : qnan();
            }
            put_drafter(F, j, f);
        } else {
            const int j = s - nd;
            const ScanGroup &G = p.grp[gt];
            SoftState acc;
            float g;
            bool bad;
            const int64_t r = (gt ? pv.rows0 : 0) + static_cast<int64_t>(i) * G.npos + j;
            if (SHARD)
                merge_row_shards(p, r, (j < gamma) ? __ldg(d.tokens + ob + j) : -1, j < gamma, acc, g, bad);
            else
                merge_row(p, pv, r, acc, g, bad);
            put_target(F, j, row_final(p, G, j, b, acc, g, bad, leader));
        }
    }
    if (dec) {
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            const int j = tid + k * NT;
            if (j < gamma) {
                F.x[j] = xj[k];
                F.guard[j] = gj[k];
            }
        }
        if (tid == 0) {
            s_force = force_b;
            s_D = D_b;
        }
    }
    dec_sync<NT>();
    if (!dec) return;
    const bool sched = d.do_sched && has_d;

    if (sampling) {
        // ---- phase 2 (every CTA): the strict accepted length L ----
        if (warp == 0) {
            const int L = rule_first_reject(d, F, 0, b, lane);
            if (lane == 0) {
                s_L[0] = L;
                s_corr[0] = F.t_am[L];
            }
        } else if (warp == 1 && sched) {
            // pair 0 decides whether this block commits its verified tokens
            int Kh, K, Do;
            sched_pair(d, F, 0, s_force != 0, s_D, lane, Kh, K, Do);
            if (lane == 0) s_K0 = K;
        }
        __shared__ float s_warp[2 * NW];
        __shared__ int s_is_last, s_seg, s_thr, s_thr_last, s_tok;
        __shared__ df s_rem;
        __shared__ df s_cum[kDrawMaxSeg];
        if (tid == 0) {
            s_thr = INT32_MAX;
            s_thr_last = -1;
        }
        dec_sync<NT>();

        if (SHARD) {
            // ---- vocabulary-sharded: this CTA's segment of this slice's draw
            // row -- the residual (or bonus) weights' per-thread prefixes,
            // published for shard_draw_kernel, and the segment's p_t mass; the
            // last segment to arrive sums the segments' masses in order into
            // this slice's masses for the exchange between ranks ----
            const int L = s_L[0];
            const char *zt_row = d.zt + (bo + L) * d.stride_bytes;
            const char *zd_row = (L < gamma) ? d.zd + (ob + L) * d.stride_bytes : nullptr;
            const DrawCtx c = draw_ctx(zt_row, zd_row, df{F.t_lh[L], F.t_ll[L]},
                                       (L < gamma) ? df{F.d_lh[L], F.d_ll[L]} : df{0.f, 0.f});
            const int vpt = seg_vec / NT;
            const int sv0 = seg * seg_vec, sv1 = min(p.RV, sv0 + seg_vec);
            const int vb = min(sv1, sv0 + tid * vpt), ve = min(sv1, vb + vpt);
            float tot_r, tot_p;
            const float incl = cta_incl_scan<NT>(run_sum<DT>(c, vb, ve, p.V), s_warp, &tot_r);
            d.res_pref[(static_cast<int64_t>(b) * kDrawMaxSeg + seg) * NT + tid] = incl;
            if (L < gamma) {
                DrawCtx ct = c;
                ct.zd_row = nullptr;
                (void)cta_incl_scan<NT>(run_sum<DT>(ct, vb, ve, p.V), s_warp, &tot_p);
            } else {
                tot_p = tot_r;
            }
            if (tid == 0) d.shard_ptot[static_cast<int64_t>(b) * kDrawMaxSeg + seg] = tot_p;
            dec_sync<NT>();
            if (tid == 0) {
                // (as in the one-GPU draw: release of this segment's stores,
                // acquire of the others' for the last arriver)
                const uint32_t old = atom_add_acq_rel_gpu(d.res_count + b, 1u);
                s_is_last = (old == static_cast<uint32_t>(nseg - 1)) ? 1 : 0;
            }
            dec_sync<NT>();
            if (s_is_last && warp == 0) {
                df cr = df{0.f, 0.f}, cp = df{0.f, 0.f};
                for (int s0 = 0; s0 < nseg; s0 += 32) {
                    const int sg = s0 + lane;
                    const int64_t at = static_cast<int64_t>(b) * kDrawMaxSeg + sg;
                    const float tr = (sg < nseg) ? __ldcg(d.res_pref + at * NT + NT - 1) : 0.f;
                    const float tq = (sg < nseg) ? __ldcg(d.shard_ptot + at) : 0.f;
                    const df xr = df_add(cr, warp_prefix_df(df{tr, 0.f}, lane));
                    const df xq = df_add(cp, warp_prefix_df(df{tq, 0.f}, lane));
                    cr.hi = __shfl_sync(0xFFFFFFFFu, xr.hi, 31);
                    cr.lo = __shfl_sync(0xFFFFFFFFu, xr.lo, 31);
                    cp.hi = __shfl_sync(0xFFFFFFFFu, xq.hi, 31);
                    cp.lo = __shfl_sync(0xFFFFFFFFu, xq.lo, 31);
                }
                if (lane == 0) {
                    d.shard_mass[2 * b] = cr.hi + cr.lo;
                    d.shard_mass[2 * b + 1] = cp.hi + cp.lo;
                    d.res_count[b] = 0u;   // leave the counter at zero for the next call
                }
            }
            if (leader) {
                const bool commit = sched && s_K0 == 0;
                if (tid == 0) {
                    ShardDraw sd;
                    sd.L = L;
                    sd.commit = commit ? 1 : 0;
                    sd.t_lh = F.t_lh[L];
                    sd.t_ll = F.t_ll[L];
                    sd.d_lh = (L < gamma) ? F.d_lh[L] : 0.f;
                    sd.d_ll = (L < gamma) ? F.d_ll[L] : 0.f;
                    sd.pad[0] = sd.pad[1] = 0;
                    d.shard_state[b] = sd;
                }
                if (warp == 0) {
                    // the drawn token's place stays -1 until the draw
                    if (lane == 0) {
                        if (d.L_strict) d.L_strict[b] = L;
                        if (d.n_strict) d.n_strict[b] = L + 1;
                        if (commit && d.commit_n) d.commit_n[b] = L + 1;
                    }
                    if (d.tok_strict) write_tokens(lane, gamma, d.tok_strict + bo, F.x, L, -1);
                    if (commit && d.commit_tokens) write_tokens(lane, gamma, d.commit_tokens + bo, F.x, L, -1);
                }
            }
        } else {
        // ---- phase 3 (every CTA): its segment of the draw row at position L
        // (the residual row, or the bonus row when every position passed) ----
        const int L = s_L[0];
        const char *zt_row = d.zt + (bo + L) * d.stride_bytes;
        const char *zd_row = (L < gamma) ? d.zd + (ob + L) * d.stride_bytes : nullptr;
        const DrawCtx c = draw_ctx(zt_row, zd_row, df{F.t_lh[L], F.t_ll[L]},
                                   (L < gamma) ? df{F.d_lh[L], F.d_ll[L]} : df{0.f, 0.f});
        const int vpt = seg_vec / NT;
        const int64_t pair = static_cast<int64_t>(i) * nseg + seg;
        {
            const int v0 = seg * seg_vec, v1 = min(p.RV, v0 + seg_vec);
            const int vb = min(v1, v0 + tid * vpt), ve = min(v1, vb + vpt);
            float ts;
            if (s_stage) {
                // the segment of both draw rows through shared memory in
                // chunks of stage_vec vectors: one round trip per chunk (under
                // a concurrent streaming pass each dependent round trip is
                // long); every thread sums its run chunk by chunk, in order
                ts = 0.f;
                const uint4 *gt = reinterpret_cast<const uint4 *>(zt_row);
                const uint4 *gdr = zd_row ? reinterpret_cast<const uint4 *>(zd_row) : nullptr;
                for (int c0 = v0; c0 < v1; c0 += stage_vec) {
                    const int c1 = min(v1, c0 + stage_vec);
                    for (int q = tid; q < c1 - c0; q += NT) {
                        cp_async16(s_stage + q, gt + c0 + q);
                        if (gdr) cp_async16(s_stage + stage_vec + q, gdr + c0 + q);
                    }
                    cp_async_wait_all();
                    dec_sync<NT>();
                    ts = stage_sum<DT>(c, s_stage, s_stage + stage_vec, max(vb, c0) - c0, min(ve, c1) - c0, c0,
                                       p.V, ts);
                    dec_sync<NT>();   // (the next chunk overwrites the stage)
                }
            } else {
                ts = run_sum<DT>(c, vb, ve, p.V);
            }
            float tot;
            const float incl = cta_incl_scan<NT>(ts, s_warp, &tot);
            (void)tot;
            d.res_pref[pair * NT + tid] = incl;   // this thread's inclusive prefix in the segment
            dec_sync<NT>();
            if (tid == 0) {
                // the barrier above orders every thread's prefix store before
                // this release; the acquire half orders the last arriver's
                // reads of the other segments' prefixes after their releases
                const uint32_t old = atom_add_acq_rel_gpu(d.res_count + i, 1u);
                s_is_last = (old == static_cast<uint32_t>(nseg - 1)) ? 1 : 0;
            }
            dec_sync<NT>();
        }
        if (s_is_last) {
            // the last segment to arrive completes the draw: every segment's
            // prefixes in one round trip (a segment's total is its last prefix)
            const float4 *src =
                reinterpret_cast<const float4 *>(d.res_pref + static_cast<int64_t>(i) * nseg * NT);
            for (int q = tid; q < nseg * (NT / 4); q += NT) cp_async16(s_pref_all + 4 * q, src + q);
            cp_async_wait_all();
            dec_sync<NT>();
            if (warp == 0) {
                // R = sum of the segment totals and their inclusive prefix sums
                // (double-floats); the first segment whose prefix exceeds u * R
                int last_seg;   // the last segment of positive mass
                const df Rm = segment_cum<NT>(s_pref_all, nseg, s_cum, lane, last_seg);
                const uint32_t jj = (L < gamma) ? static_cast<uint32_t>(L + 1) : static_cast<uint32_t>(gamma + 1);
                const float u = philox_uniform(d.seed, jj, static_cast<uint32_t>(b), d.round,
                                               (L < gamma) ? kPurposeResid : kPurposeBonus);
                const df target = df_mul_f(Rm, u);
                int sel = -1;
                if (Rm.hi > 0.f) {
                    __syncwarp();
                    sel = segment_pick<NT>(s_pref_all, nseg, s_cum, target, lane);
                }
                if (lane == 0) {
                    if (sel >= 0) {
                        s_seg = sel;
                        s_rem = (sel > 0) ? df_sub(target, s_cum[sel - 1]) : target;   // u R minus the mass before sel
                    } else {
                        // rounding left no segment (-> the row's last positive
                        // entry: an infinite remainder), or there is no mass (-1)
                        s_seg = (Rm.hi > 0.f) ? last_seg : -1;
                        s_rem = df{__int_as_float(0x7F800000), 0.f};
                    }
                    d.res_count[i] = 0u;   // leave the workspace zeroed
                }
            }
            dec_sync<NT>();
            int tok;
            const int sel = s_seg;
            if (sel >= 0) {
                // the thread of segment sel whose run holds u R, from the
                // inclusive prefixes that segment's CTA published, then the entry
                tok = segment_find<DT, NT>(c, s_pref_all, sel, s_rem, seg_vec, p.RV, p.V, &s_thr, &s_thr_last, &s_tok);
            } else {
                // the residual has no mass (only through rounding): draw from p_t
                // of the same row, whole row in this CTA, same inverse-CDF rule
                DrawCtx ct = c;
                ct.zd_row = nullptr;
                const int vrow = (p.RV + NT - 1) / NT;
                const int vb = min(p.RV, tid * vrow), ve = min(p.RV, vb + vrow);
                float tot;
                (void)cta_incl_scan<NT>(run_sum<DT>(ct, vb, ve, p.V), s_warp, &tot);
                const float u = philox_uniform(d.seed, static_cast<uint32_t>(L + 1), static_cast<uint32_t>(b),
                                               d.round, kPurposeResid);
                tok = (tot > 0.f)
                          ? cta_find<DT, NT>(ct, 0, p.RV, vrow, p.V, df_mul_f(df{tot, 0.f}, u), s_warp, &s_thr, &s_tok)
                          : -1;
            }
            if (warp == 0) {
                if (lane == 0) {
                    if (d.L_strict) d.L_strict[b] = L;
                    if (d.n_strict) d.n_strict[b] = L + 1;
                }
                if (d.tok_strict) write_tokens(lane, gamma, d.tok_strict + bo, F.x, L, tok);
                if (sched && s_K0 == 0) {
                    // commit under pair 0: this block was not skipped
                    if (lane == 0 && d.commit_n) d.commit_n[b] = L + 1;
                    if (d.commit_tokens) write_tokens(lane, gamma, d.commit_tokens + bo, F.x, L, tok);
                }
            }
        }
        }
        if (SHARD && !leader) return;
        dec_sync<NT>();
    }

    // ---- every other rule (a warp per rule), the schedule (a warp per
    // threshold pair) and the agreement counters: under the sampling rule the
    // block's draw segments share these tasks round robin (every team holds
    // the block's facts), otherwise the one team takes them all; then the
    // leader writes the remaining commits ----
    const int R = 1 + d.n_ell + d.n_k;
    const int S = (sampling && !SHARD) ? nseg : 1, me = (sampling && !SHARD) ? seg : 0;
    for (int ir = warp;; ir += NW) {
        const int r = me + ir * S;   // this team's share of the rules
        if (r >= R) break;
        if (r == 0) {
            if (!d.do_strict || sampling) continue;   // sampling: completed by the draw
            const int L = rule_first_reject(d, F, 0, b, lane);
            if (lane == 0) {
                s_L[0] = L;
                s_corr[0] = F.t_am[L];
                if (d.L_strict) d.L_strict[b] = L;
                if (d.n_strict) d.n_strict[b] = L + 1;
            }
            if (d.tok_strict) write_tokens(lane, gamma, d.tok_strict + bo, F.x, L, F.t_am[L]);
        } else {
            const int L = rule_first_reject(d, F, r, b, lane);
            const int corr = F.t_am[L];   // target argmax at the first rejection, or of the bonus row
            const bool len = r <= d.n_ell;
            const int64_t o = static_cast<int64_t>(len ? r - 1 : r - 1 - d.n_ell) * p.B + b;
            int32_t *Lo = len ? d.L_len : d.L_topk, *no = len ? d.n_len : d.n_topk;
            int32_t *to = len ? d.tok_len : d.tok_topk;
            if (lane == 0) {
                if (Lo) Lo[o] = L;
                if (no) no[o] = L + 1;
            }
            if (to) write_tokens(lane, gamma, to + o * (gamma + 1), F.x, L, corr);
        }
    }
    if (!sched) return;
    dec_sync<NT>();   // s_L[0] of a greedy strict rule
    const int t0 = ((me - R) % S + S) % S;   // pair t goes to team (R + t) mod S
    for (int it = warp;; it += NW) {
        const int t = t0 + it * S;
        if (t >= d.n_tau) break;
        int Kh, K, Do;
        sched_pair(d, F, t, s_force != 0, s_D, lane, Kh, K, Do);
        if (lane == 0) {
            if (t == 0) s_K0 = K;
            const int64_t o = static_cast<int64_t>(t) * p.B + b;
            if (d.K_hat) d.K_hat[o] = Kh;
            if (d.K) d.K[o] = K;
            if (d.D_out) d.D_out[o] = Do;
            if (d.agreement && K > 0 && d.do_strict) {
                const int L = s_L[0];
                unsigned long long *a = reinterpret_cast<unsigned long long *>(d.agreement + 4 * t);
                atomicAdd(a + 0, static_cast<unsigned long long>(min(K, L)));
                atomicAdd(a + 1, static_cast<unsigned long long>(K));
                atomicAdd(a + 2, static_cast<unsigned long long>(K <= L ? 1 : 0));
                atomicAdd(a + 3, 1ull);
            }
        }
    }
    if (!leader) return;
    dec_sync<NT>();
    if (warp == 0) {
        // tokens committed by a fused round: a skipped block commits x_1..x_K
        // (pair 0); a greedy strict block its verified tokens
        const int K0 = s_K0;
        if (K0 > 0 || (d.do_strict && !sampling)) {
            const int Lc = (K0 > 0) ? K0 : s_L[0];
            const int corr = (K0 > 0) ? -1 : s_corr[0];
            if (lane == 0 && d.commit_n) d.commit_n[b] = (K0 > 0) ? K0 : s_L[0] + 1;
            if (d.commit_tokens) write_tokens(lane, gamma, d.commit_tokens + bo, F.x, Lc, corr);
        }
    }
}

}  // namespace

}  // namespace sdd
