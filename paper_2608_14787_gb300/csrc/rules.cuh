// rules.cuh -- what the decide kernel computes for one block of gamma draft
// positions once every logit has been streamed:
//
//  * row finalisation -- merge a row's per-warp partials (warp order), then
//    LSE as a double-float from an fp32 log, q = p(x_j), log q, maxprob and
//    entropy (the confidence quantities of Sec. 4.2) and the target facts;
//  * per-position acceptance tests -- Strict SDD (Sec. 3.1: greedy, or the
//    speculative-sampling acceptance test it cites), lenience (App. A.6,
//    Eq. 9), top-k (App. A.6);
//  * sched_step / sched_final -- the skip policy of Sec. 4.1: the local gate,
//    then Eq. 3 with the raw / conditional / marginal signals of Sec. 4.2, then
//    K_min, staleness and guards;
//  * periodic_khat -- the confidence-free periodic baseline of the appendix's
//    periodic-skipping paragraph (an attempt every P rounds, same guards);
//  * merge_row_t<true> / feat_final -- the extended features of App. A.7: a
//    drafter row's five largest entries merged from its pieces' lists (loaded
//    with its partials), then the probability margin and the top-5 mass.
//
// Everything here is fp32 or double-float (common.cuh): fp64 instructions
// issue at a small fraction of the fp32 rate on this part.
#pragma once

#include "internal.h"

namespace sdd {

// ---------------------------------------------------------------------------
// Row finalisation
// ---------------------------------------------------------------------------
// Facts of one finalised row.
struct RowFacts {
    df lse;
    float M, g, q, logq;
    int32_t argmax, rank;
};

__device__ __forceinline__ RowFacts facts_invalid() {
    RowFacts f;
    f.lse = df{qnan(), 0.f};
    f.M = f.g = f.q = f.logq = qnan();
    f.argmax = -1;
    f.rank = INT32_MAX;
    return f;
}

// A partial written by the streaming grid: read through L2.
__device__ __forceinline__ Partial load_partial(const Partial *p) {
    union {
        uint4 v[2];
        Partial q;
    } u;
    u.v[0] = __ldcg(reinterpret_cast<const uint4 *>(p));
    u.v[1] = __ldcg(reinterpret_cast<const uint4 *>(p) + 1);
    return u.q;
}

// Merged state of global row r, whose pieces were streamed by warps fw..lw
// (partial of warp w at index r + w), merged in warp order, four loads in
// flight at a time.  The row's first piece carries its token logit; any piece
// flags an out-of-range token.  FEAT (drafter rows of the feature call): also
// the row's five largest entries t, merged from the pieces' lists (p.feat,
// indexed like the partials) loaded in the same batches.
template <bool FEAT>
__device__ __forceinline__ void merge_row_t(const ScanParams &p, const PartView &pv, int64_t r, SoftState &acc,
                                            float &g, bool &tok_bad, float (&t)[5]) {
    const int64_t fw = part_owner(p, pv, r * p.RV), lw = part_owner(p, pv, (r + 1) * p.RV - 1);
    acc = soft_identity();
    g = qnan();
    tok_bad = false;
    if (FEAT) {
#pragma unroll
        for (int k = 0; k < 5; ++k) t[k] = -INFINITY;
    }
    for (int64_t w0 = fw; w0 <= lw; w0 += 4) {
        Partial pt[4];
        uint4 fv[4][2];   // FEAT: the pieces' top-5 lists, loaded in the same batch
#pragma unroll
        for (int u = 0; u < 4; ++u)
            if (w0 + u <= lw) {
                pt[u] = load_partial(p.partials + r + w0 + u);
                if (FEAT) {
                    fv[u][0] = __ldcg(reinterpret_cast<const uint4 *>(p.feat + r + w0 + u));
                    fv[u][1] = __ldcg(reinterpret_cast<const uint4 *>(p.feat + r + w0 + u) + 1);
                }
            }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            if (w0 + u > lw) break;
            if (w0 + u == fw) g = pt[u].g;
            tok_bad |= pt[u].rank < 0;
            SoftState o;
            o.m = pt[u].m;
            o.r = pt[u].r;
            o.t2 = pt[u].t2;
            o.sh = pt[u].sh;
            o.sl = pt[u].sl;
            o.amax = pt[u].amax;
            o.rank = max(pt[u].rank, 0);
            acc = soft_merge(acc, o);
            if (FEAT) {
                const float f[5] = {__uint_as_float(fv[u][0].x), __uint_as_float(fv[u][0].y),
                                    __uint_as_float(fv[u][0].z), __uint_as_float(fv[u][0].w),
                                    __uint_as_float(fv[u][1].x)};
#pragma unroll
                for (int i = 0; i < 5; ++i) {
                    float z = f[i];
#pragma unroll
                    for (int k = 0; k < 5; ++k) {   // insert z into the descending list
                        const float hi = fmaxf(t[k], z), lo = fminf(t[k], z);
                        t[k] = hi;
                        z = lo;
                    }
                }
            }
        }
    }
}
__device__ __forceinline__ void merge_row(const ScanParams &p, const PartView &pv, int64_t r, SoftState &acc, float &g,
                                          bool &tok_bad) {
    float t[5];
    merge_row_t<false>(p, pv, r, acc, g, tok_bad, t);
}

// Vocabulary-sharded rows: the merged state of row r from the S slices'
// records (slice order), the drafted token's logit from the slice that holds
// it, a token outside [0, V) flagged by any slice, and -- target rows with a
// token -- its rank among the whole row's logits (entries above it, or equal
// at a lower index), counted over the union of the slices' largest entries:
// the kcap largest of the row all lie in that union, so the count is exact
// up to the saturation at kcap.
__device__ __forceinline__ void merge_row_shards(const ScanParams &p, int64_t r, int tok, bool rank, SoftState &acc,
                                                 float &g, bool &tok_bad) {
    acc = soft_identity();
    g = qnan();
    tok_bad = false;
    for (int s = 0; s < p.n_shards; ++s) {
        const sdd_shard_partial *rec = p.shard + static_cast<int64_t>(s) * p.shard_rows + r;
        SoftState o;
        o.m = rec->m;
        o.r = rec->r;
        o.t2 = rec->t2;
        o.sh = rec->sh;
        o.sl = rec->sl;
        o.amax = rec->amax;
        o.rank = 0;
        acc = soft_merge(acc, o);
        const int info = rec->info;
        if (info & 1) g = rec->g;
        if (info & 2) tok_bad = true;
    }
    if (rank && !tok_bad && !isnan(g)) {
        int cnt = 0;
        for (int s = 0; s < p.n_shards; ++s) {
            const sdd_shard_partial *rec = p.shard + static_cast<int64_t>(s) * p.shard_rows + r;
            const int nc = min((rec->info >> 8) & 0xFF, SDD_SHARD_KMAX);
            for (int k = 0; k < nc; ++k) {
                const float z = rec->cz[k];
                cnt += (z > g || (z == g && rec->cv[k] < tok)) ? 1 : 0;
            }
        }
        acc.rank = min(cnt, p.kcap);
    }
}

// Final results of position j of block b (group G) from its merged state, by
// one thread.  `write`: also store the drafter user outputs and raise status
// flags (one CTA per block does).
__device__ __forceinline__ RowFacts row_final(const ScanParams &p, const ScanGroup &G, int j, int b,
                                              const SoftState &acc, float g, bool tok_bad, bool write) {
    const bool has_tok = j < p.gamma;
    const bool tok_ok = has_tok && !tok_bad;
    const float S0 = acc.sh + acc.sl;
    const bool valid = isfinite(acc.m) && acc.m > clamp_floor() && isfinite(S0) && S0 > 0.f;
    const int64_t o = static_cast<int64_t>(b) * p.gamma + j;
    const bool outs = write && G.kind == 0;
    RowFacts f = facts_invalid();
    if (valid) {
        // The lane that held the row maximum M took its term as ex2(y_M) with
        // y_M = M log2(e) - ceil(M log2(e)) (its reference when M arrived).  On a
        // peaked row that one term dominates S, so its MUFU error is replaced
        // by the exact 2^y_M = e0 exp(y_M ln 2 - ln e0) ~ e0 (1 + delta).
        // ln(S + corr) = ln S + corr / S to 2^-43 (|corr / S| < 2^-21), so the
        // two logarithms are independent.
        const float rM = ceilf(acc.m * kLog2e);
        const float yM = fmaf(acc.m, kLog2e, -rM);
        const float e0 = ex2(yM);
        const df ln2 = df{kLn2Hi, kLn2Lo};
        const df lnS0 = ln_df(acc.sh, acc.sl);
        const df delta = df_sub(df_mul_f(ln2, yM), ln_df(e0, 0.f));
        const float corr = e0 * (delta.hi + delta.lo) * pow2f_int(rM - acc.r);
        const float S = S0 + corr;
        // LSE = r ln 2 + ln S (S relative to the reference r)
        const df lnS = df_add(lnS0, df{__fdividef(corr, S0), 0.f});
        f.lse = df_add(df_mul_f(ln2, acc.r), lnS);
        f.M = acc.m;
        f.g = tok_ok ? g : qnan();
        const df dq = df_sub(df{f.g, 0.f}, f.lse);
        f.logq = dq.hi + dq.lo;
        const float eq = expf(dq.hi);
        f.q = fmaf(eq, dq.lo, eq);
        f.argmax = acc.amax;
        f.rank = min(acc.rank, p.kcap);
        if (outs) {
            if (G.q) G.q[o] = f.q;
            if (G.logq) G.logq[o] = f.logq;
            if (G.maxprob) {
                const df dm = df_sub(df{acc.m, 0.f}, f.lse);
                const float em = expf(dm.hi);
                G.maxprob[o] = fmaf(em, dm.lo, em);
            }
            if (G.lse) G.lse[o] = static_cast<double>(f.lse.hi) + static_cast<double>(f.lse.lo);
            // H = ln S' - ln 2 t2 / S with S' = S 2^-dM the sum against the
            // row maximum, dM = M log2(e) - r (a double-float: TwoProd and
            // TwoSum), and t2 already against the maximum: on a peaked row
            // both terms are small, so nothing cancels
            if (G.entropy) {
                const float pm = acc.m * kLog2e;
                const float pe = fmaf(acc.m, kLog2e, -pm);
                float dh, dl;
                two_sum(pm, -acc.r, dh, dl);
                const df ln2df = df{kLn2Hi, kLn2Lo};
                const df dMln2 = df_add(df_mul_f(ln2df, dh), df{(dl + pe) * kLn2, 0.f});
                const df lnSp = df_sub(lnS, dMln2);
                G.entropy[o] = (lnSp.hi + lnSp.lo) - kLn2 * acc.t2 / S;
            }
            if (G.argmax) G.argmax[o] = acc.amax;
        }
    } else {
        if (outs) {
            if (G.q) G.q[o] = qnan();
            if (G.logq) G.logq[o] = qnan();
            if (G.maxprob) G.maxprob[o] = qnan();
            if (G.lse) G.lse[o] = __longlong_as_double(0x7FF8000000000000ll);
            if (G.entropy) G.entropy[o] = qnan();
            if (G.argmax) G.argmax[o] = -1;
        }
        if (write) status_or(p.status, SDD_DEV_NONFINITE);
    }
    if (has_tok && !tok_ok) {
        f.q = f.logq = f.g = qnan();
        f.rank = INT32_MAX;
        if (write) status_or(p.status, SDD_DEV_BAD_TOKEN);
    }
    return f;
}

// Extended features of a drafter row (user index o) from its five largest
// entries t and LSE: margin = p_(1) - p_(2), top5 = p_(1) + ... + p_(5) (an
// entry that is not there contributes exp(-inf) = 0), by one thread.
__device__ __forceinline__ void feat_final(const ScanGroup &G, int64_t o, const float (&t)[5], df lse) {
    float margin = qnan(), top5 = qnan();
    if (!isnan(lse.hi)) {
        float pk[5];
#pragma unroll
        for (int k = 0; k < 5; ++k) {
            const df d = df_sub(df{t[k], 0.f}, lse);
            const float e = expf(d.hi);
            pk[k] = (t[k] == -INFINITY) ? 0.f : fmaf(e, d.lo, e);
        }
        margin = pk[0] - pk[1];
        top5 = (((pk[4] + pk[3]) + pk[2]) + pk[1]) + pk[0];
    }
    if (G.margin) G.margin[o] = margin;
    if (G.top5) G.top5[o] = top5;
}

// ---------------------------------------------------------------------------
// The facts of one block, in shared memory (position j on index j)
// ---------------------------------------------------------------------------
struct BlockFacts {
    // target rows, positions 0..gamma (gamma = bonus row)
    float t_lh[SDD_MAX_GAMMA + 1], t_ll[SDD_MAX_GAMMA + 1], t_M[SDD_MAX_GAMMA + 1], t_g[SDD_MAX_GAMMA + 1];
    int32_t t_am[SDD_MAX_GAMMA + 1], t_rk[SDD_MAX_GAMMA + 1];
    // drafter rows (or, with no drafter rows streamed, the caller's LSE and logit)
    float d_lh[SDD_MAX_GAMMA], d_ll[SDD_MAX_GAMMA], d_g[SDD_MAX_GAMMA], d_q[SDD_MAX_GAMMA], d_lq[SDD_MAX_GAMMA];
    int32_t x[SDD_MAX_GAMMA];       // drafted tokens
    uint8_t guard[SDD_MAX_GAMMA];   // guard flags (0 without a guard array)
};

__device__ __forceinline__ void put_target(BlockFacts &F, int j, const RowFacts &f) {
    F.t_lh[j] = f.lse.hi;
    F.t_ll[j] = f.lse.lo;
    F.t_M[j] = f.M;
    F.t_g[j] = f.g;
    F.t_am[j] = f.argmax;
    F.t_rk[j] = f.rank;
}
__device__ __forceinline__ void put_drafter(BlockFacts &F, int j, const RowFacts &f) {
    F.d_lh[j] = f.lse.hi;
    F.d_ll[j] = f.lse.lo;
    F.d_g[j] = f.g;
    F.d_q[j] = f.q;
    F.d_lq[j] = f.logq;
}

// Rules evaluated per block: rule 0 strict, 1..n_ell lenience, then top-k.
constexpr int kMaxRules = 1 + 2 * SDD_MAX_GRID;

// Acceptance of draft position j (< gamma) of block b under rule r.
__device__ __forceinline__ bool rule_accept(const DecideParams &d, const BlockFacts &F, int r, int j, int b) {
    if (r == 0) {
        if (d.greedy) return F.t_rk[j] == 0;
        // speculative sampling: accept iff u <= min(1, p_t(x_j) / p_d(x_j)), with
        // log r = (g_t - g_d) - (LSE_t - LSE_d)
        const df lr = df_sub(df_diff(F.t_g[j], F.d_g[j]), df_sub(df{F.t_lh[j], F.t_ll[j]}, df{F.d_lh[j], F.d_ll[j]}));
        const float u = philox_uniform(d.seed, static_cast<uint32_t>(j + 1), static_cast<uint32_t>(b), d.round,
                                       kPurposeAccept);
        return df_ge(lr, df{0.f, 0.f}) || (u <= expf(lr.hi));
    }
    if (r <= d.n_ell) {
        const int e = r - 1;
        if (d.ell_one[e]) return F.t_rk[j] == 0;
        return df_ge(df_diff(F.t_g[j], F.t_M[j]), d.ell_thr[e]);   // ln p_t(x_j) - ln max p_t >= ln ell
    }
    return F.t_rk[j] < d.kval[r - 1 - d.n_ell];
}

// First rejected position of rule r (gamma if none), by one warp.
__device__ __forceinline__ int rule_first_reject(const DecideParams &d, const BlockFacts &F, int r, int b, int lane) {
    const int gamma = d.gamma;
    for (int c = 0; c < gamma; c += 32) {
        const int j = c + lane;
        const bool rej = (j < gamma) && !rule_accept(d, F, r, j, b);
        const unsigned bal = __ballot_sync(0xFFFFFFFFu, rej);
        if (bal) return c + __ffs(bal) - 1;
    }
    return gamma;
}

// x_1..x_L, then `corr`, then -1, into a [gamma+1] token list, by one warp.
__device__ __forceinline__ void write_tokens(int lane, int gamma, int32_t *dst, const int32_t *x, int L, int corr) {
    for (int j = lane; j <= gamma; j += 32) dst[j] = (j < L) ? x[j] : (j == L ? corr : -1);
}

// Inclusive prefix sum of one double-float per lane (lane order).
__device__ __forceinline__ df warp_prefix_df(df v, int lane) {
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        df t;
        t.hi = __shfl_up_sync(0xFFFFFFFFu, v.hi, off);
        t.lo = __shfl_up_sync(0xFFFFFFFFu, v.lo, off);
        if (lane >= off) v = df_add(t, v);
    }
    return v;
}

// One chunk (positions c .. c+31, this lane's position j = c + lane, `in` iff
// j < gamma) of the skip policy for one threshold pair.  kb = leading
// positions passing the local gate so far (gamma while no position failed),
// best = largest prefix length meeting Eq. 3 so far; both warp-uniform.
// S = inclusive prefix sum of ln q through position j.
__device__ __forceinline__ void sched_step(int c, int lane, int gamma, bool in, float qj, bool guard_j, const df &S,
                                           const df &eta_loc, const df &log_eta_c, int signal, int &kb, int &best) {
    if (kb < c) return;   // the gate failed in an earlier chunk
    const bool fail = in && (guard_j || !isfinite(qj) || !df_ge(df{qj, 0.f}, eta_loc));
    const unsigned bal = __ballot_sync(0xFFFFFFFFu, fail);
    if (kb == gamma && bal) kb = c + __ffs(bal) - 1;
    if (signal == SDD_SIG_MARGINAL) return;
    const int j = c + lane;
    bool pass = false;
    if (in && j < kb)
        pass = (signal == SDD_SIG_RAW) ? df_ge(S, df_mul_f(log_eta_c, static_cast<float>(j + 1)))
                                       : df_ge(S, log_eta_c);
    const unsigned bal2 = __ballot_sync(0xFFFFFFFFu, pass);
    if (bal2) best = c + 32 - __clz(bal2);
}

// K_hat of the periodic skipping baseline (the appendix's confidence-free
// schedule), by one warp: rounds with round mod period = period - 1 attempt
// K_skip tokens, every other round none; the prefix stops before the first
// guarded position (guarded(j) for position j < gamma).
template <typename Guard>
__device__ __forceinline__ int periodic_khat(int gamma, int period, int K_skip, uint64_t round, Guard guarded,
                                             int lane) {
    if (period < 1 || round % static_cast<uint64_t>(period) != static_cast<uint64_t>(period - 1)) return 0;
    int kb = gamma;
    for (int c = 0; c < gamma; c += 32) {
        const int j = c + lane;
        const unsigned bal = __ballot_sync(0xFFFFFFFFu, j < gamma && guarded(j));
        if (bal) {
            kb = c + __ffs(bal) - 1;
            break;
        }
    }
    return min(K_skip, kb);
}

// K_min / staleness gate of Sec. 4.1 on a block's K_hat.
__device__ __forceinline__ void sched_final(int K_hat, int D, int K_min, int S_max, int &K, int &D_out) {
    K = (D < S_max && K_hat > 0 && K_hat >= K_min) ? K_hat : 0;
    D_out = (K > 0) ? D + K : 0;
}

}  // namespace sdd
