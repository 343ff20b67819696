/*
 * sdd_oracle.c -- plain, slow fp64 CPU oracle for the logits-side path of
 * verifier-skipping speculative diffusion decoding (Luo, Sandler, Fioretto,
 * "From Positionwise Confidence to Prefix Scheduling: Verifier Skipping in
 * Speculative Decoding", arXiv 2608.14787).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call, link or
 * execute this file; only the tests, the smoke check and the benchmark's CPU
 * baseline leg use it.  It shares no code, header, table or constant with the
 * CUDA library.
 *
 * Every quantity is computed in IEEE fp64 with plain loops, in the order the
 * paper states it.  Inputs are converted exactly from bf16 or fp32 to fp64.
 * Build with -ffp-contract=off so that x86-64 and aarch64 round identically.
 *
 * Parity-pinning status of each function is stated in its comment; the pins
 * live in tests/test_oracle_*.py.
 */
#include <math.h>
#include <stdlib.h>
#include <stdint.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* Exact element conversion.                                                 */
/* ------------------------------------------------------------------------ */
enum { ORC_F32 = 0, ORC_BF16 = 1 };

static double orc_load(const void *base, int dtype, int64_t idx) {
    if (dtype == ORC_BF16) {
        uint16_t h = ((const uint16_t *)base)[idx];
        uint32_t bits = ((uint32_t)h) << 16; /* bf16 is the top half of fp32 */
        float f;
        memcpy(&f, &bits, sizeof f);
        return (double)f;
    } else {
        return (double)((const float *)base)[idx];
    }
}

/* ------------------------------------------------------------------------ */
/* Philox4x32-10 counter-based generator (Salmon, Moraes, Dror, Shaw,        */
/* "Parallel random numbers: as easy as 1, 2, 3", SC'11, Sec. 4).  The paper  */
/* under study draws no random numbers of its own (its runs are greedy); the  */
/* sampling rule it cites (Leviathan et al.) needs uniforms, which both this  */
/* oracle and the device library derive from this generator.                */
/* Pinned by the published known-answer vectors (tests/golden/).             */
/* ------------------------------------------------------------------------ */
static void orc_mulhilo32(uint32_t a, uint32_t b, uint32_t *hi, uint32_t *lo) {
    uint64_t p = (uint64_t)a * (uint64_t)b;
    *hi = (uint32_t)(p >> 32);
    *lo = (uint32_t)p;
}

void orc_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2], uint32_t out[4]) {
    /* Multipliers and Weyl key increments as published for Philox-4x32. */
    const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u;
    const uint32_t W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;
    uint32_t c0 = ctr_in[0], c1 = ctr_in[1], c2 = ctr_in[2], c3 = ctr_in[3];
    uint32_t k0 = key_in[0], k1 = key_in[1];
    for (int round = 0; round < 10; ++round) {
        if (round > 0) { /* key schedule: bump before every round but the first */
            k0 += W0;
            k1 += W1;
        }
        uint32_t hi0, lo0, hi1, lo1;
        orc_mulhilo32(M0, c0, &hi0, &lo0);
        orc_mulhilo32(M1, c2, &hi1, &lo1);
        uint32_t n0 = hi1 ^ c1 ^ k0;
        uint32_t n1 = lo1;
        uint32_t n2 = hi0 ^ c3 ^ k1;
        uint32_t n3 = lo0;
        c0 = n0; c1 = n1; c2 = n2; c3 = n3;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* Stream map: key = (seed_lo, seed_hi); counter = (j, b, round_lo,
 * purpose | round_hi << 8).  Word 0 becomes u = ((x >> 8) | 1) * 2^-24, an odd
 * multiple of 2^-24: exactly representable in fp32 and fp64, inside (0, 1). */
double orc_uniform(uint64_t seed, uint32_t j, uint32_t b, uint64_t round, uint32_t purpose) {
    uint32_t ctr[4], key[2], out[4];
    ctr[0] = j;
    ctr[1] = b;
    ctr[2] = (uint32_t)round;
    ctr[3] = (purpose & 0xFFu) | ((uint32_t)(round >> 32) << 8);
    key[0] = (uint32_t)seed;
    key[1] = (uint32_t)(seed >> 32);
    orc_philox4x32_10(ctr, key, out);
    uint32_t odd = (out[0] >> 8) | 1u;
    return ldexp((double)odd, -24);
}

/* Many uniforms at once (a plain loop over orc_uniform, for tests that need
 * millions of draws). */
void orc_uniform_many(int64_t n, uint64_t seed, const uint32_t *j, const uint32_t *b,
                      const uint64_t *round, const uint32_t *purpose, double *out) {
    for (int64_t i = 0; i < n; ++i) out[i] = orc_uniform(seed, j[i], b[i], round[i], purpose[i]);
}

/* ------------------------------------------------------------------------ */
/* Per-row softmax statistics (Sec. 4.2, raw confidence q_j = p_draft(x_j);   */
/* App. A.7 lists top-1 probability and entropy among the drafter features).  */
/* Two-pass plain definition: m = max z, LSE = m + ln sum exp(z - m),         */
/* p(v) = exp(z(v) - LSE), maxprob = exp(m - LSE), H = -sum p ln p,          */
/* argmax = lowest index attaining m, q = p(token), logq = z(token) - LSE.   */
/* Logits are clamped from below at -2^23 (z <- max(z, -2^23); -inf too), so */
/* an entry at or below the floor contributes exp(-2^23 - m), which is 0 in  */
/* fp64 unless the row's maximum m lies within ~745 of the floor.  A row     */
/* with NaN or +inf anywhere, or whose clamped maximum is the floor itself   */
/* (every entry -inf or at most -2^23), has no distribution: all its outputs */
/* are NaN and argmax is -1.                                                 */
/* Pinned by closed forms, by fp64 library softmax/logsumexp/entr, and by    */
/* rows below the floor.                                                     */
/* ------------------------------------------------------------------------ */
static const double orc_floor = -8388608.0; /* -2^23 */

static double orc_clamp(double z) { return (z < orc_floor) ? orc_floor : z; }

void orc_row_stats(const void *logits, int dtype, int64_t n_rows, int64_t V, int64_t row_stride,
                   const int32_t *tokens, /* [n_rows] or NULL */
                   double *out_m, double *out_lse, double *out_q, double *out_logq,
                   double *out_maxprob, double *out_entropy, int32_t *out_argmax) {
    for (int64_t r = 0; r < n_rows; ++r) {
        int64_t base = r * row_stride;
        double m = -INFINITY;
        int64_t amax = -1;
        int bad = 0;
        for (int64_t v = 0; v < V; ++v) {
            double z = orc_load(logits, dtype, base + v);
            if (isnan(z) || (isinf(z) && z > 0)) bad = 1;
            z = orc_clamp(z);
            if (z > m) { m = z; amax = v; }
        }
        if (!(m > orc_floor)) bad = 1;
        int64_t tok = tokens ? (int64_t)tokens[r] : -1;
        if (tokens && (tok < 0 || tok >= V)) bad = 1;
        if (bad) {
            if (out_m) out_m[r] = NAN;
            if (out_lse) out_lse[r] = NAN;
            if (out_q) out_q[r] = NAN;
            if (out_logq) out_logq[r] = NAN;
            if (out_maxprob) out_maxprob[r] = NAN;
            if (out_entropy) out_entropy[r] = NAN;
            if (out_argmax) out_argmax[r] = -1;
            continue;
        }
        double s = 0.0;
        for (int64_t v = 0; v < V; ++v) s += exp(orc_clamp(orc_load(logits, dtype, base + v)) - m);
        double lse = m + log(s);
        double H = 0.0;
        for (int64_t v = 0; v < V; ++v) {
            double z = orc_clamp(orc_load(logits, dtype, base + v));
            double p = exp(z - lse);
            if (p > 0.0) H -= p * (z - lse);
        }
        if (out_m) out_m[r] = m;
        if (out_lse) out_lse[r] = lse;
        if (out_maxprob) out_maxprob[r] = exp(m - lse);
        if (out_entropy) out_entropy[r] = H;
        if (out_argmax) out_argmax[r] = (int32_t)amax;
        if (tokens) {
            double zt = orc_clamp(orc_load(logits, dtype, base + tok));
            if (out_q) out_q[r] = exp(zt - lse);
            if (out_logq) out_logq[r] = zt - lse;
        } else {
            if (out_q) out_q[r] = NAN;
            if (out_logq) out_logq[r] = NAN;
        }
    }
}

/* ------------------------------------------------------------------------ */
/* Extended pre-verification features of a drafter row (App. A.7's list:    */
/* probability margin and top-5 probability mass; top-1 probability, its    */
/* log and the entropy come from orc_row_stats).  With p_(1) >= p_(2) >= ...  */
/* the probabilities in descending order (ties kept with multiplicity):      */
/*   margin = p_(1) - p_(2)       (p_(2) = 0 when V = 1)                     */
/*   top5   = p_(1) + ... + p_(min(5, V))                                   */
/* Logits are clamped from below at -2^23 as everywhere in the path.  A row  */
/* with NaN or +inf, or with only -inf, has no distribution: NaN features.   */
/* Parity pinned in tests/test_oracle_stats.py (closed forms, a library      */
/* sort + logsumexp).                                                       */
/* ------------------------------------------------------------------------ */
void orc_row_features(const void *logits, int dtype, int64_t n_rows, int64_t V, int64_t row_stride,
                      double *out_margin, double *out_top5) {
    for (int64_t r = 0; r < n_rows; ++r) {
        int64_t base = r * row_stride;
        double top[5] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY, -INFINITY};
        double m = -INFINITY;
        int bad = 0;
        for (int64_t v = 0; v < V; ++v) {
            double z = orc_load(logits, dtype, base + v);
            if (isnan(z) || (isinf(z) && z > 0)) bad = 1;
            z = orc_clamp(z);
            if (z > m) m = z;
        }
        if (!(m > orc_floor)) bad = 1;
        if (bad) {
            out_margin[r] = NAN;
            out_top5[r] = NAN;
            continue;
        }
        double s = 0.0;
        for (int64_t v = 0; v < V; ++v) {
            double z = orc_load(logits, dtype, base + v);
            z = orc_clamp(z);
            s += exp(z - m);
            /* insert z into the descending list of the 5 largest values */
            for (int i = 0; i < 5; ++i) {
                if (z > top[i]) {
                    for (int k = 4; k > i; --k) top[k] = top[k - 1];
                    top[i] = z;
                    break;
                }
            }
        }
        double lse = m + log(s);
        int n = V < 5 ? (int)V : 5;
        double t5 = 0.0;
        for (int i = 0; i < n; ++i) t5 += exp(top[i] - lse);
        double p1 = exp(top[0] - lse), p2 = (V > 1) ? exp(top[1] - lse) : 0.0;
        out_margin[r] = p1 - p2;
        out_top5[r] = t5;
    }
}

/* Normalised probabilities of one row, p(v) = exp(z(v) - LSE) with the     */
/* logits clamped at -2^23 as above, fp64 (the softmax the strict rule's     */
/* residual max(0, p_t - p_d) and bonus draw are built from, Sec. 3.1).      */
/* Pinned against fp64 library softmax on random, peaked and masked rows.   */
void orc_row_probs(const void *logits, int dtype, int64_t V, int64_t offset, double *p) {
    double m = -INFINITY;
    for (int64_t v = 0; v < V; ++v) {
        double z = orc_clamp(orc_load(logits, dtype, offset + v));
        if (z > m) m = z;
    }
    double s = 0.0;
    for (int64_t v = 0; v < V; ++v) s += exp(orc_clamp(orc_load(logits, dtype, offset + v)) - m);
    double lse = m + log(s);
    for (int64_t v = 0; v < V; ++v) p[v] = exp(orc_clamp(orc_load(logits, dtype, offset + v)) - lse);
}

/* Rank of `token` in one row under the order (larger logit first, then lower
 * index first): #{v : z(v) > z(t)} + #{v < t : z(v) = z(t)}.  Rank 0 is the
 * greedy argmax; the top-k rule of App. A.6 (the drafted token is one of the
 * target's k largest logits) is rank < k. */
int64_t orc_rank(const void *logits, int dtype, int64_t V, int64_t offset, int64_t token) {
    double g = orc_load(logits, dtype, offset + token);
    int64_t rank = 0;
    for (int64_t v = 0; v < V; ++v) {
        double z = orc_load(logits, dtype, offset + v);
        if (z > g || (z == g && v < token)) rank += 1;
    }
    return rank;
}

/* ------------------------------------------------------------------------ */
/* Prefix skip policy (Sec. 4.1 Eq. 3 and the commit rule after it; signals  */
/* of Sec. 4.2).  For batch row b with position scores q_1..q_gamma:         */
/*   B_k = min_{j<=k} q_j                                                    */
/*   raw:         C_k = (prod_{j<=k} q_j)^(1/k)                              */
/*   marginal:    C_k = min_{j<=k} q_j   (so both gates use max(eta_b,eta_c))*/
/*   conditional: C_k = prod_{j<=k} q_j                                      */
/*   K_hat = max{k : B_k >= eta_b and C_k >= eta_c and no guarded position   */
/*               among 1..k}, max of the empty set = 0.                      */
/*   Commit: if D >= S_max -> strict (K = 0); else skip iff K_hat > 0 and    */
/*   K_hat >= K_min; a skip sets K = K_hat and D += K, a strict round sets   */
/*   K = 0 and D = 0.  A non-finite score is an invalid score: that position */
/*   is guarded.  force_strict marks a shortened final block.  eta_b >= 1 or */
/*   eta_c >= 1 disables skipping (K_hat = K = 0), so that the threshold     */
/*   limit reproduces Strict SDD exactly even when an fp32 score rounds to 1.*/
/* Signals: 0 raw, 1 marginal, 2 conditional.                                */
/* margin[b] = smallest |compared quantity - its threshold| over the         */
/* comparisons that decide K_hat (+inf when none is made).                   */
/* ------------------------------------------------------------------------ */
void orc_schedule(const double *q, int B, int gamma, int signal, double eta_b, double eta_c,
                  int K_min, int S_max, const uint8_t *guard, const uint8_t *force_strict,
                  const int32_t *D_in, int32_t *K_hat_out, int32_t *K_out, int32_t *D_out,
                  double *margin_out) {
    for (int b = 0; b < B; ++b) {
        const double *qb = q + (int64_t)b * gamma;
        double margin = INFINITY;
        int K_hat = 0;
        int disabled = (force_strict && force_strict[b]) || eta_b >= 1.0 || eta_c >= 1.0;
        if (!disabled) {
            double Bk = INFINITY;      /* running min of q */
            double logsum = 0.0;       /* sum of ln q */
            int blocked = 0;           /* a guarded / invalid position has been passed */
            for (int k = 1; k <= gamma; ++k) {
                double qk = qb[k - 1];
                int guarded = (guard && guard[(int64_t)b * gamma + (k - 1)]) || !isfinite(qk);
                if (guarded) blocked = 1;
                if (blocked) break; /* every longer prefix contains this position */
                if (qk < Bk) Bk = qk;
                logsum += log(qk);
                double Ck;
                if (signal == 0)
                    Ck = exp(logsum / (double)k);
                else if (signal == 1)
                    Ck = Bk;
                else
                    Ck = exp(logsum);
                double eb = (signal == 1) ? fmax(eta_b, eta_c) : eta_b;
                double ec = (signal == 1) ? fmax(eta_b, eta_c) : eta_c;
                int pass_b = Bk >= eb;
                int pass_c = Ck >= ec;
                double mb = fabs(Bk - eb), mc = fabs(Ck - ec);
                if (mb < margin) margin = mb;
                if (pass_b && mc < margin) margin = mc;
                if (!pass_b) break; /* B_k is non-increasing: no longer prefix passes */
                if (pass_c) K_hat = k;
            }
        }
        int D = D_in ? D_in[b] : 0;
        int K = 0;
        if (!disabled && D < S_max && K_hat > 0 && K_hat >= K_min) K = K_hat;
        K_hat_out[b] = K_hat;
        K_out[b] = K;
        if (D_out) D_out[b] = (K > 0) ? D + K : 0;
        if (margin_out) margin_out[b] = margin;
    }
}

/* ------------------------------------------------------------------------ */
/* Periodic skipping baseline (appendix, periodic-skipping paragraph): no    */
/* confidence.  A skip of K_skip tokens is attempted once every P rounds --  */
/* in the rounds with round mod P = P - 1 (reading: P - 1 strict rounds      */
/* precede each attempt) -- and every other round is strict.  The attempt    */
/* meets the guards of the confidence policy: it cannot cover a guarded      */
/* position (the prefix ends before the first one), a shortened final block  */
/* (force_strict) has none, and the commit rule of Sec. 4.1 follows (D >=    */
/* S_max forces strict; skip iff K_hat > 0 and K_hat >= K_min; D += K or D = */
/* 0).  Parity pinned by the closed forms in tests/test_oracle_schedule.py.  */
/* ------------------------------------------------------------------------ */
void orc_schedule_periodic(int B, int gamma, int P, int K_skip, uint64_t round, int K_min, int S_max,
                           const uint8_t *guard, const uint8_t *force_strict, const int32_t *D_in,
                           int32_t *K_hat_out, int32_t *K_out, int32_t *D_out) {
    int attempt = (round % (uint64_t)P) == (uint64_t)(P - 1);
    for (int b = 0; b < B; ++b) {
        int K_hat = 0;
        if (attempt && !(force_strict && force_strict[b])) {
            /* longest prefix of length <= min(K_skip, gamma) with no guarded position */
            int limit = K_skip < gamma ? K_skip : gamma;
            for (int k = 1; k <= limit; ++k) {
                if (guard && guard[(int64_t)b * gamma + (k - 1)]) break;
                K_hat = k;
            }
        }
        int D = D_in ? D_in[b] : 0;
        int K = (D < S_max && K_hat > 0 && K_hat >= K_min) ? K_hat : 0;
        K_hat_out[b] = K_hat;
        K_out[b] = K;
        if (D_out) D_out[b] = (K > 0) ? D + K : 0;
    }
}

/* ------------------------------------------------------------------------ */
/* Inverse-CDF draw over non-negative weights w[0..V) in ascending index     */
/* order: the smallest v with sum_{x<=v} w(x) > u * R, R = sum w.  If        */
/* rounding leaves no such v, the last v with positive weight.  Returns -1   */
/* when R is not positive.  margin = min(|uR - C(v)|, |uR - C(v-1)|) / R.    */
/* Pinned against a library searchsorted on an fp64 cumulative sum.          */
/* ------------------------------------------------------------------------ */
int64_t orc_inverse_cdf(const double *w, int64_t V, double u, double *margin) {
    double R = 0.0;
    for (int64_t v = 0; v < V; ++v) R += w[v];
    if (!(R > 0.0)) {
        if (margin) *margin = INFINITY;
        return -1;
    }
    double target = u * R;
    double cum = 0.0, prev = 0.0;
    int64_t last_pos = -1;
    for (int64_t v = 0; v < V; ++v) {
        if (w[v] > 0.0) last_pos = v;
        prev = cum;
        cum += w[v];
        if (w[v] > 0.0 && cum > target) {
            if (margin) *margin = fmin(fabs(target - cum), fabs(target - prev)) / R;
            return v;
        }
    }
    if (margin) *margin = 0.0;
    return last_pos;
}

/* ------------------------------------------------------------------------ */
/* Strict SDD verification, sampling form (Sec. 3.1: the standard rule of    */
/* speculative decoding, Leviathan et al.).  pt: [gamma+1][V] target         */
/* probabilities (row gamma is the bonus row), pd: [gamma][V] drafter        */
/* probabilities, x: drafted tokens.  For j = 1..gamma accept x_j iff        */
/* u_j <= min(1, pt_j(x_j) / pd_j(x_j)); L = number accepted before the      */
/* first rejection.  If L < gamma the next token is drawn from the residual  */
/* norm(max(0, pt_{L+1} - pd_{L+1})) with u_res (from pt_{L+1} if that       */
/* residual has no mass); if L = gamma a bonus token is drawn from           */
/* pt_{gamma+1} with u_bonus.  Committed = x_1..x_L followed by that token.  */
/* margin = smallest |u_j - r_j| over the compared positions, and the        */
/* inverse-CDF margin of the final draw.                                     */
/* Pinned by exact enumeration of the output law for V <= 8, gamma <= 3.     */
/* ------------------------------------------------------------------------ */
void orc_verify_strict_sample(const double *pt, const double *pd, const int32_t *x, int gamma,
                              int64_t V, const double *u_acc, double u_res, double u_bonus,
                              double *w_scratch, /* [V] caller-provided */
                              int32_t *L_out, int32_t *tokens, double *margin_out) {
    double margin = INFINITY;
    int L = gamma;
    for (int j = 0; j < gamma; ++j) {
        double ptx = pt[(int64_t)j * V + x[j]];
        double pdx = pd[(int64_t)j * V + x[j]];
        double r = (pdx > 0.0) ? ptx / pdx : INFINITY;
        if (isfinite(r) && fabs(u_acc[j] - r) < margin) margin = fabs(u_acc[j] - r);
        if (!(u_acc[j] <= r)) { L = j; break; }
    }
    for (int j = 0; j < L; ++j) tokens[j] = x[j];
    int64_t tok;
    double mcdf = INFINITY;
    if (L < gamma) {
        const double *ptr = pt + (int64_t)L * V, *pdr = pd + (int64_t)L * V;
        double R = 0.0;
        for (int64_t v = 0; v < V; ++v) {
            w_scratch[v] = fmax(0.0, ptr[v] - pdr[v]);
            R += w_scratch[v];
        }
        if (R > 0.0)
            tok = orc_inverse_cdf(w_scratch, V, u_res, &mcdf);
        else
            tok = orc_inverse_cdf(ptr, V, u_res, &mcdf);
    } else {
        tok = orc_inverse_cdf(pt + (int64_t)gamma * V, V, u_bonus, &mcdf);
    }
    if (mcdf < margin) margin = mcdf;
    tokens[L] = (int32_t)tok;
    for (int j = L + 1; j <= gamma; ++j) tokens[j] = -1;
    *L_out = L;
    if (margin_out) *margin_out = margin;
}

/* ------------------------------------------------------------------------ */
/* Greedy-family acceptance on target logits (the paper's runs are greedy,   */
/* Sec. 5.1).  For each position j = 1..gamma the caller supplies           */
/*   rank_j  (orc_rank of x_j in target row j),                              */
/*   gap_j   = z_j(x_j) - max_v z_j(v),                                      */
/* and for each row j = 1..gamma+1 the target argmax.  Rules:                */
/*   mode 0 strict greedy: accept iff x_j is the target argmax (rank 0);     */
/*   mode 1 lenience (App. A.6 Eq. 9): accept iff gap_j >= log(ell), with    */
/*          ell = 1 handled by the strict argmax comparison;                 */
/*   mode 2 top-k (App. A.6): accept iff rank_j < k.                          */
/* The longest accepted prefix is committed, followed by the target argmax   */
/* at the first rejected row, or at the bonus row if all gamma pass.         */
/* margin = smallest |gap_j - log ell| over compared positions (mode 1).      */
/* ------------------------------------------------------------------------ */
void orc_verify_greedy_family(int mode, double param, int gamma, const int32_t *x,
                              const int64_t *rank, const double *gap, const int32_t *target_argmax,
                              int32_t *L_out, int32_t *tokens, double *margin_out) {
    double margin = INFINITY;
    int L = gamma;
    double log_ell = (mode == 1) ? log(param) : 0.0;
    for (int j = 0; j < gamma; ++j) {
        int ok;
        if (mode == 0) {
            ok = rank[j] == 0;
        } else if (mode == 1) {
            if (param == 1.0) {
                ok = rank[j] == 0;
            } else {
                double d = fabs(gap[j] - log_ell);
                if (d < margin) margin = d;
                ok = gap[j] >= log_ell;
            }
        } else {
            ok = rank[j] < (int64_t)param;
        }
        if (!ok) { L = j; break; }
    }
    for (int j = 0; j < L; ++j) tokens[j] = x[j];
    tokens[L] = target_argmax[L];
    for (int j = L + 1; j <= gamma; ++j) tokens[j] = -1;
    *L_out = L;
    if (margin_out) *margin_out = margin;
}

/* ------------------------------------------------------------------------ */
/* Agreement with strict verification (Sec. 3.2, Eq. 1 and Eq. 2).  Over the */
/* rounds A with K_b > 0: sum min(K_b, L_b), sum K_b, count of K_b <= L_b,   */
/* and |A|.  StrictToken = acc[0]/acc[1], FullPrefix = acc[2]/acc[3].        */
/* ------------------------------------------------------------------------ */
void orc_agreement(const int32_t *K, const int32_t *L, int B, int64_t acc[4]) {
    for (int b = 0; b < B; ++b) {
        if (K[b] <= 0) continue;
        acc[0] += (K[b] < L[b]) ? K[b] : L[b];
        acc[1] += K[b];
        acc[2] += (K[b] <= L[b]) ? 1 : 0;
        acc[3] += 1;
    }
}

/* ------------------------------------------------------------------------ */
/* Stand-in survival scorer of the decode-loop workload: per position, from   */
/* the drafter hidden state h (K values), s = sigmoid(w2 . GELU(W1 h + b1) +  */
/* b2) with N hidden units, GELU(z) = z Phi(z) = z (1 + erf(z / sqrt 2)) / 2. */
/* The paper's learned scorer (App. A.7) has this form with more layers and   */
/* trained weights; the stand-in is random-init.  W1 is [N, K] (one row per  */
/* hidden unit), h is [M, K]; both bf16 bits, converted exactly.             */
/* ------------------------------------------------------------------------ */
void orc_survival_mlp(const uint16_t *h, int M, int K, const uint16_t *W1, const float *b1, const uint16_t *w2,
                      double b2, int N, double *out) {
    for (int m = 0; m < M; ++m) {
        double t = b2;
        for (int n = 0; n < N; ++n) {
            double z = (double)b1[n];
            for (int k = 0; k < K; ++k)
                z += orc_load(W1, ORC_BF16, (int64_t)n * K + k) * orc_load(h, ORC_BF16, (int64_t)m * K + k);
            const double gelu = 0.5 * z * (1.0 + erf(z / sqrt(2.0)));
            t += orc_load(w2, ORC_BF16, n) * gelu;
        }
        out[m] = 1.0 / (1.0 + exp(-t));
    }
}

/* ------------------------------------------------------------------------ */
/* The learned scorer's shape (App. A.7): an MLP K -> N -> N -> N -> 1 with   */
/* GELU hidden layers, on the concatenated input x = [hidden state ; scalar  */
/* features] (K = 3584 + 19 in the paper), random-init stand-in weights:     */
/*   a1 = GELU(W1 x + b1), a2 = GELU(W2 a1 + b2), a3 = GELU(W3 a2 + b3),      */
/*   s  = sigmoid(w4 . a3 + b4).                                             */
/* Every activation stays in fp64: the paper fixes no precision for the     */
/* scorer (dropout is a training-time op and is absent here).  W1 is [N, K], */
/* W2 and W3 [N, N] (one row per output unit), w4 [N]: bf16 bits.            */
/* Pinned in tests/test_oracle_mlp.py (closed forms of single-path nets,     */
/* zero weights, hidden-unit permutation invariance, a library fp64 chain). */
/* ------------------------------------------------------------------------ */
static double orc_gelu(double z) { return 0.5 * z * (1.0 + erf(z / sqrt(2.0))); }

void orc_scorer_deep(const uint16_t *x, int M, int K, const uint16_t *W1, const float *b1, const uint16_t *W2,
                     const float *b2, const uint16_t *W3, const float *b3, const uint16_t *w4, double b4, int N,
                     double *out, double *a1, double *a2) {
    /* a1, a2: caller scratch of N doubles each */
    for (int m = 0; m < M; ++m) {
        for (int n = 0; n < N; ++n) {
            double z = (double)b1[n];
            for (int k = 0; k < K; ++k)
                z += orc_load(W1, ORC_BF16, (int64_t)n * K + k) * orc_load(x, ORC_BF16, (int64_t)m * K + k);
            a1[n] = orc_gelu(z);
        }
        for (int n = 0; n < N; ++n) {
            double z = (double)b2[n];
            for (int k = 0; k < N; ++k) z += orc_load(W2, ORC_BF16, (int64_t)n * N + k) * a1[k];
            a2[n] = orc_gelu(z);
        }
        double t = b4;
        for (int n = 0; n < N; ++n) {
            double z = (double)b3[n];
            for (int k = 0; k < N; ++k) z += orc_load(W3, ORC_BF16, (int64_t)n * N + k) * a2[k];
            t += orc_load(w4, ORC_BF16, n) * orc_gelu(z);
        }
        out[m] = 1.0 / (1.0 + exp(-t));
    }
}

/* ------------------------------------------------------------------------ */
/* Permutation diagnostic (Sec. 5, H1 mechanism, Table 1) on logged blocks:  */
/* scores q[B][gamma] (fp64), strict accepted lengths L[B].  For each        */
/* repetition r and position j (1-based), the blocks valid at j -- all for   */
/* the raw and marginal signals, those with L >= j - 1 for the conditional   */
/* one -- exchange their (score, label) pairs by a uniformly random          */
/* permutation; the others keep theirs.  The feasible prefix length of every */
/* block is then K_hat of orc_schedule for (eta_b, eta_c) (the gates before  */
/* K_min or staleness).  sums[r] = sum of the feasible prefixes under        */
/* permutation r; sums[n_rep] = the sum in the logged order.                 */
/* The permutation of (r, j): the valid blocks in index order, shuffled by   */
/* Fisher-Yates from the top; slot i swaps with floor(w (i+1) / 2^32), w the */
/* first Philox4x32-10 word of key seed and counter (i, j - 1, r, 3).  The   */
/* t-th valid block takes the score of the t-th entry of the shuffle.        */
/* Parity pinned in tests/test_oracle_diag.py (column-constant and identical */
/* rows are invariant, permutations preserve every column's multiset, a      */
/* closed form of the independent-position expectation).                    */
/* ------------------------------------------------------------------------ */
/* The shuffle of (r, j) on its own: perm[0..n) starts as 0..n-1 and slot i */
/* (from n - 1 down to 1) swaps with k = floor(w (i + 1) / 2^32), w the first */
/* Philox word of counter (i, j0, r, 3), so k is uniform on 0..i (Fisher-    */
/* Yates; Durstenfeld's in-place form).  j0 = j - 1 is the 0-based position. */
/* Pinned by a chi-square test over all n! permutations for n <= 4.          */
void orc_shuffle(int n, uint64_t seed, int j0, int r, int32_t *perm) {
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    for (int t = 0; t < n; ++t) perm[t] = t;
    for (int i = n - 1; i > 0; --i) {
        uint32_t ctr[4] = {(uint32_t)i, (uint32_t)j0, (uint32_t)r, 3u}, out[4];
        orc_philox4x32_10(ctr, key, out);
        int k = (int)(((uint64_t)out[0] * (uint64_t)(i + 1)) >> 32);
        int32_t tmp = perm[i];
        perm[i] = perm[k];
        perm[k] = tmp;
    }
}

void orc_permutation_diagnostic(const double *q, const int32_t *L, int B, int gamma, int signal, double eta_b,
                                double eta_c, int n_rep, uint64_t seed, int64_t *sums, double *qp, int32_t *list,
                                int32_t *Khat, int32_t *K, int32_t *D) {
    /* qp: scratch [B * gamma]; list: scratch [B]; Khat, K, D: scratch [B] */
    for (int r = 0; r <= n_rep; ++r) {
        for (int b = 0; b < B; ++b)
            for (int j = 0; j < gamma; ++j) qp[(int64_t)b * gamma + j] = q[(int64_t)b * gamma + j];
        if (r < n_rep) {
            for (int j = 0; j < gamma; ++j) {
                int n = 0;
                for (int b = 0; b < B; ++b)
                    if (signal != 2 || L[b] >= j) list[n++] = b;
                int32_t *perm = (int32_t *)malloc(sizeof(int32_t) * (n > 0 ? n : 1));
                orc_shuffle(n, seed, j, r, perm);
                /* the t-th valid block takes the score of valid block perm[t] */
                for (int t = 0; t < n; ++t)
                    qp[(int64_t)list[t] * gamma + j] = q[(int64_t)list[perm[t]] * gamma + j];
                free(perm);
            }
        }
        orc_schedule(qp, B, gamma, signal, eta_b, eta_c, 0, 0x7FFFFFFF, NULL, NULL, NULL, Khat, K, D, NULL);
        int64_t sum = 0;
        for (int b = 0; b < B; ++b) sum += Khat[b];
        sums[r] = sum;
    }
}
