// rules.cuh -- warp-level decisions for one block of gamma draft positions,
// evaluated by the warp that finalises the block's last row (inside the
// streaming kernel) or by the stand-alone schedule kernel.
//
//  * schedule_block -- the skip policy of Sec. 4.1: Eq. 3 with the three
//    confidence signals of Sec. 4.2, then K_min / staleness / guards.
//  * block_decide   -- Strict SDD (Sec. 3.1: greedy, or the acceptance test of
//    the speculative-sampling rule it cites), lenience (App. A.6 Eq. 9), top-k
//    (App. A.6), the schedule of a fused round, the agreement counters of
//    Sec. 3.2 (Eq. 1-2) and the tokens committed by skipped blocks.
#pragma once

#include "internal.h"

namespace sdd {

__device__ __forceinline__ float qnan() { return __int_as_float(0x7FC00000); }

// A row record written by another SM during this launch: read through L2.
__device__ __forceinline__ RowRec load_rec(const RowRec *p) {
    union {
        uint4 v[2];
        RowRec r;
    } u;
    u.v[0] = __ldcg(reinterpret_cast<const uint4 *>(p));
    u.v[1] = __ldcg(reinterpret_cast<const uint4 *>(p) + 1);
    return u.r;
}

template <int DT>
__device__ __forceinline__ float logit_at(const char *rowp, int v) {
    if (DT == SDD_BF16) {
        const uint16_t h = __ldg(reinterpret_cast<const unsigned short *>(rowp) + v);
        return __uint_as_float(static_cast<uint32_t>(h) << 16);
    } else {
        return __ldg(reinterpret_cast<const float *>(rowp) + v);
    }
}

// Skip policy for one block and one threshold pair, by one warp.  q and logq
// (nullable) are read at q[j * stride] for the block's gamma positions; guard
// is nullable.
__device__ __forceinline__ void schedule_block(int lane, int gamma, const float *q, const float *logq, int stride,
                                               const uint8_t *guard, bool off, int D, int signal, double eta_loc,
                                               double log_eta_c, int K_min, int S_max, int &K_hat, int &K,
                                               int &D_out) {
    if (off) {
        K_hat = 0;
        K = 0;
        D_out = 0;
        return;
    }
    // local gate and guards: kb = number of leading positions that pass
    int kb = gamma;
    for (int c = 0; c < gamma; c += 32) {
        const int j = c + lane;
        bool fail = false;
        if (j < gamma) {
            const float qj = __ldcg(q + static_cast<int64_t>(j) * stride);
            fail = (guard && guard[j]) || !isfinite(qj) || !(static_cast<double>(qj) >= eta_loc);
        }
        const unsigned bal = __ballot_sync(0xFFFFFFFFu, fail);
        if (bal) {
            kb = c + __ffs(bal) - 1;
            break;
        }
    }
    int best = 0;
    if (signal == SDD_SIG_MARGINAL) {
        best = kb;
    } else {
        // prefix sums of ln q in fp64; raw: S_k >= k ln eta_c, conditional: S_k >= ln eta_c
        double carry = 0.0;
        for (int c = 0; c < kb; c += 32) {
            const int j = c + lane;
            double v = 0.0;
            if (j < kb)
                v = logq ? static_cast<double>(__ldcg(logq + static_cast<int64_t>(j) * stride))
                         : static_cast<double>(logf(__ldcg(q + static_cast<int64_t>(j) * stride)));
#pragma unroll
            for (int off2 = 1; off2 < 32; off2 <<= 1) {
                const double t = __shfl_up_sync(0xFFFFFFFFu, v, off2);
                if (lane >= off2) v += t;
            }
            const double Sk = carry + v;
            const bool pass = (j < kb) && ((signal == SDD_SIG_RAW) ? (Sk >= static_cast<double>(j + 1) * log_eta_c)
                                                                    : (Sk >= log_eta_c));
            const unsigned bal = __ballot_sync(0xFFFFFFFFu, pass);
            if (bal) best = c + 32 - __clz(bal);
            carry = __shfl_sync(0xFFFFFFFFu, Sk, 31);
        }
    }
    K_hat = best;
    K = (D < S_max && best > 0 && best >= K_min) ? best : 0;
    D_out = (K > 0) ? D + K : 0;
}

// First failing position (0-based) of a per-position acceptance predicate,
// gamma if none fails.
template <class Accept>
__device__ __forceinline__ int first_reject(int lane, int gamma, Accept accept) {
    for (int c = 0; c < gamma; c += 32) {
        const int j = c + lane;
        const bool fail = (j < gamma) && !accept(j);
        const unsigned bal = __ballot_sync(0xFFFFFFFFu, fail);
        if (bal) return c + __ffs(bal) - 1;
    }
    return gamma;
}

// x_1..x_L, then `corr`, then -1, into a [gamma+1] token list.
__device__ __forceinline__ void write_tokens(int lane, int gamma, int32_t *dst, const int32_t *xb, int L, int corr) {
    for (int j = lane; j <= gamma; j += 32) dst[j] = (j < L) ? __ldg(xb + j) : (j == L ? corr : -1);
}

// Rules evaluated together, one chunk of 32 positions at a time: the block's
// records are read once per chunk and every rule tests its acceptance on them;
// a rule's correction token (the target argmax at its first rejection) is
// taken from the lane holding that position.
constexpr int kMaxRules = 1 + 2 * SDD_MAX_GRID;

template <int DT>
__device__ void block_decide(const DecideParams &p, int i, int lane, int *s_L, int *s_corr) {
    const int gamma = p.gamma;
    const int b = p.bidx ? __ldg(p.bidx + i) : i;
    if (b < 0 || b >= p.B) return;   // flagged by the streaming pass
    const RowRec *tr = p.trec + static_cast<int64_t>(i) * (gamma + 1);
    const int32_t *xb = p.tokens + static_cast<int64_t>(b) * gamma;
    const int64_t bo = static_cast<int64_t>(b) * (gamma + 1);
    const bool sampling = p.do_strict && !p.greedy;
    // rule r: 0 strict, 1..n_ell lenience, then top-k
    const int n_rules = 1 + p.n_ell + p.n_k;
    for (int r = lane; r < n_rules; r += 32) s_L[r] = -1;
    __syncwarp();
    const int bonus_argmax = load_rec(tr + gamma).argmax;
    int remaining = (p.do_strict ? 1 : 0) + p.n_ell + p.n_k;
    for (int c = 0; c < gamma && remaining > 0; c += 32) {
        const int j = c + lane;
        const bool in = j < gamma;
        RowRec t{};
        if (in) t = load_rec(tr + j);
        auto settle = [&](int r, bool accept) {
            if (s_L[r] >= 0) return;
            const unsigned bal = __ballot_sync(0xFFFFFFFFu, in && !accept);
            if (bal) {
                const int f = __ffs(bal) - 1;
                const int corr = __shfl_sync(0xFFFFFFFFu, t.argmax, f);
                if (lane == 0) {
                    s_L[r] = c + f;
                    s_corr[r] = corr;
                }
                __syncwarp();
                --remaining;
            }
        };
        if (p.do_strict) {
            bool acc = true;
            if (in) {
                if (!sampling) {
                    acc = t.rank == 0;
                } else {
                    double lse_d;
                    float gd;
                    if (p.drec) {
                        const RowRec d = load_rec(p.drec + static_cast<int64_t>(i) * gamma + j);
                        lse_d = d.lse;
                        gd = d.g;
                    } else {
                        const int xj = __ldg(xb + j);
                        const char *zdr = p.zd + (static_cast<int64_t>(b) * gamma + j) * p.stride_bytes;
                        lse_d = __ldg(p.d_lse + static_cast<int64_t>(b) * gamma + j);
                        gd = (xj >= 0 && xj < p.V) ? fmax_nan(logit_at<DT>(zdr, xj), clamp_floor()) : qnan();
                    }
                    // log r = log p_t(x_j) - log p_d(x_j) = (g_t - g_d) - (LSE_t - LSE_d)
                    const double lr = static_cast<double>(t.g - gd) - (t.lse - lse_d);
                    const float u = philox_uniform(p.seed, static_cast<uint32_t>(j + 1), static_cast<uint32_t>(b),
                                                   p.round, kPurposeAccept);
                    acc = (lr >= 0.0) || (u <= expf(static_cast<float>(lr)));
                }
            }
            settle(0, acc);
        }
        for (int r = 0; r < p.n_ell; ++r)
            settle(1 + r, p.ell_one[r] ? (t.rank == 0) : (static_cast<double>(t.g - t.M) >= p.ell_thr[r]));
        for (int r = 0; r < p.n_k; ++r) settle(1 + p.n_ell + r, t.rank < p.kval[r]);
    }
    __syncwarp();
    auto rule_L = [&](int r) { return s_L[r] >= 0 ? s_L[r] : gamma; };
    auto rule_corr = [&](int r) { return s_L[r] >= 0 ? s_corr[r] : bonus_argmax; };
    // ---- outputs of the rules ----
    int L = gamma;
    if (p.do_strict) {
        L = rule_L(0);
        if (!sampling) {
            if (lane == 0) {
                if (p.L_strict) p.L_strict[b] = L;
                if (p.n_strict) p.n_strict[b] = L + 1;
            }
            if (p.tok_strict) write_tokens(lane, gamma, p.tok_strict + bo, xb, L, rule_corr(0));
        } else if (lane == 0) {
            p.blk_L[i] = L;   // the draw kernel completes the block
        }
    }
    for (int r = 0; r < p.n_ell; ++r) {
        const int Lr = rule_L(1 + r);
        const int64_t o = static_cast<int64_t>(r) * p.B + b;
        if (lane == 0) {
            if (p.L_len) p.L_len[o] = Lr;
            if (p.n_len) p.n_len[o] = Lr + 1;
        }
        if (p.tok_len) write_tokens(lane, gamma, p.tok_len + o * (gamma + 1), xb, Lr, rule_corr(1 + r));
    }
    for (int r = 0; r < p.n_k; ++r) {
        const int Lr = rule_L(1 + p.n_ell + r);
        const int64_t o = static_cast<int64_t>(r) * p.B + b;
        if (lane == 0) {
            if (p.L_topk) p.L_topk[o] = Lr;
            if (p.n_topk) p.n_topk[o] = Lr + 1;
        }
        if (p.tok_topk) write_tokens(lane, gamma, p.tok_topk + o * (gamma + 1), xb, Lr, rule_corr(1 + p.n_ell + r));
    }
    // ---- fused round: schedule, agreement, tokens of skipped blocks ----
    if (p.do_sched) {
        const RowRec *dr = p.drec + static_cast<int64_t>(i) * gamma;
        const bool force = p.force_strict && p.force_strict[b];
        const int D = p.D_in ? p.D_in[b] : 0;
        const float *qv = &dr->q;
        const float *lqv = &dr->logq;
        constexpr int kRecFloats = sizeof(RowRec) / sizeof(float);
        for (int t = 0; t < p.n_tau; ++t) {
            int Kh, K, Do;
            schedule_block(lane, gamma, qv, lqv, kRecFloats, p.guard ? p.guard + static_cast<int64_t>(b) * gamma : nullptr,
                           force || p.tau_off[t], D, p.signal, p.eta_loc[t], p.log_eta_c[t], p.K_min, p.S_max, Kh, K,
                           Do);
            if (lane == 0) {
                const int64_t o = static_cast<int64_t>(t) * p.B + b;
                if (p.K_hat) p.K_hat[o] = Kh;
                if (p.K) p.K[o] = K;
                if (p.D_out) p.D_out[o] = Do;
                if (p.agreement && K > 0 && p.do_strict) {
                    unsigned long long *a = reinterpret_cast<unsigned long long *>(p.agreement + 4 * t);
                    atomicAdd(a + 0, static_cast<unsigned long long>(min(K, L)));
                    atomicAdd(a + 1, static_cast<unsigned long long>(K));
                    atomicAdd(a + 2, static_cast<unsigned long long>(K <= L ? 1 : 0));
                    atomicAdd(a + 3, 1ull);
                }
            }
            if (t == 0) {
                if (lane == 0) p.k0[i] = K;   // read by the draw kernel
                const bool skip = K > 0;
                if (skip || (p.do_strict && !sampling)) {
                    // skipped: x_1..x_K; greedy strict: the verified tokens
                    const int Lc = skip ? K : L;
                    const int corr = skip ? -1 : rule_corr(0);
                    if (lane == 0 && p.commit_n) p.commit_n[b] = skip ? K : L + 1;
                    if (p.commit_tokens) write_tokens(lane, gamma, p.commit_tokens + bo, xb, Lc, corr);
                }
            }
        }
    }
}

}  // namespace sdd
