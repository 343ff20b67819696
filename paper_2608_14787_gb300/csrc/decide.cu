// decide.cu -- the per-block decisions of the path, after the streaming pass.
//
//  * schedule_block   -- the skip policy of Sec. 4.1 (Eq. 3, K_min, staleness)
//                        with the three confidence signals of Sec. 4.2.
//  * decide_kernel    -- acceptance under Strict SDD (Sec. 3.1; greedy, or the
//                        speculative-sampling rule it cites), lenience (App. A.6
//                        Eq. 9) and top-k (App. A.6) from the target facts; the
//                        residual / bonus inverse-CDF draw of the sampling rule
//                        split over several CTAs per block; and, for a fused
//                        round, the schedule, the committed tokens and the
//                        agreement counters of Sec. 3.2 (Eq. 1-2).
//  * schedule_kernel, agreement_kernel, commit_kernel -- the same pieces as
//                        stand-alone entry points.
#include "internal.h"

namespace sdd {

namespace {

__device__ __forceinline__ float nanf_() { return __int_as_float(0x7FC00000); }

// Skip policy for one block and one threshold pair, by one warp.
// q, logq (nullable), guard (nullable) point at the block's gamma positions.
__device__ void schedule_block(int lane, int gamma, const float *q, const float *logq, const uint8_t *guard,
                               bool off, int D, int signal, double eta_loc, double log_eta_c, int K_min,
                               int S_max, int &K_hat, int &K, int &D_out) {
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
            const float qj = q[j];
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
            if (j < kb) v = logq ? static_cast<double>(logq[j]) : static_cast<double>(logf(q[j]));
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

template <int DT>
__device__ __forceinline__ float load_logit(const char *rowp, int v) {
    if (DT == SDD_BF16) {
        const uint16_t h = __ldg(reinterpret_cast<const unsigned short *>(rowp) + v);
        return __uint_as_float(static_cast<uint32_t>(h) << 16);
    } else {
        return __ldg(reinterpret_cast<const float *>(rowp) + v);
    }
}

// Weights of the sampling draw for the EPV entries of one 16-byte vector.
//   residual: p_t - p_d = p_d (exp(D(v)) - 1) with the log-ratio
//             D(v) = (z_t(v) - z_d(v)) - (LSE_t - LSE_d); the LSE difference is
//             applied as two fp32 terms (hi + lo) and the difference by expm1, so
//             no cancellation between near-equal p_t and p_d loses precision;
//             p_d(v) = 2^(z_d(v) log2(e) - r_d) up to the common factor of the row;
//   bonus (zd_row == nullptr): 2^(z_t(v) log2(e) - r_t).
// Returns the fp32 sum of the entries in ascending order (the draw and the
// totals use this same order).
template <int DT>
__device__ __forceinline__ float vec_weights(const char *zt_row, const char *zd_row, int vec, int V, float nrt,
                                             float nrd, float d_hi, float d_lo, float (&w)[8]) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    const uint4 a = __ldg(reinterpret_cast<const uint4 *>(zt_row) + vec);
    uint4 d = make_uint4(0, 0, 0, 0);
    if (zd_row) d = __ldg(reinterpret_cast<const uint4 *>(zd_row) + vec);
    const uint32_t *ua = reinterpret_cast<const uint32_t *>(&a);
    const uint32_t *ud = reinterpret_cast<const uint32_t *>(&d);
    float sum = 0.f;
#pragma unroll
    for (int e = 0; e < EPV; ++e) {
        float zt, zd;
        if (DT == SDD_BF16) {
            zt = (e & 1) ? bf16_hi(ua[e >> 1]) : bf16_lo(ua[e >> 1]);
            zd = (e & 1) ? bf16_hi(ud[e >> 1]) : bf16_lo(ud[e >> 1]);
        } else {
            zt = __uint_as_float(ua[e]);
            zd = __uint_as_float(ud[e]);
        }
        zt = fmax_nan(zt, clamp_floor());
        zd = fmax_nan(zd, clamp_floor());
        float wv;
        if (zd_row) {
            const float dv = ((zt - zd) - d_hi) - d_lo;
            wv = (dv > 0.f) ? ex2(fmaf(zd, kLog2e, nrd)) * expm1f(dv) : 0.f;
        } else {
            wv = ex2(fmaf(zt, kLog2e, nrt));
        }
        if (vec * EPV + e >= V) wv = 0.f;
        w[e] = wv;
        sum += wv;
    }
    return sum;
}

// Inclusive block scan of one double per thread (kResidThreads threads).
__device__ __forceinline__ double block_incl_scan(double v, double *warp_tot, double &block_total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const double t = __shfl_up_sync(0xFFFFFFFFu, v, off);
        if (lane >= off) v += t;
    }
    if (lane == 31) warp_tot[warp] = v;
    __syncthreads();
    double base = 0.0, tot = 0.0;
    for (int w = 0; w < kResidThreads / 32; ++w) {
        if (w < warp) base += warp_tot[w];
        tot += warp_tot[w];
    }
    __syncthreads();
    block_total = tot;
    return base + v;
}

struct DrawCtx {
    const char *zt_row, *zd_row;
    float nrt, nrd, d_hi, d_lo;
};

// One pass over vectors [v0, v1) of the draw row.  With find == false returns
// the weight total (and the last positive index); with find == true returns
// the index of the first entry whose running sum exceeds `target` (or -1).
template <int DT>
__device__ double draw_pass(const DrawCtx &c, int v0, int v1, int V, bool find, double target, int &last_pos,
                            int &found, double *warp_tot, int *s_first) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    double carry = 0.0;
    last_pos = -1;
    found = -1;
    for (int base = v0; base < v1; base += kResidThreads) {
        const int vec = base + threadIdx.x;
        float w[8];
        float vs_f = 0.f;
        if (vec < v1) vs_f = vec_weights<DT>(c.zt_row, c.zd_row, vec, V, c.nrt, c.nrd, c.d_hi, c.d_lo, w);
        if (vec < v1)
            for (int e = 0; e < EPV; ++e)
                if (w[e] > 0.f) last_pos = vec * EPV + e;
        const double vs = static_cast<double>(vs_f);
        double tot;
        const double incl = block_incl_scan(vs, warp_tot, tot);
        if (find) {
            if (threadIdx.x == 0) *s_first = INT32_MAX;
            __syncthreads();
            if (vec < v1 && carry + incl > target) atomicMin(s_first, static_cast<int>(threadIdx.x));
            __syncthreads();
            const int tf = *s_first;
            if (tf != INT32_MAX) {
                if (static_cast<int>(threadIdx.x) == tf) {
                    const double before = carry + (incl - vs);
                    float part = 0.f;
                    int pick = -1, lastp = -1;
                    for (int e = 0; e < EPV; ++e) {
                        if (w[e] > 0.f) lastp = vec * EPV + e;
                        part += w[e];
                        if (w[e] > 0.f && before + static_cast<double>(part) > target) {
                            pick = vec * EPV + e;
                            break;
                        }
                    }
                    *s_first = (pick >= 0) ? pick : lastp;
                }
                __syncthreads();
                found = *s_first;
                __syncthreads();
                return carry;
            }
        }
        carry += tot;
    }
    return carry;
}

// Draw-row context from the two rows' fp64 log-normalisers.
__device__ __forceinline__ DrawCtx draw_ctx(const char *zt_row, const char *zd_row, double lse_t, double lse_d) {
    DrawCtx c;
    c.zt_row = zt_row;
    c.zd_row = zd_row;
    c.nrt = -ceilf(static_cast<float>(lse_t * kLog2ed));
    c.nrd = 0.f;
    c.d_hi = 0.f;
    c.d_lo = 0.f;
    if (zd_row) {
        c.nrd = -ceilf(static_cast<float>(lse_d * kLog2ed));
        const double D = lse_t - lse_d;
        c.d_hi = static_cast<float>(D);
        c.d_lo = static_cast<float>(D - static_cast<double>(c.d_hi));
    }
    return c;
}

template <int DT>
__global__ void __launch_bounds__(kResidThreads) decide_kernel(const __grid_constant__ DecideParams p) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    const int i = blockIdx.x;     // listed block
    const int seg = blockIdx.y;   // residual segment
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int gamma = p.gamma;
    int b = p.bidx ? __ldg(p.bidx + i) : i;
    const bool b_ok = (b >= 0 && b < p.B);
    if (!b_ok) {
        if (seg == 0 && threadIdx.x == 0) status_or(p.status, SDD_DEV_BAD_TOKEN);
        return;
    }
    const RowRec *tr = p.trec + static_cast<int64_t>(i) * (gamma + 1);
    const int32_t *xb = p.tokens + static_cast<int64_t>(b) * gamma;

    __shared__ int s_L;              // strict accepted length
    __shared__ double s_lse[2];      // LSE of the target and drafter draw rows
    __shared__ double s_warp[kResidThreads / 32];
    __shared__ int s_first;
    __shared__ double s_tot[kResidMaxSeg];
    __shared__ int s_last[kResidMaxSeg];

    // ---- acceptance decisions (warp 0) ----
    if (warp == 0) {
        int L = gamma;
        if (p.do_strict) {
            for (int c = 0; c < gamma; c += 32) {
                const int j = c + lane;
                bool fail = false;
                if (j < gamma) {
                    const RowRec t = tr[j];
                    if (p.greedy) {
                        fail = !(t.rank == 0);
                    } else {
                        double lse_d;
                        float gd;
                        if (p.drec) {
                            const RowRec d = p.drec[static_cast<int64_t>(i) * gamma + j];
                            lse_d = d.lse;
                            gd = d.g;
                        } else {
                            const char *zdr = p.zd + (static_cast<int64_t>(b) * gamma + j) * p.stride_bytes;
                            const int xj = xb[j];
                            lse_d = __ldg(p.d_lse + static_cast<int64_t>(b) * gamma + j);
                            gd = (xj >= 0 && xj < p.V) ? fmax_nan(load_logit<DT>(zdr, xj), clamp_floor()) : nanf_();
                        }
                        // log r = log p_t(x_j) - log p_d(x_j) = (g_t - g_d) - (LSE_t - LSE_d), in fp64
                        const double lr = (static_cast<double>(t.g) - static_cast<double>(gd)) - (t.lse - lse_d);
                        const float u = philox_uniform(p.seed, static_cast<uint32_t>(j + 1), static_cast<uint32_t>(b),
                                                       p.round, kPurposeAccept);
                        const bool acc = (lr >= 0.0) || (u <= expf(static_cast<float>(lr)));
                        fail = !acc;
                    }
                }
                const unsigned bal = __ballot_sync(0xFFFFFFFFu, fail);
                if (bal) {
                    L = c + __ffs(bal) - 1;
                    break;
                }
            }
            if (lane == 0) s_L = L;
        }
        // greedy-family rules are complete here: write them from segment 0
        if (seg == 0) {
            auto emit = [&](int32_t *Lp, int32_t *tok, int32_t *np, int Lr) {
                const int corr = tr[Lr].argmax;
                if (lane == 0) {
                    if (Lp) Lp[b] = Lr;
                    if (np) np[b] = Lr + 1;
                }
                if (tok)
                    for (int j = lane; j <= gamma; j += 32)
                        tok[static_cast<int64_t>(b) * (gamma + 1) + j] = (j < Lr) ? xb[j] : (j == Lr ? corr : -1);
            };
            if (p.do_strict && p.greedy) emit(p.L_strict, p.tok_strict, p.n_strict, L);
            for (int r = 0; r < p.n_ell; ++r) {
                int Lr = gamma;
                for (int c = 0; c < gamma; c += 32) {
                    const int j = c + lane;
                    bool fail = false;
                    if (j < gamma) {
                        const RowRec t = tr[j];
                        fail = p.ell_one[r] ? !(t.rank == 0) : !(static_cast<double>(t.g - t.M) >= p.ell_thr[r]);
                    }
                    const unsigned bal = __ballot_sync(0xFFFFFFFFu, fail);
                    if (bal) {
                        Lr = c + __ffs(bal) - 1;
                        break;
                    }
                }
                const int64_t o = static_cast<int64_t>(r) * p.B;
                emit(p.L_len ? p.L_len + o : nullptr, p.tok_len ? p.tok_len + o * (gamma + 1) : nullptr,
                     p.n_len ? p.n_len + o : nullptr, Lr);
            }
            for (int r = 0; r < p.n_k; ++r) {
                int Lr = gamma;
                for (int c = 0; c < gamma; c += 32) {
                    const int j = c + lane;
                    bool fail = false;
                    if (j < gamma) fail = !(tr[j].rank < p.kval[r]);
                    const unsigned bal = __ballot_sync(0xFFFFFFFFu, fail);
                    if (bal) {
                        Lr = c + __ffs(bal) - 1;
                        break;
                    }
                }
                const int64_t o = static_cast<int64_t>(r) * p.B;
                emit(p.L_topk ? p.L_topk + o : nullptr, p.tok_topk ? p.tok_topk + o * (gamma + 1) : nullptr,
                     p.n_topk ? p.n_topk + o : nullptr, Lr);
            }
            // fused round: schedule, agreement and the tokens of skipped blocks
            if (p.do_sched) {
                const RowRec *dr = p.drec + static_cast<int64_t>(i) * gamma;
                // gather q / logq of the block into registers-by-lane via shared memory is not
                // needed: schedule_block reads them through these small strided views
                __shared__ float s_q[SDD_MAX_GAMMA], s_lq[SDD_MAX_GAMMA];
                for (int j = lane; j < gamma; j += 32) {
                    s_q[j] = dr[j].q;
                    s_lq[j] = dr[j].logq;
                }
                __syncwarp();
                const bool force = p.force_strict && p.force_strict[b];
                const int D = p.D_in ? p.D_in[b] : 0;
                for (int t = 0; t < p.n_tau; ++t) {
                    int Kh, K, Do;
                    schedule_block(lane, gamma, s_q, s_lq,
                                   p.guard ? p.guard + static_cast<int64_t>(b) * gamma : nullptr,
                                   force || p.tau_off[t], D, p.signal, p.eta_loc[t], p.log_eta_c[t], p.K_min, p.S_max,
                                   Kh, K, Do);
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
                        const bool skip = K > 0;
                        if (lane == 0) p.k0[i] = K;   // read by the CTA that completes the sampling draw
                        if (skip || (p.do_strict && p.greedy)) {
                            // skipped: commit x_1..x_K; greedy strict: the verified tokens
                            const int Lc = skip ? K : L;
                            const int corr = skip ? -1 : tr[L].argmax;
                            if (lane == 0 && p.commit_n) p.commit_n[b] = skip ? K : L + 1;
                            if (p.commit_tokens)
                                for (int j = lane; j <= gamma; j += 32)
                                    p.commit_tokens[static_cast<int64_t>(b) * (gamma + 1) + j] =
                                        (j < Lc) ? xb[j] : (j == Lc ? corr : -1);
                        }
                    }
                }
            }
        }
    }
    __syncthreads();
    if (!p.do_strict || p.greedy) return;

    // ---- sampling: residual (L < gamma) or bonus (L = gamma) inverse-CDF draw ----
    const int L = s_L;
    if (threadIdx.x == 0) {
        s_lse[0] = tr[L].lse;
        s_lse[1] = 0.0;
        if (L < gamma)
            s_lse[1] = p.drec ? p.drec[static_cast<int64_t>(i) * gamma + L].lse
                              : __ldg(p.d_lse + static_cast<int64_t>(b) * gamma + L);
    }
    __syncthreads();
    const DrawCtx c = draw_ctx(p.zt + (static_cast<int64_t>(b) * (gamma + 1) + L) * p.stride_bytes,
                               (L < gamma) ? p.zd + (static_cast<int64_t>(b) * gamma + L) * p.stride_bytes : nullptr,
                               s_lse[0], s_lse[1]);
    const int v0 = seg * p.seg_vec, v1 = min(p.RV, v0 + p.seg_vec);
    int last_pos, found;
    const double tot = (v0 < v1) ? draw_pass<DT>(c, v0, v1, p.V, false, 0.0, last_pos, found, s_warp, &s_first) : 0.0;
    // publish this segment's total (and last positive entry) and count arrivals
    int lp = last_pos;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) lp = max(lp, __shfl_xor_sync(0xFFFFFFFFu, lp, off));
    __shared__ int s_lpw[kResidThreads / 32];
    if (lane == 0) s_lpw[warp] = lp;
    __syncthreads();
    __shared__ int s_is_last;
    if (threadIdx.x == 0) {
        int lpb = -1;
        for (int w = 0; w < kResidThreads / 32; ++w) lpb = max(lpb, s_lpw[w]);
        p.res_total[static_cast<int64_t>(i) * p.nseg + seg] = tot;
        p.res_last[static_cast<int64_t>(i) * p.nseg + seg] = lpb;
        __threadfence();
        const uint32_t old = atomicAdd(p.res_count + i, 1u);
        s_is_last = (old == static_cast<uint32_t>(p.nseg - 1)) ? 1 : 0;
    }
    __syncthreads();
    if (!s_is_last) return;
    __threadfence();
    // the last segment to arrive completes the draw for this block
    if (threadIdx.x < p.nseg) {
        s_tot[threadIdx.x] = __ldcg(p.res_total + static_cast<int64_t>(i) * p.nseg + threadIdx.x);
        s_last[threadIdx.x] = __ldcg(p.res_last + static_cast<int64_t>(i) * p.nseg + threadIdx.x);
    }
    __syncthreads();
    __shared__ int s_seg, s_lastp;
    __shared__ double s_target, s_before;
    if (threadIdx.x == 0) {
        double R = 0.0;
        int lastp = -1;
        for (int s = 0; s < p.nseg; ++s) {
            R += s_tot[s];
            lastp = max(lastp, s_last[s]);
        }
        const uint32_t jj = (L < gamma) ? static_cast<uint32_t>(L + 1) : static_cast<uint32_t>(gamma + 1);
        const float u = philox_uniform(p.seed, jj, static_cast<uint32_t>(b), p.round,
                                       (L < gamma) ? kPurposeResid : kPurposeBonus);
        const double target = static_cast<double>(u) * R;
        int sel = -2;   // -2: none (rounding) -> last positive; -3: no mass
        double before = 0.0, cum = 0.0;
        if (!(R > 0.0)) {
            sel = -3;
        } else {
            for (int s = 0; s < p.nseg; ++s) {
                if (cum + s_tot[s] > target && s_tot[s] > 0.0) {
                    sel = s;
                    before = cum;
                    break;
                }
                cum += s_tot[s];
            }
        }
        s_seg = sel;
        s_target = target;
        s_before = before;
        s_lastp = lastp;
        p.res_count[i] = 0u;   // leave the workspace zeroed
    }
    __syncthreads();
    int tok = -1;
    if (s_seg >= 0) {
        const int sv0 = s_seg * p.seg_vec, sv1 = min(p.RV, sv0 + p.seg_vec);
        const int lastp = s_lastp;
        int lp2, fnd;
        (void)draw_pass<DT>(c, sv0, sv1, p.V, true, s_target - s_before, lp2, fnd, s_warp, &s_first);
        tok = (fnd >= 0) ? fnd : lastp;
    } else if (s_seg == -2) {
        tok = s_lastp;
    } else {
        // the residual has no mass (only possible through rounding): draw from p_t of
        // this row, whole row in this CTA, same inverse-CDF rule
        DrawCtx ct = c;
        ct.zd_row = nullptr;
        int lp3, fnd;
        __syncthreads();
        const double R = draw_pass<DT>(ct, 0, p.RV, p.V, false, 0.0, lp3, fnd, s_warp, &s_first);
        const float u = philox_uniform(p.seed, static_cast<uint32_t>(L + 1), static_cast<uint32_t>(b), p.round,
                                       kPurposeResid);
        if (R > 0.0) {
            (void)draw_pass<DT>(ct, 0, p.RV, p.V, true, static_cast<double>(u) * R, lp3, fnd, s_warp, &s_first);
            tok = fnd;
        }
    }
    if (warp == 0) {
        if (lane == 0) {
            if (p.L_strict) p.L_strict[b] = L;
            if (p.n_strict) p.n_strict[b] = L + 1;
        }
        if (p.tok_strict)
            for (int j = lane; j <= gamma; j += 32)
                p.tok_strict[static_cast<int64_t>(b) * (gamma + 1) + j] = (j < L) ? xb[j] : (j == L ? tok : -1);
        if (p.do_sched) {
            // commit under pair 0 when that schedule did not skip this block
            const int K0 = __ldcg(p.k0 + i);
            if (K0 == 0) {
                if (lane == 0 && p.commit_n) p.commit_n[b] = L + 1;
                if (p.commit_tokens)
                    for (int j = lane; j <= gamma; j += 32)
                        p.commit_tokens[static_cast<int64_t>(b) * (gamma + 1) + j] =
                            (j < L) ? xb[j] : (j == L ? tok : -1);
            }
        }
    }
    (void)EPV;
}

__global__ void schedule_kernel(const __grid_constant__ ScheduleParams p) {
    const int lane = threadIdx.x & 31;
    const int64_t w = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    if (w >= static_cast<int64_t>(p.B) * p.n_tau) return;
    const int t = static_cast<int>(w / p.B), b = static_cast<int>(w % p.B);
    const int64_t o = static_cast<int64_t>(b) * p.gamma;
    const bool force = p.force_strict && p.force_strict[b];
    const int D = p.D_in ? p.D_in[b] : 0;
    int Kh, K, Do;
    schedule_block(lane, p.gamma, p.q + o, p.logq ? p.logq + o : nullptr, p.guard ? p.guard + o : nullptr,
                   force || p.tau_off[t], D, p.signal, p.eta_loc[t], p.log_eta_c[t], p.K_min, p.S_max, Kh, K, Do);
    if (lane == 0) {
        const int64_t oo = static_cast<int64_t>(t) * p.B + b;
        p.K_hat[oo] = Kh;
        p.K[oo] = K;
        if (p.D_out) p.D_out[oo] = Do;
    }
}

__global__ void agreement_kernel(const int32_t *K, const int32_t *L, int B, int n_tau, long long *acc) {
    const int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= static_cast<int64_t>(B) * n_tau) return;
    const int t = static_cast<int>(idx / B), b = static_cast<int>(idx % B);
    const int k = K[idx], l = L[b];
    if (k <= 0) return;
    unsigned long long *a = reinterpret_cast<unsigned long long *>(acc + 4 * t);
    atomicAdd(a + 0, static_cast<unsigned long long>(min(k, l)));
    atomicAdd(a + 1, static_cast<unsigned long long>(k));
    atomicAdd(a + 2, static_cast<unsigned long long>(k <= l ? 1 : 0));
    atomicAdd(a + 3, 1ull);
}

__global__ void commit_kernel(const int32_t *K, const int32_t *x, const int32_t *vt, const int32_t *vn, int B,
                              int gamma, int32_t *out_t, int32_t *out_n) {
    const int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= static_cast<int64_t>(B) * (gamma + 1)) return;
    const int b = static_cast<int>(idx / (gamma + 1)), j = static_cast<int>(idx % (gamma + 1));
    const int k = K[b];
    if (k > 0) {
        out_t[idx] = (j < k) ? x[static_cast<int64_t>(b) * gamma + j] : -1;
        if (j == 0) out_n[b] = k;
    } else {
        out_t[idx] = vt[idx];
        if (j == 0) out_n[b] = vn[b];
    }
}

__global__ void uniforms_kernel(uint64_t seed, const uint32_t *j, const uint32_t *b, const uint64_t *round,
                                const uint32_t *purpose, int64_t n, float *u) {
    const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i < n) u[i] = philox_uniform(seed, j[i], b[i], round[i], purpose[i]);
}

}  // namespace

cudaError_t launch_uniforms(uint64_t seed, const uint32_t *j, const uint32_t *b, const uint64_t *round,
                            const uint32_t *purpose, int64_t n, float *u, cudaStream_t stream) {
    if (n == 0) return cudaSuccess;
    uniforms_kernel<<<static_cast<unsigned>((n + 255) / 256), 256, 0, stream>>>(seed, j, b, round, purpose, n, u);
    return cudaGetLastError();
}

cudaError_t launch_decide(const DecideParams &p, cudaStream_t stream) {
    if (p.nb == 0) return cudaSuccess;
    const dim3 grid(p.nb, p.nseg);
    if (p.dtype == SDD_BF16)
        decide_kernel<SDD_BF16><<<grid, kResidThreads, 0, stream>>>(p);
    else
        decide_kernel<SDD_F32><<<grid, kResidThreads, 0, stream>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_schedule(const ScheduleParams &p, cudaStream_t stream) {
    const int64_t warps = static_cast<int64_t>(p.B) * p.n_tau;
    if (warps == 0) return cudaSuccess;
    const int64_t blocks = (warps * 32 + 255) / 256;
    schedule_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_agreement(const int32_t *K, const int32_t *L, int B, int n_tau, long long *acc,
                             cudaStream_t stream) {
    const int64_t n = static_cast<int64_t>(B) * n_tau;
    if (n == 0) return cudaSuccess;
    agreement_kernel<<<static_cast<unsigned>((n + 255) / 256), 256, 0, stream>>>(K, L, B, n_tau, acc);
    return cudaGetLastError();
}

cudaError_t launch_commit(const int32_t *K, const int32_t *x, const int32_t *vt, const int32_t *vn, int B,
                          int gamma, int32_t *out_t, int32_t *out_n, cudaStream_t stream) {
    const int64_t n = static_cast<int64_t>(B) * (gamma + 1);
    if (n == 0) return cudaSuccess;
    commit_kernel<<<static_cast<unsigned>((n + 255) / 256), 256, 0, stream>>>(K, x, vt, vn, B, gamma, out_t, out_n);
    return cudaGetLastError();
}

}  // namespace sdd
