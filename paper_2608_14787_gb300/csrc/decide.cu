// decide.cu -- the kernels that run after (or beside) the streaming pass.
//
//  * draw_kernel      -- the inverse-CDF draw of the speculative-sampling rule
//                        cited by Sec. 3.1: at the first rejected position the
//                        residual norm(max(0, p_t - p_d)), or, when the whole
//                        block is accepted, p_t of the bonus row.  The draw row
//                        is split into segments, one CTA each; the last segment
//                        to finish (atomic arrival, no waiting) locates the
//                        segment holding u * R and rescans it.
//  * schedule_kernel  -- the skip policy of Sec. 4.1 as a stand-alone call.
//  * agreement_kernel, commit_kernel, uniforms_kernel -- small stand-alone calls.
#include "rules.cuh"

namespace sdd {

namespace {

// Draw-row context: integer references and the hi/lo LSE difference.
struct DrawCtx {
    const char *zt_row, *zd_row;
    float nrt, nrd, d_hi, d_lo;
};

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

// Weights of the draw for the EPV entries of one 16-byte vector.
//   residual: p_t - p_d = p_d (exp(D(v)) - 1) with the log-ratio
//             D(v) = (z_t(v) - z_d(v)) - (LSE_t - LSE_d); the LSE difference is
//             applied as two fp32 terms (hi + lo) and the difference by expm1, so
//             no cancellation between near-equal p_t and p_d loses precision;
//             p_d(v) = 2^(z_d(v) log2(e) - r_d) up to the common factor of the row;
//   bonus (zd_row == nullptr): 2^(z_t(v) log2(e) - r_t).
// Returns the fp32 sum of the entries in ascending order.
template <int DT>
__device__ __forceinline__ float vec_weights(const DrawCtx &c, uint4 a, uint4 d, int vec, int V, float (&w)[8]) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
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
        if (c.zd_row) {
            const float dv = ((zt - zd) - c.d_hi) - c.d_lo;
            wv = 0.f;
            if (dv > 0.f) wv = ex2(fmaf(zd, kLog2e, c.nrd)) * expm1_pos(dv);
        } else {
            wv = ex2(fmaf(zt, kLog2e, c.nrt));
        }
        if (vec * EPV + e >= V) wv = 0.f;
        w[e] = wv;
        sum += wv;
    }
    return sum;
}

// Inclusive scan of one fp32 value per thread over the CTA (kDrawThreads).
// Returns the thread's inclusive value; *total receives the CTA total.
__device__ __forceinline__ float cta_incl_scan(float v, float *warp_tot, float *total) {
    constexpr int NW = kDrawThreads / 32;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const float t = __shfl_up_sync(0xFFFFFFFFu, v, off);
        if (lane >= off) v += t;
    }
    if (lane == 31) warp_tot[warp] = v;
    __syncthreads();
    if (threadIdx.x < 32) {
        float t = (lane < NW) ? warp_tot[lane] : 0.f;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const float s = __shfl_up_sync(0xFFFFFFFFu, t, off);
            if (lane >= off) t += s;
        }
        if (lane < NW) warp_tot[NW + lane] = t;   // inclusive prefix of the warp totals
    }
    __syncthreads();
    const float r = ((warp > 0) ? warp_tot[NW + warp - 1] : 0.f) + v;
    *total = warp_tot[2 * NW - 1];
    __syncthreads();
    return r;
}

// Sum (fp32, ascending order) of the draw weights of vectors [vb, ve).
template <int DT>
__device__ __forceinline__ float run_sum(const DrawCtx &c, int vb, int ve, int V, int &last_pos) {
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
                for (int e = 0; e < EPV; ++e) {
                    sum += w[e];
                    if (w[e] > 0.f) last_pos = vec * EPV + e;
                }
            }
        }
    }
    return sum;
}

// The first entry of vectors [vb, ve) whose running sum, starting at `start`,
// exceeds `target` (same order and arithmetic as run_sum); -1 if none.
template <int DT>
__device__ __forceinline__ int run_find(const DrawCtx &c, int vb, int ve, int V, double start, double target,
                                        int &last_pos) {
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
                if (start + static_cast<double>(sum) > target) return vec * EPV + e;
            }
        }
    }
    return -1;
}

// Inverse CDF over vectors [v0, v1) of the draw row, one contiguous run of
// `vpt` vectors per thread: returns the drawn index (or the last positive
// entry if rounding leaves none), identical in every thread.
template <int DT>
__device__ int cta_find(const DrawCtx &c, int v0, int v1, int vpt, int V, double before, double target,
                        float *s_warp, int *s_thr, int *s_tok) {
    const int vb = min(v1, v0 + static_cast<int>(threadIdx.x) * vpt), ve = min(v1, vb + vpt);
    int lastp = -1;
    const float ts = run_sum<DT>(c, vb, ve, V, lastp);
    float tot;
    const float incl = cta_incl_scan(ts, s_warp, &tot);
    if (threadIdx.x == 0) *s_thr = INT32_MAX;
    __syncthreads();
    const bool mine = (ve > vb) && (before + static_cast<double>(incl) > target);
    const unsigned bal = __ballot_sync(0xFFFFFFFFu, mine);
    if ((threadIdx.x & 31) == 0 && bal) atomicMin(s_thr, static_cast<int>(threadIdx.x) + __ffs(bal) - 1);
    __syncthreads();
    const int thr = *s_thr;
    if (thr == INT32_MAX) return -1;
    if (static_cast<int>(threadIdx.x) == thr) {
        int lp = -1;
        const int pick = run_find<DT>(c, vb, ve, V, before + static_cast<double>(incl - ts), target, lp);
        *s_tok = (pick >= 0) ? pick : lp;
    }
    __syncthreads();
    return *s_tok;
}

template <int DT>
__global__ void __launch_bounds__(kDrawThreads) draw_kernel(const __grid_constant__ DrawParams p) {
    const int i = blockIdx.x;       // listed block
    const int seg = blockIdx.y;     // segment of the draw row
    const int gamma = p.gamma;
    const int b = p.bidx ? __ldg(p.bidx + i) : i;
    if (b < 0 || b >= p.B) return;  // flagged by the streaming pass
    __shared__ float s_warp[2 * (kDrawThreads / 32)];
    __shared__ int s_is_last, s_seg, s_lastp, s_thr, s_tok, s_L;
    __shared__ double s_target, s_before;
    __shared__ double s_tot[kDrawMaxSeg];
    __shared__ int s_last[kDrawMaxSeg];
    __shared__ DrawCtx s_ctx;

    // the draw row and its context, once per CTA
    if (threadIdx.x == 0) {
        const int L = p.blk_L[i];
        const double lse_t = p.trec[static_cast<int64_t>(i) * (gamma + 1) + L].lse;
        double lse_d = 0.0;
        if (L < gamma)
            lse_d = p.drec ? p.drec[static_cast<int64_t>(i) * gamma + L].lse
                           : p.d_lse[static_cast<int64_t>(b) * gamma + L];
        const char *zt_row = p.zt + (static_cast<int64_t>(b) * (gamma + 1) + L) * p.stride_bytes;
        const char *zd_row = (L < gamma) ? p.zd + (static_cast<int64_t>(b) * gamma + L) * p.stride_bytes : nullptr;
        s_ctx = draw_ctx(zt_row, zd_row, lse_t, lse_d);
        s_L = L;
        s_lastp = -1;
    }
    __syncthreads();
    const DrawCtx c = s_ctx;
    const int L = s_L;
    const int vpt = p.seg_vec / kDrawThreads;

    // first pass: this segment's weight total and last positive entry
    const int v0 = seg * p.seg_vec, v1 = min(p.RV, v0 + p.seg_vec);
    int last_pos = -1;
    {
        const int vb = min(v1, v0 + static_cast<int>(threadIdx.x) * vpt), ve = min(v1, vb + vpt);
        const float ts = run_sum<DT>(c, vb, ve, p.V, last_pos);
        float tot;
        (void)cta_incl_scan(ts, s_warp, &tot);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) last_pos = max(last_pos, __shfl_xor_sync(0xFFFFFFFFu, last_pos, off));
        if ((threadIdx.x & 31) == 0) atomicMax(&s_lastp, last_pos);
        __syncthreads();
        if (threadIdx.x == 0) {
            p.res_total[static_cast<int64_t>(i) * p.nseg + seg] = static_cast<double>(tot);
            p.res_last[static_cast<int64_t>(i) * p.nseg + seg] = s_lastp;
            __threadfence();
            const uint32_t old = atomicAdd(p.res_count + i, 1u);
            s_is_last = (old == static_cast<uint32_t>(p.nseg - 1)) ? 1 : 0;
        }
        __syncthreads();
    }
    if (!s_is_last) return;
    __threadfence();
    // the last segment to arrive completes the draw: locate the segment holding u * R
    for (int s = threadIdx.x; s < p.nseg; s += kDrawThreads) {
        s_tot[s] = __ldcg(p.res_total + static_cast<int64_t>(i) * p.nseg + s);
        s_last[s] = __ldcg(p.res_last + static_cast<int64_t>(i) * p.nseg + s);
    }
    __syncthreads();
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
        int sel = (R > 0.0) ? -2 : -3;   // -2: rounding left none (last positive), -3: no mass
        double cum = 0.0, before = 0.0;
        if (R > 0.0) {
            for (int s = 0; s < p.nseg; ++s) {
                const double t = s_tot[s];
                if (t > 0.0 && cum + t > target) {
                    sel = s;
                    before = cum;
                    break;
                }
                cum += t;
            }
        }
        s_seg = sel;
        s_target = target;
        s_before = before;
        s_lastp = lastp;
        p.res_count[i] = 0u;   // leave the workspace zeroed
    }
    __syncthreads();
    int tok;
    if (s_seg >= 0) {
        const int sv0 = s_seg * p.seg_vec, sv1 = min(p.RV, sv0 + p.seg_vec);
        tok = cta_find<DT>(c, sv0, sv1, vpt, p.V, s_before, s_target, s_warp, &s_thr, &s_tok);
        if (tok < 0) tok = s_lastp;
    } else if (s_seg == -2) {
        tok = s_lastp;
    } else {
        // the residual has no mass (only through rounding): draw from p_t of the
        // same row, whole row in this CTA, same inverse-CDF rule
        DrawCtx ct = c;
        ct.zd_row = nullptr;
        const int vrow = (p.RV + kDrawThreads - 1) / kDrawThreads;
        const int vb = min(p.RV, static_cast<int>(threadIdx.x) * vrow), ve = min(p.RV, vb + vrow);
        int lp = -1;
        float tot;
        (void)cta_incl_scan(run_sum<DT>(ct, vb, ve, p.V, lp), s_warp, &tot);
        const float u = philox_uniform(p.seed, static_cast<uint32_t>(L + 1), static_cast<uint32_t>(b), p.round,
                                       kPurposeResid);
        tok = (tot > 0.f) ? cta_find<DT>(ct, 0, p.RV, vrow, p.V, 0.0, static_cast<double>(u) * tot, s_warp, &s_thr, &s_tok)
                          : -1;
    }
    if (threadIdx.x < 32) {
        const int lane = threadIdx.x;
        const int32_t *xb = p.tokens + static_cast<int64_t>(b) * gamma;
        const int64_t bo = static_cast<int64_t>(b) * (gamma + 1);
        if (lane == 0) {
            if (p.L_strict) p.L_strict[b] = L;
            if (p.n_strict) p.n_strict[b] = L + 1;
        }
        if (p.tok_strict) write_tokens(lane, gamma, p.tok_strict + bo, xb, L, tok);
        if (p.k0 && p.k0[i] == 0) {
            // commit under pair 0: this block was not skipped
            if (lane == 0 && p.commit_n) p.commit_n[b] = L + 1;
            if (p.commit_tokens) write_tokens(lane, gamma, p.commit_tokens + bo, xb, L, tok);
        }
    }
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
    schedule_block(lane, p.gamma, p.q + o, p.logq ? p.logq + o : nullptr, 1, p.guard ? p.guard + o : nullptr,
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

cudaError_t launch_draw(const DrawParams &p, cudaStream_t stream) {
    if (p.nb == 0) return cudaSuccess;
    const dim3 grid(p.nb, p.nseg);
    if (p.dtype == SDD_BF16)
        draw_kernel<SDD_BF16><<<grid, kDrawThreads, 0, stream>>>(p);
    else
        draw_kernel<SDD_F32><<<grid, kDrawThreads, 0, stream>>>(p);
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

cudaError_t launch_uniforms(uint64_t seed, const uint32_t *j, const uint32_t *b, const uint64_t *round,
                            const uint32_t *purpose, int64_t n, float *u, cudaStream_t stream) {
    if (n == 0) return cudaSuccess;
    uniforms_kernel<<<static_cast<unsigned>((n + 255) / 256), 256, 0, stream>>>(seed, j, b, round, purpose, n, u);
    return cudaGetLastError();
}

}  // namespace sdd
