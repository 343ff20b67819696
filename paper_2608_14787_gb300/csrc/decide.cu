// decide.cu -- the kernels that run after (or beside) the streaming pass
// (the per-CTA decide work and its helpers are in decide.cuh).
//  * decide_kernel    -- one CTA per (listed block, draw segment), launched as
//                        a programmatic dependent of the streaming grid.
//  * shard_draw_kernel -- the vocabulary-sharded round's draw.
//  * schedule_kernel  -- the skip policy of Sec. 4.1 as a stand-alone call.
//  * agreement_kernel, commit_kernel, uniforms_kernel, select_rows_kernel --
//                        small stand-alone calls.
#include "decide.cuh"

namespace sdd {

namespace {

// One CTA per (listed block, draw segment), behind the streaming grid that
// wrote the partials (FEAT, SHARD: as decide_cta).  Separate instantiations,
// so that the fused round keeps the smallest kernel.
template <int DT, bool FEAT, bool SHARD = false>
__global__ void __launch_bounds__(kDecThreads) decide_kernel(const __grid_constant__ ScanParams p) {
    extern __shared__ float s_pref_all[];   // [nseg][kDecThreads]: every segment's prefixes (last CTA)
    griddep_wait();   // launched behind the streaming grid that wrote the partials
    const PartView pv = part_view(p);
    const DecGeom geo = dec_geom(p, pv, p.dec.enabled && p.dec.do_strict && !p.dec.greedy && !SHARD);
    decide_cta<DT, FEAT, SHARD>(p, pv, geo, s_pref_all);
}

// Vocabulary-sharded draw, one CTA per block, after every slice's masses of
// the block's draw row have been exchanged (Sec. 3.1's resampling rule: the
// inverse CDF in ascending vocabulary order).  Warp 0 takes double-float
// prefix sums of the slices' masses in slice order and locates u R exactly
// as the one-GPU draw locates a segment (no residual mass -> p_t of the same
// row; rounding past the last slice -> the last slice of positive mass, its
// last positive entry).  Only the rank whose slice holds the draw goes on:
// it finds the entry in its slice and writes the token at position L.
constexpr int kMaxShards = 64;

template <int DT>
__global__ void __launch_bounds__(kDecThreads) shard_draw_kernel(const __grid_constant__ ShardParams sp) {
    constexpr int NW = kDecThreads / 32;
    const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int gamma = sp.gamma, S = sp.n_shards;
    __shared__ float s_warp[2 * NW];
    __shared__ df s_cum[kMaxShards];
    __shared__ df s_cseg[kDrawMaxSeg];
    __shared__ int s_sel, s_col, s_thr, s_last, s_tok, s_seg;
    __shared__ df s_rem, s_rem2;
    extern __shared__ float s_pref_all[];   // [nseg][kDecThreads]: the decide's prefixes of this slice's draw row
    if (tid == 0) {
        s_thr = INT32_MAX;
        s_last = -1;
    }
    const ShardDraw st = sp.state[b];
    const int L = st.L;
    if (warp == 0) {
        const uint32_t jj = (L < gamma) ? static_cast<uint32_t>(L + 1) : static_cast<uint32_t>(gamma + 1);
        const float u = philox_uniform(sp.seed, jj, static_cast<uint32_t>(b), sp.round,
                                       (L < gamma) ? kPurposeResid : kPurposeBonus);
        int col = 0, last = -1;
        df R = df{0.f, 0.f};
        for (int pass = 0; pass < 2; ++pass) {
            col = pass;
            df carry = df{0.f, 0.f};
            last = -1;
            for (int s0 = 0; s0 < S; s0 += 32) {
                const int sg = s0 + lane;
                const float t = (sg < S) ? sp.mass_all[(static_cast<int64_t>(sg) * sp.B + b) * 2 + col] : 0.f;
                const df cum = df_add(carry, warp_prefix_df(df{t, 0.f}, lane));
                if (sg < S) s_cum[sg] = cum;
                if (t > 0.f) last = sg;
                carry.hi = __shfl_sync(0xFFFFFFFFu, cum.hi, 31);
                carry.lo = __shfl_sync(0xFFFFFFFFu, cum.lo, 31);
            }
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) last = max(last, __shfl_xor_sync(0xFFFFFFFFu, last, off));
            R = carry;
            // the residual has no mass (only through rounding): p_t of the same row
            if (R.hi > 0.f || L >= gamma) break;
        }
        __syncwarp();
        const df target = df_mul_f(R, u);
        int sel = -1;
        if (R.hi > 0.f) {
            for (int s0 = 0; s0 < S; s0 += 32) {
                const int sg = s0 + lane;
                const bool hit = (sg < S) && sp.mass_all[(static_cast<int64_t>(sg) * sp.B + b) * 2 + col] > 0.f &&
                                 !df_ge(target, s_cum[sg]);
                const unsigned bal = __ballot_sync(0xFFFFFFFFu, hit);
                if (bal) {
                    sel = s0 + __ffs(bal) - 1;
                    break;
                }
            }
        }
        if (lane == 0) {
            s_col = col;
            if (sel >= 0) {
                s_sel = sel;
                s_rem = (sel > 0) ? df_sub(target, s_cum[sel - 1]) : target;
            } else {
                s_sel = (R.hi > 0.f) ? last : -1;
                s_rem = df{__int_as_float(0x7F800000), 0.f};
            }
        }
    }
    dec_sync();
    if (s_sel != sp.shard) return;   // another rank's slice holds this block's draw
    const int64_t bo = static_cast<int64_t>(b) * (gamma + 1);
    const char *zt_row = sp.zt + (bo + L) * sp.stride_bytes;
    const char *zd_row = (L < gamma && s_col == 0) ? sp.zd + (static_cast<int64_t>(b) * gamma + L) * sp.stride_bytes
                                                   : nullptr;
    const DrawCtx c = draw_ctx(zt_row, zd_row, df{st.t_lh, st.t_ll}, zd_row ? df{st.d_lh, st.d_ll} : df{0.f, 0.f});
    int tok;
    if (s_col == 0) {
        // the residual (or bonus) weights: the segment, thread and entry from
        // the prefixes sdd_shard_decide published (the sums this slice's
        // mass was made of), as the one-GPU draw locates its token
        const float4 *src =
            reinterpret_cast<const float4 *>(sp.res_pref + static_cast<int64_t>(b) * kDrawMaxSeg * kDecThreads);
        for (int q = tid; q < sp.nseg * (kDecThreads / 4); q += kDecThreads) cp_async16(s_pref_all + 4 * q, src + q);
        cp_async_wait_all();
        dec_sync();
        if (warp == 0) {
            int last_seg;
            (void)segment_cum(s_pref_all, sp.nseg, s_cseg, lane, last_seg);
            __syncwarp();
            const df rem = s_rem;
            const int sel = segment_pick(s_pref_all, sp.nseg, s_cseg, rem, lane);
            if (lane == 0) {
                if (sel >= 0) {
                    s_seg = sel;
                    s_rem2 = (sel > 0) ? df_sub(rem, s_cseg[sel - 1]) : rem;
                } else {
                    // rounding (or an infinite remainder): the slice's last positive entry
                    s_seg = last_seg;
                    s_rem2 = df{__int_as_float(0x7F800000), 0.f};
                }
            }
        }
        dec_sync();
        tok = (s_seg >= 0) ? segment_find<DT>(c, s_pref_all, s_seg, s_rem2, sp.seg_vec, sp.RVs, sp.Vs, &s_thr, &s_last,
                                              &s_tok)
                           : -1;
    } else {
        // p_t of the row (the residual had no mass, only through rounding): the whole slice here
        tok = slice_find<DT>(c, sp.RVs, sp.Vs, s_rem, s_warp, &s_thr, &s_last, &s_tok);
    }
    if (tid == 0) {
        const int t = (tok >= 0) ? sp.v0 + tok : -1;
        if (sp.tok_strict) sp.tok_strict[bo + L] = t;
        if (st.commit && sp.commit_tokens) sp.commit_tokens[bo + L] = t;
    }
}

__global__ void schedule_kernel(const __grid_constant__ ScheduleParams p) {
    const int lane = threadIdx.x & 31;
    const int64_t w = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    if (w >= static_cast<int64_t>(p.B) * p.n_tau) return;
    const int t = static_cast<int>(w / p.B), b = static_cast<int>(w % p.B);
    const int gamma = p.gamma;
    const int64_t o = static_cast<int64_t>(b) * gamma;
    const bool force = p.force_strict && p.force_strict[b];
    const int D = p.D_in ? p.D_in[b] : 0;
    int Kh = 0, K = 0, Do = 0;
    if (p.signal == SDD_SIG_PERIODIC) {
        if (!force) {
            Kh = periodic_khat(gamma, p.period[t], p.K_skip, p.round,
                               [&](int j) { return p.guard && p.guard[o + j] != 0; }, lane);
            sched_final(Kh, D, p.K_min, p.S_max, K, Do);
        }
    } else if (!(force || p.tau_off[t])) {
        int kb = gamma, best = 0;
        df carry = df{0.f, 0.f};
        for (int c = 0; c < gamma && kb >= c; c += 32) {
            const int j = c + lane;
            const bool in = j < gamma;
            const float qj = in ? p.q[o + j] : 0.f;
            const float lq = in ? (p.logq ? p.logq[o + j] : logf(qj)) : 0.f;
            const bool guard_j = in && p.guard && p.guard[o + j];
            const df S = df_add(carry, warp_prefix_df(df{lq, 0.f}, lane));
            carry.hi = __shfl_sync(0xFFFFFFFFu, S.hi, 31);
            carry.lo = __shfl_sync(0xFFFFFFFFu, S.lo, 31);
            sched_step(c, lane, gamma, in, qj, guard_j, S, p.eta_loc[t], p.log_eta_c[t], p.signal, kb, best);
        }
        Kh = (p.signal == SDD_SIG_MARGINAL) ? kb : best;
        sched_final(Kh, D, p.K_min, p.S_max, K, Do);
    }
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

int decide_max_ctas_per_sm() {
    int n = 0;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, decide_kernel<SDD_BF16, false>, kDecThreads, 0);
    return n;
}

// Opt both instantiations in to the prefix staging area of the draw.
cudaError_t decide_prepare_device() {
    constexpr int bytes = kDrawMaxSeg * kDecThreads * static_cast<int>(sizeof(float));
    void (*const kernels[])(ScanParams) = {decide_kernel<SDD_BF16, false>, decide_kernel<SDD_F32, false>,
                                           decide_kernel<SDD_BF16, true>, decide_kernel<SDD_F32, true>,
                                           decide_kernel<SDD_BF16, false, true>, decide_kernel<SDD_F32, false, true>};
    for (auto k : kernels) {
        const cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
        if (e != cudaSuccess) return e;
    }
    void (*const draws[])(ShardParams) = {shard_draw_kernel<SDD_BF16>, shard_draw_kernel<SDD_F32>};
    for (auto k : draws) {
        const cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

cudaError_t launch_decide(const ScanParams &p, cudaStream_t stream) {
    const int nb = p.grp[0].nb;
    if (nb == 0) return cudaSuccess;
    const bool draw = p.dec.enabled && p.dec.do_strict && !p.dec.greedy;
    // a device block count: a one-dimensional grid cut on the device (dec_geom)
    const bool dev_geom = draw && p.nb_dev != nullptr && p.shard == nullptr;
    const int nseg = draw ? (dev_geom ? std::min(kDrawMaxSeg, std::max(p.dec.dec_ctas, 1)) : p.dec.nseg) : 1;
    const size_t smem = draw ? static_cast<size_t>(nseg) * kDecThreads * sizeof(float) : 0;
    const dim3 grid = dev_geom ? dim3(static_cast<unsigned>(std::max(p.dec.dec_ctas, nb))) : dim3(nb, nseg);
    const bool bf = p.dtype == SDD_BF16, feat = p.feat != nullptr;
    void (*const k)(ScanParams) = (p.shard != nullptr)
                                      ? (bf ? decide_kernel<SDD_BF16, false, true> : decide_kernel<SDD_F32, false, true>)
                                  : feat ? (bf ? decide_kernel<SDD_BF16, true> : decide_kernel<SDD_F32, true>)
                                         : (bf ? decide_kernel<SDD_BF16, false> : decide_kernel<SDD_F32, false>);
    return launch_dependent(k, grid, dim3(kDecThreads), smem, stream, p);
}

// The blocks that go to the verifier: K[b] == 0, in ascending order, by one
// CTA (a ballot and a running offset per chunk of 1024).
__global__ void __launch_bounds__(1024) select_rows_kernel(const int32_t *K, int B, int32_t *rows, int32_t *n_rows) {
    __shared__ int s_warp[32];
    __shared__ int s_base;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) s_base = 0;
    __syncthreads();
    for (int c0 = 0; c0 < B; c0 += 1024) {
        const int b = c0 + tid;
        const bool sel = b < B && K[b] == 0;
        const unsigned bal = __ballot_sync(0xFFFFFFFFu, sel);
        if (lane == 0) s_warp[warp] = __popc(bal);
        __syncthreads();
        int before = s_base;
        for (int w = 0; w < warp; ++w) before += s_warp[w];
        if (sel) rows[before + __popc(bal & ((1u << lane) - 1u))] = b;
        __syncthreads();
        if (tid == 0) {
            int tot = 0;
            for (int w = 0; w < 32; ++w) tot += s_warp[w];
            s_base += tot;
        }
        __syncthreads();
    }
    if (tid == 0) *n_rows = s_base;
}

cudaError_t launch_select_rows(const int32_t *K, int B, int32_t *rows, int32_t *n_rows, cudaStream_t stream) {
    select_rows_kernel<<<1, 1024, 0, stream>>>(K, B, rows, n_rows);
    return cudaGetLastError();
}

cudaError_t launch_shard_draw(const ShardParams &sp, cudaStream_t stream) {
    if (sp.B == 0) return cudaSuccess;
    const size_t smem = static_cast<size_t>(sp.nseg) * kDecThreads * sizeof(float);
    if (sp.dtype == SDD_BF16)
        shard_draw_kernel<SDD_BF16><<<sp.B, kDecThreads, smem, stream>>>(sp);
    else
        shard_draw_kernel<SDD_F32><<<sp.B, kDecThreads, smem, stream>>>(sp);
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
