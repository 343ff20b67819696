// scan.cu -- the streaming pass of the path: one read of every drafter and
// target logit, producing per-row softmax statistics.
//
// What it computes (per row of logits z over the vocabulary):
//   M = max z, S = sum exp(z - M), T2 = sum exp(z - M) (z - M) log2(e),
//   the lowest index attaining M, and for target rows the saturated rank of
//   the drafted token x: #{v : z(v) > z(x)} + #{v < x : z(v) = z(x)}.
// From these the merging warp derives the quantities of Sec. 4.2 (raw
// confidence q = p_draft(x_j), LSE, maxprob, entropy) and the target facts that
// the acceptance rules of Sec. 3.1 and App. A.6 read.
//
// How: the rows of the call are laid end to end as one sequence of 16-byte
// vectors, split into contiguous, equal ranges, one per warp (perfect balance,
// no per-tile scheduling).  Each warp streams its range through a private
// ring of 4 KiB shared-memory tiles filled by 1D bulk copies (cp.async.bulk +
// mbarrier), keeps an online-softmax state per lane, reduces it across the
// warp at the end of each row piece and publishes a 32-byte partial.  The
// last warp to finish a row (atomic arrival counter, no waiting) merges the
// row's partials in a fixed order and writes the row's results.
#include "internal.h"

namespace sdd {

namespace {

struct Cursor {
    int64_t v;     // absolute vector index
    int64_t r;     // row
    int32_t k;     // vector offset inside the row
};

__device__ __forceinline__ void row_locate(const ScanParams &p, int64_t r, int &gi, int64_t &lr, int &j, int &b,
                                           bool &b_ok) {
    gi = (r >= p.rows0) ? 1 : 0;
    lr = gi ? r - p.rows0 : r;
    const ScanGroup &G = p.grp[gi];
    const int64_t i = lr / G.npos;
    j = static_cast<int>(lr - i * G.npos);
    b = G.bidx ? __ldg(G.bidx + i) : static_cast<int>(i);
    b_ok = (b >= 0 && b < p.B);
    if (!b_ok) b = 0;  // keep every address inside the tensor; the row is flagged at the end
}

__device__ __forceinline__ const char *row_base(const ScanParams &p, int64_t r) {
    int gi, j, b;
    int64_t lr;
    bool ok;
    row_locate(p, r, gi, lr, j, b, ok);
    const ScanGroup &G = p.grp[gi];
    return G.base + (static_cast<int64_t>(b) * G.npos + j) * G.stride_bytes;
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

template <int DT>
__device__ __forceinline__ float elem(const uint4 (&w)[kVPL], int i, int e) {
    const uint32_t *u = reinterpret_cast<const uint32_t *>(&w[i]);
    if (DT == SDD_BF16) return (e & 1) ? bf16_hi(u[e >> 1]) : bf16_lo(u[e >> 1]);
    return __uint_as_float(u[e]);
}

// Process one tile: the lane's vectors are lane, lane+32, ... of the tile.
template <int DT, bool kTarget>
__device__ __forceinline__ void process_tile(const uint4 *tile, int n, int k0, int lane, int tail, bool row_end,
                                             SoftState &st, float g, int tok, int kcap) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    uint4 w[kVPL];
#pragma unroll
    for (int i = 0; i < kVPL; ++i) {
        const int idx = lane + 32 * i;
        if (idx < n) {
            w[i] = tile[idx];
            if (row_end && tail && idx == n - 1) mask_tail<DT>(w[i], tail);
        } else {
            w[i] = make_uint4(kNegInfPairBf16, kNegInfPairBf16, kNegInfPairBf16, kNegInfPairBf16);
            if (DT != SDD_BF16) w[i] = make_uint4(0xFF800000u, 0xFF800000u, 0xFF800000u, 0xFF800000u);
        }
    }
    // clamp from below (NaN-propagating) and take the tile maximum
    float cm;
    if (DT == SDD_BF16) {
        uint32_t mx = kClampPairBf16;
#pragma unroll
        for (int i = 0; i < kVPL; ++i) {
            uint32_t *u = reinterpret_cast<uint32_t *>(&w[i]);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                u[q] = bf16x2_max_nan(u[q], kClampPairBf16);
                mx = bf16x2_max_nan(mx, u[q]);
            }
        }
        cm = fmax_nan(bf16_lo(mx), bf16_hi(mx));
    } else {
        const float fl = clamp_floor();
        cm = fl;
#pragma unroll
        for (int i = 0; i < kVPL; ++i) {
            float *f = reinterpret_cast<float *>(&w[i]);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                f[q] = fmax_nan(f[q], fl);
                cm = fmax_nan(cm, f[q]);
            }
        }
    }
    // a new running maximum: rescale and locate its first occurrence
    if (cm > st.m) {
        const float d = (st.m - cm) * kLog2e;
        const float sc = ex2(d);
        st.t2 = st.t2 * sc + (st.s * sc) * d;
        st.s *= sc;
        st.m = cm;
        int found = INT32_MAX;
#pragma unroll
        for (int i = 0; i < kVPL; ++i)
#pragma unroll
            for (int e = 0; e < EPV; ++e)
                if (found == INT32_MAX && elem<DT>(w, i, e) == cm) found = (k0 + lane + 32 * i) * EPV + e;
        st.amax = found;
    }
    // exp-sum (and entropy accumulator for drafter rows) on packed fp32 pairs
    const f2_t m2 = f2_pack(st.m, st.m);
    const f2_t l2 = f2_pack(kLog2e, kLog2e);
    f2_t as = 0ull, at = 0ull;
#pragma unroll
    for (int i = 0; i < kVPL; ++i) {
        const uint32_t *u = reinterpret_cast<const uint32_t *>(&w[i]);
#pragma unroll
        for (int q = 0; q < (DT == SDD_BF16 ? 4 : 2); ++q) {
            f2_t z2;
            if (DT == SDD_BF16)
                z2 = f2_pack(bf16_lo(u[q]), bf16_hi(u[q]));
            else
                z2 = f2_pack(__uint_as_float(u[2 * q]), __uint_as_float(u[2 * q + 1]));
            const f2_t y2 = f2_mul(f2_sub(z2, m2), l2);
            float y0, y1;
            f2_unpack(y2, y0, y1);
            const f2_t e2 = f2_pack(ex2(y0), ex2(y1));
            as = f2_add(as, e2);
            if (!kTarget) at = f2_fma(e2, y2, at);
        }
    }
    float a0, a1;
    f2_unpack(as, a0, a1);
    st.s += a0 + a1;
    if (!kTarget) {
        f2_unpack(at, a0, a1);
        st.t2 += a0 + a1;
    }
    // rank of the drafted token (target rows): only tiles that can hold an
    // entry >= g are inspected, and a lane stops once its count reaches kcap
    if (kTarget && tok >= 0 && cm >= g && st.rank < kcap) {
        int cnt = 0;
#pragma unroll
        for (int i = 0; i < kVPL; ++i)
#pragma unroll
            for (int e = 0; e < EPV; ++e) {
                const float z = elem<DT>(w, i, e);
                const int idx = (k0 + lane + 32 * i) * EPV + e;
                cnt += (z > g || (z == g && idx < tok)) ? 1 : 0;
            }
        st.rank += cnt;
    }
}

// Final results of row r from its merged state (whole warp calls; lane 0 writes).
template <int DT>
__device__ void finalize_row(const ScanParams &p, int64_t r, SoftState st, int lane) {
    int gi, j, b;
    int64_t lr;
    bool b_ok;
    row_locate(p, r, gi, lr, j, b, b_ok);
    const ScanGroup &G = p.grp[gi];
    const char *rowp = G.base + (static_cast<int64_t>(b) * G.npos + j) * G.stride_bytes;
    const bool has_tok = j < p.gamma;
    int tok = has_tok ? __ldg(p.tokens + static_cast<int64_t>(b) * p.gamma + j) : -1;
    const bool tok_ok = has_tok && tok >= 0 && tok < p.V;
    const bool valid = b_ok && isfinite(st.m) && st.m > clamp_floor() && isfinite(st.s) && st.s > 0.f;
    if (lane != 0) return;
    float g = __int_as_float(0x7FC00000);
    if (tok_ok) g = fmax_nan(load_logit<DT>(rowp, tok), clamp_floor());
    RowRec rec;
    const float nanf_ = __int_as_float(0x7FC00000);
    if (valid) {
        const float lnS = logf(st.s);
        rec.M = st.m;
        rec.S = st.s;
        rec.g = g;
        rec.gap = g - st.m;
        rec.q = ex2((g - st.m) * kLog2e) / st.s;
        rec.logq = (g - st.m) - lnS;
        rec.argmax = st.amax;
        rec.rank = min(st.rank, p.kcap);
        if (G.kind == 0 && b_ok) {
            const int64_t o = static_cast<int64_t>(b) * p.gamma + j;
            if (G.q) G.q[o] = tok_ok ? rec.q : nanf_;
            if (G.logq) G.logq[o] = tok_ok ? rec.logq : nanf_;
            if (G.maxprob) G.maxprob[o] = 1.f / st.s;
            if (G.lse) G.lse[o] = st.m + lnS;
            if (G.entropy) G.entropy[o] = lnS - (st.t2 * kLn2) / st.s;
            if (G.argmax) G.argmax[o] = st.amax;
        }
    } else {
        rec.M = rec.S = rec.g = rec.gap = rec.q = rec.logq = nanf_;
        rec.argmax = -1;
        rec.rank = INT32_MAX;
        if (G.kind == 0 && b_ok) {
            const int64_t o = static_cast<int64_t>(b) * p.gamma + j;
            if (G.q) G.q[o] = nanf_;
            if (G.logq) G.logq[o] = nanf_;
            if (G.maxprob) G.maxprob[o] = nanf_;
            if (G.lse) G.lse[o] = nanf_;
            if (G.entropy) G.entropy[o] = nanf_;
            if (G.argmax) G.argmax[o] = -1;
        }
        if (b_ok) status_or(p.status, SDD_DEV_NONFINITE);
    }
    if (has_tok && !tok_ok) {
        rec.q = rec.logq = rec.g = rec.gap = nanf_;
        rec.rank = INT32_MAX;
    }
    if ((has_tok && !tok_ok) || !b_ok) status_or(p.status, SDD_DEV_BAD_TOKEN);
    G.rec[lr] = rec;
}

template <int DT>
__global__ void __launch_bounds__(kThreads, 2) scan_kernel(const __grid_constant__ ScanParams p) {
    extern __shared__ __align__(128) unsigned char smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t gw = static_cast<int64_t>(blockIdx.x) * kWarpsPerCta + warp;
    if (gw >= p.W) return;
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    const int tail = p.V % EPV;  // valid entries of the last vector of a row (0 = full)

    unsigned char *ring = smem + warp * (kStages * kTileBytes);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kWarpsPerCta * kStages * kTileBytes) + warp * kStages;
    if (lane == 0) {
#pragma unroll
        for (int s = 0; s < kStages; ++s) mbar_init(&bars[s], 1);
        fence_mbar_init();
    }
    __syncwarp();

    const int64_t v0 = part_start(gw, p.T, p.W), v1 = part_start(gw + 1, p.T, p.W);
    Cursor pc{v0, v0 / p.RV, 0};
    pc.k = static_cast<int32_t>(v0 - pc.r * p.RV);
    Cursor cc = pc;
    const char *prow = row_base(p, pc.r);
    uint32_t pending = 0;  // slots with a copy in flight
    uint32_t phase = 0;    // parity bit per slot

    auto issue = [&](int slot) {
        const int n = static_cast<int>(min(static_cast<int64_t>(min(kTileVec, p.RV - pc.k)), v1 - pc.v));
        if (lane == 0) {
            fence_proxy_async_smem();
            mbar_arrive_expect_tx(&bars[slot], static_cast<uint32_t>(n) * 16u);
            bulk_g2s(ring + slot * kTileBytes, prow + static_cast<int64_t>(pc.k) * 16, static_cast<uint32_t>(n) * 16u,
                     &bars[slot]);
        }
        pending |= 1u << slot;
        pc.v += n;
        pc.k += n;
        if (pc.k == p.RV && pc.v < v1) {
            pc.k = 0;
            pc.r += 1;
            prow = row_base(p, pc.r);
        }
    };
    for (int s = 0; s < kStages && pc.v < v1; ++s) issue(s);

    SoftState st;
    bool in_piece = false;
    int kind = 0, tok = -1;
    float g = 0.f;
    int slot = 0;
    bool timed_out = false;
    while (cc.v < v1) {
        const int n = static_cast<int>(min(static_cast<int64_t>(min(kTileVec, p.RV - cc.k)), v1 - cc.v));
        if (!in_piece) {
            st.m = clamp_floor();
            st.s = 0.f;
            st.t2 = 0.f;
            st.amax = INT32_MAX;
            st.rank = 0;
            int gi, j, b;
            int64_t lr;
            bool ok;
            row_locate(p, cc.r, gi, lr, j, b, ok);
            kind = p.grp[gi].kind;
            tok = -1;
            g = 0.f;
            if (kind == 1 && j < p.gamma) {
                tok = __ldg(p.tokens + static_cast<int64_t>(b) * p.gamma + j);
                if (tok >= 0 && tok < p.V) {
                    const char *rowp = p.grp[gi].base + (static_cast<int64_t>(b) * p.grp[gi].npos + j) *
                                                            p.grp[gi].stride_bytes;
                    g = fmax_nan(load_logit<DT>(rowp, tok), clamp_floor());
                } else {
                    tok = -1;
                }
            }
            in_piece = true;
        }
        if (!mbar_wait_bounded(&bars[slot], (phase >> slot) & 1u, kWaitPolls)) {
            timed_out = true;
            break;
        }
        const uint4 *tile = reinterpret_cast<const uint4 *>(ring + slot * kTileBytes);
        const bool row_end = (cc.k + n == p.RV);
        if (kind == 1)
            process_tile<DT, true>(tile, n, cc.k, lane, tail, row_end, st, g, tok, p.kcap);
        else
            process_tile<DT, false>(tile, n, cc.k, lane, tail, row_end, st, g, tok, p.kcap);
        __syncwarp();
        phase ^= 1u << slot;
        pending &= ~(1u << slot);
        if (pc.v < v1) issue(slot);
        slot = (slot + 1 == kStages) ? 0 : slot + 1;
        cc.v += n;
        cc.k += n;
        if (row_end || cc.v == v1) {
            // end of this warp's piece of row cc.r
            SoftState red = soft_warp_reduce(st);
            const int64_t fw = part_owner(cc.r * p.RV, p.T, p.W);
            const int64_t lw = part_owner((cc.r + 1) * p.RV - 1, p.T, p.W);
            if (fw == lw) {
                finalize_row<DT>(p, cc.r, red, lane);
            } else {
                if (lane == 0) {
                    Partial pt;
                    pt.m = red.m;
                    pt.s = red.s;
                    pt.t2 = red.t2;
                    pt.amax = red.amax;
                    pt.rank = red.rank;
                    pt.pad0 = pt.pad1 = pt.pad2 = 0;
                    p.partials[cc.r + gw] = pt;
                }
                uint32_t old = 0;
                if (lane == 0) {
                    __threadfence();
                    old = atomicAdd(p.counters + cc.r, 1u);
                }
                old = __shfl_sync(0xFFFFFFFFu, old, 0);
                if (old == static_cast<uint32_t>(lw - fw)) {
                    __threadfence();
                    SoftState acc;
                    acc.m = clamp_floor();
                    acc.s = 0.f;
                    acc.t2 = 0.f;
                    acc.amax = INT32_MAX;
                    acc.rank = 0;
                    for (int64_t w = fw + lane; w <= lw; w += 32) {
                        const Partial *pp = p.partials + cc.r + w;
                        SoftState o;
                        o.m = __ldcg(&pp->m);
                        o.s = __ldcg(&pp->s);
                        o.t2 = __ldcg(&pp->t2);
                        o.amax = __ldcg(&pp->amax);
                        o.rank = __ldcg(&pp->rank);
                        acc = soft_merge(acc, o);
                    }
                    acc = soft_warp_reduce(acc);
                    if (lane == 0) p.counters[cc.r] = 0u;  // leave the workspace zeroed
                    finalize_row<DT>(p, cc.r, acc, lane);
                }
            }
            in_piece = false;
            if (row_end) {
                cc.k = 0;
                cc.r += 1;
            }
        }
    }
    if (timed_out) {
        status_or(p.status, SDD_DEV_TIMEOUT);
        // let every copy still in flight land before the CTA's shared memory goes away
        for (int s = 0; s < kStages; ++s)
            if (pending & (1u << s)) (void)mbar_wait_bounded(&bars[s], (phase >> s) & 1u, kWaitPolls);
    }
}

}  // namespace

int scan_max_ctas_per_sm() {
    int n = 0;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, scan_kernel<SDD_BF16>, kThreads, kScanSmem);
    return n;
}

// Opt both instantiations in to their dynamic shared memory on the current device.
cudaError_t scan_prepare_device() {
    cudaError_t e = cudaFuncSetAttribute(scan_kernel<SDD_BF16>, cudaFuncAttributeMaxDynamicSharedMemorySize, kScanSmem);
    if (e != cudaSuccess) return e;
    return cudaFuncSetAttribute(scan_kernel<SDD_F32>, cudaFuncAttributeMaxDynamicSharedMemorySize, kScanSmem);
}

cudaError_t launch_scan(const ScanParams &p, int grid, cudaStream_t stream) {
    if (p.dtype == SDD_BF16)
        scan_kernel<SDD_BF16><<<grid, kThreads, kScanSmem, stream>>>(p);
    else
        scan_kernel<SDD_F32><<<grid, kThreads, kScanSmem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace sdd
