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
#include "rules.cuh"

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

// A tile that is not full, or that ends a row whose length is not a whole
// number of vectors, is completed in shared memory with -inf entries so that
// the hot loop can read every vector of the tile unconditionally.
template <int DT>
__device__ __noinline__ void pad_tile(uint4 *tile, int n, int lane, bool row_end, int tail) {
    const uint4 ninf = (DT == SDD_BF16) ? make_uint4(kNegInfPairBf16, kNegInfPairBf16, kNegInfPairBf16, kNegInfPairBf16)
                                        : make_uint4(0xFF800000u, 0xFF800000u, 0xFF800000u, 0xFF800000u);
    for (int idx = n + lane; idx < kTileVec; idx += 32) tile[idx] = ninf;
    if (row_end && tail && lane == ((n - 1) & 31)) {
        uint4 w = tile[n - 1];
        mask_tail<DT>(w, tail);
        tile[n - 1] = w;
    }
    __syncwarp();
}

// Entries of the lane's vectors in a (full, padded) tile that rank before the
// drafted token tok: value above g, or equal to g at a lower index.
template <int DT>
__device__ __noinline__ int count_before(const uint4 *tile, int n, int k0, int lane, float g, int tok) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    int cnt = 0;
#pragma unroll 1
    for (int i = 0; i < kVPL; ++i) {
        const int idx = lane + 32 * i;
        if (idx >= n) break;
        const uint4 w = clamp_vec<DT>(tile[idx]);
#pragma unroll
        for (int e = 0; e < EPV; ++e) {
            const float z = vec_elem<DT>(w, e);
            const int v = (k0 + idx) * EPV + e;
            cnt += (z > g || (z == g && v < tok)) ? 1 : 0;
        }
    }
    return cnt;
}

// Resolve a lane's argmax: the first of its entries equal to m inside the tile
// that starts at vector k0 of the row (re-read from global memory; the row's
// padding and entries past V are excluded).
template <int DT>
__device__ __noinline__ int first_index(const char *rowp, int k0, int lane, int RV, int V, float m) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
#pragma unroll 1
    for (int i = 0; i < kVPL; ++i) {
        const int vec = k0 + lane + 32 * i;
        if (vec >= RV) break;
        const uint4 w = clamp_vec<DT>(__ldg(reinterpret_cast<const uint4 *>(rowp) + vec));
#pragma unroll
        for (int e = 0; e < EPV; ++e)
            if (vec * EPV + e < V && vec_elem<DT>(w, e) == m) return vec * EPV + e;
    }
    return INT32_MAX;
}

// Process one full tile: the lane's vectors are lane, lane+32, ... of the tile.
// Sums are relative to the integer reference st.r (log2 units), so a new
// maximum rescales by an exact power of two.  A new maximum only records the
// tile (st.amax = k0); the exact index is resolved once at the end of the piece.
// Error-free sum of two fp32 values (Knuth's TwoSum): a + b = s + err exactly.
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &err) {
    s = a + b;
    const float bb = s - a;
    err = (a - (s - bb)) + (b - bb);
}

// The lane's running exp-sum is kept as an unevaluated fp32 pair (hi, lo)
// (compensated summation), so the hot loop needs no fp64 arithmetic; the pair
// is folded into st.s (fp64) at the end of each row piece.
template <int DT>
__device__ __forceinline__ float process_tile(const uint4 *tile, int k0, int lane, SoftState &st, float &s_hi,
                                              float &s_lo) {
    uint4 w[kVPL];
#pragma unroll
    for (int i = 0; i < kVPL; ++i) w[i] = clamp_vec<DT>(tile[lane + 32 * i]);
    float cm;
    if (DT == SDD_BF16) {
        uint32_t mx = kClampPairBf16;
#pragma unroll
        for (int i = 0; i < kVPL; ++i) {
            const uint32_t *u = reinterpret_cast<const uint32_t *>(&w[i]);
#pragma unroll
            for (int q = 0; q < 4; ++q) mx = bf16x2_max_nan(mx, u[q]);
        }
        cm = fmax_nan(bf16_lo(mx), bf16_hi(mx));
    } else {
        cm = clamp_floor();
#pragma unroll
        for (int i = 0; i < kVPL; ++i) {
            const float *f = reinterpret_cast<const float *>(&w[i]);
#pragma unroll
            for (int q = 0; q < 4; ++q) cm = fmax_nan(cm, f[q]);
        }
    }
    if (cm > st.m) {
        st.amax = k0;
        st.m = cm;
        const float rn = ceilf(cm * kLog2e);
        if (rn > st.r) {
            const float k = st.r - rn;
            const float sc = pow2f_int(k);   // exact power of two (0 below the normal range)
            st.t2 = sc * (st.t2 + k * (s_hi + s_lo));
            s_hi *= sc;
            s_lo *= sc;
            st.r = rn;
        }
    }
    // y = z log2(e) - r; s += 2^y; t2 += 2^y y   (two accumulators each)
    const float nr = -st.r;
    float s0 = 0.f, s1 = 0.f, t0 = 0.f, t1 = 0.f;
#pragma unroll
    for (int i = 0; i < kVPL; ++i) {
        const uint32_t *u = reinterpret_cast<const uint32_t *>(&w[i]);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            if (DT == SDD_BF16) {
                const float y0 = fmaf(bf16_lo(u[q]), kLog2e, nr);
                const float y1 = fmaf(bf16_hi(u[q]), kLog2e, nr);
                const float e0 = ex2(y0), e1 = ex2(y1);
                s0 += e0;
                t0 = fmaf(e0, y0, t0);
                s1 += e1;
                t1 = fmaf(e1, y1, t1);
            } else {
                const float y0 = fmaf(__uint_as_float(u[q]), kLog2e, nr);
                const float e0 = ex2(y0);
                if (q & 1) {
                    s1 += e0;
                    t1 = fmaf(e0, y0, t1);
                } else {
                    s0 += e0;
                    t0 = fmaf(e0, y0, t0);
                }
            }
        }
    }
    float e1, e2, h;
    two_sum(s_hi, s0, h, e1);
    two_sum(h, s1, s_hi, e2);
    s_lo += e1 + e2;
    st.t2 += t0 + t1;
    return cm;
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
    const bool valid = b_ok && isfinite(st.m) && st.m > clamp_floor() && isfinite(st.s) && st.s > 0.0;
    if (lane != 0) return;
    const float nanf_ = __int_as_float(0x7FC00000);
    float g = nanf_;
    if (tok_ok) g = fmax_nan(load_logit<DT>(rowp, tok), clamp_floor());
    RowRec rec;
    const int64_t o = static_cast<int64_t>(b) * p.gamma + j;
    if (valid) {
        // The lane that held the row maximum M took its term as ex2(y_M) with
        // y_M = M log2(e) - ceil(M log2(e)) (its reference when M arrived).  On a
        // peaked row that one term dominates S, so its MUFU approximation error
        // is replaced by the exact power of two (scaled to the final reference).
        const float rM = ceilf(st.m * kLog2e);
        const float yM = fmaf(st.m, kLog2e, -rM);
        const double S = st.s + (exp2(static_cast<double>(yM)) - static_cast<double>(ex2(yM))) * pow2d_int(rM - st.r);
        st.s = S;
        // all in fp64: LSE = r ln2 + ln S (S relative to the reference r)
        const double lnS = log(st.s);
        const double lse = static_cast<double>(st.r) * kLn2d + lnS;
        rec.lse = lse;
        rec.M = st.m;
        rec.g = g;
        rec.logq = static_cast<float>(static_cast<double>(g) - lse);
        rec.q = static_cast<float>(exp(static_cast<double>(g) - lse));
        rec.argmax = st.amax;
        rec.rank = min(st.rank, p.kcap);
        if (G.kind == 0 && b_ok) {
            if (G.q) G.q[o] = tok_ok ? rec.q : nanf_;
            if (G.logq) G.logq[o] = tok_ok ? rec.logq : nanf_;
            if (G.maxprob) G.maxprob[o] = static_cast<float>(exp(static_cast<double>(st.m) - lse));
            if (G.lse) G.lse[o] = lse;
            if (G.entropy) G.entropy[o] = static_cast<float>(lnS - kLn2d * static_cast<double>(st.t2) / st.s);
            if (G.argmax) G.argmax[o] = st.amax;
        }
    } else {
        rec.lse = __longlong_as_double(0x7FF8000000000000ll);
        rec.M = rec.g = rec.q = rec.logq = nanf_;
        rec.argmax = -1;
        rec.rank = INT32_MAX;
        if (G.kind == 0 && b_ok) {
            if (G.q) G.q[o] = nanf_;
            if (G.logq) G.logq[o] = nanf_;
            if (G.maxprob) G.maxprob[o] = nanf_;
            if (G.lse) G.lse[o] = rec.lse;
            if (G.entropy) G.entropy[o] = nanf_;
            if (G.argmax) G.argmax[o] = -1;
        }
        if (b_ok) status_or(p.status, SDD_DEV_NONFINITE);
    }
    if (has_tok && !tok_ok) {
        rec.q = rec.logq = rec.g = nanf_;
        rec.rank = INT32_MAX;
    }
    if ((has_tok && !tok_ok) || !b_ok) status_or(p.status, SDD_DEV_BAD_TOKEN);
    G.rec[lr] = rec;
}

// A row of list block i is final: count it, and let the warp that completes
// the block evaluate the block's decisions (rules.cuh).
template <int DT>
__device__ __forceinline__ void block_arrive(const ScanParams &p, int64_t r, int lane) {
    const int gi = (r >= p.rows0) ? 1 : 0;
    const int64_t lr = gi ? r - p.rows0 : r;
    const int i = static_cast<int>(lr / p.grp[gi].npos);
    __syncwarp();
    uint32_t old = 0;
    if (lane == 0) {
        __threadfence();
        old = atomicAdd(p.dec.blk_count + i, 1u);
    }
    old = __shfl_sync(0xFFFFFFFFu, old, 0);
    if (old == static_cast<uint32_t>(p.dec.rows_per_block - 1)) {
        __threadfence();
        __shared__ int s_rule_L[kWarpsPerCta][kMaxRules], s_rule_corr[kWarpsPerCta][kMaxRules];
        const int w = threadIdx.x >> 5;
        block_decide<DT>(p.dec, i, lane, s_rule_L[w], s_rule_corr[w]);
        if (lane == 0) p.dec.blk_count[i] = 0u;   // leave the workspace zeroed
    }
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
            // the slot's previous contents were consumed into registers before the
            // warp reached this point (__syncwarp), so the copy may overwrite it
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

    SoftState st = soft_identity();
    float s_hi = 0.f, s_lo = 0.f;   // the lane's exp-sum as an fp32 pair
    bool in_piece = false;
    int tok = -1;          // drafted token of the current target row (-1: none)
    float g = 0.f;         // its clamped logit
    bool rank_on = false;  // warp-uniform: the rank of tok is still below kcap
    int wrank = 0;         // warp-uniform running rank count
    const char *crow = nullptr;
    int slot = 0;
    bool timed_out = false;
    while (cc.v < v1) {
        const int n = static_cast<int>(min(static_cast<int64_t>(min(kTileVec, p.RV - cc.k)), v1 - cc.v));
        if (!in_piece) {
            st = soft_identity();
            s_hi = 0.f;
            s_lo = 0.f;
            int gi, j, b;
            int64_t lr;
            bool ok;
            row_locate(p, cc.r, gi, lr, j, b, ok);
            const ScanGroup &G = p.grp[gi];
            crow = G.base + (static_cast<int64_t>(b) * G.npos + j) * G.stride_bytes;
            tok = -1;
            g = 0.f;
            if (G.kind == 1 && j < p.gamma) {
                const int t = __ldg(p.tokens + static_cast<int64_t>(b) * p.gamma + j);
                if (t >= 0 && t < p.V) {
                    tok = t;
                    g = fmax_nan(load_logit<DT>(crow, t), clamp_floor());
                }
            }
            rank_on = tok >= 0;
            wrank = 0;
            in_piece = true;
        }
        if (!mbar_wait_bounded(&bars[slot], (phase >> slot) & 1u, kWaitPolls)) {
            timed_out = true;
            break;
        }
        uint4 *tile = reinterpret_cast<uint4 *>(ring + slot * kTileBytes);
        const bool row_end = (cc.k + n == p.RV);
        if (n < kTileVec || (row_end && tail)) pad_tile<DT>(tile, n, lane, row_end, tail);
        const float cm = process_tile<DT>(tile, cc.k, lane, st, s_hi, s_lo);
        if (rank_on) {
            const bool want = cm >= g;
            if (__any_sync(0xFFFFFFFFu, want)) {
                int c = want ? count_before<DT>(tile, n, cc.k, lane, g, tok) : 0;
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) c += __shfl_xor_sync(0xFFFFFFFFu, c, off);
                wrank += c;
                if (wrank >= p.kcap) rank_on = false;
            }
        }
        __syncwarp();
        phase ^= 1u << slot;
        pending &= ~(1u << slot);
        if (n < kTileVec || (row_end && tail)) fence_proxy_async_smem();  // generic writes of pad_tile
        if (pc.v < v1) issue(slot);
        slot = (slot + 1 == kStages) ? 0 : slot + 1;
        cc.v += n;
        cc.k += n;
        if (row_end || cc.v == v1) {
            // end of this warp's piece of row cc.r: exact argmax of the piece,
            // then the warp's partial state
            float M = st.m;
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) M = fmax_nan(M, __shfl_xor_sync(0xFFFFFFFFu, M, off));
            int idx = INT32_MAX;
            if (st.m == M && st.amax != INT32_MAX) idx = first_index<DT>(crow, st.amax, lane, p.RV, p.V, M);
            st.amax = idx;
            st.rank = (lane == 0) ? wrank : 0;
            st.s = static_cast<double>(s_hi) + static_cast<double>(s_lo);
            SoftState red = soft_warp_reduce(st);
            const int64_t fw = part_owner(cc.r * p.RV, p.T, p.W);
            const int64_t lw = part_owner((cc.r + 1) * p.RV - 1, p.T, p.W);
            if (fw == lw) {
                finalize_row<DT>(p, cc.r, red, lane);
                if (p.dec.enabled) block_arrive<DT>(p, cc.r, lane);
            } else {
                if (lane == 0) {
                    Partial pt;
                    pt.m = red.m;
                    pt.r = red.r;
                    pt.t2 = red.t2;
                    pt.amax = red.amax;
                    pt.rank = red.rank;
                    pt.pad = 0;
                    pt.s = red.s;
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
                    SoftState acc = soft_identity();
                    for (int64_t w = fw + lane; w <= lw; w += 32) {
                        const Partial *pp = p.partials + cc.r + w;
                        SoftState o;
                        o.m = __ldcg(&pp->m);
                        o.r = __ldcg(&pp->r);
                        o.t2 = __ldcg(&pp->t2);
                        o.s = __ldcg(&pp->s);
                        o.amax = __ldcg(&pp->amax);
                        o.rank = __ldcg(&pp->rank);
                        acc = soft_merge(acc, o);
                    }
                    acc = soft_warp_reduce(acc);
                    if (lane == 0) p.counters[cc.r] = 0u;  // leave the workspace zeroed
                    finalize_row<DT>(p, cc.r, acc, lane);
                    if (p.dec.enabled) block_arrive<DT>(p, cc.r, lane);
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
