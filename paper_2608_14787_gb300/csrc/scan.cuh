// scan.cuh -- the streaming pass of the path: one read of every drafter and
// target logit, producing per-row partial softmax statistics.
//
// What it computes (per row of logits z over the vocabulary):
//   M = max z, S = sum exp(z - M), T2 = sum exp(z - M) (z - M) log2(e),
//   the lowest index attaining M, and for target rows the saturated rank of
//   the drafted token x: #{v : z(v) > z(x)} + #{v < x : z(v) = z(x)}.
// From these follow the quantities of Sec. 4.2 (raw confidence q = p_draft(x_j),
// LSE, maxprob, entropy) and the target facts that the acceptance rules of
// Sec. 3.1 and App. A.6 read.
//
// How: the rows of the call are laid end to end as one sequence of 16-byte
// vectors, split into contiguous ranges of equal cost, one per warp (a drafter
// vector weighs 10, a target vector 9: the drafter rows' entropy accumulator
// costs more; no per-tile scheduling).  Each warp streams its range through a
// private ring of two 4 KiB shared-memory tiles filled by 1D bulk copies
// (cp.async.bulk + mbarrier), keeps an online-softmax state per lane (packed
// f32x2 arithmetic, exp-sums as double-floats), reduces it across the warp at
// the end of each row piece and publishes a 32-byte partial.  The feature
// instantiation also publishes each drafter row piece's five largest entries
// (group_update / group_top5 below).
// The decide kernel (decide.cu) merges each row's partials and finalises the
// rows; keeping that out of the streaming work keeps it free of register
// spills.  Included by scan.cu (the streaming kernel) and pipe.cu (the
// pipelined round).
#pragma once

#include "internal.h"

namespace sdd {

namespace {

struct Cursor {
    int64_t v;     // absolute vector index
    int64_t r;     // row
    int32_t k;     // vector offset inside the row
};

__device__ __forceinline__ void row_locate(const ScanParams &p, const PartView &pv, int64_t r, int &gi, int64_t &lr,
                                           int &j, int &b, bool &b_ok) {
    gi = (r >= pv.rows0) ? 1 : 0;
    lr = gi ? r - pv.rows0 : r;
    const ScanGroup &G = p.grp[gi];
    const int64_t i = fast_div(lr, p.divNpos[gi]);
    j = static_cast<int>(lr - i * G.npos);
    b = G.bidx ? __ldg(G.bidx + i) : static_cast<int>(i);
    b_ok = (b >= 0 && b < p.B);
    if (!b_ok) b = 0;  // keep every address inside the tensor; the row is flagged at the end
}

__device__ __forceinline__ const char *row_base(const ScanParams &p, const PartView &pv, int64_t r) {
    int gi, j, b;
    int64_t lr;
    bool ok;
    row_locate(p, pv, r, gi, lr, j, b, ok);
    const ScanGroup &G = p.grp[gi];
    return G.base + (static_cast<int64_t>(b) * G.npos + j) * G.stride_bytes;
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
    if (DT == SDD_BF16 && g > clamp_floor()) {
        // Packed compares, two entries per instruction (g is a bf16 value above
        // the clamp value, so clamping cannot change a comparison, and padded
        // entries are -inf).  Entries equal to g rank before the token only at a
        // lower index: counted one by one, in the rare tiles that hold any.
        const uint32_t gb = __float_as_uint(g) >> 16, g2 = gb | (gb << 16);
        int cnt = 0;
        uint32_t eq = 0;
#pragma unroll
        for (int i = 0; i < kVPL; ++i) {
            const uint4 w = tile[lane + 32 * i];
            const uint32_t u[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                cnt += __popc(bf16x2_gt(u[q], g2) & 0x00010001u);
                eq |= bf16x2_eq(u[q], g2);
            }
        }
        if (eq) {
#pragma unroll 1
            for (int i = 0; i < kVPL; ++i) {
                const uint4 w = tile[lane + 32 * i];
#pragma unroll
                for (int e = 0; e < EPV; ++e)
                    cnt += (vec_elem<DT>(w, e) == g && (k0 + lane + 32 * i) * EPV + e < tok) ? 1 : 0;
            }
        }
        return cnt;
    }
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
// that starts at vector k0 of the row (re-read from global memory, all loads
// issued before the first compare; the row's padding and entries past V are
// excluded).
template <int DT>
__device__ __noinline__ int first_index(const char *rowp, int k0, int lane, int RV, int V, float m) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    uint4 w[kVPL];
#pragma unroll
    for (int i = 0; i < kVPL; ++i) {
        const int vec = k0 + lane + 32 * i;
        w[i] = (vec < RV) ? __ldg(reinterpret_cast<const uint4 *>(rowp) + vec) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int i = 0; i < kVPL; ++i) {
        const int vec = k0 + lane + 32 * i;
        if (vec >= RV) break;
        const uint4 c = clamp_vec<DT>(w[i]);
#pragma unroll
        for (int e = 0; e < EPV; ++e)
            if (vec * EPV + e < V && vec_elem<DT>(c, e) == m) return vec * EPV + e;
    }
    return INT32_MAX;
}

// Process one full tile: the lane's vectors are lane, lane+32, ... of the tile.
// Sums are relative to the integer reference st.r (log2 units), so a new
// maximum rescales by an exact power of two.  A new maximum only records the
// tile (st.amax = k0); the exact index is resolved once at the end of the piece.
// Pairs of entries go through the packed f32x2 pipe: y = z log2(e) - r,
// s += 2^y and, for drafter rows (ENT), t2 += 2^y (z - m) log2(e), m the
// lane's maximum (so the dominant term of a peaked row adds 0).  Drafter entries are
// clamped first (so a masked entry adds 0 * finite to t2); target rows need no
// clamp (2^-inf = 0 and the maximum starts at the clamp value).  The lane's
// exp-sum is an fp32 pair (s_hi, s_lo) updated by TwoSum once per tile.
// Returns the lane's tile maximum (clamp value included).
template <int DT, bool ENT>
__device__ __forceinline__ float process_tile(const uint4 *tile, int k0, int lane, SoftState &st, float &s_hi,
                                              float &s_lo) {
    // pass 1: the tile maximum (clamp value included)
    float cm;
    if (DT == SDD_BF16) {
        uint32_t mx = kClampPairBf16;
#pragma unroll
        for (int i = 0; i < kVPL; ++i) {
            const uint4 w = tile[lane + 32 * i];
            const uint32_t vm = bf16x2_max_nan(bf16x2_max_nan(w.x, w.y), bf16x2_max_nan(w.z, w.w));
            mx = bf16x2_max_nan(mx, vm);
        }
        cm = fmax_nan(bf16_lo(mx), bf16_hi(mx));
    } else {
        cm = clamp_floor();
#pragma unroll
        for (int i = 0; i < kVPL; ++i) {
            const uint4 w = tile[lane + 32 * i];
            const float vm = fmax_nan(fmax_nan(__uint_as_float(w.x), __uint_as_float(w.y)),
                                      fmax_nan(__uint_as_float(w.z), __uint_as_float(w.w)));
            cm = fmax_nan(cm, vm);
        }
    }
    if (cm > st.m) {
        st.amax = k0;
        // the entropy accumulator is kept against the lane's maximum: a new
        // maximum shifts it by (m_old - m_new) log2(e) per unit of the sum
        if (ENT) st.t2 = fmaf((st.m - cm) * kLog2e, s_hi + s_lo, st.t2);
        st.m = cm;
        const float rn = ceilf(cm * kLog2e);
        if (rn > st.r) {
            const float k = st.r - rn;
            const float sc = pow2f_int(k);   // exact power of two (0 below the normal range)
            if (ENT) st.t2 *= sc;
            s_hi *= sc;
            s_lo *= sc;
            st.r = rn;
        }
    }
    // pass 2: the exp-sums, the vectors re-read from shared memory two at a
    // time; unrolled, so the reads of later steps issue ahead of the
    // arithmetic of earlier ones
    const float nr = -st.r;
    const f2_t L2 = f2_pack(kLog2e, kLog2e), NR = f2_pack(nr, nr);
    // the lane maximum's own y (the same fma as an entry's): y - DM is an
    // entry's (z - m) log2(e), exactly 0 for the maximum itself
    const float dm = fmaf(st.m, kLog2e, nr);
    const f2_t DM = f2_pack(dm, dm);
    f2_t sa = f2_pack(0.f, 0.f), sb = sa, ta = sa, tb = sa;
    constexpr int PAIRS = (DT == SDD_BF16) ? 4 : 2;   // entry pairs per 16-byte vector
#pragma unroll
    for (int i = 0; i < kVPL; i += 2) {
        uint4 w[2];
        w[0] = tile[lane + 32 * i];
        w[1] = tile[lane + 32 * (i + 1)];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            if (ENT) w[h] = clamp_vec<DT>(w[h]);
            const uint32_t *u = reinterpret_cast<const uint32_t *>(&w[h]);
#pragma unroll
            for (int q = 0; q < PAIRS; ++q) {
                const f2_t z = (DT == SDD_BF16) ? f2_pack(bf16_lo(u[q]), bf16_hi(u[q]))
                                                : f2_pack(__uint_as_float(u[2 * q]), __uint_as_float(u[2 * q + 1]));
                const f2_t y = f2_fma(z, L2, NR);
                float y0, y1;
                f2_unpack(y, y0, y1);
                const f2_t e = f2_pack(ex2(y0), ex2(y1));
                if (q & 1) {
                    sb = f2_add(sb, e);
                    if (ENT) tb = f2_fma(e, f2_sub(y, DM), tb);
                } else {
                    sa = f2_add(sa, e);
                    if (ENT) ta = f2_fma(e, f2_sub(y, DM), ta);
                }
            }
        }
    }
    float s0, s1;
    f2_unpack(f2_add(sa, sb), s0, s1);
    if (ENT) {
        // A tile dominated by one term (the others sum to < 1/16 of it: the
        // lane holding the peak of a peaked row) loses those others' low bits
        // next to it, and they make the row's entropy.  Such a lane's terms
        // are re-summed by the whole warp -- the maximum counted apart, the
        // others summed among themselves -- from shared memory (rare: about
        // one lane-tile per peaked row).
        const float ecm = ex2(fmaf(cm, kLog2e, nr));
        unsigned dom = __ballot_sync(0xFFFFFFFFu, s0 + s1 < 1.0625f * ecm && cm > clamp_floor());
        while (dom) {
            const int src = __ffs(dom) - 1;
            dom &= dom - 1;
            // src's tile maximum and reference (every lane has its own)
            const float cms = __shfl_sync(0xFFFFFFFFu, cm, src);
            const float nrs = __shfl_sync(0xFFFFFFFFu, nr, src);
            // src's 8 vectors, 8 bf16 (or 4 fp32) entries each: lane l takes
            // entries l and l + 32 of them
            constexpr int EN = kVPL * 2 * PAIRS;   // entries of one lane-tile
            float small = 0.f, nmax = 0.f;
#pragma unroll
            for (int t = lane; t < EN; t += 32) {
                const int i = t / (2 * PAIRS), k = t % (2 * PAIRS);
                const uint4 w = clamp_vec<DT>(tile[src + 32 * i]);
                const int wi = (DT == SDD_BF16) ? (k >> 1) : k;   // (word picked by selects, not by index)
                const uint32_t uw = (wi < 2) ? ((wi == 0) ? w.x : w.y) : ((wi == 2) ? w.z : w.w);
                const float z = (DT == SDD_BF16) ? ((k & 1) ? bf16_hi(uw) : bf16_lo(uw)) : __uint_as_float(uw);
                if (z == cms)
                    nmax += 1.f;
                else
                    small += ex2(fmaf(z, kLog2e, nrs));
            }
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
                small += __shfl_xor_sync(0xFFFFFFFFu, small, off);
                nmax += __shfl_xor_sync(0xFFFFFFFFu, nmax, off);
            }
            if (lane == src) {
                s0 = nmax * ecm;   // (nmax <= 64: exact)
                s1 = small;
            }
        }
    }
    float e1, e2, h;
    two_sum(s_hi, s0, h, e1);
    two_sum(h, s1, s_hi, e2);
    s_lo += e1 + e2;
    if (ENT) {
        float t0, t1;
        f2_unpack(f2_add(ta, tb), t0, t1);
        st.t2 += t0 + t1;
    }
    return cm;
}

// Extended features (drafter rows): the five largest clamped entries of a
// piece, with multiplicity.  A group is one lane's kVPL vectors of one tile.
// The five largest entries lie in the five groups with the largest maxima:
// every other group's maximum is at most the fifth largest group maximum,
// which those five groups' maxima reach, so an entry outside them can only
// tie the fifth largest entry.  While the piece streams, each lane keeps its
// five largest tile maxima (order-preserving integer keys) with the tiles'
// first vectors -- one compare per tile; at the piece's end the warp merges
// the lanes' lists (five integer max reductions), re-reads the five groups
// (40 vectors) from global memory and takes their five largest entries.
__device__ __forceinline__ uint32_t fkey(float f) {
    const uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float fkey_inv(uint32_t k) {
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// The lane's tile maximum cm of the tile starting at row vector k0 into its
// list (ck descending, ct the tiles; key 0 = empty).
__device__ __forceinline__ void group_update(float cm, int k0, uint32_t (&ck)[5], int (&ct)[5]) {
    uint32_t key = fkey(cm);
    if (key <= ck[4]) return;
    int k = k0;
#pragma unroll
    for (int j = 0; j < 5; ++j)
        if (key > ck[j]) {
            const uint32_t tk = ck[j];
            const int tt = ct[j];
            ck[j] = key;
            ct[j] = k;
            key = tk;
            k = tt;
        }
}

// The five largest clamped entries (descending; -inf where the piece has
// fewer) of the piece [kb, ke) of row rowp, warp-uniform, from the lanes'
// group lists.  The 40 vectors of the five groups are loaded (two per lane)
// before `between` runs, so their round trip overlaps whatever it waits on.
template <int DT, class Between>
__device__ __forceinline__ void group_top5(const char *rowp, int kb, int ke, int V, int lane, uint32_t (&ck)[5],
                                           int (&ct)[5], float (&t)[5], Between between) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    // (the rounds are rolled loops shifting their results in: this code runs
    // once per piece, and its instructions are fetched while L2 is busy)
    int gl[5], gk[5];   // the five groups: lane and tile
#pragma unroll
    for (int k = 0; k < 5; ++k) {
        gl[k] = 0;
        gk[k] = -1;
        t[k] = -INFINITY;
    }
#pragma unroll 1
    for (int k = 0; k < 5; ++k) {
        const uint32_t m = __reduce_max_sync(0xFFFFFFFFu, ck[0]);
        const int owner = __ffs(__ballot_sync(0xFFFFFFFFu, ck[0] == m)) - 1;
        const int tile = __shfl_sync(0xFFFFFFFFu, ct[0], owner);   // -1 when every list is empty
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            gl[j] = gl[j + 1];
            gk[j] = gk[j + 1];
        }
        gl[4] = owner;
        gk[4] = tile;
        if (lane == owner) {
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                ck[j] = ck[j + 1];
                ct[j] = ct[j + 1];
            }
            ck[4] = 0u;
            ct[4] = -1;
        }
    }
    // vector u (0..39) of the groups: group u / 8, its (u % 8)-th vector;
    // lane q takes u = q and u = q + 32
    int vec[2];
    uint4 w[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int u = lane + 32 * h;
        const int g = u >> 3, j = u & 7;
        int gk_ = -1, gl_ = 0;
#pragma unroll
        for (int k = 0; k < 5; ++k)
            if (g == k) {
                gk_ = gk[k];
                gl_ = gl[k];
            }
        const int v = (gk_ >= 0) ? gk_ + gl_ + 32 * j : -1;
        vec[h] = (u < 40 && v >= kb && v < ke) ? v : -1;
        w[h] = (vec[h] >= 0) ? __ldg(reinterpret_cast<const uint4 *>(rowp) + vec[h]) : make_uint4(0, 0, 0, 0);
    }
    between();
    float e[2 * EPV];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const uint4 c = clamp_vec<DT>(w[h]);
#pragma unroll
        for (int j = 0; j < EPV; ++j)
            e[h * EPV + j] = (vec[h] >= 0 && vec[h] * EPV + j < V) ? vec_elem<DT>(c, j) : -INFINITY;
    }
#pragma unroll 1
    for (int k = 0; k < 5; ++k) {   // five rounds: the warp's largest remaining entry
        float lm = e[0];
#pragma unroll
        for (int j = 1; j < 2 * EPV; ++j) lm = fmaxf(lm, e[j]);
        const uint32_t m = __reduce_max_sync(0xFFFFFFFFu, fkey(lm));
#pragma unroll
        for (int j = 0; j < 4; ++j) t[j] = t[j + 1];
        t[4] = fkey_inv(m);
        const int owner = __ffs(__ballot_sync(0xFFFFFFFFu, fkey(lm) == m)) - 1;
        if (lane == owner) {
            bool done = false;
#pragma unroll
            for (int j = 0; j < 2 * EPV; ++j)
                if (!done && fkey(e[j]) == m) {
                    e[j] = -INFINITY;
                    done = true;
                }
        }
    }
}

// Drafted token of global row r, if the row has one (load issued, not waited on).
struct RowTok {
    int t;
    bool has;
};
__device__ __forceinline__ RowTok row_token(const ScanParams &p, const PartView &pv, int64_t r) {
    RowTok x{0, false};
    if (r < pv.rows) {
        int gi, j, b;
        int64_t lr;
        bool ok;
        row_locate(p, pv, r, gi, lr, j, b, ok);
        if (j < p.gamma) {
            x.t = __ldg(p.tokens + static_cast<int64_t>(b) * p.gamma + j);
            x.has = true;
        }
    }
    return x;
}
// Clamped logit of row r at its drafted token (NaN if none or out of range).
template <int DT>
__device__ __forceinline__ float token_logit(const ScanParams &p, const PartView &pv, int64_t r, RowTok x) {
    if (!x.has || x.t < 0 || x.t >= p.V) return __int_as_float(0x7FC00000);
    return fmax_nan(logit_at<DT>(row_base(p, pv, r), x.t), clamp_floor());
}

// The streaming work of one warp of the CTA, streaming warp gw (below p.W;
// blockIdx.x * p.wpc + warp - p.warp0), once the work ahead of it in the
// stream has completed.  smem is the CTA's ring area, ring_bytes(STAGES,
// n_rings): one ring of STAGES tiles per streaming warp, then their barriers;
// this warp's is ring ring_idx.  FEAT: also the five largest logits of
// every drafter row piece (extended features); without it the code is
// unchanged.
template <int DT, bool FEAT, int STAGES = kStages>
__device__ __forceinline__ void scan_warp(const ScanParams &p, unsigned char *smem, int64_t gw, int ring_idx,
                                          int n_rings) {
    constexpr int kStages = STAGES;
    const int lane = threadIdx.x & 31;
    const PartView pv = part_view(p);
    if (gw >= pv.W) return;   // (a device block count can leave warps without work)
    // The sampling draw's arrival counters of this call's blocks start at zero
    // (the decide kernel behind this one reads them only after this grid has
    // completed), so the workspace needs no zero fill and calls of any shape
    // that fits it may follow one another.
    if (gw == 0 && p.dec.enabled && p.dec.res_count != nullptr)
        for (int i = lane; i < pv.nb; i += 32) p.dec.res_count[i] = 0u;
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    const int tail = p.V % EPV;  // valid entries of the last vector of a row (0 = full)

    unsigned char *ring = smem + ring_idx * (kStages * kTileBytes);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + n_rings * kStages * kTileBytes) + ring_idx * kStages;
    if (lane == 0) {
#pragma unroll
        for (int s = 0; s < kStages; ++s) mbar_init(&bars[s], 1);
        fence_mbar_init();
    }
    __syncwarp();

    const int64_t v0 = part_start(p, pv, gw), v1 = part_start(p, pv, gw + 1);
    Cursor pc{v0, fast_div(v0, p.divRV), 0};
    pc.k = static_cast<int32_t>(v0 - pc.r * p.RV);
    Cursor cc = pc;
    const char *prow = row_base(p, pv, pc.r);
    const uint64_t pol = l2_evict_first_policy();   // the logits are read once
    uint32_t pending = 0;  // slots with a copy in flight
    uint32_t phase = 0;    // parity bit per slot
    bool drop = p.drop_copy != 0 && gw == 0;   // test hook: this warp's first copy is never issued

    auto issue = [&](int slot) {
        const int n = static_cast<int>(min(static_cast<int64_t>(min(kTileVec, p.RV - pc.k)), v1 - pc.v));
        if (drop) {
            // nothing will ever complete this slot's barrier: the consumer's
            // bounded wait runs out (no copy is in flight for the drain)
            drop = false;
        } else {
            if (lane == 0) {
            // the slot's previous contents were consumed into registers before the
            // warp reached this point (__syncwarp), so the copy may overwrite it
                mbar_arrive_expect_tx(&bars[slot], static_cast<uint32_t>(n) * 16u);
                bulk_g2s(ring + slot * kTileBytes, prow + static_cast<int64_t>(pc.k) * 16,
                         static_cast<uint32_t>(n) * 16u, &bars[slot], pol);
            }
            pending |= 1u << slot;
        }
        pc.v += n;
        pc.k += n;
        if (pc.k == p.RV && pc.v < v1) {
            pc.k = 0;
            pc.r += 1;
            prow = row_base(p, pv, pc.r);
        }
    };
    for (int s = 0; s < kStages && pc.v < v1; ++s) issue(s);

    // Drafted tokens and their logits run ahead of the stream: the token two
    // rows ahead and the logit one row ahead are in flight while the current
    // piece streams, so no piece start waits on a dependent pair of loads.
    RowTok tokA = row_token(p, pv, cc.r), tokB = row_token(p, pv, cc.r + 1);
    float gA = token_logit<DT>(p, pv, cc.r, tokA);

    SoftState st = soft_identity();
    uint32_t ck[5];        // FEAT: the lane's five largest tile maxima of the piece (keys) ...
    int ct[5];             // ... and their tiles' first vectors (drafter rows)
    int kb = 0;            // FEAT: the piece's first vector in the row
    float s_hi = 0.f, s_lo = 0.f;   // the lane's exp-sum as an fp32 pair
    bool in_piece = false;
    bool ent = false;      // warp-uniform: drafter row (entropy accumulator, clamped entries)
    int tok = -1;          // drafted token of the current row (-1: none or out of range)
    bool tok_bad = false;  // the row has a drafted token outside [0, V)
    float g = 0.f;         // its clamped logit (NaN if none)
    bool rank_on = false;  // warp-uniform: target row whose token's rank is still below kcap
    int wrank = 0;         // warp-uniform running rank count
    const char *crow = nullptr;
    int slot = 0;
    bool timed_out = false;
    while (cc.v < v1) {
        const int n = static_cast<int>(min(static_cast<int64_t>(min(kTileVec, p.RV - cc.k)), v1 - cc.v));
        if (!in_piece) {
            st = soft_identity();
            if (FEAT) {
#pragma unroll
                for (int k = 0; k < 5; ++k) {
                    ck[k] = 0u;
                    ct[k] = -1;
                }
                kb = cc.k;
            }
            s_hi = 0.f;
            s_lo = 0.f;
            int gi, j, b;
            int64_t lr;
            bool ok;
            row_locate(p, pv, cc.r, gi, lr, j, b, ok);
            const ScanGroup &G = p.grp[gi];
            crow = G.base + (static_cast<int64_t>(b) * G.npos + j) * G.stride_bytes;
            ent = G.kind == 0;
            const bool tok_ok = tokA.has && tokA.t >= 0 && tokA.t < p.V;
            tok = tok_ok ? tokA.t : -1;
            tok_bad = tokA.has && !tok_ok;
            g = gA;
            // advance the prefetch: logit of the next row, token of the one after
            gA = token_logit<DT>(p, pv, cc.r + 1, tokB);
            tokA = tokB;
            tokB = row_token(p, pv, cc.r + 2);
            rank_on = !ent && tok >= 0;
            wrank = 0;
            in_piece = true;
        }
        // warp-uniform outcome: a phase that one lane saw complete is complete for all
        if (!__any_sync(0xFFFFFFFFu, mbar_wait_bounded(&bars[slot], (phase >> slot) & 1u, p.wait_polls))) {
            timed_out = true;
            break;
        }
        uint4 *tile = reinterpret_cast<uint4 *>(ring + slot * kTileBytes);
        const bool row_end = (cc.k + n == p.RV);
        if (n < kTileVec || (row_end && tail)) pad_tile<DT>(tile, n, lane, row_end, tail);
        const float cm = ent ? process_tile<DT, true>(tile, cc.k, lane, st, s_hi, s_lo)
                             : process_tile<DT, false>(tile, cc.k, lane, st, s_hi, s_lo);
        if (FEAT && ent) group_update(cm, cc.k, ck, ct);
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
            auto resolve = [&]() {
                if (st.m == M && st.amax != INT32_MAX) idx = first_index<DT>(crow, st.amax, lane, p.RV, p.V, M);
            };
            float top[5];
            if (FEAT && ent)
                group_top5<DT>(crow, kb, cc.k, p.V, lane, ck, ct, top, resolve);   // (cc.k: the piece's end)
            else
                resolve();
            st.amax = idx;
            st.rank = (lane == 0) ? wrank : 0;
            st.sh = s_hi;
            st.sl = s_lo;
            const SoftState red = soft_warp_reduce(st);
            if (FEAT && ent) {
                if (lane == 0) {
                FeatPartial fp;
#pragma unroll
                for (int k = 0; k < 5; ++k) fp.top[k] = top[k];
                fp.pad[0] = fp.pad[1] = fp.pad[2] = 0.f;
                p.feat[cc.r + gw] = fp;
                }
            }
            if (lane == 0) {
                Partial pt;
                pt.m = red.m;
                pt.r = red.r;
                pt.t2 = red.t2;
                pt.sh = red.sh;
                pt.sl = red.sl;
                pt.amax = red.amax;
                pt.rank = tok_bad ? -1 : red.rank;
                pt.g = g;
                p.partials[cc.r + gw] = pt;
            }
            in_piece = false;
            if (row_end) {
                cc.k = 0;
                cc.r += 1;
            }
        }
    }
    if (timed_out) {
        if (lane == 0) status_or(p.status, SDD_DEV_TIMEOUT);
        // let every copy still in flight land before the CTA's shared memory
        // goes away (the full limit, whatever the ring waits were given)
        for (int s = 0; s < kStages; ++s)
            if (pending & (1u << s)) (void)mbar_wait_bounded(&bars[s], (phase >> s) & 1u, kWaitPolls);
    }
}

}  // namespace

}  // namespace sdd
