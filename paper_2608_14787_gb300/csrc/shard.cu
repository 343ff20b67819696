// shard.cu -- the per-slice half of the vocabulary-sharded round (a
// tensor-parallel LM head: each rank holds one contiguous vocabulary slice
// [v0, v1) of every drafter and target row).
//
//  * shard_partials_kernel -- one CTA per row of the slice.  Each thread
//    streams its 16-byte vectors (ascending), keeping the online-softmax state
//    of its entries relative to an integer reference in log2 units (a new
//    maximum rescales the sums by an exact power of two), the first index of
//    its maximum and the drafter entropy accumulator; on target rows of a
//    round with the top-k rule each warp keeps its kcap highest-ranked
//    vectors in a list held one key per lane.  The CTA merges the threads'
//    states in thread order and selects the slice's kcap largest entries
//    (value descending, index ascending), then one thread writes the row's
//    record.  Logits are floored at -2^23 as in the
//    streaming kernel; entries past the slice width weigh nothing.
//
// The records of all slices are merged, and every rule of the round runs, in
// decide_kernel (rules.cuh: merge_row_shards); the draw that follows the
// exchange of the slices' draw-row masses is shard_draw_kernel (decide.cu).
#include "rules.cuh"

namespace sdd {

namespace {

// One CTA of four warps per row and eight CTAs per SM (64 registers): a c3
// slice holds 1,040 rows, one wave on 152 SMs.  (With 256-thread CTAs, four
// per SM, and per-thread candidate lists in shared memory, a half-vocabulary
// slice took 84 us; as here, ~55 us.)
constexpr int kShardThreads = 128;
constexpr int kShardMinCtas = 8;
constexpr int kShardU = 4;   // 16-byte vectors per thread in flight

// Order key of a candidate: larger value first, then lower index (an
// unsigned comparison of the keys is that order; a real entry's key is > 0).
__device__ __forceinline__ uint64_t cand_key(float z, int v) {
    uint32_t u = __float_as_uint(z);
    u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
    return (static_cast<uint64_t>(u) << 32) | static_cast<uint32_t>(~static_cast<uint32_t>(v));
}
__device__ __forceinline__ float cand_value(uint64_t key) {
    const uint32_t e = static_cast<uint32_t>(key >> 32);
    return __uint_as_float((e & 0x80000000u) ? (e & 0x7FFFFFFFu) : ~e);
}
__device__ __forceinline__ int cand_index(uint64_t key) {
    return static_cast<int>(~static_cast<uint32_t>(key));
}

__device__ __forceinline__ uint64_t warp_max_u64(uint64_t v) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const uint64_t o = __shfl_xor_sync(0xFFFFFFFFu, v, off);
        v = (o > v) ? o : v;
    }
    return v;
}

// The rare paths of the per-element work, kept out of line so that the
// common path is not compiled into predicated copies of them.
//
// The first index (ascending) of the value m in one vector whose entries
// start at index idx0; m is one of them.
template <int DT>
__device__ __noinline__ int vector_first_index(uint4 w, int idx0, float m) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    for (int e = 0; e < EPV; ++e)
        if (vec_elem_sel<DT>(w, e) == m) return idx0 + e;
    return INT32_MAX;
}

// One key into a warp's candidate list: lane k < kl holds the list's k-th
// key (descending; 0 = empty), every lane returns its new entry.
__device__ __forceinline__ uint64_t warp_list_insert(uint64_t lk, uint64_t key, int kl, int lane) {
    const int pos = __popc(__ballot_sync(0xFFFFFFFFu, lk > key));   // keys ranking before it
    const uint64_t up = __shfl_up_sync(0xFFFFFFFFu, lk, 1);
    if (lane < kl && lane > pos) return up;
    if (lane < kl && lane == pos) return key;
    return lk;
}

// The running state of one thread's entries of a row.
struct ShardAcc {
    SoftState st;
    float s_hi, s_lo;   // exp-sum relative to 2^r, as an unevaluated pair
    bool nan;
    uint64_t lk;        // candidate rows: this lane's entry of the warp's list
    float wthr;         // value of the list's last key once full, else -inf
};

// One chunk (kShardU vectors per lane, lane-contiguous) of a row.  DRAFT: a
// drafter row (entropy accumulator, compensated sums); CANDL: a target row
// of a round with the top-k rule (the warp's candidate list); FULL: every
// vector of the warp's chunk lies inside the slice and before a ragged last
// vector (no guards).  Warp-uniform: every lane of the warp runs the same
// chunk, lanes past the end on floored -inf vectors that weigh nothing.
template <int DT, bool DRAFT, bool CANDL, bool FULL>
__device__ __forceinline__ void shard_chunk(const char *row, const ShardParams &sp, int v0, int kl, int lane,
                                            ShardAcc &a) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    constexpr int PAIRS = EPV / 2;
    uint4 w[kShardU];
    float vm[kShardU];   // each vector's maximum (floored; NaN kept)
#pragma unroll
    for (int u = 0; u < kShardU; ++u) {
        const int vec = v0 + u * kShardThreads;
        if (FULL || vec < sp.RVs) {
            w[u] = __ldcs(reinterpret_cast<const uint4 *>(row) + vec);
        } else {
            const uint32_t ni = (DT == SDD_BF16) ? kNegInfPairBf16 : 0xFF800000u;
            w[u] = make_uint4(ni, ni, ni, ni);
        }
    }
    float cm = clamp_floor();
#pragma unroll
    for (int u = 0; u < kShardU; ++u) {
        const int vec = v0 + u * kShardThreads;
        if (!FULL && vec < sp.RVs && (vec + 1) * EPV > sp.Vs) mask_tail<DT>(w[u], sp.Vs - vec * EPV);
        w[u] = clamp_vec<DT>(w[u]);   // entries past the slice and masked ones: the floor
        const uint32_t *q = reinterpret_cast<const uint32_t *>(&w[u]);
        if (DT == SDD_BF16) {
            const uint32_t m2 = bf16x2_max_nan(bf16x2_max_nan(q[0], q[1]), bf16x2_max_nan(q[2], q[3]));
            vm[u] = fmax_nan(bf16_lo(m2), bf16_hi(m2));
        } else {
            vm[u] = fmax_nan(fmax_nan(__uint_as_float(q[0]), __uint_as_float(q[1])),
                             fmax_nan(__uint_as_float(q[2]), __uint_as_float(q[3])));
        }
        cm = fmax_nan(cm, vm[u]);
    }
    a.nan |= isnan(cm);
    if (cm > a.st.m) {
        // a new maximum (rare): its first index, in the first vector that holds it
        int us = kShardU - 1;
#pragma unroll
        for (int u = kShardU - 2; u >= 0; --u) us = (vm[u] == cm) ? u : us;
        uint4 ws = w[kShardU - 1];
#pragma unroll
        for (int u = kShardU - 2; u >= 0; --u) ws = (u == us) ? w[u] : ws;
        a.st.amax = vector_first_index<DT>(ws, (v0 + us * kShardThreads) * EPV, cm);
        // t2 against the maximum (as in the streaming kernel)
        if (DRAFT) a.st.t2 = fmaf((a.st.m - cm) * kLog2e, a.s_hi + a.s_lo, a.st.t2);
        a.st.m = cm;
        const float rn = ceilf(cm * kLog2e);
        if (rn > a.st.r) {
            const float sc = pow2f_int(a.st.r - rn);   // exact power of two (0 below the normal range)
            if (DRAFT) a.st.t2 *= sc;
            a.s_hi *= sc;
            a.s_lo *= sc;
            a.st.r = rn;
        }
    }
    if (CANDL) {
#pragma unroll
        for (int u = 0; u < kShardU; ++u) {
            const int vec = v0 + u * kShardThreads;
            // (a vector tying the last key has a larger index: it ranks after it)
            unsigned pend = __ballot_sync(0xFFFFFFFFu, vm[u] > a.wthr && (FULL || vec < sp.RVs));
            if (pend) {
                const uint64_t mine = cand_key(vm[u], vec);
                while (pend) {
                    const int src = __ffs(pend) - 1;
                    pend &= pend - 1;
                    a.lk = warp_list_insert(a.lk, __shfl_sync(0xFFFFFFFFu, mine, src), kl, lane);
                }
                const uint64_t last = __shfl_sync(0xFFFFFFFFu, a.lk, kl - 1);
                a.wthr = (last != 0ull) ? cand_value(last) : -INFINITY;
            }
        }
    }
    // the exp-sums, two entries at a time (drafter rows: compensated, so
    // that the small terms of a peaked row survive next to its peak)
    const f2_t L2 = f2_pack(kLog2e, kLog2e);
    const float nr = -a.st.r;
    const f2_t NR = f2_pack(nr, nr);
    const float dm = fmaf(a.st.m, kLog2e, nr);
    const f2_t DM = f2_pack(dm, dm);
    f2_t sa = f2_pack(0.f, 0.f), ca = sa, ta = sa;
#pragma unroll
    for (int u = 0; u < kShardU; ++u) {
        const uint32_t *q = reinterpret_cast<const uint32_t *>(&w[u]);
#pragma unroll
        for (int h = 0; h < PAIRS; ++h) {
            const f2_t z = (DT == SDD_BF16) ? f2_pack(bf16_lo(q[h]), bf16_hi(q[h]))
                                            : f2_pack(__uint_as_float(q[2 * h]), __uint_as_float(q[2 * h + 1]));
            const f2_t y = f2_fma(z, L2, NR);
            float y0, y1;
            f2_unpack(y, y0, y1);
            const f2_t e = f2_pack(ex2(y0), ex2(y1));
            if (DRAFT) {
                const f2_t yk = f2_sub(e, ca), t = f2_add(sa, yk);
                ca = f2_sub(f2_sub(t, sa), yk);
                sa = t;
                ta = f2_fma(e, f2_sub(y, DM), ta);
            } else {
                sa = f2_add(sa, e);
            }
        }
    }
    float a0, a1, h, e1, e2;
    f2_unpack(sa, a0, a1);
    two_sum(a.s_hi, a0, h, e1);
    two_sum(h, a1, a.s_hi, e2);
    if (DRAFT) {
        float c0, c1, t0, t1;
        f2_unpack(ca, c0, c1);
        f2_unpack(ta, t0, t1);
        a.s_lo += (e1 + e2) - (c0 + c1);
        a.st.t2 += t0 + t1;
    } else {
        a.s_lo += e1 + e2;
    }
}

// A thread's part of a row: chunks v0 = tid + c * kShardThreads * kShardU,
// run while the warp's first lane is inside the row.
template <int DT, bool DRAFT, bool CANDL>
__device__ __forceinline__ ShardAcc shard_row(const char *row, const ShardParams &sp, int kl, int tid) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    const int lane = tid & 31;
    ShardAcc a;
    a.st = soft_identity();
    a.s_hi = a.s_lo = 0.f;
    a.nan = false;
    a.lk = 0ull;
    a.wthr = -INFINITY;
    const int rvf = (sp.Vs % EPV == 0) ? sp.RVs : sp.RVs - 1;   // vectors wholly inside the slice
    for (int v0 = tid; v0 - lane < sp.RVs; v0 += kShardThreads * kShardU) {
        if ((v0 - lane) + 31 + (kShardU - 1) * kShardThreads < rvf)
            shard_chunk<DT, DRAFT, CANDL, true>(row, sp, v0, kl, lane, a);
        else
            shard_chunk<DT, DRAFT, CANDL, false>(row, sp, v0, kl, lane, a);
    }
    return a;
}

template <int DT, bool CAND>
__global__ void __launch_bounds__(kShardThreads, kShardMinCtas) shard_partials_kernel(const __grid_constant__ ShardParams sp) {
    constexpr int EPV = (DT == SDD_BF16) ? 8 : 4;
    constexpr int NW = kShardThreads / 32;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t r = blockIdx.x;
    const int64_t nd = static_cast<int64_t>(sp.B) * sp.gamma;
    const bool drafter = r < nd;
    const char *row;
    int tok = -1;
    bool has_tok;
    if (drafter) {
        row = sp.zd + r * sp.stride_bytes;
        tok = __ldg(sp.tokens + r);
        has_tok = true;
    } else {
        const int64_t rr = r - nd;
        const int b = static_cast<int>(rr / (sp.gamma + 1)), j = static_cast<int>(rr % (sp.gamma + 1));
        row = sp.zt + rr * sp.stride_bytes;
        has_tok = j < sp.gamma;
        if (has_tok) tok = __ldg(sp.tokens + static_cast<int64_t>(b) * sp.gamma + j);
    }
    const bool tok_out = has_tok && (tok < 0 || tok >= sp.V);
    const bool in_slice = has_tok && !tok_out && tok >= sp.v0 && tok < sp.v0 + sp.Vs;
    const bool cand = CAND && !drafter;

    // target rows: the warp's kcap highest-ranked vectors, ranked by their
    // maximum (larger first, then lower vector index), held one key per lane
    // in descending order.  The kcap largest entries of the slice lie in the
    // slice's kcap highest-ranked vectors (an entry outside them has kcap
    // vectors ranked above its own, each holding an entry that ranks before
    // it), so the CTA selects those vectors at the end and takes the kcap
    // largest of their entries.
    const int kl = cand ? sp.kcap : 0;   // list length
    ShardAcc acc = drafter ? shard_row<DT, true, false>(row, sp, 0, tid)
                           : (cand ? shard_row<DT, false, CAND>(row, sp, kl, tid)
                                   : shard_row<DT, false, false>(row, sp, 0, tid));
    SoftState st = acc.st;
    const uint64_t lk = acc.lk;
    const bool nan = acc.nan;
    const float s_hi = acc.s_hi, s_lo = acc.s_lo;
    if (nan) st.m = qnan();
    st.sh = s_hi;
    st.sl = s_lo;
    st.rank = 0;

    // CTA merge of the threads' states, in thread order
    __shared__ SoftState s_st[NW];
    const SoftState wst = soft_warp_reduce(st);
    if (lane == 0) s_st[warp] = wst;

    // the slice's kcap highest-ranked vectors: the warps' lists in shared
    // memory, kcap rounds of a warp maximum over them (one warp); then the
    // kcap largest entries of those vectors (one warp, kcap rounds)
    __shared__ uint64_t s_wl[NW * SDD_SHARD_KMAX];
    __shared__ uint64_t s_top[SDD_SHARD_KMAX];
    __shared__ uint64_t s_ent[SDD_SHARD_KMAX * 8];
    const int kc = cand ? sp.kcap : 0;
    if (lane < kc) s_wl[warp * SDD_SHARD_KMAX + lane] = lk;
    __syncthreads();
    if (kc > 0 && warp == 0) {
        constexpr int PER = (NW * SDD_SHARD_KMAX + 31) / 32;
        uint64_t mk[PER];
#pragma unroll
        for (int t = 0; t < PER; ++t) {
            const int i = lane + 32 * t;
            mk[t] = (i < NW * SDD_SHARD_KMAX && (i % SDD_SHARD_KMAX) < kc) ? s_wl[i] : 0ull;
        }
        for (int round = 0; round < kc; ++round) {
            uint64_t mine = 0ull;
#pragma unroll
            for (int t = 0; t < PER; ++t) mine = (mk[t] > mine) ? mk[t] : mine;
            const uint64_t best = warp_max_u64(mine);
#pragma unroll
            for (int t = 0; t < PER; ++t) mk[t] = (best != 0ull && mk[t] == best) ? 0ull : mk[t];   // unique keys
            if (lane == 0) s_top[round] = best;
        }
    }
    __syncthreads();
    if (kc > 0) {
        // the entries of the selected vectors (re-read: kc x 16 bytes), keyed by value and global index
        if (tid < kc) {
            const uint64_t vk = s_top[tid];
            uint4 wv = make_uint4(0, 0, 0, 0);
            const int vec = (vk != 0ull) ? cand_index(vk) : -1;
            if (vec >= 0) wv = clamp_vec<DT>(__ldg(reinterpret_cast<const uint4 *>(row) + vec));
#pragma unroll
            for (int e = 0; e < EPV; ++e) {
                const int idx = vec * EPV + e;
                const float x = vec_elem<DT>(wv, e);
                s_ent[tid * 8 + e] = (vec >= 0 && idx < sp.Vs && !isnan(x)) ? cand_key(x, sp.v0 + idx) : 0ull;
            }
#pragma unroll
            for (int e = EPV; e < 8; ++e) s_ent[tid * 8 + e] = 0ull;
        }
        __syncthreads();
        if (warp == 0) {
            const int n = kc * 8;
            for (int round = 0; round < kc; ++round) {
                uint64_t mine = 0ull;
                int at = -1;
                for (int t = lane; t < n; t += 32)
                    if (s_ent[t] > mine) {
                        mine = s_ent[t];
                        at = t;
                    }
                const uint64_t best = warp_max_u64(mine);
                if (best != 0ull && mine == best) s_ent[at] = 0ull;   // unique keys: one lane takes it
                if (lane == 0) s_top[round] = best;
                __syncwarp();
            }
        }
    }
    __syncthreads();   // (every warp's state in s_st; the selection done)

    if (tid == 0) {
        SoftState a = s_st[0];
#pragma unroll
        for (int q = 1; q < NW; ++q) a = soft_merge(a, s_st[q]);
        sdd_shard_partial rec;
        rec.m = a.m;
        rec.r = a.r;
        rec.t2 = a.t2;
        rec.sh = a.sh;
        rec.sl = a.sl;
        rec.amax = (a.amax == INT32_MAX) ? INT32_MAX : sp.v0 + a.amax;
        rec.g = qnan();
        if (in_slice) {
            const int li = tok - sp.v0;
            float x;
            if (DT == SDD_BF16) {
                const uint16_t h = __ldg(reinterpret_cast<const unsigned short *>(row) + li);
                x = __uint_as_float(static_cast<uint32_t>(h) << 16);
            } else {
                x = __ldg(reinterpret_cast<const float *>(row) + li);
            }
            rec.g = fmax_nan(x, clamp_floor());
        }
        int nc = 0;
#pragma unroll
        for (int k = 0; k < SDD_SHARD_KMAX; ++k) {
            const uint64_t key = (k < kc) ? s_top[k] : 0ull;
            rec.cz[k] = (key != 0ull) ? cand_value(key) : -INFINITY;
            rec.cv[k] = (key != 0ull) ? cand_index(key) : INT32_MAX;
            nc += (key != 0ull) ? 1 : 0;
        }
        rec.info = (in_slice ? 1 : 0) | (tok_out ? 2 : 0) | (nc << 8);
        sp.out[r] = rec;
    }
}

}  // namespace

cudaError_t launch_shard_partials(const ShardParams &sp, cudaStream_t stream) {
    const int64_t rows = static_cast<int64_t>(sp.B) * (2 * sp.gamma + 1);
    if (rows == 0) return cudaSuccess;
    const bool bf = sp.dtype == SDD_BF16, cand = sp.kcap > 0;
    void (*const k)(ShardParams) = bf ? (cand ? shard_partials_kernel<SDD_BF16, true> : shard_partials_kernel<SDD_BF16, false>)
                                      : (cand ? shard_partials_kernel<SDD_F32, true> : shard_partials_kernel<SDD_F32, false>);
    k<<<static_cast<unsigned>(rows), kShardThreads, 0, stream>>>(sp);
    return cudaGetLastError();
}

}  // namespace sdd
