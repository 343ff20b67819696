// shard.cu -- the per-slice half of the vocabulary-sharded round (a
// tensor-parallel LM head: each rank holds one contiguous vocabulary slice
// [v0, v1) of every drafter and target row).
//
//  * shard_partials_kernel -- one CTA per row of the slice.  Each thread
//    streams its 16-byte vectors (ascending), keeping the online-softmax state
//    of its entries relative to an integer reference in log2 units (a new
//    maximum rescales the sums by an exact power of two), the first index of
//    its maximum, the drafter entropy accumulator, and -- target rows of a
//    round with the top-k rule -- its SDD_SHARD_KMAX largest entries.  The CTA
//    merges the threads' states in thread order and selects the slice's kcap
//    largest entries (value descending, index ascending), then one thread
//    writes the row's record.  Logits are floored at -2^23 as in the
//    streaming kernel; entries past the slice width weigh nothing.
//
// The records of all slices are merged, and every rule of the round runs, in
// decide_kernel (rules.cuh: merge_row_shards); the draw that follows the
// exchange of the slices' draw-row masses is shard_draw_kernel (decide.cu).
#include "rules.cuh"

namespace sdd {

namespace {

constexpr int kShardThreads = 256;
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

struct CandList {
    int n;       // keys held (at most kl)
    float thr;   // value of the last key once the list is full, else -inf
};

// One key into a thread's candidate list (keys descending, kl long, entry k
// at ck[k * kShardThreads]), inserted from the tail.
__device__ __noinline__ CandList cand_insert_key(uint64_t *ck, uint64_t key, int kl, CandList c) {
    int k = min(c.n, kl - 1);   // the slot it takes, moved up past smaller keys
    while (k > 0 && ck[(k - 1) * kShardThreads] < key) {
        ck[k * kShardThreads] = ck[(k - 1) * kShardThreads];
        --k;
    }
    ck[k * kShardThreads] = key;
    c.n = min(c.n + 1, kl);
    if (c.n == kl) c.thr = cand_value(ck[(kl - 1) * kShardThreads]);
    return c;
}

template <int DT, bool CAND>
__global__ void __launch_bounds__(kShardThreads) shard_partials_kernel(const __grid_constant__ ShardParams sp) {
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

    SoftState st = soft_identity();
    bool nan = false;
    float s_hi = 0.f, s_lo = 0.f;
    // target rows: the thread's kcap highest-ranked vectors, ranked by their
    // maximum (larger first, then lower vector index), keys in descending order
    // in shared memory, inserted from the tail.  The kcap largest entries of
    // the slice lie in the slice's kcap highest-ranked vectors (an entry
    // outside them has kcap vectors ranked above its own, each holding an
    // entry that ranks before it), so the CTA selects those vectors at the end
    // and takes the kcap largest of their entries.
    __shared__ uint64_t s_ck[SDD_SHARD_KMAX][kShardThreads];
    uint64_t *ck = &s_ck[0][tid];   // entry k at ck[k * kShardThreads]
    const int kl = cand ? sp.kcap : 0;   // list length
    CandList cl{0, -INFINITY};
    constexpr int PAIRS = EPV / 2;
    const f2_t L2 = f2_pack(kLog2e, kLog2e);

    for (int v0 = tid; v0 < sp.RVs; v0 += kShardThreads * kShardU) {
        uint4 w[kShardU];
        float vm[kShardU];   // each vector's maximum (floored; NaN kept)
#pragma unroll
        for (int u = 0; u < kShardU; ++u) {
            const int vec = v0 + u * kShardThreads;
            if (vec < sp.RVs) {
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
            if (vec < sp.RVs && (vec + 1) * EPV > sp.Vs) mask_tail<DT>(w[u], sp.Vs - vec * EPV);
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
        nan |= isnan(cm);
        if (cm > st.m) {
            // a new maximum (rare): its first index, in the first vector that holds it
            int us = kShardU - 1;
#pragma unroll
            for (int u = kShardU - 2; u >= 0; --u) us = (vm[u] == cm) ? u : us;
            uint4 ws = w[kShardU - 1];
#pragma unroll
            for (int u = kShardU - 2; u >= 0; --u) ws = (u == us) ? w[u] : ws;
            st.amax = vector_first_index<DT>(ws, (v0 + us * kShardThreads) * EPV, cm);
            // t2 against the maximum (as in the streaming kernel)
            if (drafter) st.t2 = fmaf((st.m - cm) * kLog2e, s_hi + s_lo, st.t2);
            st.m = cm;
            const float rn = ceilf(cm * kLog2e);
            if (rn > st.r) {
                const float k = st.r - rn;
                const float sc = pow2f_int(k);   // exact power of two (0 below the normal range)
                if (drafter) st.t2 *= sc;
                s_hi *= sc;
                s_lo *= sc;
                st.r = rn;
            }
        }
        if (cand) {
#pragma unroll
            for (int u = 0; u < kShardU; ++u) {
                const int vec = v0 + u * kShardThreads;
                // (a vector tying the last key comes later: it ranks after it)
                if (vm[u] > cl.thr && vec < sp.RVs) cl = cand_insert_key(ck, cand_key(vm[u], vec), kl, cl);
            }
        }
        // the exp-sums, two entries at a time (drafter rows: compensated, so
        // that the small terms of a peaked row survive next to its peak)
        const float nr = -st.r;
        const f2_t NR = f2_pack(nr, nr);
        const float dm = fmaf(st.m, kLog2e, nr);
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
                if (drafter) {
                    const f2_t yk = f2_sub(e, ca), t = f2_add(sa, yk);
                    ca = f2_sub(f2_sub(t, sa), yk);
                    sa = t;
                    ta = f2_fma(e, f2_sub(y, DM), ta);
                } else {
                    sa = f2_add(sa, e);
                }
            }
        }
        float a0, a1, c0, c1, t0, t1, h, e1, e2;
        f2_unpack(sa, a0, a1);
        f2_unpack(ca, c0, c1);
        f2_unpack(ta, t0, t1);
        two_sum(s_hi, a0, h, e1);
        two_sum(h, a1, s_hi, e2);
        s_lo += (e1 + e2) - (c0 + c1);
        st.t2 += t0 + t1;
    }
    if (nan) st.m = qnan();
    st.sh = s_hi;
    st.sl = s_lo;
    st.rank = 0;

    // CTA merge of the threads' states, in thread order
    __shared__ SoftState s_st[NW];
    const SoftState wst = soft_warp_reduce(st);
    if (lane == 0) s_st[warp] = wst;

    // the slice's kcap highest-ranked vectors: kcap rounds of a CTA-wide
    // maximum of the threads' list heads, the winner popping its head; then
    // the kcap largest entries of those vectors (one warp, kcap rounds)
    __shared__ uint64_t s_wmax[NW];
    __shared__ uint64_t s_top[SDD_SHARD_KMAX];
    __shared__ uint64_t s_ent[SDD_SHARD_KMAX * 8];
    const int kc = cand ? sp.kcap : 0;
    int head = 0;   // the thread's next unselected key
    for (int round = 0; round < kc; ++round) {
        const uint64_t mine = (head < cl.n) ? ck[head * kShardThreads] : 0ull;
        const uint64_t m = warp_max_u64(mine);
        if (lane == 0) s_wmax[warp] = m;
        __syncthreads();
        uint64_t best = 0ull;
#pragma unroll
        for (int q = 0; q < NW; ++q) best = (s_wmax[q] > best) ? s_wmax[q] : best;
        if (tid == 0) s_top[round] = best;
        if (best != 0ull && mine == best) ++head;   // keys are unique: one thread pops
        __syncthreads();
    }
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
