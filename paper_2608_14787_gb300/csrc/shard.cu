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
    float mr = clamp_floor();   // running maximum (first index in amax)
    bool nan = false;
    float s_hi = 0.f, s_lo = 0.f;
    uint64_t ck[SDD_SHARD_KMAX];
#pragma unroll
    for (int k = 0; k < SDD_SHARD_KMAX; ++k) ck[k] = 0ull;

    for (int v0 = tid; v0 < sp.RVs; v0 += kShardThreads * kShardU) {
        uint4 w[kShardU];
#pragma unroll
        for (int u = 0; u < kShardU; ++u) {
            const int vec = v0 + u * kShardThreads;
            w[u] = (vec < sp.RVs) ? __ldcs(reinterpret_cast<const uint4 *>(row) + vec) : make_uint4(0, 0, 0, 0);
        }
        // the chunk's entries (floored; NaN kept), its maximum and first index
        float z[kShardU * EPV];
        bool ok[kShardU * EPV];
        float cm = clamp_floor();
#pragma unroll
        for (int u = 0; u < kShardU; ++u) {
            const int vec = v0 + u * kShardThreads;
            const uint32_t *q = reinterpret_cast<const uint32_t *>(&w[u]);
#pragma unroll
            for (int e = 0; e < EPV; ++e) {
                const int i = u * EPV + e;
                const int idx = vec * EPV + e;
                ok[i] = vec < sp.RVs && idx < sp.Vs;
                float x = (DT == SDD_BF16) ? ((e & 1) ? bf16_hi(q[e >> 1]) : bf16_lo(q[e >> 1])) : __uint_as_float(q[e]);
                x = fmax_nan(x, clamp_floor());
                z[i] = x;
                if (ok[i]) {
                    nan |= isnan(x);
                    cm = fmax_nan(cm, x);
                    if (x > mr) {
                        mr = x;
                        st.amax = idx;
                    }
                    if (cand && !isnan(x)) {
                        uint64_t key = cand_key(x, sp.v0 + idx);
                        if (key > ck[SDD_SHARD_KMAX - 1]) {
#pragma unroll
                            for (int k = 0; k < SDD_SHARD_KMAX; ++k) {
                                const uint64_t a = ck[k];
                                ck[k] = (key > a) ? key : a;
                                key = (key > a) ? a : key;
                            }
                        }
                    }
                }
            }
        }
        if (cm > st.m) {
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
        const float nr = -st.r;
        const float dm = fmaf(st.m, kLog2e, nr);
        float sa = 0.f, ca = 0.f, ta = 0.f;   // compensated (Kahan) exp-sum
#pragma unroll
        for (int i = 0; i < kShardU * EPV; ++i) {
            if (ok[i]) {
                const float y = fmaf(z[i], kLog2e, nr);
                const float e = ex2(y);
                const float yk = e - ca, t = sa + yk;
                ca = (t - sa) - yk;
                sa = t;
                if (drafter) ta = fmaf(e, y - dm, ta);
            }
        }
        float h, e1;
        two_sum(s_hi, sa, h, e1);
        s_hi = h;
        s_lo += e1 - ca;
        st.t2 += ta;
    }
    if (nan) st.m = qnan();
    st.sh = s_hi;
    st.sl = s_lo;
    st.rank = 0;

    // CTA merge of the threads' states, in thread order
    __shared__ SoftState s_st[NW];
    const SoftState wst = soft_warp_reduce(st);
    if (lane == 0) s_st[warp] = wst;

    // the slice's kcap largest entries: kcap rounds of a CTA-wide maximum of
    // the threads' list heads, the winner popping its head
    __shared__ uint64_t s_wmax[NW];
    __shared__ uint64_t s_top[SDD_SHARD_KMAX];
    const int kc = cand ? sp.kcap : 0;
    for (int round = 0; round < kc; ++round) {
        const uint64_t m = warp_max_u64(ck[0]);
        if (lane == 0) s_wmax[warp] = m;
        __syncthreads();
        uint64_t best = 0ull;
#pragma unroll
        for (int q = 0; q < NW; ++q) best = (s_wmax[q] > best) ? s_wmax[q] : best;
        if (tid == 0) s_top[round] = best;
        if (best != 0ull && ck[0] == best) {   // keys are unique: one thread pops
#pragma unroll
            for (int k = 0; k + 1 < SDD_SHARD_KMAX; ++k) ck[k] = ck[k + 1];
            ck[SDD_SHARD_KMAX - 1] = 0ull;
        }
        __syncthreads();
    }
    __syncthreads();

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
