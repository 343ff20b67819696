// diag.cu -- offline diagnostics over logged blocks (scores q [B, gamma] and
// strict accepted lengths L [B] of Strict SDD / shadow-verified rounds):
//
//  * the permutation diagnostic behind Table 1 (Sec. 5, H1 mechanism): at every
//    position j the (score, label) pairs are permuted across the blocks valid
//    there (all blocks; for the conditional signal those with L >= j - 1, j
//    1-based), which keeps every positionwise distribution and breaks the
//    association of positions within a block; the feasible prefix length
//    (Eq. 3's gates, before K_min or staleness) is recomputed per block;
//  * positionwise offline metrics (App. offline metrics): BCE of the scores
//    against the labels 1{L >= j}, the position-only baseline (the positive
//    rate at j), and AUROC (Mann-Whitney, ties count one half).
//
// perm_build_kernel  -- one CTA per (repetition, position): Fisher-Yates over
//                       the valid blocks in shared memory (order-preserving
//                       compaction by ballots; Philox partners drawn in
//                       parallel, the swaps in order by one thread; 64
//                       threads, so that 32 CTAs interleave on an SM); it
//                       writes the permuted scores of its position.
// perm_prefix_kernel -- one warp per (repetition, block): the gates of Eq. 3 on
//                       the permuted scores (the schedule's own arithmetic),
//                       integer sums per repetition (exact, order-free).
// metrics_kernel     -- one CTA per position: fp64 BCE sums, integer pair counts.
#include "rules.cuh"

namespace sdd {
namespace {

constexpr uint32_t kPurposePerm = 3;
constexpr int kDiagThreads = 256;
// The permutation builder's CTAs are small so that 32 of them share an SM:
// each spends most of its time in one thread's serial swap loop, and the SM
// interleaves those loops.
constexpr int kPermThreads = 64;

// Logs of at most this many blocks are shuffled by the parallel construction
// below; longer ones by the serial swap loop.
constexpr int kPermPar = 4096;

// Shared memory of the permutation builder for B logged blocks: the block
// list [B], the validity bits of position j [ceil(B/32) words] and their
// exclusive prefix popcounts [ceil(B/32)]; for B <= kPermPar the parallel
// construction's arrays: one [B] of 32-bit bucket bounds and four [B] of
// 16-bit indices (small, so that ~23 CTAs share an SM).
__host__ __device__ inline size_t perm_smem_bytes(int B) {
    const size_t words = (static_cast<size_t>(B) + 31) / 32;
    const size_t par = (B <= kPermPar) ? static_cast<size_t>(B) * (sizeof(int32_t) + 4 * sizeof(int16_t)) : 0;
    return (static_cast<size_t>(B) + 2 * words) * sizeof(int32_t) + par;
}

__global__ void __launch_bounds__(kPermThreads) perm_build_kernel(const float *q, const int32_t *L, int B, int gamma,
                                                                  int n_rep, int conditional, uint64_t seed,
                                                                  float *pq) {
    extern __shared__ int32_t s_dyn[];
    int32_t *s_list = s_dyn;                                               // the valid blocks, then their shuffle
    uint32_t *s_mask = reinterpret_cast<uint32_t *>(s_dyn + B);            // validity bits
    int32_t *s_wpre = s_dyn + B + (B + 31) / 32;                           // valid blocks before each word
    __shared__ __align__(16) int32_t s_k[kPermThreads];   // swap partners of the current batch of slots
    __shared__ int s_n;
    const int r = blockIdx.x / gamma, j = blockIdx.x % gamma;
    const int tid = threadIdx.x, lane = tid & 31;
    const int words = (B + 31) / 32;
    float *row = pq + (static_cast<int64_t>(r) * gamma + j) * B;
    // validity bits (the loads of several chunks in flight together)
#pragma unroll 4
    for (int c = 0; c < B; c += kPermThreads) {
        const int b = c + tid;
        const bool v = b < B && (!conditional || __ldg(L + b) >= j);
        const unsigned m = __ballot_sync(0xFFFFFFFFu, v);
        if (lane == 0 && b < B) s_mask[b >> 5] = m;   // (b: the warp's first block, a multiple of 32)
    }
    __syncthreads();
    // exclusive prefix popcounts of the words (one warp)
    if (tid < 32) {
        int carry = 0;
        for (int w0 = 0; w0 < words; w0 += 32) {
            const int w = w0 + lane;
            const int c = (w < words) ? __popc(s_mask[w]) : 0;
            int incl = c;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int t = __shfl_up_sync(0xFFFFFFFFu, incl, off);
                if (lane >= off) incl += t;
            }
            if (w < words) s_wpre[w] = carry + incl - c;
            carry += __shfl_sync(0xFFFFFFFFu, incl, 31);
        }
        if (lane == 0) s_n = carry;
    }
    __syncthreads();
    const int n = s_n;
    // the valid blocks in index order (the order defines the draw)
    for (int b = tid; b < B; b += kPermThreads) {
        const uint32_t m = s_mask[b >> 5], bit = 1u << (b & 31);
        if (m & bit) s_list[s_wpre[b >> 5] + __popc(m & (bit - 1u))] = b;
    }
    __syncthreads();
    // Fisher-Yates from the top: slot i swaps with k_i = floor(w (i + 1) / 2^32),
    // w the first Philox word of counter (i, j, r, purpose), for i = n-1 .. 1.
    const uint2 key = make_uint2(static_cast<uint32_t>(seed), static_cast<uint32_t>(seed >> 32));
    if (n > 1 && B <= kPermPar) {   // (the shared-memory layout follows B, not n)
        // The same permutation without the serial loop.  Step a moves the
        // value then at slot a to slot k_a and fixes slot a.  Let P(s) be the
        // value at slot s just before step s (slot 0: at the end); the last
        // step before a that wrote slot s is the smallest a' > a with
        // k_a' = s, and it wrote P(a').  So, with bucket(s) = {a : k_a = s}:
        //   P(s) = P(min{a' in bucket(s), a' > s}), or the original s_list[s];
        //   final[a] = P(min{a' in bucket(k_a), a' > a}), or s_list[k_a];
        //   final[0] = P(0).
        // P follows the "first step above" chains to their ends (pointer
        // jumping); buckets come from a counting sort, each sorted by index.
        int32_t *s_cnt = s_wpre + words;                          // bucket sizes, starts, then ends
        int16_t *s_kk = reinterpret_cast<int16_t *>(s_cnt + B);   // k_a
        int16_t *s_bkt = s_kk + B;                                // steps by bucket; later the final list
        int16_t *s_nxt = s_bkt + B;                               // next step of the bucket above a (-1: none)
        int16_t *s_ptr = s_nxt + B;                               // chain links, then chain ends
        __shared__ int32_t s_part[kPermThreads];
        for (int t = tid; t < n; t += kPermThreads) s_cnt[t] = 0;
        __syncthreads();
        for (int a = 1 + tid; a < n; a += kPermThreads) {
            const uint4 o = philox4x32_10(make_uint4(static_cast<uint32_t>(a), static_cast<uint32_t>(j),
                                                     static_cast<uint32_t>(r), kPurposePerm),
                                          key);
            const int k = static_cast<int>((static_cast<uint64_t>(o.x) * static_cast<uint64_t>(a + 1)) >> 32);
            s_kk[a] = static_cast<int16_t>(k);
            atomicAdd(&s_cnt[k], 1);
        }
        __syncthreads();
        // bucket starts: exclusive prefix of the sizes (chunks per thread)
        const int chunk = (n + kPermThreads - 1) / kPermThreads;
        const int c0 = min(n, tid * chunk), c1 = min(n, c0 + chunk);
        int sum = 0;
        for (int t = c0; t < c1; ++t) sum += s_cnt[t];
        s_part[tid] = sum;
        __syncthreads();
        if (tid == 0) {
            int run = 0;
            for (int t = 0; t < kPermThreads; ++t) {
                const int v = s_part[t];
                s_part[t] = run;
                run += v;
            }
        }
        __syncthreads();
        int run = s_part[tid];
        for (int t = c0; t < c1; ++t) {
            const int v = s_cnt[t];
            s_cnt[t] = run;
            run += v;
        }
        __syncthreads();
        // scatter (the starts advance to the ends: bucket t is [end(t-1), end(t)))
        for (int a = 1 + tid; a < n; a += kPermThreads)
            s_bkt[atomicAdd(&s_cnt[s_kk[a]], 1)] = static_cast<int16_t>(a);
        __syncthreads();
        // per slot: its bucket sorted, successors, the first step above the slot
        for (int t = tid; t < n; t += kPermThreads) {
            const int b0 = (t > 0) ? s_cnt[t - 1] : 0, b1 = s_cnt[t];
            for (int u = b0 + 1; u < b1; ++u) {   // insertion sort (buckets hold ~1 step)
                const int v = s_bkt[u];
                int w = u - 1;
                while (w >= b0 && s_bkt[w] > v) {
                    s_bkt[w + 1] = s_bkt[w];
                    --w;
                }
                s_bkt[w + 1] = static_cast<int16_t>(v);
            }
            int above = t;   // the chain ends here when no step above t targets t
            for (int u = b0; u < b1; ++u) {
                const int v = s_bkt[u];
                s_nxt[v] = (u + 1 < b1) ? s_bkt[u + 1] : static_cast<int16_t>(-1);
                if (above == t && v > t) above = v;
            }
            s_ptr[t] = static_cast<int16_t>(above);
        }
        __syncthreads();
        for (int span = 1; span < n; span <<= 1) {   // pointer jumping to the chain ends
            for (int t = tid; t < n; t += kPermThreads) s_ptr[t] = s_ptr[s_ptr[t]];
            __syncthreads();
        }
        for (int a = tid; a < n; a += kPermThreads) {
            int v;
            if (a == 0) {
                v = s_list[s_ptr[0]];
            } else {
                const int na = s_nxt[a];
                v = (na >= 0) ? s_list[s_ptr[na]] : s_list[s_kk[a]];
            }
            s_bkt[a] = static_cast<int16_t>(v);
        }
        __syncthreads();
        for (int a = tid; a < n; a += kPermThreads) s_list[a] = s_bkt[a];
        __syncthreads();
    } else {
        // serial: the partners of kPermThreads slots drawn in parallel, the swaps
        // then in order
        for (int top = n - 1; top > 0; top -= kPermThreads) {
            const int i = top - tid;
            if (i > 0) {
                const uint4 o = philox4x32_10(make_uint4(static_cast<uint32_t>(i), static_cast<uint32_t>(j),
                                                         static_cast<uint32_t>(r), kPurposePerm),
                                              key);
                s_k[tid] = static_cast<int32_t>((static_cast<uint64_t>(o.x) * static_cast<uint64_t>(i + 1)) >> 32);
            }
            __syncthreads();
            if (tid == 0) {
                // slots top, top - 1, ..., top - cnt + 1 (all > 0); x carries the
                // value at slot a, re-read after each swap (which may have written
                // slot a - 1), so one shared-memory round trip bounds an iteration;
                // the partners come four at a time
                const int cnt = min(kPermThreads, top);
                int32_t x = s_list[top];
                for (int u = 0; u < cnt; u += 4) {
                    const int4 kk = *reinterpret_cast<const int4 *>(s_k + u);
                    const int ks[4] = {kk.x, kk.y, kk.z, kk.w};
#pragma unroll
                    for (int h = 0; h < 4; ++h) {
                        if (u + h >= cnt) break;
                        const int a = top - u - h, k = ks[h];
                        const int32_t y = (k == a) ? x : s_list[k];
                        s_list[k] = x;
                        s_list[a] = y;
                        x = s_list[a - 1];
                    }
                }
            }
            __syncthreads();
        }
    }
    // block b (the t-th valid block) takes the score of block s_list[t]; others
    // keep theirs: the permuted scores of position j, gathered here so that the
    // prefix kernel reads each with one load
    for (int b = tid; b < B; b += kPermThreads) {
        const uint32_t m = s_mask[b >> 5], bit = 1u << (b & 31);
        const int src = (m & bit) ? s_list[s_wpre[b >> 5] + __popc(m & (bit - 1u))] : b;
        row[b] = __ldg(q + static_cast<int64_t>(src) * gamma + j);
    }
}

__global__ void perm_prefix_kernel(const float *q, const float *pq, int B, int gamma, int n_rep, int signal,
                                   df eta_loc, df log_eta_c, unsigned long long *sums) {
    const int lane = threadIdx.x & 31;
    const int64_t w = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    if (w >= static_cast<int64_t>(n_rep + 1) * B) return;
    const int r = static_cast<int>(w / B), b = static_cast<int>(w % B);   // r == n_rep: the logged order
    int kb = gamma, best = 0;
    df carry = df{0.f, 0.f};
    for (int c = 0; c < gamma && kb >= c; c += 32) {
        const int j = c + lane;
        const bool in = j < gamma;
        const float qj = !in ? 0.f
                         : (r < n_rep) ? __ldg(pq + (static_cast<int64_t>(r) * gamma + j) * B + b)
                                       : __ldg(q + static_cast<int64_t>(b) * gamma + j);
        const float lq = in ? logf(qj) : 0.f;
        const df S = df_add(carry, warp_prefix_df(df{lq, 0.f}, lane));
        carry.hi = __shfl_sync(0xFFFFFFFFu, S.hi, 31);
        carry.lo = __shfl_sync(0xFFFFFFFFu, S.lo, 31);
        sched_step(c, lane, gamma, in, qj, false, S, eta_loc, log_eta_c, signal, kb, best);
    }
    const int Kh = (signal == SDD_SIG_MARGINAL) ? kb : best;
    if (lane == 0) atomicAdd(sums + r, static_cast<unsigned long long>(Kh));
}

__global__ void __launch_bounds__(kDiagThreads) metrics_kernel(const float *q, const int32_t *L, int B, int gamma,
                                                               int conditional, double *bce, double *bce_base,
                                                               double *auroc, int32_t *n_pos, int32_t *n_neg) {
    const int j = blockIdx.x;
    __shared__ double s_bce[kDiagThreads];
    __shared__ unsigned long long s_np[kDiagThreads], s_nn[kDiagThreads], s_gt[kDiagThreads], s_eq[kDiagThreads];
    double sb = 0.0;
    unsigned long long np = 0, nn = 0, gt = 0, eq = 0;
    for (int b = threadIdx.x; b < B; b += kDiagThreads) {
        const int l = __ldg(L + b);
        if (conditional && l < j) continue;
        const bool y = l >= j + 1;
        const double qc = fmin(fmax(static_cast<double>(__ldg(q + static_cast<int64_t>(b) * gamma + j)), 1e-7),
                               1.0 - 1e-7);
        sb -= y ? log(qc) : log1p(-qc);
        if (y) {
            ++np;
            const float qi = __ldg(q + static_cast<int64_t>(b) * gamma + j);
            for (int k = 0; k < B; ++k) {   // every valid negative
                const int lk = __ldg(L + k);
                if ((conditional && lk < j) || lk >= j + 1) continue;
                const float qk = __ldg(q + static_cast<int64_t>(k) * gamma + j);
                gt += qi > qk;
                eq += qi == qk;
            }
        } else {
            ++nn;
        }
    }
    s_bce[threadIdx.x] = sb;
    s_np[threadIdx.x] = np;
    s_nn[threadIdx.x] = nn;
    s_gt[threadIdx.x] = gt;
    s_eq[threadIdx.x] = eq;
    __syncthreads();
    for (int h = kDiagThreads / 2; h > 0; h >>= 1) {   // fixed-order tree: deterministic sums
        if (threadIdx.x < h) {
            s_bce[threadIdx.x] += s_bce[threadIdx.x + h];
            s_np[threadIdx.x] += s_np[threadIdx.x + h];
            s_nn[threadIdx.x] += s_nn[threadIdx.x + h];
            s_gt[threadIdx.x] += s_gt[threadIdx.x + h];
            s_eq[threadIdx.x] += s_eq[threadIdx.x + h];
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        const double P = static_cast<double>(s_np[0]), N = static_cast<double>(s_nn[0]), n = P + N;
        const double nan = __longlong_as_double(0x7FF8000000000000ll);
        bce[j] = (n > 0) ? s_bce[0] / n : nan;
        const double pr = (n > 0) ? P / n : nan;
        bce_base[j] = (n > 0) ? ((pr > 0.0 && pr < 1.0) ? -(pr * log(pr) + (1.0 - pr) * log1p(-pr)) : 0.0) : nan;
        auroc[j] = (P > 0 && N > 0) ? (static_cast<double>(s_gt[0]) + 0.5 * static_cast<double>(s_eq[0])) / (P * N)
                                    : nan;
        if (n_pos) n_pos[j] = static_cast<int32_t>(s_np[0]);
        if (n_neg) n_neg[j] = static_cast<int32_t>(s_nn[0]);
    }
}

}  // namespace

cudaError_t launch_perm_diag(const float *q, const int32_t *L, int B, int gamma, int signal, df eta_loc,
                             df log_eta_c, int n_rep, uint64_t seed, float *pq, unsigned long long *sums,
                             cudaStream_t stream) {
    cudaError_t e = cudaMemsetAsync(sums, 0, sizeof(unsigned long long) * (n_rep + 1), stream);
    if (e != cudaSuccess) return e;
    const size_t smem = perm_smem_bytes(B);
    if (smem > 48 * 1024) {
        e = cudaFuncSetAttribute(perm_build_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(smem));
        if (e != cudaSuccess) return e;
    }
    if (n_rep > 0) {
        perm_build_kernel<<<n_rep * gamma, kPermThreads, smem, stream>>>(q, L, B, gamma, n_rep,
                                                                        signal == SDD_SIG_CONDITIONAL, seed, pq);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    const int64_t warps = static_cast<int64_t>(n_rep + 1) * B;
    perm_prefix_kernel<<<static_cast<unsigned>((warps * 32 + 255) / 256), 256, 0, stream>>>(
        q, pq, B, gamma, n_rep, signal, eta_loc, log_eta_c, sums);
    return cudaGetLastError();
}

cudaError_t launch_position_metrics(const float *q, const int32_t *L, int B, int gamma, int conditional, double *bce,
                                    double *bce_base, double *auroc, int32_t *n_pos, int32_t *n_neg,
                                    cudaStream_t stream) {
    metrics_kernel<<<gamma, kDiagThreads, 0, stream>>>(q, L, B, gamma, conditional, bce, bce_base, auroc, n_pos,
                                                       n_neg);
    return cudaGetLastError();
}

}  // namespace sdd
