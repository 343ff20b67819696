// mlp.cu -- the learned-scorer stand-ins of the decode-loop workload on the
// 5th-generation tensor cores (App. A.7's form, random weights):
//
//   one layer:  s[m] = sigmoid(w2 . GELU(W1 h[m] + b1) + b2),
//   deep:       a1 = bf16(GELU(W1 [h ; f] + b1)), a2 = bf16(GELU(W2 a1 + b2)),
//               s[m] = sigmoid(w4 . GELU(W3 a2 + b3) + b4),
//   GELU(z) = z Phi(z) (erf form), fp32 accumulation throughout,
//
// and the scalar-feature block f of the deep scorer's input.
//
// First layer (mlp_kernel): a cluster of S = 4 CTAs per 128-row tile splits K;
// each CTA streams its K quarter through a four-stage ring of 48 KiB (A tile
// 128 x 64, B tile 256 x 64, K-major, 128-byte swizzle) filled by 2D TMA, one
// thread issues tcgen05.mma.kind::f16 (M = 128, N = 256, K = 16) into a
// 256-column TMEM accumulator; the partial accumulators meet through an L2
// workspace (stores, one cluster barrier, bulk copies) and CTA q finishes
// output columns [64 q, 64 q + 64) with the fused epilogue.
// Layers 2-3 of the deep scorer (mlp_tail_kernel): a cluster of four CTAs per
// tile, each computing 64 output columns of both layers, a2 through the
// workspace and back by TMA.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <mutex>

#include "internal.h"

namespace sdd {
namespace {

constexpr int kMlpN = 256;           // hidden units = UMMA N
constexpr int kMlpBM = 128;          // rows per CTA = UMMA M
constexpr int kMlpBK = 64;           // K per stage: 64 bf16 = one 128-byte swizzle row
constexpr int kMlpStages = 4;
constexpr int kMlpThreads = 512;     // warp 0 lane 0: TMA producer; warp 1 lane 0: MMA issuer; all: epilogue
constexpr uint32_t kATileBytes = kMlpBM * kMlpBK * 2;   // 16 KiB
constexpr uint32_t kBTileBytes = kMlpN * kMlpBK * 2;    // 32 KiB
constexpr uint32_t kStageBytes = kATileBytes + kBTileBytes;
constexpr int kMlpSmem = kMlpStages * kStageBytes + 1024 + 256;   // + alignment slack + barriers
constexpr uint32_t kTmemCols = 256;

struct MlpParams {
    int32_t M, K;
    int32_t Ka;             // K columns of the first A operand (the rest come from the second)
    const float *b1;        // [256]
    const uint16_t *w2;     // [256] bf16 bits (head mode)
    float b2;
    float *out;             // [M] (head mode)
    uint16_t *act;          // [M, 256] bf16 bits: GELU(W1 x + b1) (activation mode)
    float *ws;              // [tiles][S][256][128] fp32: partial accumulators (column-major per source CTA)
    int32_t *status;
};

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int c0, int c1, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
        : "memory");
}

// Shared-memory matrix descriptor of a K-major operand tile with the 128-byte
// swizzle: rows of 128 bytes, 8-row core groups 1024 bytes apart (SBO); the
// leading-dimension offset is unused for this layout; descriptor version 1.
__device__ __forceinline__ uint64_t umma_desc_sw128(uint32_t addr) {
    uint64_t d = static_cast<uint64_t>((addr >> 4) & 0x3FFFu);
    d |= static_cast<uint64_t>(1) << 16;                // LBO (unused): 16 bytes
    d |= static_cast<uint64_t>(1024 >> 4) << 32;        // SBO: 1024 bytes
    d |= static_cast<uint64_t>(1) << 46;                // version
    d |= static_cast<uint64_t>(2) << 61;                // 128-byte swizzle
    return d;
}

// Instruction descriptor of kind::f16: fp32 D, bf16 A and B, both K-major, N, M = 128.
__host__ __device__ constexpr uint32_t idesc_f16(int n) {
    return (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(n >> 3) << 17) |
           (static_cast<uint32_t>(kMlpBM >> 4) << 24);
}

template <int N = kMlpN>
__device__ __forceinline__ void umma_f16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc_f16(N)), "r"(accumulate)
        : "memory");
}

// Arrive on `bar` once every tcgen05 operation this thread issued so far completes.
__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 16 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
// 16 columns of this thread's TMEM lane, or zeros when the accumulator is not valid.
__device__ __forceinline__ void tmem_ld16_or0(bool ok, uint32_t taddr, uint32_t (&v)[16]) {
    if (ok) {
        tmem_ld16(taddr, v);
    } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) v[j] = 0u;
    }
}

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Address of the same shared-memory location in cluster CTA `rank`.
__device__ __forceinline__ uint32_t map_rank(uint32_t addr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}
// Orders this thread's generic-proxy global stores before later async-proxy
// (TMA) reads of them, by any thread that synchronises with this one.
__device__ __forceinline__ void fence_proxy_async_global() {
    asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Untiled global -> shared bulk copy (16-byte aligned, size a multiple of 16).
__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

__device__ __forceinline__ void st_cluster_f32(uint32_t addr, float a) {
    asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(addr), "f"(a) : "memory");
}

// Two fp32 values rounded to bf16 (round to nearest even), packed (a low).
__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
    uint32_t d;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(b), "f"(a));
    return d;
}

__device__ __forceinline__ float gelu_erf(float z) { return 0.5f * z * (1.f + erff(z * 0.70710678118654752f)); }

// Grid: (M tiles x S) CTAs in clusters of S along x (S = 1, 2 or 4 splits of
// K).  CTA rank r of a cluster multiplies K slices [r nk/S, (r+1) nk/S) of its
// 128-row tile into its own TMEM.  Columns [q W, (q+1) W) of the tile (W =
// 256/S) are finished by CTA q: every CTA stores the other columns of its
// partial to the workspace (L2; distributed shared memory moves these 96 KiB
// per CTA several times slower), a cluster barrier orders the stores before
// the loads, and each CTA sums the S partials of its columns in rank order
// (its own from TMEM) and runs the epilogue.
//
// The A operand is the concatenation [A1 | A2] along K: slices below p.Ka come
// from tmA, the rest from tmA2 (the scalar features of the deep scorer).
// HEAD: the epilogue fuses GELU, the w2 dot product and the sigmoid (one
// float per row); otherwise it writes the layer's activations GELU(z + b1)
// as bf16 rows of p.act for the next layer.
template <int S, bool HEAD>
__global__ void __launch_bounds__(kMlpThreads, 1) mlp_kernel(const __grid_constant__ CUtensorMap tmA,
                                                            const __grid_constant__ CUtensorMap tmA2,
                                                            const __grid_constant__ CUtensorMap tmB,
                                                            const __grid_constant__ MlpParams p) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                            ~static_cast<uintptr_t>(1023));
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + kMlpStages * kStageBytes);
    uint64_t *empty = full + kMlpStages;
    uint64_t *done = empty + kMlpStages;
    uint64_t *xfer = done + 1;   // the other CTAs' partials of this CTA's columns have landed
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(done + 2);
    __shared__ int s_abort;
    __shared__ float s_b1[kMlpN], s_w2[kMlpN];   // epilogue constants, widened once per CTA
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t rank = (S > 1) ? cluster_rank() : 0u;
    const int m0 = (blockIdx.x / S) * kMlpBM;
    const int nk = p.K / kMlpBK / S;           // K slices of this CTA
    const int kt0 = static_cast<int>(rank) * nk;

    if (tid == 0) {
        for (int s = 0; s < kMlpStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        mbar_init(done, 1);
        mbar_init(xfer, 1);
        fence_mbar_init();
        s_abort = 0;
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(tmem_slot)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    // launched as a programmatic dependent: the setup above overlaps the end
    // of the work ahead in the stream; nothing is read before that completes
    griddep_wait();
    for (int n = tid; n < kMlpN; n += kMlpThreads) {
        s_b1[n] = __ldg(p.b1 + n);
        s_w2[n] = HEAD ? __uint_as_float(static_cast<uint32_t>(__ldg(p.w2 + n)) << 16) : 0.f;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // TMA producer: stage s holds K slice kt0 + t of the A tile (rows
        // m0..m0+127) and of the B tile (all 256 hidden units)
        int t = 0;
        for (; t < nk; ++t) {
            const int s = t % kMlpStages;
            const uint32_t ph = static_cast<uint32_t>(t / kMlpStages) & 1u;
            if (t >= kMlpStages && !mbar_wait_bounded(&empty[s], ph ^ 1u, kWaitPolls)) {
                s_abort = 1;
                break;
            }
            mbar_arrive_expect_tx(&full[s], kStageBytes);
            const uint32_t a = smem_addr(smem + s * kStageBytes);
            const int k = (kt0 + t) * kMlpBK;
            if (k < p.Ka)
                tma_load_2d(a, &tmA, k, m0, smem_addr(&full[s]));
            else
                tma_load_2d(a, &tmA2, k - p.Ka, m0, smem_addr(&full[s]));
            tma_load_2d(a + kATileBytes, &tmB, k, 0, smem_addr(&full[s]));
        }
        // let every issued load land before the ring is reused or the CTA
        // leaves (already true unless a wait gave up): the last load per stage
        for (int s = 0; s < kMlpStages && s < t; ++s) {
            const int last = ((t - 1 - s) / kMlpStages) * kMlpStages + s;
            (void)mbar_wait_bounded(&full[s], static_cast<uint32_t>(last / kMlpStages) & 1u, kWaitPolls);
        }
    } else if (warp == 1 && lane == 0) {
        // MMA issuer: four K = 16 steps per stage, the 128-byte rows advanced
        // by 32 bytes per step
        for (int t = 0; t < nk; ++t) {
            const int s = t % kMlpStages;
            const uint32_t ph = static_cast<uint32_t>(t / kMlpStages) & 1u;
            if (!mbar_wait_bounded(&full[s], ph, kWaitPolls)) {
                s_abort = 1;
                break;
            }
            tc_fence_after();
            const uint32_t a = smem_addr(smem + s * kStageBytes), b = a + kATileBytes;
#pragma unroll
            for (int kk = 0; kk < kMlpBK / 16; ++kk)
                umma_f16(tmem, umma_desc_sw128(a + kk * 32), umma_desc_sw128(b + kk * 32), (t | kk) != 0 ? 1u : 0u);
            umma_commit(smem_addr(&empty[s]));   // the stage is free once these MMAs have read it
        }
        umma_commit(smem_addr(done));            // the accumulator is complete
    }
    __syncwarp();

    // Exchange through the workspace.  CTA q of the cluster finishes the
    // column block [q W, (q + 1) W) (W = 256 / S) of all 128 rows: its own
    // partial of the block stays in its TMEM, every other column of its
    // partial goes to ws[tile][q][column][row] (a warp's 32 rows of one column
    // are 128 contiguous bytes), from where the owner of the column copies it.
    // Warp w reads TMEM lanes 32 (w % 4) .. + 31 (tile rows); the four warps
    // of a lane quarter share the columns in 16-column chunks.
    constexpr int W = kMlpN / S;
    const bool ok = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(done, 0u, kWaitPolls));
    tc_fence_after();
    if (!ok) s_abort = 1;
    griddep_launch_dependents();   // the next layer's setup and weight loads may start
    const int quarter = warp & 3, part = warp >> 2;
    const int row = quarter * 32 + lane;
    const uint32_t tbase = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    float *ws_tile = p.ws + static_cast<int64_t>(blockIdx.x / S) * S * kMlpN * kMlpBM;
    if (S > 1) {
        float *mine = ws_tile + static_cast<int64_t>(rank) * kMlpN * kMlpBM;
        int idx = 0;   // remote chunks in column order, round robin over the quarter's four warps
#pragma unroll 1
        for (int c = 0; c < kMlpN; c += 16) {
            if (c / W == static_cast<int>(rank)) continue;
            if ((idx++ & 3) != part) continue;
            uint32_t v[16];
            tmem_ld16_or0(ok, tbase + c, v);
#pragma unroll
            for (int j = 0; j < 16; ++j) __stcg(mine + (c + j) * kMlpBM + row, __uint_as_float(v[j]));
        }
        fence_proxy_async_global();   // the stores, before the bulk copies of the other CTAs read them
        cluster_sync();               // every partial of the tile is in the workspace (release / acquire)
        if (tid == 0) {
            // the S - 1 other partials of this CTA's columns (W x 128 fp32, contiguous
            // in the column-major workspace) into slots of the idle stage ring
            constexpr uint32_t kBlock = W * kMlpBM * sizeof(float);
            mbar_arrive_expect_tx(xfer, (S - 1) * kBlock);
            for (int r = 0; r < S; ++r)
                if (r != static_cast<int>(rank))
                    bulk_load(smem_addr(smem + r * kBlock),
                              ws_tile + (static_cast<int64_t>(r) * kMlpN + static_cast<int>(rank) * W) * kMlpBM, kBlock,
                              smem_addr(xfer));
        }
    }
    const bool okx = (S == 1) || __all_sync(0xFFFFFFFFu, mbar_wait_bounded(xfer, 0u, kWaitPolls));
    if (!okx) s_abort = 1;
    const float *recv = reinterpret_cast<const float *>(smem);   // [S][W columns][128 rows]

    // epilogue: z = the partials summed in rank order, then bias and GELU;
    // this warp's columns [rank W + part W / 4, + W / 4) of its 32 rows
    const int grow = m0 + row;
    float t2 = 0.f;   // HEAD: this thread's part of the w2 dot product
#pragma unroll 1
    for (int c = static_cast<int>(rank) * W + part * (W / 4); c < static_cast<int>(rank) * W + (part + 1) * (W / 4);
         c += 16) {
        uint32_t own[16];
        tmem_ld16_or0(ok, tbase + c, own);
        float rem[S][16];
#pragma unroll
        for (int r = 0; r < S; ++r)
            if (r != static_cast<int>(rank)) {
                const float *src = recv + (r * W + c - static_cast<int>(rank) * W) * kMlpBM + row;
#pragma unroll
                for (int j = 0; j < 16; ++j) rem[r][j] = src[j * kMlpBM];
            }
        float g[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            float z = 0.f;
#pragma unroll
            for (int r = 0; r < S; ++r) {
                const float x = (r == static_cast<int>(rank)) ? __uint_as_float(own[j]) : rem[r][j];
                z = (r == 0) ? x : z + x;
            }
            const int n = c + j;
            g[j] = gelu_erf(z + s_b1[n]);
            if (HEAD) t2 = fmaf(s_w2[n], g[j], t2);
        }
        if (!HEAD && ok && grow < p.M) {
            // 16 bf16 activations (round to nearest even) in two 16-byte stores
            uint32_t w[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) w[q] = pack_bf16x2(g[2 * q], g[2 * q + 1]);
            uint4 *dst = reinterpret_cast<uint4 *>(p.act + static_cast<int64_t>(grow) * kMlpN + c);
            dst[0] = make_uint4(w[0], w[1], w[2], w[3]);
            dst[1] = make_uint4(w[4], w[5], w[6], w[7]);
        }
    }
    if (HEAD) {
        // the row's dot product: the four warps of the quarter in order, then
        // the S column blocks in rank order (CTA 0 of the cluster finishes)
        __shared__ float s_part[3][kMlpBM];
        __shared__ float s_head[S][kMlpBM];
        if (part > 0) s_part[part - 1][row] = t2;
        __syncthreads();
        if (part == 0) {
            const float t = ((t2 + s_part[0][row]) + s_part[1][row]) + s_part[2][row];
            if (S > 1)
                st_cluster_f32(map_rank(smem_addr(&s_head[rank][row]), 0u), t);
            else
                s_head[0][row] = t;
        }
        if (S > 1)
            cluster_sync();
        else
            __syncthreads();
        if (rank == 0 && part == 0 && ok && grow < p.M) {
            float t = s_head[0][row];
#pragma unroll
            for (int r = 1; r < S; ++r) t += s_head[r][row];
            p.out[grow] = 1.f / (1.f + expf(-(t + p.b2)));
        }
    }
    tc_fence_before();
    __syncthreads();
    if (tid == 0 && s_abort) status_or(p.status, SDD_DEV_TIMEOUT);
    if (S > 1 && tid == 0 && !okx) (void)mbar_wait_bounded(xfer, 0u, kWaitPolls);   // copies still in flight
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
}

// ---------------------------------------------------------------------------
// Layers 2 and 3 and the head of the deep scorer (K -> 256 -> 256 -> 256 -> 1):
// a cluster of four CTAs per 128-row tile, CTA q producing output columns
// [64 q, 64 q + 64) of both layers, so that the GELU epilogues (ALU-bound:
// 32 K activations per tile and layer) spread over four SMs.
//   1. TMA: the tile's first-layer activations a1 (128 x 256 bf16, four
//      64-column slices, 128-byte swizzle), rows [64 q, +64) of W2 and of W3.
//   2. z2 = W2_q a1 (M = 128, N = 64) into TMEM columns 0..63; the epilogue
//      writes a2 = bf16(GELU(z2 + b2)) for its 64 columns to the workspace.
//   3. Cluster barrier; every CTA loads the whole a2 tile back by TMA (L2)
//      into the swizzled K-major layout over a1.
//   4. z3 = W3_q a2 into TMEM columns 64..127; each row's dot product
//      w4 . GELU(z3 + b3) over the CTA's 64 columns goes to CTA 0, which adds
//      the four in rank order, adds b4 and applies the sigmoid.
// ---------------------------------------------------------------------------
constexpr int kTailCluster = 4;
constexpr int kTailN = kMlpN / kTailCluster;               // 64 output columns per CTA
constexpr uint32_t kTailASlice = kMlpBM * kMlpBK * 2;      // 16 KiB: 128 rows x 64 bf16
constexpr uint32_t kTailWSlice = kTailN * kMlpBK * 2;      // 8 KiB: 64 rows x 64 bf16
constexpr int kTailSlices = kMlpN / kMlpBK;                // 4
constexpr uint32_t kTailA = kTailSlices * kTailASlice;     // 64 KiB
constexpr uint32_t kTailW = kTailSlices * kTailWSlice;     // 32 KiB
constexpr int kTailSmem = kTailA + 2 * kTailW + 1024 + 256;
constexpr uint32_t kTailTmemCols = 128;
constexpr int kTailThreads = 512;   // 16 warps: four per TMEM lane quarter, 16 columns each

struct TailParams {
    int32_t M;
    const float *b2, *b3;   // [256]
    const uint16_t *w4;     // [256] bf16 bits
    float b4;
    uint16_t *a2;           // [tiles * 128, 256] bf16 bits (workspace)
    float *out;             // [M]
    int32_t *status;
};

__global__ void __launch_bounds__(kTailThreads, 1) mlp_tail_kernel(const __grid_constant__ CUtensorMap tmAct,
                                                                 const __grid_constant__ CUtensorMap tmW2,
                                                                 const __grid_constant__ CUtensorMap tmW3,
                                                                 const __grid_constant__ CUtensorMap tmAct2,
                                                                 const __grid_constant__ TailParams p) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                            ~static_cast<uintptr_t>(1023));
    unsigned char *bufA = smem, *bufW2 = smem + kTailA, *bufW3 = smem + kTailA + kTailW;
    uint64_t *bar = reinterpret_cast<uint64_t *>(smem + kTailA + 2 * kTailW);
    uint64_t *fullA = bar, *fullW2 = bar + 1, *fullW3 = bar + 2, *mma2 = bar + 3, *mma3 = bar + 4, *fullA2 = bar + 5;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bar + 6);
    __shared__ int s_abort;
    __shared__ float s_b2[kTailN], s_b3[kTailN], s_w4[kTailN];
    __shared__ float s_part[3][kMlpBM];             // warps 1..3 of a quarter: their parts of each row's dot product
    __shared__ float s_head[kTailCluster][kMlpBM];  // (CTA 0) each CTA's dot product of each row
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t rank = cluster_rank();
    const int m0 = (blockIdx.x / kTailCluster) * kMlpBM;
    const int n0 = static_cast<int>(rank) * kTailN;
    for (int n = tid; n < kTailN; n += kTailThreads) {
        s_b2[n] = __ldg(p.b2 + n0 + n);
        s_b3[n] = __ldg(p.b3 + n0 + n);
        s_w4[n] = __uint_as_float(static_cast<uint32_t>(__ldg(p.w4 + n0 + n)) << 16);
    }
    if (tid == 0) {
        for (int i = 0; i < 6; ++i) mbar_init(&bar[i], 1);
        fence_mbar_init();
        s_abort = 0;
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(tmem_slot)),
                     "r"(kTailTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (tid == 0) {
        // the weights do not depend on the first layer: loaded while it finishes
        mbar_arrive_expect_tx(fullW2, kTailW);
        for (int c = 0; c < kTailSlices; ++c)
            tma_load_2d(smem_addr(bufW2 + c * kTailWSlice), &tmW2, c * kMlpBK, n0, smem_addr(fullW2));
        mbar_arrive_expect_tx(fullW3, kTailW);
        for (int c = 0; c < kTailSlices; ++c)
            tma_load_2d(smem_addr(bufW3 + c * kTailWSlice), &tmW3, c * kMlpBK, n0, smem_addr(fullW3));
    }
    // launched as a programmatic dependent of the first layer: a1 (and the
    // workspace, which a2 overwrites) only once that grid has completed
    griddep_wait();
    if (tid == 0) {
        mbar_arrive_expect_tx(fullA, kTailA);
        for (int c = 0; c < kTailSlices; ++c)
            tma_load_2d(smem_addr(bufA + c * kTailASlice), &tmAct, c * kMlpBK, m0, smem_addr(fullA));
    } else if (warp == 1 && lane == 0) {
        const bool okA = mbar_wait_bounded(fullA, 0u, kWaitPolls), okB = mbar_wait_bounded(fullW2, 0u, kWaitPolls);
        if (okA && okB) {
            tc_fence_after();
#pragma unroll 1
            for (int c = 0; c < kTailSlices; ++c)
#pragma unroll
                for (int kk = 0; kk < kMlpBK / 16; ++kk)
                    umma_f16<kTailN>(tmem, umma_desc_sw128(smem_addr(bufA + c * kTailASlice) + kk * 32),
                                     umma_desc_sw128(smem_addr(bufW2 + c * kTailWSlice) + kk * 32),
                                     (c | kk) != 0 ? 1u : 0u);
        } else {
            s_abort = 1;
        }
        umma_commit(smem_addr(mma2));   // (arrives at once when nothing was issued)
    }
    __syncwarp();

    // layer-2 epilogue: warp w reads TMEM lanes 32 (w % 4) .. + 31 (tile
    // rows), columns 16 (w / 4) .. + 15 of this CTA's 64
    const int quarter = warp & 3, part = warp >> 2;
    const int row = quarter * 32 + lane;
    const uint32_t tlane = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    bool ok = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(mma2, 0u, kWaitPolls));
    tc_fence_after();
    {
        uint32_t v[16];
        tmem_ld16_or0(ok, tlane + part * 16, v);
        uint32_t w[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const int j = 2 * q;
            w[q] = pack_bf16x2(gelu_erf(__uint_as_float(v[j]) + s_b2[part * 16 + j]),
                               gelu_erf(__uint_as_float(v[j + 1]) + s_b2[part * 16 + j + 1]));
        }
        uint4 *dst = reinterpret_cast<uint4 *>(p.a2 + static_cast<int64_t>(m0 + row) * kMlpN + n0 + part * 16);
        __stcg(dst, make_uint4(w[0], w[1], w[2], w[3]));
        __stcg(dst + 1, make_uint4(w[4], w[5], w[6], w[7]));
    }
    fence_proxy_async_global();   // the stores, before the other CTAs' TMA loads read them
    cluster_sync();               // the four column blocks of a2 are in the workspace (release / acquire)

    // the a2 tile into bufA (a1 was consumed by the finished layer-2 MMAs)
    if (tid == 0) {
        mbar_arrive_expect_tx(fullA2, kTailA);
        for (int c = 0; c < kTailSlices; ++c)
            tma_load_2d(smem_addr(bufA + c * kTailASlice), &tmAct2, c * kMlpBK, m0, smem_addr(fullA2));
    }
    if (warp == 1 && lane == 0) {
        if (ok && mbar_wait_bounded(fullA2, 0u, kWaitPolls) && mbar_wait_bounded(fullW3, 0u, kWaitPolls)) {
            tc_fence_after();
#pragma unroll 1
            for (int c = 0; c < kTailSlices; ++c)
#pragma unroll
                for (int kk = 0; kk < kMlpBK / 16; ++kk)
                    umma_f16<kTailN>(tmem + kTailN, umma_desc_sw128(smem_addr(bufA + c * kTailASlice) + kk * 32),
                                     umma_desc_sw128(smem_addr(bufW3 + c * kTailWSlice) + kk * 32),
                                     (c | kk) != 0 ? 1u : 0u);
        } else {
            s_abort = 1;
        }
        umma_commit(smem_addr(mma3));
    }
    __syncwarp();

    // layer-3 epilogue and head: this thread's part of the row's dot product
    ok = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(mma3, 0u, kWaitPolls)) && ok;
    tc_fence_after();
    griddep_launch_dependents();   // whatever follows may set up (it still waits for this grid)
    float t = 0.f;
    {
        uint32_t v[16];
        tmem_ld16_or0(ok, tlane + kTailN + part * 16, v);
#pragma unroll
        for (int j = 0; j < 16; ++j)
            t = fmaf(s_w4[part * 16 + j], gelu_erf(__uint_as_float(v[j]) + s_b3[part * 16 + j]), t);
    }
    if (part > 0) s_part[part - 1][row] = t;
    tc_fence_before();
    __syncthreads();
    if (part == 0)
        st_cluster_f32(map_rank(smem_addr(&s_head[rank][row]), 0u),
                       ((t + s_part[0][row]) + s_part[1][row]) + s_part[2][row]);
    cluster_sync();   // CTA 0 holds the four parts of every row
    if (rank == 0 && part == 0 && ok && m0 + row < p.M)
        p.out[m0 + row] = 1.f / (1.f + expf(-((((s_head[0][row] + s_head[1][row]) + s_head[2][row]) +
                                                s_head[3][row]) + p.b4)));
    if (tid == 0) {
        // every load this CTA issued has landed before its shared memory goes away
        for (int i : {0, 1, 2, 5}) (void)mbar_wait_bounded(&bar[i], 0u, kWaitPolls);
        if (s_abort || !ok) status_or(p.status, SDD_DEV_TIMEOUT);
    }
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTailTmemCols)
                     : "memory");
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    }
    return fn;
}

// Row-major bf16 [rows, K] as a 2D tensor map with (64 x box_rows) boxes and the 128-byte swizzle.
bool make_map(CUtensorMap *map, const void *base, int64_t rows, int K, int box_rows) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
    if (!enc) return false;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(K) * 2};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(kMlpBK), static_cast<cuuint32_t>(box_rows)};
    const cuuint32_t estr[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Encoded maps of recent (address, rows, K) operands: a decode loop passes the
// same weights every round and often the same hidden-state buffer.
struct MapCache {
    struct Entry {
        const void *base;
        int64_t rows;
        int K, box;
        CUtensorMap map;
    };
    static constexpr int kSlots = 8;
    Entry e[kSlots];
    int n = 0, next = 0;
    std::mutex mu;
    bool get(CUtensorMap *out, const void *base, int64_t rows, int K, int box) {
        std::lock_guard<std::mutex> g(mu);
        for (int i = 0; i < n; ++i)
            if (e[i].base == base && e[i].rows == rows && e[i].K == K && e[i].box == box) {
                *out = e[i].map;
                return true;
            }
        if (!make_map(out, base, rows, K, box)) return false;
        e[next] = Entry{base, rows, K, box, *out};
        next = (next + 1) % kSlots;
        n = n < kSlots ? n + 1 : n;
        return true;
    }
};
MapCache g_maps;
constexpr int kMaxDevices = 64;
std::atomic<int> g_attr_ready[kMaxDevices];

// Per-device opt-in of every kernel here to its dynamic shared memory.
cudaError_t mlp_prepare() {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    if (g_attr_ready[dev].load(std::memory_order_acquire)) return cudaSuccess;
    for (auto fn : {mlp_kernel<1, true>, mlp_kernel<2, true>, mlp_kernel<4, true>, mlp_kernel<1, false>,
                    mlp_kernel<2, false>, mlp_kernel<4, false>}) {
        e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kMlpSmem);
        if (e != cudaSuccess) return e;
    }
    e = cudaFuncSetAttribute(mlp_tail_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kTailSmem);
    if (e != cudaSuccess) return e;
    g_attr_ready[dev].store(1, std::memory_order_release);
    return cudaSuccess;
}

// The first layer: A = [A1 | A2] (A2 may be absent: Ka = K), W1 [256, K].
// head: fused GELU / w2 / sigmoid into out; else bf16 activations into act.
cudaError_t launch_layer1(const void *a1, int Ka, const void *a2, int M, int K, const void *W1, const float *b1,
                          const void *w2, float b2, float *out, uint16_t *act, bool head, float *ws, int32_t *status,
                          cudaStream_t stream, const char **why) {
    CUtensorMap tmA, tmA2, tmB;
    if (!g_maps.get(&tmA, a1, M, Ka, kMlpBM) || !g_maps.get(&tmB, W1, kMlpN, K, kMlpN) ||
        !g_maps.get(&tmA2, a2 ? a2 : a1, M, a2 ? K - Ka : Ka, kMlpBM)) {
        *why = "cuTensorMapEncodeTiled failed";
        return cudaErrorInvalidValue;
    }
    cudaError_t e = mlp_prepare();
    if (e != cudaSuccess) return e;
    // split K four ways when the slices divide evenly (more SMs, no reloads)
    const int nk = K / kMlpBK;
    const int S = (nk % 4 == 0 && nk >= 8) ? 4 : (nk % 2 == 0 && nk >= 4) ? 2 : 1;
    MlpParams p;
    p.M = M;
    p.K = K;
    p.Ka = Ka;
    p.b1 = b1;
    p.w2 = static_cast<const uint16_t *>(w2);
    p.b2 = b2;
    p.out = out;
    p.act = act;
    p.ws = ws;
    p.status = status;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(((M + kMlpBM - 1) / kMlpBM) * S);
    cfg.blockDim = dim3(kMlpThreads);
    cfg.dynamicSmemBytes = kMlpSmem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = S;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // setup overlaps the work ahead
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    if (head) {
        if (S == 4) return cudaLaunchKernelEx(&cfg, mlp_kernel<4, true>, tmA, tmA2, tmB, p);
        if (S == 2) return cudaLaunchKernelEx(&cfg, mlp_kernel<2, true>, tmA, tmA2, tmB, p);
        return cudaLaunchKernelEx(&cfg, mlp_kernel<1, true>, tmA, tmA2, tmB, p);
    }
    if (S == 4) return cudaLaunchKernelEx(&cfg, mlp_kernel<4, false>, tmA, tmA2, tmB, p);
    if (S == 2) return cudaLaunchKernelEx(&cfg, mlp_kernel<2, false>, tmA, tmA2, tmB, p);
    return cudaLaunchKernelEx(&cfg, mlp_kernel<1, false>, tmA, tmA2, tmB, p);
}

}  // namespace

size_t mlp_workspace_bytes(int M) {
    const int64_t tiles = (static_cast<int64_t>(M) + kMlpBM - 1) / kMlpBM;
    return static_cast<size_t>(tiles) * 4 * kMlpN * kMlpBM * sizeof(float);   // K split at most four ways
}

cudaError_t launch_mlp(const void *h, int M, int K, const void *W1, const float *b1, const void *w2, float b2,
                       float *out, void *ws, int32_t *status, cudaStream_t stream, const char **why) {
    *why = nullptr;
    if (M == 0) return cudaSuccess;
    return launch_layer1(h, K, nullptr, M, K, W1, b1, w2, b2, out, nullptr, true, static_cast<float *>(ws), status,
                         stream, why);
}

cudaError_t launch_scorer_deep(const void *h, int Kh, const void *f, int M, const void *W1, const float *b1,
                               const void *W2, const float *b2, const void *W3, const float *b3, const void *w4,
                               float b4, uint16_t *act, float *out, void *ws, int32_t *status, cudaStream_t stream,
                               const char **why) {
    *why = nullptr;
    if (M == 0) return cudaSuccess;
    cudaError_t e = launch_layer1(h, Kh, f, M, Kh + kMlpN, W1, b1, nullptr, 0.f, nullptr, act, false,
                                  static_cast<float *>(ws), status, stream, why);
    if (e != cudaSuccess || *why) return e;
    const int64_t rows_pad = ((static_cast<int64_t>(M) + kMlpBM - 1) / kMlpBM) * kMlpBM;
    CUtensorMap tmAct, tmW2, tmW3, tmAct2;
    if (!g_maps.get(&tmAct, act, M, kMlpN, kMlpBM) || !g_maps.get(&tmW2, W2, kMlpN, kMlpN, kTailN) ||
        !g_maps.get(&tmW3, W3, kMlpN, kMlpN, kTailN) || !g_maps.get(&tmAct2, ws, rows_pad, kMlpN, kMlpBM)) {
        *why = "cuTensorMapEncodeTiled failed";
        return cudaErrorInvalidValue;
    }
    TailParams p;
    p.M = M;
    p.b2 = b2;
    p.b3 = b3;
    p.w4 = static_cast<const uint16_t *>(w4);
    p.b4 = b4;
    p.a2 = static_cast<uint16_t *>(ws);   // the first layer's partials are dead once it has finished
    p.out = out;
    p.status = status;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(((M + kMlpBM - 1) / kMlpBM) * kTailCluster);
    cfg.blockDim = dim3(kTailThreads);
    cfg.dynamicSmemBytes = kTailSmem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kTailCluster;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // weight loads overlap the first layer
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, mlp_tail_kernel, tmAct, tmW2, tmW3, tmAct2, p);
}

// ---------------------------------------------------------------------------
// The learned scorer's scalar-feature block (App. A.7's list): one warp per
// position writes its 256 bf16 columns (lane u: columns 8u .. 8u + 7), zero
// except the logits-side features and the position ones.
// ---------------------------------------------------------------------------
namespace {
__global__ void scorer_features_kernel(const float *maxprob, const float *entropy, const float *margin,
                                       const float *top5, int64_t M, int gamma, float gen, uint16_t *f) {
    const int64_t w = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (w >= M) return;
    float v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = 0.f;
    if (lane == 0) {   // columns 4..7: top-1 probability, its log, entropy, its negative
        const float mp = __ldg(maxprob + w), h = __ldg(entropy + w);
        v[4] = mp;
        v[5] = logf(mp);
        v[6] = h;
        v[7] = -h;
    } else if (lane == 1) {   // columns 8, 9: margin, top-5 mass; 14, 15: block position, generated length
        v[0] = __ldg(margin + w);
        v[1] = __ldg(top5 + w);
        v[6] = static_cast<float>(w % gamma) / static_cast<float>(gamma);
        v[7] = gen;
    }
    const uint4 u = make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]), pack_bf16x2(v[4], v[5]),
                               pack_bf16x2(v[6], v[7]));
    reinterpret_cast<uint4 *>(f + w * kMlpN)[lane] = u;
}
}  // namespace

cudaError_t launch_scorer_features(const float *maxprob, const float *entropy, const float *margin, const float *top5,
                                   int64_t M, int gamma, float gen, uint16_t *f, cudaStream_t stream) {
    if (M == 0) return cudaSuccess;
    const int64_t threads = M * 32;
    scorer_features_kernel<<<static_cast<unsigned>((threads + 255) / 256), 256, 0, stream>>>(
        maxprob, entropy, margin, top5, M, gamma, gen, f);
    return cudaGetLastError();
}

}  // namespace sdd
