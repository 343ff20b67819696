// mlp.cu -- the stand-in survival scorer of the decode-loop workload on the
// 5th-generation tensor cores:
//
//   s[m] = sigmoid(w2 . GELU(W1 h[m] + b1) + b2),  GELU(z) = z Phi(z) (erf form),
//
// for h [M, K] bf16 (drafter hidden states), W1 [256, K] bf16 (one row per
// hidden unit), b1 fp32 [256], w2 bf16 [256], b2 fp32 -- the form of the
// learned scorer of App. A.7 with one hidden layer and random weights.
//
// One CTA per 128-row tile computes the whole 128 x 256 product W1 h on
// tcgen05: a four-stage ring of 48 KiB (A tile 128 x 64, B tile 256 x 64, both
// K-major with the 128-byte swizzle) filled by 2D TMA loads; one thread issues
// tcgen05.mma.kind::f16 (M = 128, N = 256, K = 16, fp32 accumulate) into a
// 256-column TMEM accumulator and commits each stage back to the producer;
// then four warps read their 32 rows from TMEM (tcgen05.ld) and fuse bias,
// GELU, the w2 dot product and the sigmoid, writing one float per row.
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
constexpr int kMlpThreads = 256;     // warp 0 lane 0: TMA producer; warp 1 lane 0: MMA issuer; all: epilogue
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

// Instruction descriptor of kind::f16: fp32 D, bf16 A and B, both K-major, N, M.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(kMlpN >> 3) << 17) |
                            (static_cast<uint32_t>(kMlpBM >> 4) << 24);

__device__ __forceinline__ void umma_f16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate)
        : "memory");
}

// Arrive on `bar` once every tcgen05 operation this thread issued so far completes.
__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 32 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]),
          "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]),
          "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
          "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
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
__device__ __forceinline__ void st_cluster_v4(uint32_t addr, float a, float b, float c, float d) {
    asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(a), "f"(b), "f"(c), "f"(d)
                 : "memory");
}

// Two fp32 values rounded to bf16 (round to nearest even), packed (a low).
__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
    uint32_t d;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(b), "f"(a));
    return d;
}

// Row stride (floats) of a partial accumulator dumped to shared memory: a
// multiple of 4 for 16-byte accesses, 4 mod 32 so that 8 consecutive rows
// cover all banks.
constexpr int kAccStride = kMlpN + 4;

// Grid: (M tiles x S) CTAs in clusters of S along x (S = 1, 2 or 4 splits of
// K).  CTA rank r of a cluster multiplies K slices [r nk/S, (r+1) nk/S) of its
// 128-row tile into its own TMEM.  Rows [q R, (q+1) R) of the tile (R = 128/S)
// are finished by CTA q: once every CTA of the cluster has finished its
// mainloop (cluster barrier), every CTA pushes its partial of those rows into
// slot r of CTA q's receive area (distributed shared-memory stores over the
// idle stage ring); after a second cluster barrier each CTA sums its S slots
// locally and runs the epilogue.
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
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(done + 1);
    __shared__ int s_abort;
    __shared__ float s_b1[kMlpN], s_w2[kMlpN];   // epilogue constants, widened once per CTA
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    for (int n = tid; n < kMlpN; n += kMlpThreads) {
        s_b1[n] = __ldg(p.b1 + n);
        s_w2[n] = HEAD ? __uint_as_float(static_cast<uint32_t>(__ldg(p.w2 + n)) << 16) : 0.f;
    }
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
        fence_mbar_init();
        s_abort = 0;
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(tmem_slot)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
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

    // push the partial accumulator: warp w reads TMEM lanes 32 (w % 4) ..
    // 32 (w % 4) + 31 (tile rows, all finished by CTA q = 32 (w % 4) / R), columns
    // half w / 4
    const bool ok = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(done, 0u, kWaitPolls));
    tc_fence_after();
    if (!ok) s_abort = 1;
    constexpr int R = kMlpBM / S;
    float *recv = reinterpret_cast<float *>(smem);   // [S slots][R rows][kAccStride], over the idle ring
    if (S > 1) cluster_sync();   // every CTA's ring is idle before any partial is pushed into it
    {
        const int quarter = warp & 3, half = warp >> 2;
        const int dest = (quarter * 32) / R;
        const int drow = quarter * 32 - dest * R + lane;
        const uint32_t local = smem_addr(recv + (static_cast<int>(rank) * R + drow) * kAccStride);
        const uint32_t dst = (S > 1) ? map_rank(local, static_cast<uint32_t>(dest)) : local;
        const uint32_t tbase = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
#pragma unroll 1
        for (int c = half * (kMlpN / 2); c < (half + 1) * (kMlpN / 2); c += 32) {
            uint32_t v[32];
            if (ok) {
                tmem_ld32(tbase + c, v);
            } else {
#pragma unroll
                for (int j = 0; j < 32; ++j) v[j] = 0u;
            }
#pragma unroll
            for (int j = 0; j < 8; ++j)
                st_cluster_v4(dst + (c + 4 * j) * 4, __uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                              __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
        }
    }
    tc_fence_before();
    if (S > 1)
        cluster_sync();   // every pushed partial has landed (release / acquire)
    else
        __syncthreads();

    // epilogue: the R rows of this CTA, P = kMlpThreads / R threads per row;
    // thread p of a row takes the 16-byte column chunks p, p + P, p + 2P, ...
    // (the row's threads read consecutive chunks: no bank conflicts)
    {
        constexpr int P = kMlpThreads / R;
        const int lrow = tid / P;
        const int pp = tid % P;
        const int grow = m0 + static_cast<int>(rank) * R + lrow;
        float t2 = 0.f;
#pragma unroll 4
        for (int ch = pp; ch < kMlpN / 4; ch += P) {
            const int c = 4 * ch;
            float4 z = *reinterpret_cast<const float4 *>(recv + lrow * kAccStride + c);
#pragma unroll
            for (int q = 1; q < S; ++q) {
                const float4 v = *reinterpret_cast<const float4 *>(recv + (q * R + lrow) * kAccStride + c);
                z.x += v.x;
                z.y += v.y;
                z.z += v.z;
                z.w += v.w;
            }
            const float zz[4] = {z.x, z.y, z.z, z.w};
            float gg[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int n = c + e;
                const float u = zz[e] + s_b1[n];
                gg[e] = 0.5f * u * (1.f + erff(u * 0.70710678118654752f));
                if (HEAD) t2 = fmaf(s_w2[n], gg[e], t2);
            }
            if (!HEAD && ok && grow < p.M) {
                // four bf16 activations (round to nearest even) in one 8-byte store
                const uint32_t lo = pack_bf16x2(gg[0], gg[1]), hi = pack_bf16x2(gg[2], gg[3]);
                *reinterpret_cast<uint2 *>(p.act + static_cast<int64_t>(grow) * kMlpN + c) = make_uint2(lo, hi);
            }
        }
        if (HEAD) {
            for (int off = 1; off < P; off <<= 1) t2 += __shfl_xor_sync(0xFFFFFFFFu, t2, off);
            if (tid % P == 0 && ok && grow < p.M) p.out[grow] = 1.f / (1.f + expf(-(t2 + p.b2)));
        }
    }
    __syncthreads();
    if (tid == 0 && s_abort) status_or(p.status, SDD_DEV_TIMEOUT);
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
}

// ---------------------------------------------------------------------------
// Layers 2 and 3 and the head of the deep scorer (K -> 256 -> 256 -> 256 -> 1):
// one CTA per 128-row tile.  The tile's first-layer activations (128 x 256
// bf16, four 64-column slices with the 128-byte swizzle) and W2 (256 x 256)
// arrive by TMA; z2 = W2 a1 goes to TMEM columns 0..255; the epilogue writes
// a2 = bf16(GELU(z2 + b2)) back over a1 in the same swizzled K-major layout
// (16-byte unit u of row r at r * 128 + (u ^ (r % 8)) * 16 within a slice)
// while W3 replaces W2; z3 = W3 a2 goes to TMEM columns 256..511; the last
// epilogue computes sigmoid(w4 . GELU(z3 + b3) + b4) per row.
// ---------------------------------------------------------------------------
constexpr uint32_t kTailASlice = kMlpBM * kMlpBK * 2;      // 16 KiB: 128 rows x 64 bf16
constexpr uint32_t kTailBSlice = kMlpN * kMlpBK * 2;       // 32 KiB: 256 rows x 64 bf16
constexpr int kTailSlices = kMlpN / kMlpBK;                // 4
constexpr uint32_t kTailA = kTailSlices * kTailASlice;     // 64 KiB
constexpr uint32_t kTailB = kTailSlices * kTailBSlice;     // 128 KiB
constexpr int kTailSmem = kTailA + kTailB + 1024 + 256;
constexpr uint32_t kTailTmemCols = 512;
constexpr int kTailThreads = 512;   // 16 warps: four per TMEM lane quarter, 64 columns each

struct TailParams {
    int32_t M;
    const float *b2, *b3;      // [256]
    const uint16_t *w4;        // [256] bf16 bits
    float b4;
    float *out;                // [M]
    int32_t *status;
};

__global__ void __launch_bounds__(kTailThreads, 1) mlp_tail_kernel(const __grid_constant__ CUtensorMap tmAct,
                                                                 const __grid_constant__ CUtensorMap tmW2,
                                                                 const __grid_constant__ CUtensorMap tmW3,
                                                                 const __grid_constant__ TailParams p) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                            ~static_cast<uintptr_t>(1023));
    unsigned char *bufA = smem, *bufB = smem + kTailA;
    uint64_t *bar = reinterpret_cast<uint64_t *>(smem + kTailA + kTailB);
    uint64_t *fullA = bar, *fullW2 = bar + 1, *fullW3 = bar + 2, *mma2 = bar + 3, *mma3 = bar + 4;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bar + 5);
    __shared__ int s_abort;
    __shared__ float s_b2[kMlpN], s_b3[kMlpN], s_w4[kMlpN];
    __shared__ float s_part[3][kMlpBM];   // column parts 1..3 of each row's dot product
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int m0 = blockIdx.x * kMlpBM;
    for (int n = tid; n < kMlpN; n += kTailThreads) {
        s_b2[n] = __ldg(p.b2 + n);
        s_b3[n] = __ldg(p.b3 + n);
        s_w4[n] = __uint_as_float(static_cast<uint32_t>(__ldg(p.w4 + n)) << 16);
    }
    if (tid == 0) {
        for (int i = 0; i < 5; ++i) mbar_init(&bar[i], 1);
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
        mbar_arrive_expect_tx(fullA, kTailA);
        for (int c = 0; c < kTailSlices; ++c)
            tma_load_2d(smem_addr(bufA + c * kTailASlice), &tmAct, c * kMlpBK, m0, smem_addr(fullA));
        mbar_arrive_expect_tx(fullW2, kTailB);
        for (int c = 0; c < kTailSlices; ++c)
            tma_load_2d(smem_addr(bufB + c * kTailBSlice), &tmW2, c * kMlpBK, 0, smem_addr(fullW2));
    } else if (warp == 1 && lane == 0) {
        const bool okA = mbar_wait_bounded(fullA, 0u, kWaitPolls), okB = mbar_wait_bounded(fullW2, 0u, kWaitPolls);
        if (okA && okB) {
            tc_fence_after();
#pragma unroll 1
            for (int c = 0; c < kTailSlices; ++c)
#pragma unroll
                for (int kk = 0; kk < kMlpBK / 16; ++kk)
                    umma_f16(tmem, umma_desc_sw128(smem_addr(bufA + c * kTailASlice) + kk * 32),
                             umma_desc_sw128(smem_addr(bufB + c * kTailBSlice) + kk * 32), (c | kk) != 0 ? 1u : 0u);
        } else {
            s_abort = 1;
        }
        umma_commit(smem_addr(mma2));   // (arrives at once when nothing was issued)
    }
    __syncwarp();

    // layer-2 epilogue: warp w reads TMEM lanes 32 (w % 4) .. + 31 (tile rows),
    // columns 64 (w / 4) .. + 63
    const int quarter = warp & 3, part = warp >> 2;
    const int row = quarter * 32 + lane;
    const uint32_t tlane = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    bool ok = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(mma2, 0u, kWaitPolls));
    tc_fence_after();
    if (tid == 0 && ok) {
        // W2 has been read: W3 takes its place
        mbar_arrive_expect_tx(fullW3, kTailB);
        for (int c = 0; c < kTailSlices; ++c)
            tma_load_2d(smem_addr(bufB + c * kTailBSlice), &tmW3, c * kMlpBK, 0, smem_addr(fullW3));
    }
#pragma unroll 1
    for (int cb = 0; cb < 2; ++cb) {
        const int n0 = part * 64 + cb * 32;
        uint32_t v[32];
        if (ok) {
            tmem_ld32(tlane + n0, v);
        } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = 0u;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {   // four 16-byte units of 8 activations
            uint32_t w[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                float g[2];
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const int j = u * 8 + q * 2 + e;
                    const float z = __uint_as_float(v[j]) + s_b2[n0 + j];
                    g[e] = 0.5f * z * (1.f + erff(z * 0.70710678118654752f));
                }
                w[q] = pack_bf16x2(g[0], g[1]);
            }
            const int n = n0 + u * 8;                       // first column of the unit
            const int slice = n / kMlpBK, unit = (n % kMlpBK) / 8;
            unsigned char *dst = bufA + slice * kTailASlice + row * 128 + ((unit ^ (row & 7)) * 16);
            *reinterpret_cast<uint4 *>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
    fence_proxy_async_smem();   // the generic writes of a2, before the tensor cores read them
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    if (warp == 1 && lane == 0) {
        // (W3 was requested iff ok; its load has landed before the CTA can leave)
        if (ok && mbar_wait_bounded(fullW3, 0u, kWaitPolls)) {
            tc_fence_after();
#pragma unroll 1
            for (int c = 0; c < kTailSlices; ++c)
#pragma unroll
                for (int kk = 0; kk < kMlpBK / 16; ++kk)
                    umma_f16(tmem + 256, umma_desc_sw128(smem_addr(bufA + c * kTailASlice) + kk * 32),
                             umma_desc_sw128(smem_addr(bufB + c * kTailBSlice) + kk * 32), (c | kk) != 0 ? 1u : 0u);
        } else {
            s_abort = 1;
        }
        umma_commit(smem_addr(mma3));
    }
    __syncwarp();

    // layer-3 epilogue and head: each thread's dot product over its 64
    // columns, the four parts of a row added through shared memory
    ok = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(mma3, 0u, kWaitPolls)) && ok;
    tc_fence_after();
    float t = 0.f;
#pragma unroll 1
    for (int cb = 0; cb < 2; ++cb) {
        const int n0 = part * 64 + cb * 32;
        uint32_t v[32];
        if (ok) {
            tmem_ld32(tlane + 256 + n0, v);
        } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = 0u;
        }
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            const float z = __uint_as_float(v[j]) + s_b3[n0 + j];
            t = fmaf(s_w4[n0 + j], 0.5f * z * (1.f + erff(z * 0.70710678118654752f)), t);
        }
    }
    if (part > 0) s_part[part - 1][row] = t;
    tc_fence_before();
    __syncthreads();
    if (part == 0 && ok && m0 + row < p.M)
        p.out[m0 + row] = 1.f / (1.f + expf(-(((t + s_part[0][row]) + s_part[1][row]) + s_part[2][row] + p.b4)));
    if (tid == 0 && (s_abort || !ok)) status_or(p.status, SDD_DEV_TIMEOUT);
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
                          const void *w2, float b2, float *out, uint16_t *act, bool head, int32_t *status,
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
    p.status = status;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(((M + kMlpBM - 1) / kMlpBM) * S);
    cfg.blockDim = dim3(kMlpThreads);
    cfg.dynamicSmemBytes = kMlpSmem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = S;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
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

cudaError_t launch_mlp(const void *h, int M, int K, const void *W1, const float *b1, const void *w2, float b2,
                       float *out, int32_t *status, cudaStream_t stream, const char **why) {
    *why = nullptr;
    if (M == 0) return cudaSuccess;
    return launch_layer1(h, K, nullptr, M, K, W1, b1, w2, b2, out, nullptr, true, status, stream, why);
}

cudaError_t launch_scorer_deep(const void *h, int Kh, const void *f, int M, const void *W1, const float *b1,
                               const void *W2, const float *b2, const void *W3, const float *b3, const void *w4,
                               float b4, uint16_t *act, float *out, int32_t *status, cudaStream_t stream,
                               const char **why) {
    *why = nullptr;
    if (M == 0) return cudaSuccess;
    cudaError_t e = launch_layer1(h, Kh, f, M, Kh + kMlpN, W1, b1, nullptr, 0.f, nullptr, act, false, status,
                                  stream, why);
    if (e != cudaSuccess || *why) return e;
    CUtensorMap tmAct, tmW2, tmW3;
    if (!g_maps.get(&tmAct, act, M, kMlpN, kMlpBM) || !g_maps.get(&tmW2, W2, kMlpN, kMlpN, kMlpN) ||
        !g_maps.get(&tmW3, W3, kMlpN, kMlpN, kMlpN)) {
        *why = "cuTensorMapEncodeTiled failed";
        return cudaErrorInvalidValue;
    }
    TailParams p;
    p.M = M;
    p.b2 = b2;
    p.b3 = b3;
    p.w4 = static_cast<const uint16_t *>(w4);
    p.b4 = b4;
    p.out = out;
    p.status = status;
    mlp_tail_kernel<<<(M + kMlpBM - 1) / kMlpBM, kTailThreads, kTailSmem, stream>>>(tmAct, tmW2, tmW3, p);
    return cudaGetLastError();
}

}  // namespace sdd
