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

#include "internal.h"

namespace sdd {
namespace {

constexpr int kMlpN = 256;           // hidden units = UMMA N
constexpr int kMlpBM = 128;          // rows per CTA = UMMA M
constexpr int kMlpBK = 64;           // K per stage: 64 bf16 = one 128-byte swizzle row
constexpr int kMlpStages = 4;
constexpr int kMlpThreads = 128;     // warp 0 lane 0: TMA producer; warp 1 lane 0: MMA issuer; all: epilogue
constexpr uint32_t kATileBytes = kMlpBM * kMlpBK * 2;   // 16 KiB
constexpr uint32_t kBTileBytes = kMlpN * kMlpBK * 2;    // 32 KiB
constexpr uint32_t kStageBytes = kATileBytes + kBTileBytes;
constexpr int kMlpSmem = kMlpStages * kStageBytes + 1024 + 256;   // + alignment slack + barriers
constexpr uint32_t kTmemCols = 256;

struct MlpParams {
    int32_t M, K;
    const float *b1;        // [256]
    const uint16_t *w2;     // [256] bf16 bits
    float b2;
    float *out;             // [M]
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

__global__ void __launch_bounds__(kMlpThreads, 1) mlp_kernel(const __grid_constant__ CUtensorMap tmA,
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
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int m0 = blockIdx.x * kMlpBM;
    const int nk = p.K / kMlpBK;

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
        // TMA producer: stage s holds K slice t of the A tile (rows m0..m0+127)
        // and of the B tile (all 256 hidden units)
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
            tma_load_2d(a, &tmA, t * kMlpBK, m0, smem_addr(&full[s]));
            tma_load_2d(a + kATileBytes, &tmB, t * kMlpBK, 0, smem_addr(&full[s]));
        }
        // let every issued load land before the CTA can leave (already true
        // unless a wait gave up): the last load into each stage
        for (int s = 0; s < kMlpStages && s < t; ++s) {
            const int last = ((t - 1 - s) / kMlpStages) * kMlpStages + s;   // last load issued into stage s
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

    // epilogue: thread (warp w, lane l) owns row 32 w + l of the tile = TMEM lane 32 w + l
    // warp-uniform, since tcgen05.ld below is a .sync.aligned warp instruction
    const bool ok = __all_sync(0xFFFFFFFFu, mbar_wait_bounded(done, 0u, kWaitPolls));
    tc_fence_after();
    if (!ok) s_abort = 1;
    const int row = warp * 32 + lane;
    float t2 = p.b2;
    if (ok) {
        const uint32_t tbase = tmem + (static_cast<uint32_t>(warp * 32) << 16);
#pragma unroll 1
        for (int c = 0; c < kMlpN; c += 32) {
            uint32_t v[32];
            tmem_ld32(tbase + c, v);
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                const float z = __uint_as_float(v[j]) + __ldg(p.b1 + c + j);
                const float g = 0.5f * z * (1.f + erff(z * 0.70710678118654752f));
                const float w = __uint_as_float(static_cast<uint32_t>(__ldg(p.w2 + c + j)) << 16);
                t2 = fmaf(w, g, t2);
            }
        }
        if (m0 + row < p.M) p.out[m0 + row] = 1.f / (1.f + expf(-t2));
    }
    tc_fence_before();
    __syncthreads();
    if (tid == 0 && s_abort) status_or(p.status, SDD_DEV_TIMEOUT);
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
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

}  // namespace

cudaError_t launch_mlp(const void *h, int M, int K, const void *W1, const float *b1, const void *w2, float b2,
                       float *out, int32_t *status, cudaStream_t stream, const char **why) {
    *why = nullptr;
    if (M == 0) return cudaSuccess;
    CUtensorMap tmA, tmB;
    if (!make_map(&tmA, h, M, K, kMlpBM) || !make_map(&tmB, W1, kMlpN, K, kMlpN)) {
        *why = "cuTensorMapEncodeTiled failed";
        return cudaErrorInvalidValue;
    }
    // per function and device; cheap, so set on every call
    cudaError_t e = cudaFuncSetAttribute(mlp_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kMlpSmem);
    if (e != cudaSuccess) return e;
    MlpParams p;
    p.M = M;
    p.K = K;
    p.b1 = b1;
    p.w2 = static_cast<const uint16_t *>(w2);
    p.b2 = b2;
    p.out = out;
    p.status = status;
    mlp_kernel<<<(M + kMlpBM - 1) / kMlpBM, kMlpThreads, kMlpSmem, stream>>>(tmA, tmB, p);
    return cudaGetLastError();
}

}  // namespace sdd
