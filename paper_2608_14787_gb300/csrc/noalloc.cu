// noalloc.cu -- sdd_confidence_noalloc: the drafter-row statistics of
// sdd_confidence for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc (or any allocating routine) at the point
// where they need the statistics: code running inside a CUDA graph capture, a
// framework whose device memory is owned by a fixed arena, or an embedded
// host loop without an allocator.  This entry point takes no workspace.  Its
// scratch -- the per-warp partial states of the streaming kernel -- lives in one file-scope device array of fixed size that every GPU
// which loads this library holds until the process exits.
#include <algorithm>
#include <atomic>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include "internal.h"

namespace sdd {
namespace {

// Capacity: up to kNoAllocMaxRows drafter rows (B * gamma) per call, streamed
// by at most kNoAllocMaxWarps warps.
constexpr int kNoAllocMaxRows = 8192;
constexpr int kNoAllocMaxWarps = 4096;
constexpr size_t kPartialBytes = static_cast<size_t>(kNoAllocMaxRows + kNoAllocMaxWarps) * sizeof(Partial);
constexpr size_t kScratchBytes = kPartialBytes;  // 384 KiB

// The scratch.  In host code this name is only a stand-in for the device
// symbol: its device address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

sdd_status_t na_fail(sdd_status_t s, const char *fmt, ...) __attribute__((format(printf, 2, 3)));
sdd_status_t na_fail(sdd_status_t s, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    set_last_error(buf);   // reported by sdd_last_error()
    return s;
}

// Per-device set-up, done once per device (with that device current) by the
// first call on it: the device address of g_scratch and the launch geometry.
constexpr int kMaxDevices = 64;
struct NoAllocDev {
    unsigned char *scratch;
    int W_max;
};
NoAllocDev g_na_dev[kMaxDevices];
std::atomic<int> g_na_ready[kMaxDevices];

sdd_status_t noalloc_setup(NoAllocDev &out) {
    int d = 0;
    cudaError_t e = cudaGetDevice(&d);
    if (e != cudaSuccess) return na_fail(SDD_ERR_CUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
    if (d < 0 || d >= kMaxDevices) return na_fail(SDD_ERR_UNSUPPORTED, "device ordinal %d out of range", d);
    if (!g_na_ready[d].load(std::memory_order_acquire)) {
        NoAllocDev nd{};
        void *ptr = nullptr;
        e = cudaGetSymbolAddress(&ptr, g_scratch);
        if (e != cudaSuccess) return na_fail(SDD_ERR_CUDA, "cudaGetSymbolAddress: %s", cudaGetErrorString(e));
        nd.scratch = static_cast<unsigned char *>(ptr);
        int sms = 0;
        e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, d);
        if (e != cudaSuccess) return na_fail(SDD_ERR_CUDA, "cudaDeviceGetAttribute: %s", cudaGetErrorString(e));
        e = scan_prepare_device();
        if (e != cudaSuccess) return na_fail(SDD_ERR_CUDA, "cudaFuncSetAttribute: %s", cudaGetErrorString(e));
        const int ctas = scan_max_ctas_per_sm();
        if (ctas < 1) return na_fail(SDD_ERR_UNSUPPORTED, "streaming kernel does not fit on this device");
        nd.W_max = std::min(sms * ctas * kWarpsPerCta, kNoAllocMaxWarps);
        g_na_dev[d] = nd;
        g_na_ready[d].store(1, std::memory_order_release);
    }
    out = g_na_dev[d];
    return SDD_OK;
}

}  // namespace
}  // namespace sdd

using namespace sdd;

extern "C" {

sdd_status_t sdd_confidence_noalloc(const void *draft_logits, sdd_dtype_t dtype, int B, int gamma, int V,
                                    int64_t row_stride, const int32_t *draft_tokens, float *q, float *logq,
                                    float *maxprob, double *lse, float *entropy, int32_t *argmax, int32_t *status,
                                    sdd_stream_t stream) {
    if (dtype != SDD_F32 && dtype != SDD_BF16) return na_fail(SDD_ERR_INVALID_ARGUMENT, "dtype %d unknown", dtype);
    if (B < 0) return na_fail(SDD_ERR_INVALID_ARGUMENT, "B = %d < 0", B);
    if (gamma < 1 || gamma > SDD_MAX_GAMMA)
        return na_fail(SDD_ERR_INVALID_ARGUMENT, "gamma = %d outside [1, %d]", gamma, SDD_MAX_GAMMA);
    if (V < 1) return na_fail(SDD_ERR_INVALID_ARGUMENT, "V = %d < 1", V);
    const int esz = (dtype == SDD_BF16) ? 2 : 4;
    if (row_stride < V || (row_stride * esz) % 16 != 0 || row_stride * esz > (int64_t(1) << 31))
        return na_fail(SDD_ERR_INVALID_ARGUMENT,
                       "row_stride must be >= V, a multiple of 16 bytes and at most 2 GiB per row");
    const int64_t rows = static_cast<int64_t>(B) * gamma;
    if (rows > kNoAllocMaxRows)
        return na_fail(SDD_ERR_INVALID_ARGUMENT,
                       "B * gamma = %lld exceeds the %d rows of the fixed scratch of sdd_confidence_noalloc; "
                       "split the batch or use sdd_confidence with a workspace",
                       static_cast<long long>(rows), kNoAllocMaxRows);
    if (rows == 0) return SDD_OK;
    if (!draft_logits || reinterpret_cast<uintptr_t>(draft_logits) % 16 != 0)
        return na_fail(SDD_ERR_INVALID_ARGUMENT, "draft_logits is NULL or not 16-byte aligned");
    if (!draft_tokens || !q) return na_fail(SDD_ERR_INVALID_ARGUMENT, "draft_tokens and q must not be NULL");

    NoAllocDev nd;
    sdd_status_t s = noalloc_setup(nd);
    if (s != SDD_OK) return s;
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);

    ScanParams p;
    std::memset(&p, 0, sizeof p);
    p.n_groups = 1;
    p.dtype = dtype;
    p.V = V;
    p.RV = static_cast<int32_t>((static_cast<int64_t>(V) * esz + 15) / 16);
    p.gamma = gamma;
    p.kcap = 1;
    p.B = B;
    p.tokens = draft_tokens;
    p.partials = reinterpret_cast<Partial *>(nd.scratch);
    p.status = status;
    ScanGroup &G = p.grp[0];
    G.base = static_cast<const char *>(draft_logits);
    G.stride_bytes = row_stride * esz;
    G.npos = gamma;
    G.kind = 0;
    G.nb = B;
    G.q = q;
    G.logq = logq;
    G.maxprob = maxprob;
    G.lse = lse;
    G.entropy = entropy;
    G.argmax = argmax;
    p.rows0 = rows;
    p.rows = rows;
    p.T = rows * p.RV;
    const int64_t W = scan_warps(nd.W_max, p.T, p.rows);
    p.W = static_cast<int32_t>(W);
    set_divisors(p);
    if (static_cast<double>(p.C) * static_cast<double>(W) >= 9.007199254740992e15)   // 2^53
        return na_fail(SDD_ERR_UNSUPPORTED, "%lld vectors of logits exceed the index arithmetic", (long long)p.T);

    cudaError_t e = launch_scan(p, static_cast<int>((W + kWarpsPerCta - 1) / kWarpsPerCta), st);
    if (e != cudaSuccess) return na_fail(SDD_ERR_CUDA, "scan launch: %s", cudaGetErrorString(e));
    e = launch_decide(p, st);   // row finalisation only (no decisions)
    if (e != cudaSuccess) return na_fail(SDD_ERR_CUDA, "decide launch: %s", cudaGetErrorString(e));
    return SDD_OK;
}

}  // extern "C"
