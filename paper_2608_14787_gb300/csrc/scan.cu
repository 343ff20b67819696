// scan.cu -- the streaming kernel (the per-warp work is in scan.cuh).
#include <atomic>

#include "scan.cuh"

namespace sdd {

namespace {

// FEAT: also the five largest logits of every drafter row piece (extended
// features); the kernel without it is unchanged.
template <int DT, bool FEAT>
__global__ void __launch_bounds__(kThreads, 1) scan_kernel(const __grid_constant__ ScanParams p) {
    extern __shared__ __align__(128) unsigned char smem[];
    const int64_t gw = static_cast<int64_t>(blockIdx.x) * kWarpsPerCta + (threadIdx.x >> 5);
    if (gw >= p.W) return;
    // launched as a programmatic dependent of whatever precedes it in the
    // stream: nothing is read or written before that work has completed
    griddep_wait();
    scan_warp<DT, FEAT>(p, smem, gw, threadIdx.x >> 5, kWarpsPerCta);
}

}  // namespace

int scan_max_ctas_per_sm() {
    int n = 0;
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, scan_kernel<SDD_BF16, false>, kThreads, kScanSmem);
    return n;
}

// Opt both instantiations in to their dynamic shared memory on the current device.
cudaError_t scan_prepare_device() {
    void (*const kernels[])(ScanParams) = {scan_kernel<SDD_BF16, false>, scan_kernel<SDD_F32, false>,
                                           scan_kernel<SDD_BF16, true>, scan_kernel<SDD_F32, true>};
    for (auto k : kernels) {
        const cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, kScanSmem);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

// The launch overhead of the streaming grid overlaps the tail of the work
// ahead of it in the stream (the kernel waits for that work to complete).
namespace {
std::atomic<uint32_t> g_wait_polls{0};
std::atomic<int> g_drop_copy{0};
}  // namespace

void set_scan_wait_hooks(uint32_t polls, int drop_copy) {
    g_wait_polls.store(polls, std::memory_order_relaxed);
    g_drop_copy.store(drop_copy ? 1 : 0, std::memory_order_relaxed);
}

cudaError_t launch_scan(const ScanParams &p, int grid, cudaStream_t stream) {
    const bool bf = p.dtype == SDD_BF16, feat = p.feat != nullptr;
    void (*const k)(ScanParams) = feat ? (bf ? scan_kernel<SDD_BF16, true> : scan_kernel<SDD_F32, true>)
                                       : (bf ? scan_kernel<SDD_BF16, false> : scan_kernel<SDD_F32, false>);
    ScanParams q = p;
    const uint32_t polls = g_wait_polls.load(std::memory_order_relaxed);
    q.wait_polls = polls ? polls : kWaitPolls;
    q.drop_copy = g_drop_copy.load(std::memory_order_relaxed);
    return launch_dependent(k, dim3(grid), dim3(kThreads), kScanSmem, stream, q);
}

}  // namespace sdd
