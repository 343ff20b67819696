// pipe.cu -- the pipelined round (sdd_block_pipelined): one launch that
// streams round n's logits and, on the same SMs, finishes round n-1.
//
// A round of the fused path is a streaming pass (every logit once, HBM-bound)
// followed by the decide work (row finalisation, the acceptance rules, the
// schedule, the sampling draw), which is latency-bound: behind its own
// streaming pass it leaves the memory system idle for most of its ~12 us.
// Rounds over independent batches need not wait for one another, so here the
// decide work of round n-1 runs beside the streaming pass of round n: in every
// CTA, the first warps (a team of kPipeTeam = 64 threads; kPipeTeamSmall =
// 128 when round n is a small, latency-bound one) do one (block, draw
// segment) item of round n-1's decide work (decide_cta, its barrier over the
// team only) while the other warps stream round n, the rows divided among
// them.  Measured on GB300 (16 blocks of 32 positions, V = 151,936 bf16, back
// to back): 61.2 us per round against 69.0 us for the streaming and decide
// kernels in turn.  A team of eight decide warps beside eight streaming warps
// (which then streamed a share cut to its decide time) gave 71-75 us, four
// decide warps beside twelve 63.5-64.0 us; with two, a decide item takes ~42
// us under the concurrent stream, still before the streaming warps end.
// Round n-1's partials were written by the previous launch on the stream,
// which has completed when this grid passes griddepcontrol.wait.
#include <algorithm>
#include <atomic>
#include <cstring>

#include "scan.cuh"
#include "decide.cuh"

namespace sdd {

namespace {

struct PipeParams {
    ScanParams next;    // the round streamed by this launch (unused when has_next == 0)
    ScanParams prev;    // the round decided by this launch (unused when has_prev == 0)
    int32_t has_next, has_prev;
    int32_t n_items;    // decide items of prev: blocks x draw segments
    int32_t stage_vec;  // vectors per row of a team's staged chunk of its draw segment (0: none)
};

// The first TEAM threads: prev's decide items of this CTA.  Out of line, so
// that its register allocation stays apart from the streaming loop's.
template <int DT, int TEAM>
__device__ __noinline__ void pipe_decide(const PipeParams &pp, float *s_pref_all) {
    const ScanParams &p = pp.prev;
    const PartView pv = part_view(p);
    // after the segments' prefixes: the staged draw segment (16-byte aligned)
    uint4 *s_stage = pp.stage_vec ? reinterpret_cast<uint4 *>(s_pref_all + p.dec.nseg * TEAM) : nullptr;
    for (int item = blockIdx.x; item < pp.n_items; item += gridDim.x) {
        const DecGeom geo{item / p.dec.nseg, item % p.dec.nseg, p.dec.nseg, p.dec.seg_vec};
        decide_cta<DT, false, false, TEAM>(p, pv, geo, s_pref_all, s_stage, pp.stage_vec);
        dec_sync<TEAM>();   // the team's shared memory serves its next item
    }
}

// The streaming warps' rings, indexed by streaming warp: two stages each, as
// in the streaming kernel (three measured slower here too: 64.5 against 63.9
// us per round).
constexpr int kPipeStages = 2;
__host__ __device__ constexpr int pipe_rings(int team) { return ring_bytes(kPipeStages, kWarpsPerCta - team / 32); }

// DTN, DTP: the logits' types of next and prev (rounds of either type may
// follow one another); TEAM: the decide team, the first TEAM threads (next's
// streaming pass runs on the other warps: next.warp0 == TEAM / 32).
template <int DTN, int DTP, int TEAM>
__global__ void __launch_bounds__(kThreads, 1) pipe_kernel(const __grid_constant__ PipeParams pp) {
    extern __shared__ __align__(128) unsigned char smem[];
    // behind the previous launch on the stream (it streamed prev)
    griddep_wait();
    if (threadIdx.x < TEAM) {
        if (pp.has_prev) pipe_decide<DTP, TEAM>(pp, reinterpret_cast<float *>(smem + pipe_rings(TEAM)));
        return;
    }
    constexpr int kTeamWarps = TEAM / 32, kStreamWarps = kWarpsPerCta - kTeamWarps;
    const int warp = threadIdx.x >> 5;
    const int64_t gw = static_cast<int64_t>(blockIdx.x) * kStreamWarps + (warp - kTeamWarps);
    if (pp.has_next && gw < pp.next.W)
        scan_warp<DTN, false, kPipeStages>(pp.next, smem, gw, warp - kTeamWarps, kStreamWarps);
}

using PipeKernel = void (*)(PipeParams);
// [next is bf16][prev is bf16][team: kPipeTeam, kPipeTeamSmall]
const PipeKernel kPipeKernels[2][2][2] = {
    {{pipe_kernel<SDD_F32, SDD_F32, kPipeTeam>, pipe_kernel<SDD_F32, SDD_F32, kPipeTeamSmall>},
     {pipe_kernel<SDD_F32, SDD_BF16, kPipeTeam>, pipe_kernel<SDD_F32, SDD_BF16, kPipeTeamSmall>}},
    {{pipe_kernel<SDD_BF16, SDD_F32, kPipeTeam>, pipe_kernel<SDD_BF16, SDD_F32, kPipeTeamSmall>},
     {pipe_kernel<SDD_BF16, SDD_BF16, kPipeTeam>, pipe_kernel<SDD_BF16, SDD_BF16, kPipeTeamSmall>}}};

// The dynamic shared memory a pipelined launch may use on this device (the
// per-block opt-in limit less the kernels' static shared memory).
std::atomic<int> g_pipe_smem{0};

}  // namespace

cudaError_t pipe_prepare_device() {
    int dev = 0, optin = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    size_t stat = 0;
    for (const auto &plane : kPipeKernels)
        for (const auto &row : plane)
            for (PipeKernel k : row) {
                cudaFuncAttributes fa;
                if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, k);
                if (e == cudaSuccess) stat = std::max(stat, fa.sharedSizeBytes);
            }
    if (e != cudaSuccess) return e;
    const int dyn = optin - static_cast<int>(stat);
    for (const auto &plane : kPipeKernels)
        for (const auto &row : plane)
            for (PipeKernel k : row) {
                e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn);
                if (e != cudaSuccess) return e;
            }
    g_pipe_smem.store(dyn, std::memory_order_relaxed);
    return cudaSuccess;
}

// next: streamed on warps next->warp0..15 (next->warp0 = the decide team's
// warps: kPipeTeam / 32 or kPipeTeamSmall / 32); grid: next's streaming grid;
// prev (or null): decided by the team, prev->dec.nseg / seg_vec its blocks'
// draw segments over that grid for that team (one item per CTA while they
// fit).
cudaError_t launch_pipe(const ScanParams *next, const ScanParams *prev, int grid, cudaStream_t stream) {
    const int team = 32 * next->warp0;
    const int ti = (team == kPipeTeamSmall) ? 1 : 0;
    if (team != kPipeTeam && team != kPipeTeamSmall) return cudaErrorInvalidValue;
    PipeParams pp;
    std::memset(&pp, 0, sizeof pp);
    pp.next = *next;
    pp.has_next = 1;
    pp.next.wait_polls = kWaitPolls;
    size_t smem = static_cast<size_t>(ti ? pipe_rings(kPipeTeamSmall) : pipe_rings(kPipeTeam));
    if (prev) {
        pp.prev = *prev;
        pp.has_prev = 1;
        const bool draw = prev->dec.enabled && prev->dec.do_strict && !prev->dec.greedy;
        const int nseg = draw ? prev->dec.nseg : 1;
        pp.prev.dec.nseg = nseg;
        pp.n_items = prev->grp[0].nb * nseg;
        if (draw) {
            smem += static_cast<size_t>(nseg) * team * sizeof(float);
            // chunks of both draw rows' segments in the shared memory left
            // beside the rings (the whole segment when it fits)
            const size_t room = static_cast<size_t>(g_pipe_smem.load(std::memory_order_relaxed)) - smem;
            const int chunk = static_cast<int>(std::min<size_t>(prev->dec.seg_vec, room / 32));
            if (chunk >= team) {
                pp.stage_vec = chunk;
                smem += 2 * static_cast<size_t>(chunk) * 16;
            }
        }
    }
    if (grid <= 0) return cudaSuccess;
    const int dn = next->dtype == SDD_BF16, dp = (prev ? prev->dtype : next->dtype) == SDD_BF16;
    return launch_dependent(kPipeKernels[dn][dp][ti], dim3(grid), dim3(kThreads), smem, stream, pp);
}

}  // namespace sdd
