// internal.h -- launch parameters shared between the C-ABI layer (api.cu,
// noalloc.cu) and the kernels (scan.cu, decide.cu).  Not part of the public ABI.
#pragma once

#include <algorithm>
#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/sdd.h"
#include "common.cuh"

namespace sdd {

// Streaming pass geometry: each warp owns a private ring of kStages tiles of
// kVPL 16-byte vectors per lane, filled by 1D bulk copies.
constexpr int kWarpsPerCta = 16;
constexpr int kThreads = kWarpsPerCta * 32;
constexpr int kVPL = 8;                       // 16-byte vectors per lane per tile
constexpr int kTileVec = 32 * kVPL;           // vectors per warp tile
constexpr int kTileBytes = kTileVec * 16;     // 4 KiB
constexpr int kStages = 2;
// Shared memory of the rings of `warps` streaming warps with `stages` tiles each.
__host__ __device__ constexpr int ring_bytes(int stages, int warps) { return warps * stages * (kTileBytes + 8); }
constexpr int kScanSmem = ring_bytes(kStages, kWarpsPerCta);
constexpr uint32_t kWaitPolls = 1u << 24;     // bounded mbarrier wait (seconds of polling)

// Division by a per-launch constant d >= 1 without the 64-bit integer division
// routine (a called subroutine, slow on this part): floor(n / d) =
// umulhi(n, M) >> s with s = floor(log2 d) and M = ceil(2^(64+s) / d), exact for
// every 0 <= n < 2^53 (M d - 2^(64+s) < d <= 2^(s+1) <= 2^(64+s-53)); a power
// of two is a plain shift.  Built on the host (make_fastdiv).
struct FastDiv {
    uint64_t M;
    uint32_t s;
    uint32_t pow2;   // d = 2^s
};

inline FastDiv make_fastdiv(uint64_t d) {
    FastDiv f{0, 0, 0};
    while ((static_cast<uint64_t>(2) << f.s) <= d && f.s < 63) ++f.s;   // s = floor(log2 d)
    if ((d & (d - 1)) == 0) {
        f.pow2 = 1;
        return f;
    }
    const unsigned __int128 num = static_cast<unsigned __int128>(1) << (64 + f.s);
    f.M = static_cast<uint64_t>((num + d - 1) / d);
    return f;
}

// Decide kernel geometry: one CTA of kDecThreads per (listed block, draw
// segment); each draw segment is a run of whole 256-vector chunks of the draw
// row, at most kDrawMaxSeg per block (the last CTA of a block stages every
// segment's kDecThreads prefixes in shared memory: 1 KiB per segment).
constexpr int kDecThreads = 256;
constexpr int kDrawMaxSeg = 64;

// Vocabulary-sharded draw: what the decide kernel leaves, per block, for the
// draw that follows the exchange of the slices' draw-row masses (shard.cu).
struct ShardDraw {
    int32_t L;          // strict accepted length (the draw row is L, or gamma for the bonus row)
    int32_t commit;     // the block's verified tokens are committed (pair 0 did not skip it)
    float t_lh, t_ll;   // LSE of the target draw row (double-float)
    float d_lh, d_ll;   // LSE of the drafter draw row (residual only)
    int32_t pad[2];
};

// Per-block finalisation and decisions (decide.cu, rules.cuh).  Thresholds
// are double-floats split on the host from their fp64 values.
struct DecideParams {
    int32_t enabled;               // evaluate block decisions after finalising the rows
    int32_t B, gamma, V;
    int64_t stride_bytes;
    const char *zt, *zd;           // target / drafter logits (draw rows, stand-alone acceptance)
    const int32_t *tokens;         // [B, gamma]
    const double *d_lse;           // [B, gamma] drafter LSE (user array) when no drafter rows are streamed
    // strict
    int32_t do_strict, greedy;
    uint64_t seed, round;
    int32_t *L_strict, *tok_strict, *n_strict;
    // lenience
    int32_t n_ell;
    int32_t ell_one[SDD_MAX_GRID];
    df ell_thr[SDD_MAX_GRID];      // ln(ell)
    int32_t *L_len, *tok_len, *n_len;
    // top-k
    int32_t n_k;
    int32_t kval[SDD_MAX_GRID];
    int32_t *L_topk, *tok_topk, *n_topk;
    // schedule (fused round)
    int32_t do_sched, signal, n_tau, K_min, S_max;
    int32_t period[SDD_MAX_GRID], K_skip;   // SDD_SIG_PERIODIC
    int32_t tau_off[SDD_MAX_GRID];
    df eta_loc[SDD_MAX_GRID];
    df log_eta_c[SDD_MAX_GRID];
    const uint8_t *guard, *force_strict;
    const int32_t *D_in;
    int32_t *K_hat, *K, *D_out;
    int32_t *commit_tokens, *commit_n;
    long long *agreement;
    // sampling draw (residual / bonus inverse CDF), workspace
    int32_t nseg, seg_vec;         // segments per block and vectors per segment
    int32_t dec_ctas;              // decide CTAs resident at once (the draw's one-wave budget)
    float *res_pref;               // [nb, nseg, kDecThreads] per-thread inclusive prefix sums
    uint32_t *res_count;           // [nb] (zero between calls)
    // vocabulary-sharded decide: this slice's draw-row masses [B][2] (residual
    // or bonus weights, then p_t weights) and the per-block draw state
    float *shard_mass;
    ShardDraw *shard_state;
    float *shard_ptot;             // [B][kDrawMaxSeg] each draw segment's p_t mass (this slice)
};

// One set of rows streamed by the scan kernel (drafter rows or target rows).
// Both groups of a launch list the same blocks in the same order.
struct ScanGroup {
    const char *base;        // logits [B, npos, row_stride]
    int64_t stride_bytes;    // row_stride * element size
    int32_t npos;            // rows per block: gamma (drafter) or gamma+1 (target)
    int32_t kind;            // 0 = drafter (entropy), 1 = target (rank)
    int32_t nb;              // blocks in this group (after compaction)
    int32_t pad;
    const int32_t *bidx;     // [nb] batch index of each listed block, or nullptr (= identity)
    // drafter user outputs, indexed (b * gamma + j); any may be nullptr
    float *q, *logq, *maxprob, *entropy;
    double *lse;
    int32_t *argmax;
    float *margin, *top5;    // extended features (only with ScanParams::feat)
};

struct ScanParams {
    ScanGroup grp[2];
    int32_t n_groups;
    int32_t dtype;           // SDD_F32 / SDD_BF16
    int32_t V;
    int32_t RV;              // 16-byte vectors per row (ceil)
    int32_t gamma;
    int32_t kcap;            // rank saturation (>= 1)
    int32_t B;
    int32_t W;               // active warps
    int64_t rows0;           // rows of group 0
    int64_t rows;            // rows of all groups
    int64_t T;               // total vectors = rows * RV
    // Cost-balanced partition: a vector of a group-g row costs wt[g] units
    // (drafter rows carry the entropy work), and the first vector of every row
    // R more (a piece's end and the next piece's start); P[g] = wt[g] RV + R is
    // a whole row's cost; T0 = rows0 * RV, C = total cost.
    int32_t wt[2];
    int64_t R, P[2];
    int64_t T0, C;
    FastDiv divC, divW, divRV, divNpos[2], divWt[2], divP[2];   // division by C, W, RV, grp[g].npos, wt[g], P[g]
    // The streaming warps of a CTA: warps warp0 .. warp0 + wpc - 1, global
    // streaming warp blockIdx.x * wpc + (warp - warp0) (set_divisors: all 16;
    // the pipelined round: warps kPipeWarps-15, the others run the previous
    // round's decide work).
    int32_t warp0, wpc;
    const int32_t *tokens;   // [B, gamma]
    // When set, the number of listed blocks is read from this device word at
    // launch (at most grp[g].nb, which then sizes the grid): rows, T, T0, C
    // and the active warps follow from it on the device (PartView).
    const int32_t *nb_dev;
    Partial *partials;       // [rows + W]
    FeatPartial *feat;       // [rows + W], or nullptr: no extended features
    int32_t *status;
    // vocabulary-sharded decide: the S slices' records [S][rows] replace the
    // warp partials; V and RV then describe this rank's slice
    const sdd_shard_partial *shard;
    int32_t n_shards;
    int32_t shard_v0;        // first vocabulary index of this rank's slice
    int64_t shard_rows;      // records per slice (B * (2 gamma + 1))
    uint32_t wait_polls;     // polls of a ring wait before the warp gives up (set at launch)
    int32_t drop_copy;       // failure-detection test hook: warp 0 never issues its first copy
    DecideParams dec;
};

struct ScheduleParams {
    const float *q, *logq;
    int32_t B, gamma, signal, n_tau, K_min, S_max;
    int32_t period[SDD_MAX_GRID], K_skip;   // SDD_SIG_PERIODIC
    uint64_t round;
    int32_t tau_off[SDD_MAX_GRID];
    df eta_loc[SDD_MAX_GRID];
    df log_eta_c[SDD_MAX_GRID];
    const uint8_t *guard, *force_strict;
    const int32_t *D_in;
    int32_t *K_hat, *K, *D_out;
};

// The streaming kernel (grid = warps / kWarpsPerCta CTAs).
cudaError_t launch_scan(const ScanParams &p, int grid, cudaStream_t stream);
// Failure-detection test hooks of the streaming kernel, read at each launch:
// the ring waits' poll limit (0 = kWaitPolls) and the dropped first copy.
void set_scan_wait_hooks(uint32_t polls, int drop_copy);
// The decide kernel over (listed blocks, p.dec.nseg) CTAs, launched as a
// programmatic dependent of the streaming kernel.
cudaError_t launch_decide(const ScanParams &p, cudaStream_t stream);
// The pipelined round (pipe.cu): next's streaming pass over `grid` CTAs and,
// on the first next->warp0 warps of the same CTAs, prev's decide work (prev
// may be null).
cudaError_t launch_pipe(const ScanParams *next, const ScanParams *prev, int grid, cudaStream_t stream);
cudaError_t launch_schedule(const ScheduleParams &p, cudaStream_t stream);
// Vocabulary-sharded path (shard.cu): the slice's per-row records, and the
// draw once every slice's draw-row mass is known.
struct ShardParams {
    const char *zd, *zt;     // this slice of the drafter [B, gamma, .] and target [B, gamma+1, .] logits
    int64_t stride_bytes;
    int32_t dtype, B, gamma;
    int32_t Vs, RVs;         // slice width and its 16-byte vectors
    int32_t v0, V;           // first index of the slice, full vocabulary
    int32_t kcap;            // candidates kept per target row (0: none)
    const int32_t *tokens;   // [B, gamma]
    sdd_shard_partial *out;  // [B gamma + B (gamma + 1)]
    int32_t *status;
    // draw
    int32_t n_shards, shard;
    const float *mass_all;   // [n_shards][B][2]
    const ShardDraw *state;  // [B]
    const float *res_pref;   // [B][kDrawMaxSeg][kDecThreads] the decide's per-thread prefixes of the draw row
    int32_t nseg, seg_vec;   // its segments of the slice's draw row
    uint64_t seed, round;
    int32_t *tok_strict, *commit_tokens;
};
cudaError_t launch_shard_partials(const ShardParams &sp, cudaStream_t stream);
cudaError_t launch_shard_draw(const ShardParams &sp, cudaStream_t stream);
cudaError_t launch_agreement(const int32_t *K, const int32_t *L, int B, int n_tau, long long *acc,
                             cudaStream_t stream);
// The batch indices b with K[b] == 0, ascending, and their count (one CTA).
cudaError_t launch_select_rows(const int32_t *K, int B, int32_t *rows, int32_t *n_rows, cudaStream_t stream);
cudaError_t launch_commit(const int32_t *K, const int32_t *x, const int32_t *vt, const int32_t *vn, int B,
                          int gamma, int32_t *out_t, int32_t *out_n, cudaStream_t stream);
cudaError_t launch_uniforms(uint64_t seed, const uint32_t *j, const uint32_t *b, const uint64_t *round,
                            const uint32_t *purpose, int64_t n, float *u, cudaStream_t stream);
// Relative per-vector cost of streaming a drafter row (online softmax plus
// the entropy accumulator) and a target row (online softmax plus the rank
// count), measured on GB300: 10 : 9.
constexpr int32_t kCostDrafter = 10, kCostTarget = 9;
// Extra cost of a row's first vector, in vectors of the heavier group: the
// end of a warp's piece of a row (exact argmax re-read, reduction, partial)
// and the next piece's start.  Per-warp globaltimer stamps (one 16-block
// round): warps whose range crosses a row boundary ended 3.2 us after those
// whose range does not.  Measured on GB300 (16-block round, back to back):
// 0 -> 69.08 us, 200 -> 68.68, 400 -> 68.62, 700 -> 69.21.
constexpr int64_t kRowStartVec = 400;

// Warps of a launch over T vectors in `rows` rows with at most W_max warps:
// at least two vectors per warp, so that with the cost weights every warp's
// share of the cost holds at least one vector start (no empty warp inside a
// row), and at most kPiecesPerRow warps per row on average, so that the
// decide kernel merges few partials per row.  The cap binds only for small
// calls (one block of 32 rows: 16 instead of ~37 pieces per row): measured
// on GB300, a one-block round at V = 151,936 took 31.5 instead of 34.5 us
// and the 8 x 32,000 fp32 block 27.9 instead of 68 us (cap 8: 35.8 / 26.6;
// cap 32: 33.4 / 32.1); the 16-block round is unchanged.
constexpr int64_t kPiecesPerRow = 16;
__host__ __device__ inline int32_t scan_warps(int64_t W_max, int64_t T, int64_t rows) {
    int64_t w = W_max < T / 2 ? W_max : T / 2;
    if (w > rows * kPiecesPerRow) w = rows * kPiecesPerRow;
    return static_cast<int32_t>(w > 1 ? w : 1);
}

// The pipelined round (sdd_block_pipelined): the first warps of every CTA (a
// team of 64 threads, or 128 after a round of at most kPipeSmallBytes of
// logits) run the previous round's decide work while the others stream.  A
// round that small is latency-bound: its decide items are few and each takes
// longer than its streaming pass (GB300, one 32 x 151,936 bf16 block: 23.8
// us per round with a 128-thread team, 27.9 us with 64; one 8 x 32,000 fp32
// block: 22.8 / 24.2 us), while at 16 blocks the two more streaming warps
// win (61.2 against 63.5 us).
constexpr int kPipeTeam = 64, kPipeTeamSmall = 128;
constexpr int64_t kPipeSmallBytes = int64_t(64) << 20;
// The pipelined pass's cost weights (drafter, target vector), as kCostDrafter
// and kCostTarget for the streaming kernel: on fourteen warps beside the
// decide work the drafter rows' entropy work weighs more (GB300, 16-block
// round: 10 : 9 62.3 us, 21 : 18 61.2, 11 : 9 61.5, 23 : 18 62.2, 12 : 9 63.5;
// with 10 : 9 the CTAs streaming drafter rows ended ~2.5 us after the others).
constexpr int32_t kPipeCostDrafter = 21, kPipeCostTarget = 18;

// The cost weights and division constants of a launch whose groups, rows, T
// and W are set (host), all 16 warps of a CTA streaming.  The magic divisions
// are exact while C * W < 2^53 (the callers check it).
inline void set_divisors(ScanParams &p, int32_t cost_drafter = kCostDrafter, int32_t cost_target = kCostTarget) {
    const bool mixed = p.n_groups == 2 && p.grp[0].kind != p.grp[1].kind;
    for (int g = 0; g < 2; ++g) p.wt[g] = mixed ? (p.grp[g].kind == 0 ? cost_drafter : cost_target) : 1;
    const int64_t wmax = std::max(p.wt[0], p.wt[1]), wmin = std::min(p.wt[0], p.wt[1]);
    // The row-start cost must leave every warp at least one vector start: a
    // warp's share of the cost, at least a row's cost over kPiecesPerRow
    // (scan_warps; also for a smaller device block count), has to exceed the
    // largest single vector's cost R + wmax: wmin RV + R >= kPiecesPerRow
    // (R + 2 wmax).  Rows too short for that (and too short to be cut at all)
    // get no row-start cost.
    int64_t R = kRowStartVec * wmax;
    if (p.RV < 2 * kPiecesPerRow || wmin * p.RV + R < kPiecesPerRow * (R + 2 * wmax)) R = 0;
    p.R = R;
    for (int g = 0; g < 2; ++g) p.P[g] = p.wt[g] * p.RV + R;
    p.T0 = p.rows0 * p.RV;
    p.C = p.rows0 * p.P[0] + (p.rows - p.rows0) * p.P[1];
    p.divC = make_fastdiv(static_cast<uint64_t>(p.C > 0 ? p.C : 1));
    for (int g = 0; g < 2; ++g) p.divWt[g] = make_fastdiv(static_cast<uint64_t>(p.wt[g]));
    for (int g = 0; g < 2; ++g) p.divP[g] = make_fastdiv(static_cast<uint64_t>(p.P[g] > 0 ? p.P[g] : 1));
    p.divW = make_fastdiv(static_cast<uint64_t>(p.W > 0 ? p.W : 1));
    p.divRV = make_fastdiv(static_cast<uint64_t>(p.RV > 0 ? p.RV : 1));
    for (int g = 0; g < 2; ++g) p.divNpos[g] = make_fastdiv(static_cast<uint64_t>(p.grp[g].npos > 0 ? p.grp[g].npos : 1));
    p.warp0 = 0;
    p.wpc = kWarpsPerCta;
}

// Offline diagnostics (diag.cu).  perm: [n_rep, gamma, B] int32 scratch;
// sums: [n_rep + 1] feasible-prefix sums (the last: the logged order).
cudaError_t launch_perm_diag(const float *q, const int32_t *L, int B, int gamma, int signal, df eta_loc,
                             df log_eta_c, int n_rep, uint64_t seed, float *pq, unsigned long long *sums,
                             cudaStream_t stream);
cudaError_t launch_position_metrics(const float *q, const int32_t *L, int B, int gamma, int conditional, double *bce,
                                    double *bce_base, double *auroc, int32_t *n_pos, int32_t *n_neg,
                                    cudaStream_t stream);

// The learned scorer's scalar-feature block (mlp.cu), bf16 [M, 256].
cudaError_t launch_scorer_features(const float *maxprob, const float *entropy, const float *margin, const float *top5,
                                   int64_t M, int gamma, float gen, uint16_t *f, cudaStream_t stream);
// Device scratch of the scorers (mlp.cu) for M rows: the split-K partials of
// the first layer, later the deep scorer's second-layer activations.
size_t mlp_workspace_bytes(int M);
// The stand-in survival scorer (mlp.cu); *why names a host-side failure.
cudaError_t launch_mlp(const void *h, int M, int K, const void *W1, const float *b1, const void *w2, float b2,
                       float *out, void *ws, int32_t *status, cudaStream_t stream, const char **why);
// The deep scorer (mlp.cu): layer 1 over [h | f] into act, then layers 2, 3 and the head.
cudaError_t launch_scorer_deep(const void *h, int Kh, const void *f, int M, const void *W1, const float *b1,
                               const void *W2, const float *b2, const void *W3, const float *b3, const void *w4,
                               float b4, uint16_t *act, float *out, void *ws, int32_t *status,
                               cudaStream_t stream, const char **why);
int scan_max_ctas_per_sm();
int decide_max_ctas_per_sm();
cudaError_t scan_prepare_device();
cudaError_t decide_prepare_device();
cudaError_t pipe_prepare_device();
void set_last_error(const char *msg);  // message returned by sdd_last_error()

__device__ __forceinline__ int64_t fast_div(int64_t n, const FastDiv &f) {
    const uint64_t u = static_cast<uint64_t>(n);
    return static_cast<int64_t>(f.pow2 ? (u >> f.s) : (__umul64hi(u, f.M) >> f.s));
}

// make_fastdiv on the device (a 128-bit division, once per warp).
__device__ __forceinline__ FastDiv make_fastdiv_dev(uint64_t d) {
    FastDiv f{0, 63u - static_cast<uint32_t>(__clzll(static_cast<long long>(d))), 0};
    if ((d & (d - 1)) == 0) {
        f.pow2 = 1;
        return f;
    }
    const unsigned __int128 num = static_cast<unsigned __int128>(1) << (64 + f.s);
    f.M = static_cast<uint64_t>((num + d - 1) / d);
    return f;
}

// The launch's partition: from the parameters, or -- with a device block
// count -- computed on the device the way the host computes it.
struct PartView {
    int64_t nb, rows0, rows, T, T0, C;
    int32_t W;
    FastDiv divC, divW;
};

__device__ __forceinline__ PartView part_view(const ScanParams &p) {
    PartView v;
    if (p.nb_dev == nullptr) {
        v.nb = p.grp[0].nb;
        v.rows0 = p.rows0;
        v.rows = p.rows;
        v.T = p.T;
        v.T0 = p.T0;
        v.C = p.C;
        v.W = p.W;
        v.divC = p.divC;
        v.divW = p.divW;
        return v;
    }
    v.nb = min(max(static_cast<int64_t>(*p.nb_dev), static_cast<int64_t>(0)), static_cast<int64_t>(p.grp[0].nb));
    v.rows0 = v.nb * p.grp[0].npos;
    v.rows = v.rows0 + (p.n_groups > 1 ? v.nb * p.grp[1].npos : 0);
    v.T = v.rows * p.RV;
    v.T0 = v.rows0 * p.RV;
    v.C = v.rows0 * p.P[0] + (v.rows - v.rows0) * p.P[1];
    v.W = scan_warps(p.W, v.T, v.rows);
    v.divC = make_fastdiv_dev(static_cast<uint64_t>(v.C > 0 ? v.C : 1));
    v.divW = make_fastdiv_dev(static_cast<uint64_t>(v.W));
    return v;
}

// Index arithmetic of the cost-balanced contiguous partition of the T
// vectors over W warps.  Vector v occupies the cost interval [cost(v),
// cost(v+1)): a group-g vector costs wt[g] and a row's first vector R more,
// so cost(v) = (whole rows before v's row) + (R + k wt[g] for the k >= 1
// vectors of v's row before it, 0 for k = 0), rows of group 0 first.  Warp w
// owns the costs [floor(w C / W), floor((w+1) C / W)) and so the vectors whose
// cost interval starts there: [start(w), start(w+1)) with start(w) the first
// vector of cost >= floor(w C / W).  Requires C W < 2^53 (checked by the host).
__device__ __forceinline__ int64_t part_start(const ScanParams &p, const PartView &v, int64_t w) {
    const int64_t c = fast_div(w * v.C, v.divW);
    const int64_t c0 = v.rows0 * p.P[0];   // the cost of group 0
    const int g = (c <= c0) ? 0 : 1;
    const int64_t cg = g ? c - c0 : c;
    const int64_t r = fast_div(cg, p.divP[g]);   // whole rows of the group before it
    const int64_t rem = cg - r * p.P[g];
    int64_t k = 0;
    if (rem > 0) k = (rem <= p.R) ? 1 : fast_div(rem - p.R + p.wt[g] - 1, p.divWt[g]);
    return (g ? v.T0 : 0) + r * p.RV + k;
}
// The warp owning vector v.
__device__ __forceinline__ int64_t part_owner(const ScanParams &p, const PartView &pv, int64_t v) {
    const int g = (v < pv.T0) ? 0 : 1;
    const int64_t u = g ? v - pv.T0 : v;
    const int64_t r = fast_div(u, p.divRV);
    const int64_t k = u - r * p.RV;
    const int64_t cost = (g ? pv.rows0 * p.P[0] : 0) + r * p.P[g] + (k > 0 ? p.R + k * p.wt[g] : 0);
    return fast_div((cost + 1) * pv.W - 1, pv.divC);
}

}  // namespace sdd
