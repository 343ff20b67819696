/*
 * sdd.h -- C ABI of the GB300 (sm_103a) logits-side path of verifier-skipping
 * speculative diffusion decoding (Luo, Sandler, Fioretto, "From Positionwise
 * Confidence to Prefix Scheduling: Verifier Skipping in Speculative Decoding",
 * arXiv 2608.14787).
 *
 * The path has two halves around the verifier call of one decoding round:
 *   pre-verify   drafter logits -> per-position confidence -> committed prefix
 *                length K for each threshold pair (skip the verifier, or not);
 *   post-verify  target logits  -> accepted length L and committed tokens
 *                under Strict SDD, lenience or top-k acceptance.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * Pointers.  Unless a parameter says "host", every array pointer is DEVICE
 *   memory owned by the caller.  The library never allocates or frees memory,
 *   keeps no state between calls and may be called from several host threads.
 * Layout.  Logits are row-major [B, P, row_stride] with P = gamma drafter
 *   positions or gamma+1 target positions (the last target row serves the bonus
 *   token); element v of position j of batch row b sits at
 *   ((b * P) + j) * row_stride + v.  V <= row_stride is the vocabulary size.
 *   The base address must be 16-byte aligned and row_stride * element size a
 *   multiple of 16 bytes; the padding elements V..row_stride-1 are never read
 *   into any result.  Per-position arrays are [B, gamma] row-major, per-block
 *   arrays [B], threshold-grid outputs [n, B] (grid index outermost).
 * Streams.  Every call only enqueues work on `stream` (a cudaStream_t; NULL is
 *   the legacy default stream) and returns without synchronising.
 * Workspace.  Calls that take `workspace` need at least sdd_workspace_size()
 *   bytes of device memory for their (B, gamma, V), 256-byte aligned; it holds
 *   the streaming kernel's per-warp partial statistics and the sampling draw's
 *   per-segment prefix sums and arrival counters.  Its contents need no
 *   initialisation: every call writes what it reads and resets the arrival
 *   counters of its blocks before its draw, so one workspace serves any
 *   sequence of stream-ordered calls whose shapes it is large enough for (also
 *   after a call whose device status reports SDD_DEV_TIMEOUT).  Calls that may
 *   overlap on the GPU (different streams) need separate workspaces.
 * Errors.  The return value reports host-side problems only: invalid
 *   arguments are detected before anything is enqueued (SDD_ERR_INVALID_ARGUMENT)
 *   and launch failures return SDD_ERR_CUDA.  Conditions found while the
 *   kernels run are OR-ed into the caller's device word `*status` (bits
 *   SDD_DEV_*; the caller clears it); no kernel traps.  sdd_last_error()
 *   returns a message for the calling thread's last non-OK return;
 *   sdd_status_from_device() reads the device word into a return value.
 * Dtypes.  Logits are SDD_F32 or SDD_BF16; all arithmetic is fp32, with
 *   double-float (unevaluated fp32 pairs, about 48 significant bits) where sums,
 *   log-normalisers and threshold comparisons need more; fp64 results (lse) are
 *   converted from those pairs.
 * Kernels.  Each statistics, verification or block call enqueues the
 *   streaming kernel (one read of the logits) and then the decide kernel
 *   (row finalisation, decisions, draws) as a programmatic dependent launch.
 */
#ifndef SDD_H
#define SDD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define SDD_API __attribute__((visibility("default")))
#else
#define SDD_API
#endif

/* Same type as cudaStream_t. */
typedef struct CUstream_st *sdd_stream_t;

typedef enum {
    SDD_OK = 0,
    SDD_ERR_INVALID_ARGUMENT = 1,
    SDD_ERR_UNSUPPORTED = 2,
    SDD_ERR_CUDA = 3,
    SDD_ERR_WORKSPACE = 4,
    SDD_ERR_DEVICE = 5      /* sdd_status_from_device: a device status bit was set */
} sdd_status_t;

typedef enum { SDD_F32 = 0, SDD_BF16 = 1 } sdd_dtype_t;

/* Confidence signals of Sec. 4.2, and the confidence-free periodic skipping
 * baseline of the appendix (its parameters are a period per pair and a skip
 * length; see sdd_schedule_periodic). */
typedef enum { SDD_SIG_RAW = 0, SDD_SIG_MARGINAL = 1, SDD_SIG_CONDITIONAL = 2, SDD_SIG_PERIODIC = 3 } sdd_signal_t;

/* Bits of the device status word. */
#define SDD_DEV_NONFINITE 1u  /* a logits row held NaN or +inf, or only -inf      */
#define SDD_DEV_BAD_TOKEN 2u  /* a drafted token or row index was out of range   */
#define SDD_DEV_TIMEOUT 4u    /* a bounded wait on a tile copy gave up           */

/* Limits. */
#define SDD_MAX_GAMMA 128
#define SDD_MAX_GRID 32       /* threshold pairs, lenience values or k values per call */

/* ABI version (major * 10000 + minor * 100 + patch). */
SDD_API int sdd_version(void);

/* Message describing the calling thread's last non-OK return ("" if none). */
SDD_API const char *sdd_last_error(void);

/* The device status word `status` (int32 in device memory) of the calls
 * enqueued on `stream` so far, read once they complete (this call
 * synchronises the stream): *bits (host) receives its SDD_DEV_* bits.
 * Returns SDD_OK when no bit is set, SDD_ERR_DEVICE when one is (the message
 * of sdd_last_error() names them), SDD_ERR_CUDA if the read fails,
 * SDD_ERR_INVALID_ARGUMENT for a NULL pointer.  clear != 0 zeroes the word
 * after the read (stream-ordered, before this call returns). */
SDD_API sdd_status_t sdd_status_from_device(int32_t *status, int clear, uint32_t *bits, sdd_stream_t stream);

/*
 * sdd_workspace_size -- bytes of device scratch that any entry
 * point needs for blocks of this shape on the CURRENT device (the figure
 * depends on its SM count).  B, gamma, V as in the calls below.
 */
SDD_API sdd_status_t sdd_workspace_size(int B, int gamma, int V, size_t *bytes);

/*
 * sdd_confidence -- pre-verify statistics of the drafter rows (Sec. 4.2).
 * For each position (b, j), with z the drafter logits of that row and x_j the
 * drafted token:
 *   q       = p_draft(x_j) = exp(z(x_j) - LSE)      (raw confidence, Sec. 4.2)
 *   logq    = z(x_j) - LSE
 *   maxprob = max_v p(v)                            (top-1 probability, App. A.7)
 *   lse     = log sum_v exp(z(v)), in fp64 (the exact normaliser the sampling
 *             rule of sdd_verify_strict needs)
 *   entropy = -sum_v p(v) ln p(v), in nats          (App. A.7 feature)
 *   argmax  = lowest index attaining max_v z(v)
 * All outputs are [B, gamma]; every one but q may be NULL.  Finite logits
 * below -2^23 are treated as masked (-inf).  A row with NaN or
 * +inf logits, or only -inf, yields NaN statistics, argmax -1 and sets
 * SDD_DEV_NONFINITE; a drafted token outside [0, V) yields NaN q/logq and sets
 * SDD_DEV_BAD_TOKEN.  One streaming pass reads every logit exactly once.
 */
SDD_API sdd_status_t sdd_confidence(const void *draft_logits, sdd_dtype_t dtype, int B, int gamma, int V,
                            int64_t row_stride, const int32_t *draft_tokens, float *q, float *logq,
                            float *maxprob, double *lse, float *entropy, int32_t *argmax,
                            void *workspace, size_t workspace_bytes, int32_t *status,
                            sdd_stream_t stream);

/*
 * sdd_confidence_features -- sdd_confidence plus two more of the learned
 * scorer's pre-verification features (App. A.7) from the same single read of
 * the drafter logits: with p_(1) >= p_(2) >= ... the row's probabilities in
 * descending order (ties kept with multiplicity),
 *   margin[b, j] = p_(1) - p_(2)   (p_(2) = 0 when V = 1),
 *   top5[b, j]   = p_(1) + ... + p_(min(5, V))   (top-5 probability mass),
 * both fp32 [B, gamma], NaN for a row without a distribution (as q).  The
 * streaming pass additionally keeps each lane's five largest entries; the
 * other arguments, outputs and errors are those of sdd_confidence (margin and
 * top5 must not be NULL).
 */
SDD_API sdd_status_t sdd_confidence_features(const void *draft_logits, sdd_dtype_t dtype, int B, int gamma, int V,
                                             int64_t row_stride, const int32_t *draft_tokens, float *q,
                                             float *logq, float *maxprob, double *lse, float *entropy,
                                             int32_t *argmax, float *margin, float *top5, void *workspace,
                                             size_t workspace_bytes, int32_t *status, sdd_stream_t stream);

/*
 * sdd_schedule_prefix -- the skip policy of Sec. 4.1 for n_tau threshold pairs
 * (Eq. 3 and the commit rule that follows it).  For batch row b and pair t:
 *   B_k = min_{j<=k} q_j;  C_k = (prod q)^(1/k) (RAW), min_{j<=k} q_j (MARGINAL),
 *   prod_{j<=k} q_j (CONDITIONAL, computed in log space);
 *   K_hat = max{k : B_k >= eta_b[t], C_k >= eta_c[t], no guarded position in 1..k}
 *   (0 if none; for MARGINAL both gates use max(eta_b, eta_c)).
 *   If D_in[b] >= S_max the round is strict; otherwise it skips iff K_hat > 0 and
 *   K_hat >= K_min.  A skip writes K = K_hat and D_out = D_in + K; a strict round
 *   writes K = 0 and D_out = 0 (every verifier call resets D).
 * Readings fixed by this library: positions whose score is not finite count as
 * guarded (an invalid score); force_strict[b] != 0 (a shortened final block)
 * forces K_hat = K = 0; a pair with eta_b >= 1 or eta_c >= 1 disables skipping
 * (K_hat = K = 0), so the threshold limit reproduces Strict SDD exactly.
 *   q       [B, gamma] scores in [0, 1]: raw confidence from sdd_confidence, or
 *           the output of a learned survival scorer.
 *   logq    [B, gamma] natural log of q, or NULL (then log q is taken here).
 *   eta_b, eta_c  HOST arrays [n_tau], 1 <= n_tau <= SDD_MAX_GRID.
 *   guard   [B, gamma] uint8, nonzero = this position may not be skipped; NULL = none.
 *   force_strict [B] uint8 or NULL.  D_in [B] staleness counters (NULL = all 0).
 *   K_hat, K [n_tau, B]; D_out [n_tau, B] or NULL.
 */
SDD_API sdd_status_t sdd_schedule_prefix(const float *q, const float *logq, int B, int gamma,
                                 sdd_signal_t signal, const double *eta_b, const double *eta_c,
                                 int n_tau, int K_min, int S_max, const uint8_t *guard,
                                 const uint8_t *force_strict, const int32_t *D_in, int32_t *K_hat,
                                 int32_t *K, int32_t *D_out, int32_t *status, sdd_stream_t stream);

/*
 * sdd_schedule_periodic -- the confidence-free periodic skipping baseline (the
 * appendix's periodic-skipping paragraph and table): a skip of K_skip tokens is
 * attempted once every period[t] rounds, all other rounds are strict, and an
 * attempt meets the same guards as sdd_schedule_prefix.  For batch row b, pair t:
 *   attempt = (round mod period[t] == period[t] - 1)   (reading: period[t] - 1
 *             strict rounds precede each attempt; round counts from 0);
 *   K_hat   = attempt ? min(K_skip, gamma, first guarded position - 1) : 0
 *             (the prefix stops before a guarded position; force_strict[b]
 *             forces K_hat = 0);
 *   then the commit rule of sdd_schedule_prefix: D_in[b] >= S_max forces a
 *   strict round, otherwise the block skips iff K_hat > 0 and K_hat >= K_min
 *   (with K_min = K_skip a guarded prefix cancels the attempt).
 *   period  HOST [n_p], each >= 1, 1 <= n_p <= SDD_MAX_GRID.  K_skip >= 1.
 *   guard, force_strict, D_in, K_hat, K, D_out: as for sdd_schedule_prefix
 *   ([n_p, B] outputs).  No scores are read.
 */
SDD_API sdd_status_t sdd_schedule_periodic(int B, int gamma, const int32_t *period, int n_p, int K_skip,
                                           uint64_t round, int K_min, int S_max, const uint8_t *guard,
                                           const uint8_t *force_strict, const int32_t *D_in, int32_t *K_hat,
                                           int32_t *K, int32_t *D_out, int32_t *status, sdd_stream_t stream);

/*
 * Offline diagnostics over logged blocks: per block b its position scores
 * q[b, 0..gamma) (fp32, device) and its strict accepted length L[b] (int32,
 * device; from Strict SDD or the shadow verifier), j below 1-based.
 *
 * sdd_permutation_diagnostic -- the permutation test of Sec. 5 (H1 mechanism,
 * Table 1): n_rep times, at every position j the (score, label) pairs are
 * permuted across the blocks valid there -- all blocks for RAW and MARGINAL,
 * those with L >= j - 1 for CONDITIONAL -- which keeps every positionwise
 * distribution (so every positionwise metric) and breaks the association of
 * positions within a block; then the feasible prefix length of every block
 * is recomputed: K_hat of sdd_schedule_prefix for the pair (eta_b, eta_c)
 * before K_min or staleness.  Permutation r of position j is a Fisher-Yates
 * shuffle of the valid blocks in index order: slot i (from the top) swaps
 * with floor(w (i + 1) / 2^32), w the first word of Philox4x32-10 with key
 * seed and counter (i, j - 1, r, 3) (the map of sdd_uniforms, purpose 3).
 * Writes sums[r] = sum over blocks of the feasible prefix length under
 * permutation r (r < n_rep) and sums[n_rep] = that sum in the logged order
 * (int64, device); the means are sums / B.  Workspace: at least
 * sdd_permutation_workspace_size(B, gamma, n_rep) bytes (device).  B <= 50000.
 */
SDD_API sdd_status_t sdd_permutation_workspace_size(int B, int gamma, int n_rep, size_t *bytes);
SDD_API sdd_status_t sdd_permutation_diagnostic(const float *q, const int32_t *L, int B, int gamma,
                                                sdd_signal_t signal, double eta_b, double eta_c, int n_rep,
                                                uint64_t seed, int64_t *sums, void *workspace,
                                                size_t workspace_bytes, sdd_stream_t stream);

/*
 * sdd_position_metrics -- positionwise offline metrics (Sec. 5 H1, App. offline
 * metrics) of the scores against the labels y = 1{L >= j} at each position j,
 * over all blocks (conditional = 0: marginal survival, raw confidence) or the
 * blocks with L >= j - 1 (conditional != 0): for position j (index j - 1)
 *   bce[j]      = -mean(y ln q' + (1 - y) ln(1 - q')), q' = q clamped to [1e-7, 1 - 1e-7];
 *   bce_base[j] = the same for the position-only predictor (the positive rate
 *                 at j on these blocks): -(p ln p + (1 - p) ln(1 - p));
 *   auroc[j]    = (#{q_pos > q_neg} + #{q_pos = q_neg} / 2) / (n_pos n_neg),
 *                 NaN without positives or negatives;
 *   n_pos, n_neg [gamma] int32 (may be NULL).  bce, bce_base, auroc fp64 [gamma], device.
 */
SDD_API sdd_status_t sdd_position_metrics(const float *q, const int32_t *L, int B, int gamma, int conditional,
                                          double *bce, double *bce_base, double *auroc, int32_t *n_pos,
                                          int32_t *n_neg, sdd_stream_t stream);

/*
 * sdd_verify_strict -- Strict SDD verification (Sec. 3.1: the standard rule of
 * speculative decoding) of the blocks listed in rows[0..n_rows) (all B blocks
 * when rows is NULL; then n_rows must be B, or 0 for an empty list, which
 * enqueues nothing).
 *   greedy != 0 (the paper's runs, Sec. 5.1): accept x_j iff it is the lowest-
 *     index argmax of target row j; the token after the accepted prefix is the
 *     target argmax of row L+1 (row gamma+1 when all gamma are accepted).
 *   greedy == 0 (sampling): accept x_j iff u_j <= p_t(x_j) / p_d(x_j) with
 *     u_j = U(seed, j, b, round, 0); at the first rejection draw from
 *     norm(max(0, p_t - p_d)) of that row by inverse CDF in ascending token order
 *     with U(seed, L+1, b, round, 1) (from p_t when that residual has no mass);
 *     when all gamma are accepted draw the bonus token from p_t of row gamma+1
 *     with U(seed, gamma+1, b, round, 2).
 *   U(seed, j, b, round, purpose): Philox4x32-10 (Salmon et al., SC'11) with key
 *     (seed low, seed high 32 bits) and counter (j, b, round low 32,
 *     purpose | round high 32 << 8); u = ((word0 >> 8) | 1) * 2^-24.
 * Inputs: target_logits [B, gamma+1, row_stride]; draft_logits [B, gamma,
 *   row_stride] and draft_lse [B, gamma] (fp64, as written by sdd_confidence;
 *   both may be NULL when greedy != 0); draft_tokens [B, gamma].
 * Outputs, written only at the listed rows b: L [B] accepted length;
 *   tokens [B, gamma+1] = x_1..x_L, the drawn token, then -1; n_commit [B] = L+1.
 */
SDD_API sdd_status_t sdd_verify_strict(const void *target_logits, const void *draft_logits,
                               sdd_dtype_t dtype, int B, int gamma, int V, int64_t row_stride,
                               const int32_t *draft_tokens, const double *draft_lse, int greedy, uint64_t seed,
                               uint64_t round, const int32_t *rows, int n_rows, int32_t *L,
                               int32_t *tokens, int32_t *n_commit, void *workspace,
                               size_t workspace_bytes, int32_t *status, sdd_stream_t stream);

/*
 * sdd_select_rows -- the blocks a decode loop sends to the verifier (Sec. 4.1:
 * every block the skip policy did not skip): rows[0..n) = the indices b with
 * K[b] == 0 in ascending order, *n_rows = n (K [B], rows [B], n_rows: device).
 * With sdd_verify_strict_listed this keeps the verifier's row list on the
 * device, so that a loop round needs no host round trip.
 */
SDD_API sdd_status_t sdd_select_rows(const int32_t *K, int B, int32_t *rows, int32_t *n_rows, sdd_stream_t stream);

/*
 * sdd_verify_strict_listed -- sdd_verify_strict of the blocks rows[0..n) with
 * the count n read from device memory when the kernels run (*n_rows, at most
 * B; rows: device [B]), e.g. as written by sdd_select_rows on the same
 * stream.  The launch covers up to B blocks and the streaming pass splits
 * the listed blocks' target rows over the warps on the device.  Arguments and
 * outputs otherwise as sdd_verify_strict (draft_lse required for sampling).
 */
SDD_API sdd_status_t sdd_verify_strict_listed(const void *target_logits, const void *draft_logits,
                                              sdd_dtype_t dtype, int B, int gamma, int V, int64_t row_stride,
                                              const int32_t *draft_tokens, const double *draft_lse, int greedy,
                                              uint64_t seed, uint64_t round, const int32_t *rows,
                                              const int32_t *n_rows, int32_t *L, int32_t *tokens, int32_t *n_commit,
                                              void *workspace, size_t workspace_bytes, int32_t *status,
                                              sdd_stream_t stream);

/*
 * sdd_verify_lenient -- lenience acceptance (App. A.6 Eq. 9) for n_ell values in
 * one read of the target rows: accept x_j iff z_j(x_j) - max_v z_j(v) >= log ell,
 * except that ell = 1 uses the strict argmax comparison.  The longest accepted
 * prefix is committed, then the target argmax of the first rejected row (of
 * row gamma+1 when all are accepted).  ell: HOST array [n_ell] in the paper's
 * convention 0 < ell <= 1.  Outputs [n_ell, B], tokens [n_ell, B, gamma+1],
 * written only at the listed rows.
 */
SDD_API sdd_status_t sdd_verify_lenient(const void *target_logits, sdd_dtype_t dtype, int B, int gamma,
                                int V, int64_t row_stride, const int32_t *draft_tokens,
                                const double *ell, int n_ell, const int32_t *rows, int n_rows,
                                int32_t *L, int32_t *tokens, int32_t *n_commit, void *workspace,
                                size_t workspace_bytes, int32_t *status, sdd_stream_t stream);

/*
 * sdd_verify_topk -- top-k acceptance (App. A.6) for n_k values in one read of
 * the target rows: accept x_j iff it is among the k largest target logits of row
 * j, ranking ties by lower token index (so k = 1 is strict greedy).  Prefix and
 * correction/bonus as for lenience.  k: HOST array [n_k], 1 <= k <= 1024.
 */
SDD_API sdd_status_t sdd_verify_topk(const void *target_logits, sdd_dtype_t dtype, int B, int gamma, int V,
                             int64_t row_stride, const int32_t *draft_tokens, const int32_t *k,
                             int n_k, const int32_t *rows, int n_rows, int32_t *L, int32_t *tokens,
                             int32_t *n_commit, void *workspace, size_t workspace_bytes,
                             int32_t *status, sdd_stream_t stream);

/*
 * sdd_agreement -- accumulate the agreement counters of Sec. 3.2 for n_tau
 * schedules against the strict (shadow) accepted lengths L_strict [B]:
 * for each t, over the rows b with K[t, b] > 0 (the set A of Eq. 1-2),
 *   acc[t, 0] += min(K, L);  acc[t, 1] += K;  acc[t, 2] += (K <= L);  acc[t, 3] += 1.
 * StrictToken = acc[t,0] / acc[t,1] (Eq. 1); FullPrefix = acc[t,2] / acc[t,3] (Eq. 2).
 * acc: device int64 [n_tau, 4], added to (never cleared here).
 */
SDD_API sdd_status_t sdd_agreement(const int32_t *K, const int32_t *L_strict, int B, int n_tau,
                           int64_t *acc, sdd_stream_t stream);

/*
 * sdd_commit -- the tokens a round commits (Sec. 4.1): a skipped block (K[b] > 0)
 * commits x_1..x_K without a verifier call; any other block commits the verified
 * tokens.  K [B] (one schedule), draft_tokens [B, gamma], verified_tokens
 * [B, gamma+1] and verified_n [B] from a verify call.  Writes out_tokens
 * [B, gamma+1] (-1 padded) and out_n [B].
 */
SDD_API sdd_status_t sdd_commit(const int32_t *K, const int32_t *draft_tokens, const int32_t *verified_tokens,
                        const int32_t *verified_n, int B, int gamma, int32_t *out_tokens,
                        int32_t *out_n, sdd_stream_t stream);

/*
 * sdd_test_wait_hooks -- failure-detection test hooks (the paper has no
 * counterpart: they test the library's bounded device waits).  They apply to
 * the streaming kernel of every call this process enqueues afterwards, from
 * any thread, until changed:
 *   polls      the number of polls after which a wait for a tile copy gives
 *              up (each poll may suspend the warp briefly); 0 restores the
 *              default of 2^24 polls (seconds).  Copies still in flight when a
 *              warp gives up are always waited for with the default limit.
 *   drop_copy  nonzero: the first warp of each launch never issues its first
 *              tile copy, so its wait runs out -- the call returns normally,
 *              its device status gets SDD_DEV_TIMEOUT, its results are
 *              undefined, and the context, the workspace and later calls stay
 *              usable.  0: normal operation.
 * Returns SDD_OK.  Meant for tests; leave both at 0 in production.
 */
SDD_API sdd_status_t sdd_test_wait_hooks(uint32_t polls, int drop_copy);

/*
 * sdd_uniforms -- the uniforms U(seed, j, b, round, purpose) that the sampling
 * rule of sdd_verify_strict draws (Philox4x32-10 map stated there), for n
 * counters given as device arrays j, b, purpose [n] (uint32) and round [n]
 * (uint64).  Writes u [n] (fp32, exact).  Lets a caller reproduce or audit
 * the draws of a round.
 */
SDD_API sdd_status_t sdd_uniforms(uint64_t seed, const uint32_t *j, const uint32_t *b, const uint64_t *round,
                                  const uint32_t *purpose, int64_t n, float *u, sdd_stream_t stream);

/*
 * sdd_scorer_features -- the scalar-feature block of the learned scorer's input
 * (the feature list of App. A.7) for B*gamma drafter positions, in the column
 * order of that list:
 *   f [B*gamma, SDD_MLP_HIDDEN] bf16 (round to nearest even), row-major,
 *     16-byte aligned; every column is written: 4 top-1 probability (maxprob),
 *     5 its natural log, 6 entropy, 7 its negative, 8 probability margin,
 *     9 top-5 mass, 14 block position j / gamma, 15 generated length
 *     round / 256; every other column 0 (the paper's diffusion-model
 *     quantities -- reveal step and rank, parallelism, step-0 values -- have
 *     no counterpart here).
 *   maxprob, entropy, margin, top5 [B, gamma] fp32: the outputs of
 *     sdd_confidence_features.  round >= 0.
 * One launch.  The block is the f argument of sdd_scorer_deep.
 */
SDD_API sdd_status_t sdd_scorer_features(const float *maxprob, const float *entropy, const float *margin,
                                         const float *top5, int B, int gamma, int64_t round, void *f,
                                         sdd_stream_t stream);

/*
 * sdd_scorer_workspace_size -- bytes of device scratch that sdd_survival_mlp
 * and sdd_scorer_deep need for M positions (512 KiB per 128 positions: the
 * first layer's split-K partial accumulators, later the deep scorer's
 * second-layer activations).  No zero fill is needed; calls that may overlap
 * on the GPU need separate workspaces.
 */
SDD_API sdd_status_t sdd_scorer_workspace_size(int M, size_t *bytes);

/*
 * sdd_survival_mlp -- a learned-style survival score per draft position (the
 * form of the scorer of App. A.7 with one hidden layer; the decode-loop
 * workload uses it with random weights as a stand-in for the trained one):
 *   s[m] = sigmoid(w2 . GELU(W1 h[m] + b1) + b2),  GELU(z) = z Phi(z) (erf form),
 * for M positions (m = b * gamma + j).  The scores feed sdd_schedule_prefix as q
 * (the conditional survival signal of Sec. 4.2 treats them as per-position
 * survival probabilities).  The product W1 h runs on the tensor cores (bf16
 * inputs, fp32 accumulation).
 *   h   [M, K] bf16, row-major, 16-byte aligned (drafter hidden states);
 *       K a positive multiple of SDD_MLP_KSTEP.
 *   W1  [SDD_MLP_HIDDEN, K] bf16, row-major (one row per hidden unit), 16-byte aligned.
 *   b1  [SDD_MLP_HIDDEN] fp32; w2 [SDD_MLP_HIDDEN] bf16; b2 a host scalar.
 *   s   [M] fp32 output.
 *   workspace  device scratch of sdd_scorer_workspace_size(M) bytes, 16-byte
 *       aligned (SDD_ERR_INVALID_ARGUMENT if smaller).
 * One launch: 128-position tiles, K split over a cluster of up to four CTAs
 * whose partial products meet in the workspace.  Needs an sm_10x device
 * (returns SDD_ERR_UNSUPPORTED otherwise).  A bounded wait that gives up sets
 * SDD_DEV_TIMEOUT in *status (s is then undefined).
 */
#define SDD_MLP_HIDDEN 256
#define SDD_MLP_KSTEP 64
SDD_API sdd_status_t sdd_survival_mlp(const void *h, int M, int K, const void *W1, const float *b1, const void *w2,
                                      float b2, float *s, void *workspace, size_t workspace_bytes, int32_t *status,
                                      sdd_stream_t stream);

/*
 * sdd_scorer_deep -- the learned scorer's shape of App. A.7 (K -> 256 -> 256 ->
 * 256 -> 1, GELU hidden layers; dropout is a training-time op) per draft
 * position, with stand-in weights, on the concatenated input
 * x[m] = [h[m] ; f[m]] (drafter hidden state and scalar features):
 *   a1 = bf16(GELU(W1 x + b1)),  a2 = bf16(GELU(W2 a1 + b2)),
 *   s[m] = sigmoid(w4 . GELU(W3 a2 + b3) + b4).
 * a1 and a2 are rounded to bf16 (nearest even): the tensor cores take them as
 * bf16 operands (fp32 accumulation throughout).
 *   h    [M, Kh] bf16, row-major, 16-byte aligned; Kh a positive multiple of
 *        SDD_MLP_KSTEP (3584 in the paper).
 *   f    [M, SDD_MLP_HIDDEN] bf16: the scalar features in the first columns
 *        (19 in the paper), zeros after them.
 *   W1   [SDD_MLP_HIDDEN, Kh + SDD_MLP_HIDDEN] bf16 (columns Kh.. weigh f; the
 *        columns of f's zero padding should be zero too).
 *   W2, W3 [SDD_MLP_HIDDEN, SDD_MLP_HIDDEN] bf16 (one row per output unit);
 *   b1, b2, b3 [SDD_MLP_HIDDEN] fp32; w4 [SDD_MLP_HIDDEN] bf16; b4 a host scalar.
 *   act  [M, SDD_MLP_HIDDEN] bf16 caller scratch (receives a1), 16-byte aligned.
 *   s    [M] fp32 output.
 *   workspace  device scratch of sdd_scorer_workspace_size(M) bytes, 16-byte
 *        aligned (receives the first layer's partials, then a2).
 * Two launches on the stream: the first layer (K split over a 4-CTA cluster as
 * in sdd_survival_mlp), then layers 2 and 3 and the head, a 4-CTA cluster per
 * 128 positions (each CTA 64 of the 256 columns of both layers).  Needs an
 * sm_10x device; a bounded wait that gives up sets SDD_DEV_TIMEOUT in *status.
 */
SDD_API sdd_status_t sdd_scorer_deep(const void *h, int Kh, const void *f, int M, const void *W1, const float *b1,
                                     const void *W2, const float *b2, const void *W3, const float *b3,
                                     const void *w4, float b4, void *act, float *s, void *workspace,
                                     size_t workspace_bytes, int32_t *status, sdd_stream_t stream);

/*
 * sdd_confidence_noalloc -- sdd_confidence without a workspace, for callers
 * that cannot allocate device memory where they need the statistics: code
 * running inside CUDA stream capture (where cudaMalloc is not allowed),
 * programs whose device memory is a fixed arena owned by a framework, or host
 * loops that have no allocator at hand.  The paper has no counterpart; this is
 * a deployment convenience.
 * Same arguments, outputs, status bits and results as sdd_confidence, minus
 * the workspace.  The scratch is one file-scope device array of 384 KiB that
 * every GPU loading this library holds until the process exits; it serves
 * B * gamma <= 8192 drafter rows per call (larger batches are rejected with
 * SDD_ERR_INVALID_ARGUMENT before anything is enqueued).  The first call on a
 * device looks up the array's device address and the launch geometry for that
 * device (make that first call, on each device, before any stream capture).
 * Every call runs the same streaming and decide kernels as sdd_confidence.  All
 * calls share the one array, so
 * calls that may overlap on the GPU (different streams, or host threads without
 * ordering between them) race on it: order them on one stream.  No allocating
 * routine is called.
 */
SDD_API sdd_status_t sdd_confidence_noalloc(const void *draft_logits, sdd_dtype_t dtype, int B, int gamma, int V,
                                            int64_t row_stride, const int32_t *draft_tokens, float *q, float *logq,
                                            float *maxprob, double *lse, float *entropy, int32_t *argmax,
                                            int32_t *status, sdd_stream_t stream);

/*
 * sdd_block -- one round of the whole path over B blocks, fused so that every
 * drafter and target logit is read once: confidence (sdd_confidence), the skip
 * schedule for n_tau pairs (sdd_schedule_prefix), strict verification of every
 * block as the shadow verifier of Sec. 3.2 (sdd_verify_strict, sampling or
 * greedy), lenience for n_ell values and top-k for n_k values on the same target
 * read, agreement counters for every pair, and the tokens committed under pair
 * 0.  Array meanings and layouts are those of the single-purpose calls; NULL
 * output pointers are skipped.  sdd_block runs sdd_block_scan then
 * sdd_block_decide on the same stream, with the same args.  sdd_block_scan
 * streams every logit once into per-warp partial statistics (the workspace);
 * sdd_block_decide finalises every row, evaluates each block's rules,
 * schedule, agreement counters and commits, and draws the sampling rule's
 * residual / bonus tokens.  The two halves are exported so that a caller can
 * time the streaming pass alone; sdd_block_decide must follow the
 * sdd_block_scan of the same args on the same stream.
 */
typedef struct sdd_block_args {
    /* inputs */
    const void *draft_logits;      /* [B, gamma, row_stride]   */
    const void *target_logits;     /* [B, gamma+1, row_stride] */
    const int32_t *draft_tokens;   /* [B, gamma] */
    int32_t dtype;                 /* sdd_dtype_t */
    int32_t B, gamma, V;
    int64_t row_stride;
    /* schedule (Sec. 4.1) */
    int32_t signal;                /* sdd_signal_t */
    int32_t n_tau;                 /* 1..SDD_MAX_GRID */
    const double *eta_b;           /* HOST [n_tau] (not read for SDD_SIG_PERIODIC) */
    const double *eta_c;           /* HOST [n_tau] (not read for SDD_SIG_PERIODIC) */
    const int32_t *period;         /* HOST [n_tau], SDD_SIG_PERIODIC only (else NULL) */
    int32_t K_skip;                /* SDD_SIG_PERIODIC only */
    int32_t reserved1;
    int32_t K_min, S_max;
    const uint8_t *guard;          /* [B, gamma] or NULL */
    const uint8_t *force_strict;   /* [B] or NULL */
    const int32_t *D_in;           /* [B] or NULL */
    /* strict verification */
    int32_t greedy;
    int32_t reserved0;
    uint64_t seed, round;
    /* lenience / top-k grids */
    int32_t n_ell, n_k;            /* 0..SDD_MAX_GRID each */
    const double *ell;             /* HOST [n_ell], 0 < ell <= 1 */
    const int32_t *topk;           /* HOST [n_k] */
    /* outputs: confidence [B, gamma] (lse in fp64) */
    float *q, *logq, *maxprob;
    double *lse;
    float *entropy;
    int32_t *argmax;
    /* outputs: schedule [n_tau, B] */
    int32_t *K_hat, *K, *D_out;
    /* outputs: strict [B], [B, gamma+1], [B] */
    int32_t *L_strict, *tokens_strict, *n_strict;
    /* outputs: lenience [n_ell, B], [n_ell, B, gamma+1], [n_ell, B] */
    int32_t *L_lenient, *tokens_lenient, *n_lenient;
    /* outputs: top-k [n_k, B], [n_k, B, gamma+1], [n_k, B] */
    int32_t *L_topk, *tokens_topk, *n_topk;
    /* outputs: commit under pair 0: [B, gamma+1], [B] */
    int32_t *commit_tokens, *commit_n;
    /* agreement counters [n_tau, 4] (added to), or NULL */
    int64_t *agreement;
    /* scratch and status */
    void *workspace;
    size_t workspace_bytes;
    int32_t *status;
} sdd_block_args;

SDD_API sdd_status_t sdd_block(const sdd_block_args *args, sdd_stream_t stream);
SDD_API sdd_status_t sdd_block_scan(const sdd_block_args *args, sdd_stream_t stream);
SDD_API sdd_status_t sdd_block_decide(const sdd_block_args *args, sdd_stream_t stream);

/*
 * sdd_block_pipelined -- rounds of sdd_block over independent batches, two at
 * a time in one launch (no counterpart in the paper: it computes what
 * sdd_block computes, Sec. 3.1, 3.2 and 4.1, scheduled differently on the
 * GPU): the streaming pass of `next` and, on the same SMs,
 * the decide work (sdd_block_decide's) of `prev`, whose streaming pass ran
 * in the previous sdd_block_pipelined call on this stream.  The decide work
 * of a round is latency-bound (row finalisation, the rules, the sampling
 * draw); beside the next round's streaming pass it costs little of the
 * memory bandwidth, instead of leaving the memory system idle behind its own
 * pass.  A sequence of rounds r_0 .. r_n on one stream runs as
 *     sdd_block_pipelined(&r_0, NULL), sdd_block_pipelined(&r_1, &r_0), ...,
 *     sdd_block_pipelined(&r_n, &r_(n-1)), sdd_block_pipelined(NULL, &r_n);
 * the outputs of r_i are complete when the work of the call that names it as
 * prev has completed.
 *   next -- args as for sdd_block (NULL: decide prev only, the last call).
 *   prev -- the args that were `next` in the previous call on this stream,
 *           unchanged, with their inputs still in place (the draw reads two
 *           of its rows again) and its workspace untouched since (NULL: the
 *           first call).  Its streaming pass must have been made by this
 *           call: the pipelined pass divides the rows among warps
 *           differently from sdd_block_scan.
 * Rounds of more than 512 MiB of logits, whose decide work is a small part of
 * their time, run as sdd_block_scan (in the call that names them as next) and
 * sdd_block_decide (in the call that names them as prev) instead.
 * next and prev must use different workspaces and different output arrays.
 * Results are those of sdd_block on the same args: the same decisions and
 * tokens (outside the 1e-6 near-threshold band of the float comparisons) and
 * the same statistics up to rounding (the rows' pieces differ).
 * Errors: SDD_ERR_INVALID_ARGUMENT for both NULL, a shared workspace or any
 * error of sdd_block's arguments; as sdd_block otherwise.
 */
SDD_API sdd_status_t sdd_block_pipelined(const sdd_block_args *next, const sdd_block_args *prev,
                                         sdd_stream_t stream);

/*
 * Vocabulary-sharded round (a tensor-parallel LM head).  The paper runs its
 * verifier on one GPU and reads its logits in fp32 (App. A.8); when the
 * drafter's and verifier's logits are instead split by vocabulary over S
 * ranks -- rank s holding the contiguous slice [v0_s, v1_s) of every row,
 * slices in ascending order covering [0, V) -- the same round of sdd_block
 * runs as follows, with results identical to sdd_block's on the whole rows:
 *
 *   1. every rank: sdd_shard_partials on its slice -> one record per row;
 *   2. exchange: all-gather the records, [S][rows] in slice order;
 *   3. every rank: sdd_shard_decide -> all of sdd_block's outputs (identical
 *      on every rank), except, under strict sampling, the token drawn at the
 *      first rejection or the bonus row, left -1; plus this slice's masses
 *      of that draw row, [B][2] floats;
 *   4. (strict sampling) exchange: all-gather the masses, [S][B][2];
 *   5. (strict sampling) every rank: sdd_shard_draw -> the rank whose slice
 *      holds the draw writes the token into tokens_strict (and commit_tokens
 *      when the block is committed); the others write nothing;
 *   6. (strict sampling) exchange: element-wise MAX all-reduce of
 *      tokens_strict and commit_tokens (the missing entries are -1).
 *
 * A record: the slice's online-softmax state of the row with global indices,
 * the drafted token's logit when the token lies in the slice, and, for target
 * rows when the top-k rule runs, the slice's largest logits (value
 * descending, index ascending) -- the kcap largest of the whole row lie among
 * them, so the merged rank of the drafted token is exact up to kcap.  Records
 * are plain bytes: no pointers, the same on every rank.
 */
#define SDD_SHARD_KMAX 16

typedef struct sdd_shard_partial {
    float m;                      /* largest logit of the slice (floored at -2^23) */
    float r;                      /* integer reference of the sums, in log2 units */
    float t2;                     /* entropy accumulator relative to r (drafter rows) */
    float sh, sl;                 /* sum of 2^(z log2(e) - r) over the slice, as hi + lo */
    int32_t amax;                 /* global index of the slice's first largest logit */
    float g;                      /* the drafted token's logit if it lies in the slice */
    int32_t info;                 /* bit 0: token in the slice; bit 1: token outside [0, V);
                                     bits 8..15: number of candidates */
    float cz[SDD_SHARD_KMAX];     /* target rows: the slice's largest logits */
    int32_t cv[SDD_SHARD_KMAX];   /* their global indices */
} sdd_shard_partial;              /* 160 bytes */

/*
 * sdd_shard_workspace_size -- bytes of device scratch that sdd_shard_decide
 * leaves for sdd_shard_draw: per block the accepted length and the draw row's
 * log-normalisers (32 bytes), an arrival counter, and for up to 64 segments
 * of this slice's draw row their p_t masses and per-thread prefix sums
 * (256 floats each); about 66 KiB per block.  Zero-filled once before its
 * first use (every sdd_shard_decide leaves its counters at zero again);
 * 16-byte aligned.
 */
SDD_API sdd_status_t sdd_shard_workspace_size(int B, size_t *bytes);

/*
 * sdd_shard_partials -- step 1.  args as for sdd_block except: draft_logits
 * and target_logits hold this rank's slice, [B, gamma, row_stride] and
 * [B, gamma+1, row_stride] with columns 0..(v1-v0-1) = vocabulary entries
 * v0..v1-1 (v1 - v0 <= row_stride); V is the whole vocabulary; draft_tokens
 * are global indices; the top-k values (topk, n_k <= SDD_MAX_GRID) fix how
 * many candidates a record keeps (the largest k, at most SDD_SHARD_KMAX).
 * Only these fields and status are read.  out: [B*gamma + B*(gamma+1)]
 * records, drafter rows (b, j) at b*gamma + j, then target rows (b, j) at
 * B*gamma + b*(gamma+1) + j (device memory).
 */
SDD_API sdd_status_t sdd_shard_partials(const sdd_block_args *args, int v0, int v1, sdd_shard_partial *out,
                                        sdd_stream_t stream);

/*
 * sdd_shard_decide -- step 3.  args as for sdd_block (outputs included)
 * except: logits and V as for sdd_shard_partials, workspace = at least
 * sdd_shard_workspace_size(B) bytes.  all: [n_shards][rows] records of step
 * 2 (slice order); v0, v1 this rank's slice.  mass: [B][2] floats (device):
 * this slice's mass of each block's draw row (the residual max(0, p_t - p_d)
 * at the first rejection, or p_t of the bonus row; then p_t of that row),
 * written under strict sampling only.  n_shards <= 64.
 */
SDD_API sdd_status_t sdd_shard_decide(const sdd_block_args *args, int v0, int v1, int n_shards,
                                      const sdd_shard_partial *all, float *mass, sdd_stream_t stream);

/*
 * sdd_shard_draw -- step 5 (strict sampling only).  args, v0, v1, n_shards
 * as for sdd_shard_decide, the same workspace after it; shard: this rank's
 * index; mass_all: [n_shards][B][2] floats of step 4.  Locates, in slice order,
 * the slice holding u R of the inverse-CDF draw (R: the row's total mass) and,
 * on that slice's rank, the token, written at position L of tokens_strict and,
 * when the block is committed, of commit_tokens.
 */
SDD_API sdd_status_t sdd_shard_draw(const sdd_block_args *args, int v0, int v1, int n_shards, int shard,
                                    const float *mass_all, sdd_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* SDD_H */
