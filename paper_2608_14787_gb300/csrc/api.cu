// api.cu -- the C ABI declared in include/sdd.h: argument checks, workspace
// layout and kernel launches.  Every check that can fail runs before anything
// is enqueued; nothing here allocates device memory.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>

#include "internal.h"

namespace sdd {
namespace {

thread_local std::string g_err;

sdd_status_t fail(sdd_status_t s, const char *fmt, ...) __attribute__((format(printf, 2, 3)));
sdd_status_t fail(sdd_status_t s, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_err = buf;
    return s;
}

sdd_status_t cuda_fail(cudaError_t e, const char *what) {
    return fail(SDD_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

// Per-device launch facts, filled on first use (benign race: same values).
constexpr int kMaxDevices = 64;
struct DevInfo {
    int sms;
    int ctas_per_sm;        // streaming kernel
    int dec_ctas_per_sm;    // decide kernel
};
DevInfo g_dev[kMaxDevices];
std::atomic<int> g_dev_ready[kMaxDevices];

sdd_status_t device_info(DevInfo &out) {
    int d = 0;
    cudaError_t e = cudaGetDevice(&d);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (d < 0 || d >= kMaxDevices) return fail(SDD_ERR_UNSUPPORTED, "device ordinal %d out of range", d);
    if (!g_dev_ready[d].load(std::memory_order_acquire)) {
        DevInfo di{};
        e = cudaDeviceGetAttribute(&di.sms, cudaDevAttrMultiProcessorCount, d);
        if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
        e = scan_prepare_device();
        if (e == cudaSuccess) e = decide_prepare_device();
        if (e == cudaSuccess) e = pipe_prepare_device();
        if (e != cudaSuccess) return cuda_fail(e, "cudaFuncSetAttribute");
        di.ctas_per_sm = scan_max_ctas_per_sm();
        if (di.ctas_per_sm < 1) return fail(SDD_ERR_UNSUPPORTED, "streaming kernel does not fit on this device");
        di.dec_ctas_per_sm = decide_max_ctas_per_sm();
        if (di.dec_ctas_per_sm < 1) return fail(SDD_ERR_UNSUPPORTED, "decide kernel does not fit on this device");
        g_dev[d] = di;
        g_dev_ready[d].store(1, std::memory_order_release);
    }
    out = g_dev[d];
    return SDD_OK;
}

inline size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

// Workspace layout for blocks of shape (B, gamma) on a device with W_max warps.
struct Layout {
    size_t partials, feat, res_pref, res_count, total;
};

Layout layout(int64_t B, int64_t gamma, int64_t W_max, int64_t dec_ctas) {
    Layout L{};
    const int64_t rows = B * (2 * gamma + 1);
    size_t o = 0;
    auto take = [&](size_t bytes) {
        const size_t at = o;
        o = align256(o + bytes);
        return at;
    };
    L.partials = take(static_cast<size_t>(rows + W_max) * sizeof(Partial));
    L.feat = take(static_cast<size_t>(rows + W_max) * sizeof(FeatPartial));
    // nb * nseg <= max(resident decide CTAs, B) (see init_dec)
    L.res_pref = take(static_cast<size_t>(std::max(dec_ctas, B)) * kDecThreads * sizeof(float));
    L.res_count = take(static_cast<size_t>(B) * sizeof(uint32_t));
    L.total = o;
    return L;
}

int esize(int dtype) { return dtype == SDD_BF16 ? 2 : 4; }

sdd_status_t check_shape(sdd_dtype_t dtype, int B, int gamma, int V, int64_t row_stride) {
    if (dtype != SDD_F32 && dtype != SDD_BF16) return fail(SDD_ERR_INVALID_ARGUMENT, "dtype %d unknown", dtype);
    if (B < 0) return fail(SDD_ERR_INVALID_ARGUMENT, "B = %d < 0", B);
    if (gamma < 1 || gamma > SDD_MAX_GAMMA)
        return fail(SDD_ERR_INVALID_ARGUMENT, "gamma = %d outside [1, %d]", gamma, SDD_MAX_GAMMA);
    if (V < 1) return fail(SDD_ERR_INVALID_ARGUMENT, "V = %d < 1", V);
    if (row_stride < V) return fail(SDD_ERR_INVALID_ARGUMENT, "row_stride %lld < V %d", (long long)row_stride, V);
    if ((row_stride * esize(dtype)) % 16 != 0)
        return fail(SDD_ERR_INVALID_ARGUMENT, "row_stride * element size must be a multiple of 16 bytes");
    if (row_stride * esize(dtype) > (int64_t(1) << 31))
        return fail(SDD_ERR_INVALID_ARGUMENT, "rows longer than 2 GiB are not supported");
    return SDD_OK;
}

sdd_status_t check_ptr16(const void *p, const char *name) {
    if (!p) return fail(SDD_ERR_INVALID_ARGUMENT, "%s is NULL", name);
    if (reinterpret_cast<uintptr_t>(p) % 16 != 0) return fail(SDD_ERR_INVALID_ARGUMENT, "%s is not 16-byte aligned", name);
    return SDD_OK;
}

struct Work {
    char *base;
    Layout L;
    int W_max;
    int sms;
    int dec_ctas;   // decide-kernel CTAs resident at once on the device
};

sdd_status_t get_work(void *workspace, size_t bytes, int B, int gamma, Work &w) {
    DevInfo di;
    sdd_status_t s = device_info(di);
    if (s != SDD_OK) return s;
    w.W_max = di.sms * di.ctas_per_sm * kWarpsPerCta;
    w.sms = di.sms;
    w.dec_ctas = di.sms * di.dec_ctas_per_sm;
    w.L = layout(B, gamma, w.W_max, w.dec_ctas);
    if (!workspace) return fail(SDD_ERR_WORKSPACE, "workspace is NULL");
    if (reinterpret_cast<uintptr_t>(workspace) % 256 != 0)
        return fail(SDD_ERR_WORKSPACE, "workspace is not 256-byte aligned");
    if (bytes < w.L.total)
        return fail(SDD_ERR_WORKSPACE, "workspace has %zu bytes, %zu needed", bytes, w.L.total);
    w.base = static_cast<char *>(workspace);
    return SDD_OK;
}

void init_scan(ScanParams &p, const Work &w, sdd_dtype_t dtype, int B, int gamma, int V, const int32_t *tokens,
               int32_t *status) {
    std::memset(&p, 0, sizeof p);
    p.dtype = dtype;
    p.V = V;
    p.RV = static_cast<int32_t>((static_cast<int64_t>(V) * esize(dtype) + 15) / 16);
    p.gamma = gamma;
    p.kcap = 1;
    p.B = B;
    p.tokens = tokens;
    p.partials = reinterpret_cast<Partial *>(w.base + w.L.partials);
    p.status = status;
}

// Fill in the totals of a ScanParams whose groups are set.
void finish_params(ScanParams &p, const Work &w) {
    p.rows0 = static_cast<int64_t>(p.grp[0].nb) * p.grp[0].npos;
    p.rows = p.rows0 + (p.n_groups > 1 ? static_cast<int64_t>(p.grp[1].nb) * p.grp[1].npos : 0);
    p.T = p.rows * p.RV;
    p.W = scan_warps(w.W_max, p.T, p.rows);
    set_divisors(p);
}

// The streaming kernel over the rows of p.
sdd_status_t run_scan(const ScanParams &p, cudaStream_t stream) {
    if (p.T == 0) return SDD_OK;
    if (static_cast<double>(p.C) * static_cast<double>(p.W) >= 9.007199254740992e15)   // 2^53
        return fail(SDD_ERR_UNSUPPORTED, "%lld vectors of logits exceed the index arithmetic", (long long)p.T);
    const int grid = static_cast<int>((static_cast<int64_t>(p.W) + kWarpsPerCta - 1) / kWarpsPerCta);
    cudaError_t e = launch_scan(p, grid, stream);
    if (e != cudaSuccess) return cuda_fail(e, "scan launch");
    return SDD_OK;
}

// The decide kernel (row finalisation, decisions, draws) behind the streaming kernel.
sdd_status_t run_decide(const ScanParams &p, cudaStream_t stream) {
    if (p.T == 0) return SDD_OK;
    cudaError_t e = launch_decide(p, stream);
    if (e != cudaSuccess) return cuda_fail(e, "decide launch");
    return SDD_OK;
}

// The decide kernel of a vocabulary-sharded round (no streaming pass before it).
sdd_status_t run_decide_shard(const ScanParams &p, cudaStream_t stream) {
    cudaError_t e = launch_decide(p, stream);
    if (e != cudaSuccess) return cuda_fail(e, "decide launch");
    return SDD_OK;
}

// The draw geometry of nb blocks over `budget` decide teams of nt threads:
// each draw row of RV vectors is cut into nseg segments of whole nt-vector chunks, as
// many as keep nb * nseg teams within the budget (at least two vectors per
// thread, at most kDrawMaxSeg segments).
void draw_segments(int RV, int nb, int budget, int nt, int32_t &nseg, int32_t &seg_vec) {
    const int want = std::max(1, std::min(kDrawMaxSeg, budget / std::max(nb, 1)));
    const int per_thread = std::max(2, (RV + nt * want - 1) / (nt * want));
    seg_vec = per_thread * nt;
    nseg = (RV + seg_vec - 1) / seg_vec;
}

// Block decisions and, for the sampling rule, the draw geometry over the
// decide CTAs resident in one wave.
void init_dec(DecideParams &d, const Work &w, sdd_dtype_t dtype, int B, int gamma, int V, int64_t row_stride,
              const int32_t *tokens, int nb) {
    d.enabled = 1;
    d.B = B;
    d.gamma = gamma;
    d.V = V;
    d.stride_bytes = row_stride * esize(dtype);
    d.tokens = tokens;
    d.res_pref = reinterpret_cast<float *>(w.base + w.L.res_pref);
    d.res_count = reinterpret_cast<uint32_t *>(w.base + w.L.res_count);
    d.dec_ctas = w.dec_ctas;
    const int RV = static_cast<int>((static_cast<int64_t>(V) * esize(dtype) + 15) / 16);
    draw_segments(RV, nb, w.dec_ctas, kDecThreads, d.nseg, d.seg_vec);
}

sdd_status_t set_thresholds(int signal, const double *eta_b, const double *eta_c, int n_tau, df *eta_loc,
                            df *log_eta_c, int32_t *tau_off) {
    if (n_tau < 1 || n_tau > SDD_MAX_GRID)
        return fail(SDD_ERR_INVALID_ARGUMENT, "n_tau = %d outside [1, %d]", n_tau, SDD_MAX_GRID);
    if (!eta_b || !eta_c) return fail(SDD_ERR_INVALID_ARGUMENT, "eta_b / eta_c are NULL");
    if (signal != SDD_SIG_RAW && signal != SDD_SIG_MARGINAL && signal != SDD_SIG_CONDITIONAL)
        return fail(SDD_ERR_INVALID_ARGUMENT, "signal %d unknown", signal);
    for (int t = 0; t < n_tau; ++t) {
        const double eb = eta_b[t], ec = eta_c[t];
        if (std::isnan(eb) || std::isnan(ec)) return fail(SDD_ERR_INVALID_ARGUMENT, "threshold %d is NaN", t);
        tau_off[t] = (eb >= 1.0 || ec >= 1.0) ? 1 : 0;
        const double em = std::max(eb, ec);
        eta_loc[t] = df_from_double((signal == SDD_SIG_MARGINAL) ? em : eb);
        log_eta_c[t] = df_from_double((ec > 0.0) ? std::log(ec) : -INFINITY);
    }
    return SDD_OK;
}

// Periods and skip length of the periodic baseline, validated.
sdd_status_t set_periods(const int32_t *period, int n_p, int K_skip, int32_t *out) {
    if (n_p < 1 || n_p > SDD_MAX_GRID)
        return fail(SDD_ERR_INVALID_ARGUMENT, "%d periods outside [1, %d]", n_p, SDD_MAX_GRID);
    if (!period) return fail(SDD_ERR_INVALID_ARGUMENT, "period is NULL");
    if (K_skip < 1) return fail(SDD_ERR_INVALID_ARGUMENT, "K_skip = %d < 1", K_skip);
    for (int t = 0; t < n_p; ++t) {
        if (period[t] < 1) return fail(SDD_ERR_INVALID_ARGUMENT, "period[%d] = %d < 1", t, period[t]);
        out[t] = period[t];
    }
    return SDD_OK;
}

sdd_status_t set_ell(DecideParams &d, const double *ell, int n_ell) {
    if (n_ell < 0 || n_ell > SDD_MAX_GRID)
        return fail(SDD_ERR_INVALID_ARGUMENT, "n_ell = %d outside [0, %d]", n_ell, SDD_MAX_GRID);
    if (n_ell > 0 && !ell) return fail(SDD_ERR_INVALID_ARGUMENT, "ell is NULL");
    d.n_ell = n_ell;
    for (int r = 0; r < n_ell; ++r) {
        if (!(ell[r] > 0.0 && ell[r] <= 1.0))
            return fail(SDD_ERR_INVALID_ARGUMENT, "ell[%d] = %g outside (0, 1] (paper convention)", r, ell[r]);
        d.ell_one[r] = (ell[r] == 1.0) ? 1 : 0;
        d.ell_thr[r] = df_from_double(std::log(ell[r]));
    }
    return SDD_OK;
}

sdd_status_t set_topk(DecideParams &d, const int32_t *k, int n_k, int &kcap) {
    if (n_k < 0 || n_k > SDD_MAX_GRID) return fail(SDD_ERR_INVALID_ARGUMENT, "n_k = %d outside [0, %d]", n_k, SDD_MAX_GRID);
    if (n_k > 0 && !k) return fail(SDD_ERR_INVALID_ARGUMENT, "k is NULL");
    d.n_k = n_k;
    for (int r = 0; r < n_k; ++r) {
        if (k[r] < 1 || k[r] > 1024) return fail(SDD_ERR_INVALID_ARGUMENT, "k[%d] = %d outside [1, 1024]", r, k[r]);
        d.kval[r] = k[r];
        kcap = std::max(kcap, static_cast<int>(k[r]));
    }
    return SDD_OK;
}

sdd_status_t check_rows(const int32_t *rows, int n_rows, int B) {
    if (n_rows == 0) return SDD_OK;   // nothing to verify: rows may be NULL
    if (rows == nullptr && n_rows != B)
        return fail(SDD_ERR_INVALID_ARGUMENT, "rows is NULL but n_rows = %d != B = %d", n_rows, B);
    if (n_rows < 0 || n_rows > B) return fail(SDD_ERR_INVALID_ARGUMENT, "n_rows = %d outside [0, B]", n_rows);
    return SDD_OK;
}

#define SDD_TRY(expr)                         \
    do {                                      \
        sdd_status_t _s = (expr);             \
        if (_s != SDD_OK) return _s;          \
    } while (0)

// Target-row scan (post-verify) for the listed blocks; the block decisions in
// `dec` run inside the same launch.
sdd_status_t target_scan(const Work &w, const void *target_logits, sdd_dtype_t dtype, int B, int gamma, int V,
                         int64_t row_stride, const int32_t *tokens, const int32_t *rows, int n_rows, int kcap,
                         const DecideParams &dec, int32_t *status, cudaStream_t stream,
                         const int32_t *nb_dev = nullptr) {
    ScanParams p;
    init_scan(p, w, dtype, B, gamma, V, tokens, status);
    p.n_groups = 1;
    p.kcap = kcap;
    p.nb_dev = nb_dev;   // the listed-block count, read on the device (n_rows is then its maximum)
    ScanGroup &G = p.grp[0];
    G.base = static_cast<const char *>(target_logits);
    G.stride_bytes = row_stride * esize(dtype);
    G.npos = gamma + 1;
    G.kind = 1;
    G.nb = n_rows;
    G.bidx = rows;
    p.dec = dec;
    finish_params(p, w);
    SDD_TRY(run_scan(p, stream));
    return run_decide(p, stream);
}

}  // namespace

void set_last_error(const char *msg) { g_err = msg; }

}  // namespace sdd

using namespace sdd;

extern "C" {

int sdd_version(void) { return 100; }

const char *sdd_last_error(void) { return g_err.c_str(); }

sdd_status_t sdd_status_from_device(int32_t *status, int clear, uint32_t *bits, sdd_stream_t stream) {
    if (!status || !bits) return fail(SDD_ERR_INVALID_ARGUMENT, "status / bits is NULL");
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    int32_t h = 0;
    cudaError_t e = cudaMemcpyAsync(&h, status, sizeof h, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess && clear) e = cudaMemsetAsync(status, 0, sizeof h, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, "device status read");
    *bits = static_cast<uint32_t>(h);
    if (h == 0) return SDD_OK;
    return fail(SDD_ERR_DEVICE, "device status 0x%x:%s%s%s", static_cast<unsigned>(h),
                (h & SDD_DEV_NONFINITE) ? " non-finite row" : "", (h & SDD_DEV_BAD_TOKEN) ? " token out of range" : "",
                (h & SDD_DEV_TIMEOUT) ? " bounded wait expired" : "");
}

sdd_status_t sdd_workspace_size(int B, int gamma, int V, size_t *bytes) {
    if (!bytes) return fail(SDD_ERR_INVALID_ARGUMENT, "bytes is NULL");
    SDD_TRY(check_shape(SDD_BF16, B, gamma, V, ((static_cast<int64_t>(V) + 7) / 8) * 8));
    DevInfo di;
    SDD_TRY(device_info(di));
    *bytes = layout(B, gamma, static_cast<int64_t>(di.sms) * di.ctas_per_sm * kWarpsPerCta,
                    static_cast<int64_t>(di.sms) * di.dec_ctas_per_sm).total;
    return SDD_OK;
}

// The drafter statistics, with the extended features when margin or top5 is set.
static sdd_status_t confidence_impl(const void *draft_logits, sdd_dtype_t dtype, int B, int gamma, int V,
                                    int64_t row_stride, const int32_t *draft_tokens, float *q, float *logq,
                                    float *maxprob, double *lse, float *entropy, int32_t *argmax, float *margin,
                                    float *top5, void *workspace, size_t workspace_bytes, int32_t *status,
                                    sdd_stream_t stream) {
    SDD_TRY(check_shape(dtype, B, gamma, V, row_stride));
    if (B == 0) return SDD_OK;
    SDD_TRY(check_ptr16(draft_logits, "draft_logits"));
    if (!draft_tokens) return fail(SDD_ERR_INVALID_ARGUMENT, "draft_tokens is NULL");
    if (!q) return fail(SDD_ERR_INVALID_ARGUMENT, "q is NULL");
    Work w;
    SDD_TRY(get_work(workspace, workspace_bytes, B, gamma, w));
    ScanParams p;
    init_scan(p, w, dtype, B, gamma, V, draft_tokens, status);
    p.n_groups = 1;
    ScanGroup &G = p.grp[0];
    G.base = static_cast<const char *>(draft_logits);
    G.stride_bytes = row_stride * esize(dtype);
    G.npos = gamma;
    G.kind = 0;
    G.nb = B;
    G.q = q;
    G.logq = logq;
    G.maxprob = maxprob;
    G.lse = lse;
    G.entropy = entropy;
    G.argmax = argmax;
    if (margin || top5) {
        G.margin = margin;
        G.top5 = top5;
        p.feat = reinterpret_cast<FeatPartial *>(w.base + w.L.feat);
    }
    finish_params(p, w);
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    SDD_TRY(run_scan(p, st));
    return run_decide(p, st);
}

sdd_status_t sdd_confidence(const void *draft_logits, sdd_dtype_t dtype, int B, int gamma, int V,
                            int64_t row_stride, const int32_t *draft_tokens, float *q, float *logq,
                            float *maxprob, double *lse, float *entropy, int32_t *argmax, void *workspace,
                            size_t workspace_bytes, int32_t *status, sdd_stream_t stream) {
    return confidence_impl(draft_logits, dtype, B, gamma, V, row_stride, draft_tokens, q, logq, maxprob, lse, entropy,
                           argmax, nullptr, nullptr, workspace, workspace_bytes, status, stream);
}

sdd_status_t sdd_confidence_features(const void *draft_logits, sdd_dtype_t dtype, int B, int gamma, int V,
                                     int64_t row_stride, const int32_t *draft_tokens, float *q, float *logq,
                                     float *maxprob, double *lse, float *entropy, int32_t *argmax, float *margin,
                                     float *top5, void *workspace, size_t workspace_bytes, int32_t *status,
                                     sdd_stream_t stream) {
    if (!margin || !top5) return fail(SDD_ERR_INVALID_ARGUMENT, "margin and top5 must not be NULL");
    return confidence_impl(draft_logits, dtype, B, gamma, V, row_stride, draft_tokens, q, logq, maxprob, lse, entropy,
                           argmax, margin, top5, workspace, workspace_bytes, status, stream);
}

sdd_status_t sdd_schedule_prefix(const float *q, const float *logq, int B, int gamma, sdd_signal_t signal,
                                 const double *eta_b, const double *eta_c, int n_tau, int K_min, int S_max,
                                 const uint8_t *guard, const uint8_t *force_strict, const int32_t *D_in,
                                 int32_t *K_hat, int32_t *K, int32_t *D_out, int32_t *status, sdd_stream_t stream) {
    (void)status;
    if (B < 0) return fail(SDD_ERR_INVALID_ARGUMENT, "B = %d < 0", B);
    if (gamma < 1 || gamma > SDD_MAX_GAMMA)
        return fail(SDD_ERR_INVALID_ARGUMENT, "gamma = %d outside [1, %d]", gamma, SDD_MAX_GAMMA);
    ScheduleParams p;
    std::memset(&p, 0, sizeof p);
    SDD_TRY(set_thresholds(signal, eta_b, eta_c, n_tau, p.eta_loc, p.log_eta_c, p.tau_off));
    if (B == 0) return SDD_OK;
    if (!q || !K_hat || !K) return fail(SDD_ERR_INVALID_ARGUMENT, "q, K_hat and K must not be NULL");
    p.q = q;
    p.logq = logq;
    p.B = B;
    p.gamma = gamma;
    p.signal = signal;
    p.n_tau = n_tau;
    p.K_min = K_min;
    p.S_max = S_max;
    p.guard = guard;
    p.force_strict = force_strict;
    p.D_in = D_in;
    p.K_hat = K_hat;
    p.K = K;
    p.D_out = D_out;
    cudaError_t e = launch_schedule(p, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "schedule launch");
    return SDD_OK;
}

sdd_status_t sdd_schedule_periodic(int B, int gamma, const int32_t *period, int n_p, int K_skip, uint64_t round,
                                   int K_min, int S_max, const uint8_t *guard, const uint8_t *force_strict,
                                   const int32_t *D_in, int32_t *K_hat, int32_t *K, int32_t *D_out, int32_t *status,
                                   sdd_stream_t stream) {
    (void)status;
    if (B < 0) return fail(SDD_ERR_INVALID_ARGUMENT, "B = %d < 0", B);
    if (gamma < 1 || gamma > SDD_MAX_GAMMA)
        return fail(SDD_ERR_INVALID_ARGUMENT, "gamma = %d outside [1, %d]", gamma, SDD_MAX_GAMMA);
    ScheduleParams p;
    std::memset(&p, 0, sizeof p);
    SDD_TRY(set_periods(period, n_p, K_skip, p.period));
    if (B == 0) return SDD_OK;
    if (!K_hat || !K) return fail(SDD_ERR_INVALID_ARGUMENT, "K_hat and K must not be NULL");
    p.B = B;
    p.gamma = gamma;
    p.signal = SDD_SIG_PERIODIC;
    p.n_tau = n_p;
    p.K_skip = K_skip;
    p.round = round;
    p.K_min = K_min;
    p.S_max = S_max;
    p.guard = guard;
    p.force_strict = force_strict;
    p.D_in = D_in;
    p.K_hat = K_hat;
    p.K = K;
    p.D_out = D_out;
    cudaError_t e = launch_schedule(p, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "schedule launch");
    return SDD_OK;
}

sdd_status_t sdd_verify_strict(const void *target_logits, const void *draft_logits, sdd_dtype_t dtype, int B,
                               int gamma, int V, int64_t row_stride, const int32_t *draft_tokens,
                               const double *draft_lse, int greedy, uint64_t seed, uint64_t round, const int32_t *rows,
                               int n_rows, int32_t *L, int32_t *tokens, int32_t *n_commit, void *workspace,
                               size_t workspace_bytes, int32_t *status, sdd_stream_t stream) {
    SDD_TRY(check_shape(dtype, B, gamma, V, row_stride));
    SDD_TRY(check_rows(rows, n_rows, B));
    if (n_rows == 0) return SDD_OK;
    SDD_TRY(check_ptr16(target_logits, "target_logits"));
    if (!draft_tokens) return fail(SDD_ERR_INVALID_ARGUMENT, "draft_tokens is NULL");
    if (!greedy) {
        SDD_TRY(check_ptr16(draft_logits, "draft_logits"));
        if (!draft_lse) return fail(SDD_ERR_INVALID_ARGUMENT, "sampling needs draft_lse");
    }
    Work w;
    SDD_TRY(get_work(workspace, workspace_bytes, B, gamma, w));
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    DecideParams d;
    std::memset(&d, 0, sizeof d);
    init_dec(d, w, dtype, B, gamma, V, row_stride, draft_tokens, n_rows);
    d.zt = static_cast<const char *>(target_logits);
    d.zd = static_cast<const char *>(draft_logits);
    d.d_lse = draft_lse;
    d.do_strict = 1;
    d.greedy = greedy ? 1 : 0;
    d.seed = seed;
    d.round = round;
    d.L_strict = L;
    d.tok_strict = tokens;
    d.n_strict = n_commit;
    return target_scan(w, target_logits, dtype, B, gamma, V, row_stride, draft_tokens, rows, n_rows, 1, d, status, st);
}

sdd_status_t sdd_verify_strict_listed(const void *target_logits, const void *draft_logits, sdd_dtype_t dtype, int B,
                                      int gamma, int V, int64_t row_stride, const int32_t *draft_tokens,
                                      const double *draft_lse, int greedy, uint64_t seed, uint64_t round,
                                      const int32_t *rows, const int32_t *n_rows, int32_t *L, int32_t *tokens,
                                      int32_t *n_commit, void *workspace, size_t workspace_bytes, int32_t *status,
                                      sdd_stream_t stream) {
    SDD_TRY(check_shape(dtype, B, gamma, V, row_stride));
    if (B == 0) return SDD_OK;
    if (!rows || !n_rows) return fail(SDD_ERR_INVALID_ARGUMENT, "rows and n_rows must not be NULL");
    SDD_TRY(check_ptr16(target_logits, "target_logits"));
    if (!draft_tokens) return fail(SDD_ERR_INVALID_ARGUMENT, "draft_tokens is NULL");
    if (!greedy) {
        SDD_TRY(check_ptr16(draft_logits, "draft_logits"));
        if (!draft_lse) return fail(SDD_ERR_INVALID_ARGUMENT, "sampling needs draft_lse");
    }
    Work w;
    SDD_TRY(get_work(workspace, workspace_bytes, B, gamma, w));
    DecideParams d;
    std::memset(&d, 0, sizeof d);
    init_dec(d, w, dtype, B, gamma, V, row_stride, draft_tokens, B);
    d.zt = static_cast<const char *>(target_logits);
    d.zd = static_cast<const char *>(draft_logits);
    d.d_lse = draft_lse;
    d.do_strict = 1;
    d.greedy = greedy ? 1 : 0;
    d.seed = seed;
    d.round = round;
    d.L_strict = L;
    d.tok_strict = tokens;
    d.n_strict = n_commit;
    return target_scan(w, target_logits, dtype, B, gamma, V, row_stride, draft_tokens, rows, B, 1, d, status,
                       reinterpret_cast<cudaStream_t>(stream), n_rows);
}

sdd_status_t sdd_select_rows(const int32_t *K, int B, int32_t *rows, int32_t *n_rows, sdd_stream_t stream) {
    if (B < 0) return fail(SDD_ERR_INVALID_ARGUMENT, "B = %d < 0", B);
    if (!rows || !n_rows || (B > 0 && !K)) return fail(SDD_ERR_INVALID_ARGUMENT, "K, rows and n_rows must not be NULL");
    cudaError_t e = launch_select_rows(K, B, rows, n_rows, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "select rows launch");
    return SDD_OK;
}

sdd_status_t sdd_verify_lenient(const void *target_logits, sdd_dtype_t dtype, int B, int gamma, int V,
                                int64_t row_stride, const int32_t *draft_tokens, const double *ell, int n_ell,
                                const int32_t *rows, int n_rows, int32_t *L, int32_t *tokens, int32_t *n_commit,
                                void *workspace, size_t workspace_bytes, int32_t *status, sdd_stream_t stream) {
    SDD_TRY(check_shape(dtype, B, gamma, V, row_stride));
    SDD_TRY(check_rows(rows, n_rows, B));
    DecideParams d;
    std::memset(&d, 0, sizeof d);
    SDD_TRY(set_ell(d, ell, n_ell));
    if (n_ell < 1) return fail(SDD_ERR_INVALID_ARGUMENT, "n_ell must be >= 1");
    if (n_rows == 0) return SDD_OK;
    SDD_TRY(check_ptr16(target_logits, "target_logits"));
    if (!draft_tokens) return fail(SDD_ERR_INVALID_ARGUMENT, "draft_tokens is NULL");
    Work w;
    SDD_TRY(get_work(workspace, workspace_bytes, B, gamma, w));
    init_dec(d, w, dtype, B, gamma, V, row_stride, draft_tokens, n_rows);
    d.L_len = L;
    d.tok_len = tokens;
    d.n_len = n_commit;
    return target_scan(w, target_logits, dtype, B, gamma, V, row_stride, draft_tokens, rows, n_rows, 1, d, status,
                       reinterpret_cast<cudaStream_t>(stream));
}

sdd_status_t sdd_verify_topk(const void *target_logits, sdd_dtype_t dtype, int B, int gamma, int V,
                             int64_t row_stride, const int32_t *draft_tokens, const int32_t *k, int n_k,
                             const int32_t *rows, int n_rows, int32_t *L, int32_t *tokens, int32_t *n_commit,
                             void *workspace, size_t workspace_bytes, int32_t *status, sdd_stream_t stream) {
    SDD_TRY(check_shape(dtype, B, gamma, V, row_stride));
    SDD_TRY(check_rows(rows, n_rows, B));
    DecideParams d;
    std::memset(&d, 0, sizeof d);
    int kcap = 1;
    SDD_TRY(set_topk(d, k, n_k, kcap));
    if (n_k < 1) return fail(SDD_ERR_INVALID_ARGUMENT, "n_k must be >= 1");
    if (n_rows == 0) return SDD_OK;
    SDD_TRY(check_ptr16(target_logits, "target_logits"));
    if (!draft_tokens) return fail(SDD_ERR_INVALID_ARGUMENT, "draft_tokens is NULL");
    Work w;
    SDD_TRY(get_work(workspace, workspace_bytes, B, gamma, w));
    init_dec(d, w, dtype, B, gamma, V, row_stride, draft_tokens, n_rows);
    d.L_topk = L;
    d.tok_topk = tokens;
    d.n_topk = n_commit;
    return target_scan(w, target_logits, dtype, B, gamma, V, row_stride, draft_tokens, rows, n_rows, kcap, d, status,
                       reinterpret_cast<cudaStream_t>(stream));
}

sdd_status_t sdd_agreement(const int32_t *K, const int32_t *L_strict, int B, int n_tau, int64_t *acc,
                           sdd_stream_t stream) {
    if (B < 0 || n_tau < 0) return fail(SDD_ERR_INVALID_ARGUMENT, "B and n_tau must be >= 0");
    if (B == 0 || n_tau == 0) return SDD_OK;
    if (!K || !L_strict || !acc) return fail(SDD_ERR_INVALID_ARGUMENT, "K, L_strict and acc must not be NULL");
    cudaError_t e = launch_agreement(K, L_strict, B, n_tau, reinterpret_cast<long long *>(acc),
                                     reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "agreement launch");
    return SDD_OK;
}

sdd_status_t sdd_commit(const int32_t *K, const int32_t *draft_tokens, const int32_t *verified_tokens,
                        const int32_t *verified_n, int B, int gamma, int32_t *out_tokens, int32_t *out_n,
                        sdd_stream_t stream) {
    if (B < 0 || gamma < 1 || gamma > SDD_MAX_GAMMA) return fail(SDD_ERR_INVALID_ARGUMENT, "bad B or gamma");
    if (B == 0) return SDD_OK;
    if (!K || !draft_tokens || !verified_tokens || !verified_n || !out_tokens || !out_n)
        return fail(SDD_ERR_INVALID_ARGUMENT, "NULL array");
    cudaError_t e = launch_commit(K, draft_tokens, verified_tokens, verified_n, B, gamma, out_tokens, out_n,
                                  reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "commit launch");
    return SDD_OK;
}

sdd_status_t sdd_uniforms(uint64_t seed, const uint32_t *j, const uint32_t *b, const uint64_t *round,
                          const uint32_t *purpose, int64_t n, float *u, sdd_stream_t stream) {
    if (n < 0) return fail(SDD_ERR_INVALID_ARGUMENT, "n < 0");
    if (n == 0) return SDD_OK;
    if (!j || !b || !round || !purpose || !u) return fail(SDD_ERR_INVALID_ARGUMENT, "NULL array");
    cudaError_t e = launch_uniforms(seed, j, b, round, purpose, n, u, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "uniforms launch");
    return SDD_OK;
}

sdd_status_t sdd_test_wait_hooks(uint32_t polls, int drop_copy) {
    set_scan_wait_hooks(polls, drop_copy);
    return SDD_OK;
}

sdd_status_t sdd_scorer_features(const float *maxprob, const float *entropy, const float *margin,
                                 const float *top5, int B, int gamma, int64_t round, void *f, sdd_stream_t stream) {
    if (B < 0 || gamma < 1 || gamma > SDD_MAX_GAMMA)
        return fail(SDD_ERR_INVALID_ARGUMENT, "B = %d / gamma = %d out of range", B, gamma);
    if (round < 0) return fail(SDD_ERR_INVALID_ARGUMENT, "round = %lld < 0", static_cast<long long>(round));
    if (B == 0) return SDD_OK;
    if (!maxprob || !entropy || !margin || !top5)
        return fail(SDD_ERR_INVALID_ARGUMENT, "maxprob, entropy, margin and top5 must not be NULL");
    SDD_TRY(check_ptr16(f, "f"));
    const cudaError_t e =
        launch_scorer_features(maxprob, entropy, margin, top5, static_cast<int64_t>(B) * gamma, gamma,
                               static_cast<float>(static_cast<double>(round) / 256.0), static_cast<uint16_t *>(f),
                               reinterpret_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? SDD_OK : cuda_fail(e, "scorer features launch");
}

sdd_status_t sdd_scorer_workspace_size(int M, size_t *bytes) {
    if (!bytes) return fail(SDD_ERR_INVALID_ARGUMENT, "bytes is NULL");
    if (M < 0) return fail(SDD_ERR_INVALID_ARGUMENT, "M = %d < 0", M);
    *bytes = mlp_workspace_bytes(M);
    return SDD_OK;
}

// The scorers' workspace: present, 16-byte aligned and large enough for M rows.
static sdd_status_t check_scorer_ws(int M, const void *workspace, size_t workspace_bytes) {
    SDD_TRY(check_ptr16(workspace, "workspace"));
    const size_t need = mlp_workspace_bytes(M);
    if (workspace_bytes < need)
        return fail(SDD_ERR_INVALID_ARGUMENT, "workspace of %zu bytes < %zu needed", workspace_bytes, need);
    return SDD_OK;
}

sdd_status_t sdd_survival_mlp(const void *h, int M, int K, const void *W1, const float *b1, const void *w2, float b2,
                              float *s, void *workspace, size_t workspace_bytes, int32_t *status,
                              sdd_stream_t stream) {
    if (M < 0) return fail(SDD_ERR_INVALID_ARGUMENT, "M = %d < 0", M);
    if (K < SDD_MLP_KSTEP || K % SDD_MLP_KSTEP != 0)
        return fail(SDD_ERR_INVALID_ARGUMENT, "K = %d is not a positive multiple of %d", K, SDD_MLP_KSTEP);
    if (M == 0) return SDD_OK;
    SDD_TRY(check_ptr16(h, "h"));
    SDD_TRY(check_ptr16(W1, "W1"));
    if (!b1 || !w2 || !s) return fail(SDD_ERR_INVALID_ARGUMENT, "b1, w2 and s must not be NULL");
    SDD_TRY(check_scorer_ws(M, workspace, workspace_bytes));
    int d = 0;
    cudaError_t e = cudaGetDevice(&d);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    int major = 0, minor = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, d);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, d);
    if (major != 10) return fail(SDD_ERR_UNSUPPORTED, "tcgen05 scorer needs an sm_10x device (found sm_%d%d)", major, minor);
    const char *why = nullptr;
    e = launch_mlp(h, M, K, W1, b1, w2, b2, s, workspace, status, reinterpret_cast<cudaStream_t>(stream), &why);
    if (why) return fail(SDD_ERR_CUDA, "survival scorer: %s", why);
    if (e != cudaSuccess) return cuda_fail(e, "survival scorer launch");
    return SDD_OK;
}

sdd_status_t sdd_scorer_deep(const void *h, int Kh, const void *f, int M, const void *W1, const float *b1,
                             const void *W2, const float *b2, const void *W3, const float *b3, const void *w4,
                             float b4, void *act, float *s, void *workspace, size_t workspace_bytes,
                             int32_t *status, sdd_stream_t stream) {
    if (M < 0) return fail(SDD_ERR_INVALID_ARGUMENT, "M = %d < 0", M);
    if (Kh < SDD_MLP_KSTEP || Kh % SDD_MLP_KSTEP != 0)
        return fail(SDD_ERR_INVALID_ARGUMENT, "Kh = %d is not a positive multiple of %d", Kh, SDD_MLP_KSTEP);
    if (M == 0) return SDD_OK;
    SDD_TRY(check_ptr16(h, "h"));
    SDD_TRY(check_ptr16(f, "f"));
    SDD_TRY(check_ptr16(W1, "W1"));
    SDD_TRY(check_ptr16(W2, "W2"));
    SDD_TRY(check_ptr16(W3, "W3"));
    SDD_TRY(check_ptr16(act, "act"));
    if (!b1 || !b2 || !b3 || !w4 || !s) return fail(SDD_ERR_INVALID_ARGUMENT, "b1, b2, b3, w4 and s must not be NULL");
    SDD_TRY(check_scorer_ws(M, workspace, workspace_bytes));
    int d = 0;
    cudaError_t e = cudaGetDevice(&d);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    int major = 0, minor = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, d);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, d);
    if (major != 10) return fail(SDD_ERR_UNSUPPORTED, "tcgen05 scorer needs an sm_10x device (found sm_%d%d)", major, minor);
    const char *why = nullptr;
    e = launch_scorer_deep(h, Kh, f, M, W1, b1, W2, b2, W3, b3, w4, b4, static_cast<uint16_t *>(act), s, workspace,
                           status, reinterpret_cast<cudaStream_t>(stream), &why);
    if (why) return fail(SDD_ERR_CUDA, "deep scorer: %s", why);
    if (e != cudaSuccess) return cuda_fail(e, "deep scorer launch");
    return SDD_OK;
}

sdd_status_t sdd_permutation_workspace_size(int B, int gamma, int n_rep, size_t *bytes) {
    if (!bytes) return fail(SDD_ERR_INVALID_ARGUMENT, "bytes is NULL");
    if (B < 0 || gamma < 1 || gamma > SDD_MAX_GAMMA || n_rep < 0)
        return fail(SDD_ERR_INVALID_ARGUMENT, "B = %d, gamma = %d, n_rep = %d out of range", B, gamma, n_rep);
    *bytes = align256(static_cast<size_t>(n_rep) * gamma * B * sizeof(float)) +
             align256(static_cast<size_t>(n_rep + 1) * sizeof(unsigned long long));
    return SDD_OK;
}

sdd_status_t sdd_permutation_diagnostic(const float *q, const int32_t *L, int B, int gamma, sdd_signal_t signal,
                                        double eta_b, double eta_c, int n_rep, uint64_t seed, int64_t *sums,
                                        void *workspace, size_t workspace_bytes, sdd_stream_t stream) {
    if (B < 0 || gamma < 1 || gamma > SDD_MAX_GAMMA)
        return fail(SDD_ERR_INVALID_ARGUMENT, "B = %d / gamma = %d out of range", B, gamma);
    if (n_rep < 0 || n_rep > 100000) return fail(SDD_ERR_INVALID_ARGUMENT, "n_rep = %d out of range", n_rep);
    if (B > 50000) return fail(SDD_ERR_UNSUPPORTED, "B = %d logged blocks exceed 50000 (one shared-memory list)", B);
    df eta_loc, log_eta_c;
    int32_t off = 0;
    SDD_TRY(set_thresholds(signal, &eta_b, &eta_c, 1, &eta_loc, &log_eta_c, &off));
    if (B == 0) return SDD_OK;
    if (!q || !L || !sums) return fail(SDD_ERR_INVALID_ARGUMENT, "q, L and sums must not be NULL");
    size_t need = 0;
    SDD_TRY(sdd_permutation_workspace_size(B, gamma, n_rep, &need));
    if (!workspace || workspace_bytes < need)
        return fail(SDD_ERR_INVALID_ARGUMENT, "workspace of %zu bytes < %zu needed", workspace_bytes, need);
    if (off) {   // a threshold >= 1 disables skipping: every feasible prefix is 0
        cudaError_t e = cudaMemsetAsync(sums, 0, sizeof(int64_t) * (n_rep + 1), reinterpret_cast<cudaStream_t>(stream));
        return e == cudaSuccess ? SDD_OK : cuda_fail(e, "memset");
    }
    unsigned char *base = static_cast<unsigned char *>(workspace);
    float *pq = reinterpret_cast<float *>(base);   // the permuted scores, [n_rep][gamma][B]
    unsigned long long *acc = reinterpret_cast<unsigned long long *>(
        base + align256(static_cast<size_t>(n_rep) * gamma * B * sizeof(float)));
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e = launch_perm_diag(q, L, B, gamma, signal, eta_loc, log_eta_c, n_rep, seed, pq, acc, st);
    if (e != cudaSuccess) return cuda_fail(e, "permutation diagnostic launch");
    e = cudaMemcpyAsync(sums, acc, sizeof(int64_t) * (n_rep + 1), cudaMemcpyDeviceToDevice, st);
    return e == cudaSuccess ? SDD_OK : cuda_fail(e, "copy");
}

sdd_status_t sdd_position_metrics(const float *q, const int32_t *L, int B, int gamma, int conditional, double *bce,
                                  double *bce_base, double *auroc, int32_t *n_pos, int32_t *n_neg,
                                  sdd_stream_t stream) {
    if (B < 0 || gamma < 1 || gamma > SDD_MAX_GAMMA)
        return fail(SDD_ERR_INVALID_ARGUMENT, "B = %d / gamma = %d out of range", B, gamma);
    if (!q || !L || !bce || !bce_base || !auroc)
        return fail(SDD_ERR_INVALID_ARGUMENT, "q, L, bce, bce_base and auroc must not be NULL");
    cudaError_t e = launch_position_metrics(q, L, B, gamma, conditional ? 1 : 0, bce, bce_base, auroc, n_pos, n_neg,
                                            reinterpret_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? SDD_OK : cuda_fail(e, "position metrics launch");
}

static sdd_status_t block_check(const sdd_block_args *a) {
    if (!a) return fail(SDD_ERR_INVALID_ARGUMENT, "args is NULL");
    SDD_TRY(check_shape(static_cast<sdd_dtype_t>(a->dtype), a->B, a->gamma, a->V, a->row_stride));
    if (a->B == 0) return SDD_OK;
    SDD_TRY(check_ptr16(a->draft_logits, "draft_logits"));
    SDD_TRY(check_ptr16(a->target_logits, "target_logits"));
    if (!a->draft_tokens) return fail(SDD_ERR_INVALID_ARGUMENT, "draft_tokens is NULL");
    return SDD_OK;
}

// The launch parameters of one fused round, from its arguments (both halves
// of sdd_block build the same ones).  Sets *empty when there is nothing to do.
static sdd_status_t block_params(const sdd_block_args *a, ScanParams &p, bool *empty) {
    SDD_TRY(block_check(a));
    const sdd_dtype_t dt = static_cast<sdd_dtype_t>(a->dtype);
    DecideParams d;
    std::memset(&d, 0, sizeof d);
    if (a->signal == SDD_SIG_PERIODIC) {
        SDD_TRY(set_periods(a->period, a->n_tau, a->K_skip, d.period));
        d.K_skip = a->K_skip;
    } else {
        SDD_TRY(set_thresholds(a->signal, a->eta_b, a->eta_c, a->n_tau, d.eta_loc, d.log_eta_c, d.tau_off));
    }
    SDD_TRY(set_ell(d, a->ell, a->n_ell));
    int kcap = 1;
    SDD_TRY(set_topk(d, a->topk, a->n_k, kcap));
    *empty = a->B == 0;
    if (*empty) return SDD_OK;
    Work w;
    SDD_TRY(get_work(a->workspace, a->workspace_bytes, a->B, a->gamma, w));
    init_scan(p, w, dt, a->B, a->gamma, a->V, a->draft_tokens, a->status);
    p.n_groups = 2;
    p.kcap = kcap;
    ScanGroup &D = p.grp[0];
    D.base = static_cast<const char *>(a->draft_logits);
    D.stride_bytes = a->row_stride * esize(dt);
    D.npos = a->gamma;
    D.kind = 0;
    D.nb = a->B;
    D.q = a->q;
    D.logq = a->logq;
    D.maxprob = a->maxprob;
    D.lse = a->lse;
    D.entropy = a->entropy;
    D.argmax = a->argmax;
    ScanGroup &T = p.grp[1];
    T.base = static_cast<const char *>(a->target_logits);
    T.stride_bytes = a->row_stride * esize(dt);
    T.npos = a->gamma + 1;
    T.kind = 1;
    T.nb = a->B;
    init_dec(d, w, dt, a->B, a->gamma, a->V, a->row_stride, a->draft_tokens, a->B);
    d.zt = static_cast<const char *>(a->target_logits);
    d.zd = static_cast<const char *>(a->draft_logits);
    d.do_strict = 1;
    d.greedy = a->greedy ? 1 : 0;
    d.seed = a->seed;
    d.round = a->round;
    d.L_strict = a->L_strict;
    d.tok_strict = a->tokens_strict;
    d.n_strict = a->n_strict;
    d.L_len = a->L_lenient;
    d.tok_len = a->tokens_lenient;
    d.n_len = a->n_lenient;
    d.L_topk = a->L_topk;
    d.tok_topk = a->tokens_topk;
    d.n_topk = a->n_topk;
    d.do_sched = 1;
    d.signal = a->signal;
    d.n_tau = a->n_tau;
    d.K_min = a->K_min;
    d.S_max = a->S_max;
    d.guard = a->guard;
    d.force_strict = a->force_strict;
    d.D_in = a->D_in;
    d.K_hat = a->K_hat;
    d.K = a->K;
    d.D_out = a->D_out;
    d.commit_tokens = a->commit_tokens;
    d.commit_n = a->commit_n;
    d.agreement = reinterpret_cast<long long *>(a->agreement);
    p.dec = d;
    finish_params(p, w);
    return SDD_OK;
}

// ---------------------------------------------------------------------------
// Vocabulary-sharded round
// ---------------------------------------------------------------------------
static sdd_status_t shard_check(const sdd_block_args *a, int v0, int v1) {
    if (!a) return fail(SDD_ERR_INVALID_ARGUMENT, "args is NULL");
    const sdd_dtype_t dt = static_cast<sdd_dtype_t>(a->dtype);
    if (dt != SDD_F32 && dt != SDD_BF16) return fail(SDD_ERR_INVALID_ARGUMENT, "dtype %d unknown", a->dtype);
    if (a->B < 0) return fail(SDD_ERR_INVALID_ARGUMENT, "B = %d < 0", a->B);
    if (a->gamma < 1 || a->gamma > SDD_MAX_GAMMA)
        return fail(SDD_ERR_INVALID_ARGUMENT, "gamma = %d outside [1, %d]", a->gamma, SDD_MAX_GAMMA);
    if (a->V < 1) return fail(SDD_ERR_INVALID_ARGUMENT, "V = %d < 1", a->V);
    if (v0 < 0 || v1 <= v0 || v1 > a->V)
        return fail(SDD_ERR_INVALID_ARGUMENT, "slice [%d, %d) is empty or outside [0, V = %d)", v0, v1, a->V);
    const int w = v1 - v0;
    if (a->row_stride < w)
        return fail(SDD_ERR_INVALID_ARGUMENT, "row_stride %lld < slice width %d", (long long)a->row_stride, w);
    if ((a->row_stride * esize(dt)) % 16 != 0)
        return fail(SDD_ERR_INVALID_ARGUMENT, "row_stride * element size must be a multiple of 16 bytes");
    if (a->row_stride * esize(dt) > (int64_t(1) << 31))
        return fail(SDD_ERR_INVALID_ARGUMENT, "rows longer than 2 GiB are not supported");
    if (a->B == 0) return SDD_OK;
    SDD_TRY(check_ptr16(a->draft_logits, "draft_logits"));
    SDD_TRY(check_ptr16(a->target_logits, "target_logits"));
    if (!a->draft_tokens) return fail(SDD_ERR_INVALID_ARGUMENT, "draft_tokens is NULL");
    return SDD_OK;
}

static sdd_status_t shard_kcap(const sdd_block_args *a, int &kcap) {
    DecideParams d;
    std::memset(&d, 0, sizeof d);
    int kc = 1;
    SDD_TRY(set_topk(d, a->topk, a->n_k, kc));
    if (a->n_k > 0 && kc > SDD_SHARD_KMAX)
        return fail(SDD_ERR_UNSUPPORTED, "top-k with k = %d: the sharded round keeps at most %d candidates", kc,
                    SDD_SHARD_KMAX);
    kcap = (a->n_k > 0) ? kc : 0;
    return SDD_OK;
}

// The sharded round's workspace: per block the draw state, the draw's
// arrival counter, each draw segment's p_t mass and each segment's per-thread
// prefix sums (at most kDrawMaxSeg segments of kDecThreads runs per block).
struct ShardWs {
    size_t state, count, ptot, pref, total;
};
static ShardWs shard_ws_layout(int B) {
    auto up = [](size_t v, size_t a) { return (v + a - 1) / a * a; };
    const size_t b = static_cast<size_t>(B);
    ShardWs w;
    w.state = 0;
    w.count = up(b * sizeof(ShardDraw), 16);
    w.ptot = up(w.count + b * sizeof(uint32_t), 16);
    w.pref = up(w.ptot + b * kDrawMaxSeg * sizeof(float), 16);
    w.total = w.pref + b * kDrawMaxSeg * kDecThreads * sizeof(float);
    return w;
}

// Draw segments of a slice's draw rows (RV vectors) for B blocks, cut the way
// init_dec cuts one-GPU draw rows: as many as keep B * nseg decide CTAs
// resident at once, at least two vectors per thread, at most kDrawMaxSeg.
static void shard_segments(int B, int RV, int dec_ctas, int32_t &nseg, int32_t &seg_vec) {
    const int want = std::max(1, std::min(kDrawMaxSeg, dec_ctas / std::max(B, 1)));
    const int per_thread = std::max(2, (RV + kDecThreads * want - 1) / (kDecThreads * want));
    seg_vec = per_thread * kDecThreads;
    nseg = (RV + seg_vec - 1) / seg_vec;
}

sdd_status_t sdd_shard_workspace_size(int B, size_t *bytes) {
    if (!bytes) return fail(SDD_ERR_INVALID_ARGUMENT, "bytes is NULL");
    if (B < 0) return fail(SDD_ERR_INVALID_ARGUMENT, "B = %d < 0", B);
    *bytes = shard_ws_layout(B).total;
    return SDD_OK;
}

static void shard_geometry(ShardParams &sp, const sdd_block_args *a, int v0, int v1) {
    std::memset(&sp, 0, sizeof sp);
    const sdd_dtype_t dt = static_cast<sdd_dtype_t>(a->dtype);
    sp.zd = static_cast<const char *>(a->draft_logits);
    sp.zt = static_cast<const char *>(a->target_logits);
    sp.stride_bytes = a->row_stride * esize(dt);
    sp.dtype = dt;
    sp.B = a->B;
    sp.gamma = a->gamma;
    sp.Vs = v1 - v0;
    sp.RVs = static_cast<int32_t>((static_cast<int64_t>(sp.Vs) * esize(dt) + 15) / 16);
    sp.v0 = v0;
    sp.V = a->V;
    sp.tokens = a->draft_tokens;
    sp.status = a->status;
}

sdd_status_t sdd_shard_partials(const sdd_block_args *a, int v0, int v1, sdd_shard_partial *out,
                                sdd_stream_t stream) {
    SDD_TRY(shard_check(a, v0, v1));
    int kcap = 0;
    SDD_TRY(shard_kcap(a, kcap));
    if (a->B == 0) return SDD_OK;
    if (!out) return fail(SDD_ERR_INVALID_ARGUMENT, "out is NULL");
    ShardParams sp;
    shard_geometry(sp, a, v0, v1);
    sp.kcap = kcap;
    sp.out = out;
    cudaError_t e = launch_shard_partials(sp, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "shard partials launch");
    return SDD_OK;
}

static sdd_status_t shard_state_ws(const sdd_block_args *a) {
    size_t need = 0;
    SDD_TRY(sdd_shard_workspace_size(a->B, &need));
    if (!a->workspace) return fail(SDD_ERR_WORKSPACE, "workspace is NULL");
    if (reinterpret_cast<uintptr_t>(a->workspace) % 16 != 0)
        return fail(SDD_ERR_WORKSPACE, "workspace is not 16-byte aligned");
    if (a->workspace_bytes < need)
        return fail(SDD_ERR_WORKSPACE, "workspace has %zu bytes, %zu needed", a->workspace_bytes, need);
    return SDD_OK;
}

sdd_status_t sdd_shard_decide(const sdd_block_args *a, int v0, int v1, int n_shards, const sdd_shard_partial *all,
                              float *mass, sdd_stream_t stream) {
    SDD_TRY(shard_check(a, v0, v1));
    if (n_shards < 1 || n_shards > 64) return fail(SDD_ERR_INVALID_ARGUMENT, "n_shards = %d outside [1, 64]", n_shards);
    int kcap = 0;
    SDD_TRY(shard_kcap(a, kcap));
    const sdd_dtype_t dt = static_cast<sdd_dtype_t>(a->dtype);
    DecideParams d;
    std::memset(&d, 0, sizeof d);
    if (a->signal == SDD_SIG_PERIODIC) {
        SDD_TRY(set_periods(a->period, a->n_tau, a->K_skip, d.period));
        d.K_skip = a->K_skip;
    } else {
        SDD_TRY(set_thresholds(a->signal, a->eta_b, a->eta_c, a->n_tau, d.eta_loc, d.log_eta_c, d.tau_off));
    }
    SDD_TRY(set_ell(d, a->ell, a->n_ell));
    int kc = 1;
    SDD_TRY(set_topk(d, a->topk, a->n_k, kc));
    if (a->B == 0) return SDD_OK;
    if (!all) return fail(SDD_ERR_INVALID_ARGUMENT, "all is NULL");
    const bool sampling = !a->greedy;
    if (sampling && !mass) return fail(SDD_ERR_INVALID_ARGUMENT, "mass is NULL (strict sampling)");
    SDD_TRY(shard_state_ws(a));
    ScanParams p;
    std::memset(&p, 0, sizeof p);
    p.dtype = dt;
    p.V = v1 - v0;
    p.RV = static_cast<int32_t>((static_cast<int64_t>(p.V) * esize(dt) + 15) / 16);
    p.gamma = a->gamma;
    p.kcap = std::max(1, kcap);
    p.B = a->B;
    p.tokens = a->draft_tokens;
    p.status = a->status;
    p.n_groups = 2;
    ScanGroup &D = p.grp[0];
    D.base = static_cast<const char *>(a->draft_logits);
    D.stride_bytes = a->row_stride * esize(dt);
    D.npos = a->gamma;
    D.kind = 0;
    D.nb = a->B;
    D.q = a->q;
    D.logq = a->logq;
    D.maxprob = a->maxprob;
    D.lse = a->lse;
    D.entropy = a->entropy;
    D.argmax = a->argmax;
    ScanGroup &T = p.grp[1];
    T.base = static_cast<const char *>(a->target_logits);
    T.stride_bytes = a->row_stride * esize(dt);
    T.npos = a->gamma + 1;
    T.kind = 1;
    T.nb = a->B;
    p.rows0 = static_cast<int64_t>(a->B) * a->gamma;
    p.rows = static_cast<int64_t>(a->B) * (2 * a->gamma + 1);
    p.shard = all;
    p.n_shards = n_shards;
    p.shard_v0 = v0;
    p.shard_rows = p.rows;
    d.enabled = 1;
    d.B = a->B;
    d.gamma = a->gamma;
    d.V = p.V;
    d.stride_bytes = a->row_stride * esize(dt);
    d.tokens = a->draft_tokens;
    DevInfo di;
    SDD_TRY(device_info(di));   // the kernels' attributes are set on this device
    const ShardWs L = shard_ws_layout(a->B);
    char *ws = static_cast<char *>(a->workspace);
    d.dec_ctas = di.sms * di.dec_ctas_per_sm;
    shard_segments(a->B, p.RV, d.dec_ctas, d.nseg, d.seg_vec);
    d.res_pref = reinterpret_cast<float *>(ws + L.pref);
    d.res_count = reinterpret_cast<uint32_t *>(ws + L.count);
    d.shard_ptot = reinterpret_cast<float *>(ws + L.ptot);
    d.zt = static_cast<const char *>(a->target_logits);
    d.zd = static_cast<const char *>(a->draft_logits);
    d.do_strict = 1;
    d.greedy = a->greedy ? 1 : 0;
    d.seed = a->seed;
    d.round = a->round;
    d.L_strict = a->L_strict;
    d.tok_strict = a->tokens_strict;
    d.n_strict = a->n_strict;
    d.L_len = a->L_lenient;
    d.tok_len = a->tokens_lenient;
    d.n_len = a->n_lenient;
    d.L_topk = a->L_topk;
    d.tok_topk = a->tokens_topk;
    d.n_topk = a->n_topk;
    d.do_sched = 1;
    d.signal = a->signal;
    d.n_tau = a->n_tau;
    d.K_min = a->K_min;
    d.S_max = a->S_max;
    d.guard = a->guard;
    d.force_strict = a->force_strict;
    d.D_in = a->D_in;
    d.K_hat = a->K_hat;
    d.K = a->K;
    d.D_out = a->D_out;
    d.commit_tokens = a->commit_tokens;
    d.commit_n = a->commit_n;
    d.agreement = reinterpret_cast<long long *>(a->agreement);
    d.shard_mass = mass;
    d.shard_state = reinterpret_cast<ShardDraw *>(ws + L.state);
    p.dec = d;
    return run_decide_shard(p, reinterpret_cast<cudaStream_t>(stream));
}

sdd_status_t sdd_shard_draw(const sdd_block_args *a, int v0, int v1, int n_shards, int shard, const float *mass_all,
                            sdd_stream_t stream) {
    SDD_TRY(shard_check(a, v0, v1));
    if (n_shards < 1 || n_shards > 64) return fail(SDD_ERR_INVALID_ARGUMENT, "n_shards = %d outside [1, 64]", n_shards);
    if (shard < 0 || shard >= n_shards)
        return fail(SDD_ERR_INVALID_ARGUMENT, "shard = %d outside [0, %d)", shard, n_shards);
    if (a->B == 0 || a->greedy) return SDD_OK;   // only strict sampling draws
    if (!mass_all) return fail(SDD_ERR_INVALID_ARGUMENT, "mass_all is NULL");
    SDD_TRY(shard_state_ws(a));
    ShardParams sp;
    shard_geometry(sp, a, v0, v1);
    sp.n_shards = n_shards;
    sp.shard = shard;
    sp.mass_all = mass_all;
    DevInfo di;
    SDD_TRY(device_info(di));   // the kernels' attributes are set on this device
    const ShardWs L = shard_ws_layout(a->B);
    const char *ws = static_cast<const char *>(a->workspace);
    sp.state = reinterpret_cast<const ShardDraw *>(ws + L.state);
    sp.res_pref = reinterpret_cast<const float *>(ws + L.pref);
    shard_segments(a->B, sp.RVs, di.sms * di.dec_ctas_per_sm, sp.nseg, sp.seg_vec);
    sp.seed = a->seed;
    sp.round = a->round;
    sp.tok_strict = a->tokens_strict;
    sp.commit_tokens = a->commit_tokens;
    cudaError_t e = launch_shard_draw(sp, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "shard draw launch");
    return SDD_OK;
}

sdd_status_t sdd_block_scan(const sdd_block_args *a, sdd_stream_t stream) {
    ScanParams p;
    bool empty = false;
    SDD_TRY(block_params(a, p, &empty));
    if (empty) return SDD_OK;
    return run_scan(p, reinterpret_cast<cudaStream_t>(stream));
}

sdd_status_t sdd_block_decide(const sdd_block_args *a, sdd_stream_t stream) {
    ScanParams p;
    bool empty = false;
    SDD_TRY(block_params(a, p, &empty));
    if (empty) return SDD_OK;
    return run_decide(p, reinterpret_cast<cudaStream_t>(stream));
}

sdd_status_t sdd_block(const sdd_block_args *a, sdd_stream_t stream) {
    SDD_TRY(sdd_block_scan(a, stream));
    return sdd_block_decide(a, stream);
}

// Rounds of at most this many bytes of logits run in the pipelined kernel;
// larger ones stream on all sixteen warps of each CTA (sdd_block_scan) and are
// decided by the decide kernel in the next call.  Measured on GB300 (rows of
// 32 positions over V = 151,936 bf16, blocks/s pipelined kernel / two
// kernels): B = 16 (316 MB) 257 k / 232 k, B = 24 (474 MB) 274.5 k / 257.4 k,
// B = 32 (632 MB) 254.9 k / 272.4 k, B = 40 (790 MB) 256.5 k / 282.4 k: the
// decide kernel's fixed tail matters less as the round grows, while fourteen
// streaming warps and the decide work beside them trail sixteen warps alone.
constexpr int64_t kPipeMaxBytes = int64_t(512) << 20;

// A pipelined round's launch parameters: sdd_block's, streamed by warps
// kPipeWarps..15 of each CTA when the round is at most kPipeMaxBytes (the same
// when the round is streamed and when it is decided).
static sdd_status_t pipe_params(const sdd_block_args *a, ScanParams &p, bool *empty) {
    SDD_TRY(block_params(a, p, empty));
    if (*empty || p.T * 16 > kPipeMaxBytes) return SDD_OK;
    Work w;
    SDD_TRY(get_work(a->workspace, a->workspace_bytes, a->B, a->gamma, w));
    // the decide team beside this round's streaming pass (warps 0 .. warp0-1)
    const int team_warps = (p.T * 16 <= kPipeSmallBytes ? kPipeTeamSmall : kPipeTeam) / 32;
    const int wpc = kWarpsPerCta - team_warps;
    p.W = scan_warps(w.W_max / kWarpsPerCta * wpc, p.T, p.rows);
    set_divisors(p, kPipeCostDrafter, kPipeCostTarget);
    p.warp0 = team_warps;
    p.wpc = wpc;
    return SDD_OK;
}

sdd_status_t sdd_block_pipelined(const sdd_block_args *next, const sdd_block_args *prev, sdd_stream_t stream) {
    if (!next && !prev) return fail(SDD_ERR_INVALID_ARGUMENT, "next and prev are both NULL");
    if (next && prev && next->B > 0 && prev->B > 0 && next->workspace == prev->workspace)
        return fail(SDD_ERR_INVALID_ARGUMENT, "next and prev share a workspace");
    ScanParams pn, pp;
    bool en = true, ep = true;
    if (next) SDD_TRY(pipe_params(next, pn, &en));
    if (prev) SDD_TRY(pipe_params(prev, pp, &ep));
    const cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (en) return ep ? SDD_OK : run_decide(pp, st);   // the last round of a sequence: decide only
    if (pn.wpc == kWarpsPerCta) {
        // a large round: prev's decide kernel, then next's streaming kernel
        if (!ep) SDD_TRY(run_decide(pp, st));
        return run_scan(pn, st);
    }
    if (static_cast<double>(pn.C) * static_cast<double>(pn.W) >= 9.007199254740992e15)   // 2^53
        return fail(SDD_ERR_UNSUPPORTED, "%lld vectors of logits exceed the index arithmetic", (long long)pn.T);
    const int grid = static_cast<int>((static_cast<int64_t>(pn.W) + pn.wpc - 1) / pn.wpc);
    // prev's draw segments over this grid's CTAs, one (block, segment) item each
    if (!ep) draw_segments(pp.RV, pp.grp[0].nb, grid, 32 * pn.warp0, pp.dec.nseg, pp.dec.seg_vec);
    const cudaError_t e = launch_pipe(&pn, ep ? nullptr : &pp, grid, st);
    if (e != cudaSuccess) return cuda_fail(e, "pipelined round launch");
    return SDD_OK;
}

}  // extern "C"
