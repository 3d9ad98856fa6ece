// Host side of libaloco: argument checks, the scalar Outer Optimizer
// Correction (Sec. 3.2; App. B.2-B.4), the per-device workspace, the launch
// of the fused pass and the finalisation of D_t and C_t
// (Eq. adaptive-h-core-diagnostics).
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <memory>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/aloco.h"
#include "aloco_internal.h"

namespace {

thread_local std::string t_err;

int fail(int code, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    t_err = buf;
    return code;
}

int cuda_fail(cudaError_t e, const char *what) {
    return fail(ALOCO_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorString(e),
                cudaGetErrorName(e));
}

// ------------------------------------------------------------- schedule

bool schedule_ok(const aloco_schedule_t *s, std::string *why) {
    if (!s) { *why = "schedule is NULL"; return false; }
    if (!(std::isfinite(s->peak_lr) && s->peak_lr >= 0.0)) {
        *why = "peak_lr must be finite and >= 0"; return false;
    }
    if (s->kind == ALOCO_SCHED_CONSTANT) return true;
    if (s->kind != ALOCO_SCHED_COSINE && s->kind != ALOCO_SCHED_LINEAR) {
        *why = "unknown schedule kind"; return false;
    }
    if (!(std::isfinite(s->final_lr) && s->final_lr >= 0.0)) {
        *why = "final_lr must be finite and >= 0"; return false;
    }
    if (s->warmup_steps < 0 || s->total_steps <= s->warmup_steps) {
        *why = "need 0 <= warmup_steps < total_steps"; return false;
    }
    return true;
}

// Inner learning rate at global step k (Tab. training settings).
double lr_at(const aloco_schedule_t &s, int64_t k) {
    if (s.kind == ALOCO_SCHED_CONSTANT) return s.peak_lr;
    if (k < s.warmup_steps)
        return s.peak_lr * (double)(k + 1) / (double)s.warmup_steps;
    if (k >= s.total_steps) return s.final_lr;
    const double f = (double)(k - s.warmup_steps) /
                     (double)(s.total_steps - s.warmup_steps);
    if (s.kind == ALOCO_SCHED_COSINE)
        return s.final_lr +
               0.5 * (s.peak_lr - s.final_lr) * (1.0 + std::cos(M_PI * f));
    return s.peak_lr + (s.final_lr - s.peak_lr) * f;
}

// sum_{h=1..H} lr(t0 + h - 1), Neumaier-compensated.  Segments where the
// rate is constant (constant schedule, the tail after total_steps) are
// summed as a product.
double lr_mass(const aloco_schedule_t &s, int64_t t0, int64_t H) {
    if (H <= 0) return 0.0;
    if (s.kind == ALOCO_SCHED_CONSTANT) return (double)H * s.peak_lr;
    const int64_t end = t0 + H;  // exclusive
    const int64_t vary_end = end < s.total_steps ? end : s.total_steps;
    double sum = 0.0, comp = 0.0;
    for (int64_t k = t0; k < vary_end; ++k) {
        const double x = lr_at(s, k);
        const double t = sum + x;
        comp += std::fabs(sum) >= std::fabs(x) ? (sum - t) + x : (x - t) + sum;
        sum = t;
    }
    const int64_t tail_begin = t0 > s.total_steps ? t0 : s.total_steps;
    if (end > tail_begin) {
        const double x = (double)(end - tail_begin) * s.final_lr;
        const double t = sum + x;
        comp += std::fabs(sum) >= std::fabs(x) ? (sum - t) + x : (x - t) + sum;
        sum = t;
    }
    return sum + comp;
}

// ----------------------------------------------------------- correction

int correction_impl(const aloco_schedule_t *sched, int64_t step,
                    int64_t H_sel, int64_t H_base, double outer_lr,
                    double outer_beta, const aloco_opts_t &o,
                    aloco_correction_t *out) {
    std::string why;
    if (!schedule_ok(sched, &why)) return fail(ALOCO_ERR_ARG, "%s", why.c_str());
    if (H_sel < 1 || H_base < 1)
        return fail(ALOCO_ERR_ARG, "H_sel (%lld) and H_base (%lld) must be >= 1",
                    (long long)H_sel, (long long)H_base);
    if (step < 0) return fail(ALOCO_ERR_ARG, "step must be >= 0");
    if (!std::isfinite(outer_lr)) return fail(ALOCO_ERR_ARG, "outer_lr must be finite");
    if (o.blocks_per_sm < 0)
        return fail(ALOCO_ERR_ARG, "blocks_per_sm must be >= 0");
    if (o.pass < ALOCO_PASS_AUTO || o.pass > ALOCO_PASS_TILE)
        return fail(ALOCO_ERR_ARG, "unknown pass %d", o.pass);
    if (o.mode != ALOCO_CORR_FULL && o.mode != ALOCO_CORR_MOMENTUM_ONLY &&
        o.mode != ALOCO_CORR_NONE)
        return fail(ALOCO_ERR_ARG, "unknown correction mode %d", o.mode);
    const bool beta_ok = o.mode == ALOCO_CORR_NONE
                             ? (outer_beta >= 0.0 && outer_beta < 1.0)
                             : (outer_beta > 0.0 && outer_beta < 1.0);
    if (!beta_ok)
        return fail(ALOCO_ERR_ARG, "outer_beta %g out of range for mode %d",
                    outer_beta, o.mode);
    if (!(o.eps > 0.0 && std::isfinite(o.eps)))
        return fail(ALOCO_ERR_ARG, "eps must be finite and > 0");
    if (!(o.mu_min >= 0.0 && o.mu_min <= o.mu_max && o.mu_max < 1.0))
        return fail(ALOCO_ERR_ARG, "need 0 <= mu_min <= mu_max < 1");
    if (!(o.kappa_max >= 1.0 && std::isfinite(o.kappa_max)))
        return fail(ALOCO_ERR_ARG, "kappa_max must be finite and >= 1");

    aloco_correction_t c;
    // Eq. app-outer-correction-lr-masses: both previews start at s_t = step.
    c.lam_sel = lr_mass(*sched, step, H_sel);
    c.lam_base = lr_mass(*sched, step, H_base);
    // Eq. app-outer-correction-ratios.
    c.rho_unc = c.lam_sel / (c.lam_base + o.eps);
    c.rho = std::fmax(c.rho_unc, 1.0);
    if (o.mode == ALOCO_CORR_NONE) {
        c.mu_t = outer_beta;
        c.kappa_t = 1.0;
        c.eta_out = outer_lr;
    } else {
        // Momentum retention mu_base^rho, clipped (Sec. 3.2; App. B.4).
        c.mu_t = std::fmin(std::fmax(std::pow(outer_beta, c.rho), o.mu_min),
                           o.mu_max);
        if (o.mode == ALOCO_CORR_MOMENTUM_ONLY) {
            c.kappa_t = 1.0;
            c.eta_out = outer_lr;
        } else {
            // Eq. app-outer-step-scale, Eq. app-adjusted-outer-learning-rate.
            c.kappa_t = std::fmin(c.rho, o.kappa_max);
            c.eta_out = outer_lr * c.kappa_t * (1.0 - c.mu_t) / (1.0 - outer_beta);
        }
    }
    // Eq. normalized-pseudo-gradient with rho + eps (App. B.3).
    c.inv_norm = o.normalize ? 1.0 / (c.rho + o.eps) : 1.0;
    *out = c;
    return ALOCO_OK;
}

// ------------------------------------------------------------ workspace

// Layout of the device workspace of one device (one allocation).
struct Workspace {
    std::mutex mu;
    bool ready = false;
    int device = -1;
    int sm_count = 0;
    int max_grid = 0;
    char *dev = nullptr;                  // device block
    double *partials = nullptr;           // [max_grid * (MAX_WORKERS + 1)]
    unsigned long long *nf_partials = nullptr;  // [max_grid]
    double *totals = nullptr;             // kTotalsSlots: totals, nf, error
    unsigned long long *nf_total = nullptr;
    unsigned int *error = nullptr;
    unsigned int *ticket = nullptr;
    double *adam = nullptr;               // AdamW: [max_grid] partials, then
                                          // [2 * MAX_WORKERS] norms and factors
    char *i8 = nullptr;                   // INT8 round scratch (grown on demand)
    size_t i8_cap = 0;
    double *host = nullptr;               // pinned readback of totals + nf
    // device-mapped page-locked page the round kernels publish their totals
    // and sequence number to (kTotals + 1 slots), and its device address
    double *stats_host = nullptr;
    double *stats_dev = nullptr;
    unsigned long long seq = 0;           // rounds launched on this workspace
    cudaEvent_t ev0 = nullptr, ev1 = nullptr;
    cudaEvent_t ev_block = nullptr;       // blocking-sync event (ALOCO_WAIT_BLOCK)
    // host-memory round (aloco_sync_host): staging slots and per-chunk totals
    char *hs = nullptr;                   // device, grown on demand
    size_t hs_cap = 0;
    double *hs_host = nullptr;            // pinned per-chunk totals
    size_t hs_host_cap = 0;               // doubles
    cudaStream_t hs_in = nullptr, hs_out = nullptr;
    cudaEvent_t hs_start = nullptr, hs_end = nullptr;
    cudaEvent_t hs_loaded[3] = {}, hs_computed[3] = {}, hs_free[3] = {};
};

constexpr int kTotals = aloco::kTotalsSlots;
// pinned read-back slots: the round's totals, or AdamW's norms and factors
constexpr int kHostSlots = kTotals > 2 * ALOCO_MAX_WORKERS ? kTotals : 2 * ALOCO_MAX_WORKERS;

std::mutex g_registry_mu;
std::vector<std::unique_ptr<Workspace>> g_registry;

Workspace *workspace_for(int device) {
    std::lock_guard<std::mutex> lk(g_registry_mu);
    if ((int)g_registry.size() <= device) g_registry.resize(device + 1);
    if (!g_registry[device]) g_registry[device].reset(new Workspace());
    return g_registry[device].get();
}

// Allocate on first use (caller holds ws->mu, device is current).
int ensure_ready(Workspace *ws, int device) {
    if (ws->ready) return ALOCO_OK;
    cudaError_t e = cudaDeviceGetAttribute(&ws->sm_count,
                                           cudaDevAttrMultiProcessorCount, device);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
    int max_threads = 0;
    e = cudaDeviceGetAttribute(&max_threads,
                               cudaDevAttrMaxThreadsPerMultiProcessor, device);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
    ws->max_grid = ws->sm_count * (max_threads / aloco::kBlock);
    const size_t n_part = (size_t)ws->max_grid * (ALOCO_MAX_WORKERS + 1);
    const size_t n_adam = (size_t)ws->max_grid + 2 * ALOCO_MAX_WORKERS;
    const size_t bytes = n_part * sizeof(double) +
                         (size_t)ws->max_grid * sizeof(unsigned long long) +
                         kTotals * sizeof(double) + n_adam * sizeof(double) + 256;
    e = cudaMalloc((void **)&ws->dev, bytes);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(ALOCO_ERR_NOMEM, "workspace cudaMalloc(%zu): %s", bytes,
                    cudaGetErrorString(e));
    }
    char *p = ws->dev;
    ws->partials = (double *)p;
    p += n_part * sizeof(double);
    ws->nf_partials = (unsigned long long *)p;
    p += (size_t)ws->max_grid * sizeof(unsigned long long);
    ws->totals = (double *)p;
    ws->nf_total = (unsigned long long *)(ws->totals + aloco::kNfSlot);
    ws->error = (unsigned int *)(ws->totals + aloco::kErrorSlot);
    p += kTotals * sizeof(double);
    ws->adam = (double *)p;
    p += n_adam * sizeof(double);
    ws->ticket = (unsigned int *)p;
    e = cudaMemset(ws->dev, 0, bytes);
    if (e == cudaSuccess) e = cudaMallocHost((void **)&ws->host, kHostSlots * sizeof(double));
    if (e == cudaSuccess)
        e = cudaHostAlloc((void **)&ws->stats_host, (kTotals + 1) * sizeof(double),
                          cudaHostAllocMapped);
    if (e == cudaSuccess) {
        std::memset(ws->stats_host, 0, (kTotals + 1) * sizeof(double));
        e = cudaHostGetDevicePointer((void **)&ws->stats_dev, ws->stats_host, 0);
    }
    if (e == cudaSuccess) e = cudaEventCreate(&ws->ev0);
    if (e == cudaSuccess) e = cudaEventCreate(&ws->ev1);
    if (e == cudaSuccess)
        e = cudaEventCreateWithFlags(&ws->ev_block,
                                     cudaEventBlockingSync | cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        cudaGetLastError();
        return cuda_fail(e, "workspace setup");
    }
    ws->device = device;
    ws->ready = true;
    return ALOCO_OK;
}

// Wait until the round kernel has published round `seq` to `page` (see
// SyncArgs::stats_out).  The last block publishes after every block's
// outputs are written, so on return the outputs are complete, and work
// queued later on the stream runs after the kernel.  The stream is polled
// every few hundred reads: a launch that fails or ends without publishing
// returns an error instead of waiting on.
int wait_published(const double *page, unsigned long long seq, cudaStream_t stream) {
    const volatile unsigned long long *flag =
        reinterpret_cast<const volatile unsigned long long *>(page + aloco::kSeqSlot);
    for (unsigned it = 1;; ++it) {
        if (*flag == seq) break;
        if ((it & 255) == 0) {
            const cudaError_t q = cudaStreamQuery(stream);
            if (q == cudaErrorNotReady) continue;
            if (q != cudaSuccess) return cuda_fail(q, "round");
            if (*flag == seq) break;
            return fail(ALOCO_ERR_CUDA, "the round ended without publishing its statistics");
        }
    }
    std::atomic_thread_fence(std::memory_order_acquire);
    return ALOCO_OK;
}

// ALOCO_WAIT_BLOCK: sleep on a blocking-sync event recorded behind the
// kernel, then check that the round published its statistics.
int wait_blocking(const double *page, unsigned long long seq, cudaStream_t stream,
                  cudaEvent_t ev) {
    cudaError_t e = cudaEventRecord(ev, stream);
    if (e == cudaSuccess) e = cudaEventSynchronize(ev);
    if (e != cudaSuccess) return cuda_fail(e, "round");
    std::atomic_thread_fence(std::memory_order_acquire);
    const volatile unsigned long long *flag =
        reinterpret_cast<const volatile unsigned long long *>(page + aloco::kSeqSlot);
    if (*flag != seq)
        return fail(ALOCO_ERR_CUDA, "the round ended without publishing its statistics");
    return ALOCO_OK;
}

// --------------------------------------------------------- buffer checks

typedef CUresult (*GetAddressRangeFn)(CUdeviceptr *, size_t *, CUdeviceptr);

GetAddressRangeFn address_range_fn() {
    static GetAddressRangeFn fn = [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuMemGetAddressRange", &p, 12000,
                                             cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess) {
            cudaGetLastError();
            return (GetAddressRangeFn) nullptr;
        }
        return (GetAddressRangeFn)p;
    }();
    return fn;
}

}  // namespace

// Helpers with external linkage: also used by the allocation-free entry
// point (aloco_noalloc.cu).
// Testing hook of aloco_test_stall_tile: consumed by the calling thread's
// next bulk-copy, tile or fused INT8 round.
thread_local int64_t t_test_stall_tile1 = 0;

namespace aloco {

bool use_int8_fused(int pass, int M, aloco_dtype dtype) {
    if (!int8_fused_fits(M, dtype)) return false;
    if (pass == ALOCO_PASS_INT8_FUSED) return true;
    if (pass == ALOCO_PASS_INT8_SPLIT) return false;
    return true;  // AUTO
}


bool use_tile(int pass, int M, aloco_dtype dtype, int64_t n, int64_t nvec) {
    if (!sync_tile_fits(M, n, nvec)) return false;
    if (pass == ALOCO_PASS_TILE) return true;
    if (pass != ALOCO_PASS_AUTO) return false;
    // AUTO, as measured on GB300 (fraction of the measured copy peak): from
    // 2^27 parameters the tile pass leads for bf16 replicas (0.97-0.98
    // against 0.94) and for fp32 with M = 1 or M >= 5 (0.96-0.98 against
    // 0.94-0.95); at fp32 M = 2..4 the two passes tie within 0.5 %.  On
    // smaller rounds the CTAs of the tile pass move through their blocks in
    // step, so HBM idles while they compute, and the register pass leads.
    // M = 9..16 from 2^27 too: fp32 0.99-1.00 against 0.95-0.97 (M >= 12),
    // bf16 0.96-0.97 against 0.955-0.963 (M <= 12); bf16 M >= 13 spills
    // registers in the tile pass and stays on the register pass.
    if (n < ((int64_t)1 << 27)) return false;
    if (dtype == ALOCO_BF16) return M <= 12;
    return M == 1 || M >= 5;
}

bool use_tma(int pass, int M, aloco_dtype dtype, int64_t nvec) {
    if (M < 1 || M > 16 || nvec < kTmaTilePacks) return false;
    if (pass == ALOCO_PASS_BULK_COPY) return true;
    if (pass == ALOCO_PASS_REGISTERS) return false;
    // AUTO: on GB300 the tuned register-streaming pass matched or beat the
    // bulk-copy ring on every full-size workload measured (150M x 8 fp32:
    // 0.94 against 0.92 of the measured copy peak; 3B x 8 bf16: 0.94 each).
    (void)dtype;
    return false;
}

// Record an error message for aloco_last_error() and return `code`.
int report_error(int code, const char *msg) { return fail(code, "%s", msg); }

// The buffer must be device (or managed) memory of `device`, and when the
// driver can tell, [p, p + bytes) must lie inside one allocation.
int check_buffer(const void *p, size_t bytes, int device, const char *name) {
    cudaPointerAttributes at;
    cudaError_t e = cudaPointerGetAttributes(&at, p);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(ALOCO_ERR_ARG, "%s: not a CUDA pointer (%s)", name,
                    cudaGetErrorString(e));
    }
    if (at.type != cudaMemoryTypeDevice && at.type != cudaMemoryTypeManaged)
        return fail(ALOCO_ERR_ARG, "%s: not device memory", name);
    if (at.type == cudaMemoryTypeDevice && at.device != device)
        return fail(ALOCO_ERR_ARG, "%s: lives on device %d, current device is %d",
                    name, at.device, device);
    if (GetAddressRangeFn fn = address_range_fn()) {
        CUdeviceptr base = 0;
        size_t size = 0;
        if (fn(&base, &size, (CUdeviceptr)p) == CUDA_SUCCESS && size > 0) {
            if ((uintptr_t)p + bytes > (uintptr_t)base + size)
                return fail(ALOCO_ERR_ARG,
                            "%s: %zu bytes from %p run past the end of its "
                            "allocation (%zu bytes at %p)",
                            name, bytes, p, size, (void *)base);
        }
    }
    return ALOCO_OK;
}

void fill_default_opts(aloco_opts_t *o) {
    std::memset(o, 0, sizeof *o);
    o->mu_min = 0.45;
    o->mu_max = 0.90;
    o->kappa_max = 1.6;
    o->eps = 1e-8;
    o->normalize = 0;
    o->mode = ALOCO_CORR_FULL;
    o->time_kernel = 0;
    o->blocks_per_sm = 0;
    o->stream = nullptr;
    o->pass = ALOCO_PASS_AUTO;
    o->wait = ALOCO_WAIT_SPIN;
}

// x ~= hi + lo with hi = fl32(x), lo = fl32(x - hi).
void split_coef(double x, float *hi, float *lo) {
    *hi = (float)x;
    *lo = (float)(x - (double)*hi);
}

void finalize_stats(const double *totals, unsigned long long nf, int M,
                    double eps, double b_scale, aloco_stats_t *st) {
    double sum = 0.0;
    for (int m = 0; m < M; ++m) {
        st->drift[m] = totals[m];
        sum += totals[m];
    }
    st->D = sum / (double)M;
    st->mean_sq_norm = totals[M] * b_scale;
    st->C = (double)M * st->mean_sq_norm / (st->D + eps);
    st->nonfinite = (int64_t)nf;
}

}  // namespace aloco

using aloco::check_buffer;
using aloco::fill_default_opts;
using aloco::finalize_stats;
using aloco::split_coef;

// ================================================================ C ABI

extern "C" {

void aloco_default_opts(aloco_opts_t *opts) {
    if (opts) fill_default_opts(opts);
}

double aloco_inner_lr_accum(const aloco_schedule_t *schedule, int64_t t0,
                            int64_t H) {
    std::string why;
    if (!schedule_ok(schedule, &why) || t0 < 0 || H < 0) {
        fail(ALOCO_ERR_ARG, "aloco_inner_lr_accum: %s",
             why.empty() ? "t0 and H must be >= 0" : why.c_str());
        return std::nan("");
    }
    return lr_mass(*schedule, t0, H);
}

int aloco_correction(const aloco_schedule_t *schedule, int64_t step,
                     int64_t H_sel, int64_t H_base, double outer_lr,
                     double outer_beta, const aloco_opts_t *opts,
                     aloco_correction_t *out) {
    aloco_opts_t o;
    if (opts) o = *opts; else fill_default_opts(&o);
    if (!out) return fail(ALOCO_ERR_ARG, "out is NULL");
    return correction_impl(schedule, step, H_sel, H_base, outer_lr, outer_beta,
                           o, out);
}

int aloco_sync(float *global, float *momentum, void *const *locals, size_t N,
               int M, aloco_dtype dtype, int64_t H_sel, int64_t H_base,
               int64_t step, const aloco_schedule_t *schedule, double outer_lr,
               double outer_beta, aloco_stats_t *stats_out) {
    return aloco_sync_ex(global, momentum, locals, N, M, dtype, H_sel, H_base,
                         step, schedule, outer_lr, outer_beta, nullptr,
                         stats_out);
}

}  // extern "C"

namespace {

// Build the part table of an INT8 round (NULL parts: one part of N).
int build_parts(const int64_t *parts, int n_parts, size_t N, aloco::Int8Parts *P) {
    if (!parts) {
        n_parts = 1;
    } else if (n_parts < 1 || n_parts > aloco::kInt8MaxParts) {
        return fail(ALOCO_ERR_ARG, "n_parts = %d outside [1, %d]", n_parts,
                    aloco::kInt8MaxParts);
    }
    P->n_parts = n_parts;
    P->off[0] = 0;
    P->blk[0] = 0;
    for (int p = 0; p < n_parts; ++p) {
        const int64_t sz = parts ? parts[p] : (int64_t)N;
        if (sz < 1) return fail(ALOCO_ERR_ARG, "part %d has size %lld", p, (long long)sz);
        P->off[p + 1] = P->off[p] + sz;
        P->blk[p + 1] = P->blk[p] + (sz + 4095) / 4096;
    }
    if ((size_t)P->off[n_parts] != N)
        return fail(ALOCO_ERR_ARG, "parts add up to %lld, not N = %zu",
                    (long long)P->off[n_parts], N);
    return ALOCO_OK;
}

// The partials of a shard from the round's totals block.
void fill_partials(const double *totals, unsigned long long nf, int M, double eps,
                   double sq_scale, const aloco_correction_t &corr, int64_t n,
                   aloco_partials_t *p) {
    std::memset(p, 0, sizeof *p);
    for (int m = 0; m < M; ++m) p->drift[m] = totals ? totals[m] : 0.0;
    p->sum_sq = totals ? totals[M] : 0.0;
    p->sq_scale = sq_scale;
    p->eps = eps;
    p->corr = corr;
    p->nonfinite = (int64_t)nf;
    p->n = n;
    p->M = M;
    p->kernel_ms = -1.f;
}

// One round: the plain pass (parts == NULL && !int8) or the INT8-
// communicated pass.  With partials_out, the round's totals are returned
// as a shard's partial sums instead of being finished into D and C.
int sync_impl(float *global, float *momentum, void *const *locals, size_t N,
              int M, aloco_dtype dtype, int64_t H_sel, int64_t H_base,
              int64_t step, const aloco_schedule_t *schedule, double outer_lr,
              double outer_beta, bool int8, const int64_t *parts, int n_parts,
              const aloco_opts_t *opts, aloco_stats_t *stats_out,
              aloco_partials_t *partials_out = nullptr) {
    aloco_opts_t o;
    if (opts) o = *opts; else fill_default_opts(&o);
    aloco_stats_t local_stats;
    aloco_stats_t *st = stats_out ? stats_out : &local_stats;
    if (o.wait != ALOCO_WAIT_SPIN && o.wait != ALOCO_WAIT_BLOCK)
        return fail(ALOCO_ERR_ARG, "unknown wait mode %d", o.wait);

    // ---------------------------------------------------- arguments
    if (M < 1 || M > (int8 ? 16 : ALOCO_MAX_WORKERS))
        return fail(ALOCO_ERR_ARG, "M = %d outside [1, %d]", M,
                    int8 ? 16 : ALOCO_MAX_WORKERS);
    if (dtype != ALOCO_F32 && dtype != ALOCO_BF16)
        return fail(ALOCO_ERR_ARG, "unknown replica dtype %d", (int)dtype);
    const bool int8_pass = o.pass == ALOCO_PASS_INT8_SPLIT || o.pass == ALOCO_PASS_INT8_FUSED;
    if (int8 ? (o.pass == ALOCO_PASS_REGISTERS || o.pass == ALOCO_PASS_BULK_COPY ||
                o.pass == ALOCO_PASS_TILE)
             : int8_pass)
        return fail(ALOCO_ERR_ARG, "pass %d does not apply to this round", o.pass);
    if (int8 && o.pass == ALOCO_PASS_INT8_FUSED && !aloco::int8_fused_fits(M, dtype))
        return fail(ALOCO_ERR_ARG, "the fused INT8 round takes M <= 16");
    if (N > (size_t)INT64_MAX / 8) return fail(ALOCO_ERR_ARG, "N too large");
    if (N > 0 && (!global || !momentum || !locals))
        return fail(ALOCO_ERR_ARG, "NULL buffer");
    for (int m = 0; N > 0 && m < M; ++m)
        if (!locals[m]) return fail(ALOCO_ERR_ARG, "locals[%d] is NULL", m);
    aloco_correction_t corr;
    int rc = correction_impl(schedule, step, H_sel, H_base, outer_lr,
                             outer_beta, o, &corr);
    if (rc != ALOCO_OK) return rc;

    static thread_local aloco::Int8Parts P;
    if (int8 && (rc = build_parts(parts, n_parts, N, &P)) != ALOCO_OK) return rc;

    std::memset(st, 0, sizeof *st);
    st->corr = corr;
    st->M = M;
    st->kernel_ms = -1.f;
    const double sq_scale = int8 ? 1.0 : 1.0 / ((double)M * (double)M);
    if (N == 0) {
        if (partials_out) fill_partials(nullptr, 0, M, o.eps, sq_scale, corr, 0, partials_out);
        t_err.clear();
        return ALOCO_OK;
    }

    const size_t rsz = dtype == ALOCO_F32 ? 4 : 2;
    // Pairwise overlap check of the M + 2 byte ranges.
    {
        std::vector<std::pair<uintptr_t, size_t>> r;
        r.push_back({(uintptr_t)global, N * 4});
        r.push_back({(uintptr_t)momentum, N * 4});
        for (int m = 0; m < M; ++m) r.push_back({(uintptr_t)locals[m], N * rsz});
        for (size_t i = 0; i < r.size(); ++i)
            for (size_t j = i + 1; j < r.size(); ++j)
                if (r[i].first < r[j].first + r[j].second &&
                    r[j].first < r[i].first + r[i].second)
                    return fail(ALOCO_ERR_ALIAS, "buffers %zu and %zu overlap", i, j);
    }
    if (((uintptr_t)global | (uintptr_t)momentum) & 3)
        return fail(ALOCO_ERR_ARG, "global/momentum not 4-byte aligned");
    for (int m = 0; m < M; ++m)
        if ((uintptr_t)locals[m] & (rsz - 1))
            return fail(ALOCO_ERR_ARG, "locals[%d] not %zu-byte aligned", m, rsz);

    int device = 0;
    cudaError_t e = cudaGetDevice(&device);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    Workspace *ws = workspace_for(device);
    std::lock_guard<std::mutex> lk(ws->mu);
    rc = ensure_ready(ws, device);
    if (rc != ALOCO_OK) return rc;

    if ((rc = check_buffer(global, N * 4, device, "global")) != ALOCO_OK) return rc;
    if ((rc = check_buffer(momentum, N * 4, device, "momentum")) != ALOCO_OK) return rc;
    for (int m = 0; m < M; ++m) {
        char name[32];
        snprintf(name, sizeof name, "locals[%d]", m);
        if ((rc = check_buffer(locals[m], N * rsz, device, name)) != ALOCO_OK)
            return rc;
    }

    // ------------------------------------------------------- launch
    aloco::SyncArgs a;
    std::memset(&a, 0, sizeof a);
    a.g = global;
    a.v = momentum;
    uintptr_t align_or = (uintptr_t)global | (uintptr_t)momentum;
    for (int m = 0; m < M; ++m) {
        a.x[m] = locals[m];
        align_or |= (uintptr_t)locals[m];
    }
    const int pack = aloco::pack_elems(dtype);
    a.n = (int64_t)N;
    a.nvec = (align_or & 15) == 0 ? (int64_t)(N / pack) : 0;
    // plain pass: Dtil = (inv/M) sum_m Delta_m; INT8 pass: Dtil = inv * mean
    split_coef(int8 ? corr.inv_norm : corr.inv_norm / (double)M, &a.c_hi, &a.c_lo);
    split_coef(corr.mu_t, &a.mu_hi, &a.mu_lo);
    split_coef(-corr.eta_out, &a.neg_eta_hi, &a.neg_eta_lo);
    a.M = M;
    a.partials = ws->partials;
    a.nf_partials = ws->nf_partials;
    a.ticket = ws->ticket;
    a.totals = ws->totals;
    a.nf_total = ws->nf_total;

    const int64_t work = a.nvec > 0 ? a.nvec : a.n;
    aloco::LaunchPlan plan;
    const bool tile = !int8 && aloco::use_tile(o.pass, M, dtype, a.n, a.nvec);
    const bool tma = !int8 && !tile && aloco::use_tma(o.pass, M, dtype, a.nvec);
    const bool fused = int8 && aloco::use_int8_fused(o.pass, M, dtype);
    if (fused || tile) {
        plan.grid = 0;
        plan.block = 0;
        plan.kernel = nullptr;
    } else if (int8) {
        // scratch of the two INT8 passes: per-block worker scales and the
        // per-CTA drift energies of pass 1 (grown on demand, kept cached)
        const size_t need = (size_t)P.blk[P.n_parts] * M * sizeof(float) + 256 +
                            (size_t)ws->max_grid * 16 * sizeof(double);
        if (ws->i8_cap < need) {
            if (ws->i8) cudaFree(ws->i8);
            ws->i8 = nullptr;
            ws->i8_cap = 0;
            e = cudaMalloc((void **)&ws->i8, need);
            if (e != cudaSuccess) {
                cudaGetLastError();
                return fail(ALOCO_ERR_NOMEM, "INT8 scratch cudaMalloc(%zu): %s", need,
                            cudaGetErrorString(e));
            }
            ws->i8_cap = need;
        }
        plan.grid = 0;
        plan.block = 0;
        plan.kernel = nullptr;
    } else if (tma)
        e = dtype == ALOCO_F32 ? aloco::plan_sync_tma_f32(M, a.nvec, ws->sm_count, &plan)
                               : aloco::plan_sync_tma_bf16(M, a.nvec, ws->sm_count, &plan);
    else
        e = dtype == ALOCO_F32
                ? aloco::plan_sync_f32(M, work, ws->sm_count, o.blocks_per_sm, &plan)
                : aloco::plan_sync_bf16(M, work, ws->sm_count, o.blocks_per_sm, &plan);
    if (e != cudaSuccess) return cuda_fail(e, "launch plan");
    a.n_tiles = plan.tiles;
    a.stages = plan.stages;
    a.error = ws->error;
    a.stats_out = ws->stats_dev;
    a.seq = ++ws->seq;
    if (tma || fused || tile) {
        a.test_stall_tile1 = t_test_stall_tile1;
        t_test_stall_tile1 = 0;
    }
    if (plan.grid > ws->max_grid)
        return fail(ALOCO_ERR_CUDA, "grid %d exceeds workspace %d", plan.grid,
                    ws->max_grid);

    cudaStream_t stream = (cudaStream_t)o.stream;
    if (o.time_kernel && (e = cudaEventRecord(ws->ev0, stream)) != cudaSuccess)
        return cuda_fail(e, "cudaEventRecord");
    if (fused) {
        e = aloco::launch_int8_fused(a, P, dtype, ws->sm_count, ws->max_grid, stream,
                                     &plan.grid);
    } else if (tile) {
        e = aloco::launch_sync_tile(a, dtype, ws->sm_count, ws->max_grid, stream, &plan.grid);
    } else if (int8) {
        double *e_rows = reinterpret_cast<double *>(ws->i8);
        unsigned *bmax = reinterpret_cast<unsigned *>(
            ws->i8 + (size_t)ws->max_grid * 16 * sizeof(double));
        e = aloco::launch_int8_round(a, P, dtype, ws->sm_count, bmax, e_rows,
                                     ws->max_grid, stream, &plan.grid);
    } else {
        void *params[] = {&a};
        e = cudaLaunchKernel(plan.kernel, dim3(plan.grid), dim3(plan.block), params,
                             plan.smem, stream);
    }
    if (e != cudaSuccess) return cuda_fail(e, "fused sync launch");
    if (o.time_kernel && (e = cudaEventRecord(ws->ev1, stream)) != cudaSuccess)
        return cuda_fail(e, "cudaEventRecord");
    rc = o.wait == ALOCO_WAIT_BLOCK
             ? wait_blocking(ws->stats_host, a.seq, stream, ws->ev_block)
             : wait_published(ws->stats_host, a.seq, stream);
    if (rc != ALOCO_OK) return rc;

    unsigned long long nf;
    std::memcpy(&nf, ws->stats_host + aloco::kNfSlot, sizeof nf);
    unsigned int perr;
    std::memcpy(&perr, ws->stats_host + aloco::kErrorSlot, sizeof perr);
    if (perr != 0) {
        cudaMemsetAsync(ws->error, 0, sizeof(unsigned int), stream);
        cudaStreamSynchronize(stream);
        cudaGetLastError();
        return fail(ALOCO_ERR_CUDA,
                    "bulk-copy pipeline wait timed out; outputs are incomplete");
    }
    finalize_stats(ws->stats_host, nf, M, o.eps, sq_scale, st);
    st->grid = plan.grid;
    st->pass_used = fused ? ALOCO_PASS_INT8_FUSED
                    : int8 ? ALOCO_PASS_INT8_SPLIT
                    : tile ? ALOCO_PASS_TILE
                    : tma  ? ALOCO_PASS_BULK_COPY
                           : ALOCO_PASS_REGISTERS;
    if (o.time_kernel) {
        float ms = -1.f;
        if (cudaEventSynchronize(ws->ev1) == cudaSuccess &&
            cudaEventElapsedTime(&ms, ws->ev0, ws->ev1) == cudaSuccess)
            st->kernel_ms = ms;
        else
            cudaGetLastError();
    }
    if (partials_out) {
        fill_partials(ws->stats_host, nf, M, o.eps, sq_scale, corr, (int64_t)N,
                      partials_out);
        partials_out->pass_used = st->pass_used;
        partials_out->kernel_ms = st->kernel_ms;
        if (nf > 0)
            return fail(ALOCO_ERR_NONFINITE, "shard produced %llu non-finite elements", nf);
        t_err.clear();
        return ALOCO_OK;
    }
    if (st->nonfinite > 0 || !std::isfinite(st->D) || !std::isfinite(st->C))
        return fail(ALOCO_ERR_NONFINITE,
                    "round produced %lld non-finite elements (D=%g, C=%g)",
                    (long long)st->nonfinite, st->D, st->C);
    t_err.clear();
    return ALOCO_OK;
}

}  // namespace

extern "C" {

int aloco_sync_ex(float *global, float *momentum, void *const *locals,
                  size_t N, int M, aloco_dtype dtype, int64_t H_sel,
                  int64_t H_base, int64_t step,
                  const aloco_schedule_t *schedule, double outer_lr,
                  double outer_beta, const aloco_opts_t *opts,
                  aloco_stats_t *stats_out) {
    return sync_impl(global, momentum, locals, N, M, dtype, H_sel, H_base, step,
                     schedule, outer_lr, outer_beta, false, nullptr, 0, opts,
                     stats_out);
}

int aloco_sync_int8(float *global, float *momentum, void *const *locals,
                    size_t N, int M, aloco_dtype dtype, int64_t H_sel,
                    int64_t H_base, int64_t step,
                    const aloco_schedule_t *schedule, double outer_lr,
                    double outer_beta, const int64_t *part_sizes, int n_parts,
                    const aloco_opts_t *opts, aloco_stats_t *stats_out) {
    return sync_impl(global, momentum, locals, N, M, dtype, H_sel, H_base, step,
                     schedule, outer_lr, outer_beta, true, part_sizes, n_parts,
                     opts, stats_out);
}

int aloco_sync_shard(float *global, float *momentum, void *const *locals,
                     size_t n_shard, int M, aloco_dtype dtype, int64_t H_sel,
                     int64_t H_base, int64_t step, const aloco_schedule_t *schedule,
                     double outer_lr, double outer_beta, const aloco_opts_t *opts,
                     aloco_partials_t *partials_out) {
    if (!partials_out) return fail(ALOCO_ERR_ARG, "partials_out is NULL");
    aloco_stats_t st;
    return sync_impl(global, momentum, locals, n_shard, M, dtype, H_sel, H_base, step,
                     schedule, outer_lr, outer_beta, false, nullptr, 0, opts, &st,
                     partials_out);
}

int aloco_sync_int8_shard(float *global, float *momentum, void *const *locals,
                          size_t n_shard, int M, aloco_dtype dtype, int64_t H_sel,
                          int64_t H_base, int64_t step, const aloco_schedule_t *schedule,
                          double outer_lr, double outer_beta, const int64_t *part_sizes,
                          int n_parts, const aloco_opts_t *opts,
                          aloco_partials_t *partials_out) {
    if (!partials_out) return fail(ALOCO_ERR_ARG, "partials_out is NULL");
    aloco_stats_t st;
    return sync_impl(global, momentum, locals, n_shard, M, dtype, H_sel, H_base, step,
                     schedule, outer_lr, outer_beta, true, part_sizes, n_parts, opts, &st,
                     partials_out);
}

int aloco_combine_partials(const aloco_partials_t *shards, int n_shards,
                           aloco_stats_t *stats_out) {
    if (!shards || n_shards < 1) return fail(ALOCO_ERR_ARG, "need n_shards >= 1 partials");
    if (!stats_out) return fail(ALOCO_ERR_ARG, "stats_out is NULL");
    const aloco_partials_t &p0 = shards[0];
    const int M = p0.M;
    if (M < 1 || M > ALOCO_MAX_WORKERS)
        return fail(ALOCO_ERR_ARG, "shard 0: M = %d outside [1, %d]", M, ALOCO_MAX_WORKERS);
    for (int k = 1; k < n_shards; ++k) {
        const aloco_partials_t &p = shards[k];
        if (p.M != M || p.eps != p0.eps || p.sq_scale != p0.sq_scale ||
            std::memcmp(&p.corr, &p0.corr, sizeof p.corr) != 0)
            return fail(ALOCO_ERR_ARG,
                        "shard %d does not belong to the round of shard 0 (M, eps, "
                        "aggregate scale or correction context differ)", k);
    }
    // fixed shard order: every holder adds the same values in the same order
    double tot[ALOCO_MAX_WORKERS + 1] = {};
    unsigned long long nf = 0;
    float ms = -1.f;
    int pass_used = 0;
    for (int k = 0; k < n_shards; ++k) {
        const aloco_partials_t &p = shards[k];
        if (p.nonfinite < 0) return fail(ALOCO_ERR_ARG, "shard %d: negative count", k);
        for (int m = 0; m < M; ++m) tot[m] += p.drift[m];
        tot[M] += p.sum_sq;
        nf += (unsigned long long)p.nonfinite;
        if (p.kernel_ms > ms) ms = p.kernel_ms;
        if (!pass_used && p.n > 0) pass_used = p.pass_used;
    }
    std::memset(stats_out, 0, sizeof *stats_out);
    finalize_stats(tot, nf, M, p0.eps, p0.sq_scale, stats_out);
    stats_out->corr = p0.corr;
    stats_out->M = M;
    stats_out->grid = n_shards;
    stats_out->kernel_ms = ms;
    stats_out->pass_used = pass_used;
    if (stats_out->nonfinite > 0 || !std::isfinite(stats_out->D) ||
        !std::isfinite(stats_out->C))
        return fail(ALOCO_ERR_NONFINITE,
                    "combined round has %lld non-finite elements (D=%g, C=%g)",
                    (long long)stats_out->nonfinite, stats_out->D, stats_out->C);
    t_err.clear();
    return ALOCO_OK;
}

int64_t aloco_int8_num_blocks(const int64_t *part_sizes, int n_parts) {
    if (!part_sizes || n_parts < 1) {
        fail(ALOCO_ERR_ARG, "part_sizes is NULL or n_parts < 1");
        return -1;
    }
    int64_t nb = 0;
    for (int p = 0; p < n_parts; ++p) {
        if (part_sizes[p] < 1) {
            fail(ALOCO_ERR_ARG, "part %d has size %lld", p, (long long)part_sizes[p]);
            return -1;
        }
        nb += (part_sizes[p] + 4095) / 4096;
    }
    return nb;
}

}  // extern "C"

namespace {

// Common set-up of the stand-alone codec calls.
int codec_setup(size_t N, const int64_t *parts, int n_parts, aloco::Int8Parts *P,
                int *sm_count) {
    if (N == 0) return fail(ALOCO_ERR_ARG, "N must be >= 1");
    int rc = build_parts(parts, n_parts, N, P);
    if (rc != ALOCO_OK) return rc;
    int device = 0;
    cudaError_t e = cudaGetDevice(&device);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    e = cudaDeviceGetAttribute(sm_count, cudaDevAttrMultiProcessorCount, device);
    if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
    return ALOCO_OK;
}

}  // namespace

extern "C" {

int aloco_int8_encode(const float *x, size_t N, const int64_t *part_sizes,
                      int n_parts, int8_t *codes, float *scales, float *decoded,
                      void *stream) {
    if (!x || !codes || !scales) return fail(ALOCO_ERR_ARG, "NULL buffer");
    static thread_local aloco::Int8Parts P;
    int sms = 0;
    int rc = codec_setup(N, part_sizes, n_parts, &P, &sms);
    if (rc != ALOCO_OK) return rc;
    int device = 0;
    cudaGetDevice(&device);
    if ((rc = check_buffer(x, N * 4, device, "x")) != ALOCO_OK) return rc;
    if ((rc = check_buffer(codes, N, device, "codes")) != ALOCO_OK) return rc;
    if ((rc = check_buffer(scales, (size_t)P.blk[P.n_parts] * 4, device, "scales")) != ALOCO_OK)
        return rc;
    if (decoded && (rc = check_buffer(decoded, N * 4, device, "decoded")) != ALOCO_OK)
        return rc;
    const bool vec = (((uintptr_t)x | (uintptr_t)decoded) & 15) == 0 &&
                     ((uintptr_t)codes & 3) == 0;
    cudaError_t e = aloco::launch_int8_encode(x, codes, scales, decoded, vec, P, sms,
                                              (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "int8 encode launch");
    t_err.clear();
    return ALOCO_OK;
}

int aloco_int8_decode(const int8_t *codes, const float *scales, size_t N,
                      const int64_t *part_sizes, int n_parts, float *out,
                      void *stream) {
    if (!codes || !scales || !out) return fail(ALOCO_ERR_ARG, "NULL buffer");
    static thread_local aloco::Int8Parts P;
    int sms = 0;
    int rc = codec_setup(N, part_sizes, n_parts, &P, &sms);
    if (rc != ALOCO_OK) return rc;
    int device = 0;
    cudaGetDevice(&device);
    if ((rc = check_buffer(codes, N, device, "codes")) != ALOCO_OK) return rc;
    if ((rc = check_buffer(scales, (size_t)P.blk[P.n_parts] * 4, device, "scales")) != ALOCO_OK)
        return rc;
    if ((rc = check_buffer(out, N * 4, device, "out")) != ALOCO_OK) return rc;
    const bool vec = ((uintptr_t)out & 15) == 0 && ((uintptr_t)codes & 3) == 0;
    cudaError_t e = aloco::launch_int8_decode(codes, scales, out, vec, P, sms,
                                              (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, "int8 decode launch");
    t_err.clear();
    return ALOCO_OK;
}

int aloco_sync_host(float *global, float *momentum, const void *const *locals,
                    size_t N, int M, aloco_dtype dtype, int64_t H_sel,
                    int64_t H_base, int64_t step, const aloco_schedule_t *schedule,
                    double outer_lr, double outer_beta, size_t chunk_elems,
                    const aloco_opts_t *opts, aloco_stats_t *stats_out) {
    constexpr int kSlots = 3;
    aloco_opts_t o;
    if (opts) o = *opts; else fill_default_opts(&o);
    aloco_stats_t local_stats;
    aloco_stats_t *st = stats_out ? stats_out : &local_stats;
    if (M < 1 || M > ALOCO_MAX_WORKERS)
        return fail(ALOCO_ERR_ARG, "M = %d outside [1, %d]", M, ALOCO_MAX_WORKERS);
    if (dtype != ALOCO_F32 && dtype != ALOCO_BF16)
        return fail(ALOCO_ERR_ARG, "unknown replica dtype %d", (int)dtype);
    if (o.pass != ALOCO_PASS_AUTO && o.pass != ALOCO_PASS_REGISTERS)
        return fail(ALOCO_ERR_ARG, "the host-memory round runs the register pass; pass %d "
                    "does not apply", o.pass);
    if (N > (size_t)INT64_MAX / 8) return fail(ALOCO_ERR_ARG, "N too large");
    if (N > 0 && (!global || !momentum || !locals))
        return fail(ALOCO_ERR_ARG, "NULL buffer");
    for (int m = 0; N > 0 && m < M; ++m)
        if (!locals[m]) return fail(ALOCO_ERR_ARG, "locals[%d] is NULL", m);
    aloco_correction_t corr;
    int rc = correction_impl(schedule, step, H_sel, H_base, outer_lr, outer_beta, o, &corr);
    if (rc != ALOCO_OK) return rc;
    std::memset(st, 0, sizeof *st);
    st->corr = corr;
    st->M = M;
    st->kernel_ms = -1.f;
    if (N == 0) {
        t_err.clear();
        return ALOCO_OK;
    }
    const size_t rsz = dtype == ALOCO_F32 ? 4 : 2;
    {
        std::vector<std::pair<uintptr_t, size_t>> r;
        r.push_back({(uintptr_t)global, N * 4});
        r.push_back({(uintptr_t)momentum, N * 4});
        for (int m = 0; m < M; ++m) r.push_back({(uintptr_t)locals[m], N * rsz});
        for (size_t i = 0; i < r.size(); ++i)
            for (size_t j = i + 1; j < r.size(); ++j)
                if (r[i].first < r[j].first + r[j].second &&
                    r[j].first < r[i].first + r[i].second)
                    return fail(ALOCO_ERR_ALIAS, "buffers %zu and %zu overlap", i, j);
    }
    if (((uintptr_t)global | (uintptr_t)momentum) & 3)
        return fail(ALOCO_ERR_ARG, "global/momentum not 4-byte aligned");
    for (int m = 0; m < M; ++m)
        if ((uintptr_t)locals[m] & (rsz - 1))
            return fail(ALOCO_ERR_ARG, "locals[%d] not %zu-byte aligned", m, rsz);
    {
        const void *ptrs[2 + ALOCO_MAX_WORKERS] = {global, momentum};
        for (int m = 0; m < M; ++m) ptrs[2 + m] = locals[m];
        for (int i = 0; i < M + 2; ++i) {
            cudaPointerAttributes at;
            cudaError_t e = cudaPointerGetAttributes(&at, ptrs[i]);
            if (e != cudaSuccess) cudaGetLastError();
            if (e != cudaSuccess || at.type != cudaMemoryTypeHost)
                return fail(ALOCO_ERR_ARG,
                            "buffer %d is not page-locked host memory (allocate it with "
                            "cudaMallocHost or register it with cudaHostRegister)", i);
        }
    }
    size_t chunk = chunk_elems ? chunk_elems : ((size_t)1 << 24);
    chunk = (chunk + 7) / 8 * 8;
    if (chunk > N) chunk = (N + 7) / 8 * 8;
    const size_t n_chunks = (N + chunk - 1) / chunk;

    int device = 0;
    cudaError_t e = cudaGetDevice(&device);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    Workspace *ws = workspace_for(device);
    std::lock_guard<std::mutex> lk(ws->mu);
    rc = ensure_ready(ws, device);
    if (rc != ALOCO_OK) return rc;

    // streams, events and staging (grown on demand, kept until shutdown)
    if (!ws->hs_in) {
        e = cudaStreamCreateWithFlags(&ws->hs_in, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&ws->hs_out, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ws->hs_start, cudaEventDisableTiming);
        if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ws->hs_end, cudaEventDisableTiming);
        for (int k = 0; e == cudaSuccess && k < kSlots; ++k) {
            e = cudaEventCreateWithFlags(&ws->hs_loaded[k], cudaEventDisableTiming);
            if (e == cudaSuccess)
                e = cudaEventCreateWithFlags(&ws->hs_computed[k], cudaEventDisableTiming);
            if (e == cudaSuccess) e = cudaEventCreateWithFlags(&ws->hs_free[k], cudaEventDisableTiming);
        }
        if (e != cudaSuccess) return cuda_fail(e, "host-round streams and events");
    }
    auto up256 = [](size_t b) { return (b + 255) / 256 * 256; };
    const size_t arr4 = up256(chunk * 4), arrx = up256(chunk * rsz);
    const size_t slot_bytes = 2 * arr4 + (size_t)M * arrx;
    const size_t tot_bytes = n_chunks * aloco::kTotalsSlots * sizeof(double);
    const size_t need = kSlots * slot_bytes + up256(tot_bytes);
    if (ws->hs_cap < need) {
        if (ws->hs) cudaFree(ws->hs);
        ws->hs = nullptr;
        ws->hs_cap = 0;
        e = cudaMalloc((void **)&ws->hs, need);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return fail(ALOCO_ERR_NOMEM, "host-round staging cudaMalloc(%zu): %s", need,
                        cudaGetErrorString(e));
        }
        ws->hs_cap = need;
    }
    const size_t host_need = n_chunks * aloco::kTotalsSlots;
    if (ws->hs_host_cap < host_need) {
        if (ws->hs_host) cudaFreeHost(ws->hs_host);
        ws->hs_host = nullptr;
        ws->hs_host_cap = 0;
        e = cudaMallocHost((void **)&ws->hs_host, host_need * sizeof(double));
        if (e != cudaSuccess) {
            cudaGetLastError();
            return fail(ALOCO_ERR_NOMEM, "host-round read-back cudaMallocHost: %s",
                        cudaGetErrorString(e));
        }
        ws->hs_host_cap = host_need;
    }
    double *chunk_totals = reinterpret_cast<double *>(ws->hs + kSlots * slot_bytes);

    aloco::SyncArgs a;
    std::memset(&a, 0, sizeof a);
    split_coef(corr.inv_norm / (double)M, &a.c_hi, &a.c_lo);
    split_coef(corr.mu_t, &a.mu_hi, &a.mu_lo);
    split_coef(-corr.eta_out, &a.neg_eta_hi, &a.neg_eta_lo);
    a.M = M;
    a.partials = ws->partials;
    a.nf_partials = ws->nf_partials;
    a.ticket = ws->ticket;
    a.totals = ws->totals;
    a.nf_total = ws->nf_total;
    a.error = ws->error;
    const int pack = aloco::pack_elems(dtype);

    cudaStream_t main_s = (cudaStream_t)o.stream;
    auto ck = [&](cudaError_t err, const char *what) -> int {
        if (err == cudaSuccess) return ALOCO_OK;
        cudaStreamSynchronize(ws->hs_in);
        cudaStreamSynchronize(ws->hs_out);
        cudaStreamSynchronize(main_s);
        return cuda_fail(err, what);
    };
    if (o.time_kernel && (rc = ck(cudaEventRecord(ws->ev0, main_s), "cudaEventRecord")))
        return rc;
    // the copies start after the work already queued on the caller's stream
    if ((rc = ck(cudaEventRecord(ws->hs_start, main_s), "cudaEventRecord")) ||
        (rc = ck(cudaStreamWaitEvent(ws->hs_in, ws->hs_start, 0), "cudaStreamWaitEvent")) ||
        (rc = ck(cudaStreamWaitEvent(ws->hs_out, ws->hs_start, 0), "cudaStreamWaitEvent")))
        return rc;
    for (size_t c = 0; c < n_chunks; ++c) {
        const int k = (int)(c % kSlots);
        const size_t off = c * chunk;
        const size_t n = std::min(chunk, N - off);
        char *slot = ws->hs + k * slot_bytes;
        float *sg = reinterpret_cast<float *>(slot);
        float *sv = reinterpret_cast<float *>(slot + arr4);
        char *sx = slot + 2 * arr4;
        if (c >= (size_t)kSlots &&
            (rc = ck(cudaStreamWaitEvent(ws->hs_in, ws->hs_free[k], 0), "cudaStreamWaitEvent")))
            return rc;
        rc = ck(cudaMemcpyAsync(sg, global + off, n * 4, cudaMemcpyHostToDevice, ws->hs_in),
                "host-round copy in");
        if (!rc)
            rc = ck(cudaMemcpyAsync(sv, momentum + off, n * 4, cudaMemcpyHostToDevice,
                                    ws->hs_in), "host-round copy in");
        for (int m = 0; !rc && m < M; ++m)
            rc = ck(cudaMemcpyAsync(sx + m * arrx,
                                    static_cast<const char *>(locals[m]) + off * rsz, n * rsz,
                                    cudaMemcpyHostToDevice, ws->hs_in), "host-round copy in");
        if (!rc) rc = ck(cudaEventRecord(ws->hs_loaded[k], ws->hs_in), "cudaEventRecord");
        if (!rc) rc = ck(cudaStreamWaitEvent(main_s, ws->hs_loaded[k], 0), "cudaStreamWaitEvent");
        if (rc) return rc;

        a.g = sg;
        a.v = sv;
        for (int m = 0; m < M; ++m) a.x[m] = sx + m * arrx;
        a.n = (int64_t)n;
        a.nvec = (int64_t)(n / pack);
        aloco::LaunchPlan plan;
        e = dtype == ALOCO_F32
                ? aloco::plan_sync_f32(M, a.nvec > 0 ? a.nvec : a.n, ws->sm_count,
                                       o.blocks_per_sm, &plan)
                : aloco::plan_sync_bf16(M, a.nvec > 0 ? a.nvec : a.n, ws->sm_count,
                                        o.blocks_per_sm, &plan);
        if ((rc = ck(e, "launch plan"))) return rc;
        a.n_tiles = plan.tiles;
        a.stages = plan.stages;
        void *params[] = {&a};
        rc = ck(cudaLaunchKernel(plan.kernel, dim3(plan.grid), dim3(plan.block), params,
                                 plan.smem, main_s), "host-round kernel launch");
        if (!rc)
            rc = ck(cudaMemcpyAsync(chunk_totals + c * aloco::kTotalsSlots, ws->totals,
                                    aloco::kTotalsSlots * sizeof(double),
                                    cudaMemcpyDeviceToDevice, main_s), "chunk totals");
        if (!rc) rc = ck(cudaEventRecord(ws->hs_computed[k], main_s), "cudaEventRecord");
        if (!rc)
            rc = ck(cudaStreamWaitEvent(ws->hs_out, ws->hs_computed[k], 0), "cudaStreamWaitEvent");
        if (!rc)
            rc = ck(cudaMemcpyAsync(global + off, sg, n * 4, cudaMemcpyDeviceToHost, ws->hs_out),
                    "host-round copy out");
        if (!rc)
            rc = ck(cudaMemcpyAsync(momentum + off, sv, n * 4, cudaMemcpyDeviceToHost,
                                    ws->hs_out), "host-round copy out");
        if (!rc) rc = ck(cudaEventRecord(ws->hs_free[k], ws->hs_out), "cudaEventRecord");
        if (rc) return rc;
    }
    rc = ck(cudaMemcpyAsync(ws->hs_host, chunk_totals, tot_bytes, cudaMemcpyDeviceToHost, main_s),
            "statistics readback");
    if (!rc) rc = ck(cudaEventRecord(ws->hs_end, ws->hs_out), "cudaEventRecord");
    if (!rc) rc = ck(cudaStreamWaitEvent(main_s, ws->hs_end, 0), "cudaStreamWaitEvent");
    if (!rc && o.time_kernel) rc = ck(cudaEventRecord(ws->ev1, main_s), "cudaEventRecord");
    if (rc) return rc;
    if ((rc = ck(cudaStreamSynchronize(main_s), "host round"))) return rc;

    // totals of the chunks, added in chunk order
    double tot[aloco::kTotalsSlots] = {};
    unsigned long long nf = 0;
    for (size_t c = 0; c < n_chunks; ++c) {
        const double *t = ws->hs_host + c * aloco::kTotalsSlots;
        for (int m = 0; m <= M; ++m) tot[m] += t[m];
        unsigned long long nfc;
        std::memcpy(&nfc, t + aloco::kNfSlot, sizeof nfc);
        nf += nfc;
    }
    finalize_stats(tot, nf, M, o.eps, 1.0 / ((double)M * (double)M), st);
    st->grid = (int)n_chunks;
    st->pass_used = ALOCO_PASS_REGISTERS;
    if (o.time_kernel) {
        float ms = -1.f;
        if (cudaEventElapsedTime(&ms, ws->ev0, ws->ev1) == cudaSuccess)
            st->kernel_ms = ms;
        else
            cudaGetLastError();
    }
    if (st->nonfinite > 0 || !std::isfinite(st->D) || !std::isfinite(st->C))
        return fail(ALOCO_ERR_NONFINITE, "round produced %lld non-finite elements (D=%g, C=%g)",
                    (long long)st->nonfinite, st->D, st->C);
    t_err.clear();
    return ALOCO_OK;
}

static int adamw_impl(void *const *params, const void *const *grads,
                      float *const *exp_avg, float *const *exp_avg_sq, size_t N,
                      int M, aloco_dtype param_dtype, aloco_dtype grad_dtype,
                      const aloco_adamw_cfg_t *cfg, const double *norms_in,
                      const aloco_opts_t *opts, aloco_adamw_stats_t *stats_out);

int aloco_adamw_step(void *const *params, const void *const *grads,
                     float *const *exp_avg, float *const *exp_avg_sq, size_t N,
                     int M, aloco_dtype param_dtype, aloco_dtype grad_dtype,
                     const aloco_adamw_cfg_t *cfg, const aloco_opts_t *opts,
                     aloco_adamw_stats_t *stats_out) {
    return adamw_impl(params, grads, exp_avg, exp_avg_sq, N, M, param_dtype, grad_dtype,
                      cfg, nullptr, opts, stats_out);
}

int aloco_adamw_step_normed(void *const *params, const void *const *grads,
                            float *const *exp_avg, float *const *exp_avg_sq, size_t N,
                            int M, aloco_dtype param_dtype, aloco_dtype grad_dtype,
                            const aloco_adamw_cfg_t *cfg, const double *grad_norms,
                            const aloco_opts_t *opts, aloco_adamw_stats_t *stats_out) {
    if (!grad_norms) return fail(ALOCO_ERR_ARG, "NULL grad_norms");
    return adamw_impl(params, grads, exp_avg, exp_avg_sq, N, M, param_dtype, grad_dtype,
                      cfg, grad_norms, opts, stats_out);
}

void aloco_adamw_default_cfg(aloco_adamw_cfg_t *cfg) {
    if (!cfg) return;
    std::memset(cfg, 0, sizeof *cfg);
    cfg->lr = 4e-4;
    cfg->beta1 = 0.9;
    cfg->beta2 = 0.95;
    cfg->eps = 1e-8;
    cfg->weight_decay = 0.1;
    cfg->max_grad_norm = 1.0;
    cfg->step = 1;
}

static int adamw_impl(void *const *params, const void *const *grads,
                      float *const *exp_avg, float *const *exp_avg_sq, size_t N,
                      int M, aloco_dtype param_dtype, aloco_dtype grad_dtype,
                      const aloco_adamw_cfg_t *cfg, const double *norms_in,
                      const aloco_opts_t *opts, aloco_adamw_stats_t *stats_out) {
    aloco_opts_t o;
    if (opts) o = *opts; else fill_default_opts(&o);
    if (!cfg) return fail(ALOCO_ERR_ARG, "NULL cfg");
    if (M < 1 || M > ALOCO_MAX_WORKERS)
        return fail(ALOCO_ERR_ARG, "M = %d outside [1, %d]", M, ALOCO_MAX_WORKERS);
    if ((param_dtype != ALOCO_F32 && param_dtype != ALOCO_BF16) ||
        (grad_dtype != ALOCO_F32 && grad_dtype != ALOCO_BF16))
        return fail(ALOCO_ERR_ARG, "unknown dtype (params %d, grads %d)",
                    (int)param_dtype, (int)grad_dtype);
    const aloco_adamw_cfg_t &c = *cfg;
    if (!(std::isfinite(c.lr) && c.lr >= 0.0))
        return fail(ALOCO_ERR_ARG, "lr = %g must be finite and >= 0", c.lr);
    if (!(c.beta1 >= 0.0 && c.beta1 < 1.0) || !(c.beta2 >= 0.0 && c.beta2 < 1.0))
        return fail(ALOCO_ERR_ARG, "betas (%g, %g) must lie in [0, 1)", c.beta1, c.beta2);
    if (!(std::isfinite(c.eps) && c.eps > 0.0))
        return fail(ALOCO_ERR_ARG, "eps = %g must be finite and > 0", c.eps);
    if (!(std::isfinite(c.weight_decay) && c.weight_decay >= 0.0))
        return fail(ALOCO_ERR_ARG, "weight_decay = %g must be finite and >= 0",
                    c.weight_decay);
    if (!std::isfinite(c.max_grad_norm))
        return fail(ALOCO_ERR_ARG, "max_grad_norm must be finite");
    if (c.step < 1) return fail(ALOCO_ERR_ARG, "step = %lld must be >= 1", (long long)c.step);
    // clipping factors from given norms: the update kernel's formula, in
    // the same double arithmetic
    double given_clip[ALOCO_MAX_WORKERS];
    if (norms_in) {
        for (int m = 0; m < M; ++m) {
            const double nm = norms_in[m];
            if (!(std::isfinite(nm) && nm >= 0.0))
                return fail(ALOCO_ERR_ARG, "grad_norms[%d] = %g must be finite and >= 0", m, nm);
            double cf = 1.0;
            if (c.max_grad_norm > 0.0) {
                cf = c.max_grad_norm / (nm + 1e-6);
                if (cf > 1.0) cf = 1.0;
            }
            given_clip[m] = cf;
        }
    }
    if (o.blocks_per_sm < 0)
        return fail(ALOCO_ERR_ARG, "blocks_per_sm = %d must be >= 0", o.blocks_per_sm);
    if (N > (size_t)INT64_MAX / 8) return fail(ALOCO_ERR_ARG, "N too large");
    if (N > 0 && (!params || !grads || !exp_avg || !exp_avg_sq))
        return fail(ALOCO_ERR_ARG, "NULL pointer array");
    for (int m = 0; N > 0 && m < M; ++m)
        if (!params[m] || !grads[m] || !exp_avg[m] || !exp_avg_sq[m])
            return fail(ALOCO_ERR_ARG, "NULL buffer for replica %d", m);

    aloco_adamw_stats_t local;
    aloco_adamw_stats_t *st = stats_out ? stats_out : &local;
    std::memset(st, 0, sizeof *st);
    st->M = M;
    st->kernel_ms = -1.f;
    for (int m = 0; m < M; ++m) {
        st->clip[m] = norms_in ? given_clip[m] : 1.0;
        if (norms_in) st->grad_norm[m] = norms_in[m];
    }
    if (N == 0) {
        t_err.clear();
        return ALOCO_OK;
    }

    const size_t psz = param_dtype == ALOCO_F32 ? 4 : 2;
    const size_t gsz = grad_dtype == ALOCO_F32 ? 4 : 2;
    // Updated buffers may overlap nothing; gradients may be shared by
    // replicas (read only) but may not overlap an updated buffer.
    {
        std::vector<std::pair<uintptr_t, size_t>> upd, rd;
        for (int m = 0; m < M; ++m) {
            upd.push_back({(uintptr_t)params[m], N * psz});
            upd.push_back({(uintptr_t)exp_avg[m], N * 4});
            upd.push_back({(uintptr_t)exp_avg_sq[m], N * 4});
            rd.push_back({(uintptr_t)grads[m], N * gsz});
        }
        auto hit = [](const std::pair<uintptr_t, size_t> &a,
                      const std::pair<uintptr_t, size_t> &b) {
            return a.first < b.first + b.second && b.first < a.first + a.second;
        };
        for (size_t i = 0; i < upd.size(); ++i) {
            for (size_t j = i + 1; j < upd.size(); ++j)
                if (hit(upd[i], upd[j]))
                    return fail(ALOCO_ERR_ALIAS, "updated buffers %zu and %zu overlap", i, j);
            for (size_t j = 0; j < rd.size(); ++j)
                if (hit(upd[i], rd[j]))
                    return fail(ALOCO_ERR_ALIAS, "grads[%zu] overlaps an updated buffer", j);
        }
    }
    uintptr_t align_or = 0;
    for (int m = 0; m < M; ++m) {
        if (((uintptr_t)params[m] & (psz - 1)) || ((uintptr_t)grads[m] & (gsz - 1)) ||
            ((uintptr_t)exp_avg[m] & 3) || ((uintptr_t)exp_avg_sq[m] & 3))
            return fail(ALOCO_ERR_ARG, "replica %d: buffer not aligned to its element", m);
        align_or |= (uintptr_t)params[m] | (uintptr_t)grads[m] |
                    (uintptr_t)exp_avg[m] | (uintptr_t)exp_avg_sq[m];
    }

    int device = 0;
    cudaError_t e = cudaGetDevice(&device);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    Workspace *ws = workspace_for(device);
    std::lock_guard<std::mutex> lk(ws->mu);
    int rc = ensure_ready(ws, device);
    if (rc != ALOCO_OK) return rc;
    for (int m = 0; m < M; ++m) {
        char name[40];
        snprintf(name, sizeof name, "params[%d]", m);
        if ((rc = check_buffer(params[m], N * psz, device, name)) != ALOCO_OK) return rc;
        snprintf(name, sizeof name, "grads[%d]", m);
        if ((rc = check_buffer(grads[m], N * gsz, device, name)) != ALOCO_OK) return rc;
        snprintf(name, sizeof name, "exp_avg[%d]", m);
        if ((rc = check_buffer(exp_avg[m], N * 4, device, name)) != ALOCO_OK) return rc;
        snprintf(name, sizeof name, "exp_avg_sq[%d]", m);
        if ((rc = check_buffer(exp_avg_sq[m], N * 4, device, name)) != ALOCO_OK) return rc;
    }

    aloco::AdamArgs a;
    std::memset(&a, 0, sizeof a);
    for (int m = 0; m < M; ++m) {
        a.x[m] = params[m];
        a.g[m] = grads[m];
        a.m1[m] = exp_avg[m];
        a.m2[m] = exp_avg_sq[m];
    }
    a.n = (int64_t)N;
    a.nunit = (align_or & 15) == 0 ? (int64_t)(N / 4) : 0;
    a.M = M;
    const double bc1 = 1.0 - std::pow(c.beta1, (double)c.step);
    const double bc2 = 1.0 - std::pow(c.beta2, (double)c.step);
    a.beta1 = (float)c.beta1;
    a.omb1 = (float)(1.0 - c.beta1);
    a.beta2 = (float)c.beta2;
    a.omb2 = (float)(1.0 - c.beta2);
    a.decay = (float)(1.0 - c.lr * c.weight_decay);
    a.neg_step = (float)(-c.lr / bc1);
    a.inv_sqrt_bc2 = (float)(1.0 / std::sqrt(bc2));
    a.eps = (float)c.eps;
    a.max_norm = c.max_grad_norm;
    a.partials = ws->adam;
    a.out = ws->adam + ws->max_grid;
    if (norms_in) {
        a.given = 1;
        for (int m = 0; m < M; ++m) a.clip[m] = (float)given_clip[m];
    }

    // norm pass: up to the workspace's max_grid blocks over all workers;
    // update pass: SMs x blocks_per_sm blocks (default 4) over all workers
    const int64_t work = a.nunit > 0 ? a.nunit : a.n;
    const int64_t per_thread = (int64_t)aloco::kBlock;
    int64_t g1 = ws->max_grid / M;
    g1 = std::min<int64_t>(g1, (work + per_thread - 1) / per_thread);
    a.g1 = (int)std::max<int64_t>(g1, 1);
    const int bps = o.blocks_per_sm > 0 ? o.blocks_per_sm : 4;
    int64_t g2 = ((int64_t)ws->sm_count * bps + M - 1) / M;
    g2 = std::min<int64_t>(g2, (work + 2 * per_thread - 1) / (2 * per_thread));
    g2 = std::max<int64_t>(g2, 1);
    if (g2 > 65535) g2 = 65535;

    cudaStream_t stream = (cudaStream_t)o.stream;
    const bool timed = o.time_kernel && stats_out;
    if (timed && (e = cudaEventRecord(ws->ev0, stream)) != cudaSuccess)
        return cuda_fail(e, "cudaEventRecord");
    e = aloco::launch_adamw(a, param_dtype, grad_dtype, (int)g2, stream);
    if (e != cudaSuccess) return cuda_fail(e, "AdamW launch");
    if (timed && (e = cudaEventRecord(ws->ev1, stream)) != cudaSuccess)
        return cuda_fail(e, "cudaEventRecord");
    st->grid = (int)(g2 * M);
    if (stats_out && norms_in) {
        if (timed) {
            if ((e = cudaEventSynchronize(ws->ev1)) != cudaSuccess)
                return cuda_fail(e, "AdamW step");
            float ms = -1.f;
            if (cudaEventElapsedTime(&ms, ws->ev0, ws->ev1) == cudaSuccess)
                st->kernel_ms = ms;
            else
                cudaGetLastError();
        }
    } else if (stats_out) {
        e = cudaMemcpyAsync(ws->host, a.out, 2 * ALOCO_MAX_WORKERS * sizeof(double),
                            cudaMemcpyDeviceToHost, stream);
        if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
        if (e != cudaSuccess) return cuda_fail(e, "AdamW step");
        for (int m = 0; m < M; ++m) {
            st->grad_norm[m] = ws->host[m];
            st->clip[m] = ws->host[ALOCO_MAX_WORKERS + m];
        }
        if (timed) {
            float ms = -1.f;
            if (cudaEventElapsedTime(&ms, ws->ev0, ws->ev1) == cudaSuccess)
                st->kernel_ms = ms;
            else
                cudaGetLastError();
        }
    }
    t_err.clear();
    return ALOCO_OK;
}

void aloco_test_stall_tile(int64_t tile) { t_test_stall_tile1 = tile >= 0 ? tile + 1 : 0; }

const char *aloco_last_error(void) { return t_err.c_str(); }

void aloco_shutdown(void) {
    std::lock_guard<std::mutex> lk(g_registry_mu);
    int prev = -1;
    cudaGetDevice(&prev);
    for (auto &ws : g_registry) {
        if (!ws) continue;
        std::lock_guard<std::mutex> lk2(ws->mu);
        if (!ws->ready) continue;
        cudaSetDevice(ws->device);
        cudaDeviceSynchronize();
        if (ws->ev0) cudaEventDestroy(ws->ev0);
        if (ws->ev1) cudaEventDestroy(ws->ev1);
        if (ws->ev_block) cudaEventDestroy(ws->ev_block);
        ws->ev_block = nullptr;
        if (ws->host) cudaFreeHost(ws->host);
        if (ws->stats_host) cudaFreeHost(ws->stats_host);
        if (ws->dev) cudaFree(ws->dev);
        if (ws->i8) cudaFree(ws->i8);
        ws->i8 = nullptr;
        ws->i8_cap = 0;
        if (ws->hs) cudaFree(ws->hs);
        if (ws->hs_host) cudaFreeHost(ws->hs_host);
        ws->hs = nullptr;
        ws->hs_cap = 0;
        ws->hs_host = nullptr;
        ws->hs_host_cap = 0;
        cudaEvent_t *evs[] = {&ws->hs_start, &ws->hs_end};
        for (cudaEvent_t *ev : evs)
            if (*ev) cudaEventDestroy(*ev), *ev = nullptr;
        for (int k = 0; k < 3; ++k) {
            for (cudaEvent_t *ev : {&ws->hs_loaded[k], &ws->hs_computed[k], &ws->hs_free[k]})
                if (*ev) cudaEventDestroy(*ev), *ev = nullptr;
        }
        if (ws->hs_in) cudaStreamDestroy(ws->hs_in);
        if (ws->hs_out) cudaStreamDestroy(ws->hs_out);
        ws->hs_in = ws->hs_out = nullptr;
        ws->ev0 = ws->ev1 = nullptr;
        ws->host = nullptr;
        ws->stats_host = nullptr;
        ws->stats_dev = nullptr;
        ws->dev = nullptr;
        ws->ready = false;
    }
    if (prev >= 0) cudaSetDevice(prev);
    cudaGetLastError();
}

int aloco_version(void) { return 100; }

}  // extern "C"
