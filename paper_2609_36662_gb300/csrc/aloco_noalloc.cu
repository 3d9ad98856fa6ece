// aloco_sync_noalloc: the outer synchronisation round without any memory
// allocation by the library.
//
// aloco_sync_ex keeps a per-device workspace that it allocates with
// cudaMalloc / cudaMallocHost on first use.  Some callers cannot let a
// library allocate: frameworks that reserve the whole device memory up front
// and hand it out from their own pools, deployments whose memory footprint
// must be fixed when the library is loaded, and loops that cannot afford the
// implicit device synchronisation of cudaMalloc / cudaFree.  For them this
// entry point runs the same fused kernel as aloco_sync_ex, chosen by the same
// rule (the tile pass, the bulk-copy pass or the register pass) and launched
// with the same grid, with its scratch (per-block partial sums, the
// last-block ticket and the totals) in a file-scope __device__ array that
// exists, on every device that loads the library, from module load until the
// process exits.  It calls no cudaMalloc, cudaFree, cudaMallocHost or other
// allocating routine; the statistics come back through a plain
// cudaMemcpyAsync into a buffer on the caller's stack, followed by a stream
// synchronisation, so a call cannot be part of a stream capture.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "../../include/aloco.h"
#include "aloco_internal.h"

namespace {

// Block partials the scratch can hold: one row of M + 1 fp64 values per
// block.  The register and bulk-copy passes cap their residency at the
// kernel's occupancy, whatever opts->blocks_per_sm asks for, so they use at
// most SMs x 8 blocks (256-thread blocks, 2048 threads per SM); the tile
// pass uses at most SMs x 4.  On a 152-SM GB300 that is 1216 rows; only a
// device with more than 256 SMs could be refused.
constexpr int kScratchBlocks = ALOCO_NOALLOC_MAX_BLOCKS;

struct NoallocScratch {
    double partials[kScratchBlocks * (ALOCO_MAX_WORKERS + 1)];
    unsigned long long nf_partials[kScratchBlocks];
    double totals[aloco::kTotalsSlots];  // M + 1 totals, nf count, error word
    unsigned int ticket;
};

// The scratch itself.  In host code this name is only a host-side stand-in
// for the device symbol: its device address comes from cudaGetSymbolAddress.
static __device__ __align__(256) NoallocScratch g_scratch;

constexpr int kMaxDevices = 64;
std::mutex g_mu[kMaxDevices];
NoallocScratch *g_addr[kMaxDevices];  // device address per device, or null
int g_sms[kMaxDevices];

// Once per device, with that device current: resolve the scratch address.
int setup_device(int device) {
    if (g_addr[device]) return ALOCO_OK;
    void *ptr = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&ptr, g_scratch);
    if (e != cudaSuccess || ptr == nullptr) {
        cudaGetLastError();
        char msg[160];
        snprintf(msg, sizeof msg, "cudaGetSymbolAddress(scratch): %s",
                 cudaGetErrorString(e));
        return aloco::report_error(ALOCO_ERR_CUDA, msg);
    }
    int sms = 0;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, device);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return aloco::report_error(ALOCO_ERR_CUDA, "cudaDeviceGetAttribute");
    }
    g_sms[device] = sms;
    g_addr[device] = static_cast<NoallocScratch *>(ptr);
    return ALOCO_OK;
}

int errf(int code, const char *fmt, ...) __attribute__((format(printf, 2, 3)));
int errf(int code, const char *fmt, ...) {
    char buf[256];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    return aloco::report_error(code, buf);
}

}  // namespace

extern "C" int aloco_sync_noalloc(float *global, float *momentum,
                                  void *const *locals, size_t N, int M,
                                  aloco_dtype dtype, int64_t H_sel,
                                  int64_t H_base, int64_t step,
                                  const aloco_schedule_t *schedule,
                                  double outer_lr, double outer_beta,
                                  const aloco_opts_t *opts,
                                  aloco_stats_t *stats_out) {
    aloco_opts_t o;
    if (opts) o = *opts; else aloco::fill_default_opts(&o);
    aloco_stats_t local_stats;
    aloco_stats_t *st = stats_out ? stats_out : &local_stats;

    if (M < 1 || M > ALOCO_MAX_WORKERS)
        return errf(ALOCO_ERR_ARG, "M = %d outside [1, %d]", M, ALOCO_MAX_WORKERS);
    if (dtype != ALOCO_F32 && dtype != ALOCO_BF16)
        return errf(ALOCO_ERR_ARG, "unknown replica dtype %d", (int)dtype);
    if (o.pass == ALOCO_PASS_INT8_SPLIT || o.pass == ALOCO_PASS_INT8_FUSED)
        return errf(ALOCO_ERR_ARG, "pass %d does not apply to this round", o.pass);
    if (N > (size_t)INT64_MAX / 8) return errf(ALOCO_ERR_ARG, "N too large");
    if (N > 0 && (!global || !momentum || !locals))
        return errf(ALOCO_ERR_ARG, "NULL buffer");
    for (int m = 0; N > 0 && m < M; ++m)
        if (!locals[m]) return errf(ALOCO_ERR_ARG, "locals[%d] is NULL", m);
    aloco_correction_t corr;
    int rc = aloco_correction(schedule, step, H_sel, H_base, outer_lr,
                              outer_beta, &o, &corr);
    if (rc != ALOCO_OK) return rc;

    std::memset(st, 0, sizeof *st);
    st->corr = corr;
    st->M = M;
    st->kernel_ms = -1.f;
    if (N == 0) return ALOCO_OK;

    const size_t rsz = dtype == ALOCO_F32 ? 4 : 2;
    {
        uintptr_t base[ALOCO_MAX_WORKERS + 2];
        size_t len[ALOCO_MAX_WORKERS + 2];
        base[0] = (uintptr_t)global;
        len[0] = N * 4;
        base[1] = (uintptr_t)momentum;
        len[1] = N * 4;
        for (int m = 0; m < M; ++m) {
            base[m + 2] = (uintptr_t)locals[m];
            len[m + 2] = N * rsz;
        }
        for (int i = 0; i < M + 2; ++i)
            for (int j = i + 1; j < M + 2; ++j)
                if (base[i] < base[j] + len[j] && base[j] < base[i] + len[i])
                    return errf(ALOCO_ERR_ALIAS, "buffers %d and %d overlap", i, j);
    }
    if (((uintptr_t)global | (uintptr_t)momentum) & 3)
        return errf(ALOCO_ERR_ARG, "global/momentum not 4-byte aligned");
    for (int m = 0; m < M; ++m)
        if ((uintptr_t)locals[m] & (rsz - 1))
            return errf(ALOCO_ERR_ARG, "locals[%d] not %zu-byte aligned", m, rsz);

    int device = 0;
    cudaError_t e = cudaGetDevice(&device);
    if (e != cudaSuccess || device < 0 || device >= kMaxDevices) {
        cudaGetLastError();
        return errf(ALOCO_ERR_CUDA, "cudaGetDevice failed or device out of range");
    }
    cudaStream_t stream = (cudaStream_t)o.stream;
    {
        // the call ends with a stream synchronisation, which a capture
        // cannot contain: refuse before any other CUDA call
        cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
        e = cudaStreamIsCapturing(stream, &cap);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return errf(ALOCO_ERR_CUDA, "cudaStreamIsCapturing: %s", cudaGetErrorString(e));
        }
        if (cap != cudaStreamCaptureStatusNone)
            return errf(ALOCO_ERR_ARG,
                        "aloco_sync_noalloc cannot run under stream capture: it "
                        "waits for its round with a stream synchronisation");
    }
    std::lock_guard<std::mutex> lk(g_mu[device]);
    if ((rc = setup_device(device)) != ALOCO_OK) return rc;
    if ((rc = aloco::check_buffer(global, N * 4, device, "global")) != ALOCO_OK)
        return rc;
    if ((rc = aloco::check_buffer(momentum, N * 4, device, "momentum")) != ALOCO_OK)
        return rc;
    for (int m = 0; m < M; ++m) {
        char name[32];
        snprintf(name, sizeof name, "locals[%d]", m);
        if ((rc = aloco::check_buffer(locals[m], N * rsz, device, name)) != ALOCO_OK)
            return rc;
    }

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
    aloco::split_coef(corr.inv_norm / (double)M, &a.c_hi, &a.c_lo);
    aloco::split_coef(corr.mu_t, &a.mu_hi, &a.mu_lo);
    aloco::split_coef(-corr.eta_out, &a.neg_eta_hi, &a.neg_eta_lo);
    a.M = M;

    const int64_t work = a.nvec > 0 ? a.nvec : a.n;
    aloco::LaunchPlan plan;
    // the same choice of kernel as aloco_sync_ex
    const bool tile = aloco::use_tile(o.pass, M, dtype, a.n, a.nvec);
    const bool tma = !tile && aloco::use_tma(o.pass, M, dtype, a.nvec);
    plan.grid = 0;
    plan.block = 0;
    plan.kernel = nullptr;
    e = cudaSuccess;
    if (tile)
        ;  // launch_sync_tile picks its grid below (at most SMs x 4 CTAs)
    else if (tma)
        e = dtype == ALOCO_F32
                ? aloco::plan_sync_tma_f32(M, a.nvec, g_sms[device], &plan)
                : aloco::plan_sync_tma_bf16(M, a.nvec, g_sms[device], &plan);
    else
        e = dtype == ALOCO_F32
                ? aloco::plan_sync_f32(M, work, g_sms[device], o.blocks_per_sm, &plan)
                : aloco::plan_sync_bf16(M, work, g_sms[device], o.blocks_per_sm, &plan);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return errf(ALOCO_ERR_CUDA, "launch plan: %s", cudaGetErrorString(e));
    }
    if (plan.grid > kScratchBlocks)
        return errf(ALOCO_ERR_ARG,
                    "this round needs %d blocks of partial sums; the "
                    "allocation-free scratch holds %d (ALOCO_NOALLOC_MAX_BLOCKS)",
                    plan.grid, kScratchBlocks);

    NoallocScratch *s = g_addr[device];
    a.partials = s->partials;
    a.nf_partials = s->nf_partials;
    a.ticket = &s->ticket;
    a.totals = s->totals;
    a.nf_total = (unsigned long long *)(s->totals + aloco::kNfSlot);
    a.error = (unsigned int *)(s->totals + aloco::kErrorSlot);
    a.n_tiles = plan.tiles;
    a.stages = plan.stages;

    // The ticket and the error word must start at zero; every partial row
    // and total used by this launch is written by it before it is read.
    e = cudaMemsetAsync(&s->ticket, 0, sizeof(unsigned int), stream);
    if (e == cudaSuccess)
        e = cudaMemsetAsync(a.error, 0, sizeof(unsigned int), stream);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return errf(ALOCO_ERR_CUDA, "ticket reset: %s", cudaGetErrorString(e));
    }
    if (tile) {
        e = aloco::launch_sync_tile(a, dtype, g_sms[device], kScratchBlocks, stream,
                                    &plan.grid);
    } else {
        void *params[] = {&a};
        e = cudaLaunchKernel(plan.kernel, dim3(plan.grid), dim3(plan.block), params,
                             plan.smem, stream);
    }
    if (e != cudaSuccess) {
        cudaGetLastError();
        return errf(ALOCO_ERR_CUDA, "fused sync launch: %s", cudaGetErrorString(e));
    }
    double host[aloco::kTotalsSlots];
    e = cudaMemcpyAsync(host, s->totals, sizeof host, cudaMemcpyDeviceToHost,
                        stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return errf(ALOCO_ERR_CUDA, "round: %s", cudaGetErrorString(e));
    }
    unsigned long long nf;
    std::memcpy(&nf, host + aloco::kNfSlot, sizeof nf);
    unsigned int perr;
    std::memcpy(&perr, host + aloco::kErrorSlot, sizeof perr);
    if (perr != 0)
        return errf(ALOCO_ERR_CUDA,
                    "bulk-copy pipeline wait timed out; outputs are incomplete");
    aloco::finalize_stats(host, nf, M, o.eps, 1.0 / ((double)M * (double)M), st);
    st->grid = plan.grid;
    st->pass_used = tile ? ALOCO_PASS_TILE : tma ? ALOCO_PASS_BULK_COPY : ALOCO_PASS_REGISTERS;
    if (st->nonfinite > 0 || !std::isfinite(st->D) || !std::isfinite(st->C))
        return errf(ALOCO_ERR_NONFINITE,
                    "round produced %lld non-finite elements (D=%g, C=%g)",
                    (long long)st->nonfinite, st->D, st->C);
    aloco::report_error(ALOCO_OK, "");
    return ALOCO_OK;
}
