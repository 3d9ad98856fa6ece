/*
 * aloco.h -- C ABI of libaloco: the AutoLoCo outer synchronisation round
 * (arxiv 2609.36662) on one GB300 GPU.
 *
 * One call runs the whole round of Algorithm 1 ("Synchronization and
 * corrected outer update" plus the D_t / C_t part of "Interval evaluation")
 * for M worker replicas that live in the memory of one GPU:
 *
 *   Delta_m = theta - x_m                       pseudo-gradients (Alg. 1)
 *   Dbar    = (1/M) sum_m Delta_m               synchronisation (Alg. 1)
 *   D       = (1/M) sum_m ||Delta_m||^2         local-drift energy
 *   C       = M ||Dbar||^2 / (D + eps)          aggregation coherence
 *                                               (Eq. adaptive-h-core-diagnostics)
 *   Dtil    = Dbar / (rho + eps)  (optional)    (Eq. normalized-pseudo-gradient,
 *                                                App. B.3)
 *   v'      = mu_t v + Dtil
 *   d       = Dtil + mu_t v'
 *   theta'  = theta - eta_out d                 (Eq. autoloco-corrected-nesterov)
 *   x_m     = theta'   for every m              replica reset (Alg. 1)
 *
 * with rho, mu_t, kappa_t and eta_out from the Outer Optimizer Correction
 * (Sec. 3.2; App. B.2 and B.4), evaluated on the host from exact previews of
 * the inner learning-rate schedule.  The elementwise work is one fused CUDA
 * pass that reads theta, v and every replica once and writes each once.
 *
 * Conventions shared by every entry point:
 *   - All N-element buffers are caller-owned DEVICE memory on the current
 *     CUDA device and are updated in place.  `locals` is a HOST array of M
 *     device pointers.  Buffers must not overlap one another.
 *   - theta ("global") and v ("momentum") are fp32; replicas are fp32 or
 *     bf16 (aloco_dtype).  Element n of every buffer is parameter n of the
 *     flattened parameter vector.
 *   - Return value: ALOCO_OK (0) or a negative aloco_status.  Arguments are
 *     validated before any work is enqueued; on ALOCO_ERR_ARG and
 *     ALOCO_ERR_ALIAS no buffer is touched.  aloco_last_error() returns a
 *     thread-local message describing the last failure.  The library never
 *     exits or traps.
 *   - Work is enqueued on opts->stream (NULL: the legacy default stream).
 *     aloco_sync / aloco_sync_ex return after the round has completed on
 *     that stream (they wait for the statistics, a few hundred bytes).
 *   - Statistics are reduced in a fixed order, so repeated calls on the same
 *     inputs, device and build return bit-identical results.
 */
#ifndef ALOCO_H
#define ALOCO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ALOCO_MAX_WORKERS 32

/* Replica storage type.  theta and v are always fp32 (the paper keeps FP32
 * master weights and outer state, App. E.1 and App. G.1). */
typedef enum { ALOCO_F32 = 0, ALOCO_BF16 = 1 } aloco_dtype;

typedef enum {
    ALOCO_OK = 0,
    ALOCO_ERR_ARG = -1,       /* invalid argument; nothing was touched     */
    ALOCO_ERR_CUDA = -2,      /* a CUDA runtime call failed                */
    ALOCO_ERR_NONFINITE = -3, /* round completed; some outputs are NaN/Inf */
    ALOCO_ERR_ALIAS = -4,     /* two buffers overlap; nothing was touched  */
    ALOCO_ERR_NOMEM = -5      /* workspace allocation failed               */
} aloco_status;

/* Inner learning-rate schedule (Tab. training settings: cosine decay with a
 * linear warm-up).  For global inner step s (0-based):
 *   s <  warmup_steps:            lr = peak_lr * (s + 1) / warmup_steps
 *   warmup_steps <= s < total:    cosine:  final + (peak - final)(1 + cos(pi f))/2
 *                                 linear:  peak + (final - peak) f
 *                                 with f = (s - warmup) / (total - warmup)
 *   s >= total_steps:             lr = final_lr
 *   kind CONSTANT:                lr = peak_lr for every s.
 * total_steps counts the warm-up.  Requirements: 0 <= warmup_steps <
 * total_steps (any values for CONSTANT), finite non-negative rates. */
typedef enum {
    ALOCO_SCHED_COSINE = 0,
    ALOCO_SCHED_CONSTANT = 1,
    ALOCO_SCHED_LINEAR = 2
} aloco_sched_kind;

typedef struct aloco_schedule {
    int32_t kind; /* aloco_sched_kind */
    int32_t reserved;
    double peak_lr;
    double final_lr;
    int64_t warmup_steps;
    int64_t total_steps;
} aloco_schedule_t;

/* Which parts of the Outer Optimizer Correction run (Tab. component
 * ablation; App. E.4):
 *   FULL           mu_t = clip(mu_base^rho, mu_min, mu_max),
 *                  eta_out = eta_base kappa_t (1 - mu_t)/(1 - mu_base)
 *   MOMENTUM_ONLY  mu_t as FULL, eta_out = eta_base
 *   NONE           mu_t = mu_base, eta_out = eta_base (DiLoCo's outer step)
 * Pseudo-gradient normalisation is switched independently
 * (aloco_opts_t.normalize; App. B.3). */
typedef enum {
    ALOCO_CORR_FULL = 0,
    ALOCO_CORR_MOMENTUM_ONLY = 1,
    ALOCO_CORR_NONE = 2
} aloco_corr_mode;

/* The implementations of the fused pass.  All compute the same round with
 * the same per-element arithmetic (theta', v' and the replicas agree bit
 * for bit); they differ in how data reaches the SMs.
 *   REGISTERS  every thread streams 16-byte loads of theta, v and the
 *              replicas straight into registers (any M, any alignment);
 *   BULK_COPY  a producer warp per SM stages 4-8 KB tiles of every array in
 *              a shared-memory ring with cp.async.bulk and mbarriers, and
 *              consumer warps compute from shared memory (M <= 16, 16-byte
 *              aligned buffers; otherwise REGISTERS runs);
 *   TILE       CTAs stage whole blocks of every array with cp.async.bulk,
 *              write theta' once to a shared-memory tile and store the
 *              replica reset as M bulk copies of it (M <= 16, 16-byte
 *              aligned buffers, N >= 4096; otherwise REGISTERS runs);
 *   AUTO       the fastest as measured on GB300 for (M, dtype, N): TILE
 *              from 2^27 parameters for bf16 replicas with M <= 12 and for
 *              fp32 with M = 1 or 5..16, else REGISTERS.
 * The INT8-communicated round (aloco_sync_int8) has two forms of its own:
 *   INT8_SPLIT a block-scale kernel, then an apply kernel that reads the
 *              replicas again (any M <= 16);
 *   INT8_FUSED one kernel that stages each block of the replicas (and of
 *              theta and v, for the shapes where that measured faster) in
 *              shared memory, reading every array once (any M <= 16; above
 *              8 fp32 replicas it stages each block's replicas in groups);
 *   AUTO       the form measured faster on GB300 for (M, dtype).
 * The two INT8 forms give the same theta', v' and replicas bit for bit.
 * aloco_sync / aloco_sync_ex reject the INT8 values and aloco_sync_int8 the
 * REGISTERS / BULK_COPY / TILE values with ALOCO_ERR_ARG. */
typedef enum {
    ALOCO_PASS_AUTO = 0,
    ALOCO_PASS_REGISTERS = 1,
    ALOCO_PASS_BULK_COPY = 2,
    ALOCO_PASS_INT8_SPLIT = 3,
    ALOCO_PASS_INT8_FUSED = 4,
    ALOCO_PASS_TILE = 5
} aloco_pass;

/* How a round call waits for its kernel (aloco_sync_ex, aloco_sync_int8 and
 * the shard calls):
 *   SPIN   the calling thread polls the device-mapped page that the round's
 *          last block publishes its statistics to, checking the stream every
 *          few hundred reads.  Lowest latency (the call returns a few
 *          microseconds after the last block), but the thread keeps one host
 *          core busy for the whole round, including any time the stream is
 *          queued behind earlier work.
 *   BLOCK  the call records a blocking-sync CUDA event behind the kernel and
 *          waits on it: the thread sleeps until the round has completed, then
 *          reads the same published statistics.  For callers that run the
 *          round on a busy stream or need the core; each call pays the
 *          event's wake-up latency.
 * Outputs and statistics are the same in both modes. */
typedef enum { ALOCO_WAIT_SPIN = 0, ALOCO_WAIT_BLOCK = 1 } aloco_wait;

/* Options.  aloco_default_opts() fills the paper's settings
 * (Tab. AutoLoCo configuration): mu_min 0.45, mu_max 0.90, kappa_max 1.6,
 * eps 1e-8, normalize off, FULL correction, no kernel timing, the tuned
 * launch configuration, default stream, AUTO pass, SPIN wait.  Passing NULL
 * where an opts pointer is accepted means these defaults. */
typedef struct aloco_opts {
    double mu_min;
    double mu_max;
    double kappa_max;
    double eps;           /* the paper's numerical constant epsilon, > 0     */
    int32_t normalize;    /* 1: Dtil = Dbar / (rho + eps)                    */
    int32_t mode;         /* aloco_corr_mode                                 */
    int32_t time_kernel;  /* 1: stats_out->kernel_ms = duration of the fused
                             pass, from CUDA events on the launch stream     */
    int32_t blocks_per_sm;/* resident blocks per SM of the fused pass; 0 =
                             the library's tuned choice for (M, dtype).  It
                             is capped at what the kernel's registers allow.
                             The grid fixes the order of the fp64 partial
                             sums, so a different value can change the
                             statistics in their last bits.                  */
    void *stream;         /* cudaStream_t; NULL = legacy default stream      */
    int32_t pass;         /* aloco_pass: which fused kernel runs the round   */
    int32_t wait;         /* aloco_wait: how the host waits for the round    */
} aloco_opts_t;

/* Correction context of one interval (App. B.2, B.4). */
typedef struct aloco_correction {
    double lam_sel;  /* Lambda_t      = sum_{h=1..H_sel}  lr(step + h - 1)   */
    double lam_base; /* Lambda_t^base = sum_{h=1..H_base} lr(step + h - 1)   */
    double rho_unc;  /* Lambda_t / (Lambda_t^base + eps)                     */
    double rho;      /* max(rho_unc, 1)                                      */
    double mu_t;     /* outer momentum applied this round                    */
    double kappa_t;  /* bounded outer-step scale                             */
    double eta_out;  /* outer learning rate applied this round               */
    double inv_norm; /* 1 / (rho + eps) with normalisation, else 1           */
} aloco_correction_t;

/* Statistics of one round. */
typedef struct aloco_stats {
    double D;                         /* local-drift energy D_t              */
    double C;                         /* aggregation coherence C_t           */
    double mean_sq_norm;              /* ||Dbar||_2^2                        */
    double drift[ALOCO_MAX_WORKERS];  /* ||Delta_m||_2^2, m < M              */
    aloco_correction_t corr;          /* the correction context applied      */
    int64_t nonfinite;                /* elements whose theta' or v' is not
                                         finite                              */
    int32_t M;
    int32_t grid;                     /* CUDA blocks of the fused pass       */
    float kernel_ms;                  /* fused-pass duration, or -1          */
    int32_t pass_used;                /* aloco_pass that ran (0 if no kernel) */
} aloco_stats_t;

/* Fill *opts with the defaults listed above. */
void aloco_default_opts(aloco_opts_t *opts);

/* Accumulated inner learning rate over an interval of H local steps that
 * starts at global inner step t0 (0-based):
 *   sum_{h=1..H} lr(t0 + h - 1)          (Eq. app-outer-correction-lr-masses)
 * Host-only, no GPU needed.  Returns NaN when schedule is NULL or invalid,
 * t0 < 0 or H < 0; H = 0 gives 0. */
double aloco_inner_lr_accum(const aloco_schedule_t *schedule, int64_t t0,
                            int64_t H);

/* The scalar correction context of an interval starting at global inner
 * step `step` with selected horizon H_sel and base horizon H_base (both in
 * executable steps; Sec. 3.2, Eq. outer-correction-ratio,
 * Eq. adjusted-outer-learning-rate; App. B.2-B.4).  outer_lr is
 * eta_base^out, outer_beta is mu_base.  Host-only.  Requirements: H_sel >=
 * 1, H_base >= 1, step >= 0, outer_lr finite, 0 < outer_beta < 1 for FULL
 * and MOMENTUM_ONLY, 0 <= outer_beta < 1 for NONE, 0 <= mu_min <= mu_max
 * < 1, kappa_max >= 1, eps > 0. */
int aloco_correction(const aloco_schedule_t *schedule, int64_t step,
                     int64_t H_sel, int64_t H_base, double outer_lr,
                     double outer_beta, const aloco_opts_t *opts,
                     aloco_correction_t *out);

/* One outer synchronisation round with default options (see
 * aloco_sync_ex).  Equivalent to aloco_sync_ex(..., NULL). */
int aloco_sync(float *global, float *momentum, void *const *locals,
               size_t N, int M, aloco_dtype dtype, int64_t H_sel,
               int64_t H_base, int64_t step,
               const aloco_schedule_t *schedule, double outer_lr,
               double outer_beta, aloco_stats_t *stats_out);

/* One outer synchronisation round (Algorithm 1: synchronisation, corrected
 * Nesterov outer update, replica reset, D_t and C_t).
 *   global    [N] fp32 device   theta_t in, theta_{t+1} out
 *   momentum  [N] fp32 device   v_{t-1} in, v_t out
 *   locals    host array of M device pointers; locals[m] is [N] of `dtype`,
 *             worker m's endpoint theta^(m)_{t,H} in, theta_{t+1} out
 *             (bf16: theta_{t+1} rounded to nearest even)
 *   N         parameters (0 is allowed: no kernel runs, statistics are 0)
 *   M         workers, 1 <= M <= ALOCO_MAX_WORKERS
 *   H_sel, H_base, step   executable horizons and the 0-based global inner
 *             step at which the interval began (App. B.2)
 *   schedule  inner learning-rate schedule
 *   outer_lr, outer_beta  eta_base^out and mu_base
 *   opts      NULL or options (see aloco_opts_t)
 *   stats_out NULL or host memory for the statistics
 * Buffers of any 4-byte (fp32) / 2-byte (bf16) alignment are accepted;
 * when all of them are 16-byte aligned the fused pass uses 16-byte vector
 * accesses.  Returns ALOCO_ERR_NONFINITE when some theta' or v' is NaN/Inf
 * (outputs and statistics are still written; the paper's controller treats
 * a non-finite statistic as a reduction signal, App. A.2).
 * Completion: the call returns once the round's last block has published
 * the statistics, which it does after every block has written its outputs.
 * The kernel may still be retiring on opts->stream; work queued there
 * later runs after it, and work on other streams that must follow the
 * round should wait on that stream.  The INT8 round (aloco_sync_int8)
 * behaves the same way.
 * Thread safety: calls for the same device are serialised internally. */
int aloco_sync_ex(float *global, float *momentum, void *const *locals,
                  size_t N, int M, aloco_dtype dtype, int64_t H_sel,
                  int64_t H_base, int64_t step,
                  const aloco_schedule_t *schedule, double outer_lr,
                  double outer_beta, const aloco_opts_t *opts,
                  aloco_stats_t *stats_out);

/* One outer round (as aloco_sync_ex, Algorithm 1) on state that lives in
 * host memory: theta, v and the M replicas are page-locked host arrays
 * (cudaMallocHost, or registered with cudaHostRegister); any other memory
 * is ALOCO_ERR_ARG.  The library streams them through cached device
 * staging in chunks of chunk_elems elements (0 = 2^24; rounded up to a
 * multiple of 8), overlapping the host-to-device copy of one chunk, the
 * fused kernel on another and the device-to-host copy of theta' and v' of a
 * third, on two internal copy streams and opts->stream.
 *   global, momentum  in: theta, v; out: theta', v' (fp32, N each);
 *   locals            in only: the replicas' endpoints.  The host replicas
 *                     are NOT reset; the reset replicas equal theta', which
 *                     the caller hands to its workers.
 * Per-element results are bit-identical to aloco_sync_ex on the same
 * inputs; the statistics differ only in the grouping of their partial sums
 * (fp32 per thread, then fp64), so in their last few fp32 bits.  The register
 * pass runs (opts->pass AUTO or REGISTERS; BULK_COPY is ALOCO_ERR_ARG).
 * The call returns when theta', v' and the statistics are in place.  The
 * device staging (3 chunks of (8 + M * element size) bytes each) is
 * allocated on first use, kept until aloco_shutdown, and shared by the
 * device's calls, which therefore must not overlap. */
int aloco_sync_host(float *global, float *momentum, const void *const *locals,
                    size_t N, int M, aloco_dtype dtype, int64_t H_sel,
                    int64_t H_base, int64_t step,
                    const aloco_schedule_t *schedule, double outer_lr,
                    double outer_beta, size_t chunk_elems,
                    const aloco_opts_t *opts, aloco_stats_t *stats_out);

/* ------------------------------------------------------------------------
 * Sharded rounds (the synchronisation of Algorithm 1 over a parameter vector
 * split into contiguous shards, for instance one shard per GPU).
 *
 * Every element of the round depends only on its own inputs and the round's
 * scalars (rho, mu_t, eta_out come from the schedule, not from the data), so
 * a shard can run the whole fused pass on its own range.  Only D_t and C_t
 * (Eq. adaptive-h-core-diagnostics) are sums over the whole vector: each
 * shard returns its partial sums, the shards' partials are exchanged (an
 * all-gather of one small struct per shard), and every holder combines them
 * in the same fixed shard order, so all of them obtain the same statistics.
 * ---------------------------------------------------------------------- */

/* Partial sums of one shard of a round, before combination. */
typedef struct aloco_partials {
    double drift[ALOCO_MAX_WORKERS];  /* sum over the shard of Delta_m^2      */
    double sum_sq;                    /* sum over the shard of the squared
                                         aggregate, in the pass's own units   */
    double sq_scale;                  /* factor that turns the summed sum_sq
                                         into ||Dbar||^2 (1/M^2 for the plain
                                         round, which sums (sum_m Delta_m)^2;
                                         1 for the INT8 round)                */
    double eps;                       /* opts->eps of the shard               */
    aloco_correction_t corr;          /* correction context applied           */
    int64_t nonfinite;                /* elements whose theta' or v' is not
                                         finite                               */
    int64_t n;                        /* elements of the shard                */
    int32_t M;
    int32_t pass_used;                /* aloco_pass that ran (0: empty shard) */
    float kernel_ms;                  /* fused-pass duration, or -1           */
    int32_t reserved;
} aloco_partials_t;

/* One shard of an outer round: aloco_sync_ex on the n_shard elements that
 * global, momentum and locals[m] point to (the shard's first element), but
 * instead of the finished statistics it returns the shard's partial sums in
 * *partials_out (required).  theta', v' and the replica reset of the shard are
 * written in place and equal aloco_sync_ex's on the same elements bit for bit
 * (the fused pass is elementwise); only the grouping of the partial sums
 * differs from an unsharded round.  The kernel is chosen for the shard's size
 * (see aloco_pass); shards whose pointers are 16-byte aligned keep the
 * vector paths.  n_shard = 0 is allowed (no kernel runs; zero partials with
 * the correction context).  Returns ALOCO_ERR_NONFINITE, with the partials
 * filled, when the shard produced a non-finite theta' or v'.  Other
 * arguments, errors and the wait as aloco_sync_ex. */
int aloco_sync_shard(float *global, float *momentum, void *const *locals,
                     size_t n_shard, int M, aloco_dtype dtype, int64_t H_sel,
                     int64_t H_base, int64_t step,
                     const aloco_schedule_t *schedule, double outer_lr,
                     double outer_beta, const aloco_opts_t *opts,
                     aloco_partials_t *partials_out);

/* The INT8-communicated round (aloco_sync_int8) on one shard.  The shard's
 * part_sizes describe the tensor parts it holds; codec blocks restart at
 * every part, so a shard made of whole tensor parts encodes exactly the
 * blocks the unsharded round would.  Partials as aloco_sync_shard. */
int aloco_sync_int8_shard(float *global, float *momentum, void *const *locals,
                          size_t n_shard, int M, aloco_dtype dtype,
                          int64_t H_sel, int64_t H_base, int64_t step,
                          const aloco_schedule_t *schedule, double outer_lr,
                          double outer_beta, const int64_t *part_sizes,
                          int n_parts, const aloco_opts_t *opts,
                          aloco_partials_t *partials_out);

/* Combine the partials of n_shards >= 1 shards of one round (host only, no
 * GPU): the drift energies, the squared aggregate and the non-finite counts
 * are added shard by shard in array order, then
 *   D = (1/M) sum_m drift_m,  ||Dbar||^2 = sq_scale sum_sq,
 *   C = M ||Dbar||^2 / (D + eps)          (Eq. adaptive-h-core-diagnostics).
 * Every holder that combines the same partials in the same order obtains
 * bit-identical statistics.  stats_out->grid is n_shards, kernel_ms the
 * largest shard's time (or -1), pass_used the first non-empty shard's.
 * ALOCO_ERR_ARG when the shards disagree on M, eps, sq_scale or the
 * correction context (they are not shards of one round); ALOCO_ERR_NONFINITE,
 * with the statistics filled, when any shard counted a non-finite element or
 * D or C is not finite. */
int aloco_combine_partials(const aloco_partials_t *shards, int n_shards,
                           aloco_stats_t *stats_out);

/* ------------------------------------------------------------------------
 * INT8 pseudo-gradient communication (App. G.1).
 *
 * Blocks: the flattened vector is a sequence of tensor parts (part_sizes,
 * n_parts <= 1024; NULL means one part of N); each part is cut into
 * consecutive blocks of at most 4096 elements starting at its first
 * element.  Codec, in FP32: scale = max|y| / 127 per block (1 for an all-zero
 * block; kept within [FLT_MIN, FLT_MAX / 127]), q = y / scale rounded to the
 * nearest integer with ties to even and clipped to [-127, 127], decoded value
 * q * scale.  One worker's payload per sync is N bytes of codes plus 4 bytes
 * per block (aloco_int8_num_blocks).
 * ---------------------------------------------------------------------- */

/* Number of codec blocks of a vector made of the given parts, or -1. */
int64_t aloco_int8_num_blocks(const int64_t *part_sizes, int n_parts);

/* Encode an fp32 device vector x[N]: codes[N] (int8), scales[num_blocks]
 * (fp32) and, when decoded != NULL, decoded[N] = codes * scale.  Device
 * buffers; enqueued on `stream` (cudaStream_t, NULL = default) without
 * waiting. */
int aloco_int8_encode(const float *x, size_t N, const int64_t *part_sizes,
                      int n_parts, int8_t *codes, float *scales,
                      float *decoded, void *stream);

/* Decode codes[N] with scales[num_blocks] into out[N] (device buffers,
 * enqueued on `stream`). */
int aloco_int8_decode(const int8_t *codes, const float *scales, size_t N,
                      const int64_t *part_sizes, int n_parts, float *out,
                      void *stream);

/* One outer round with INT8-communicated pseudo-gradients (App. G.1): every
 * worker's FP32 pseudo-gradient is encoded and decoded blockwise, the decoded
 * contributions are averaged in FP32 (in worker order), the mean is encoded
 * and decoded once, and that aggregate drives the corrected Nesterov step and
 * the replica reset.  D_t and the drift energies use the pre-quantisation
 * pseudo-gradients, C_t and ||Dbar||^2 the decoded aggregate.  Arguments as
 * aloco_sync_ex plus the parts; M <= 16; opts->pass selects the form
 * (AUTO, INT8_SPLIT or INT8_FUSED; see aloco_pass) and blocks_per_sm does
 * not apply. */
int aloco_sync_int8(float *global, float *momentum, void *const *locals,
                    size_t N, int M, aloco_dtype dtype, int64_t H_sel,
                    int64_t H_base, int64_t step,
                    const aloco_schedule_t *schedule, double outer_lr,
                    double outer_beta, const int64_t *part_sizes, int n_parts,
                    const aloco_opts_t *opts, aloco_stats_t *stats_out);

/* ------------------------------------------------------------------------
 * Inner optimizer (Sec. 2, Eq. diloco-local-trajectory: every worker takes
 * H local AdamW steps between synchronisations; Tab. training settings:
 * AdamW coefficients (0.9, 0.95) for C4 and (0.9, 0.999) for SFT, weight
 * decay 0.1 / 0, gradient-norm clipping 1.0, FP32 master parameters and
 * optimizer states).  The paper's runs compute the gradients from data; this
 * library takes them as inputs, so a caller can drive whole intervals on one
 * GPU with synthetic gradients.
 *
 * One step on each of the M replicas:
 *   c_m = min(1, max_grad_norm / (||g_m|| + 1e-6))   (1 if max_grad_norm <= 0)
 *   m'  = beta1 m + (1 - beta1) c_m g
 *   v'  = beta2 v + (1 - beta2) (c_m g)^2
 *   x'  = x - lr weight_decay x
 *           - lr (m' / (1 - beta1^step)) / (sqrt(v' / (1 - beta2^step)) + eps)
 * in fp32 arithmetic per element; ||g_m|| is summed in fp64 over the whole
 * replica in a fixed order.
 * ---------------------------------------------------------------------- */

typedef struct aloco_adamw_cfg {
    double lr;             /* this step's inner learning rate eta_{t,h} > 0  */
    double beta1;          /* first-moment coefficient, in [0, 1)            */
    double beta2;          /* second-moment coefficient, in [0, 1)           */
    double eps;            /* denominator guard, > 0                         */
    double weight_decay;   /* decoupled decay coefficient, >= 0              */
    double max_grad_norm;  /* per-replica clipping threshold; <= 0: none     */
    int64_t step;          /* 1-based index of this step (bias correction)   */
} aloco_adamw_cfg_t;

/* Per-replica results of one step. */
typedef struct aloco_adamw_stats {
    double grad_norm[ALOCO_MAX_WORKERS];  /* ||g_m|| before clipping         */
    double clip[ALOCO_MAX_WORKERS];       /* c_m applied                     */
    int32_t M;
    int32_t grid;                         /* CUDA blocks of the update pass  */
    float kernel_ms;                      /* both passes, or -1              */
    int32_t reserved;
} aloco_adamw_stats_t;

/* The C4 pre-training settings: lr 4e-4, (0.9, 0.95), eps 1e-8, weight
 * decay 0.1, clipping at 1.0, step 1. */
void aloco_adamw_default_cfg(aloco_adamw_cfg_t *cfg);

/* One AdamW step on M <= ALOCO_MAX_WORKERS replicas, in place.
 *   params[m]     x_m, N elements of param_dtype (fp32 or bf16; bf16 results
 *                 are rounded to nearest even), updated;
 *   grads[m]      g_m, N elements of grad_dtype, read only;
 *   exp_avg[m], exp_avg_sq[m]   m and v, fp32, updated.
 * Host arrays of M device pointers to caller-owned device memory of the
 * current device; no two updated buffers may overlap.  opts (NULL =
 * defaults) supplies the stream, kernel timing and blocks_per_sm; the
 * correction and pass fields do not apply.  With stats_out == NULL the call
 * only enqueues its two kernels; otherwise it waits for them and fills
 * *stats_out.  Returns ALOCO_OK, ALOCO_ERR_ARG / ALOCO_ERR_ALIAS before any
 * device work, or ALOCO_ERR_CUDA.  Calls on one device share its scratch:
 * steps that overlap on the GPU (different streams, no ordering) race. */
int aloco_adamw_step(void *const *params, const void *const *grads,
                     float *const *exp_avg, float *const *exp_avg_sq, size_t N,
                     int M, aloco_dtype param_dtype, aloco_dtype grad_dtype,
                     const aloco_adamw_cfg_t *cfg, const aloco_opts_t *opts,
                     aloco_adamw_stats_t *stats_out);

/* aloco_adamw_step for callers that already have the replicas' gradient
 * norms (for instance from the backward pass that produced the gradients):
 * grad_norms is a host array of M finite, non-negative values ||g_m||.  The
 * clipping factors are formed from them on the host, exactly as
 * aloco_adamw_step forms them from its own norms, and only the update pass
 * runs, reading each gradient once.  stats_out (optional) reports the given
 * norms and the factors applied; with stats_out == NULL the call only
 * enqueues.  Other arguments and errors as aloco_adamw_step. */
int aloco_adamw_step_normed(void *const *params, const void *const *grads,
                            float *const *exp_avg, float *const *exp_avg_sq,
                            size_t N, int M, aloco_dtype param_dtype,
                            aloco_dtype grad_dtype, const aloco_adamw_cfg_t *cfg,
                            const double *grad_norms, const aloco_opts_t *opts,
                            aloco_adamw_stats_t *stats_out);

/* ------------------------------------------------------------------------
 * Interval controller (Sec. 3.1; App. A).  Host-only and scalar: after each
 * completed interval it takes that interval's D_t, C_t, accumulated inner
 * learning rate and token count, assesses them against the accepted-horizon
 * reference profile and returns the horizon of the next interval, in tokens
 * and in executable steps, together with the step horizon of one base token
 * interval (the H_base argument of aloco_sync).
 *
 * Rules followed (App. A.1-A.3; Tab. AutoLoCo configuration):
 *   - the recipe horizon H_base runs through the inner-lr warm-up; from the
 *     interval that completes warm-up, ref_bootstrap finite intervals set
 *     D_ref, C_ref to geometric means; variability_intervals more intervals
 *     fill the residual histories; then one monitoring interval;
 *   - residuals r_D = log(sqrt(D)/(sqrt(D_ref) xi + eps) + eps),
 *     r_C = -log(C/(C_ref + eps) + eps), xi = Lambda/(Lambda_ref + eps)
 *     (Eqs. adaptive-h-lr-mass, adaptive-h-core-residuals); centre = median,
 *     scale = MAD of at most 16 residuals; z = max of the positive parts
 *     over the scales (Eq. adaptive-h-core-deviation);
 *   - z < 1.5 supports an increase, < 2.5 is reference consistent, < 4.0 is
 *     a moderate deviation (two in a row reduce by 1.20), otherwise severe
 *     (reduce by 1.50); a non-finite statistic takes the severe path, and
 *     consecutive severe or invalid intervals fall back to H_min
 *     (Tab. adaptive-h-assessment); only the first reference estimate skips
 *     non-finite intervals instead ("two finite intervals", App. A.1);
 *   - a supported monitoring interval proposes the longest admissible horizon
 *     whose previewed accumulated inner lr is at most 1.15 times that of the
 *     accepted horizon, or, while a rejected-horizon bound is active, the
 *     admissible horizon nearest the geometric midpoint of accepted and
 *     bound; the bound retires once its previewed exposure falls to 0.90 of
 *     the value stored when it was set;
 *   - a candidate is adopted after one supported interval, or two intervals
 *     of which the first is consistent and the second supported or
 *     consistent; a moderate or severe candidate interval is rejected and the
 *     accepted horizon restored; after adoption, return or reduction the
 *     reference is re-estimated (one interval) and its variability measured
 *     again before the next proposal;
 *   - token mapper: M_base = median token mass of the first three recipe-
 *     horizon intervals, n_hat = EMA (beta) of tokens per step; the step
 *     horizon is the multiple of q_H nearest M_base H_tok / (H_base n_hat),
 *     the identity before calibration (Eq. adaptive-h-token-mapping).
 * Horizons are admissible when they are multiples of q_H within
 * [H_min, H_max]; ties between two nearest horizons take the smaller.
 * ---------------------------------------------------------------------- */

#define ALOCO_CTRL_HISTORY 16

typedef enum {
    ALOCO_ASSESS_NONE = 0,        /* not assessed (warm-up, calibration)   */
    ALOCO_ASSESS_SUPPORTED = 1,   /* z < thr_candidate                     */
    ALOCO_ASSESS_CONSISTENT = 2,  /* z < thr_moderate                      */
    ALOCO_ASSESS_MODERATE = 3,    /* z < thr_severe                        */
    ALOCO_ASSESS_SEVERE = 4,      /* z >= thr_severe                       */
    ALOCO_ASSESS_INVALID = 5      /* a required statistic is not finite    */
} aloco_assessment;

typedef enum {
    ALOCO_PHASE_WARMUP = 0,
    ALOCO_PHASE_REFERENCE = 1,    /* estimating D_ref, C_ref, Lambda_ref   */
    ALOCO_PHASE_VARIABILITY = 2,  /* filling the residual histories        */
    ALOCO_PHASE_MONITOR = 3,      /* at the accepted horizon               */
    ALOCO_PHASE_CANDIDATE = 4,    /* first interval at a longer candidate  */
    ALOCO_PHASE_CONFIRM = 5       /* second interval at the candidate      */
} aloco_ctrl_phase;

/* Controller settings.  aloco_ctrl_default_cfg() fills the paper's shared
 * settings (Tab. AutoLoCo configuration) and the readings where the paper
 * gives no value (ref_ema, mad_scale, scale_floor, severe_fallback). */
typedef struct aloco_ctrl_cfg {
    int64_t H_base;               /* recipe token horizon (500 C4, 100 SFT)*/
    int64_t H_min, H_max;         /* token-horizon bounds                  */
    int64_t q_H;                  /* horizon quantum                       */
    int64_t warmup_steps;         /* inner-lr warm-up held at H_base       */
    double beta_tok;              /* token-density EMA coefficient, 0.9    */
    double thr_candidate;         /* 1.5 */
    double thr_moderate;          /* 2.5 */
    double thr_severe;            /* 4.0 */
    double exposure_mult;         /* 1.15 */
    double div_moderate;          /* 1.20 */
    double div_severe;            /* 1.50 */
    double retire_frac;           /* 0.90 */
    double ref_ema;               /* weight of a new interval in the
                                     log-space EMA of D_ref, C_ref (0.1)   */
    double mad_scale;             /* scale = mad_scale * MAD (1.4826)      */
    double scale_floor;           /* lower bound of a residual scale (1e-3)*/
    double eps;                   /* 1e-8 */
    int32_t mapper_bootstrap;     /* 3 */
    int32_t ref_bootstrap;        /* 2 */
    int32_t variability_intervals;/* 3 */
    int32_t severe_fallback;      /* consecutive severe/invalid -> H_min (2)*/
} aloco_ctrl_cfg_t;

/* Controller state: plain data, so it can be checkpointed by copying the
 * bytes (aloco_ctrl_save / aloco_ctrl_load add a version check). */
typedef struct aloco_ctrl_state {
    int32_t version;
    int32_t phase;                /* aloco_ctrl_phase of the next interval */
    int64_t intervals;            /* completed intervals observed          */
    int64_t H_acc;                /* accepted token horizon                */
    int64_t H_next;               /* token horizon of the next interval    */
    int64_t H_cand;               /* candidate under evaluation, 0 if none */
    int64_t bound;                /* rejected-horizon bound, 0 if none     */
    double bound_lam;             /* Lambda observed when the bound was set*/
    int32_t phase_count;          /* intervals completed in this phase     */
    int32_t ref_needed;           /* intervals the reference estimate uses */
    int32_t moderate_run;
    int32_t severe_run;
    double log_D_ref, log_C_ref, lam_ref;
    double sum_log_D, sum_log_C;  /* reference bootstrap accumulators      */
    int32_t n_hist, head;         /* residual ring (shared by D and C)     */
    double hist_D[ALOCO_CTRL_HISTORY], hist_C[ALOCO_CTRL_HISTORY];
    int32_t mapper_n, calibrated;
    double mapper_mass[8];
    double M_base, n_hat;
    double last_z, last_r_D, last_r_C;
    int32_t last_assessment;
    int32_t referenced;           /* 1 once a reference profile was set    */
} aloco_ctrl_state_t;

/* One completed interval. */
typedef struct aloco_interval_obs {
    double D;                     /* local-drift energy (aloco_stats_t.D)  */
    double C;                     /* aggregation coherence                 */
    double lam;                   /* accumulated inner lr of the interval  */
    double tokens;                /* non-padding tokens M_t it processed   */
    int64_t H_step;               /* steps it executed                     */
    int64_t step_end;             /* global inner step at which it ended   */
} aloco_interval_obs_t;

/* The controller's answer for the next interval. */
typedef struct aloco_ctrl_decision {
    int64_t H_tok;                /* token horizon H_{t+1}^tok             */
    int64_t H_step;               /* executable steps H_{t+1}^step         */
    int64_t H_ref_step;           /* steps of one base token interval      */
    int32_t assessment;           /* of the completed interval             */
    int32_t phase;                /* aloco_ctrl_phase of the next interval */
    double z, r_D, r_C;           /* z_t^max and residuals (0 if none)     */
} aloco_ctrl_decision_t;

/* Fill *cfg with the paper's settings for a recipe horizon H_base, bounds
 * [H_min, H_max], quantum q_H and an inner-lr warm-up of warmup_steps. */
void aloco_ctrl_default_cfg(aloco_ctrl_cfg_t *cfg, int64_t H_base,
                            int64_t H_min, int64_t H_max, int64_t q_H,
                            int64_t warmup_steps);

/* Start a run: the first interval executes H_base.  Returns ALOCO_ERR_ARG
 * for an inconsistent cfg (H_min <= H_base <= H_max, all multiples of q_H,
 * thresholds increasing, ...). */
int aloco_ctrl_init(aloco_ctrl_state_t *state, const aloco_ctrl_cfg_t *cfg,
                    aloco_ctrl_decision_t *first);

/* Feed one completed interval and choose the next one (App. A).  The
 * schedule is used to preview accumulated inner learning rates from
 * obs->step_end.  state is updated in place. */
int aloco_select_interval(aloco_ctrl_state_t *state,
                          const aloco_ctrl_cfg_t *cfg,
                          const aloco_interval_obs_t *obs,
                          const aloco_schedule_t *schedule,
                          aloco_ctrl_decision_t *out);

/* Serialise / restore a controller state (checkpoint and resume).  save
 * writes aloco_ctrl_state_bytes() bytes; load checks the version. */
size_t aloco_ctrl_state_bytes(void);
int aloco_ctrl_save(const aloco_ctrl_state_t *state, void *buf, size_t len);
int aloco_ctrl_load(aloco_ctrl_state_t *state, const void *buf, size_t len);

/* Block partials the scratch of aloco_sync_noalloc can hold. */
#define ALOCO_NOALLOC_MAX_BLOCKS 2048

/* aloco_sync_ex without any memory allocation by the library.
 *
 * The paper has no counterpart: this entry point exists for callers that
 * cannot let a library allocate device or pinned host memory -- frameworks
 * that reserve the whole GPU memory up front and serve it from their own
 * pools, deployments whose memory footprint must be fixed when the library
 * is loaded, and loops that cannot afford the device-wide synchronisation
 * that cudaMalloc / cudaFree imply.  aloco_sync_ex, by contrast, allocates a
 * cached per-device workspace on its first call.
 *
 * Arguments, results, status codes and numerics are those of aloco_sync_ex:
 * the kernel is chosen by the same rule from opts->pass, M, dtype and N (the
 * tile, bulk-copy or register pass; pass_used reports it) and launched with
 * the same grid, so theta', v', the replicas and the fixed-order statistics
 * equal aloco_sync_ex's bit for bit on the same inputs.  Exceptions:
 * opts->time_kernel is ignored (stats_out->kernel_ms is -1), and the call
 * cannot run under stream capture (it ends with a stream synchronisation;
 * a call on a capturing stream returns ALOCO_ERR_ARG before enqueuing
 * anything).  The caller still provides every input and output buffer.
 *
 * Scratch: the per-block partial sums live in one statically sized device
 * array inside the library (about 560 KB: ALOCO_NOALLOC_MAX_BLOCKS rows of
 * ALOCO_MAX_WORKERS + 1 doubles plus counters), which every GPU that loads
 * the library holds until the process exits.  A round that would need more
 * than ALOCO_NOALLOC_MAX_BLOCKS blocks is rejected with ALOCO_ERR_ARG and a
 * message naming both numbers.  Every pass caps its blocks at the kernel's
 * occupancy whatever opts->blocks_per_sm asks for: at most SMs x 8 blocks
 * (1216 on a 152-SM GB300), so only a device with more than 256 SMs can be
 * refused.  Statistics are read back with cudaMemcpyAsync into a buffer on
 * the calling thread's stack; no cudaMalloc, cudaFree, cudaMallocHost or
 * other allocating routine is called.
 *
 * The first call on a device resolves the scratch array's device address
 * (cudaGetSymbolAddress, with that device current).  All calls on a device
 * share the one array and it keeps the previous call's contents: each call
 * clears the counter and the error word that must start at zero, and every
 * other scratch value a round reads is written by that round first.  Rounds
 * that overlapped on the GPU would race on the array; within a process the
 * library prevents that by holding a per-device lock for the whole call,
 * which returns only after its round has completed. */
int aloco_sync_noalloc(float *global, float *momentum, void *const *locals,
                       size_t N, int M, aloco_dtype dtype, int64_t H_sel,
                       int64_t H_base, int64_t step,
                       const aloco_schedule_t *schedule, double outer_lr,
                       double outer_beta, const aloco_opts_t *opts,
                       aloco_stats_t *stats_out);

/* TESTING ONLY (failure detection without a GPU fault): the calling
 * thread's next round that runs the bulk-copy pass (aloco_sync /
 * aloco_sync_ex) or the fused INT8 pass (aloco_sync_int8) skips the copies
 * of tile `tile` (bulk-copy pass) or of codec block `tile` (fused INT8
 * pass, a whole aligned block); a negative value cancels.  That stage's
 * mbarrier then never completes, so the bounded waits on it (about 2 s) run
 * out: the block aborts, lets its copies in flight land, and the round
 * returns ALOCO_ERR_CUDA with every kernel finished and the device usable.
 * The hook is consumed by that round; no other call reads it. */
void aloco_test_stall_tile(int64_t tile);

/* Message of the last failure on the calling thread ("" if none).  The
 * pointer stays valid until the next call on this thread. */
const char *aloco_last_error(void);

/* Release the library's cached per-device workspaces (device and pinned
 * host memory).  Safe to call at any time no round is in flight. */
void aloco_shutdown(void);

/* Library version, major * 10000 + minor * 100 + patch. */
int aloco_version(void);

#ifdef __cplusplus
}
#endif

#endif /* ALOCO_H */
