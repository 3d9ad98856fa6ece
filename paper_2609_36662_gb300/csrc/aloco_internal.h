// Internal interface between the host side of libaloco (aloco_host.cpp) and
// the fused synchronisation kernels (aloco_sync_*.cu).  Not part of the ABI.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "../../include/aloco.h"

namespace aloco {

// A value computed once per device and kept for the process: function
// attributes and occupancy belong to a device's context, so launch set-up is
// cached per device (zero = not yet computed).  Devices beyond kMaxDevices
// are not cached and recompute every time.
constexpr int kMaxDevices = 64;
struct PerDevice {
    std::atomic<int> v[kMaxDevices];
    static int device() {
        int d = -1;
        if (cudaGetDevice(&d) != cudaSuccess) {
            cudaGetLastError();
            return -1;
        }
        return d >= 0 && d < kMaxDevices ? d : -1;
    }
    int get(int d) const { return d >= 0 ? v[d].load(std::memory_order_acquire) : 0; }
    void set(int d, int x) {
        if (d >= 0) v[d].store(x, std::memory_order_release);
    }
};

// Threads per block of the fused pass.
constexpr int kBlock = 256;

// Everything the fused pass needs, passed by value as a __grid_constant__
// kernel parameter (the replica pointers are uniform across the grid).
struct SyncArgs {
    float *g;                       // theta [n]
    float *v;                       // momentum [n]
    void *x[ALOCO_MAX_WORKERS];     // replicas [n] each
    int64_t n;                      // elements
    int64_t nvec;                   // packs handled by the vector loop
                                    // (0 when a buffer is not 16 B aligned)
    // Round coefficients, each as an fp32 pair hi + lo whose sum carries the
    // fp64 host value to ~2^-48 relative, so that the per-element update is
    // not biased by one fixed fp32 rounding of the coefficient.
    float c_hi, c_lo;               // inv_norm / M  (Dtil = c * sum_m Delta_m)
    float mu_hi, mu_lo;             // mu_t
    float neg_eta_hi, neg_eta_lo;   // -eta_out
    int M;
    // workspace (device)
    double *partials;               // [grid][M + 1]: sum Delta_m^2 (m < M), sum S^2
    unsigned long long *nf_partials;// [grid]
    unsigned int *ticket;           // last-block-done counter, 0 between launches
    double *totals;                 // [M + 1] fixed-order totals
    unsigned long long *nf_total;   // [1]
    // bulk-copy pass only
    int64_t n_tiles;                // whole tiles of kTmaConsumers packs
    int stages;                     // depth of the shared-memory ring
    unsigned int *error;            // set to 1 if a pipeline wait timed out
    int64_t test_stall_tile1;       // testing only: 1 + the index of a tile whose
                                    // copies the producer skips (0 = none)
    // Statistics published to the host (null: not published).  The last
    // block writes the totals block (kTotalsSlots values) to this
    // device-mapped page-locked host memory, then, after a system-scope
    // fence, `seq` to slot kSeqSlot.
    double *stats_out;
    unsigned long long seq;
};

// Slots of the totals block read back after a round (8 bytes each): M + 1
// totals, then the non-finite count, then the pipeline error word.
constexpr int kTotalsSlots = ALOCO_MAX_WORKERS + 3;
constexpr int kNfSlot = ALOCO_MAX_WORKERS + 1;
constexpr int kErrorSlot = ALOCO_MAX_WORKERS + 2;
// The published round sequence number follows the totals block.
constexpr int kSeqSlot = kTotalsSlots;

// Shared memory the bulk-copy pass may use for its ring (bytes), and the
// packs of one tile (one per consumer thread).
constexpr int kTmaSmemBudget = 224 * 1024;
constexpr int kTmaTilePacks = 256;

// Elements per vector pack: one 16-byte access of a replica.
inline int pack_elems(aloco_dtype dt) { return dt == ALOCO_F32 ? 4 : 8; }

// Launch configuration chosen for (M, dtype, n) on the current device.
struct LaunchPlan {
    const void *kernel;
    int grid;
    int block;
    int smem = 0;       // dynamic shared memory (bytes)
    int stages = 0;     // bulk-copy pass: ring depth
    int64_t tiles = 0;  // bulk-copy pass: whole tiles
};

// Pick the kernel instance and grid; returns cudaSuccess or an error.
// blocks_per_sm = 0 takes the tuned residency for (M, dtype); any other
// value is used as given, capped by the kernel's occupancy limit.
cudaError_t plan_sync_f32(int M, int64_t work_items, int sm_count,
                          int blocks_per_sm, LaunchPlan *plan);
cudaError_t plan_sync_bf16(int M, int64_t work_items, int sm_count,
                           int blocks_per_sm, LaunchPlan *plan);

// The bulk-copy (TMA) pass for 1 <= M <= 16 and 16-byte aligned buffers.
cudaError_t plan_sync_tma_f32(int M, int64_t nvec, int sm_count,
                              LaunchPlan *plan);
cudaError_t plan_sync_tma_bf16(int M, int64_t nvec, int sm_count,
                               LaunchPlan *plan);

// Whether a round of M workers (dtype) uses the bulk-copy pass, given the
// requested aloco_pass.
bool use_tma(int pass, int M, aloco_dtype dtype, int64_t nvec);
// The tile pass (aloco_sync_tile.cu): M <= 16, aligned buffers, at least one
// whole block.
bool sync_tile_fits(int M, int64_t n, int64_t nvec);
bool use_tile(int pass, int M, aloco_dtype dtype, int64_t n, int64_t nvec);
cudaError_t launch_sync_tile(const SyncArgs &a, aloco_dtype dtype, int sm_count,
                             int max_grid, cudaStream_t stream, int *grid_out);
// Whether an INT8 round of M workers (dtype) uses the fused form.
bool use_int8_fused(int pass, int M, aloco_dtype dtype);

// Tensor parts of an INT8-communicated round, passed by value to the
// kernels: part p covers elements [off[p], off[p+1]) and its codec blocks
// are blk[p] .. blk[p+1]-1.
constexpr int kInt8MaxParts = 1024;
struct Int8Parts {
    int64_t off[kInt8MaxParts + 1];
    int64_t blk[kInt8MaxParts + 1];
    int n_parts;
};

// Enqueue the split form of an INT8 round (two kernels).  bmax holds
// nblocks * M unsigned (per-block worker maxima, cleared here), e_rows
// max_grid * 16 doubles (device scratch).
cudaError_t launch_int8_round(const SyncArgs &a, const Int8Parts &P,
                              aloco_dtype dtype, int sm_count, unsigned *bmax,
                              double *e_rows, int max_grid, cudaStream_t stream,
                              int *grid_out);
// The fused form (one kernel, no scratch beyond the reduction's): only
// where int8_fused_fits(M, dtype), i.e. M <= 16.
bool int8_fused_fits(int M, aloco_dtype dtype);
cudaError_t launch_int8_fused(const SyncArgs &a, const Int8Parts &P,
                              aloco_dtype dtype, int sm_count, int max_grid,
                              cudaStream_t stream, int *grid_out);
cudaError_t launch_int8_encode(const float *x, int8_t *codes, float *scales,
                               float *decoded, bool vec_ok, const Int8Parts &P,
                               int sm_count, cudaStream_t stream);
cudaError_t launch_int8_decode(const int8_t *codes, const float *scales,
                               float *out, bool vec_ok, const Int8Parts &P,
                               int sm_count, cudaStream_t stream);

// One AdamW step on M replicas (aloco_adamw.cu), passed by value.
struct AdamArgs {
    void *x[ALOCO_MAX_WORKERS];         // parameters [n] (fp32 or bf16)
    const void *g[ALOCO_MAX_WORKERS];   // gradients [n] (fp32 or bf16)
    float *m1[ALOCO_MAX_WORKERS];       // first moments [n]
    float *m2[ALOCO_MAX_WORKERS];       // second moments [n]
    int64_t n;                          // elements per replica
    int64_t nunit;                      // 4-element units of the vector loop
                                        // (0 when a buffer is not 16 B aligned)
    int M;
    int g1;                             // norm-pass blocks per worker
    float beta1, omb1;                  // beta1, 1 - beta1
    float beta2, omb2;                  // beta2, 1 - beta2
    float decay;                        // 1 - lr * weight_decay
    float neg_step;                     // -lr / (1 - beta1^step)
    float inv_sqrt_bc2;                 // 1 / sqrt(1 - beta2^step)
    float eps;
    double max_norm;                    // clipping threshold; <= 0: none
    double *partials;                   // [M][g1] sums of g^2 (device)
    double *out;                        // [2][ALOCO_MAX_WORKERS]: norms, factors
    int given;                          // 1: clip[] holds the factors; no norm pass
    float clip[ALOCO_MAX_WORKERS];      // clipping factors when given
};

// Enqueue the norm pass (grid g1 x M) and the update pass (grid g2 x M).
cudaError_t launch_adamw(const AdamArgs &a, aloco_dtype param_dtype,
                         aloco_dtype grad_dtype, int g2, cudaStream_t stream);

// Host helpers shared by the entry points (aloco_host.cpp).
int report_error(int code, const char *msg);
int check_buffer(const void *p, size_t bytes, int device, const char *name);
void fill_default_opts(aloco_opts_t *o);
void split_coef(double x, float *hi, float *lo);
// b_scale converts the last total into ||Dbar||^2: 1/M^2 when the pass
// accumulated (sum_m Delta_m)^2, 1 when it accumulated the aggregate itself.
void finalize_stats(const double *totals, unsigned long long nf, int M,
                    double eps, double b_scale, aloco_stats_t *st);

}  // namespace aloco
