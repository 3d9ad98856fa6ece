// Fused outer-synchronisation pass with bulk-copy (TMA) staging.
//
// One persistent CTA per SM: a producer warp streams, tile by tile, the
// theta, v and replica tiles of the round into an S-stage ring in shared
// memory with cp.async.bulk (one contiguous 4 KB (fp32) / 8 KB (bf16 theta,
// v) copy per array and tile, completing on the stage's "full" mbarrier);
// eight consumer warps read the stage, form the pseudo-gradients, the
// drift-energy partials and the corrected Nesterov step exactly as the
// register-streaming kernel does, store theta', v' and the replica reset
// with 16-byte stores, and release the stage on its "empty" mbarrier.
// Bytes in flight per SM are set by the ring (S x stage bytes, ~200 KB),
// not by register occupancy.
//
// Every mbarrier wait is bounded: after ~2 s without progress the waiting
// thread raises the block's abort flag and the round's error word, the
// consumers stop, and the producer waits (again bounded) for the copies it
// still has in flight before the block exits.  The host reports the error.
#pragma once

#include "aloco_bulk.cuh"
#include "aloco_sync_kernel.cuh"

namespace aloco {

constexpr int kTmaConsumers = kTmaTilePacks;       // 8 consumer warps
constexpr int kTmaThreads = kTmaConsumers + 32;     // + 1 producer warp
constexpr int kTmaMaxStages = 8;
// Bytes of one stage: theta and v tiles (fp32) and M replica tiles.
template <bool BF16>
__host__ __device__ constexpr uint32_t tma_gv_bytes() {
    return kTmaConsumers * Pack<BF16>::E * 4;
}
__host__ __device__ constexpr uint32_t tma_x_bytes() { return kTmaConsumers * 16; }
template <bool BF16>
__host__ __device__ constexpr uint32_t tma_stage_bytes(int M) {
    return 2 * tma_gv_bytes<BF16>() + (uint32_t)M * tma_x_bytes();
}

template <int MT, bool BF16>
__global__ void __launch_bounds__(kTmaThreads, 1)
    sync_tma_kernel(const __grid_constant__ SyncArgs a) {
    static_assert(MT > 0, "the bulk-copy pass needs a compile-time M");
    using P = Pack<BF16>;
    constexpr int E = P::E;
    constexpr int M = MT;
    constexpr uint32_t kGV = tma_gv_bytes<BF16>();
    constexpr uint32_t kX = tma_x_bytes();
    constexpr uint32_t kStage = tma_stage_bytes<BF16>(M);

    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ __align__(8) unsigned long long full_bar[kTmaMaxStages];
    __shared__ __align__(8) unsigned long long empty_bar[kTmaMaxStages];
    __shared__ int abort_flag;
    volatile int *abort_v = &abort_flag;

    const int S = a.stages;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(smem_addr(&full_bar[s]), 1);
            mbar_init(smem_addr(&empty_bar[s]), kTmaConsumers);
        }
        abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

    float e32[M];
    double e64[M];
#pragma unroll
    for (int m = 0; m < M; ++m) {
        e32[m] = 0.f;
        e64[m] = 0.0;
    }
    float b32 = 0.f;
    double b64 = 0.0;
    unsigned nf = 0;
    int cnt = 0;
    const Coef k{a.c_hi, a.c_lo, a.mu_hi, a.mu_lo, a.neg_eta_hi, a.neg_eta_lo};
    auto flush = [&]() {
#pragma unroll
        for (int m = 0; m < M; ++m) {
            e64[m] += (double)e32[m];
            e32[m] = 0.f;
        }
        b64 += (double)b32;
        b32 = 0.f;
    };
    // One pack: gg / vv / X are theta, v and the M replica packs.
    auto process = [&](int64_t i, const float (&gg)[E], const float (&vv)[E],
                       const typename P::Raw (&X)[M]) {
        float s[E];
#pragma unroll
        for (int j = 0; j < E; ++j) s[j] = 0.f;
#pragma unroll
        for (int m = 0; m < M; ++m) {
            float xx[E];
            P::widen(X[m], xx);
#pragma unroll
            for (int j = 0; j < E; ++j) {
                const float d = gg[j] - xx[j];
                s[j] += d;
                e32[m] = fmaf(d, d, e32[m]);
            }
        }
        float gp[E], vp[E];
#pragma unroll
        for (int j = 0; j < E; ++j) {
            b32 = fmaf(s[j], s[j], b32);
            outer_step(k, s[j], gg[j], vv[j], gp[j], vp[j]);
            nf += not_finite(gp[j], vp[j]);
        }
        P::store(a.g, i, gp);
        P::store(a.v, i, vp);
        const typename P::Raw xo = P::narrow(gp);
#pragma unroll
        for (int m = 0; m < M; ++m) P::store_x(a.x[m], i, xo);
        if (++cnt == kFlush) {
            flush();
            cnt = 0;
        }
    };

    const int64_t G = gridDim.x, b = blockIdx.x;
    const int64_t my_tiles = b < a.n_tiles ? (a.n_tiles - 1 - b) / G + 1 : 0;
    const uint32_t ring = smem_addr(smem);

    if (warp == kTmaConsumers / 32) {
        // ------------------------------------------------------ producer
        if (lane == 0) {
            int64_t issued = 0;
            for (int64_t j = 0; j < my_tiles; ++j) {
                const int s = (int)(j % S);
                if (j >= S &&
                    !mbar_wait(smem_addr(&empty_bar[s]), (uint32_t)((j / S - 1) & 1),
                               abort_v)) {
                    *abort_v = 1;
                    atomicExch(a.error, 1u);
                    break;
                }
                if (*abort_v) break;
                const int64_t t = b + j * G;
                if (a.test_stall_tile1 != 0 && t == a.test_stall_tile1 - 1) {
                    // testing only: this stage's full barrier never completes,
                    // so the consumers' bounded wait runs out
                    issued = j + 1;
                    continue;
                }
                const uint32_t st = ring + (uint32_t)s * kStage;
                const uint32_t fb = smem_addr(&full_bar[s]);
                mbar_arrive_expect_tx(fb, kStage);
                bulk_load(st, reinterpret_cast<const char *>(a.g) + t * kGV, kGV, fb);
                bulk_load(st + kGV, reinterpret_cast<const char *>(a.v) + t * kGV, kGV,
                          fb);
#pragma unroll
                for (int m = 0; m < M; ++m)
                    bulk_load(st + 2 * kGV + m * kX,
                              reinterpret_cast<const char *>(a.x[m]) + t * kX, kX, fb);
                issued = j + 1;
            }
            if (*abort_v) {
                // let the copies still in flight land before the block exits
                const int64_t first = issued > S ? issued - S : 0;
                for (int64_t j = first; j < issued; ++j)
                    mbar_wait(smem_addr(&full_bar[j % S]), (uint32_t)((j / S) & 1),
                              nullptr);
            }
        }
    } else {
        // ----------------------------------------------------- consumers
        const int ct = threadIdx.x;
        for (int64_t j = 0; j < my_tiles; ++j) {
            const int s = (int)(j % S);
            if (!mbar_wait(smem_addr(&full_bar[s]), (uint32_t)((j / S) & 1), abort_v)) {
                *abort_v = 1;
                atomicExch(a.error, 1u);
                break;
            }
            const unsigned char *st = smem + (size_t)s * kStage;
            float gg[E], vv[E];
            typename P::Raw X[M];
            {
                const float4 *g4 = reinterpret_cast<const float4 *>(st) + ct * (E / 4);
                const float4 *v4 =
                    reinterpret_cast<const float4 *>(st + kGV) + ct * (E / 4);
#pragma unroll
                for (int q = 0; q < E / 4; ++q) {
                    const float4 gq = g4[q], vq = v4[q];
                    gg[4 * q] = gq.x; gg[4 * q + 1] = gq.y;
                    gg[4 * q + 2] = gq.z; gg[4 * q + 3] = gq.w;
                    vv[4 * q] = vq.x; vv[4 * q + 1] = vq.y;
                    vv[4 * q + 2] = vq.z; vv[4 * q + 3] = vq.w;
                }
#pragma unroll
                for (int m = 0; m < M; ++m)
                    X[m] = reinterpret_cast<const typename P::Raw *>(
                        st + 2 * kGV + m * kX)[ct];
            }
            // every consumer releases the stage once its reads are done
            mbar_arrive(smem_addr(&empty_bar[s]));
            const int64_t t = b + j * G;
            process(t * kTmaConsumers + ct, gg, vv, X);
        }
        // packs after the last whole tile, then the element-wise remainder
        if (!*abort_v) {
            const int64_t tid = b * kTmaConsumers + ct;
            const int64_t stride = G * kTmaConsumers;
            for (int64_t i = a.n_tiles * kTmaConsumers + tid; i < a.nvec; i += stride) {
                float gg[E], vv[E];
                typename P::Raw X[M];
                P::load(a.g, i, gg);
                P::load(a.v, i, vv);
#pragma unroll
                for (int m = 0; m < M; ++m) X[m] = P::load_x(a.x[m], i);
                process(i, gg, vv, X);
            }
            for (int64_t jj = a.nvec * E + tid; jj < a.n; jj += stride) {
                const float g = a.g[jj];
                const float v = a.v[jj];
                float s = 0.f;
#pragma unroll
                for (int m = 0; m < M; ++m) {
                    float x;
                    if constexpr (BF16)
                        x = __uint_as_float(
                            (uint32_t)(reinterpret_cast<const uint16_t *>(a.x[m])[jj])
                            << 16);
                    else
                        x = reinterpret_cast<const float *>(a.x[m])[jj];
                    const float d = g - x;
                    s += d;
                    e32[m] = fmaf(d, d, e32[m]);
                }
                b32 = fmaf(s, s, b32);
                float gp, vp;
                outer_step(k, s, g, v, gp, vp);
                nf += not_finite(gp, vp);
                a.g[jj] = gp;
                a.v[jj] = vp;
#pragma unroll
                for (int m = 0; m < M; ++m) {
                    if constexpr (BF16)
                        reinterpret_cast<__nv_bfloat16 *>(a.x[m])[jj] =
                            __float2bfloat16_rn(gp);
                    else
                        reinterpret_cast<float *>(a.x[m])[jj] = gp;
                }
            }
        }
    }
    flush();
    reduce_and_finish<M, kTmaThreads / 32>(a, M, e64, b64, nf);
}

// Largest ring that fits the shared-memory budget, 2..kTmaMaxStages stages.
template <bool BF16>
constexpr int tma_stages(int M, int smem_budget) {
    int s = smem_budget / (int)tma_stage_bytes<BF16>(M);
    return s > kTmaMaxStages ? kTmaMaxStages : s;
}

template <int MT, bool BF16>
cudaError_t plan_tma_one(int64_t nvec, int sm_count, int smem_budget,
                         LaunchPlan *plan) {
    static PerDevice configured;  // the shared-memory attribute, per device
    const int stages = tma_stages<BF16>(MT, smem_budget);
    if (stages < 2) return cudaErrorInvalidValue;
    const int smem = stages * (int)tma_stage_bytes<BF16>(MT);
    const int dev = PerDevice::device();
    if (!configured.get(dev)) {
        cudaError_t e = cudaFuncSetAttribute(
            sync_tma_kernel<MT, BF16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
            smem_budget);
        if (e != cudaSuccess) return e;
        configured.set(dev, 1);
    }
    const int64_t tiles = nvec / kTmaConsumers;
    plan->kernel = reinterpret_cast<const void *>(&sync_tma_kernel<MT, BF16>);
    plan->grid = sm_count;
    plan->block = kTmaThreads;
    plan->smem = smem;
    plan->stages = stages;
    plan->tiles = tiles;
    return cudaSuccess;
}

template <bool BF16>
cudaError_t plan_tma_dispatch(int M, int64_t nvec, int sm_count, int smem_budget,
                              LaunchPlan *plan) {
    switch (M) {
#define ALOCO_TMA_CASE(K) \
    case K:               \
        return plan_tma_one<K, BF16>(nvec, sm_count, smem_budget, plan);
        ALOCO_TMA_CASE(1) ALOCO_TMA_CASE(2) ALOCO_TMA_CASE(3) ALOCO_TMA_CASE(4)
        ALOCO_TMA_CASE(5) ALOCO_TMA_CASE(6) ALOCO_TMA_CASE(7) ALOCO_TMA_CASE(8)
        ALOCO_TMA_CASE(9) ALOCO_TMA_CASE(10) ALOCO_TMA_CASE(11) ALOCO_TMA_CASE(12)
        ALOCO_TMA_CASE(13) ALOCO_TMA_CASE(14) ALOCO_TMA_CASE(15) ALOCO_TMA_CASE(16)
#undef ALOCO_TMA_CASE
        default:
            return cudaErrorInvalidValue;
    }
}

}  // namespace aloco
