// Fused outer-synchronisation pass (one launch per round).
//
// Each thread walks the parameter vector with a grid stride.  Per 16-byte
// pack it loads theta, v and the M replicas once, forms the pseudo-gradients
// Delta_m = theta - x_m (Algorithm 1), their sum S, the drift-energy and
// ||sum||^2 partials (Eq. adaptive-h-core-diagnostics), applies the
// corrected Nesterov step (Eq. autoloco-corrected-nesterov, with the
// normalisation of Eq. normalized-pseudo-gradient folded into c_avg), and
// stores theta', v' and the replica reset from the same registers.
//
// Reductions are deterministic: per-thread fp32 partials are promoted to
// fp64 every kFlush packs, threads are combined by a fixed warp-shuffle tree
// and a fixed cross-warp order into one fp64 partial per block, and the last
// block to finish (atomic ticket, no spinning) sums the block partials in
// block order.  The grid depends only on (M, dtype, n, device), so a round
// on the same inputs reproduces its statistics bit for bit.
#pragma once

#include <cuda_bf16.h>
#include <float.h>

#include "aloco_internal.h"

namespace aloco {

// Packs accumulated in fp32 before promotion to fp64: at most 64 (fp32) or
// 128 (bf16) squared terms per fp32 partial.
constexpr int kFlush = 16;

__device__ __forceinline__ float4 ldcs4(const void *base, int64_t i) {
    return __ldcs(reinterpret_cast<const float4 *>(base) + i);
}
__device__ __forceinline__ uint4 ldcs4u(const void *base, int64_t i) {
    return __ldcs(reinterpret_cast<const uint4 *>(base) + i);
}
__device__ __forceinline__ void stcs4(void *base, int64_t i, float4 val) {
    __stcs(reinterpret_cast<float4 *>(base) + i, val);
}
__device__ __forceinline__ void stcs4u(void *base, int64_t i, uint4 val) {
    __stcs(reinterpret_cast<uint4 *>(base) + i, val);
}

// Exact widening of the two bf16 values packed in a 32-bit word (element
// 2k in the low half, 2k+1 in the high half).
__device__ __forceinline__ float bf16_lo(uint32_t w) {
    return __uint_as_float(w << 16);
}
__device__ __forceinline__ float bf16_hi(uint32_t w) {
    return __uint_as_float(w & 0xFFFF0000u);
}
// Round two fp32 values to bf16 (nearest even) and pack them.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&h);
}

__device__ __forceinline__ unsigned not_finite(float a, float b) {
    return (fabsf(a) <= FLT_MAX && fabsf(b) <= FLT_MAX) ? 0u : 1u;
}

// Outer step for one element given S = sum_m Delta_m:
//   Dtil = c S ; v' = mu v + Dtil ; d = Dtil + mu v' ; g' = g - eta d
// Each coefficient is applied as hi + lo: the small lo term enters the
// addend of the FMA that carries the hi product, so the coefficient's own
// fp32 rounding does not bias every element the same way.
struct Coef {
    float c_hi, c_lo, mu_hi, mu_lo, ne_hi, ne_lo;
};
__device__ __forceinline__ void outer_step(const Coef &k, float s, float g,
                                           float v, float &gp, float &vp) {
    const float dt = fmaf(s, k.c_hi, s * k.c_lo);
    vp = fmaf(k.mu_hi, v, fmaf(k.mu_lo, v, dt));
    const float d = fmaf(k.mu_hi, vp, fmaf(k.mu_lo, vp, dt));
    gp = g + fmaf(k.ne_hi, d, k.ne_lo * d);
}

template <int MT, bool BF16>
__global__ void __launch_bounds__(kBlock)
    sync_kernel(const __grid_constant__ SyncArgs a) {
    constexpr int MM = MT > 0 ? MT : ALOCO_MAX_WORKERS;
    const int M = MT > 0 ? MT : a.M;

    float e32[MM];
    double e64[MM];
#pragma unroll
    for (int m = 0; m < MM; ++m) {
        e32[m] = 0.f;
        e64[m] = 0.0;
    }
    float b32 = 0.f;
    double b64 = 0.0;
    unsigned nf = 0;
    int cnt = 0;

    const Coef k{a.c_hi, a.c_lo, a.mu_hi, a.mu_lo, a.neg_eta_hi, a.neg_eta_lo};
    const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;

    auto flush = [&]() {
#pragma unroll
        for (int m = 0; m < MM; ++m) {
            e64[m] += (double)e32[m];
            e32[m] = 0.f;
        }
        b64 += (double)b32;
        b32 = 0.f;
    };

    // ---------------------------------------------------- vector body
    if constexpr (!BF16) {
        for (int64_t i = tid; i < a.nvec; i += stride) {
            const float4 g4 = ldcs4(a.g, i);
            const float4 v4 = ldcs4(a.v, i);
            float s[4] = {0.f, 0.f, 0.f, 0.f};
            const float gg[4] = {g4.x, g4.y, g4.z, g4.w};
#pragma unroll
            for (int m = 0; m < MM; ++m) {
                if (MT == 0 && m >= M) continue;
                const float4 x4 = ldcs4(a.x[m], i);
                const float xx[4] = {x4.x, x4.y, x4.z, x4.w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float d = gg[j] - xx[j];
                    s[j] += d;
                    e32[m] = fmaf(d, d, e32[m]);
                }
            }
            const float vv[4] = {v4.x, v4.y, v4.z, v4.w};
            float gp[4], vp[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                b32 = fmaf(s[j], s[j], b32);
                outer_step(k, s[j], gg[j], vv[j], gp[j], vp[j]);
                nf += not_finite(gp[j], vp[j]);
            }
            const float4 go = make_float4(gp[0], gp[1], gp[2], gp[3]);
            stcs4(a.g, i, go);
            stcs4(a.v, i, make_float4(vp[0], vp[1], vp[2], vp[3]));
#pragma unroll
            for (int m = 0; m < MM; ++m) {
                if (MT == 0 && m >= M) continue;
                stcs4(a.x[m], i, go);
            }
            if (++cnt == kFlush) {
                flush();
                cnt = 0;
            }
        }
    } else {
        for (int64_t i = tid; i < a.nvec; i += stride) {
            const float4 g4a = ldcs4(a.g, 2 * i), g4b = ldcs4(a.g, 2 * i + 1);
            const float4 v4a = ldcs4(a.v, 2 * i), v4b = ldcs4(a.v, 2 * i + 1);
            const float gg[8] = {g4a.x, g4a.y, g4a.z, g4a.w,
                                 g4b.x, g4b.y, g4b.z, g4b.w};
            float s[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int m = 0; m < MM; ++m) {
                if (MT == 0 && m >= M) continue;
                const uint4 x4 = ldcs4u(a.x[m], i);
                const uint32_t w[4] = {x4.x, x4.y, x4.z, x4.w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float d0 = gg[2 * j] - bf16_lo(w[j]);
                    const float d1 = gg[2 * j + 1] - bf16_hi(w[j]);
                    s[2 * j] += d0;
                    s[2 * j + 1] += d1;
                    e32[m] = fmaf(d0, d0, e32[m]);
                    e32[m] = fmaf(d1, d1, e32[m]);
                }
            }
            const float vv[8] = {v4a.x, v4a.y, v4a.z, v4a.w,
                                 v4b.x, v4b.y, v4b.z, v4b.w};
            float gp[8], vp[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                b32 = fmaf(s[j], s[j], b32);
                outer_step(k, s[j], gg[j], vv[j], gp[j], vp[j]);
                nf += not_finite(gp[j], vp[j]);
            }
            stcs4(a.g, 2 * i, make_float4(gp[0], gp[1], gp[2], gp[3]));
            stcs4(a.g, 2 * i + 1, make_float4(gp[4], gp[5], gp[6], gp[7]));
            stcs4(a.v, 2 * i, make_float4(vp[0], vp[1], vp[2], vp[3]));
            stcs4(a.v, 2 * i + 1, make_float4(vp[4], vp[5], vp[6], vp[7]));
            const uint4 xo = make_uint4(
                pack_bf16x2(gp[0], gp[1]), pack_bf16x2(gp[2], gp[3]),
                pack_bf16x2(gp[4], gp[5]), pack_bf16x2(gp[6], gp[7]));
#pragma unroll
            for (int m = 0; m < MM; ++m) {
                if (MT == 0 && m >= M) continue;
                stcs4u(a.x[m], i, xo);
            }
            if (++cnt == kFlush) {
                flush();
                cnt = 0;
            }
        }
    }

    // --------------------------------------- scalar remainder / unaligned
    constexpr int PACK = BF16 ? 8 : 4;
    for (int64_t j = a.nvec * PACK + tid; j < a.n; j += stride) {
        const float g = a.g[j];
        const float v = a.v[j];
        float s = 0.f;
#pragma unroll
        for (int m = 0; m < MM; ++m) {
            if (MT == 0 && m >= M) continue;
            float x;
            if constexpr (BF16)
                x = __uint_as_float(
                    (uint32_t)(reinterpret_cast<const uint16_t *>(a.x[m])[j])
                    << 16);
            else
                x = reinterpret_cast<const float *>(a.x[m])[j];
            const float d = g - x;
            s += d;
            e32[m] = fmaf(d, d, e32[m]);
        }
        b32 = fmaf(s, s, b32);
        float gp, vp;
        outer_step(k, s, g, v, gp, vp);
        nf += not_finite(gp, vp);
        a.g[j] = gp;
        a.v[j] = vp;
#pragma unroll
        for (int m = 0; m < MM; ++m) {
            if (MT == 0 && m >= M) continue;
            if constexpr (BF16)
                reinterpret_cast<__nv_bfloat16 *>(a.x[m])[j] =
                    __float2bfloat16_rn(gp);
            else
                reinterpret_cast<float *>(a.x[m])[j] = gp;
        }
        if (++cnt == kFlush) {
            flush();
            cnt = 0;
        }
    }
    flush();

    // ------------------------------------------------ block reduction
    constexpr int kWarps = kBlock / 32;
    __shared__ double sh[kWarps][MM + 1];
    __shared__ unsigned long long shnf[kWarps];
    __shared__ bool s_last;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

    unsigned long long nfl = nf;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
#pragma unroll
        for (int m = 0; m < MM; ++m)
            e64[m] += __shfl_down_sync(0xffffffffu, e64[m], off);
        b64 += __shfl_down_sync(0xffffffffu, b64, off);
        nfl += __shfl_down_sync(0xffffffffu, nfl, off);
    }
    if (lane == 0) {
#pragma unroll
        for (int m = 0; m < MM; ++m) sh[warp][m] = e64[m];
        sh[warp][MM] = b64;
        shnf[warp] = nfl;
    }
    __syncthreads();
    const int np = M + 1;  // values per block: M energies + sum S^2
    if (threadIdx.x < np) {
        const int col = threadIdx.x < M ? threadIdx.x : MM;
        double t = 0.0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) t += sh[w][col];
        a.partials[(int64_t)blockIdx.x * np + threadIdx.x] = t;
    }
    if (threadIdx.x == kBlock - 1) {
        unsigned long long t = 0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) t += shnf[w];
        a.nf_partials[blockIdx.x] = t;
    }

    // ------------------------------------------- last block: grid total
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
        const unsigned prev = atomicAdd(a.ticket, 1u);
        s_last = (prev == gridDim.x - 1);
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();

    double acc[MM + 1];
#pragma unroll
    for (int p = 0; p <= MM; ++p) acc[p] = 0.0;
    unsigned long long nacc = 0;
    for (int b = threadIdx.x; b < (int)gridDim.x; b += kBlock) {
        const double *row = a.partials + (int64_t)b * np;
#pragma unroll
        for (int p = 0; p <= MM; ++p)
            if (p < np) acc[p] += __ldcg(row + p);
        nacc += __ldcg(a.nf_partials + b);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
#pragma unroll
        for (int p = 0; p <= MM; ++p)
            acc[p] += __shfl_down_sync(0xffffffffu, acc[p], off);
        nacc += __shfl_down_sync(0xffffffffu, nacc, off);
    }
    __syncthreads();  // sh is reused
    if (lane == 0) {
#pragma unroll
        for (int p = 0; p <= MM; ++p) sh[warp][p] = acc[p];
        shnf[warp] = nacc;
    }
    __syncthreads();
    if (threadIdx.x < np) {
        double t = 0.0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) t += sh[w][threadIdx.x];
        a.totals[threadIdx.x] = t;
    }
    if (threadIdx.x == kBlock - 1) {
        unsigned long long t = 0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) t += shnf[w];
        *a.nf_total = t;
        *a.ticket = 0u;  // ready for the next launch
    }
}

// Occupancy-sized persistent grid for one instance.
template <int MT, bool BF16>
cudaError_t plan_one(int64_t work_items, int sm_count, LaunchPlan *plan) {
    static int blocks_per_sm = 0;  // per instance, computed once
    const void *fn = reinterpret_cast<const void *>(&sync_kernel<MT, BF16>);
    if (blocks_per_sm == 0) {
        int b = 0;
        cudaError_t e =
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, sync_kernel<MT, BF16>,
                                                          kBlock, 0);
        if (e != cudaSuccess) return e;
        blocks_per_sm = b > 0 ? b : 1;
    }
    int64_t want = (work_items + kBlock - 1) / kBlock;
    int64_t full = (int64_t)sm_count * blocks_per_sm;
    int64_t grid = want < full ? want : full;
    if (grid < 1) grid = 1;
    plan->kernel = fn;
    plan->grid = (int)grid;
    plan->block = kBlock;
    return cudaSuccess;
}

template <bool BF16>
cudaError_t plan_dispatch(int M, int64_t work_items, int sm_count,
                          LaunchPlan *plan) {
    switch (M) {
#define ALOCO_CASE(K) \
    case K:           \
        return plan_one<K, BF16>(work_items, sm_count, plan);
        ALOCO_CASE(1) ALOCO_CASE(2) ALOCO_CASE(3) ALOCO_CASE(4)
        ALOCO_CASE(5) ALOCO_CASE(6) ALOCO_CASE(7) ALOCO_CASE(8)
        ALOCO_CASE(9) ALOCO_CASE(10) ALOCO_CASE(11) ALOCO_CASE(12)
        ALOCO_CASE(13) ALOCO_CASE(14) ALOCO_CASE(15) ALOCO_CASE(16)
#undef ALOCO_CASE
        default:
            return plan_one<0, BF16>(work_items, sm_count, plan);
    }
}

}  // namespace aloco
