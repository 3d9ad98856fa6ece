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

// Tuning knobs (compile-time): packs loaded per thread before any is used,
// minimum resident blocks per SM requested from the register allocator, and
// the cache policy of the streaming loads and stores.
#ifndef ALOCO_UNROLL
#define ALOCO_UNROLL 1
#endif
#ifndef ALOCO_MINB
#define ALOCO_MINB 0  // 0: the per-instance table below
#endif
#ifndef ALOCO_LD
#define ALOCO_LD 0  // 0 ld.global.cs, 1 ld.global.lu, 2 plain, 3 ld.global.cg
#endif
#ifndef ALOCO_ST
#define ALOCO_ST 0  // 0 st.global.cs, 1 plain, 2 st.global.cg
#endif

template <typename T>
__device__ __forceinline__ T ld_stream(const T *p) {
#if ALOCO_LD == 0
    return __ldcs(p);
#elif ALOCO_LD == 1
    return __ldlu(p);
#elif ALOCO_LD == 2
    return *p;
#else
    return __ldcg(p);
#endif
}
template <typename T>
__device__ __forceinline__ void st_stream(T *p, T v) {
#if ALOCO_ST == 0
    __stcs(p, v);
#elif ALOCO_ST == 1
    *p = v;
#else
    __stcg(p, v);
#endif
}

__device__ __forceinline__ float4 ldcs4(const void *base, int64_t i) {
    return ld_stream(reinterpret_cast<const float4 *>(base) + i);
}
__device__ __forceinline__ uint4 ldcs4u(const void *base, int64_t i) {
    return ld_stream(reinterpret_cast<const uint4 *>(base) + i);
}
__device__ __forceinline__ void stcs4(void *base, int64_t i, float4 val) {
    st_stream(reinterpret_cast<float4 *>(base) + i, val);
}
__device__ __forceinline__ void stcs4u(void *base, int64_t i, uint4 val) {
    st_stream(reinterpret_cast<uint4 *>(base) + i, val);
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

// One 16-byte replica access ("pack") and the matching theta / v elements.
// fp32 replicas: 4 elements, one float4 of each stream.  bf16 replicas: 8
// elements, one uint4 of each replica and two float4 of theta and v.
template <bool BF16>
struct Pack;

template <>
struct Pack<false> {
    static constexpr int E = 4;
    using Raw = float4;
    __device__ static void load(const float *p, int64_t i, float (&o)[E]) {
        const float4 t = ldcs4(p, i);
        o[0] = t.x; o[1] = t.y; o[2] = t.z; o[3] = t.w;
    }
    __device__ static void store(float *p, int64_t i, const float (&o)[E]) {
        stcs4(p, i, make_float4(o[0], o[1], o[2], o[3]));
    }
    __device__ static Raw load_x(const void *p, int64_t i) { return ldcs4(p, i); }
    __device__ static void widen(const Raw &r, float (&o)[E]) {
        o[0] = r.x; o[1] = r.y; o[2] = r.z; o[3] = r.w;
    }
    __device__ static Raw narrow(const float (&o)[E]) {
        return make_float4(o[0], o[1], o[2], o[3]);
    }
    __device__ static void store_x(void *p, int64_t i, const Raw &r) {
        stcs4(p, i, r);
    }
};

template <>
struct Pack<true> {
    static constexpr int E = 8;
    using Raw = uint4;
    __device__ static void load(const float *p, int64_t i, float (&o)[E]) {
        const float4 a = ldcs4(p, 2 * i), b = ldcs4(p, 2 * i + 1);
        o[0] = a.x; o[1] = a.y; o[2] = a.z; o[3] = a.w;
        o[4] = b.x; o[5] = b.y; o[6] = b.z; o[7] = b.w;
    }
    __device__ static void store(float *p, int64_t i, const float (&o)[E]) {
        stcs4(p, 2 * i, make_float4(o[0], o[1], o[2], o[3]));
        stcs4(p, 2 * i + 1, make_float4(o[4], o[5], o[6], o[7]));
    }
    __device__ static Raw load_x(const void *p, int64_t i) { return ldcs4u(p, i); }
    __device__ static void widen(const Raw &r, float (&o)[E]) {
        const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            o[2 * j] = bf16_lo(w[j]);
            o[2 * j + 1] = bf16_hi(w[j]);
        }
    }
    __device__ static Raw narrow(const float (&o)[E]) {
        return make_uint4(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]),
                          pack_bf16x2(o[4], o[5]), pack_bf16x2(o[6], o[7]));
    }
    __device__ static void store_x(void *p, int64_t i, const Raw &r) {
        stcs4u(p, i, r);
    }
};

// Block and grid reduction of the per-thread fp64 partials (the block's
// NW warps all call it).  Each block writes one row of M + 1 partials; the
// last block to finish (atomic ticket, no spinning) adds the rows in block
// order and resets the ticket.  The order of every addition is fixed by the
// grid alone.
template <int MM, int NW>
__device__ __forceinline__ void reduce_and_finish(const SyncArgs &a, int M,
                                                  double (&e64)[MM], double b64,
                                                  unsigned nf) {
    constexpr int kThreads = NW * 32;
    __shared__ double sh[NW][MM + 1];
    __shared__ unsigned long long shnf[NW];
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
        for (int w = 0; w < NW; ++w) t += sh[w][col];
        a.partials[(int64_t)blockIdx.x * np + threadIdx.x] = t;
    }
    if (threadIdx.x == kThreads - 1) {
        unsigned long long t = 0;
#pragma unroll
        for (int w = 0; w < NW; ++w) t += shnf[w];
        a.nf_partials[blockIdx.x] = t;
    }

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
    for (int b = threadIdx.x; b < (int)gridDim.x; b += kThreads) {
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
        for (int w = 0; w < NW; ++w) t += sh[w][threadIdx.x];
        a.totals[threadIdx.x] = t;
    }
    if (threadIdx.x == kThreads - 1) {
        unsigned long long t = 0;
#pragma unroll
        for (int w = 0; w < NW; ++w) t += shnf[w];
        *a.nf_total = t;
        *a.ticket = 0u;  // ready for the next launch
    }
    if (a.stats_out) {
        // publish the totals block to the host, then the round's number
        __syncthreads();
        if (threadIdx.x == 0) {
            volatile double *out = a.stats_out;
            for (int p = 0; p < np; ++p) out[p] = __ldcg(a.totals + p);
            out[kNfSlot] = __longlong_as_double((long long)__ldcg(a.nf_total));
            out[kErrorSlot] = __ldcg(a.totals + kErrorSlot);
            __threadfence_system();
            reinterpret_cast<volatile unsigned long long *>(a.stats_out)[kSeqSlot] = a.seq;
        }
    }
}

// Minimum resident blocks per SM the register allocator must allow (it
// bounds registers per thread to 65536 / (kBlock * value)); 0 leaves the
// choice to the compiler, which measured as good as any fixed budget.
template <int MT, bool BF16>
constexpr int min_blocks() {
    return ALOCO_MINB > 0 ? ALOCO_MINB : 0;
}

template <int MT, bool BF16>
__global__ void __launch_bounds__(kBlock, (min_blocks<MT, BF16>()))
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
    using P = Pack<BF16>;
    constexpr int E = P::E;

    // Pseudo-gradients of one replica pack: S += Delta, ||Delta_m||^2 += Delta^2.
    auto accumulate = [&](const float (&gg)[E], const typename P::Raw &raw,
                          float (&s)[E], float &e) {
        float xx[E];
        P::widen(raw, xx);
#pragma unroll
        for (int j = 0; j < E; ++j) {
            const float d = gg[j] - xx[j];
            s[j] += d;
            e = fmaf(d, d, e);
        }
    };
    // Outer step of the pack and its stores: theta', v', replica reset.
    auto finish = [&](int64_t i, const float (&gg)[E], const float (&vv)[E],
                      const float (&s)[E]) {
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
        for (int m = 0; m < MM; ++m) {
            if (MT == 0 && m >= M) continue;
            P::store_x(a.x[m], i, xo);
        }
        if (++cnt == kFlush) {
            flush();
            cnt = 0;
        }
    };

    if constexpr (MT > 0) {
        // Compile-time M: every load of the U packs is issued before any is
        // used, so (M + 2) U 16-byte loads (bf16: (M + 4) U) are in flight.
        constexpr int U = ALOCO_UNROLL;
        for (int64_t i0 = tid; i0 < a.nvec; i0 += stride * U) {
            float G[U][E], V[U][E];
            typename P::Raw X[U][MT];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int64_t i = i0 + u * stride;
                if (i >= a.nvec) continue;
                P::load(a.g, i, G[u]);
                P::load(a.v, i, V[u]);
#pragma unroll
                for (int m = 0; m < MT; ++m) X[u][m] = P::load_x(a.x[m], i);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int64_t i = i0 + u * stride;
                if (i >= a.nvec) continue;
                float s[E];
#pragma unroll
                for (int j = 0; j < E; ++j) s[j] = 0.f;
#pragma unroll
                for (int m = 0; m < MT; ++m) accumulate(G[u], X[u][m], s, e32[m]);
                finish(i, G[u], V[u], s);
            }
        }
    } else {
        // Any M up to 32: replicas are loaded in groups of 8 (independent
        // loads in flight) and consumed group by group, which bounds the
        // registers that hold loaded packs.
        constexpr int kGroup = 8;
        for (int64_t i = tid; i < a.nvec; i += stride) {
            float gg[E], vv[E], s[E];
            P::load(a.g, i, gg);
            P::load(a.v, i, vv);
#pragma unroll
            for (int j = 0; j < E; ++j) s[j] = 0.f;
#pragma unroll
            for (int m0 = 0; m0 < MM; m0 += kGroup) {
                if (m0 >= M) break;
                typename P::Raw X[kGroup];
#pragma unroll
                for (int q = 0; q < kGroup; ++q)
                    if (m0 + q < M) X[q] = P::load_x(a.x[m0 + q], i);
#pragma unroll
                for (int q = 0; q < kGroup; ++q)
                    if (m0 + q < M) accumulate(gg, X[q], s, e32[m0 + q]);
            }
            finish(i, gg, vv, s);
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

    reduce_and_finish<MM, kBlock / 32>(a, M, e64, b64, nf);
}

// Tuned residency (blocks of kBlock threads per SM) of the fused pass for
// M workers, measured on GB300 over M = 1..32 and both replica types on a
// 2^28-parameter round: fewer resident warps streaming more arrays keep
// HBM busier once M + 2 streams are in flight.  Capped by occupancy.
template <bool BF16>
constexpr int tuned_blocks_per_sm(int M) {
    if (BF16) return M <= 7 ? 2 : 1;
    return M == 1 ? 4 : M == 2 ? 3 : M <= 8 ? 2 : 1;
}

// Persistent grid for one instance: SMs x resident blocks.
template <int MT, bool BF16>
cudaError_t plan_one(int64_t work_items, int sm_count, int M, int request,
                     LaunchPlan *plan) {
    static PerDevice cache;  // per instance and device, computed once
    const void *fn = reinterpret_cast<const void *>(&sync_kernel<MT, BF16>);
    const int dev = PerDevice::device();
    int occupancy = cache.get(dev);
    if (occupancy == 0) {
        int b = 0;
        cudaError_t e =
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, sync_kernel<MT, BF16>,
                                                          kBlock, 0);
        if (e != cudaSuccess) return e;
        occupancy = b > 0 ? b : 1;
        cache.set(dev, occupancy);
    }
    int blocks_per_sm = request > 0 ? request : tuned_blocks_per_sm<BF16>(M);
    if (blocks_per_sm <= 0 || blocks_per_sm > occupancy) blocks_per_sm = occupancy;
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
                          int blocks_per_sm, LaunchPlan *plan) {
    switch (M) {
#define ALOCO_CASE(K) \
    case K:           \
        return plan_one<K, BF16>(work_items, sm_count, M, blocks_per_sm, plan);
        ALOCO_CASE(1) ALOCO_CASE(2) ALOCO_CASE(3) ALOCO_CASE(4)
        ALOCO_CASE(5) ALOCO_CASE(6) ALOCO_CASE(7) ALOCO_CASE(8)
        ALOCO_CASE(9) ALOCO_CASE(10) ALOCO_CASE(11) ALOCO_CASE(12)
        ALOCO_CASE(13) ALOCO_CASE(14) ALOCO_CASE(15) ALOCO_CASE(16)
#undef ALOCO_CASE
        default:
            return plan_one<0, BF16>(work_items, sm_count, M, blocks_per_sm,
                                     plan);
    }
}

}  // namespace aloco
