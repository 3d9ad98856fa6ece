// The workers' inner optimizer (Sec. 2, Eq. diloco-local-trajectory: H local
// AdamW steps per interval; Tab. training settings): one AdamW step with
// decoupled weight decay and per-replica gradient-norm clipping on all M
// replicas, in two streaming kernels.
//
//   norm pass    grid (G1, M): block (b, m) sums g_m^2 over its grid-stride
//                share of replica m (fp32 over up to 8 units of 4 elements,
//                then fp64) and writes one fp64 partial, partials[m][b];
//   update pass  grid (G2, M): every block of worker m first folds that
//                worker's G1 partials in a fixed order (lane-strided sums,
//                then a fixed shuffle tree) into ||g_m|| and the clipping
//                factor c_m, so all blocks agree without a device-wide sync;
//                then it streams x, g, m, v of replica m and writes x, m, v.
// When the caller supplies the norms (aloco_adamw_step_normed) the factors
// arrive with the arguments and only the update pass runs.
// Both passes are deterministic: the partition depends only on the grid.
// The update reads each array once; the gradient is read a second time by
// the norm pass, which clipping needs before any element can move.
#include "aloco_sync_kernel.cuh"

namespace aloco {

namespace {

constexpr int kUnit = 4;      // elements per thread per unit
constexpr int kNormUnits = 8; // units summed in fp32 before the fp64 add
constexpr int kUpdUnroll = 2; // units in flight per thread in the update

template <bool BF16>
__device__ __forceinline__ void load_unit(const void *p, int64_t u, float (&o)[kUnit]) {
    if constexpr (BF16) {
        const uint2 q = __ldcs(reinterpret_cast<const uint2 *>(p) + u);
        o[0] = bf16_lo(q.x); o[1] = bf16_hi(q.x);
        o[2] = bf16_lo(q.y); o[3] = bf16_hi(q.y);
    } else {
        const float4 q = __ldcs(reinterpret_cast<const float4 *>(p) + u);
        o[0] = q.x; o[1] = q.y; o[2] = q.z; o[3] = q.w;
    }
}

template <bool BF16>
__device__ __forceinline__ void store_unit(void *p, int64_t u, const float (&o)[kUnit]) {
    if constexpr (BF16) {
        __stcs(reinterpret_cast<uint2 *>(p) + u,
               make_uint2(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3])));
    } else {
        __stcs(reinterpret_cast<float4 *>(p) + u, make_float4(o[0], o[1], o[2], o[3]));
    }
}

template <bool BF16>
__device__ __forceinline__ float load_elem(const void *p, int64_t e) {
    if constexpr (BF16)
        return __uint_as_float((uint32_t)reinterpret_cast<const uint16_t *>(p)[e] << 16);
    else
        return reinterpret_cast<const float *>(p)[e];
}

template <bool BF16>
__device__ __forceinline__ void store_elem(void *p, int64_t e, float x) {
    if constexpr (BF16)
        reinterpret_cast<__nv_bfloat16 *>(p)[e] = __float2bfloat16_rn(x);
    else
        reinterpret_cast<float *>(p)[e] = x;
}

// Block-wide fp64 sum in a fixed order (warp trees, then warp 0 over warps);
// the result is valid in thread 0.
__device__ __forceinline__ double block_sum(double v) {
    __shared__ double sh[kBlock / 32];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_down_sync(0xffffffffu, v, off);
    if ((threadIdx.x & 31) == 0) sh[threadIdx.x >> 5] = v;
    __syncthreads();
    double s = 0.0;
    if (threadIdx.x == 0) {
#pragma unroll
        for (int w = 0; w < kBlock / 32; ++w) s += sh[w];
    }
    return s;
}

// One element's AdamW update in fp32.
__device__ __forceinline__ void adamw_elem(const AdamArgs &a, float c, float g, float &x,
                                           float &m1, float &m2) {
    const float gt = c * g;
    m1 = fmaf(a.beta1, m1, a.omb1 * gt);
    m2 = fmaf(a.beta2, m2, (a.omb2 * gt) * gt);
    const float denom = fmaf(sqrtf(m2), a.inv_sqrt_bc2, a.eps);
    x = fmaf(a.neg_step, m1 / denom, x * a.decay);
}

}  // namespace

template <bool GBF16>
__global__ void __launch_bounds__(kBlock) adamw_norm_kernel(const __grid_constant__ AdamArgs a) {
    const int m = blockIdx.y;
    const void *gp = a.g[m];
    const int64_t stride = (int64_t)gridDim.x * kBlock;
    double acc = 0.0;
    for (int64_t u0 = (int64_t)blockIdx.x * kBlock + threadIdx.x; u0 < a.nunit;
         u0 += kNormUnits * stride) {
        float v[kNormUnits][kUnit];
#pragma unroll
        for (int k = 0; k < kNormUnits; ++k) {
            const int64_t u = u0 + k * stride;
            if (u < a.nunit) {
                load_unit<GBF16>(gp, u, v[k]);
            } else {
#pragma unroll
                for (int j = 0; j < kUnit; ++j) v[k][j] = 0.f;
            }
        }
        float s = 0.f;
#pragma unroll
        for (int k = 0; k < kNormUnits; ++k)
#pragma unroll
            for (int j = 0; j < kUnit; ++j) s = fmaf(v[k][j], v[k][j], s);
        acc += (double)s;
    }
    for (int64_t e = a.nunit * kUnit + (int64_t)blockIdx.x * kBlock + threadIdx.x; e < a.n;
         e += stride) {
        const float x = load_elem<GBF16>(gp, e);
        acc += (double)x * (double)x;
    }
    const double s = block_sum(acc);
    if (threadIdx.x == 0) a.partials[(int64_t)m * a.g1 + blockIdx.x] = s;
}

template <bool PBF16, bool GBF16>
__global__ void __launch_bounds__(kBlock)
    adamw_update_kernel(const __grid_constant__ AdamArgs a) {
    const int m = blockIdx.y;
    __shared__ float s_clip;
    if (a.given) {
        if (threadIdx.x == 0) s_clip = a.clip[m];
    } else if (threadIdx.x < 32) {
        double s = 0.0;
        for (int b = threadIdx.x; b < a.g1; b += 32) s += a.partials[(int64_t)m * a.g1 + b];
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) s += __shfl_down_sync(0xffffffffu, s, off);
        if (threadIdx.x == 0) {
            const double norm = sqrt(s);
            double c = 1.0;
            if (a.max_norm > 0.0) {
                c = a.max_norm / (norm + 1e-6);
                if (c > 1.0) c = 1.0;
            }
            s_clip = (float)c;
            if (blockIdx.x == 0) {
                a.out[m] = norm;
                a.out[ALOCO_MAX_WORKERS + m] = c;
            }
        }
    }
    __syncthreads();
    const float c = s_clip;
    void *xp = a.x[m];
    const void *gp = a.g[m];
    float *m1p = a.m1[m];
    float *m2p = a.m2[m];
    const int64_t stride = (int64_t)gridDim.x * kBlock;
    for (int64_t u0 = (int64_t)blockIdx.x * kBlock + threadIdx.x; u0 < a.nunit;
         u0 += kUpdUnroll * stride) {
        float x[kUpdUnroll][kUnit], g[kUpdUnroll][kUnit], m1[kUpdUnroll][kUnit],
            m2[kUpdUnroll][kUnit];
        bool in[kUpdUnroll];
#pragma unroll
        for (int k = 0; k < kUpdUnroll; ++k) {
            const int64_t u = u0 + k * stride;
            in[k] = u < a.nunit;
            if (in[k]) {
                load_unit<PBF16>(xp, u, x[k]);
                load_unit<GBF16>(gp, u, g[k]);
                load_unit<false>(m1p, u, m1[k]);
                load_unit<false>(m2p, u, m2[k]);
            }
        }
#pragma unroll
        for (int k = 0; k < kUpdUnroll; ++k) {
            if (!in[k]) continue;
            const int64_t u = u0 + k * stride;
#pragma unroll
            for (int j = 0; j < kUnit; ++j) adamw_elem(a, c, g[k][j], x[k][j], m1[k][j], m2[k][j]);
            store_unit<PBF16>(xp, u, x[k]);
            store_unit<false>(m1p, u, m1[k]);
            store_unit<false>(m2p, u, m2[k]);
        }
    }
    for (int64_t e = a.nunit * kUnit + (int64_t)blockIdx.x * kBlock + threadIdx.x; e < a.n;
         e += stride) {
        float x = load_elem<PBF16>(xp, e), m1 = m1p[e], m2 = m2p[e];
        adamw_elem(a, c, load_elem<GBF16>(gp, e), x, m1, m2);
        store_elem<PBF16>(xp, e, x);
        m1p[e] = m1;
        m2p[e] = m2;
    }
}

namespace {

template <bool PBF16, bool GBF16>
cudaError_t adamw_launch(const AdamArgs &a, int g2, cudaStream_t stream) {
    const dim3 block(kBlock);
    if (!a.given) {
        adamw_norm_kernel<GBF16><<<dim3(a.g1, a.M), block, 0, stream>>>(a);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    adamw_update_kernel<PBF16, GBF16><<<dim3(g2, a.M), block, 0, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_adamw(const AdamArgs &a, aloco_dtype param_dtype,
                         aloco_dtype grad_dtype, int g2, cudaStream_t stream) {
    const bool pb = param_dtype == ALOCO_BF16, gb = grad_dtype == ALOCO_BF16;
    if (pb && gb) return adamw_launch<true, true>(a, g2, stream);
    if (pb) return adamw_launch<true, false>(a, g2, stream);
    if (gb) return adamw_launch<false, true>(a, g2, stream);
    return adamw_launch<false, false>(a, g2, stream);
}

}  // namespace aloco
