// INT8 pseudo-gradient communication (App. G.1): the blockwise codec and
// the outer round whose averaged pseudo-gradient is the decoded INT8
// aggregate.
//
// Blocks: every tensor part is cut into consecutive blocks of at most 4096
// elements starting at the part's first element.  Codec, in FP32 as the
// appendix states: scale = max|y| / 127 (1 for an all-zero block, kept in
// [FLT_MIN, FLT_MAX / 127]); q = rint(y / scale) clipped to [-127, 127]
// (0 where the quotient is NaN); decode = q * scale.  The codec's divisions,
// products and sums use the _rn intrinsics so that no FMA contraction
// changes an integer decision.
//
// Round: per block, each worker's FP32 pseudo-gradient Delta_m = theta - x_m
// is encoded and decoded; the decoded contributions are added in worker
// order and divided by M; that mean is encoded and decoded once, and the
// result drives the corrected Nesterov step.  D_t uses the pre-quantisation
// Delta_m, C_t the decoded aggregate.
#include <cuda_bf16.h>
#include <float.h>

#include <type_traits>

#include "aloco_sync_kernel.cuh"

namespace aloco {

constexpr int kI8Block = 4096;      // elements per codec block
constexpr int kI8Threads = 512;     // 8 elements per thread
constexpr int kI8PerThread = kI8Block / kI8Threads;

// Where block k lies: the part p with blk[p] <= k < blk[p + 1].
__device__ __forceinline__ void locate_block(const Int8Parts &P, int64_t k,
                                             int64_t &start, int &len) {
    int lo = 0, hi = P.n_parts - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (P.blk[mid] <= k) lo = mid; else hi = mid - 1;
    }
    start = P.off[lo] + (k - P.blk[lo]) * kI8Block;
    const int64_t end = P.off[lo + 1];
    len = (int)((end - start) < kI8Block ? (end - start) : kI8Block);
}

// Element offset (within the block) of a thread's i-th value.  fp32 data
// moves in two 16-byte slots (4 elements each) spaced 2048 elements apart,
// bf16 replicas in one 16-byte slot of 8 elements, so every warp access is
// 512 contiguous bytes.
template <bool BF16>
__device__ __forceinline__ int elem_of(int t, int i) {
    if (BF16) return 8 * t + i;
    return (i >> 2) * 2048 + 4 * t + (i & 3);
}

template <bool BF16>
__device__ __forceinline__ void load_f32(const float *p, int64_t start, int len,
                                         bool vec, int t, float (&o)[kI8PerThread]) {
#pragma unroll
    for (int i = 0; i < kI8PerThread; i += 4) {
        const int e = elem_of<BF16>(t, i);
        if (vec && e + 3 < len) {
            const float4 q = __ldcs(reinterpret_cast<const float4 *>(p + start + e));
            o[i] = q.x; o[i + 1] = q.y; o[i + 2] = q.z; o[i + 3] = q.w;
        } else {
#pragma unroll
            for (int k = 0; k < 4; ++k)
                o[i + k] = (e + k < len) ? p[start + e + k] : 0.f;
        }
    }
}

template <bool BF16>
__device__ __forceinline__ void store_f32(float *p, int64_t start, int len,
                                          bool vec, int t, const float (&o)[kI8PerThread]) {
#pragma unroll
    for (int i = 0; i < kI8PerThread; i += 4) {
        const int e = elem_of<BF16>(t, i);
        if (vec && e + 3 < len) {
            __stcs(reinterpret_cast<float4 *>(p + start + e),
                   make_float4(o[i], o[i + 1], o[i + 2], o[i + 3]));
        } else {
#pragma unroll
            for (int k = 0; k < 4; ++k)
                if (e + k < len) p[start + e + k] = o[i + k];
        }
    }
}

// Replica values (fp32, or bf16 widened exactly).
template <bool BF16>
__device__ __forceinline__ void load_rep(const void *p, int64_t start, int len,
                                         bool vec, int t, float (&o)[kI8PerThread]) {
    if constexpr (!BF16) {
        load_f32<false>(reinterpret_cast<const float *>(p), start, len, vec, t, o);
    } else {
        const uint16_t *h = reinterpret_cast<const uint16_t *>(p);
#pragma unroll
        for (int i = 0; i < kI8PerThread; i += 8) {
            const int e = elem_of<true>(t, i);
            if (vec && e + 7 < len) {
                const uint4 q = __ldcs(reinterpret_cast<const uint4 *>(h + start + e));
                const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    o[i + 2 * j] = bf16_lo(w[j]);
                    o[i + 2 * j + 1] = bf16_hi(w[j]);
                }
            } else {
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    o[i + k] = (e + k < len)
                                   ? __uint_as_float((uint32_t)h[start + e + k] << 16)
                                   : 0.f;
            }
        }
    }
}

template <bool BF16>
__device__ __forceinline__ void store_rep(void *p, int64_t start, int len, bool vec,
                                          int t, const float (&o)[kI8PerThread]) {
    if constexpr (!BF16) {
        store_f32<false>(reinterpret_cast<float *>(p), start, len, vec, t, o);
    } else {
        __nv_bfloat16 *h = reinterpret_cast<__nv_bfloat16 *>(p);
#pragma unroll
        for (int i = 0; i < kI8PerThread; i += 8) {
            const int e = elem_of<true>(t, i);
            if (vec && e + 7 < len) {
                __stcs(reinterpret_cast<uint4 *>(h + start + e),
                       make_uint4(pack_bf16x2(o[i], o[i + 1]), pack_bf16x2(o[i + 2], o[i + 3]),
                                  pack_bf16x2(o[i + 4], o[i + 5]),
                                  pack_bf16x2(o[i + 6], o[i + 7])));
            } else {
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    if (e + k < len) h[start + e + k] = __float2bfloat16_rn(o[i + k]);
            }
        }
    }
}

// Full, 16-byte aligned block: raw replica packs of one thread, loaded
// unconditionally so that a group of workers' loads is in flight at once.
template <bool BF16>
struct RawPack {
    using T = typename std::conditional<BF16, uint4, float4>::type;
    static constexpr int N = BF16 ? 1 : 2;  // 16-byte loads per thread
    T q[N];
};
template <bool BF16>
__device__ __forceinline__ RawPack<BF16> load_raw(const void *p, int64_t start, int t) {
    RawPack<BF16> r;
    if constexpr (BF16) {
        r.q[0] = __ldcs(reinterpret_cast<const uint4 *>(
            reinterpret_cast<const uint16_t *>(p) + start + 8 * t));
    } else {
        const float *f = reinterpret_cast<const float *>(p) + start + 4 * t;
        r.q[0] = __ldcs(reinterpret_cast<const float4 *>(f));
        r.q[1] = __ldcs(reinterpret_cast<const float4 *>(f + 2048));
    }
    return r;
}
template <bool BF16>
__device__ __forceinline__ void widen_raw(const RawPack<BF16> &r, float (&o)[kI8PerThread]) {
    if constexpr (BF16) {
        const uint32_t w[4] = {r.q[0].x, r.q[0].y, r.q[0].z, r.q[0].w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            o[2 * j] = bf16_lo(w[j]);
            o[2 * j + 1] = bf16_hi(w[j]);
        }
    } else {
        o[0] = r.q[0].x; o[1] = r.q[0].y; o[2] = r.q[0].z; o[3] = r.q[0].w;
        o[4] = r.q[1].x; o[5] = r.q[1].y; o[6] = r.q[1].z; o[7] = r.q[1].w;
    }
}

constexpr int kI8Warps = kI8Threads / 32;

// Tuning knobs: workers whose loads are issued together on full blocks, and
// the apply kernel's minimum resident CTAs per SM (0 = compiler's choice).
#ifndef ALOCO_I8_G_BF16
#define ALOCO_I8_G_BF16 2
#endif
#ifndef ALOCO_I8_G_F32
#define ALOCO_I8_G_F32 2
#endif
#ifndef ALOCO_I8_MINB
#define ALOCO_I8_MINB 0
#endif
#ifndef ALOCO_I8_MINB_SCALES
#define ALOCO_I8_MINB_SCALES 2
#endif
template <bool BF16>
__host__ __device__ constexpr int i8_group() { return BF16 ? ALOCO_I8_G_BF16 : ALOCO_I8_G_F32; }

// Block-wide max|y| as the bits of a non-negative float (NaN, whose bits
// exceed +inf's, wins) and, when sq != null, the block's sum of y^2: each
// warp's fp32 sum lands in sq[warp] for the caller to add in warp order.
// red[] / sq[] are double-buffered by the caller's parity so one barrier per
// reduction suffices.
__device__ __forceinline__ float block_amax(const float (&y)[kI8PerThread], bool valid_all,
                                            int len, int t, bool bf16, unsigned *red,
                                            float *sq) {
    unsigned m = 0;
    float q = 0.f;
#pragma unroll
    for (int i = 0; i < kI8PerThread; ++i) {
        const int e = bf16 ? elem_of<true>(t, i) : elem_of<false>(t, i);
        if (valid_all || e < len) {
            m = max(m, __float_as_uint(fabsf(y[i])));
            q = fmaf(y[i], y[i], q);
        }
    }
    m = __reduce_max_sync(0xffffffffu, m);
    if (sq) {
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) q += __shfl_down_sync(0xffffffffu, q, off);
    }
    if ((threadIdx.x & 31) == 0) {
        red[threadIdx.x >> 5] = m;
        if (sq) sq[threadIdx.x >> 5] = q;
    }
    __syncthreads();
    unsigned r = red[0];
#pragma unroll
    for (int w = 1; w < kI8Warps; ++w) r = max(r, red[w]);
    return __uint_as_float(r);
}

__device__ __forceinline__ float codec_scale(float amax) {
    if (amax == 0.f) return 1.f;
    float s = __fdiv_rn(amax, 127.f);
    if (s < FLT_MIN) s = FLT_MIN;
    if (s > FLT_MAX / 127.f) s = FLT_MAX / 127.f;
    return s;  // NaN stays NaN
}

// fl32(y / s) given r = fl32(1 / s), by Markstein's method: the product
// y r is corrected twice with the exact residual y - s q (one FMA each);
// with a correctly rounded reciprocal the second correction returns the
// correctly rounded quotient for every finite, non-overflowing quotient.
// Anything else (infinite or NaN operands) takes the IEEE division.
__device__ __forceinline__ float div_by_scale(float y, float s, float r) {
    const float q0 = __fmul_rn(y, r);
    const float q1 = __fmaf_rn(__fmaf_rn(-s, q0, y), r, q0);
    const float q2 = __fmaf_rn(__fmaf_rn(-s, q1, y), r, q1);
    return isfinite(q2) ? q2 : __fdiv_rn(y, s);
}

// The code of y as a float in [-127, 127] (0 where the quotient is NaN).
__device__ __forceinline__ float codec_code_f(float y, float s, float r) {
    float t = rintf(div_by_scale(y, s, r));
    if (t != t) return 0.f;
    return fminf(fmaxf(t, -127.f), 127.f);
}

__device__ __forceinline__ int codec_code(float y, float s) {
    return (int)codec_code_f(y, s, __frcp_rn(s));
}

// The same code from the product y r alone when that is provably the same
// decision: |y r - y/s| <= 2^-23 |y/s| < 2^-16 for |y r| < 127, so a
// product at least 2^-14 away from every half-integer rounds like the
// quotient.  Products nearer a half-integer, at or beyond 127, or not
// finite take the exact quotient.
__device__ __forceinline__ float codec_code_fast(float y, float s, float r) {
    const float t = __fmul_rn(y, r);
    const float n = rintf(t);
    if (fabsf(t) < 127.f && 0.5f - fabsf(t - n) > 0x1p-14f) return n;
    return codec_code_f(y, s, r);
}

// Paired fp32 arithmetic (the sm_100 family's two-lane FADD/FMUL/FFMA): each
// lane is the correctly rounded fp32 result of the scalar operation.
constexpr int kI8Pairs = kI8PerThread / 2;
__device__ __forceinline__ float2 sub2(float2 a, float2 b) {  // RN(a - b)
    return __ffma2_rn(b, make_float2(-1.f, -1.f), a);
}
__device__ __forceinline__ float2 splat2(float a) { return make_float2(a, a); }
// Paired product with explicit .rn rounding in PTX.  ptxas (CUDA 13.0) was
// measured to contract a single-use paired product into a following paired
// .rn add (a paired FMA), which skips the rounding of the decoded value q * s
// that the codec defines; a one-ulp change in the mean then moves some
// quotients across a half-integer.  So decoded values are summed with the
// scalar __fadd_rn, which is never contracted, and the paired form serves
// only products that are not added.
__device__ __forceinline__ float2 mul2_rn(float2 a, float2 b) {
    float2 r;
    asm("{\n\t.reg .b64 pa, pb, pd;\n\t"
        "mov.b64 pa, {%2, %3};\n\tmov.b64 pb, {%4, %5};\n\t"
        "mul.rn.f32x2 pd, pa, pb;\n\tmov.b64 {%0, %1}, pd;\n\t}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}

// Half-integer margin of the product test below: 0.5 - 2^-14, exact in fp32.
constexpr float kCodeMargin = 0.5f - 0x1p-14f;

// Codes of a pair from the product y r; `ok` turns false unless both are
// provably the codec's.  For the codec's own scale (max |y| over the block,
// so |y| <= max) every finite product lies below 127.5, since s and r are
// each within half an ulp of max / 127 and 127 / max; rint of it is then in
// [-127, 127] and no clipping is needed.  A product more than 2^-14 from a
// half-integer rounds like the quotient (the product is within 2^-16 of y/s,
// and fl32(y/s) within 2^-17), and infinite or NaN products fail the test.
__device__ __forceinline__ float2 code2_fast(float2 y, float r, bool &ok) {
    const float2 t = mul2_rn(y, splat2(r));
    const float2 n = make_float2(rintf(t.x), rintf(t.y));
    const float2 d = sub2(t, n);  // exact: |t - n| <= 1/2
    ok = ok && fabsf(d.x) < kCodeMargin && fabsf(d.y) < kCodeMargin;
    return n;
}

template <bool BF16>
__device__ __forceinline__ void to_pairs(const float (&f)[kI8PerThread],
                                         float2 (&o)[kI8Pairs]) {
#pragma unroll
    for (int j = 0; j < kI8Pairs; ++j) o[j] = make_float2(f[2 * j], f[2 * j + 1]);
}
template <bool BF16>
__device__ __forceinline__ void widen_pairs(const RawPack<BF16> &r, float2 (&o)[kI8Pairs]) {
    if constexpr (BF16) {
        const uint32_t w[4] = {r.q[0].x, r.q[0].y, r.q[0].z, r.q[0].w};
#pragma unroll
        for (int j = 0; j < 4; ++j) o[j] = make_float2(bf16_lo(w[j]), bf16_hi(w[j]));
    } else {
        o[0] = make_float2(r.q[0].x, r.q[0].y);
        o[1] = make_float2(r.q[0].z, r.q[0].w);
        o[2] = make_float2(r.q[1].x, r.q[1].y);
        o[3] = make_float2(r.q[1].z, r.q[1].w);
    }
}

// ------------------------------------------------------------- the round
// Two streaming passes, one CTA per 4096-element block at a time (persistent
// grid stride over blocks, 8 elements per thread, the same grid for both):
//   pass 1 reads theta and the replicas and writes, per block and worker,
//          the codec scale of Delta_m; every worker's max |Delta_m| and
//          sum Delta_m^2 are reduced together (one barrier per block), and
//          the CTA's fp64 drift energies go to e_rows[blockIdx.x];
//   pass 2 reads theta, v and the replicas again; with the scales known the
//          encode / decode / FP32 sum over workers streams freely, and only
//          the mean's block maximum needs a barrier.
// Thread q < M combines worker q's warp values in warp order, so both
// passes are deterministic.
constexpr int kMaxI8Workers = 16;

template <bool BF16>
__global__ void __launch_bounds__(kI8Threads, ALOCO_I8_MINB_SCALES)
    int8_scales_kernel(const __grid_constant__ SyncArgs a,
                       const __grid_constant__ Int8Parts P, unsigned *__restrict__ bmax,
                       double *__restrict__ e_rows) {
    // No block barrier: each warp folds its max |Delta_m| into the block's
    // slot with an atomic max on the float bits (order-independent), and
    // keeps its own energies until the end.
    constexpr int R = kI8PerThread;
    __shared__ double e_w[kI8Warps][kMaxI8Workers];
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int M = a.M;
    if (lane < kMaxI8Workers) e_w[warp][lane] = 0.0;
    __syncwarp();
    const int64_t nblocks = P.blk[P.n_parts];
    for (int64_t kb = blockIdx.x; kb < nblocks; kb += gridDim.x) {
        int64_t start;
        int len;
        locate_block(P, kb, start, len);
        const bool vec = a.nvec > 0 && (start % 8) == 0;
        const bool full = len == kI8Block;
        float gs[R];
        load_f32<BF16>(a.g, start, len, vec, t, gs);
        float2 g[kI8Pairs];
        to_pairs<BF16>(gs, g);
        // max |Delta_m| by float max while every Delta_m and the energy are
        // finite (then it equals the bit-pattern max); otherwise by the bits.
        auto worker = [&](int m, const float2 (&x)[kI8Pairs], bool all_in) {
            float mf = 0.f;
            float2 e2 = make_float2(0.f, 0.f);
            if (all_in) {
#pragma unroll
                for (int j = 0; j < kI8Pairs; ++j) {
                    const float2 d = sub2(g[j], x[j]);
                    mf = fmaxf(mf, fmaxf(fabsf(d.x), fabsf(d.y)));
                    e2 = __ffma2_rn(d, d, e2);
                }
            } else {
#pragma unroll
                for (int j = 0; j < kI8Pairs; ++j) {
                    const float2 d = sub2(g[j], x[j]);
                    const bool in0 = elem_of<BF16>(t, 2 * j) < len;
                    const bool in1 = elem_of<BF16>(t, 2 * j + 1) < len;
                    const float2 dz = make_float2(in0 ? d.x : 0.f, in1 ? d.y : 0.f);
                    mf = fmaxf(mf, fmaxf(fabsf(dz.x), fabsf(dz.y)));
                    e2 = __ffma2_rn(dz, dz, e2);
                }
            }
            float e = __fadd_rn(e2.x, e2.y);
            unsigned mx = __float_as_uint(mf);
            if (!isfinite(e)) {
                mx = 0;
#pragma unroll
                for (int j = 0; j < kI8Pairs; ++j) {
                    const float2 d = sub2(g[j], x[j]);
                    if (all_in || elem_of<BF16>(t, 2 * j) < len)
                        mx = max(mx, __float_as_uint(fabsf(d.x)));
                    if (all_in || elem_of<BF16>(t, 2 * j + 1) < len)
                        mx = max(mx, __float_as_uint(fabsf(d.y)));
                }
            }
            mx = __reduce_max_sync(0xffffffffu, mx);
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) e += __shfl_down_sync(0xffffffffu, e, off);
            if (lane == 0) {
                atomicMax(bmax + kb * M + m, mx);
                e_w[warp][m] += (double)e;
            }
        };
        if (full && vec) {
            constexpr int G = i8_group<BF16>();
            int m0 = 0;
            for (; m0 + G <= M; m0 += G) {
                RawPack<BF16> raw[G];
#pragma unroll
                for (int q = 0; q < G; ++q) raw[q] = load_raw<BF16>(a.x[m0 + q], start, t);
#pragma unroll
                for (int q = 0; q < G; ++q) {
                    float2 x[kI8Pairs];
                    widen_pairs<BF16>(raw[q], x);
                    worker(m0 + q, x, true);
                }
            }
            for (; m0 < M; ++m0) {
                float2 x[kI8Pairs];
                widen_pairs<BF16>(load_raw<BF16>(a.x[m0], start, t), x);
                worker(m0, x, true);
            }
        } else {
            for (int m = 0; m < M; ++m) {
                float xs[R];
                float2 x[kI8Pairs];
                load_rep<BF16>(a.x[m], start, len, vec, t, xs);
                to_pairs<BF16>(xs, x);
                worker(m, x, full);
            }
        }
    }
    __syncthreads();
    if (t < M) {
        double e = 0.0;
#pragma unroll
        for (int w = 0; w < kI8Warps; ++w) e += e_w[w][t];
        e_rows[(int64_t)blockIdx.x * kMaxI8Workers + t] = e;
    }
}

template <bool BF16>
__global__ void __launch_bounds__(kI8Threads, ALOCO_I8_MINB)
    int8_apply_kernel(const __grid_constant__ SyncArgs a,
                      const __grid_constant__ Int8Parts P,
                      const unsigned *__restrict__ bmax,
                      const double *__restrict__ e_rows) {
    constexpr int R = kI8PerThread;
    __shared__ unsigned red1[2][kI8Warps];
    const int t = threadIdx.x, lane = t & 31;
    const int M = a.M;
    float b32 = 0.f;
    double b64 = 0.0;
    unsigned nf = 0;
    int parity = 0;
    const Coef k{a.c_hi, a.c_lo, a.mu_hi, a.mu_lo, a.neg_eta_hi, a.neg_eta_lo};
    const int64_t nblocks = P.blk[P.n_parts];
    for (int64_t kb = blockIdx.x; kb < nblocks; kb += gridDim.x) {
        int64_t start;
        int len;
        locate_block(P, kb, start, len);
        const bool vec = a.nvec > 0 && (start % 8) == 0;
        const bool full = len == kI8Block;
        // every warp reads the workers' block maxima itself: lane m holds
        // worker m's scale and its reciprocal
        float my_s = 1.f, my_r = 1.f;
        if (lane < M) {
            my_s = codec_scale(__uint_as_float(__ldcg(bmax + kb * M + lane)));
            my_r = __frcp_rn(my_s);
        }
        float g[R];
        load_f32<BF16>(a.g, start, len, vec, t, g);
        float2 g2[kI8Pairs], sum2[kI8Pairs];
        to_pairs<BF16>(g, g2);
        // -0 + d == d for every d, so the FP32 sum in worker order starts
        // from -0 without a first-worker special case
#pragma unroll
        for (int j = 0; j < kI8Pairs; ++j) sum2[j] = splat2(-0.f);
        auto add_worker = [&](int m, const float2 (&x)[kI8Pairs]) {
            const float s = __shfl_sync(0xffffffffu, my_s, m);
            const float r = __shfl_sync(0xffffffffu, my_r, m);
            float2 n[kI8Pairs];
            bool ok = true;
#pragma unroll
            for (int j = 0; j < kI8Pairs; ++j) n[j] = code2_fast(sub2(g2[j], x[j]), r, ok);
            if (!ok) {
#pragma unroll
                for (int j = 0; j < kI8Pairs; ++j) {
                    const float2 d = sub2(g2[j], x[j]);
                    n[j] = make_float2(codec_code_f(d.x, s, r), codec_code_f(d.y, s, r));
                }
            }
            // paired product, scalar sums (see mul2_rn)
#pragma unroll
            for (int j = 0; j < kI8Pairs; ++j) {
                const float2 dec = mul2_rn(n[j], splat2(s));
                sum2[j] = make_float2(__fadd_rn(sum2[j].x, dec.x), __fadd_rn(sum2[j].y, dec.y));
            }
        };
        if (full && vec) {
            constexpr int G = i8_group<BF16>();
            int m0 = 0;
            for (; m0 + G <= M; m0 += G) {
                RawPack<BF16> raw[G];
#pragma unroll
                for (int q = 0; q < G; ++q) raw[q] = load_raw<BF16>(a.x[m0 + q], start, t);
#pragma unroll
                for (int q = 0; q < G; ++q) {
                    float2 x[kI8Pairs];
                    widen_pairs<BF16>(raw[q], x);
                    add_worker(m0 + q, x);
                }
            }
            for (; m0 < M; ++m0) {
                float2 x[kI8Pairs];
                widen_pairs<BF16>(load_raw<BF16>(a.x[m0], start, t), x);
                add_worker(m0, x);
            }
        } else {
            for (int m = 0; m < M; ++m) {
                float xs[R];
                float2 x[kI8Pairs];
                load_rep<BF16>(a.x[m], start, len, vec, t, xs);
                to_pairs<BF16>(xs, x);
                add_worker(m, x);
            }
        }
        float sum[R], v[R];
#pragma unroll
        for (int j = 0; j < kI8Pairs; ++j) {
            sum[2 * j] = sum2[j].x;
            sum[2 * j + 1] = sum2[j].y;
        }
        load_f32<BF16>(a.v, start, len, vec, t, v);
        const float fM = (float)M, rM = __frcp_rn(fM);
#pragma unroll
        for (int i = 0; i < R; ++i) sum[i] = div_by_scale(sum[i], fM, rM);
        const float s = codec_scale(block_amax(sum, full, len, t, BF16, red1[parity],
                                               nullptr));
        const float rs = __frcp_rn(s);
        parity ^= 1;
        float gp[R], vp[R];
#pragma unroll
        for (int i = 0; i < R; ++i) {
            const float dq = __fmul_rn(codec_code_fast(sum[i], s, rs), s);
            const bool in = full || elem_of<BF16>(t, i) < len;
            if (in) b32 = fmaf(dq, dq, b32);
            outer_step(k, dq, g[i], v[i], gp[i], vp[i]);
            if (in) nf += not_finite(gp[i], vp[i]);
        }
        store_f32<BF16>(a.g, start, len, vec, t, gp);
        store_f32<BF16>(a.v, start, len, vec, t, vp);
        for (int m = 0; m < M; ++m) store_rep<BF16>(a.x[m], start, len, vec, t, gp);
        b64 += (double)b32;  // at most 8 terms per thread and block
        b32 = 0.f;
    }
    double e64[kMaxI8Workers];
#pragma unroll
    for (int m = 0; m < kMaxI8Workers; ++m)
        e64[m] = (t == 0 && m < M) ? e_rows[(int64_t)blockIdx.x * kMaxI8Workers + m] : 0.0;
    reduce_and_finish<kMaxI8Workers, kI8Warps>(a, M, e64, b64, nf);
}

// ------------------------------------------------------------ the codec
__global__ void __launch_bounds__(kI8Threads)
    int8_encode_kernel(const float *__restrict__ x, int8_t *__restrict__ codes,
                       float *__restrict__ scales, float *__restrict__ decoded,
                       bool vec_ok, const __grid_constant__ Int8Parts P) {
    __shared__ unsigned red[2][kI8Warps];
    const int t = threadIdx.x;
    int parity = 0;
    const int64_t nblocks = P.blk[P.n_parts];
    for (int64_t kb = blockIdx.x; kb < nblocks; kb += gridDim.x) {
        int64_t start;
        int len;
        locate_block(P, kb, start, len);
        const bool vec = vec_ok && (start % 8) == 0;
        float y[kI8PerThread];
        load_f32<false>(x, start, len, vec, t, y);
        const float s = codec_scale(block_amax(y, len == kI8Block, len, t, false,
                                               red[parity], nullptr));
        parity ^= 1;
        if (t == 0) scales[kb] = s;
        float dq[kI8PerThread];
#pragma unroll
        for (int i = 0; i < kI8PerThread; i += 4) {
            const int e = elem_of<false>(t, i);
            int q[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                q[j] = codec_code(y[i + j], s);
                dq[i + j] = __fmul_rn((float)q[j], s);
            }
            if (vec && e + 3 < len) {
                const char4 c = make_char4((signed char)q[0], (signed char)q[1],
                                           (signed char)q[2], (signed char)q[3]);
                *reinterpret_cast<char4 *>(codes + start + e) = c;
            } else {
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    if (e + j < len) codes[start + e + j] = (int8_t)q[j];
            }
        }
        if (decoded) store_f32<false>(decoded, start, len, vec, t, dq);
    }
}

__global__ void __launch_bounds__(kI8Threads)
    int8_decode_kernel(const int8_t *__restrict__ codes, const float *__restrict__ scales,
                       float *__restrict__ out, bool vec_ok,
                       const __grid_constant__ Int8Parts P) {
    const int t = threadIdx.x;
    const int64_t nblocks = P.blk[P.n_parts];
    for (int64_t kb = blockIdx.x; kb < nblocks; kb += gridDim.x) {
        int64_t start;
        int len;
        locate_block(P, kb, start, len);
        const bool vec = vec_ok && (start % 8) == 0;
        const float s = scales[kb];
        float o[kI8PerThread];
#pragma unroll
        for (int i = 0; i < kI8PerThread; i += 4) {
            const int e = elem_of<false>(t, i);
            if (vec && e + 3 < len) {
                const char4 c = *reinterpret_cast<const char4 *>(codes + start + e);
                o[i] = __fmul_rn((float)c.x, s);
                o[i + 1] = __fmul_rn((float)c.y, s);
                o[i + 2] = __fmul_rn((float)c.z, s);
                o[i + 3] = __fmul_rn((float)c.w, s);
            } else {
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    o[i + j] = (e + j < len) ? __fmul_rn((float)codes[start + e + j], s) : 0.f;
            }
        }
        store_f32<false>(out, start, len, vec, t, o);
    }
}

// ------------------------------------------------------------- launchers
namespace {
template <bool BF16>
cudaError_t round_launch(const SyncArgs &a, const Int8Parts &P, int sm_count,
                         unsigned *bmax, double *e_rows, int max_grid,
                         cudaStream_t stream, int *grid_out) {
    static int occ = 0;
    if (occ == 0) {
        int b1 = 0, b2 = 0;
        cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
            &b1, int8_scales_kernel<BF16>, kI8Threads, 0);
        if (e == cudaSuccess)
            e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
                &b2, int8_apply_kernel<BF16>, kI8Threads, 0);
        if (e != cudaSuccess) return e;
        occ = b1 < b2 ? b1 : b2;
        if (occ < 1) occ = 1;
    }
    const int64_t nblocks = P.blk[P.n_parts];
    int64_t grid = (int64_t)sm_count * occ;
    if (grid > nblocks) grid = nblocks;
    if (grid > max_grid) grid = max_grid;
    if (grid < 1) grid = 1;
    *grid_out = (int)grid;
    cudaError_t e = cudaMemsetAsync(bmax, 0, (size_t)nblocks * a.M * sizeof(unsigned),
                                    stream);
    if (e != cudaSuccess) return e;
    int8_scales_kernel<BF16><<<(unsigned)grid, kI8Threads, 0, stream>>>(a, P, bmax,
                                                                       e_rows);
    int8_apply_kernel<BF16><<<(unsigned)grid, kI8Threads, 0, stream>>>(a, P, bmax,
                                                                      e_rows);
    return cudaGetLastError();
}
}  // namespace

cudaError_t launch_int8_round(const SyncArgs &a, const Int8Parts &P, aloco_dtype dtype,
                              int sm_count, unsigned *bmax, double *e_rows, int max_grid,
                              cudaStream_t stream, int *grid_out) {
    if (a.M < 1 || a.M > kMaxI8Workers) return cudaErrorInvalidValue;
    return dtype == ALOCO_F32
               ? round_launch<false>(a, P, sm_count, bmax, e_rows, max_grid, stream,
                                     grid_out)
               : round_launch<true>(a, P, sm_count, bmax, e_rows, max_grid, stream,
                                    grid_out);
}

cudaError_t launch_int8_encode(const float *x, int8_t *codes, float *scales,
                               float *decoded, bool vec_ok, const Int8Parts &P,
                               int sm_count, cudaStream_t stream) {
    const int64_t nblocks = P.blk[P.n_parts];
    int64_t grid = (int64_t)sm_count * 8;
    if (grid > nblocks) grid = nblocks;
    if (grid < 1) return cudaSuccess;
    int8_encode_kernel<<<(unsigned)grid, kI8Threads, 0, stream>>>(x, codes, scales,
                                                                  decoded, vec_ok, P);
    return cudaGetLastError();
}

cudaError_t launch_int8_decode(const int8_t *codes, const float *scales, float *out,
                               bool vec_ok, const Int8Parts &P, int sm_count,
                               cudaStream_t stream) {
    const int64_t nblocks = P.blk[P.n_parts];
    int64_t grid = (int64_t)sm_count * 8;
    if (grid > nblocks) grid = nblocks;
    if (grid < 1) return cudaSuccess;
    int8_decode_kernel<<<(unsigned)grid, kI8Threads, 0, stream>>>(codes, scales, out,
                                                                  vec_ok, P);
    return cudaGetLastError();
}

}  // namespace aloco
