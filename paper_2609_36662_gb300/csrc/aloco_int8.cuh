// Shared pieces of the INT8-communicated round (App. G.1): block
// geometry, per-thread loads and stores, the FP32 codec (scale, exact code,
// decode) and paired-fp32 helpers.  Included by the split (two-kernel) and
// the fused (one-kernel) round and by the stand-alone codec kernels.
#pragma once

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
constexpr int kI8Warps = kI8Threads / 32;


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

// Nearest integer, ties to even, of |t| < 2^22 on the fp32 adder: t + 1.5 *
// 2^23 has no fraction bits left, so the addition rounds t at the units
// place (to even on a tie), and subtracting the constant back is exact.
// This keeps the hot loops off the conversion instruction, which on this
// part issues at the low fp64 rate.  Explicit .rn PTX keeps the compiler
// from folding the pair away.  (A zero result is +0.)
constexpr float kRoundMagic = 12582912.f;  // 1.5 * 2^23
__device__ __forceinline__ float rint_small(float t) {
    float u, n;
    asm("add.rn.f32 %0, %1, %2;" : "=f"(u) : "f"(t), "f"(kRoundMagic));
    asm("add.rn.f32 %0, %1, %2;" : "=f"(n) : "f"(u), "f"(-kRoundMagic));
    return n;
}

// The same code from the product y r alone when that is provably the same
// decision: |y r - y/s| <= 2^-23 |y/s| < 2^-16 for |y r| < 127, so a
// product at least 2^-14 away from every half-integer rounds like the
// quotient.  Products nearer a half-integer, at or beyond 127, or not
// finite take the exact quotient.
__device__ __forceinline__ float codec_code_fast(float y, float s, float r) {
    const float t = __fmul_rn(y, r);
    const float n = rint_small(t);  // NaN or infinite t fails the test below
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
// Paired sum and product with explicit .rn rounding in PTX.  ptxas (CUDA
// 13.0) was measured to contract a single-use paired product into a
// following paired .rn add (a paired FMA), which skips the rounding of the
// decoded value q * s that the codec defines; a one-ulp change in the mean
// then moves some quotients across a half-integer.  So decoded values are
// summed with the scalar __fadd_rn, which is never contracted.  The paired
// add serves only the rounding of a product in code2_fast, where a
// contraction would round the exact product instead, and the half-integer
// margin test there covers that difference.
__device__ __forceinline__ float2 add2_rn(float2 a, float2 b) {
    float2 r;
    asm("{\n\t.reg .b64 pa, pb, pd;\n\t"
        "mov.b64 pa, {%2, %3};\n\tmov.b64 pb, {%4, %5};\n\t"
        "add.rn.f32x2 pd, pa, pb;\n\tmov.b64 {%0, %1}, pd;\n\t}"
        : "=f"(r.x), "=f"(r.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return r;
}
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
    // rint_small of both lanes; an infinite or NaN product gives a NaN
    // difference below and fails the test
    const float2 n = add2_rn(add2_rn(t, splat2(kRoundMagic)), splat2(-kRoundMagic));
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

// Workers a round may have (the statistics rows of the reduction).
constexpr int kMaxI8Workers = 16;

// A replica's raw pack of one thread for any block: the unconditional
// 16-byte load on full, aligned blocks, element loads (zero beyond the
// block's end) otherwise.  Zero-filled elements have Delta = 0 and add
// nothing to a maximum, an energy or a sum.
template <bool BF16>
__device__ __forceinline__ RawPack<BF16> load_raw_any(const void *p, int64_t start, int len,
                                                      bool fast, int t) {
    if (fast) return load_raw<BF16>(p, start, t);
    RawPack<BF16> r;
    if constexpr (BF16) {
        const uint16_t *h = reinterpret_cast<const uint16_t *>(p) + start;
        uint32_t w[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int e = 8 * t + 2 * j;
            const uint32_t lo = e < len ? h[e] : 0u;
            const uint32_t hi = e + 1 < len ? h[e + 1] : 0u;
            w[j] = lo | (hi << 16);
        }
        r.q[0] = make_uint4(w[0], w[1], w[2], w[3]);
    } else {
        const float *f = reinterpret_cast<const float *>(p) + start;
        float o[kI8PerThread];
#pragma unroll
        for (int i = 0; i < kI8PerThread; ++i) {
            const int e = elem_of<false>(t, i);
            o[i] = e < len ? f[e] : 0.f;
        }
        r.q[0] = make_float4(o[0], o[1], o[2], o[3]);
        r.q[1] = make_float4(o[4], o[5], o[6], o[7]);
    }
    return r;
}

}  // namespace aloco
