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
#include "aloco_int8.cuh"

namespace aloco {

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

// ------------------------------------------------- the round, split form
// Two streaming kernels, one CTA per 4096-element block at a time
// (persistent grid stride over blocks, 8 elements per thread, the same grid
// for both).  This form serves every M; the fused kernel
// (aloco_int8_fused.cu) replaces it where a thread can hold its packed
// replica values in registers.
//   scales reads theta and the replicas; each warp folds every worker's
//          max |Delta_m| into the block's slot with an atomic max on the
//          float bits and keeps its fp64 drift energies, written to
//          e_rows[blockIdx.x] at the end; it has no block barrier;
//   apply  reads theta, v and the replicas again; with the scales known the
//          encode / decode / FP32 sum over workers streams freely, and only
//          the mean's block maximum needs a barrier.
// Both are deterministic: maxima are order-independent, and energies are
// added in warp order.
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
    static PerDevice cache;
    const int dev = PerDevice::device();
    int occ = cache.get(dev);
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
        cache.set(dev, occ);
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
