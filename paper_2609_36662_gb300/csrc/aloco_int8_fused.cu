// The INT8-communicated round (App. G.1) in one kernel: every replica is
// read from HBM once, as in the uncompressed round.
//
// Per 4096-element block, one CTA of 512 threads (8 elements each):
//   1. each thread copies its 16-byte chunks of theta, v and the M replicas
//      into shared memory with cp.async (no register holds data in flight,
//      so all M + 2 arrays stream at once) and waits for its own copies;
//   2. each warp reduces every worker's max |Delta_m| (as float bits, NaN
//      above +inf) and its sum Delta_m^2; barrier; lanes m < M of every warp
//      fold worker m's 16 warp maxima into its scale and reciprocal;
//   3. the workers' pseudo-gradients are encoded, decoded and summed in FP32
//      worker order, reading the replicas again from shared memory;
//   4. the mean is encoded and decoded once (its block maximum is the second
//      barrier), the corrected Nesterov step runs, and theta', v' and the
//      reset replicas are stored.
// A thread reads back only the chunks it copied, so the staging needs no
// barrier of its own, and the next block's copies may start as soon as the
// thread is done with the current one.  The arithmetic of every step is the
// split form's (aloco_int8.cu), so both forms give the same codes, scales
// and outputs.  The staging takes (M + 2) x 16 KB (fp32) or (M x 8 + 32) KB
// (bf16) per CTA; worker counts beyond bf16 M = 8 or fp32 M = 4 would leave
// fewer than two CTAs per SM and use the split form.
#include <atomic>

#include "aloco_int8.cuh"

namespace aloco {

// Minimum resident CTAs per SM asked of the compiler: every instantiation
// but fp32 M = 4 fits two CTAs' registers (64 per thread) on its own, and
// bounding those makes it spill; fp32 M = 4 is held to two with a small
// spill rather than dropping to one CTA per SM.
template <int M, bool BF16>
constexpr int fused_min_blocks() { return (!BF16 && M == 4) ? 2 : 0; }

constexpr int kFusedMaxBf16 = 8;
constexpr int kFusedMaxF32 = 4;

// 16-byte asynchronous copy global -> shared (L2 only), and the wait for
// all of this thread's outstanding copies.
__device__ __forceinline__ void cp_async16(void *smem, const void *gmem) {
    const unsigned d = (unsigned)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(gmem)
                 : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

// Stage one thread's 8 elements of an fp32 array (two 16-byte chunks at the
// fp32 layout's positions) or of a bf16 replica (one chunk) in shared
// memory; element loads with zero fill where the block is short or not
// 16-byte aligned.
template <bool BF16_LAYOUT>
__device__ __forceinline__ void stage_f32(float *sm, const float *p, int64_t start, int len,
                                          bool fast, int t) {
#pragma unroll
    for (int i = 0; i < kI8PerThread; i += 4) {
        const int e = elem_of<BF16_LAYOUT>(t, i);
        if (fast) {
            cp_async16(sm + e, p + start + e);
        } else {
#pragma unroll
            for (int k = 0; k < 4; ++k) sm[e + k] = (e + k < len) ? p[start + e + k] : 0.f;
        }
    }
}
__device__ __forceinline__ void stage_bf16(uint16_t *sm, const uint16_t *p, int64_t start,
                                           int len, bool fast, int t) {
    const int e = 8 * t;
    if (fast) {
        cp_async16(sm + e, p + start + e);
    } else {
#pragma unroll
        for (int k = 0; k < 8; ++k) sm[e + k] = (e + k < len) ? p[start + e + k] : (uint16_t)0;
    }
}

// A thread's replica values, widened exactly, from its staged chunks.
template <bool BF16>
__device__ __forceinline__ void staged_pairs(const void *sm, int t, float2 (&o)[kI8Pairs]) {
    RawPack<BF16> r;
    if constexpr (BF16) {
        r.q[0] = *reinterpret_cast<const uint4 *>(reinterpret_cast<const uint16_t *>(sm) + 8 * t);
    } else {
        const float *f = reinterpret_cast<const float *>(sm);
        r.q[0] = *reinterpret_cast<const float4 *>(f + 4 * t);
        r.q[1] = *reinterpret_cast<const float4 *>(f + 2048 + 4 * t);
    }
    widen_pairs<BF16>(r, o);
}

template <bool BF16>
__device__ __forceinline__ void staged_f32(const float *sm, int t, float (&o)[kI8PerThread]) {
#pragma unroll
    for (int i = 0; i < kI8PerThread; i += 4) {
        const float4 q = *reinterpret_cast<const float4 *>(sm + elem_of<BF16>(t, i));
        o[i] = q.x; o[i + 1] = q.y; o[i + 2] = q.z; o[i + 3] = q.w;
    }
}

template <int M, bool BF16>
constexpr size_t fused_smem_bytes() {
    return (size_t)kI8Block * (2 * sizeof(float) + M * (BF16 ? 2 : 4));
}

template <int M, bool BF16>
__global__ void __launch_bounds__(kI8Threads, (fused_min_blocks<M, BF16>()))
    int8_fused_kernel(const __grid_constant__ SyncArgs a,
                      const __grid_constant__ Int8Parts P) {
    constexpr int R = kI8PerThread;
    // Single buffers suffice: red_w is read between the block's two
    // barriers and rewritten only after the second; red1 is read after the
    // second and rewritten only after the next block's first.
    __shared__ unsigned red_w[kI8Warps][M];
    __shared__ unsigned red1[kI8Warps];
    __shared__ double e_w[kI8Warps][M];
    extern __shared__ __align__(16) unsigned char stage[];
    float *sg = reinterpret_cast<float *>(stage);
    float *sv = sg + kI8Block;
    unsigned char *sx = reinterpret_cast<unsigned char *>(sv + kI8Block);
    constexpr int kRepBytes = kI8Block * (BF16 ? 2 : 4);

    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    if (lane < M) e_w[warp][lane] = 0.0;
    __syncwarp();
    float b32 = 0.f;
    double b64 = 0.0;
    unsigned nf = 0;
    const Coef k{a.c_hi, a.c_lo, a.mu_hi, a.mu_lo, a.neg_eta_hi, a.neg_eta_lo};
    const int64_t nblocks = P.blk[P.n_parts];
    for (int64_t kb = blockIdx.x; kb < nblocks; kb += gridDim.x) {
        int64_t start;
        int len;
        locate_block(P, kb, start, len);
        const bool vec = a.nvec > 0 && (start % 8) == 0;
        const bool full = len == kI8Block;
        const bool fast = full && vec;

        // 1. stage theta, the replicas and v
        stage_f32<BF16>(sg, a.g, start, len, fast, t);
#pragma unroll
        for (int m = 0; m < M; ++m) {
            if constexpr (BF16)
                stage_bf16(reinterpret_cast<uint16_t *>(sx + m * kRepBytes),
                           reinterpret_cast<const uint16_t *>(a.x[m]), start, len, fast, t);
            else
                stage_f32<false>(reinterpret_cast<float *>(sx + m * kRepBytes),
                                 reinterpret_cast<const float *>(a.x[m]), start, len, fast, t);
        }
        stage_f32<BF16>(sv, a.v, start, len, fast, t);
        cp_async_wait_all();
        float g[R];
        staged_f32<BF16>(sg, t, g);
        float2 g2[kI8Pairs];
        to_pairs<BF16>(g, g2);

        // 2. block maxima and energies of every worker
#pragma unroll
        for (int m = 0; m < M; ++m) {
            float2 x[kI8Pairs];
            staged_pairs<BF16>(sx + m * kRepBytes, t, x);
            float mf = 0.f;
            float2 e2 = make_float2(0.f, 0.f);
#pragma unroll
            for (int j = 0; j < kI8Pairs; ++j) {
                const float2 d = sub2(g2[j], x[j]);
                mf = fmaxf(mf, fmaxf(fabsf(d.x), fabsf(d.y)));
                e2 = __ffma2_rn(d, d, e2);
            }
            float e = __fadd_rn(e2.x, e2.y);
            unsigned mx = __float_as_uint(mf);
            if (!isfinite(e)) {  // a NaN or infinity: take the maximum by the bits
                mx = 0;
#pragma unroll
                for (int j = 0; j < kI8Pairs; ++j) {
                    const float2 d = sub2(g2[j], x[j]);
                    mx = max(mx, max(__float_as_uint(fabsf(d.x)), __float_as_uint(fabsf(d.y))));
                }
            }
            mx = __reduce_max_sync(0xffffffffu, mx);
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) e += __shfl_down_sync(0xffffffffu, e, off);
            if (lane == 0) {
                red_w[warp][m] = mx;
                e_w[warp][m] += (double)e;
            }
        }
        __syncthreads();
        float my_s = 1.f, my_r = 1.f;
        if (lane < M) {
            unsigned mx = red_w[0][lane];
#pragma unroll
            for (int w = 1; w < kI8Warps; ++w) mx = max(mx, red_w[w][lane]);
            my_s = codec_scale(__uint_as_float(mx));
            my_r = __frcp_rn(my_s);
        }

        // 3. encode, decode and sum in worker order
        float2 sum2[kI8Pairs];
#pragma unroll
        for (int j = 0; j < kI8Pairs; ++j) sum2[j] = splat2(-0.f);
#pragma unroll
        for (int m = 0; m < M; ++m) {
            const float s = __shfl_sync(0xffffffffu, my_s, m);
            const float r = __shfl_sync(0xffffffffu, my_r, m);
            float2 x[kI8Pairs], n[kI8Pairs];
            staged_pairs<BF16>(sx + m * kRepBytes, t, x);
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
#pragma unroll
            for (int j = 0; j < kI8Pairs; ++j) {
                const float2 dec = mul2_rn(n[j], splat2(s));
                sum2[j] = make_float2(__fadd_rn(sum2[j].x, dec.x), __fadd_rn(sum2[j].y, dec.y));
            }
        }

        // 4. the mean's codec, the outer step and the stores
        float sum[R];
#pragma unroll
        for (int j = 0; j < kI8Pairs; ++j) {
            sum[2 * j] = sum2[j].x;
            sum[2 * j + 1] = sum2[j].y;
        }
        const float fM = (float)M, rM = __frcp_rn(fM);
#pragma unroll
        for (int i = 0; i < R; ++i) sum[i] = div_by_scale(sum[i], fM, rM);
        // elements beyond a short block hold 0 and do not move the maximum
        const float s = codec_scale(block_amax(sum, true, len, t, BF16, red1, nullptr));
        const float rs = __frcp_rn(s);
        float v[R];
        staged_f32<BF16>(sv, t, v);
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
#pragma unroll
        for (int m = 0; m < M; ++m) store_rep<BF16>(a.x[m], start, len, vec, t, gp);
        b64 += (double)b32;  // at most 8 terms per thread and block
        b32 = 0.f;
    }
    __syncthreads();
    double e64[kMaxI8Workers];
#pragma unroll
    for (int m = 0; m < kMaxI8Workers; ++m) {
        double e = 0.0;
        if (t == 0 && m < M) {
#pragma unroll
            for (int w = 0; w < kI8Warps; ++w) e += e_w[w][m];
        }
        e64[m] = e;
    }
    reduce_and_finish<kMaxI8Workers, kI8Warps>(a, M, e64, b64, nf);
}

namespace {

template <int M, bool BF16>
cudaError_t fused_launch(const SyncArgs &a, const Int8Parts &P, int sm_count,
                         int max_grid, cudaStream_t stream, int *grid_out) {
    constexpr size_t smem = fused_smem_bytes<M, BF16>();
    static std::atomic<int> occ_cache{0};
    int occ = occ_cache.load(std::memory_order_relaxed);
    if (occ == 0) {
        cudaError_t e = cudaFuncSetAttribute(int8_fused_kernel<M, BF16>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e == cudaSuccess)
            e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
                &occ, int8_fused_kernel<M, BF16>, kI8Threads, smem);
        if (e != cudaSuccess) return e;
        if (occ < 1) occ = 1;
        occ_cache.store(occ, std::memory_order_relaxed);
    }
    const int64_t nblocks = P.blk[P.n_parts];
    int64_t grid = (int64_t)sm_count * occ;
    if (grid > nblocks) grid = nblocks;
    if (grid > max_grid) grid = max_grid;
    if (grid < 1) grid = 1;
    *grid_out = (int)grid;
    int8_fused_kernel<M, BF16><<<(unsigned)grid, kI8Threads, smem, stream>>>(a, P);
    return cudaGetLastError();
}

}  // namespace

bool int8_fused_fits(int M, aloco_dtype dtype) {
    return M >= 1 && M <= (dtype == ALOCO_BF16 ? kFusedMaxBf16 : kFusedMaxF32);
}

cudaError_t launch_int8_fused(const SyncArgs &a, const Int8Parts &P, aloco_dtype dtype,
                              int sm_count, int max_grid, cudaStream_t stream,
                              int *grid_out) {
    if (!int8_fused_fits(a.M, dtype)) return cudaErrorInvalidValue;
    if (dtype == ALOCO_BF16) {
        switch (a.M) {
            case 1: return fused_launch<1, true>(a, P, sm_count, max_grid, stream, grid_out);
            case 2: return fused_launch<2, true>(a, P, sm_count, max_grid, stream, grid_out);
            case 3: return fused_launch<3, true>(a, P, sm_count, max_grid, stream, grid_out);
            case 4: return fused_launch<4, true>(a, P, sm_count, max_grid, stream, grid_out);
            case 5: return fused_launch<5, true>(a, P, sm_count, max_grid, stream, grid_out);
            case 6: return fused_launch<6, true>(a, P, sm_count, max_grid, stream, grid_out);
            case 7: return fused_launch<7, true>(a, P, sm_count, max_grid, stream, grid_out);
            default: return fused_launch<8, true>(a, P, sm_count, max_grid, stream, grid_out);
        }
    }
    switch (a.M) {
        case 1: return fused_launch<1, false>(a, P, sm_count, max_grid, stream, grid_out);
        case 2: return fused_launch<2, false>(a, P, sm_count, max_grid, stream, grid_out);
        case 3: return fused_launch<3, false>(a, P, sm_count, max_grid, stream, grid_out);
        default: return fused_launch<4, false>(a, P, sm_count, max_grid, stream, grid_out);
    }
}

}  // namespace aloco
