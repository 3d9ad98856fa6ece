// The INT8-communicated round (App. G.1) in one kernel: every replica is
// read from HBM once, as in the uncompressed round.
//
// CTAs of T threads work through 4096-element codec blocks (grid stride),
// 4096 / T consecutive elements per thread: one 1024-thread CTA per SM, or
// two 512-thread CTAs per SM (bf16 except M = 2; see fused_threads).  Per
// block:
//   1. theta, v and the M replica slices are staged in shared memory with
//      cp.async; each thread copies exactly the 16- or 8-byte chunks it later
//      reads, so the staging needs no barrier, and one buffer serves: the
//      next block's copies are issued as soon as the thread has read its own
//      chunks of this block (before the mean's codec, the outer step and the
//      stores), so they overlap the rest of the block;
//   2. each warp reduces every worker's max |Delta_m| (as float bits, NaN
//      above +inf); barrier; every warp then reads the 32 warp maxima of each
//      worker lane-parallel and folds them with one warp max, and lane m
//      turns worker m's maximum into its scale and reciprocal;
//   3. the workers' pseudo-gradients are encoded, decoded and summed in FP32
//      worker order, reading the replicas again from shared memory;
//   4. the mean is encoded and decoded once (its block maximum is the second
//      barrier), the corrected Nesterov step runs, and theta', v' and the
//      reset replicas are stored.
// Drift energies sum in fp32 per thread over at most 8 blocks (32 squares)
// before each warp adds them, in a fixed order, to its fp64 row.  The
// arithmetic of every element is the split form's (aloco_int8.cu), so both
// forms give the same codes, scales and outputs.
//
// Shared memory per CTA: one staging buffer of 4096 x (8 + M x element
// size) bytes (bf16 with 1024 threads and odd M: one more worker's slot).
// A second buffer, issuing the next block's copies before this block is
// computed, measured no faster anywhere and halves the room for the 512-
// thread shape.  Worker counts beyond 8 use the split form.
#include <atomic>

#include "aloco_int8.cuh"

namespace aloco {

namespace {

constexpr int kFlushBlocks = 8;
constexpr int kFusedMax = 8;

// Threads per CTA (T) and elements per thread (4096 / T), measured on
// GB300 (2^26-parameter rounds, fraction of the measured copy peak):
//   fp32: T = 1024 (one CTA per SM) 0.78-0.87 over M = 1..8; T = 512 (two
//     CTAs per SM) 0.58-0.72;
//   bf16: T = 512 0.65-0.71 over M = 1, 3..8 against 0.60-0.67 with 1024
//     threads; at M = 2, where the 1024-thread shape's worker pair fills one
//     16-byte slot, 1024 threads 0.69 against 0.65.
// ALOCO_I8_FUSED_T = 512 or 1024 forces one shape (a tuning knob).
#ifndef ALOCO_I8_FUSED_T
#define ALOCO_I8_FUSED_T 0
#endif
template <int M, bool BF16>
constexpr int fused_threads() {
    if (ALOCO_I8_FUSED_T) return ALOCO_I8_FUSED_T;
    return (BF16 && M != 2) ? 512 : 1024;
}

// Replica staging of a thread's PER elements: fp32 workers one after
// another (16 KB each).  bf16 at 4 elements per thread: workers in pairs, a
// thread's elements of workers 2p and 2p + 1 side by side in one 16-byte
// slot, so one shared-memory load feeds both; at 8 elements per thread each
// worker's slice is already one 16-byte load, one worker after another.
template <int M, bool BF16, int T>
__host__ __device__ constexpr size_t rep_bytes() {
    return (BF16 && T == 1024) ? (size_t)((M + 1) / 2) * kI8Block * 4
                               : (size_t)M * kI8Block * (BF16 ? 2 : 4);
}
template <int M, bool BF16, int T>
__host__ __device__ constexpr size_t stage_bytes() {
    return (size_t)kI8Block * 8 + rep_bytes<M, BF16, T>();
}
template <int T>
__host__ __device__ constexpr int fused_min_ctas() { return T == 512 ? 2 : 1; }
// Byte offset of worker m's element e (of 4096) in the replica staging.
template <bool BF16, int T>
__device__ __forceinline__ int rep_off(int m, int e) {
    if constexpr (BF16 && T == 1024)
        return ((m >> 1) * T + (e >> 2)) * 16 + (m & 1) * 8 + (e & 3) * 2;
    else
        return m * kI8Block * (BF16 ? 2 : 4) + e * (BF16 ? 2 : 4);
}

__device__ __forceinline__ void cp16(void *smem, const void *gmem) {
    const unsigned d = (unsigned)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d), "l"(gmem)
                 : "memory");
}
__device__ __forceinline__ void cp8(void *smem, const void *gmem) {
    const unsigned d = (unsigned)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(d), "l"(gmem)
                 : "memory");
}
__device__ __forceinline__ void cp_commit() {
    asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Stage one block: theta, v, then the replicas; thread t copies elements
// [PER t, PER t + PER) of every array (16-byte copies; 8-byte for bf16 at 4
// elements per thread).  Short or unaligned blocks are loaded element by
// element, zero beyond the end.
template <int M, bool BF16, int T>
__device__ __forceinline__ void stage_block(unsigned char *buf, const SyncArgs &a,
                                            int64_t start, int len, bool fast, int t) {
    constexpr int PER = kI8Block / T;
    float *sg = reinterpret_cast<float *>(buf);
    float *sv = sg + kI8Block;
    unsigned char *sx = reinterpret_cast<unsigned char *>(sv + kI8Block);
    const int e = PER * t;
    if (fast) {
#pragma unroll
        for (int c = 0; c < PER; c += 4) {
            cp16(sg + e + c, a.g + start + e + c);
            cp16(sv + e + c, a.v + start + e + c);
        }
#pragma unroll
        for (int m = 0; m < M; ++m) {
            if constexpr (BF16) {
                const uint16_t *src = reinterpret_cast<const uint16_t *>(a.x[m]) + start + e;
                if constexpr (PER == 4)
                    cp8(sx + rep_off<true, T>(m, e), src);
                else
                    cp16(sx + rep_off<true, T>(m, e), src);
            } else {
#pragma unroll
                for (int c = 0; c < PER; c += 4)
                    cp16(sx + rep_off<false, T>(m, e + c),
                         reinterpret_cast<const float *>(a.x[m]) + start + e + c);
            }
        }
    } else {
#pragma unroll
        for (int k = 0; k < PER; ++k) {
            const bool in = e + k < len;
            sg[e + k] = in ? a.g[start + e + k] : 0.f;
            sv[e + k] = in ? a.v[start + e + k] : 0.f;
#pragma unroll
            for (int m = 0; m < M; ++m) {
                if constexpr (BF16)
                    *reinterpret_cast<uint16_t *>(sx + rep_off<true, T>(m, e + k)) =
                        in ? reinterpret_cast<const uint16_t *>(a.x[m])[start + e + k]
                           : (uint16_t)0;
                else
                    *reinterpret_cast<float *>(sx + rep_off<false, T>(m, e + k)) =
                        in ? reinterpret_cast<const float *>(a.x[m])[start + e + k] : 0.f;
            }
        }
    }
}

__device__ __forceinline__ void widen4(uint32_t w0, uint32_t w1, float2 *o) {
    o[0] = make_float2(bf16_lo(w0), bf16_hi(w0));
    o[1] = make_float2(bf16_lo(w1), bf16_hi(w1));
}

// A thread's replica values of workers m0 and m0 + 1 (when m0 + 1 < M),
// widened exactly, as PER / 2 pairs each.
template <int M, bool BF16, int T>
__device__ __forceinline__ void staged_reps(const unsigned char *sx, int m0, int t,
                                            float2 (&a)[kI8Block / T / 2],
                                            float2 (&b)[kI8Block / T / 2]) {
    constexpr int PER = kI8Block / T;
    const int e = PER * t;
    if constexpr (BF16 && PER == 4) {
        if (m0 + 1 < M) {
            const uint4 w = *reinterpret_cast<const uint4 *>(sx + rep_off<true, T>(m0, e));
            widen4(w.x, w.y, a);
            widen4(w.z, w.w, b);
        } else {
            const uint2 w = *reinterpret_cast<const uint2 *>(sx + rep_off<true, T>(m0, e));
            widen4(w.x, w.y, a);
        }
    } else if constexpr (BF16) {
        const uint4 w = *reinterpret_cast<const uint4 *>(sx + rep_off<true, T>(m0, e));
        widen4(w.x, w.y, a);
        widen4(w.z, w.w, a + 2);
        if (m0 + 1 < M) {
            const uint4 u = *reinterpret_cast<const uint4 *>(sx + rep_off<true, T>(m0 + 1, e));
            widen4(u.x, u.y, b);
            widen4(u.z, u.w, b + 2);
        }
    } else {
#pragma unroll
        for (int c = 0; c < PER; c += 4) {
            const float4 q = *reinterpret_cast<const float4 *>(sx + rep_off<false, T>(m0, e + c));
            a[c / 2] = make_float2(q.x, q.y);
            a[c / 2 + 1] = make_float2(q.z, q.w);
            if (m0 + 1 < M) {
                const float4 r =
                    *reinterpret_cast<const float4 *>(sx + rep_off<false, T>(m0 + 1, e + c));
                b[c / 2] = make_float2(r.x, r.y);
                b[c / 2 + 1] = make_float2(r.z, r.w);
            }
        }
    }
}

// Block-wide max |y| as float bits (NaN, whose bits exceed +inf's, wins):
// each warp's maximum goes to red[warp]; after the barrier every warp folds
// the W values with one warp max (lane w reads warp w's value).
template <int PER, int W>
__device__ __forceinline__ float block_amax(const float (&y)[PER], unsigned *red) {
    unsigned m = 0;
#pragma unroll
    for (int i = 0; i < PER; ++i) m = max(m, __float_as_uint(fabsf(y[i])));
    m = __reduce_max_sync(0xffffffffu, m);
    const int lane = threadIdx.x & 31;
    if (lane == 0) red[threadIdx.x >> 5] = m;
    __syncthreads();
    return __uint_as_float(__reduce_max_sync(0xffffffffu, lane < W ? red[lane] : 0u));
}

}  // namespace

template <int M, bool BF16, int T>
__global__ void __launch_bounds__(T, (fused_min_ctas<T>()))
    int8_fused_kernel(const __grid_constant__ SyncArgs a,
                      const __grid_constant__ Int8Parts P) {
    constexpr int PER = kI8Block / T;  // elements per thread
    constexpr int NP = PER / 2;        // pairs per thread
    constexpr int W = T / 32;          // warps
    // Single buffers suffice: red_w is read between the block's two
    // barriers and rewritten only after the second; red1 is read after the
    // second and rewritten only after the next block's first.
    __shared__ unsigned red_w[M][W];                  // [worker][warp]: conflict-free reads
    __shared__ unsigned red1[W];
    __shared__ double e_w[W][M];
    __shared__ __align__(16) float2 sr[W][M + (M & 1)];  // per warp: (scale, 1/scale)
    extern __shared__ __align__(16) unsigned char stage[];

    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    if (lane < M) e_w[warp][lane] = 0.0;
    __syncwarp();
    float e_acc[M];
#pragma unroll
    for (int m = 0; m < M; ++m) e_acc[m] = 0.f;
    int since_flush = 0;
    auto flush = [&]() {
#pragma unroll
        for (int m = 0; m < M; ++m) {
            float e = e_acc[m];
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) e += __shfl_down_sync(0xffffffffu, e, off);
            if (lane == 0) e_w[warp][m] += (double)e;
            e_acc[m] = 0.f;
        }
        since_flush = 0;
    };

    float b32 = 0.f;
    double b64 = 0.0;
    unsigned nf = 0;
    const Coef k{a.c_hi, a.c_lo, a.mu_hi, a.mu_lo, a.neg_eta_hi, a.neg_eta_lo};
    const int64_t nblocks = P.blk[P.n_parts];
    const int e0 = PER * t;

    int64_t kb = blockIdx.x;
    int64_t start = 0;
    int len = 0;
    if (kb < nblocks) {
        locate_block(P, kb, start, len);
        stage_block<M, BF16, T>(stage, a, start, len,
                                len == kI8Block && a.nvec > 0 && (start % 8) == 0, t);
        cp_commit();
    }
    for (; kb < nblocks; kb += gridDim.x) {
        const bool full = len == kI8Block;
        const bool vec = a.nvec > 0 && (start % 8) == 0;
        const int64_t nk = kb + gridDim.x;
        int64_t nstart = 0;
        int nlen = 0;
        if (nk < nblocks) locate_block(P, nk, nstart, nlen);
        cp_wait<0>();  // this thread's copies of this block
        const float *sg = reinterpret_cast<const float *>(stage);
        const float *sv = sg + kI8Block;
        const unsigned char *sx = reinterpret_cast<const unsigned char *>(sv + kI8Block);

        float g[PER];
#pragma unroll
        for (int c = 0; c < PER; c += 4) {
            const float4 q = *reinterpret_cast<const float4 *>(sg + e0 + c);
            g[c] = q.x; g[c + 1] = q.y; g[c + 2] = q.z; g[c + 3] = q.w;
        }
        float2 g2[NP];
#pragma unroll
        for (int j = 0; j < NP; ++j) g2[j] = make_float2(g[2 * j], g[2 * j + 1]);

        // 2. block maxima and energies of every worker
        auto worker_max = [&](int m, const float2 (&x)[NP]) {
            float2 d[NP];
#pragma unroll
            for (int j = 0; j < NP; ++j) d[j] = sub2(g2[j], x[j]);
            float mf = 0.f;
            float2 e2 = __fmul2_rn(d[0], d[0]);
#pragma unroll
            for (int j = 0; j < NP; ++j) {
                mf = fmaxf(mf, fmaxf(fabsf(d[j].x), fabsf(d[j].y)));
                if (j > 0) e2 = __ffma2_rn(d[j], d[j], e2);
            }
            const float e = __fadd_rn(e2.x, e2.y);
            unsigned mx = __float_as_uint(mf);
            if (!isfinite(e)) {  // a NaN or infinity: take the maximum by the bits
                mx = 0;
#pragma unroll
                for (int j = 0; j < NP; ++j)
                    mx = max(mx, max(__float_as_uint(fabsf(d[j].x)),
                                     __float_as_uint(fabsf(d[j].y))));
            }
            e_acc[m] += e;
            mx = __reduce_max_sync(0xffffffffu, mx);
            if (lane == 0) red_w[m][warp] = mx;
        };
#pragma unroll
        for (int m = 0; m < M; m += 2) {
            float2 xa[NP], xb[NP];
            staged_reps<M, BF16, T>(sx, m, t, xa, xb);
            worker_max(m, xa);
            if (m + 1 < M) worker_max(m + 1, xb);
        }
        if (++since_flush == kFlushBlocks) flush();
        __syncthreads();
        {
            // every warp folds the W warp maxima of each worker (lane w reads
            // warp w's); lane m keeps worker m's and writes its scale and
            // reciprocal to this warp's table
            unsigned mine = 0;
#pragma unroll
            for (int m = 0; m < M; ++m) {
                const unsigned w =
                    __reduce_max_sync(0xffffffffu, lane < W ? red_w[m][lane] : 0u);
                mine = lane == m ? w : mine;
            }
            if (lane < M) {
                const float sc = codec_scale(__uint_as_float(mine));
                sr[warp][lane] = make_float2(sc, __frcp_rn(sc));
            }
            __syncwarp();
        }

        // 3. encode, decode and sum in worker order
        float2 sum2[NP];
#pragma unroll
        for (int j = 0; j < NP; ++j) sum2[j] = splat2(-0.f);
        auto add_worker = [&](float2 scr, const float2 (&x)[NP]) {
            const float s = scr.x, r = scr.y;
            bool ok = true;
            float2 n[NP];
#pragma unroll
            for (int j = 0; j < NP; ++j) n[j] = code2_fast(sub2(g2[j], x[j]), r, ok);
            if (!ok) {
#pragma unroll
                for (int j = 0; j < NP; ++j) {
                    const float2 d = sub2(g2[j], x[j]);
                    n[j] = make_float2(codec_code_f(d.x, s, r), codec_code_f(d.y, s, r));
                }
            }
            // paired products, scalar sums (see mul2_rn)
#pragma unroll
            for (int j = 0; j < NP; ++j) {
                const float2 q = mul2_rn(n[j], splat2(s));
                sum2[j] = make_float2(__fadd_rn(sum2[j].x, q.x), __fadd_rn(sum2[j].y, q.y));
            }
        };
#pragma unroll
        for (int m = 0; m < M; m += 2) {
            const float4 scr = *reinterpret_cast<const float4 *>(&sr[warp][m]);
            float2 xa[NP], xb[NP];
            staged_reps<M, BF16, T>(sx, m, t, xa, xb);
            add_worker(make_float2(scr.x, scr.y), xa);
            if (m + 1 < M) add_worker(make_float2(scr.z, scr.w), xb);
        }

        // 4. the mean's codec, the outer step and the stores
        float v[PER];
#pragma unroll
        for (int c = 0; c < PER; c += 4) {
            const float4 q = *reinterpret_cast<const float4 *>(sv + e0 + c);
            v[c] = q.x; v[c + 1] = q.y; v[c + 2] = q.z; v[c + 3] = q.w;
        }
        // this thread has read all of its staged chunks: their slots take
        // the next block's copies while the rest of this block runs
        if (nk < nblocks) {
            stage_block<M, BF16, T>(stage, a, nstart, nlen,
                                    nlen == kI8Block && a.nvec > 0 && (nstart % 8) == 0, t);
            cp_commit();
        }
        float sum[PER];
#pragma unroll
        for (int j = 0; j < NP; ++j) {
            sum[2 * j] = sum2[j].x;
            sum[2 * j + 1] = sum2[j].y;
        }
        const float fM = (float)M, rM = __frcp_rn(fM);
#pragma unroll
        for (int i = 0; i < PER; ++i) sum[i] = div_by_scale(sum[i], fM, rM);
        // elements beyond a short block hold 0 and do not move the maximum
        const float s = codec_scale(block_amax<PER, W>(sum, red1));
        const float rs = __frcp_rn(s);
        float gp[PER], vp[PER];
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const float dq = __fmul_rn(codec_code_fast(sum[i], s, rs), s);
            const bool in = full || e0 + i < len;
            if (in) b32 = fmaf(dq, dq, b32);
            outer_step(k, dq, g[i], v[i], gp[i], vp[i]);
            if (in) nf += not_finite(gp[i], vp[i]);
        }
        if (full && vec) {
#pragma unroll
            for (int c = 0; c < PER; c += 4) {
                __stcs(reinterpret_cast<float4 *>(a.g + start + e0 + c),
                       make_float4(gp[c], gp[c + 1], gp[c + 2], gp[c + 3]));
                __stcs(reinterpret_cast<float4 *>(a.v + start + e0 + c),
                       make_float4(vp[c], vp[c + 1], vp[c + 2], vp[c + 3]));
            }
            if constexpr (BF16) {
                uint32_t w[NP];
#pragma unroll
                for (int j = 0; j < NP; ++j) w[j] = pack_bf16x2(gp[2 * j], gp[2 * j + 1]);
#pragma unroll
                for (int m = 0; m < M; ++m) {
                    uint16_t *dst = reinterpret_cast<uint16_t *>(a.x[m]) + start + e0;
                    if constexpr (PER == 4)
                        __stcs(reinterpret_cast<uint2 *>(dst), make_uint2(w[0], w[1]));
                    else
                        __stcs(reinterpret_cast<uint4 *>(dst), make_uint4(w[0], w[1], w[2], w[3]));
                }
            } else {
#pragma unroll
                for (int m = 0; m < M; ++m)
#pragma unroll
                    for (int c = 0; c < PER; c += 4)
                        __stcs(reinterpret_cast<float4 *>(
                                   reinterpret_cast<float *>(a.x[m]) + start + e0 + c),
                               make_float4(gp[c], gp[c + 1], gp[c + 2], gp[c + 3]));
            }
        } else {
#pragma unroll
            for (int i = 0; i < PER; ++i) {
                if (e0 + i >= len) continue;
                a.g[start + e0 + i] = gp[i];
                a.v[start + e0 + i] = vp[i];
#pragma unroll
                for (int m = 0; m < M; ++m) {
                    if constexpr (BF16)
                        reinterpret_cast<__nv_bfloat16 *>(a.x[m])[start + e0 + i] =
                            __float2bfloat16_rn(gp[i]);
                    else
                        reinterpret_cast<float *>(a.x[m])[start + e0 + i] = gp[i];
                }
            }
        }
        b64 += (double)b32;  // at most PER terms per thread and block
        b32 = 0.f;

        start = nstart;
        len = nlen;
    }
    cp_wait<0>();
    if (since_flush > 0) flush();
    __syncthreads();
    double e64[M];
#pragma unroll
    for (int m = 0; m < M; ++m) {
        double e = 0.0;
        if (t == 0) {
#pragma unroll
            for (int w = 0; w < W; ++w) e += e_w[w][m];
        }
        e64[m] = e;
    }
    reduce_and_finish<M, W>(a, M, e64, b64, nf);
}

namespace {

template <int M, bool BF16>
cudaError_t fused_launch(const SyncArgs &a, const Int8Parts &P, int sm_count,
                         int max_grid, cudaStream_t stream, int *grid_out) {
    constexpr int T = fused_threads<M, BF16>();
    constexpr size_t smem = stage_bytes<M, BF16, T>();
    static PerDevice occ_cache;  // attribute set-up and occupancy, per device
    const int dev = PerDevice::device();
    int occ = occ_cache.get(dev);
    if (occ == 0) {
        cudaError_t e = cudaFuncSetAttribute(int8_fused_kernel<M, BF16, T>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e == cudaSuccess)
            e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
                &occ, int8_fused_kernel<M, BF16, T>, T, smem);
        if (e != cudaSuccess) return e;
        if (occ < 1) occ = 1;
        occ_cache.set(dev, occ);
    }
    const int64_t nblocks = P.blk[P.n_parts];
    int64_t grid = (int64_t)sm_count * occ;
    if (grid > nblocks) grid = nblocks;
    if (grid > max_grid) grid = max_grid;
    if (grid < 1) grid = 1;
    *grid_out = (int)grid;
    int8_fused_kernel<M, BF16, T><<<(unsigned)grid, T, smem, stream>>>(a, P);
    return cudaGetLastError();
}

template <bool BF16>
cudaError_t fused_dispatch(const SyncArgs &a, const Int8Parts &P, int sm_count,
                           int max_grid, cudaStream_t stream, int *grid_out) {
    switch (a.M) {
        case 1: return fused_launch<1, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        case 2: return fused_launch<2, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        case 3: return fused_launch<3, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        case 4: return fused_launch<4, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        case 5: return fused_launch<5, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        case 6: return fused_launch<6, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        case 7: return fused_launch<7, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        default: return fused_launch<8, BF16>(a, P, sm_count, max_grid, stream, grid_out);
    }
}

}  // namespace

bool int8_fused_fits(int M, aloco_dtype dtype) {
    (void)dtype;
    return M >= 1 && M <= kFusedMax;
}

cudaError_t launch_int8_fused(const SyncArgs &a, const Int8Parts &P, aloco_dtype dtype,
                              int sm_count, int max_grid, cudaStream_t stream,
                              int *grid_out) {
    if (!int8_fused_fits(a.M, dtype)) return cudaErrorInvalidValue;
    return dtype == ALOCO_BF16 ? fused_dispatch<true>(a, P, sm_count, max_grid, stream, grid_out)
                               : fused_dispatch<false>(a, P, sm_count, max_grid, stream, grid_out);
}

}  // namespace aloco
