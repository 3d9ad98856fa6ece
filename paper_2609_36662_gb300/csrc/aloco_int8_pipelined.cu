// The pipelined form of the INT8-communicated round (App. G.1) for bf16
// replicas: the next codec block's copies overlap the current block's codec
// work.
//
// The codec of a 4096-element block needs every worker's maximum over the
// whole block before any of its values can be encoded, so each worker's
// slice is read twice from shared memory (maximum and energy, then encode,
// decode and sum).  With many workers one staged block takes most of an
// SM's shared memory, and a kernel that stages the next block only after
// the current one is encoded leaves HBM idle while it computes.  Here one
// 1024-thread CTA per SM keeps
//   - theta and v of two blocks (double buffered, 64 KB),
//   - one slot per worker for the replica slices of one block (8 KB each),
//   - the output tiles,
// and every slot has a "full" mbarrier (the bulk copy landed) and an "empty"
// mbarrier (every warp has read it for the last time in this block).  Per
// block:
//   1. theta of the block is read into registers once its buffer is full;
//   2. worker m's maximum and energy are taken as soon as its slot is full,
//      so the block's phase 2 follows the copies as they land;
//   3. barrier 1: the maxima become scales (as in the fused kernel); thread
//      0 stores the previous block's output tiles and issues the next
//      block's theta and v into the other buffer;
//   4. the workers are encoded, decoded and summed in worker order; after a
//      warp's last read of slot m it arrives on slot m's empty barrier, and
//      thread 0 issues the next block's copy into every slot it finds empty,
//      so the next block streams in while this one is encoded;
//   5. the mean's codec (barrier 2), then thread 0 issues the slots not yet
//      refilled, and the outer step writes the output tiles (theta' once, in
//      bf16; the replica reset is M bulk stores of that tile).
// Short or unaligned blocks (tensor ends) are staged by every thread,
// element by element, into its own slots.  The arithmetic of every element
// is the fused and the split form's, so all three give the same codes,
// scales and outputs bit for bit.
//
// Every wait is bounded (about 2 s).  A wait that runs out sets the round's
// error word: the CTA leaves its loop together at barrier 1, thread 0 waits
// (bounded) for the copies it issued that have not landed and for its bulk
// stores, and the host reports the error.
#include "aloco_bulk.cuh"
#include "aloco_int8.cuh"

namespace aloco {

namespace {

constexpr int kPipeT = 1024;           // threads per CTA: 4 elements each
constexpr int kPipeMinM = 2;
constexpr int kPipeMaxM = 16;
constexpr int kPipeFlush = 8;          // blocks between energy flushes
constexpr size_t kPipeSmemPerCta = 232448;
constexpr uint32_t kPipeF = kI8Block * 4;  // one fp32 array of a block
constexpr uint32_t kPipeX = kI8Block * 2;  // one bf16 replica slice

// static shared memory of the kernel and of the final reduction (a bound)
template <int M>
__host__ __device__ constexpr size_t pipe_static() {
    constexpr int W = kPipeT / 32;
    return (size_t)W * (4 * M + 4 + 8 * M + 8 * (M + 1) + 8 * (M + 1)) + 4096;
}
// theta/v double buffer and the worker slots
template <int M>
__host__ __device__ constexpr size_t pipe_in_bytes() {
    return (size_t)4 * kPipeF + (size_t)M * kPipeX;
}
// the fp32 theta' and v' tiles fit beside the bf16 theta' tile
template <int M>
__host__ __device__ constexpr bool pipe_gv() {
    return pipe_in_bytes<M>() + kPipeX + 2 * kPipeF + pipe_static<M>() <= kPipeSmemPerCta;
}
template <int M>
__host__ __device__ constexpr size_t pipe_smem() {
    return pipe_in_bytes<M>() + kPipeX + (pipe_gv<M>() ? 2 * kPipeF : 0);
}

// Block-wide max |y| as float bits (NaN, whose bits exceed +inf's, wins):
// each warp's maximum goes to red[warp]; after the barrier every warp folds
// the W values with one warp max.
template <int PER, int W>
__device__ __forceinline__ float pipe_amax(const float (&y)[PER], unsigned *red) {
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

template <int M>
__global__ void __launch_bounds__(kPipeT, 1)
    int8_pipelined_kernel(const __grid_constant__ SyncArgs a,
                     const __grid_constant__ Int8Parts P) {
    constexpr int T = kPipeT;
    constexpr int PER = kI8Block / T;  // 4 elements per thread
    constexpr int NP = PER / 2;        // pairs per thread
    constexpr int W = T / 32;
    constexpr bool GV = pipe_gv<M>();
    __shared__ unsigned red_w[M][W];                     // [worker][warp]
    __shared__ unsigned red1[W];
    __shared__ double e_w[W][M];
    __shared__ __align__(16) float2 sr[W][M + (M & 1)];  // per warp: (scale, 1/scale)
    __shared__ __align__(8) unsigned long long bar_gv[2];
    __shared__ __align__(8) unsigned long long bar_full[M];
    __shared__ __align__(8) unsigned long long bar_empty[M];
    extern __shared__ __align__(128) unsigned char smem[];
    float *gvb = reinterpret_cast<float *>(smem);      // [2][theta, v][4096]
    unsigned char *sx = smem + 4 * kPipeF;              // [M][4096] bf16
    unsigned char *ox = sx + (size_t)M * kPipeX;        // theta' (bf16)
    float *og = reinterpret_cast<float *>(ox + kPipeX);  // theta' (fp32; GV)
    float *ov = og + kI8Block;                           // v' (fp32; GV)

    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    if (lane < M) e_w[warp][lane] = 0.0;
    if (t == 0) {
        mbar_init(smem_addr(&bar_gv[0]), 1);
        mbar_init(smem_addr(&bar_gv[1]), 1);
#pragma unroll
        for (int m = 0; m < M; ++m) {
            mbar_init(smem_addr(&bar_full[m]), 1);
            mbar_init(smem_addr(&bar_empty[m]), W);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();

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
    auto bulk_block = [&](int64_t s, int l) {
        return l == kI8Block && a.nvec > 0 && (s % 8) == 0;
    };
    auto stalled = [&](int64_t kbi) {  // testing only: this block is never staged
        return a.test_stall_tile1 != 0 && kbi == a.test_stall_tile1 - 1;
    };

    // thread 0's record of copies issued and not yet seen complete (for the
    // failure path; their phases' parities are gpar[] and xpar)
    uint32_t gv_pending = 0;   // bit b: theta/v buffer b
    uint32_t x_pending = 0;    // bit m: worker slot m
    auto issue_gv = [&](int64_t kbi, int64_t s, int buf) {
        if (stalled(kbi)) return;
        const uint32_t bar = smem_addr(&bar_gv[buf]);
        float *dst = gvb + (size_t)buf * 2 * kI8Block;
        mbar_arrive_expect_tx(bar, 2 * kPipeF);
        bulk_load(smem_addr(dst), a.g + s, kPipeF, bar);
        bulk_load(smem_addr(dst + kI8Block), a.v + s, kPipeF, bar);
        gv_pending |= 1u << buf;
    };
    auto issue_x = [&](int64_t kbi, int64_t s, int m) {
        if (stalled(kbi)) return;
        const uint32_t bar = smem_addr(&bar_full[m]);
        mbar_arrive_expect_tx(bar, kPipeX);
        bulk_load(smem_addr(sx + (size_t)m * kPipeX),
                  reinterpret_cast<const unsigned char *>(a.x[m]) + s * 2, kPipeX, bar);
        x_pending |= 1u << m;
    };
    // every thread: its own 4 elements of a short or unaligned block
    auto stage_own = [&](int64_t s, int l, int buf) {
        float *dg = gvb + (size_t)buf * 2 * kI8Block;
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const int e = 4 * t + i;
            const bool in = e < l;
            dg[e] = in ? a.g[s + e] : 0.f;
            dg[kI8Block + e] = in ? a.v[s + e] : 0.f;
#pragma unroll
            for (int m = 0; m < M; ++m)
                reinterpret_cast<uint16_t *>(sx + (size_t)m * kPipeX)[e] =
                    in ? reinterpret_cast<const uint16_t *>(a.x[m])[s + e] : (uint16_t)0;
        }
        fence_proxy_async_smem();  // a later bulk copy may overwrite these bytes
    };
    auto store_tiles = [&](int64_t s) {
        if constexpr (GV) {
            bulk_store(a.g + s, smem_addr(og), kPipeF);
            bulk_store(a.v + s, smem_addr(ov), kPipeF);
        }
#pragma unroll
        for (int m = 0; m < M; ++m)
            bulk_store(reinterpret_cast<unsigned char *>(a.x[m]) + s * 2, smem_addr(ox), kPipeX);
        bulk_commit();
    };
    // a thread's values of worker slot m, widened exactly, as pairs
    auto slot = [&](int m, float2 (&o)[NP]) {
        const uint2 w = *reinterpret_cast<const uint2 *>(sx + (size_t)m * kPipeX + 8 * t);
        o[0] = make_float2(bf16_lo(w.x), bf16_hi(w.x));
        o[1] = make_float2(bf16_lo(w.y), bf16_hi(w.y));
    };

    int64_t kb = blockIdx.x;
    int64_t start = 0;
    int len = 0;
    int buf = 0;                    // theta/v buffer of the current block
    uint32_t gpar = 0u;             // bit b: parity of buffer b's next completion
    uint32_t xpar = 0u;             // parity of the worker slots' next completion
    uint32_t epar = 0u;             // parity of the empty barriers' next completion
    bool pend = false;              // the previous block's tiles wait for their stores
    int64_t pstart = 0;
    bool failed = false;
    if (kb < nblocks) {
        locate_block(P, kb, start, len);
        if (!bulk_block(start, len)) {
            stage_own(start, len, 0);
        } else if (t == 0) {
            issue_gv(kb, start, 0);
#pragma unroll
            for (int m = 0; m < M; ++m) issue_x(kb, start, m);
        }
    }
    for (; kb < nblocks; kb += gridDim.x) {
        const bool full = len == kI8Block;
        const bool bulk = bulk_block(start, len);
        const int64_t nk = kb + gridDim.x;
        int64_t nstart = 0;
        int nlen = 0;
        if (nk < nblocks) locate_block(P, nk, nstart, nlen);
        const bool next_bulk = nk < nblocks && bulk_block(nstart, nlen);
        const float *sg = gvb + (size_t)buf * 2 * kI8Block;
        const float *sv = sg + kI8Block;

        // 1. theta of the block
        bool timed_out = false;
        if (bulk) {
            timed_out = !mbar_wait(smem_addr(&bar_gv[buf]), (gpar >> buf) & 1u, nullptr);
            if (t == 0 && !timed_out) gv_pending &= ~(1u << buf);
        }
        float g[PER];
        {
            const float4 q = *reinterpret_cast<const float4 *>(sg + 4 * t);
            g[0] = q.x; g[1] = q.y; g[2] = q.z; g[3] = q.w;
        }
        float2 g2[NP];
#pragma unroll
        for (int j = 0; j < NP; ++j) g2[j] = make_float2(g[2 * j], g[2 * j + 1]);

        // 2. maxima and energies, each worker once its slot has landed
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
        for (int m = 0; m < M; ++m) {
            if (bulk && !timed_out) {
                timed_out = !mbar_wait(smem_addr(&bar_full[m]), xpar, nullptr);
                if (t == 0 && !timed_out) x_pending &= ~(1u << m);
            }
            float2 x[NP];
            slot(m, x);
            worker_max(m, x);
        }
        if (++since_flush == kPipeFlush) flush();
        // barrier 1; a wait that ran out in any thread stops the whole CTA
        // (with the parities of the phases it waited for still recorded)
        if (__syncthreads_or(timed_out)) {
            failed = true;
            break;
        }
        if (bulk) {
            gpar ^= 1u << buf;
            xpar ^= 1u;
        }
        if (t == 0) {
            // every thread wrote its part of the previous block's tiles, and
            // has finished with the other theta/v buffer
            if (pend) store_tiles(pstart);
            if (next_bulk) issue_gv(nk, nstart, buf ^ 1);
        }
        pend = false;
        {
            // every warp folds the W warp maxima of each worker (lane w reads
            // warp w's); lane m keeps worker m's and writes its scale and
            // reciprocal to this warp's table
            unsigned mine = 0;
#pragma unroll
            for (int m = 0; m < M; ++m) {
                const unsigned w = __reduce_max_sync(0xffffffffu, lane < W ? red_w[m][lane] : 0u);
                mine = lane == m ? w : mine;
            }
            if (lane < M) {
                const float sc = codec_scale(__uint_as_float(mine));
                sr[warp][lane] = make_float2(sc, __frcp_rn(sc));
            }
            __syncwarp();
        }

        // 3. encode, decode and sum in worker order; each slot is released as
        // soon as this warp has read it, and thread 0 refills the slots every
        // warp has released with the next block
        float2 sum2[NP];
#pragma unroll
        for (int j = 0; j < NP; ++j) sum2[j] = splat2(-0.f);
        uint32_t refilled = 0;  // thread 0: bit m: slot m holds the next block
#pragma unroll
        for (int m = 0; m < M; ++m) {
            const float2 scr = sr[warp][m];
            const float s = scr.x, r = scr.y;
            float2 x[NP];
            slot(m, x);
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
            if (next_bulk) {
                // this warp's last use of slot m is done (its values are in
                // the sum): release the slot
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_addr(&bar_empty[m]));
            }
            // thread 0 refills slot m - 1 if every warp has released it (the
            // others lag this warp by little); slots still held then are
            // refilled after barrier 2
            if (m >= 1 && next_bulk && t == 0 &&
                mbar_test(smem_addr(&bar_empty[m - 1]), epar)) {
                issue_x(nk, nstart, m - 1);
                refilled |= 1u << (m - 1);
            }
        }

        // 4. the mean's codec
        float sum[PER];
#pragma unroll
        for (int j = 0; j < NP; ++j) {
            sum[2 * j] = sum2[j].x;
            sum[2 * j + 1] = sum2[j].y;
        }
        const float fM = (float)M, rM = __frcp_rn(fM);
#pragma unroll
        for (int i = 0; i < PER; ++i) sum[i] = div_by_scale(sum[i], fM, rM);
        // the previous block's bulk stores have read the tiles before any
        // thread passes barrier 2 and rewrites them
        if (t == 0) bulk_wait_read();
        // barrier 2; elements beyond a short block hold 0 and do not move the
        // maximum
        const float s = codec_scale(pipe_amax<PER, W>(sum, red1));
        if (next_bulk) {
            // every warp has released every slot: the rest of the next block
            // goes in now (these waits end at once).  Should one run out
            // anyway, the slot is left unfilled, and the next block's bounded
            // wait for it stops the CTA.
            if (t == 0) {
#pragma unroll
                for (int m = 0; m < M; ++m) {
                    if ((refilled >> m) & 1u) continue;
                    if (!mbar_wait(smem_addr(&bar_empty[m]), epar, nullptr)) break;
                    issue_x(nk, nstart, m);
                }
            }
            epar ^= 1u;
        }
        const float rs = __frcp_rn(s);
        float v[PER], gp[PER], vp[PER];
        {
            const float4 q = *reinterpret_cast<const float4 *>(sv + 4 * t);
            v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
        }
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const float dq = __fmul_rn(codec_code_fast(sum[i], s, rs), s);
            const bool in = full || 4 * t + i < len;
            if (in) b32 = fmaf(dq, dq, b32);
            outer_step(k, dq, g[i], v[i], gp[i], vp[i]);
            if (in) nf += not_finite(gp[i], vp[i]);
        }

        // 5. the stores
        if (bulk) {
            *reinterpret_cast<uint2 *>(ox + 8 * t) =
                make_uint2(pack_bf16x2(gp[0], gp[1]), pack_bf16x2(gp[2], gp[3]));
            if constexpr (GV) {
                *reinterpret_cast<float4 *>(og + 4 * t) = make_float4(gp[0], gp[1], gp[2], gp[3]);
                *reinterpret_cast<float4 *>(ov + 4 * t) = make_float4(vp[0], vp[1], vp[2], vp[3]);
            } else {
                __stcs(reinterpret_cast<float4 *>(a.g + start + 4 * t),
                       make_float4(gp[0], gp[1], gp[2], gp[3]));
                __stcs(reinterpret_cast<float4 *>(a.v + start + 4 * t),
                       make_float4(vp[0], vp[1], vp[2], vp[3]));
            }
            fence_proxy_async_smem();  // the tiles are read by bulk copies
            pend = true;
            pstart = start;
        } else {
#pragma unroll
            for (int i = 0; i < PER; ++i) {
                const int e = 4 * t + i;
                if (e >= len) continue;
                a.g[start + e] = gp[i];
                a.v[start + e] = vp[i];
#pragma unroll
                for (int m = 0; m < M; ++m)
                    reinterpret_cast<__nv_bfloat16 *>(a.x[m])[start + e] =
                        __float2bfloat16_rn(gp[i]);
            }
        }
        b64 += (double)b32;
        b32 = 0.f;
        if (nk < nblocks && !next_bulk) stage_own(nstart, nlen, buf ^ 1);
        buf ^= 1;
        start = nstart;
        len = nlen;
    }
    if (failed) {
        if (t == 0) {
            atomicExch(a.error, 1u);
            // let the copies still in flight land before the CTA exits
            for (int b2 = 0; b2 < 2; ++b2)
                if ((gv_pending >> b2) & 1u)
                    mbar_wait(smem_addr(&bar_gv[b2]), (gpar >> b2) & 1u, nullptr);
#pragma unroll
            for (int m = 0; m < M; ++m)
                if (x_pending & (1u << m)) mbar_wait(smem_addr(&bar_full[m]), xpar, nullptr);
        }
    } else if (pend) {
        __syncthreads();
        if (t == 0) store_tiles(pstart);
    }
    if (t == 0) bulk_wait_all();
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

template <int M>
cudaError_t pipe_launch(const SyncArgs &a, const Int8Parts &P, int sm_count, int max_grid,
                        cudaStream_t stream, int *grid_out) {
    static_assert(pipe_smem<M>() + pipe_static<M>() <= kPipeSmemPerCta,
                  "pipelined INT8 staging exceeds shared memory");
    constexpr size_t smem = pipe_smem<M>();
    static PerDevice attr_cache;  // attribute set-up, per device
    const int dev = PerDevice::device();
    if (attr_cache.get(dev) == 0) {
        cudaError_t e = cudaFuncSetAttribute(int8_pipelined_kernel<M>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e != cudaSuccess) return e;
        attr_cache.set(dev, 1);
    }
    const int64_t nblocks = P.blk[P.n_parts];
    int64_t grid = sm_count;
    if (grid > nblocks) grid = nblocks;
    if (grid > max_grid) grid = max_grid;
    if (grid < 1) grid = 1;
    *grid_out = (int)grid;
    int8_pipelined_kernel<M><<<(unsigned)grid, kPipeT, smem, stream>>>(a, P);
    return cudaGetLastError();
}

}  // namespace

bool int8_pipelined_fits(int M, aloco_dtype dtype) {
    return dtype == ALOCO_BF16 && M >= kPipeMinM && M <= kPipeMaxM;
}

cudaError_t launch_int8_pipelined(const SyncArgs &a, const Int8Parts &P, aloco_dtype dtype,
                             int sm_count, int max_grid, cudaStream_t stream, int *grid_out) {
    if (!int8_pipelined_fits(a.M, dtype)) return cudaErrorInvalidValue;
    switch (a.M) {
        case 2: return pipe_launch<2>(a, P, sm_count, max_grid, stream, grid_out);
        case 3: return pipe_launch<3>(a, P, sm_count, max_grid, stream, grid_out);
        case 4: return pipe_launch<4>(a, P, sm_count, max_grid, stream, grid_out);
        case 5: return pipe_launch<5>(a, P, sm_count, max_grid, stream, grid_out);
        case 6: return pipe_launch<6>(a, P, sm_count, max_grid, stream, grid_out);
        case 7: return pipe_launch<7>(a, P, sm_count, max_grid, stream, grid_out);
        case 8: return pipe_launch<8>(a, P, sm_count, max_grid, stream, grid_out);
        case 9: return pipe_launch<9>(a, P, sm_count, max_grid, stream, grid_out);
        case 10: return pipe_launch<10>(a, P, sm_count, max_grid, stream, grid_out);
        case 11: return pipe_launch<11>(a, P, sm_count, max_grid, stream, grid_out);
        case 12: return pipe_launch<12>(a, P, sm_count, max_grid, stream, grid_out);
        case 13: return pipe_launch<13>(a, P, sm_count, max_grid, stream, grid_out);
        case 14: return pipe_launch<14>(a, P, sm_count, max_grid, stream, grid_out);
        case 15: return pipe_launch<15>(a, P, sm_count, max_grid, stream, grid_out);
        default: return pipe_launch<16>(a, P, sm_count, max_grid, stream, grid_out);
    }
}

}  // namespace aloco
