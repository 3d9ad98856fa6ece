// Fused outer-synchronisation pass staged through shared memory by bulk
// copies (the "tile" pass; M <= 16, 16-byte aligned buffers).
//
// The arithmetic per element is the register-streaming pass's (Algorithm 1:
// Delta_m = theta - x_m summed in worker order; the drift energies and
// ||sum||^2 of Eq. adaptive-h-core-diagnostics; the corrected Nesterov step
// of Eq. autoloco-corrected-nesterov), so theta', v' and the replica reset
// are bit-identical to that pass.  What differs is how the bytes move.
//
// CTAs of T threads walk whole blocks of 4T elements with a grid stride;
// thread t owns elements 4t .. 4t + 3 of every block.  Per block j of a CTA:
//   1. theta, v and the M replica slices arrive in one of NS shared-memory
//      stages by bulk copies (cp.async.bulk, issued by thread 0, completing
//      on the stage's mbarrier; every wait on it is bounded);
//   2. each thread reads its chunks, sums the pseudo-gradients and their
//      energies;
//   3. one barrier: the stage is free, so thread 0 issues the copies of
//      block j + NS into it, and stores block j - 1's output tiles;
//   4. the outer step runs and each thread writes its theta' (in the
//      replica type) to this block's output tile (theta' and v' in fp32 too
//      where they fit, else it stores them itself).  The replica reset is M
//      bulk stores of that one tile.
// Output tiles alternate between two sets: block j's tiles are written
// after barrier j and stored after barrier j + 1, and thread 0 waits before
// barrier j + 1 until the stores issued after barrier j (block j - 1's)
// have read their tiles, so block j + 1 may rewrite them.
// Elements after the last whole block are handled element by element.
// Drift energies sum in fp32 per thread over at most 8 blocks (32 squares)
// before each warp adds them, in a fixed order, to its fp64 row; the
// statistics agree with the register pass within the statistics tolerance.
#include "aloco_bulk.cuh"
#include "aloco_sync_kernel.cuh"

namespace aloco {

namespace {

constexpr int kTileMaxM = 16;
constexpr int kTileFlushBlocks = 8;
constexpr size_t kTileSmemPerSm = 233472;   // shared memory of one SM
constexpr size_t kTileSmemReserved = 1024;  // reserved by the system per CTA

// Tuning knobs: threads per CTA (0: the table in tile_threads; else 256,
// 512 or 1024), shared-memory stages (0: the table in tile_stages; else 1
// or 2) and the fp32 output tiles (0: where they fit; 1: never).
#ifndef ALOCO_TILE_T
#define ALOCO_TILE_T 0
#endif
#ifndef ALOCO_TILE_NS
#define ALOCO_TILE_NS 0
#endif
#ifndef ALOCO_TILE_NOGV
#define ALOCO_TILE_NOGV 0
#endif
#ifndef ALOCO_TILE_CTAS
#define ALOCO_TILE_CTAS 0  // CTAs per SM (0: the table in tile_ctas)
#endif

template <bool BF16>
__host__ __device__ constexpr int tile_es() { return BF16 ? 2 : 4; }
// CTAs per SM the shared-memory budget is planned for: 1024 threads per SM
// (64 registers a thread), except fp32 with M > 8, whose 2048-element stage
// fits one 512-thread CTA per SM
template <int M, bool BF16, int T>
__host__ __device__ constexpr int tile_ctas() {
    return ALOCO_TILE_CTAS ? ALOCO_TILE_CTAS : (!BF16 && M > 8) ? 1 : 1024 / T;
}
template <int M, bool BF16, int T>
__host__ __device__ constexpr size_t tile_budget() {
    return kTileSmemPerSm / tile_ctas<M, BF16, T>() - kTileSmemReserved;
}
// static shared memory: energy rows, the final reduction, barriers (bound)
template <int M, int T>
__host__ __device__ constexpr size_t tile_static() {
    return (size_t)(T / 32) * (16 * M + 16) + 4096;
}
template <int M, bool BF16, int T>
__host__ __device__ constexpr size_t tile_stage_bytes() {
    return (size_t)4 * T * (8 + M * tile_es<BF16>());
}
// one set of output tiles: theta' in the replica type, and with GV the
// fp32 theta' (bf16 replicas; fp32 replicas share the first tile) and v'
template <bool BF16, int T, bool GV>
__host__ __device__ constexpr size_t tile_out_bytes() {
    return (size_t)4 * T * (tile_es<BF16>() + (GV ? (BF16 ? 8 : 4) : 0));
}
template <int M, bool BF16, int T, int NS, bool GV>
__host__ __device__ constexpr size_t tile_smem() {
    return NS * tile_stage_bytes<M, BF16, T>() + 2 * tile_out_bytes<BF16, T, GV>();
}
template <int M, bool BF16, int T, int NS, bool GV>
__host__ __device__ constexpr bool tile_fit() {
    return tile_smem<M, BF16, T, NS, GV>() + tile_static<M, T>() <= tile_budget<M, BF16, T>();
}
// Shapes measured on GB300 (fraction of the measured copy peak, rounds of
// 1.4e8 - 5e8 parameters):
//   fp32: one 1024-thread CTA per SM, 0.96-0.98 for M = 1 and M = 8
//     against 0.91-0.95 for 256- and 512-thread shapes;
//   bf16 M <= 4: four 256-thread CTAs per SM with one stage, 0.98 against
//     0.95-0.97;
//   bf16 M >= 5: two 512-thread CTAs per SM with one stage, so that the
//     fp32 output tiles fit, 0.97-0.98 against 0.93-0.97.
//   M = 9..16: 512-thread CTAs with one stage (one CTA per SM for fp32,
//     two for bf16); fp32 0.99-1.00 for M = 12..16 against 0.95-0.97 for
//     the register pass, bf16 0.96-0.97 for M = 9..12 against 0.955-0.963.
template <int M, bool BF16>
__host__ __device__ constexpr int tile_threads_table() {
    return M > 8 ? 512 : !BF16 ? 1024 : (M <= 4 ? 256 : 512);
}
// a forced thread count applies where one stage of its blocks fits
template <int M, bool BF16>
__host__ __device__ constexpr int tile_threads() {
    if constexpr (ALOCO_TILE_T != 0) {
        if (tile_fit<M, BF16, ALOCO_TILE_T, 1, false>()) return ALOCO_TILE_T;
    }
    return tile_threads_table<M, BF16>();
}
template <int M, bool BF16, int T>
__host__ __device__ constexpr int tile_stages() {
    if (ALOCO_TILE_NS == 1) return 1;
    const bool two = ALOCO_TILE_NS == 2 || (!BF16 && M <= 8);
    return two && tile_fit<M, BF16, T, 2, false>() ? 2 : 1;
}
template <int M, bool BF16, int T, int NS>
__host__ __device__ constexpr bool tile_gv() {
    return !ALOCO_TILE_NOGV && tile_fit<M, BF16, T, NS, true>();
}

}  // namespace

template <int M, bool BF16, int T, int NS>
__global__ void __launch_bounds__(T, (tile_ctas<M, BF16, T>()))
    sync_tile_kernel(const __grid_constant__ SyncArgs a) {
    constexpr int W = T / 32;
    constexpr int B = 4 * T;  // elements per block
    constexpr int ES = tile_es<BF16>();
    constexpr bool GV = tile_gv<M, BF16, T, NS>();
    constexpr uint32_t kF = B * 4;   // one fp32 array of a block
    constexpr uint32_t kX = B * ES;  // one replica slice
    constexpr uint32_t kStage = 2 * kF + M * kX;
    constexpr uint32_t kOut = (uint32_t)tile_out_bytes<BF16, T, GV>();

    __shared__ double e_w[W][M];
    __shared__ __align__(8) unsigned long long full_bar[NS];
    extern __shared__ __align__(128) unsigned char smem[];

    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    if (lane < M) e_w[warp][lane] = 0.0;
    if (t == 0) {
#pragma unroll
        for (int s = 0; s < NS; ++s) mbar_init(smem_addr(&full_bar[s]), 1);
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

    const int64_t nblk = a.nvec > 0 ? a.n / B : 0;  // whole blocks
    const int64_t G = gridDim.x;
    const int64_t mine = (int64_t)blockIdx.x < nblk ? (nblk - 1 - blockIdx.x) / G + 1 : 0;
    unsigned char *out_base = smem + (size_t)NS * kStage;

    // thread 0: the bulk copies of this CTA's j-th block into stage j % NS
    int64_t skipped = -1;
    auto issue = [&](int64_t j) {
        const int64_t kb = blockIdx.x + j * G;
        if (a.test_stall_tile1 != 0 && kb == a.test_stall_tile1 - 1) {
            skipped = j;  // testing only: this stage never fills
            return;
        }
        unsigned char *st = smem + (size_t)(j % NS) * kStage;
        const uint32_t bar = smem_addr(&full_bar[j % NS]);
        mbar_arrive_expect_tx(bar, kStage);
        bulk_load(smem_addr(st), a.g + kb * B, kF, bar);
        bulk_load(smem_addr(st + kF), a.v + kb * B, kF, bar);
#pragma unroll
        for (int m = 0; m < M; ++m)
            bulk_load(smem_addr(st + 2 * kF + m * kX),
                      reinterpret_cast<const unsigned char *>(a.x[m]) + kb * B * ES, kX, bar);
    };
    // thread 0: block j's output tiles to global memory
    auto store_tiles = [&](int64_t j) {
        const int64_t kb = blockIdx.x + j * G;
        const unsigned char *ob = out_base + (size_t)(j & 1) * kOut;
        if constexpr (GV) {
            const unsigned char *og = BF16 ? ob + kX : ob;
            bulk_store(a.g + kb * B, smem_addr(og), kF);
            bulk_store(a.v + kb * B, smem_addr(og + kF), kF);
        }
#pragma unroll
        for (int m = 0; m < M; ++m)
            bulk_store(reinterpret_cast<unsigned char *>(a.x[m]) + kb * B * ES, smem_addr(ob),
                       kX);
        bulk_commit();
    };

    int64_t issued = 0, consumed = 0;  // thread 0's view
    if (t == 0) {
        issued = mine < NS ? mine : NS;
        for (int64_t j = 0; j < issued; ++j) issue(j);
    }
    bool failed = false;
    for (int64_t j = 0; j < mine; ++j) {
        const int s = (int)(j % NS);
        const unsigned char *st = smem + (size_t)s * kStage;
        const bool ok = mbar_wait(smem_addr(&full_bar[s]), (uint32_t)((j / NS) & 1), nullptr);
        if (t == 0 && ok) consumed = j + 1;

        // 2. this thread's chunks: pseudo-gradients, their sum and energies
        const float4 g4 = *reinterpret_cast<const float4 *>(st + 16 * t);
        const float4 v4 = *reinterpret_cast<const float4 *>(st + kF + 16 * t);
        const float gg[4] = {g4.x, g4.y, g4.z, g4.w};
        const float vv[4] = {v4.x, v4.y, v4.z, v4.w};
        float sm[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int m = 0; m < M; ++m) {
            float xx[4];
            const unsigned char *xp = st + 2 * kF + m * kX + 4 * t * ES;
            if constexpr (BF16) {
                const uint2 w = *reinterpret_cast<const uint2 *>(xp);
                xx[0] = bf16_lo(w.x); xx[1] = bf16_hi(w.x);
                xx[2] = bf16_lo(w.y); xx[3] = bf16_hi(w.y);
            } else {
                const float4 q = *reinterpret_cast<const float4 *>(xp);
                xx[0] = q.x; xx[1] = q.y; xx[2] = q.z; xx[3] = q.w;
            }
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float d = gg[i] - xx[i];
                sm[i] += d;
                e_acc[m] = fmaf(d, d, e_acc[m]);
            }
        }
        // the stores issued after the previous barrier have read their tiles
        if (t == 0) bulk_wait_read();
        // 3. the barrier; a wait that ran out in any thread stops the CTA
        if (__syncthreads_or(!ok)) {
            failed = true;
            break;
        }
        if (t == 0) {
            if (j >= 1) store_tiles(j - 1);
            if (j + NS < mine) {
                issue(j + NS);
                issued = j + NS + 1;
            }
        }

        // 4. the outer step and this block's tiles
        float gp[4], vp[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            b32 = fmaf(sm[i], sm[i], b32);
            outer_step(k, sm[i], gg[i], vv[i], gp[i], vp[i]);
            nf += not_finite(gp[i], vp[i]);
        }
        unsigned char *ob = out_base + (size_t)(j & 1) * kOut;
        const int64_t e = (blockIdx.x + j * G) * B + 4 * t;
        if constexpr (BF16) {
            *reinterpret_cast<uint2 *>(ob + 8 * t) =
                make_uint2(pack_bf16x2(gp[0], gp[1]), pack_bf16x2(gp[2], gp[3]));
            if constexpr (GV) {
                *reinterpret_cast<float4 *>(ob + kX + 16 * t) =
                    make_float4(gp[0], gp[1], gp[2], gp[3]);
                *reinterpret_cast<float4 *>(ob + kX + kF + 16 * t) =
                    make_float4(vp[0], vp[1], vp[2], vp[3]);
            } else {
                stcs4(a.g + e, 0, make_float4(gp[0], gp[1], gp[2], gp[3]));
                stcs4(a.v + e, 0, make_float4(vp[0], vp[1], vp[2], vp[3]));
            }
        } else {
            *reinterpret_cast<float4 *>(ob + 16 * t) = make_float4(gp[0], gp[1], gp[2], gp[3]);
            if constexpr (GV)
                *reinterpret_cast<float4 *>(ob + kF + 16 * t) =
                    make_float4(vp[0], vp[1], vp[2], vp[3]);
            else
                stcs4(a.v + e, 0, make_float4(vp[0], vp[1], vp[2], vp[3]));
            if constexpr (!GV) stcs4(a.g + e, 0, make_float4(gp[0], gp[1], gp[2], gp[3]));
        }
        fence_proxy_async_smem();  // the tiles are read by bulk copies
        if (++since_flush == kTileFlushBlocks) flush();
        b64 += (double)b32;
        b32 = 0.f;
    }
    if (failed) {
        if (t == 0) {
            atomicExch(a.error, 1u);
            // let the loads still in flight land before the CTA exits
            for (int64_t j = consumed; j < issued; ++j)
                if (j != skipped)
                    mbar_wait(smem_addr(&full_bar[j % NS]), (uint32_t)((j / NS) & 1), nullptr);
        }
    } else {
        if (mine > 0) {
            __syncthreads();
            if (t == 0) store_tiles(mine - 1);
        }
        // elements after the last whole block
        for (int64_t jj = nblk * B + (int64_t)blockIdx.x * T + t; jj < a.n; jj += G * T) {
            const float g = a.g[jj];
            const float v = a.v[jj];
            float s = 0.f;
#pragma unroll
            for (int m = 0; m < M; ++m) {
                float x;
                if constexpr (BF16)
                    x = __uint_as_float(
                        (uint32_t)(reinterpret_cast<const uint16_t *>(a.x[m])[jj]) << 16);
                else
                    x = reinterpret_cast<const float *>(a.x[m])[jj];
                const float d = g - x;
                s += d;
                e_acc[m] = fmaf(d, d, e_acc[m]);
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
                    reinterpret_cast<__nv_bfloat16 *>(a.x[m])[jj] = __float2bfloat16_rn(gp);
                else
                    reinterpret_cast<float *>(a.x[m])[jj] = gp;
            }
        }
    }
    if (t == 0) bulk_wait_all();
    flush();
    b64 += (double)b32;
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
cudaError_t tile_launch(const SyncArgs &a, int sm_count, int max_grid, cudaStream_t stream,
                        int *grid_out) {
    constexpr int T = tile_threads<M, BF16>();
    constexpr int NS = tile_stages<M, BF16, T>();
    constexpr bool GV = tile_gv<M, BF16, T, NS>();
    static_assert(tile_fit<M, BF16, T, NS, GV>(), "tile staging exceeds shared memory");
    constexpr size_t smem = tile_smem<M, BF16, T, NS, GV>();
    static PerDevice occ_cache;  // attribute set-up and occupancy, per device
    const int dev = PerDevice::device();
    int occ = occ_cache.get(dev);
    if (occ == 0) {
        cudaError_t e = cudaFuncSetAttribute(sync_tile_kernel<M, BF16, T, NS>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)smem);
        if (e == cudaSuccess)
            e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
                &occ, sync_tile_kernel<M, BF16, T, NS>, T, smem);
        if (e != cudaSuccess) return e;
        if (occ < 1) occ = 1;
        occ_cache.set(dev, occ);
    }
    const int64_t nblk = a.n / (4 * T);
    int64_t grid = (int64_t)sm_count * occ;
    if (grid > nblk) grid = nblk;
    if (grid > max_grid) grid = max_grid;
    if (grid < 1) grid = 1;
    *grid_out = (int)grid;
    sync_tile_kernel<M, BF16, T, NS><<<(unsigned)grid, T, smem, stream>>>(a);
    return cudaGetLastError();
}

template <bool BF16>
cudaError_t tile_dispatch(const SyncArgs &a, int sm_count, int max_grid, cudaStream_t stream,
                          int *grid_out) {
    switch (a.M) {
        case 1: return tile_launch<1, BF16>(a, sm_count, max_grid, stream, grid_out);
        case 2: return tile_launch<2, BF16>(a, sm_count, max_grid, stream, grid_out);
        case 3: return tile_launch<3, BF16>(a, sm_count, max_grid, stream, grid_out);
        case 4: return tile_launch<4, BF16>(a, sm_count, max_grid, stream, grid_out);
        case 5: return tile_launch<5, BF16>(a, sm_count, max_grid, stream, grid_out);
        case 6: return tile_launch<6, BF16>(a, sm_count, max_grid, stream, grid_out);
        case 7: return tile_launch<7, BF16>(a, sm_count, max_grid, stream, grid_out);
        case 8: return tile_launch<8, BF16>(a, sm_count, max_grid, stream, grid_out);
        case 9: return tile_launch<9, BF16>(a, sm_count, max_grid, stream, grid_out);
        case 10: return tile_launch<10, BF16>(a, sm_count, max_grid, stream, grid_out);
        case 11: return tile_launch<11, BF16>(a, sm_count, max_grid, stream, grid_out);
        case 12: return tile_launch<12, BF16>(a, sm_count, max_grid, stream, grid_out);
        case 13: return tile_launch<13, BF16>(a, sm_count, max_grid, stream, grid_out);
        case 14: return tile_launch<14, BF16>(a, sm_count, max_grid, stream, grid_out);
        case 15: return tile_launch<15, BF16>(a, sm_count, max_grid, stream, grid_out);
        default: return tile_launch<16, BF16>(a, sm_count, max_grid, stream, grid_out);
    }
}

}  // namespace

bool sync_tile_fits(int M, int64_t n, int64_t nvec) {
    // at least one whole block of the largest shape (4 x 1024 elements)
    return M >= 1 && M <= kTileMaxM && nvec > 0 && n >= 4096;
}

cudaError_t launch_sync_tile(const SyncArgs &a, aloco_dtype dtype, int sm_count, int max_grid,
                             cudaStream_t stream, int *grid_out) {
    if (!sync_tile_fits(a.M, a.n, a.nvec)) return cudaErrorInvalidValue;
    return dtype == ALOCO_BF16 ? tile_dispatch<true>(a, sm_count, max_grid, stream, grid_out)
                               : tile_dispatch<false>(a, sm_count, max_grid, stream, grid_out);
}

}  // namespace aloco
