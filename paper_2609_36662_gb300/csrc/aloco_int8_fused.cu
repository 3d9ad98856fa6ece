// The INT8-communicated round (App. G.1) in one kernel: every replica is
// read from HBM once, as in the uncompressed round.
//
// CTAs of T threads work through 4096-element codec blocks (grid stride),
// 4096 / T elements per thread in chunks of 4 (chunk c of thread t at
// 4t + c x 4T, so warp accesses to shared memory are contiguous): two
// 512-thread CTAs per SM where they fit (where only the staging of theta
// and v keeps them from fitting, each thread reads its theta and v from
// global memory instead; see direct_gv), else one 1024-thread CTA (see
// fused_threads).  Per block:
//   1. theta, v and the M replica slices arrive in shared memory by bulk
//      copies (cp.async.bulk, one per array, issued by thread 0 and
//      completing on the CTA's mbarrier; every thread's wait on it is
//      bounded).  Short or unaligned blocks (tensor ends) are instead staged
//      by every thread, element by element, into its own slots;
//   2. each warp reduces every worker's max |Delta_m| (as float bits, NaN
//      above +inf); barrier 1; every warp then reads the 32 warp maxima of
//      each worker lane-parallel and folds them with one warp max, and lane
//      m turns worker m's maximum into its scale and reciprocal;
//   3. the workers' pseudo-gradients are encoded, decoded and summed in FP32
//      worker order, reading the replicas again from shared memory;
//   4. the mean is encoded and decoded once (its block maximum is barrier 2).
//      Every thread has then read this block's staging, so thread 0 issues
//      the next block's bulk copies into the same buffer; they overlap the
//      outer step and the stores;
//   5. theta' is written once, in the replica type, to an output tile in
//      shared memory (theta' and v' in fp32 too where they fit), and after
//      the next block's barrier 1 thread 0 stores the tiles with bulk
//      copies: the M replica resets are M copies of one tile.  Before
//      barrier 2 of that block it waits until they have read the tiles.
// Drift energies sum in fp32 per thread over at most 8 blocks (32 squares)
// before each warp adds them, in a fixed order, to its fp64 row.  The
// arithmetic of every element is the split form's (aloco_int8.cu), so both
// forms give the same codes, scales and outputs.
//
// Shared memory per CTA: the input buffer, 4096 x (8 + G x element size)
// bytes for a group of G workers, and the output tiles, 4096 x element size
// (plus 4096 x 8 for the fp32 theta' and v' tiles where they fit; elsewhere
// threads store theta' and v' themselves).  One group holds every worker for
// bf16 and for fp32 up to M = 8; fp32 with 9 <= M <= 16 stages each block's
// replicas in groups of about three workers (see fused_group).
//
// A bounded wait that runs out (about 2 s) sets the round's error word; the
// whole CTA leaves the block loop together at the next barrier, thread 0
// lets the copies it issued land, and the host reports the error.
#include <atomic>

#include "aloco_bulk.cuh"
#include "aloco_int8.cuh"

namespace aloco {

namespace {

constexpr int kFlushBlocks = 8;
constexpr int kFusedMax = 16;

// Shared memory of one SM and the largest a CTA may take (bytes), and the
// part of each CTA's share the system reserves.
constexpr size_t kSmemPerSm = 233472;
constexpr size_t kSmemPerCta = 232448;
constexpr size_t kSmemReserved = 1024;

template <bool BF16>
__host__ __device__ constexpr int esize() { return BF16 ? 2 : 4; }
// Workers whose replica slices are staged at a time (a group), at most
// `cap` per group in groups of near-equal size.
__host__ __device__ constexpr int balanced_group(int M, int cap) {
    return (M + (M + cap - 1) / cap - 1) / ((M + cap - 1) / cap);
}
// All M for M <= 8.  Above, fp32 stages the replicas in groups on two
// 512-thread CTAs per SM: of up to 5 workers with theta and v read directly
// (grouped_direct), else of 3 with theta and v staged (0.84-0.94 of the
// copy peak for M = 9..16 against 0.54-0.60 for groups of 8 on one
// 1024-thread CTA; the split form: 0.66-0.67).  ALOCO_I8_FUSED_G caps the
// group (a tuning knob).
#ifndef ALOCO_I8_FUSED_G
#define ALOCO_I8_FUSED_G 0
#endif
// fp32 with M > 8: theta and v read directly from global memory, which
// leaves room for groups of up to 5 workers on two 512-thread CTAs per SM
// (a 16-worker block in 4 groups instead of 6).  Measured on GB300 (4e8
// parameters, fraction of the copy peak) against groups of 3 with theta and
// v staged: M = 9 0.949 (0.904), M = 12 0.878 (0.867), M = 16 0.869
// (0.808); groups of at most 4 gave 0.865, 0.880 and 0.869.
// ALOCO_I8_GDIRECT sets the group cap (0: groups of 3 with theta and v
// staged; a tuning knob).
#ifndef ALOCO_I8_GDIRECT
#define ALOCO_I8_GDIRECT 5
#endif
template <int M, bool BF16>
__host__ __device__ constexpr bool grouped_direct() {
    return ALOCO_I8_GDIRECT > 0 && !BF16 && M > 8 && ALOCO_I8_FUSED_G == 0;
}
template <int M, bool BF16>
__host__ __device__ constexpr int fused_group() {
    if (ALOCO_I8_FUSED_G) return balanced_group(M, ALOCO_I8_FUSED_G);
    if (M <= 8 || BF16) return M;
    if (grouped_direct<M, BF16>()) return balanced_group(M, ALOCO_I8_GDIRECT);
    return balanced_group(M, 3);
}
// the static shared arrays of the kernel and of the final reduction (an
// upper bound)
template <int M, int T>
__host__ __device__ constexpr size_t static_bytes() {
    return (size_t)(T / 32) * (4 * M + 4 + 8 * M + 8 * (M + 1)) + 4096;
}
// shared memory one of C CTAs per SM may take
template <int C>
__host__ __device__ constexpr size_t cta_budget() {
    return C == 1 ? kSmemPerCta : kSmemPerSm / C - kSmemReserved;
}
// Two 512-thread CTAs per SM with theta and v staged beside the replicas
// (and the replica-type output tile), or with theta and v read by every
// thread straight from global memory instead.
template <int M, bool BF16>
__host__ __device__ constexpr bool fits_two_staged() {
    return (size_t)kI8Block * (8 + fused_group<M, BF16>() * esize<BF16>()) +
               (size_t)kI8Block * esize<BF16>() + static_bytes<M, 512>() <=
           cta_budget<2>();
}
template <int M, bool BF16>
__host__ __device__ constexpr bool fits_two_direct() {
    return (size_t)kI8Block * (fused_group<M, BF16>() * esize<BF16>()) +
               (size_t)kI8Block * esize<BF16>() + static_bytes<M, 512>() <=
           cta_budget<2>();
}
// theta and v are not staged where that alone keeps two CTAs per SM from
// fitting (bf16 M = 9..12, fp32 M = 4, 5), nor for fp32 M = 2, 3: each
// thread loads its own theta (before its wait for the replicas) and v from
// global memory, the same bytes read once, and the shared memory holds the
// replicas only.  Measured on GB300 (4e8 parameters, fraction of the copy
// peak; in brackets with theta and v staged, on one 1024-thread CTA where
// two do not fit): bf16 M = 9 0.860 (0.726), M = 10 0.879 (0.738), M = 12
// 0.835 (0.737); fp32 M = 2 0.979 (0.965), M = 3 0.959 (0.921), M = 4
// 0.939 (0.903), M = 5 0.926 (0.930).  Staging stays faster for fp32 M = 1
// (0.984 against 0.931) and bf16 M <= 8 (M = 8: 0.915 against 0.839).
// bf16 M >= 13 does not fit two CTAs even so (its replicas alone take more
// than half an SM).  ALOCO_I8_DIRECT = 0 turns it off, 2 takes it wherever
// two CTAs fit (tuning knobs).
#ifndef ALOCO_I8_DIRECT
#define ALOCO_I8_DIRECT 1
#endif
template <int M, bool BF16>
__host__ __device__ constexpr bool direct_gv() {
    if (grouped_direct<M, BF16>()) return true;
    return ALOCO_I8_DIRECT && fused_group<M, BF16>() == M && fits_two_direct<M, BF16>() &&
           (ALOCO_I8_DIRECT == 2 || !fits_two_staged<M, BF16>() || (!BF16 && M >= 2));
}
// theta, v (fp32, unless read directly) and one group's replica slices of
// one block
template <int M, bool BF16>
__host__ __device__ constexpr size_t in_bytes() {
    return (size_t)kI8Block *
           ((direct_gv<M, BF16>() ? 0 : 8) + fused_group<M, BF16>() * esize<BF16>());
}
// The fp32 theta' and v' tiles fit beside the input and the replica tile.
template <int M, bool BF16, int T, int C>
__host__ __device__ constexpr bool tile_gv() {
    return in_bytes<M, BF16>() + (size_t)kI8Block * (esize<BF16>() + (BF16 ? 8 : 4)) +
               static_bytes<M, T>() <=
           cta_budget<C>();
}
template <int M, bool BF16, int T, int C>
__host__ __device__ constexpr size_t out_bytes() {
    return tile_gv<M, BF16, T, C>() ? (size_t)kI8Block * (esize<BF16>() + (BF16 ? 8 : 4))
                                    : (size_t)kI8Block * esize<BF16>();
}
template <int M, bool BF16, int T, int C>
__host__ __device__ constexpr size_t fused_smem() {
    return in_bytes<M, BF16>() + out_bytes<M, BF16, T, C>();
}
template <int M, bool BF16, int T, int C>
__host__ __device__ constexpr bool fits() {
    return fused_smem<M, BF16, T, C>() + static_bytes<M, T>() <= cta_budget<C>();
}

// Threads per CTA (T) and elements per thread (4096 / T), measured on
// GB300 (2^26-parameter rounds, fraction of the measured copy peak):
//   bf16: T = 512, two CTAs per SM, 0.85 for M <= 4 and 0.77-0.79 for
//     M = 6, 8, against 0.63-0.67 with one 1024-thread CTA, whose single
//     block in flight leaves the SM idle while the next block's copies land;
//   fp32: T = 512 0.88-0.93 for M <= 3, against 0.70-0.82 with 1024
//     threads; from M = 4 two 512-thread CTAs no longer fit.
// ALOCO_I8_FUSED_T = 512 or 1024 and ALOCO_I8_FUSED_CTAS = 1 or 2 force a
// shape (tuning knobs).
#ifndef ALOCO_I8_FUSED_T
#define ALOCO_I8_FUSED_T 0
#endif
#ifndef ALOCO_I8_FUSED_CTAS
#define ALOCO_I8_FUSED_CTAS 0
#endif
template <int M, bool BF16>
constexpr int fused_threads() {
    if (ALOCO_I8_FUSED_T == 1024) return 1024;
    if (ALOCO_I8_FUSED_T == 512 && ALOCO_I8_FUSED_CTAS == 1) return 512;
    return fits<M, BF16, 512, 2>() ? 512 : 1024;
}
// CTAs per SM the shared memory is planned for (and the register budget:
// 64 registers a thread for 1024 threads per SM, 128 for 512)
template <int M, bool BF16, int T>
__host__ __device__ constexpr int fused_ctas() {
    if (ALOCO_I8_FUSED_CTAS) return ALOCO_I8_FUSED_CTAS;
    return (T == 512 && fits<M, BF16, 512, 2>()) ? 2 : 1;
}

// A thread's replica values of staging slots m0 and m0 + 1 (when m0 + 1 <
// lim, the slots in use),
// widened exactly, as PER / 2 pairs each.  Worker m's slice starts at
// m x 4096 x element size; thread t's chunks of 4 elements sit at 4t + c x 4T.
template <int M, bool BF16, int T>
__device__ __forceinline__ void staged_reps(const unsigned char *sx, int m0, int t,
                                            float2 (&a)[kI8Block / T / 2],
                                            float2 (&b)[kI8Block / T / 2], int lim = M) {
    constexpr int PER = kI8Block / T;
    constexpr int ES = esize<BF16>();
    const unsigned char *p0 = sx + (size_t)m0 * kI8Block * ES + 4 * t * ES;
    const unsigned char *p1 = p0 + kI8Block * ES;
#pragma unroll
    for (int c = 0; c < PER / 4; ++c) {
        const int off = c * 4 * T * ES;
        if constexpr (BF16) {
            const uint2 w = *reinterpret_cast<const uint2 *>(p0 + off);
            a[2 * c] = make_float2(bf16_lo(w.x), bf16_hi(w.x));
            a[2 * c + 1] = make_float2(bf16_lo(w.y), bf16_hi(w.y));
            if (m0 + 1 < lim) {
                const uint2 u = *reinterpret_cast<const uint2 *>(p1 + off);
                b[2 * c] = make_float2(bf16_lo(u.x), bf16_hi(u.x));
                b[2 * c + 1] = make_float2(bf16_lo(u.y), bf16_hi(u.y));
            }
        } else {
            const float4 q = *reinterpret_cast<const float4 *>(p0 + off);
            a[2 * c] = make_float2(q.x, q.y);
            a[2 * c + 1] = make_float2(q.z, q.w);
            if (m0 + 1 < lim) {
                const float4 r = *reinterpret_cast<const float4 *>(p1 + off);
                b[2 * c] = make_float2(r.x, r.y);
                b[2 * c + 1] = make_float2(r.z, r.w);
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

// Fewer instructions per element-worker: the block maxima and the codes'
// half-integer margin taken with three-input maxima, and the exact-quotient
// fallback as a warp-uniform branch, against two-input maxima, a compare per
// element and a per-thread branch.  The decisions are the same either way.
// Measured on GB300 (fraction of the copy peak): bf16 M = 8 0.916 against
// 0.911 (4e8 parameters and the 3B set alike); bf16 M = 16 0.729 against
// 0.741 (24 bytes of register spills appear at 64 registers); fp32 M = 12
// unchanged.  So it is taken for bf16 with M <= 8.  ALOCO_I8_FAST = 0 turns
// it off everywhere (a tuning knob).
#ifndef ALOCO_I8_FAST
#define ALOCO_I8_FAST 1
#endif
template <int M, bool BF16>
__host__ __device__ constexpr bool i8_fast() {
    return ALOCO_I8_FAST && BF16 && M <= 8;
}

// max(a, b, c), ignoring NaN operands (as fmaxf)
__device__ __forceinline__ float max3(float a, float b, float c) {
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}
// max(a, b, c), NaN if any operand is NaN
__device__ __forceinline__ float max3_nan(float a, float b, float c) {
    float r;
    asm("max.NaN.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}
// Codes of a pair from the product y r (as code2_fast), with the distance
// of each product from its nearest integer folded into `far`: the codes are
// the codec's when far < kCodeMargin at the end (a NaN or infinite product
// makes far NaN, which fails that test).
__device__ __forceinline__ float2 code2_fast_max(float2 y, float r, float &far) {
    const float2 t = mul2_rn(y, splat2(r));
    const float2 n = add2_rn(add2_rn(t, splat2(kRoundMagic)), splat2(-kRoundMagic));
    const float2 d = sub2(t, n);  // exact: |t - n| <= 1/2
    far = max3_nan(far, fabsf(d.x), fabsf(d.y));
    return n;
}

}  // namespace

template <int M, bool BF16, int T>
__global__ void __launch_bounds__(T, (fused_ctas<M, BF16, T>()))
    int8_fused_kernel(const __grid_constant__ SyncArgs a,
                      const __grid_constant__ Int8Parts P) {
    constexpr int PER = kI8Block / T;  // elements per thread
    constexpr int NP = PER / 2;        // pairs per thread
    constexpr int W = T / 32;          // warps
    constexpr int ES = esize<BF16>();
    constexpr bool GV = tile_gv<M, BF16, T, fused_ctas<M, BF16, T>()>();
    constexpr int G = fused_group<M, BF16>();    // workers staged at a time
    constexpr int NG = (M + G - 1) / G;          // groups per block
    constexpr bool GROUPED = NG > 1;
    constexpr int EA = GROUPED ? G : M;          // energy accumulators a thread
    constexpr bool DGV = direct_gv<M, BF16>();   // theta, v read from global memory
    constexpr uint32_t kGVBytes = kI8Block * 4;  // one fp32 array of a block
    constexpr uint32_t kXBytes = kI8Block * ES;  // one replica slice
    // Single buffers suffice: red_w is read between a group's first barrier
    // and the next barrier, and rewritten only after it; red1 is read after
    // barrier 2 and rewritten only after the next block's first barrier.
    __shared__ unsigned red_w[G][W];                  // [worker][warp]: conflict-free reads
    __shared__ unsigned red1[W];
    __shared__ double e_w[W][M];
    __shared__ __align__(16) float2 sr[W][G + (G & 1)];  // per warp: (scale, 1/scale)
    __shared__ __align__(8) unsigned long long full_bar;
    extern __shared__ __align__(128) unsigned char smem[];
    float *sg = reinterpret_cast<float *>(smem);  // theta (staged only if !DGV)
    float *sv = sg + kI8Block;                      // v (staged only if !DGV)
    unsigned char *sx = smem + (DGV ? 0 : 2 * kGVBytes);
    unsigned char *ox = sx + G * kXBytes;             // theta' in the replica type
    float *og = BF16 ? reinterpret_cast<float *>(ox + kXBytes)  // theta' (fp32)
                     : reinterpret_cast<float *>(ox);
    float *ov = og + kI8Block;                         // v' (GV only)
    const uint32_t bar = smem_addr(&full_bar);

    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    if (lane < M) e_w[warp][lane] = 0.0;
    if (t == 0) {
        mbar_init(bar, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    // energies: all M workers' over up to 8 blocks, or, with groups, one
    // group's over one block
    float e_acc[EA];
#pragma unroll
    for (int m = 0; m < EA; ++m) e_acc[m] = 0.f;
    int since_flush = 0;
    auto flush_rows = [&](int m0, int n) {
#pragma unroll
        for (int m = 0; m < EA; ++m) {
            if (m >= n) break;
            float e = e_acc[m];
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) e += __shfl_down_sync(0xffffffffu, e, off);
            if (lane == 0) e_w[warp][m0 + m] += (double)e;
            e_acc[m] = 0.f;
        }
    };
    auto flush = [&]() {
        flush_rows(0, EA);
        since_flush = 0;
    };

    float b32 = 0.f;
    double b64 = 0.0;
    unsigned nf = 0;
    const Coef k{a.c_hi, a.c_lo, a.mu_hi, a.mu_lo, a.neg_eta_hi, a.neg_eta_lo};
    const int64_t nblocks = P.blk[P.n_parts];
    // thread t holds the 4-element chunks at 4t + c x 4T (c < PER / 4), so
    // every warp access to a staged array is contiguous
    auto el = [&](int i) { return (i >> 2) * (4 * T) + 4 * t + (i & 3); };
    // a thread's elements of an fp32 array read straight from global memory:
    // 16-byte streaming loads on whole aligned blocks, element loads (0
    // beyond the block's end) otherwise
    auto load_direct = [&](float (&o)[PER], const float *src, int64_t s, int l, bool whole) {
#pragma unroll
        for (int c = 0; c < PER; c += 4) {
            if (whole) {
                const float4 q = __ldcs(reinterpret_cast<const float4 *>(src + s + el(c)));
                o[c] = q.x; o[c + 1] = q.y; o[c + 2] = q.z; o[c + 3] = q.w;
            } else {
#pragma unroll
                for (int i = 0; i < 4; ++i) o[c + i] = el(c + i) < l ? src[s + el(c + i)] : 0.f;
            }
        }
    };

    // whole blocks at 16-byte aligned addresses move by bulk copies
    auto bulk_block = [&](int64_t s, int l) {
        return l == kI8Block && a.nvec > 0 && (s % 8) == 0;
    };
    bool in_flight = false;  // thread 0: bulk loads issued and not yet seen complete
    // thread 0: the bulk copies of group q of the block at s (theta and v
    // come with group 0)
    auto stage_bulk = [&](int64_t kbi, int64_t s, int q) {
        if (q == 0 && a.test_stall_tile1 != 0 && kbi == a.test_stall_tile1 - 1)
            return;  // testing only: this phase never completes
        const int m0 = q * G;
        const int gq = M - m0 < G ? M - m0 : G;
        mbar_arrive_expect_tx(bar, (q == 0 && !DGV ? 2 * kGVBytes : 0) + gq * kXBytes);
        if (q == 0 && !DGV) {
            bulk_load(smem_addr(sg), a.g + s, kGVBytes, bar);
            bulk_load(smem_addr(sv), a.v + s, kGVBytes, bar);
        }
#pragma unroll
        for (int m = 0; m < G; ++m)
            if (m < gq)
                bulk_load(smem_addr(sx + m * kXBytes),
                          reinterpret_cast<const unsigned char *>(a.x[m0 + m]) + s * ES,
                          kXBytes, bar);
        in_flight = true;
    };
    // every thread: its own elements of group q of a short or unaligned block
    auto stage_own = [&](int64_t s, int l, int q) {
        const int m0 = q * G;
        const int gq = M - m0 < G ? M - m0 : G;
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const int e = el(i);
            const bool in = e < l;
            if (q == 0 && !DGV) {
                sg[e] = in ? a.g[s + e] : 0.f;
                sv[e] = in ? a.v[s + e] : 0.f;
            }
#pragma unroll
            for (int m = 0; m < G; ++m) {
                if (m >= gq) break;
                if constexpr (BF16)
                    reinterpret_cast<uint16_t *>(sx + m * kXBytes)[e] =
                        in ? reinterpret_cast<const uint16_t *>(a.x[m0 + m])[s + e]
                           : (uint16_t)0;
                else
                    reinterpret_cast<float *>(sx + m * kXBytes)[e] =
                        in ? reinterpret_cast<const float *>(a.x[m0 + m])[s + e] : 0.f;
            }
        }
        // a later bulk copy may overwrite these bytes
        fence_proxy_async_smem();
    };
    // thread 0: the output tiles of the block at s go to global memory
    auto store_tiles = [&](int64_t s) {
        if constexpr (GV) {
            bulk_store(a.g + s, smem_addr(og), kGVBytes);
            bulk_store(a.v + s, smem_addr(ov), kGVBytes);
        }
#pragma unroll
        for (int m = 0; m < M; ++m)
            bulk_store(reinterpret_cast<unsigned char *>(a.x[m]) + s * ES, smem_addr(ox),
                       kXBytes);
        bulk_commit();
    };

    int64_t kb = blockIdx.x;
    int64_t start = 0;
    int len = 0;
    uint32_t phase = 0;
    bool pend = false;  // the previous block's tiles wait for their bulk stores
    int64_t pstart = 0;
    bool failed = false;
    if (kb < nblocks) {
        locate_block(P, kb, start, len);
        if (!bulk_block(start, len))
            stage_own(start, len, 0);
        else if (t == 0)
            stage_bulk(kb, start, 0);
    }
    for (; kb < nblocks; kb += gridDim.x) {
        const bool full = len == kI8Block;
        const bool bulk = bulk_block(start, len);
        const int64_t nk = kb + gridDim.x;
        int64_t nstart = 0;
        int nlen = 0;
        if (nk < nblocks) locate_block(P, nk, nstart, nlen);
        const bool next_bulk = nk < nblocks && bulk_block(nstart, nlen);
        float g[PER];
        float2 g2[NP];    // theta, as pairs
        float2 sum2[NP];  // the workers' decoded sum
        if constexpr (!GROUPED) {
            if constexpr (DGV) {
                // theta straight from global memory, issued before the wait
                // for the replicas so the two overlap
                load_direct(g, a.g, start, len, bulk);
            }
            bool timed_out = false;
            if (bulk) {
                timed_out = !mbar_wait(bar, phase, nullptr);
                if (t == 0 && !timed_out) in_flight = false;
                phase ^= 1;
            }

            if constexpr (!DGV) {
#pragma unroll
                for (int c = 0; c < PER; c += 4) {
                    const float4 q = *reinterpret_cast<const float4 *>(sg + el(c));
                    g[c] = q.x; g[c + 1] = q.y; g[c + 2] = q.z; g[c + 3] = q.w;
                }
            }
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
                    if constexpr (i8_fast<M, BF16>())
                        mf = max3(mf, fabsf(d[j].x), fabsf(d[j].y));
                    else
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
            // barrier 1; a wait that ran out in any thread stops the whole CTA
            if (__syncthreads_or(timed_out)) {
                failed = true;
                break;
            }
            // every thread wrote its part of the previous block's tiles before
            // the barrier
            if (pend && t == 0) store_tiles(pstart);
            pend = false;
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
#pragma unroll
            for (int j = 0; j < NP; ++j) sum2[j] = splat2(-0.f);
            auto add_worker = [&](float2 scr, const float2 (&x)[NP]) {
                const float s = scr.x, r = scr.y;
                bool ok = true;
                float2 n[NP];
                if constexpr (i8_fast<M, BF16>()) {
                    float far = 0.f;
#pragma unroll
                    for (int j = 0; j < NP; ++j) n[j] = code2_fast_max(sub2(g2[j], x[j]), r, far);
                    // warp-uniform: a lane that needs the exact quotient takes
                    // the whole warp through it (the same codes for the rest)
                    ok = !__any_sync(0xffffffffu, !(far < kCodeMargin));
                } else {
#pragma unroll
                    for (int j = 0; j < NP; ++j) n[j] = code2_fast(sub2(g2[j], x[j]), r, ok);
                }
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

        } else {
            bool stop = false;
            // 2.-3. per group of workers (one group unless fp32 M > 8)
#pragma unroll
            for (int q = 0; q < NG; ++q) {
                const int m0 = q * G;                      // first worker
                const int GQ = M - m0 < G ? M - m0 : G;    // workers in the group
                if (DGV && q == 0) load_direct(g, a.g, start, len, bulk);
                bool timed_out = false;
                if (bulk) {
                    timed_out = !mbar_wait(bar, phase, nullptr);
                    if (t == 0 && !timed_out) in_flight = false;
                    phase ^= 1;
                }
                if (q == 0) {
                    if constexpr (!DGV) {
#pragma unroll
                        for (int c = 0; c < PER; c += 4) {
                            const float4 v4 = *reinterpret_cast<const float4 *>(sg + el(c));
                            g[c] = v4.x; g[c + 1] = v4.y; g[c + 2] = v4.z; g[c + 3] = v4.w;
                        }
                    }
#pragma unroll
                    for (int j = 0; j < NP; ++j) g2[j] = make_float2(g[2 * j], g[2 * j + 1]);
                }

                // 2. block maxima and energies of the group's workers (slot m of
                // the staging holds worker m0 + m)
                auto worker_max = [&](int m, const float2 (&x)[NP]) {
                    float2 d[NP];
#pragma unroll
                    for (int j = 0; j < NP; ++j) d[j] = sub2(g2[j], x[j]);
                    float mf = 0.f;
                    float2 e2 = __fmul2_rn(d[0], d[0]);
#pragma unroll
                    for (int j = 0; j < NP; ++j) {
                        if constexpr (i8_fast<M, BF16>())
                            mf = max3(mf, fabsf(d[j].x), fabsf(d[j].y));
                        else
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
                for (int m = 0; m < G; m += 2) {
                    if (m >= GQ) break;
                    float2 xa[NP], xb[NP];
                    staged_reps<G, BF16, T>(sx, m, t, xa, xb, GQ);
                    worker_max(m, xa);
                    if (m + 1 < GQ) worker_max(m + 1, xb);
                }
                if constexpr (GROUPED)
                    flush_rows(m0, GQ);
                else if (++since_flush == kFlushBlocks)
                    flush();
                // barrier 1 (of the group); a wait that ran out in any thread
                // stops the whole CTA
                if (__syncthreads_or(timed_out)) {
                    stop = true;
                    break;
                }
                if (q == 0) {
                    // every thread wrote its part of the previous block's tiles
                    // before the barrier
                    if (pend && t == 0) store_tiles(pstart);
                    pend = false;
                }
                {
                    // every warp folds the W warp maxima of each worker (lane w
                    // reads warp w's); lane m keeps worker m's and writes its
                    // scale and reciprocal to this warp's table
                    unsigned mine = 0;
#pragma unroll
                    for (int m = 0; m < G; ++m) {
                        if (m >= GQ) break;
                        const unsigned w =
                            __reduce_max_sync(0xffffffffu, lane < W ? red_w[m][lane] : 0u);
                        mine = lane == m ? w : mine;
                    }
                    if (lane < GQ) {
                        const float sc = codec_scale(__uint_as_float(mine));
                        sr[warp][lane] = make_float2(sc, __frcp_rn(sc));
                    }
                    __syncwarp();
                }

                // 3. encode, decode and sum in worker order
                if (q == 0) {
#pragma unroll
                    for (int j = 0; j < NP; ++j) sum2[j] = splat2(-0.f);
                }
                auto add_worker = [&](float2 scr, const float2 (&x)[NP]) {
                    const float sc = scr.x, r = scr.y;
                    bool ok = true;
                    float2 n[NP];
                    if constexpr (i8_fast<M, BF16>()) {
                        float far = 0.f;
#pragma unroll
                        for (int j = 0; j < NP; ++j)
                            n[j] = code2_fast_max(sub2(g2[j], x[j]), r, far);
                        ok = !__any_sync(0xffffffffu, !(far < kCodeMargin));
                    } else {
#pragma unroll
                        for (int j = 0; j < NP; ++j) n[j] = code2_fast(sub2(g2[j], x[j]), r, ok);
                    }
                    if (!ok) {
#pragma unroll
                        for (int j = 0; j < NP; ++j) {
                            const float2 d = sub2(g2[j], x[j]);
                            n[j] = make_float2(codec_code_f(d.x, sc, r), codec_code_f(d.y, sc, r));
                        }
                    }
                    // paired products, scalar sums (see mul2_rn)
#pragma unroll
                    for (int j = 0; j < NP; ++j) {
                        const float2 qq = mul2_rn(n[j], splat2(sc));
                        sum2[j] = make_float2(__fadd_rn(sum2[j].x, qq.x), __fadd_rn(sum2[j].y, qq.y));
                    }
                };
#pragma unroll
                for (int m = 0; m < G; m += 2) {
                    if (m >= GQ) break;
                    const float4 scr = *reinterpret_cast<const float4 *>(&sr[warp][m]);
                    float2 xa[NP], xb[NP];
                    staged_reps<G, BF16, T>(sx, m, t, xa, xb, GQ);
                    add_worker(make_float2(scr.x, scr.y), xa);
                    if (m + 1 < GQ) add_worker(make_float2(scr.z, scr.w), xb);
                }
                if (q + 1 < NG) {
                    // every thread has read this group's slots and scales: the
                    // next group of the same block goes into them
                    __syncthreads();
                    if (bulk) {
                        if (t == 0) stage_bulk(kb, start, q + 1);
                    } else {
                        stage_own(start, len, q + 1);
                    }
                }
            }
            if (stop) {
                failed = true;
                break;
            }

        }
        // 4. the mean's codec
        float v[PER];
        if constexpr (DGV) {
            load_direct(v, a.v, start, len, bulk);
        } else {
#pragma unroll
            for (int c = 0; c < PER; c += 4) {
                const float4 q = *reinterpret_cast<const float4 *>(sv + el(c));
                v[c] = q.x; v[c + 1] = q.y; v[c + 2] = q.z; v[c + 3] = q.w;
            }
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
        // the previous block's bulk stores have read the tiles before any
        // thread passes barrier 2 and rewrites them
        if (t == 0) bulk_wait_read();
        // barrier 2; elements beyond a short block hold 0 and do not move
        // the maximum
        const float s = codec_scale(block_amax<PER, W>(sum, red1));
        // every thread has read this block's staging: the next block's bulk
        // copies go into the same buffer while the rest of this block runs
        // (a short or unaligned next block is staged after the stores)
        if (next_bulk && t == 0) stage_bulk(nk, nstart, 0);
        const float rs = __frcp_rn(s);
        float gp[PER], vp[PER];
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            const float dq = __fmul_rn(codec_code_fast(sum[i], s, rs), s);
            const bool in = full || el(i) < len;
            if (in) b32 = fmaf(dq, dq, b32);
            outer_step(k, dq, g[i], v[i], gp[i], vp[i]);
            if (in) nf += not_finite(gp[i], vp[i]);
        }

        // 5. the stores
        if (bulk) {
#pragma unroll
            for (int c = 0; c < PER; c += 4) {
                if constexpr (BF16) {
                    *reinterpret_cast<uint2 *>(ox + el(c) * 2) =
                        make_uint2(pack_bf16x2(gp[c], gp[c + 1]), pack_bf16x2(gp[c + 2], gp[c + 3]));
                }
                if constexpr (GV || !BF16)
                    *reinterpret_cast<float4 *>(og + el(c)) =
                        make_float4(gp[c], gp[c + 1], gp[c + 2], gp[c + 3]);
                if constexpr (GV)
                    *reinterpret_cast<float4 *>(ov + el(c)) =
                        make_float4(vp[c], vp[c + 1], vp[c + 2], vp[c + 3]);
                if constexpr (!GV) {
                    __stcs(reinterpret_cast<float4 *>(a.g + start + el(c)),
                           make_float4(gp[c], gp[c + 1], gp[c + 2], gp[c + 3]));
                    __stcs(reinterpret_cast<float4 *>(a.v + start + el(c)),
                           make_float4(vp[c], vp[c + 1], vp[c + 2], vp[c + 3]));
                }
            }
            fence_proxy_async_smem();  // the tiles are read by bulk copies
            pend = true;
            pstart = start;
        } else {
#pragma unroll
            for (int i = 0; i < PER; ++i) {
                const int e = el(i);
                if (e >= len) continue;
                a.g[start + e] = gp[i];
                a.v[start + e] = vp[i];
#pragma unroll
                for (int m = 0; m < M; ++m) {
                    if constexpr (BF16)
                        reinterpret_cast<__nv_bfloat16 *>(a.x[m])[start + e] =
                            __float2bfloat16_rn(gp[i]);
                    else
                        reinterpret_cast<float *>(a.x[m])[start + e] = gp[i];
                }
            }
        }
        b64 += (double)b32;  // at most PER terms per thread and block
        b32 = 0.f;
        if (nk < nblocks && !next_bulk) stage_own(nstart, nlen, 0);

        start = nstart;
        len = nlen;
    }
    if (failed) {
        if (t == 0) {
            atomicExch(a.error, 1u);
            // let the loads still in flight land before the CTA exits
            if (in_flight) mbar_wait(bar, phase ^ 1, nullptr);
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

template <int M, bool BF16>
cudaError_t fused_launch(const SyncArgs &a, const Int8Parts &P, int sm_count,
                         int max_grid, cudaStream_t stream, int *grid_out) {
    constexpr int T = fused_threads<M, BF16>();
    constexpr int C = fused_ctas<M, BF16, T>();
    static_assert(fits<M, BF16, T, C>(), "fused INT8 staging exceeds shared memory");
    constexpr size_t smem = fused_smem<M, BF16, T, C>();
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
        case 8: return fused_launch<8, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        case 9: return fused_launch<9, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        case 10: return fused_launch<10, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        case 11: return fused_launch<11, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        case 12: return fused_launch<12, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        case 13: return fused_launch<13, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        case 14: return fused_launch<14, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        case 15: return fused_launch<15, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        case 16: return fused_launch<16, BF16>(a, P, sm_count, max_grid, stream, grid_out);
        default: break;
    }
    return cudaErrorInvalidValue;
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
