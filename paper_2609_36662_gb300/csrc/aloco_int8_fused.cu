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
//   0. thread 0 locates the next block and, for some shapes, leaves its
//      place in shared memory for every thread (see ALOCO_I8_NEXT_SMEM);
//      where bf16 runs one CTA per SM it also asks L2 to fetch the next
//      block's arrays (see ALOCO_I8_PREFETCH);
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
//   4. the mean (the sum over M: a product where M is a power of two) is
//      encoded and decoded once on pairs (its block maximum is barrier 2).
//      Every thread has then read this block's staging, so thread 0 issues
//      the next block's bulk copies into the same buffer; they overlap the
//      outer step and the stores;
//   5. the outer step runs on pairs, 4 elements at a time, and theta' is
//      written once, in the replica type, to an output tile in shared
//      memory (theta' and v' in fp32 too where they fit); after the next
//      block's barrier 1 thread 0 stores the tiles with bulk copies: the M
//      replica resets are M copies of one tile.  Before barrier 2 of that
//      block it waits until they have read the tiles.
// Drift energies: for bf16 with more than 8 workers and fp32 with 2 or 3,
// each block's energies are summed across the warp at once (recursive
// halving) into fp64 rows; elsewhere fp32 accumulators over up to 8 blocks
// (at most 64 squares a thread) are reduced worker by worker, in a fixed
// order (see ALOCO_I8_EROW).  The squared
// decoded means take the second route in every shape.  The arithmetic of
// every element is the split form's (aloco_int8.cu): the paired operations
// round each lane as the scalar ones do, so both forms give the same codes,
// scales and outputs.
//
// Shared memory per CTA: the input buffer, 4096 x (8 + G x element size)
// bytes for a group of G workers, and the output tiles, 4096 x element size
// (plus 4096 x 8 for the fp32 theta' and v' tiles where they fit; elsewhere
// threads store theta' and v' themselves).  One group holds every worker for
// bf16 and for fp32 up to M = 8; fp32 with 9 <= M <= 16 stages each block's
// replicas in groups of at most five workers (see fused_group).
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

// A hint to bring `bytes` (multiple of 16, 16-byte aligned address) of
// global memory into L2 under the cache policy `pol` (createpolicy); nothing
// waits for it and nothing is written.
__device__ __forceinline__ void bulk_prefetch_l2_hint(const void *src, uint32_t bytes,
                                                      uint64_t pol) {
    asm volatile("cp.async.bulk.prefetch.L2.global.L2::cache_hint [%0], %1, %2;" ::"l"(src),
                 "r"(bytes), "l"(pol)
                 : "memory");
}
// A bulk load (as bulk_load) with an L2 cache policy
__device__ __forceinline__ void bulk_load_hint(uint32_t dst, const void *src, uint32_t bytes,
                                               uint32_t bar, uint64_t pol) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint "
        "[%0], [%1], %2, [%3], %4;" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(bar), "l"(pol)
        : "memory");
}
// A bulk store (as bulk_store) with an L2 cache policy
__device__ __forceinline__ void bulk_store_hint(void *dst, uint32_t src, uint32_t bytes,
                                                uint64_t pol) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group.L2::cache_hint [%0], [%1], %2, %3;" ::"l"(dst),
                 "r"(src), "r"(bytes), "l"(pol)
                 : "memory");
}
__device__ __forceinline__ uint64_t policy_evict_last() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}
__device__ __forceinline__ uint64_t policy_evict_first() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

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
// The static shared arrays of the kernel and of the final reduction, per
// warp: the group's warp maxima (4 G), the mean's (4), the energy rows
// (8 (M + 1)), the scale table (8 (G + 1)), the reduction's rows (8 (M + 1))
// and non-finite counts (8); plus 256 bytes for the mbarrier and scalars.
// An upper bound of what ptxas reports for every instantiation.
template <int M, bool BF16, int T>
__host__ __device__ constexpr size_t static_bytes() {
    return (size_t)(T / 32) *
               (4 * fused_group<M, BF16>() + 4 + 8 * (M + 1) +
                8 * (fused_group<M, BF16>() + (fused_group<M, BF16>() & 1)) + 8 * (M + 1) + 8) +
           256;
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
               (size_t)kI8Block * esize<BF16>() + static_bytes<M, BF16, 512>() <=
           cta_budget<2>();
}
template <int M, bool BF16>
__host__ __device__ constexpr bool fits_two_direct() {
    return (size_t)kI8Block * (fused_group<M, BF16>() * esize<BF16>()) +
               (size_t)kI8Block * esize<BF16>() + static_bytes<M, BF16, 512>() <=
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
// (0.984 against 0.931) and bf16 M <= 8 (M = 8: 0.915 against 0.839) except
// bf16 M = 5: measured again with the current kernel, direct loads gave bf16
// M = 5 0.953 (0.937) and lost at M = 1..4 and 6..8 (0.83-0.96 against
// 0.94-0.98), so bf16 M = 5 takes them too.
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
           (ALOCO_I8_DIRECT == 2 || !fits_two_staged<M, BF16>() || (!BF16 && M >= 2) ||
            (BF16 && M == 5));
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
               static_bytes<M, BF16, T>() <=
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
    return fused_smem<M, BF16, T, C>() + static_bytes<M, BF16, T>() <= cta_budget<C>();
}

// Blocks ahead whose arrays thread 0 asks L2 to fetch (cp.async.bulk
// .prefetch.L2) as each block starts, so that the bulk copy of the next block
// into shared memory, issued at barrier 2, reads L2 instead of HBM.  With
// one CTA per SM nothing else runs while that copy lands.  The prefetch
// marks its lines evict-last, and the copies that read a block into shared
// memory and the bulk stores mark theirs evict-first (each is used once), so
// prefetched lines stay until their copy: DRAM reads 1.016x the algorithmic
// bytes on 2^26 x 16 bf16, against 1.225x with no policies.  Measured on
// GB300 (4e8 parameters, fraction of the copy peak), one block ahead against
// none: bf16 M = 16 0.933 (0.846), M = 13 0.928 (0.818); M = 14 0.922, M = 15
// 0.925; without the policies 0.894 and 0.895 (M = 16, 13), with only the
// evict-last prefetch 0.902 and 0.899, with evict-first loads but plain
// stores 0.920 and 0.916; evict-first loads and stores on every shape lost
// 2-3 % on the shapes without prefetch.  The prefetch (before the policies)
// lost on fp32 with one CTA per SM (M = 8 0.83 against 0.99, M = 6 0.91
// against 0.95, the 150M set 0.83 against 0.95) and with two CTAs per SM
// (bf16 M = 8 0.78 against 0.95, M = 12 0.72 against 0.86, fp32 M = 16 0.65
// against 0.93); two blocks ahead lost everywhere.  -1 (default): one block
// ahead where bf16 runs one CTA per SM, none elsewhere; otherwise the
// number of blocks ahead everywhere (tuning knobs).
#ifndef ALOCO_I8_PREFETCH
#define ALOCO_I8_PREFETCH -1
#endif

// Where the next block is located: thread 0 locates it as a block starts
// and leaves it in shared memory for every thread, so the next block's
// copies go out at barrier 2 without a search before them; or thread 0
// searches at barrier 2 and every thread at the end of the block.  On flat
// vectors both cost a few instructions; which is faster depends on the code
// ptxas makes of the rest.  Measured on GB300 over every shape (fraction of
// the copy peak, shared memory against searching): the 150M set (fp32 M = 8,
// one CTA per SM, 111 tensor parts) 0.954 (0.926); bf16 M = 9 0.959 (0.896),
// M = 10 0.953 (0.886), M = 11 0.937 (0.862), M = 12 0.924 (0.918), M = 13..16
// within 0.7 %; searching: bf16 M = 6 0.946 (0.899), fp32 M = 12 0.942
// (0.884), M = 16 0.934 (0.898), M = 3 0.942 (0.930), the 3B set (bf16 M = 8)
// 0.957 (0.947), the 1B set 0.982 (0.977); the other shapes within 0.5 %.
// So shared memory where one CTA runs per SM and for bf16 with M > 8.
// ALOCO_I8_NEXT_SMEM = 0 or 1 forces either everywhere (tuning knobs).
#ifndef ALOCO_I8_NEXT_SMEM
#define ALOCO_I8_NEXT_SMEM 2
#endif

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
// bf16 on one CTA per SM (M >= 13): the shapes where the L2 prefetch and
// the mixed-precision subtraction measured faster
template <int M, bool BF16, int T>
__host__ __device__ constexpr bool bf16_one_cta() {
    return BF16 && fused_ctas<M, BF16, T>() == 1;
}

// bf16 replicas may enter theta - x through the mixed-precision FMA (bf16
// operands, fp32 addend and result): fl(theta - x) in one instruction per
// element from the staged word, with no separate widening; otherwise each
// pair is widened and subtracted with the paired FMA.  Both round every
// element the same way.  Measured on GB300 (4e8 parameters, fraction of the
// copy peak) against widened pairs: bf16 M = 9 0.956 (0.942), M = 10 0.953
// (0.920), M = 11 0.935 (0.900), M = 12 0.923 (0.881), M = 16 0.894 (0.863);
// M = 6 0.956 (0.944); M = 8 0.865 (0.952), M = 5 0.863 (0.937), M = 7 0.866
// (0.961).  ALOCO_I8_MIXED = 0 never takes it, 1 always (for bf16), 2
// (default) for bf16 with M > 8 or M = 6 (tuning knobs).
#ifndef ALOCO_I8_MIXED
#define ALOCO_I8_MIXED 2
#endif
// A pair of replica values as held between the staging and the
// subtraction: a word of two bf16 values (RAW), or two fp32 values.
template <bool RAW>
using RepPair = typename std::conditional<RAW, uint32_t, float2>::type;

// fl(theta - x) of a pair
__device__ __forceinline__ float2 dpair(float2 g, float2 x) { return sub2(g, x); }
__device__ __forceinline__ float2 dpair(float2 g, uint32_t w) {
    // x (-1) + theta, one rounding per element: the rounding of sub2's lanes
    float2 d;
    asm("{\n\t.reg .b16 lo, hi, m1;\n\t"
        "mov.b32 {lo, hi}, %2;\n\t"
        "mov.b16 m1, 0xBF80;\n\t"
        "fma.rn.f32.bf16 %0, lo, m1, %3;\n\t"
        "fma.rn.f32.bf16 %1, hi, m1, %4;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "r"(w), "f"(g.x), "f"(g.y));
    return d;
}

// A thread's replica pairs of staging slots m0 and m0 + 1 (when m0 + 1 <
// lim, the slots in use), PER / 2 pairs each.  Worker m's slice starts at
// m x 4096 x element size; thread t's chunks of 4 elements sit at 4t + c x 4T.
template <int M, bool BF16, int T, bool RAW>
__device__ __forceinline__ void staged_reps(const unsigned char *sx, int m0, int t,
                                            RepPair<RAW> (&a)[kI8Block / T / 2],
                                            RepPair<RAW> (&b)[kI8Block / T / 2], int lim = M) {
    static_assert(BF16 || !RAW, "raw words hold bf16 pairs");
    constexpr int PER = kI8Block / T;
    constexpr int ES = esize<BF16>();
    const unsigned char *p0 = sx + (size_t)m0 * kI8Block * ES + 4 * t * ES;
    const unsigned char *p1 = p0 + kI8Block * ES;
#pragma unroll
    for (int c = 0; c < PER / 4; ++c) {
        const int off = c * 4 * T * ES;
        if constexpr (BF16) {
            const uint2 w = *reinterpret_cast<const uint2 *>(p0 + off);
            const uint2 u = m0 + 1 < lim ? *reinterpret_cast<const uint2 *>(p1 + off)
                                         : make_uint2(0u, 0u);
            if constexpr (RAW) {
                a[2 * c] = w.x;
                a[2 * c + 1] = w.y;
                b[2 * c] = u.x;
                b[2 * c + 1] = u.y;
            } else {
                a[2 * c] = make_float2(bf16_lo(w.x), bf16_hi(w.x));
                a[2 * c + 1] = make_float2(bf16_lo(w.y), bf16_hi(w.y));
                if (m0 + 1 < lim) {
                    b[2 * c] = make_float2(bf16_lo(u.x), bf16_hi(u.x));
                    b[2 * c + 1] = make_float2(bf16_lo(u.y), bf16_hi(u.y));
                }
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
// it off everywhere, 2 takes it everywhere (a tuning knob).
#ifndef ALOCO_I8_FAST
#define ALOCO_I8_FAST 1
#endif
template <int M, bool BF16>
__host__ __device__ constexpr bool i8_fast() {
    return ALOCO_I8_FAST == 2 || (ALOCO_I8_FAST && BF16 && M <= 8);
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

// Block-wide max |y| of a thread's pairs, as float bits: each warp's
// maximum goes to red[warp]; after the barrier every warp folds the W values
// with one warp max.  A NaN wins (the NaN-propagating maximum gives the
// canonical NaN, whose bits exceed +inf's), as in block_amax.
template <int NP, int W>
__device__ __forceinline__ float block_amax2(const float2 (&y)[NP], unsigned *red) {
    float mf = 0.f;
#pragma unroll
    for (int j = 0; j < NP; ++j) mf = max3_nan(mf, fabsf(y[j].x), fabsf(y[j].y));
    const unsigned m = __reduce_max_sync(0xffffffffu, __float_as_uint(mf));
    const int lane = threadIdx.x & 31;
    if (lane == 0) red[threadIdx.x >> 5] = m;
    __syncthreads();
    return __uint_as_float(__reduce_max_sync(0xffffffffu, lane < W ? red[lane] : 0u));
}

// fl32(sum / M) of every pair, the quotient div_by_scale gives.  For M a
// power of two the quotient is the product with 1/M (exact): both round the
// same real number, so they agree, underflow included.  Otherwise the
// Markstein steps of div_by_scale run on pairs, and a thread with a
// non-finite quotient redoes its elements with div_by_scale itself.
template <int M, int NP>
__device__ __forceinline__ void mean_of_sum(const float2 (&sum)[NP], float2 (&mean)[NP]) {
    if constexpr ((M & (M - 1)) == 0) {
#pragma unroll
        for (int j = 0; j < NP; ++j) mean[j] = mul2_rn(sum[j], splat2(1.f / (float)M));
    } else {
        const float fM = (float)M, rM = __frcp_rn(fM);
        float bad = 0.f;
#pragma unroll
        for (int j = 0; j < NP; ++j) {
            const float2 q0 = mul2_rn(sum[j], splat2(rM));
            const float2 q1 =
                __ffma2_rn(__ffma2_rn(splat2(-fM), q0, sum[j]), splat2(rM), q0);
            mean[j] = __ffma2_rn(__ffma2_rn(splat2(-fM), q1, sum[j]), splat2(rM), q1);
            bad = max3_nan(bad, fabsf(mean[j].x), fabsf(mean[j].y));
        }
        if (!(bad <= FLT_MAX)) {
#pragma unroll
            for (int j = 0; j < NP; ++j)
                mean[j] = make_float2(div_by_scale(sum[j].x, fM, rM),
                                      div_by_scale(sum[j].y, fM, rM));
        }
    }
}

// Decoded codes fl32(code(y) s) of a thread's pairs under the block's own
// scale s (r = fl32(1/s)): the product path of code2_fast_max, and a warp
// whose products are not all provably the quotient's takes every element
// through codec_code_f (codec_code_fast's slow path); the other lanes'
// codes do not change.  Every finite product is below 127.5 here (see
// code2_fast), so no clipping is needed on the product path.
template <int NP>
__device__ __forceinline__ void decode_mean(const float2 (&y)[NP], float s, float r,
                                            float2 (&dq)[NP]) {
    float2 n[NP];
    float far = 0.f;
#pragma unroll
    for (int j = 0; j < NP; ++j) n[j] = code2_fast_max(y[j], r, far);
    if (__any_sync(0xffffffffu, !(far < kCodeMargin))) {
#pragma unroll
        for (int j = 0; j < NP; ++j)
            n[j] = make_float2(codec_code_f(y[j].x, s, r), codec_code_f(y[j].y, s, r));
    }
#pragma unroll
    for (int j = 0; j < NP; ++j) dq[j] = mul2_rn(n[j], splat2(s));
}

// outer_step on a pair: the same operations, each lane rounded as the
// scalar step rounds it.
__device__ __forceinline__ void outer_step2(const Coef &k, float2 s, float2 g, float2 v,
                                            float2 &gp, float2 &vp) {
    const float2 dt = __ffma2_rn(s, splat2(k.c_hi), __fmul2_rn(s, splat2(k.c_lo)));
    vp = __ffma2_rn(splat2(k.mu_hi), v, __ffma2_rn(splat2(k.mu_lo), v, dt));
    const float2 d = __ffma2_rn(splat2(k.mu_hi), vp, __ffma2_rn(splat2(k.mu_lo), vp, dt));
    gp = add2_rn(g, __ffma2_rn(splat2(k.ne_hi), d, __fmul2_rn(splat2(k.ne_lo), d)));
}

// Warp sums of the P values each lane holds (P a power of two, at most 32)
// by recursive halving: at each step a lane keeps the half of its values
// that its lane bit selects and adds the partner's copy of that half; the
// last steps add across the lanes that share a value.  Lane L returns the
// warp sum of value L >> (5 - log2 P).  The order is fixed (and a + b = b + a
// exactly), so every lane holding a value has the same bits.
template <int P>
__device__ __forceinline__ float warp_sum_scatter(float (&v)[P]) {
    static_assert(P >= 1 && P <= 32 && (P & (P - 1)) == 0, "P: a power of two");
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int st = 0; st < 5; ++st) {
        const int mask = 16 >> st;
        const int n = P >> st;  // values still held
        if (n > 1) {
            const bool up = (lane & mask) != 0;
#pragma unroll
            for (int i = 0; i < n / 2; ++i) {
                const float send = up ? v[i] : v[i + n / 2];
                const float keep = up ? v[i + n / 2] : v[i];
                v[i] = keep + __shfl_xor_sync(0xffffffffu, send, mask);
            }
        } else {
            v[0] += __shfl_xor_sync(0xffffffffu, v[0], mask);
        }
    }
    return v[0];
}
__host__ __device__ constexpr int pow2_at_least(int n) {
    return n <= 1 ? 1 : 2 * pow2_at_least((n + 1) / 2);
}

// The workers' energies of a block summed across the warp at once (warp
// sums by recursive halving, one fp64 row update per worker and block), so
// no per-worker accumulator stays live through the rest of the block.
// Measured on GB300 (4e8 parameters, fraction of the copy peak) against fp32
// accumulators over up to 8 blocks reduced worker by worker: bf16 M = 16
// 0.832 (0.744), M = 12 0.888 (0.861), M = 8 0.947 (0.953); fp32 M = 16
// (groups, whose energies are reduced per group and block anyway) 0.931
// (0.932); fp32 M = 3 0.958 (0.942), M = 2 0.975 (0.968), bf16 M = 5, 6, 7
// 0.917, 0.937, 0.937 (0.937, 0.944, 0.961).  Taken for bf16 with M > 8 and
// fp32 with M = 2, 3.  ALOCO_I8_EROW = 0 turns it off, 1 takes it for every
// single-group shape (tuning knobs).
#ifndef ALOCO_I8_EROW
#define ALOCO_I8_EROW 2
#endif
template <int M, bool BF16>
__host__ __device__ constexpr bool erow() {
    return ALOCO_I8_EROW == 1 ||
           (ALOCO_I8_EROW == 2 && (BF16 ? M > 8 : (M == 2 || M == 3)));
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
    // blocks between the warp reductions of the fp32 accumulators: at most
    // 64 squares a thread
    constexpr int kFlush = kFlushBlocks;
    constexpr bool GV = tile_gv<M, BF16, T, fused_ctas<M, BF16, T>()>();
    constexpr int G = fused_group<M, BF16>();    // workers staged at a time
    constexpr int NG = (M + G - 1) / G;          // groups per block
    constexpr bool GROUPED = NG > 1;
    constexpr int EA = GROUPED ? G : M;          // energy accumulators a thread
    constexpr bool DGV = direct_gv<M, BF16>();   // theta, v read from global memory
    constexpr bool EROW = !GROUPED && erow<M, BF16>();  // energies reduced every block
    constexpr int PF = ALOCO_I8_PREFETCH >= 0 ? ALOCO_I8_PREFETCH
                                              : (bf16_one_cta<M, BF16, T>() ? 1 : 0);
    constexpr bool NEXT_SMEM =
        ALOCO_I8_NEXT_SMEM == 1 ||
        (ALOCO_I8_NEXT_SMEM == 2 && (fused_ctas<M, BF16, T>() == 1 || (BF16 && M > 8)));
    // bf16 pairs reach the subtraction as raw words (see ALOCO_I8_MIXED)
    constexpr bool MIX =
        BF16 && (ALOCO_I8_MIXED == 1 || (ALOCO_I8_MIXED == 2 && (M > 8 || M == 6)));
    constexpr uint32_t kGVBytes = kI8Block * 4;  // one fp32 array of a block
    constexpr uint32_t kXBytes = kI8Block * ES;  // one replica slice
    // Single buffers suffice: red_w is read between a group's first barrier
    // and the next barrier, and rewritten only after it; red1 is read after
    // barrier 2 and rewritten only after the next block's first barrier.
    __shared__ unsigned red_w[G][W];                  // [worker][warp]: conflict-free reads
    __shared__ unsigned red1[W];
    __shared__ double e_w[W][M + 1];   // [warp][worker energies, then sum Dbar^2]
    __shared__ int64_t s_pstart;        // thread 0: start of the block whose tiles wait
    // the next block's start and length, located by thread 0 as a block
    // starts and read by every thread after barrier 1 (two slots by the
    // parity of the iteration: a slot is rewritten only after every thread
    // has passed the next barrier 1)
    __shared__ int64_t s_nstart[2];
    __shared__ int s_nlen[2];
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
    if (lane <= M) e_w[warp][lane] = 0.0;
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
    float b32 = 0.f;  // sum of squared decoded means since the last flush
    auto flush_b = [&]() {
        float e = b32;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) e += __shfl_down_sync(0xffffffffu, e, off);
        if (lane == 0) e_w[warp][M] += (double)e;
        b32 = 0.f;
    };
    // energies of one block, all M workers: warp sums by recursive halving
    // into the fp64 rows
    constexpr int EP = pow2_at_least(M);
    auto add_rows = [&](float (&eb)[EP]) {
        const float e = warp_sum_scatter<EP>(eb);
        const int w = lane >> (5 - __builtin_ctz(EP));  // the row this lane holds
        if ((lane & (32 / EP - 1)) == 0 && w < M) e_w[warp][w] += (double)e;
    };
    auto flush = [&]() {
        if constexpr (!GROUPED && !EROW) flush_rows(0, EA);
        flush_b();
        since_flush = 0;
    };

    unsigned nf = 0;
    const Coef k{a.c_hi, a.c_lo, a.mu_hi, a.mu_lo, a.neg_eta_hi, a.neg_eta_lo};
    const int nblocks = (int)P.blk[P.n_parts];  // below 2^31 - grid (host check)
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
        if constexpr (PF > 0) {
            // read once: evict these lines first, ahead of the prefetched ones
            const uint64_t pol = policy_evict_first();
            if (q == 0 && !DGV) {
                bulk_load_hint(smem_addr(sg), a.g + s, kGVBytes, bar, pol);
                bulk_load_hint(smem_addr(sv), a.v + s, kGVBytes, bar, pol);
            }
#pragma unroll
            for (int m = 0; m < G; ++m)
                if (m < gq)
                    bulk_load_hint(smem_addr(sx + m * kXBytes),
                                   reinterpret_cast<const unsigned char *>(a.x[m0 + m]) + s * ES,
                                   kXBytes, bar, pol);
        } else {
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
        }
        in_flight = true;
    };
    // thread 0: the L2 prefetch of every array of the block kbi (whole,
    // aligned blocks only)
    auto prefetch_block = [&](int64_t kbi) {
        if (kbi >= nblocks) return;
        int64_t ps;
        int pl;
        locate_block(P, kbi, ps, pl);
        if (!bulk_block(ps, pl)) return;
        const uint64_t pol = policy_evict_last();
        bulk_prefetch_l2_hint(a.g + ps, kGVBytes, pol);
        bulk_prefetch_l2_hint(a.v + ps, kGVBytes, pol);
#pragma unroll
        for (int m = 0; m < M; ++m)
            bulk_prefetch_l2_hint(reinterpret_cast<const unsigned char *>(a.x[m]) + ps * ES,
                                  kXBytes, pol);
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
        if constexpr (PF > 0) {
            // written once: evict these lines first, ahead of the prefetched ones
            const uint64_t pol = policy_evict_first();
            if constexpr (GV) {
                bulk_store_hint(a.g + s, smem_addr(og), kGVBytes, pol);
                bulk_store_hint(a.v + s, smem_addr(ov), kGVBytes, pol);
            }
#pragma unroll
            for (int m = 0; m < M; ++m)
                bulk_store_hint(reinterpret_cast<unsigned char *>(a.x[m]) + s * ES, smem_addr(ox),
                                kXBytes, pol);
        } else {
            if constexpr (GV) {
                bulk_store(a.g + s, smem_addr(og), kGVBytes);
                bulk_store(a.v + s, smem_addr(ov), kGVBytes);
            }
#pragma unroll
            for (int m = 0; m < M; ++m)
                bulk_store(reinterpret_cast<unsigned char *>(a.x[m]) + s * ES, smem_addr(ox),
                           kXBytes);
        }
        bulk_commit();
    };

    int kb = blockIdx.x;
    int64_t start = 0;
    int len = 0;
    uint32_t phase = 0;
    bool pend = false;  // the previous block's tiles wait for their bulk stores
    bool failed = false;
    if (kb < nblocks) {
        locate_block(P, kb, start, len);
        if (!bulk_block(start, len))
            stage_own(start, len, 0);
        else if (t == 0)
            stage_bulk(kb, start, 0);
    }
    int par = 0;
    for (; kb < nblocks; kb += gridDim.x, par ^= 1) {
        if (PF > 0 && t == 0) prefetch_block(kb + PF * (int64_t)gridDim.x);
        const bool full = len == kI8Block;
        const bool bulk = bulk_block(start, len);
        const int nk = kb + gridDim.x;  // the next block
        if (NEXT_SMEM && t == 0 && nk < nblocks) {
            int64_t ns;
            int nl;
            locate_block(P, nk, ns, nl);
            s_nstart[par] = ns;
            s_nlen[par] = nl;
        }
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
            float eb[EP];  // this block's energies (EROW)
#pragma unroll
            for (int m = 0; m < EP; ++m) eb[m] = 0.f;
            auto worker_max = [&](int m, const RepPair<MIX> (&x)[NP]) {
                float2 d[NP];
#pragma unroll
                for (int j = 0; j < NP; ++j) d[j] = dpair(g2[j], x[j]);
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
                if constexpr (EROW) eb[m] = e; else e_acc[m] += e;
                mx = __reduce_max_sync(0xffffffffu, mx);
                if (lane == 0) red_w[m][warp] = mx;
            };
#pragma unroll
            for (int m = 0; m < M; m += 2) {
                RepPair<MIX> xa[NP], xb[NP];
                staged_reps<M, BF16, T, MIX>(sx, m, t, xa, xb);
                worker_max(m, xa);
                if (m + 1 < M) worker_max(m + 1, xb);
            }
            if constexpr (EROW) add_rows(eb);
            if (++since_flush == kFlush) flush();
            // barrier 1; a wait that ran out in any thread stops the whole CTA
            if (__syncthreads_or(timed_out)) {
                failed = true;
                break;
            }
            // every thread wrote its part of the previous block's tiles before
            // the barrier
            if (pend && t == 0) store_tiles(s_pstart);
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
            auto add_worker = [&](float2 scr, const RepPair<MIX> (&x)[NP]) {
                const float s = scr.x, r = scr.y;
                bool ok = true;
                float2 n[NP];
                if constexpr (i8_fast<M, BF16>()) {
                    float far = 0.f;
#pragma unroll
                    for (int j = 0; j < NP; ++j) n[j] = code2_fast_max(dpair(g2[j], x[j]), r, far);
                    // warp-uniform: a lane that needs the exact quotient takes
                    // the whole warp through it (the same codes for the rest)
                    ok = !__any_sync(0xffffffffu, !(far < kCodeMargin));
                } else {
#pragma unroll
                    for (int j = 0; j < NP; ++j) n[j] = code2_fast(dpair(g2[j], x[j]), r, ok);
                }
                if (!ok) {
#pragma unroll
                    for (int j = 0; j < NP; ++j) {
                        const float2 d = dpair(g2[j], x[j]);
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
                RepPair<MIX> xa[NP], xb[NP];
                staged_reps<M, BF16, T, MIX>(sx, m, t, xa, xb);
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
                auto worker_max = [&](int m, const RepPair<MIX> (&x)[NP]) {
                    float2 d[NP];
#pragma unroll
                    for (int j = 0; j < NP; ++j) d[j] = dpair(g2[j], x[j]);
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
                    RepPair<MIX> xa[NP], xb[NP];
                    staged_reps<G, BF16, T, MIX>(sx, m, t, xa, xb, GQ);
                    worker_max(m, xa);
                    if (m + 1 < GQ) worker_max(m + 1, xb);
                }
                if constexpr (GROUPED) {
                    flush_rows(m0, GQ);
                    if (q == 0 && ++since_flush == kFlush) flush();
                } else if (++since_flush == kFlush) {
                    flush();
                }
                // barrier 1 (of the group); a wait that ran out in any thread
                // stops the whole CTA
                if (__syncthreads_or(timed_out)) {
                    stop = true;
                    break;
                }
                if (q == 0) {
                    // every thread wrote its part of the previous block's tiles
                    // before the barrier
                    if (pend && t == 0) store_tiles(s_pstart);
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
                auto add_worker = [&](float2 scr, const RepPair<MIX> (&x)[NP]) {
                    const float sc = scr.x, r = scr.y;
                    bool ok = true;
                    float2 n[NP];
                    if constexpr (i8_fast<M, BF16>()) {
                        float far = 0.f;
#pragma unroll
                        for (int j = 0; j < NP; ++j)
                            n[j] = code2_fast_max(dpair(g2[j], x[j]), r, far);
                        ok = !__any_sync(0xffffffffu, !(far < kCodeMargin));
                    } else {
#pragma unroll
                        for (int j = 0; j < NP; ++j) n[j] = code2_fast(dpair(g2[j], x[j]), r, ok);
                    }
                    if (!ok) {
#pragma unroll
                        for (int j = 0; j < NP; ++j) {
                            const float2 d = dpair(g2[j], x[j]);
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
                    RepPair<MIX> xa[NP], xb[NP];
                    staged_reps<G, BF16, T, MIX>(sx, m, t, xa, xb, GQ);
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
        float2 v2[NP];
        if constexpr (DGV) {
            float v[PER];
            load_direct(v, a.v, start, len, bulk);
#pragma unroll
            for (int j = 0; j < NP; ++j) v2[j] = make_float2(v[2 * j], v[2 * j + 1]);
        } else {
#pragma unroll
            for (int c = 0; c < PER; c += 4) {
                const float4 q = *reinterpret_cast<const float4 *>(sv + el(c));
                v2[c / 2] = make_float2(q.x, q.y);
                v2[c / 2 + 1] = make_float2(q.z, q.w);
            }
        }
        float2 mean2[NP];
        mean_of_sum<M, NP>(sum2, mean2);
        // the previous block's bulk stores have read the tiles before any
        // thread passes barrier 2 and rewrites them
        if (t == 0) bulk_wait_read();
        // barrier 2; elements beyond a short block hold 0 and do not move
        // the maximum
        const float s = codec_scale(block_amax2<NP, W>(mean2, red1));
        // every thread has read this block's staging: the next block's bulk
        // copies go into the same buffer while the rest of this block runs
        // (a short or unaligned next block is staged after the stores)
        if constexpr (NEXT_SMEM) {
            if (t == 0 && nk < nblocks && bulk_block(s_nstart[par], s_nlen[par]))
                stage_bulk(nk, s_nstart[par], 0);
        } else if (t == 0 && nk < nblocks) {
            int64_t ns;
            int nl;
            locate_block(P, nk, ns, nl);
            if (bulk_block(ns, nl)) stage_bulk(nk, ns, 0);
        }
        // decode, outer step and stores chunk by chunk (4 elements), so a
        // chunk's results alone are live
        const float rs = __frcp_rn(s);
        auto lo_hi = [](const float2 (&p)[2], int i) { return (i & 1) ? p[i >> 1].y : p[i >> 1].x; };
        float2 b2 = splat2(0.f);
#pragma unroll
        for (int c = 0; c < PER; c += 4) {
            const int j = c / 2;  // the chunk's first pair
            const float2 y[2] = {mean2[j], mean2[j + 1]};
            float2 dq[2], gp[2], vp[2];
            decode_mean<2>(y, s, rs, dq);
            // non-finite outputs are counted one by one only in a chunk
            // that has one
            float big = 0.f;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                if (full) b2 = __ffma2_rn(dq[h], dq[h], b2);
                outer_step2(k, dq[h], g2[j + h], v2[j + h], gp[h], vp[h]);
                big = max3_nan(big, fabsf(gp[h].x), fabsf(gp[h].y));
                big = max3_nan(big, fabsf(vp[h].x), fabsf(vp[h].y));
            }
            if (!full) {
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    if (el(c + i) < len) b32 = fmaf(lo_hi(dq, i), lo_hi(dq, i), b32);
            }
            if (!(big <= FLT_MAX)) {
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    if (full || el(c + i) < len) nf += not_finite(lo_hi(gp, i), lo_hi(vp, i));
            }

            // 5. the stores
            if (bulk) {
                if constexpr (BF16) {
                    *reinterpret_cast<uint2 *>(ox + el(c) * 2) =
                        make_uint2(pack_bf16x2(gp[0].x, gp[0].y), pack_bf16x2(gp[1].x, gp[1].y));
                }
                if constexpr (GV || !BF16)
                    *reinterpret_cast<float4 *>(og + el(c)) =
                        make_float4(gp[0].x, gp[0].y, gp[1].x, gp[1].y);
                if constexpr (GV)
                    *reinterpret_cast<float4 *>(ov + el(c)) =
                        make_float4(vp[0].x, vp[0].y, vp[1].x, vp[1].y);
                if constexpr (!GV) {
                    __stcs(reinterpret_cast<float4 *>(a.g + start + el(c)),
                           make_float4(gp[0].x, gp[0].y, gp[1].x, gp[1].y));
                    __stcs(reinterpret_cast<float4 *>(a.v + start + el(c)),
                           make_float4(vp[0].x, vp[0].y, vp[1].x, vp[1].y));
                }
            } else {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int e = el(c + i);
                    if (e >= len) continue;
                    const float gpi = lo_hi(gp, i);
                    a.g[start + e] = gpi;
                    a.v[start + e] = lo_hi(vp, i);
#pragma unroll
                    for (int m = 0; m < M; ++m) {
                        if constexpr (BF16)
                            reinterpret_cast<__nv_bfloat16 *>(a.x[m])[start + e] =
                                __float2bfloat16_rn(gpi);
                        else
                            reinterpret_cast<float *>(a.x[m])[start + e] = gpi;
                    }
                }
            }
        }
        if (full) b32 += __fadd_rn(b2.x, b2.y);
        if (bulk) {
            fence_proxy_async_smem();  // the tiles are read by bulk copies
            pend = true;
            if (t == 0) s_pstart = start;
        }
        if (nk < nblocks) {
            if constexpr (NEXT_SMEM) {
                start = s_nstart[par];
                len = s_nlen[par];
            } else {
                locate_block(P, nk, start, len);
            }
            if (!bulk_block(start, len)) stage_own(start, len, 0);
        }
    }
    if (failed) {
        if (t == 0) {
            atomicExch(a.error, 1u);
            // let the loads still in flight land before the CTA exits
            if (in_flight) mbar_wait(bar, phase ^ 1, nullptr);
        }
    } else if (pend) {
        __syncthreads();
        if (t == 0) store_tiles(s_pstart);
    }
    if (t == 0) bulk_wait_all();
    // the energies still in registers, and the squared means of every block
    // since the last flush (the last block's come after its flush check)
    if constexpr (!GROUPED && !EROW) {
        if (since_flush > 0) flush_rows(0, EA);
    }
    flush_b();
    __syncthreads();
    double e64[M];
    double b64 = 0.0;
    if (t == 0) {
#pragma unroll
        for (int w = 0; w < W; ++w) b64 += e_w[w][M];
    }
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
    // the kernel counts blocks in 32 bits: block + grid stays below 2^31
    if (nblocks > (int64_t)INT32_MAX - grid) return cudaErrorInvalidValue;
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
