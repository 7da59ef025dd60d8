// Full-state projection of Eq. fused_normalized_projection on the 5th-generation tensor cores:
//   part[j][t][o] = sum over the k-blocks of segment j of x[t][e] * W[e][o]   (o < nfull)
//   pstats[j][t]  = (sum x, sum x^2) over the same k-blocks
// X [T, NC] bf16 is the A operand (K-major), W is pre-packed as bf16 hi and lo rows
// Wpack[2*nfull(+pad)][NC] (B operand, K-major): one MMA of N = 2*nfull gives x*W_hi and x*W_lo,
// summed in the epilogue, i.e. the fp32 weights to ~2^-17 relative.  Tiles of 128 tokens x 64
// k-elements arrive by TMA (128-byte swizzle) into a 5-stage ring; one thread issues
// tcgen05.mma into a TMEM accumulator; four warps compute the row statistics from the staged
// tiles and, at the end of each segment, read the accumulator back with tcgen05.ld.
// Work split (stream-K): the T/128 x NC/64 k-blocks are cut into equal contiguous ranges, one per
// persistent CTA; a tile cut across CTAs gives several segments, summed later in a fixed order.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <string.h>

#include "xhc_internal.cuh"

namespace xhc {

namespace {

constexpr int BM = 128;        // tokens per tile (MMA M)
constexpr int BK = 64;         // k-elements per stage (128 bytes of bf16 = one swizzle row)
constexpr int MAXSTAGES = 8;
constexpr int NTHREADS = 192;  // warp 0 TMA, warp 1 MMA + TMEM, warps 2..5 statistics + epilogue
// a waiting thread may be suspended up to this long per try (it resumes as soon as the phase
// completes); fewer polls leave the shared-memory pipe to the TMA writes and the epilogues
constexpr uint32_t WAIT_HINT_NS = 20000;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint32_t a, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(a), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t a, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(a), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t a) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(a) : "memory");
}
// Bounded wait on a phase of an mbarrier: false once `limit` ns (global timer) have passed.
__device__ __forceinline__ bool mbar_wait(uint32_t a, uint32_t parity, uint64_t limit) {
    uint64_t t0 = 0;
    for (uint32_t it = 0;; ++it) {
        uint32_t ok;
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n"
            " selp.u32 %0, 1, 0, p;\n}\n"
            : "=r"(ok) : "r"(a), "r"(parity), "r"(WAIT_HINT_NS) : "memory");
        if (ok) return true;
        if ((it & 255u) == 255u) {
            uint64_t now;
            asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(now));
            if (t0 == 0) t0 = now;
            else if (now - t0 > limit) return false;
        }
    }
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst), "l"((uint64_t)map), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

// L2 prefetch of a 2D box (a hint: no shared memory, no completion to wait for)
__device__ __forceinline__ void tma_prefetch_2d(const CUtensorMap* map, int x, int y) {
    asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global [%0, {%1, %2}];" ::"l"((uint64_t)map), "r"(x),
                 "r"(y)
                 : "memory");
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, 8-row groups 1024 B apart.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t addr) {
    uint64_t d = 0;
    d |= (uint64_t)((addr & 0x3FFFFu) >> 4);        // start address
    d |= (uint64_t)(16u >> 4) << 16;                 // leading byte offset (unused for SW128 K-major)
    d |= (uint64_t)(1024u >> 4) << 32;               // stride byte offset: 8 rows x 128 B
    d |= (uint64_t)1 << 46;                          // descriptor version for tcgen05
    d |= (uint64_t)2 << 61;                          // swizzle: 128 B
    return d;
}

// Shared-memory matrix descriptor: MN-major operand, 128-byte swizzle.  The tile is stored as
// blocks of 64 MN-contiguous elements (one 128-byte row per K index, 8-row groups 1024 B apart);
// consecutive 64-element MN blocks are `lbo` bytes apart.
__device__ __forceinline__ uint64_t sw128_desc_mn(uint32_t addr, uint32_t lbo) {
    uint64_t d = 0;
    d |= (uint64_t)((addr & 0x3FFFFu) >> 4);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;     // leading byte offset: between MN blocks
    d |= (uint64_t)(1024u >> 4) << 32;               // stride byte offset: between 8-row K groups
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// Instruction descriptor, kind::f16: bf16 A and B, fp32 accumulator, both K-major, M x N.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, bool a_mn = false) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn ? 1u : 0u) << 15) |
           ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                         uint32_t accum) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(accum)
        : "memory");
}
__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// TMEM -> registers (32 lanes x 16 columns); the wait is in the same statement so the outputs are
// valid on exit, and there is no memory clobber so unrelated global loads can be scheduled
// around it.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float* v) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// registers -> TMEM (32 lanes x 16 columns); the caller waits with tmem_st_wait before the
// values are read again
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const float* v) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};"
        ::"r"(taddr), "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
          "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
          "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
          "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
          "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
          "r"(__float_as_uint(v[15]))
        : "memory");
}
__device__ __forceinline__ void tmem_st_wait() {
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// TMEM -> registers, 32 lanes x 8 columns (wait in the same statement, as above)
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, float* v) {
    uint32_t r[8];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7])
        : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(r[i]);
}

// The tensor cores' fp32 accumulation loses accuracy in proportion to the length of the chain of
// MMAs accumulated in one TMEM accumulator (measured: about 7e-8 of the result per 64-element
// k-block, systematic rather than random, so ~6e-5 over the ~860 k-blocks a CTA covers at
// K = 65536).  The accumulator is therefore restarted every SUB_K k-elements (a sub-segment);
// the epilogue adds the sub-segments' results in fp32 (round to nearest) into a running sum kept
// in TMEM columns [NB, NB + nfull), and writes the piece's partial once, as before.  Sub-segments
// of 4096 k-elements keep the chain's error below ~5e-6 of the result.
constexpr int SUB_K = 4096;

// TMEM columns of one CTA: the accumulator (NB) and the running sum (nfull), a power of two
__host__ __device__ inline uint32_t proj_tc_cols(int NB, int nfull) {
    const int need = NB + nfull;
    return need <= 32 ? 32u : need <= 64 ? 64u : need <= 128 ? 128u : need <= 256 ? 256u : 512u;
}

struct ProjTcArgs {
    int T, KB;          // tokens, k-blocks per tile
    int MT;             // M tiles
    long long W;        // total k-blocks
    int P;              // persistent CTAs
    int nfull;          // outputs per token (hi rows), lo rows follow
    int NB;             // B rows = MMA N total (multiple of 16)
    int nchunk;         // MMA instructions per k-step (N split in chunks of NB / nchunk <= 256)
    int nseg;           // partial slots per tile
    int stages;         // smem ring depth
    int kps;            // k-blocks of 64 per stage (projections; 1 for the weight gradients)
    uint64_t wait_ns;   // limit of every bounded wait
    int force_timeout;  // test hook: wait for a release that nothing triggers (see below)
    float* part;        // [nseg][T][nfull]
    float* pstats;      // [nseg][T][2] row sums / sums of squares of A; null: not computed
    int* err;           // set to a nonzero code when a wait gives up
};

__device__ __forceinline__ long long range_start(long long W, int P, int c) {
    return (W * c) / P;
}

// A_MN = false: rows of A are tokens, A tile = X[m*128.., kb*64..] (K-major); row statistics on.
// A_MN = true : rows of A are state elements e, K = tokens; the A tile is X[t0.., e0..] as stored
//               (two 64-wide e blocks, MN-major); no statistics (weight gradients).
template <bool A_MN>
__global__ void __launch_bounds__(NTHREADS, 2)
k_proj_tc(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
          ProjTcArgs a) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    const int STAGES = a.stages;
    unsigned char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);  // stays a shared pointer
    const int KPS = A_MN ? 1 : a.kps;               // k-blocks of 64 per stage
    const uint32_t A_BYTES = (uint32_t)KPS * BM * BK * 2;
    const uint32_t B_BYTES = (uint32_t)KPS * a.NB * BK * 2;
    const uint32_t STAGE = A_BYTES + B_BYTES;  // both multiples of 1024
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE);
    // bars[0..S) full, [S..2S) empty, [2S] acc full, [2S+1] acc empty
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 2);
    __shared__ int s_abort;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c = blockIdx.x;
    const long long g0 = range_start(a.W, a.P, c), g1 = range_start(a.W, a.P, c + 1);
    const uint32_t ncols = proj_tc_cols(a.NB, a.nfull);
    // k-block groups (g units) per sub-segment
    const int SUBG = max(1, SUB_K / (BK * KPS));

    if (threadIdx.x == 0) {
        s_abort = 0;
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_u32(&bars[s]), 1);
            mbar_init(smem_u32(&bars[STAGES + s]), 1 + 4);
        }
        mbar_init(smem_u32(&bars[2 * STAGES]), 1);
        mbar_init(smem_u32(&bars[2 * STAGES + 1]), 4);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)),
                     "r"(ncols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            // test hook (xhc_debug_set, XHC_DEBUG_FORCE_TIMEOUT): before anything is issued, wait
            // for the first release of stage 0, which needs the MMA of a load that was never
            // issued.  The waits of every role then run out with no TMA load and no MMA in
            // flight, and the kernel takes its abort path: error word set, TMEM freed, return.
            if (a.force_timeout && g0 < g1 && !mbar_wait(smem_u32(&bars[STAGES]), 0u, a.wait_ns)) {
                atomicExch(a.err, 6);
                s_abort = 1;
            }
            // stage s and phase ph of load `it`, tile m and k-block kb of g: advanced step by
            // step (no division per k-block)
            int it = 0, s = 0, m = (int)(g0 / a.KB), kb = (int)(g0 % a.KB);
            uint32_t ph = 0;
            for (long long g = g0; g < g1 && !*(volatile int*)&s_abort; ++g, ++it) {
                if (g > g0) {
                    if (++kb == a.KB) { kb = 0; ++m; }
                    if (++s == STAGES) { s = 0; ph ^= 1u; }
                }
                if (it >= STAGES && !mbar_wait(smem_u32(&bars[STAGES + s]), ph ^ 1, a.wait_ns)) {
                    atomicExch(a.err, 1);
                    s_abort = 1;
                    break;
                }
                if (*(volatile int*)&s_abort) break;
                const uint32_t full = smem_u32(&bars[s]);
                mbar_expect_tx(full, STAGE);
                unsigned char* st = smem + (size_t)s * STAGE;
                if (A_MN) {
                    tma_load_2d(smem_u32(st), &tmA, m * BM, kb * BK, full);
                    tma_load_2d(smem_u32(st + A_BYTES / 2), &tmA, m * BM + 64, kb * BK, full);
                } else {
                    for (int p2 = 0; p2 < KPS; ++p2)
                        tma_load_2d(smem_u32(st + p2 * BM * BK * 2), &tmA, (kb * KPS + p2) * BK, m * BM, full);
                }
                const int nb_box = a.NB / a.nchunk;
                for (int p2 = 0; p2 < KPS; ++p2)
                    for (int q = 0; q < a.nchunk; ++q)
                        tma_load_2d(smem_u32(st + A_BYTES + (size_t)p2 * a.NB * 128 + (size_t)q * nb_box * 128),
                                    &tmB, (kb * KPS + p2) * BK, q * nb_box, full);
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            const int nb_chunk = a.NB / a.nchunk;
            const uint32_t idesc = idesc_bf16(BM, nb_chunk, A_MN);
            int s = 0;          // stage of the next k-block and its phase, advanced per k-block
            uint32_t ph = 0;
            int seg = 0;
            long long g = g0;
            while (g < g1) {
                const int m = (int)(g / a.KB);
                const long long sub_end = (long long)m * a.KB + ((g - (long long)m * a.KB) / SUBG + 1) * SUBG;
                const long long gend = min(min(g1, (long long)(m + 1) * a.KB), sub_end);
                if (seg > 0 && !mbar_wait(smem_u32(&bars[2 * STAGES + 1]), (uint32_t)((seg - 1) & 1), a.wait_ns)) {
                    atomicExch(a.err, 2);
                    s_abort = 1;
                    break;
                }
                tc_fence_after();
                bool first = true;
                for (; g < gend; ++g) {
                    if (!mbar_wait(smem_u32(&bars[s]), ph, a.wait_ns)) {
                        atomicExch(a.err, 3);
                        s_abort = 1;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t abase = smem_u32(smem + (size_t)s * STAGE);
                    const uint32_t bbase = abase + A_BYTES;
                    for (int p2 = 0; p2 < KPS; ++p2) {
#pragma unroll
                        for (int kk = 0; kk < BK / 16; ++kk) {
                            // K-major: +32 B per 16 k-elements inside the swizzled row; MN-major:
                            // +16 K-rows of 128 B
                            const uint64_t ad = A_MN ? sw128_desc_mn(abase + kk * 2048, A_BYTES / 2)
                                                     : sw128_desc(abase + p2 * BM * BK * 2 + kk * 32);
                            for (int q = 0; q < a.nchunk; ++q) {
                                const uint64_t bd =
                                    sw128_desc(bbase + p2 * a.NB * 128 + q * nb_chunk * 128 + kk * 32);
                                mma_bf16(tmem + (uint32_t)(q * nb_chunk), ad, bd, idesc,
                                         (first && p2 == 0 && kk == 0) ? 0u : 1u);
                            }
                        }
                    }
                    first = false;
                    mma_commit(smem_u32(&bars[STAGES + s]));  // stage free once these MMAs finish
                    if (++s == STAGES) { s = 0; ph ^= 1u; }
                }
                if (*(volatile int*)&s_abort) break;
                mma_commit(smem_u32(&bars[2 * STAGES]));     // accumulator ready
                ++seg;
            }
        }
    } else {
        // ---------------- statistics + epilogue (warps 2..5) ----------------
        const int quarter = warp & 3;           // TMEM lanes this warp may access
        const int r = quarter * 32 + lane;      // tile row = token within the tile
        int s = 0;                              // stage of the next k-block and its phase
        uint32_t ph = 0;
        int seg = 0;
        long long g = g0;
        bool ok = true;
        // row sums in packed pairs, four independent accumulators each (short dependency chains,
        // half the instructions of scalar sums), over the whole piece (tile x this CTA's range)
        float2 a1[4], a2[4];
        while (g < g1 && ok) {
            const int m = (int)(g / a.KB);
            const long long piece_end = min(g1, (long long)(m + 1) * a.KB);
            const long long sub_end = (long long)m * a.KB + ((g - (long long)m * a.KB) / SUBG + 1) * SUBG;
            const long long gend = min(piece_end, sub_end);
            const bool first_sub = (g == max(g0, (long long)m * a.KB));
            const bool last_sub = (gend == piece_end);
            if (first_sub) {
#pragma unroll
                for (int e = 0; e < 4; ++e) a1[e] = a2[e] = make_float2(0.f, 0.f);
            }
            for (; g < gend; ++g) {
                if (!mbar_wait(smem_u32(&bars[s]), ph, a.wait_ns)) {
                    atomicExch(a.err, 4);
                    ok = false;
                    break;
                }
                if (!A_MN && a.pstats) {
                    // row r of the A tile: 128 bytes, logical 16-byte chunk q at position
                    // q ^ (r % 8) (128-byte swizzle).  Reading the chunks in logical order puts the
                    // 8 rows of a quarter warp on 8 different bank groups (physical order would put
                    // all 32 rows of the warp on the same 4 banks: 8-way conflicts)
                    for (int p2 = 0; p2 < KPS; ++p2) {
                        const uint4* row = reinterpret_cast<const uint4*>(smem + (size_t)s * STAGE +
                                                                          p2 * BM * BK * 2 + r * 128);
                        uint4 v[8];
#pragma unroll
                        for (int q = 0; q < 8; ++q) v[q] = row[q ^ (r & 7)];
#pragma unroll
                        for (int q = 0; q < 8; ++q) {
                            const uint32_t w[4] = {v[q].x, v[q].y, v[q].z, v[q].w};
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                const float2 f = make_float2(__uint_as_float(w[e] << 16),
                                                             __uint_as_float(w[e] & 0xffff0000u));
                                a1[e] = __fadd2_rn(a1[e], f);
                                a2[e] = __ffma2_rn(f, f, a2[e]);
                            }
                        }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&bars[STAGES + s]));
                if (++s == STAGES) { s = 0; ph ^= 1u; }
            }
            if (!ok) break;
            // the segment's slot: index of this CTA among those covering tile m
            int c0 = (int)(((long long)m * a.KB * a.P) / a.W);
            while (c0 > 0 && range_start(a.W, a.P, c0) > (long long)m * a.KB) --c0;
            while (range_start(a.W, a.P, c0 + 1) <= (long long)m * a.KB) ++c0;
            const int j = c - c0;
            if (!mbar_wait(smem_u32(&bars[2 * STAGES]), (uint32_t)(seg & 1), a.wait_ns)) {
                atomicExch(a.err, 5);
                break;
            }
            tc_fence_after();
            const int t = m * BM + r;
            float* dst = a.part + ((long long)j * a.T + t) * a.nfull;
            const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16);
            // hi columns [0, nfull), lo columns [nfull, 2 nfull); running sum of the piece's
            // sub-segments at [NB, NB + nfull)
            for (int o0 = 0; o0 < a.nfull; o0 += 16) {
                float hi[16], lo[16], sum[16];
                tmem_ld16(tl + (uint32_t)o0, hi);
                tmem_ld16(tl + (uint32_t)(a.nfull + o0), lo);
                if (first_sub) {
#pragma unroll
                    for (int q = 0; q < 16; ++q) sum[q] = hi[q] + lo[q];
                } else {
                    tmem_ld16(tl + (uint32_t)(a.NB + o0), sum);
#pragma unroll
                    for (int q = 0; q < 16; ++q) sum[q] += hi[q] + lo[q];
                }
                if (!last_sub) {
                    tmem_st16(tl + (uint32_t)(a.NB + o0), sum);
                } else if (t < a.T) {
                    const int n = min(16, a.nfull - o0);
#pragma unroll
                    for (int q = 0; q < 16; ++q)
                        if (q < n) dst[o0 + q] = sum[q];
                }
            }
            if (!last_sub) tmem_st_wait();
            if (last_sub && !A_MN && a.pstats && t < a.T) {
                const float s1 = (a1[0].x + a1[0].y) + (a1[1].x + a1[1].y) + (a1[2].x + a1[2].y) + (a1[3].x + a1[3].y);
                const float s2 = (a2[0].x + a2[0].y) + (a2[1].x + a2[1].y) + (a2[2].x + a2[2].y) + (a2[3].x + a2[3].y);
                a.pstats[((long long)j * a.T + t) * 2 + 0] = s1;
                a.pstats[((long long)j * a.T + t) * 2 + 1] = s2;
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&bars[2 * STAGES + 1]));
            ++seg;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(ncols)
                     : "memory");
    }
}

// ---------------------------------------------------------------------------------------------
// Wpack[r][e] = hi / lo bf16 parts of W[e][o] (r = o for hi, r = nfull + o for lo; 0 for pad)

__global__ void k_pack_w(WSegs W, int nfull, int NB, int K, uint16_t* __restrict__ Wpack) {
    const int e = blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= K) return;
    for (int o = 0; o < nfull; ++o) {
        const float w = seg_elem(W, e, o);
        const __nv_bfloat16 h = __float2bfloat16_rn(w);
        const float rem = w - __bfloat162float(h);
        Wpack[(int64_t)o * K + e] = __bfloat16_as_ushort(h);
        Wpack[(int64_t)(nfull + o) * K + e] = __bfloat16_as_ushort(__float2bfloat16_rn(rem));
    }
    for (int r = 2 * nfull; r < NB; ++r) Wpack[(int64_t)r * K + e] = 0;
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        cudaDriverEntryPointQueryResult q;
        void* p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (PFN_cuTensorMapEncodeTiled_v12000)p;
    }
    return fn;
}

bool make_map_box(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows,
                  uint32_t box_inner, uint32_t box_rows, uint64_t row_bytes = 0) {
    auto enc = get_encode();
    if (!enc) return false;
    cuuint64_t gdim[2] = {inner, rows};
    cuuint64_t gstride[1] = {row_bytes ? row_bytes : inner * 2};
    cuuint32_t box[2] = {box_inner, box_rows};
    cuuint32_t es[2] = {1, 1};
    CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), gdim, gstride,
                     box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint32_t box_rows) {
    return make_map_box(m, base, inner, rows, (uint32_t)BK, box_rows);
}

int num_sms() {
    static int n = 0;
    if (!n) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        if (n <= 0) n = 148;
    }
    return n;
}

}  // namespace

int proj_tc_nb(int nfull) {
    int nb = (2 * nfull + 15) / 16 * 16;
    if (nb > 256) nb = (nb + 31) / 32 * 32;  // two equal chunks, each a multiple of 16
    return nb;
}

// ring depth that fits the shared memory of one of `ctas` CTAs per SM
int proj_tc_stages_for(int NB, int kps, int ctas) {
    const size_t stage = (size_t)kps * ((size_t)BM * BK * 2 + (size_t)NB * BK * 2);
    const size_t budget = (size_t)(ctas == 2 ? 110 : 220) * 1024;
    int s = (int)((budget - 2048) / stage);
    return s > MAXSTAGES ? MAXSTAGES : s;
}

// Projections (A = X rows, K-major) with a narrow B load two k-blocks per stage, so every row of
// an A tile is read as 256 contiguous bytes (measured faster for the active projections; the wide
// full-state projection keeps one k-block per stage and two CTAs per SM); the weight gradients
// (A MN-major) already read 256 bytes per row with one k-block.  Two CTAs per SM (each with its
// own TMA ring and 256 TMEM columns) keep twice the loads in flight when two rings fit;
// otherwise (or with more than 256 accumulator columns) one CTA per SM.
ProjTcPlan plan_proj_tc(int T, int K, int nfull, int nsm, bool proj) {
    ProjTcPlan p;
    p.NB = proj_tc_nb(nfull);
    p.kps = (proj && proj_tc_stages_for(p.NB, 2, 2) >= 2) ? 2 : 1;
    p.KB = (K + BK * p.kps - 1) / (BK * p.kps);
    p.MT = (T + BM - 1) / BM;
    p.W = (long long)p.KB * p.MT;
    p.nchunk = p.NB > 256 ? 2 : 1;
    // two CTAs per SM need both rings in shared memory and both TMEM allocations (accumulator and
    // running sum) within half of the SM's 512 columns
    p.ctas = (proj_tc_cols(p.NB, nfull) <= 256 && proj_tc_stages_for(p.NB, p.kps, 2) >= 2) ? 2 : 1;
    const int sms = p.ctas * (nsm > 0 ? nsm : 148);
    long long P = std::min<long long>(sms, std::max<long long>(1, p.W / 4));
    p.P = (int)P;
    const long long per = p.W / p.P;  // >= 4
    p.nseg = (int)((p.KB + per - 1) / per) + 1;
    if (p.nseg > p.P) p.nseg = p.P;
    return p;
}

size_t proj_tc_smem(const ProjTcPlan& p) {
    const int S = proj_tc_stages_for(p.NB, p.kps, p.ctas);
    return (size_t)S * p.kps * (BM * BK * 2 + (size_t)p.NB * BK * 2) + (2 * S + 2) * 8 + 16 + 1024;
}

cudaError_t launch_pack_w(const WSegs& W, int nfull, int NB, int K, uint16_t* Wpack, cudaStream_t st) {
    k_pack_w<<<(K + 255) / 256, 256, 0, st>>>(W, nfull, NB, K, Wpack); note_launch();
    return cudaGetLastError();
}

cudaError_t launch_proj_tc(const uint16_t* X, int T, int K, const uint16_t* Wpack, int nfull,
                           const ProjTcPlan& p, float* part, float* pstats, int* err,
                           cudaStream_t st) {
    CUtensorMap ma, mb;
    if (!make_map(&ma, X, (uint64_t)K, (uint64_t)T, BM)) return cudaErrorInvalidValue;
    if (!make_map(&mb, Wpack, (uint64_t)K, (uint64_t)p.NB, (uint32_t)(p.NB / p.nchunk)))
        return cudaErrorInvalidValue;
    cudaError_t e = cudaMemsetAsync(part, 0, (size_t)p.nseg * T * nfull * sizeof(float), st);
    if (e != cudaSuccess) return e;
    if (pstats) {
        e = cudaMemsetAsync(pstats, 0, (size_t)p.nseg * T * 2 * sizeof(float), st);
        if (e != cudaSuccess) return e;
    }
    const size_t sm = proj_tc_smem(p);
    e = cudaFuncSetAttribute((const void*)k_proj_tc<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    ProjTcArgs a;
    a.T = T;
    a.KB = p.KB;
    a.MT = p.MT;
    a.W = p.W;
    a.P = p.P;
    a.nfull = nfull;
    a.NB = p.NB;
    a.nchunk = p.nchunk;
    a.nseg = p.nseg;
    a.stages = proj_tc_stages_for(p.NB, p.kps, p.ctas);
    a.kps = p.kps;
    if (a.stages < 2) return cudaErrorInvalidValue;
    a.part = part;
    a.pstats = pstats;
    a.err = err;
    a.wait_ns = debug_wait_ns();
    a.force_timeout = debug_take_force_timeout();
    k_proj_tc<false><<<p.P, NTHREADS, sm, st>>>(ma, mb, a); note_launch();
    return cudaGetLastError();
}

// dZpack[r][t]: hi / lo bf16 parts of dz[t][o] (r = o for hi, r = n + o for lo, 0 for pad), the
// K-major B operand of the weight gradient.
__global__ void k_pack_dz(const float* __restrict__ dz, int ldz, int n, int NB, int T, int Tp,
                          uint16_t* __restrict__ dzp) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= T) return;
    for (int o = 0; o < n; ++o) {
        const float w = dz[(int64_t)t * ldz + o];
        const __nv_bfloat16 h = __float2bfloat16_rn(w);
        dzp[(int64_t)o * Tp + t] = __bfloat16_as_ushort(h);
        dzp[(int64_t)(n + o) * Tp + t] = __bfloat16_as_ushort(__float2bfloat16_rn(w - __bfloat162float(h)));
    }
    for (int r = 2 * n; r < NB; ++r) dzp[(int64_t)r * Tp + t] = 0;
}

// Weight gradient on the tensor cores: part[j][e][o] = sum over the segment's tokens of
// A[t][e] dz[t][o] (A = X or the active state, [T, E] bf16), with dz split into bf16 hi/lo.
cudaError_t launch_wgrad_tc(const uint16_t* A, int T, int E, const float* dz, int ldz, int n,
                            uint16_t* dzpack, const ProjTcPlan& p, float* part, int* err,
                            cudaStream_t st) {
    const int Tp = (T + 7) / 8 * 8;  // 16-byte row stride for the tensor map
    k_pack_dz<<<(T + 255) / 256, 256, 0, st>>>(dz, ldz, n, p.NB, T, Tp, dzpack); note_launch();
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    CUtensorMap ma, mb;
    // A: [T rows, E inner], box {64 e, 64 tokens}; B: [NB rows, T inner], box {64 tokens, NB}
    if (!make_map_box(&ma, A, (uint64_t)E, (uint64_t)T, 64, BK)) return cudaErrorInvalidValue;
    if (!make_map_box(&mb, dzpack, (uint64_t)T, (uint64_t)p.NB, BK, (uint32_t)(p.NB / p.nchunk),
                      (uint64_t)Tp * 2))
        return cudaErrorInvalidValue;
    e = cudaMemsetAsync(part, 0, (size_t)p.nseg * E * n * sizeof(float), st);
    if (e != cudaSuccess) return e;
    const size_t sm = proj_tc_smem(p);
    e = cudaFuncSetAttribute((const void*)k_proj_tc<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    ProjTcArgs a;
    a.T = E;  // rows of the output
    a.KB = p.KB;
    a.MT = p.MT;
    a.W = p.W;
    a.P = p.P;
    a.nfull = n;
    a.NB = p.NB;
    a.nchunk = p.nchunk;
    a.nseg = p.nseg;
    a.stages = proj_tc_stages_for(p.NB, p.kps, p.ctas);
    a.kps = p.kps;
    if (a.stages < 2) return cudaErrorInvalidValue;
    a.part = part;
    a.pstats = nullptr;
    a.err = err;
    a.wait_ns = debug_wait_ns();
    a.force_timeout = 0;
    k_proj_tc<true><<<p.P, NTHREADS, sm, st>>>(ma, mb, a); note_launch();
    return cudaGetLastError();
}

int device_sms() { return num_sms(); }

// ---------------------------------------------------------------------------------------------
// Full-state input gradient on the tensor cores (backward of the full-state projection, of the
// norm statistics and of the dense reads):
//   dX[t][i*C + c] = base + sum_o dZ[t][o] W[i*C + c][o] + a_t + b_t x[t][i*C + c]
//   base = dX_act[t][j][c]                                  if stream i is active slot j
//        = dX[t][i*C + c] + sum_q H_pre[t][q][i] d_input_q[t][c]   otherwise
// MMA K = nfull (dZ and W in bf16: this term is a small share of dX, whose storage is bf16); the
// tiling is described at the kernel (k_dxf_tc).  The same machinery with "streams" = the k active
// slots updates dX_act in the backward of each slot's pre-map (k_dx_tc<true>).

namespace {

constexpr int DX_BN = 128;
constexpr int DX_EW = 16;                       // epilogue warps: 4 per TMEM lane quarter
constexpr int DX_THREADS = (2 + DX_EW) * 32;    // + TMA warp + MMA warp

// 16-byte global read (plain LDG: measured faster here than the non-coherent or no-allocate forms)
__device__ __forceinline__ uint4 ld_stream(const void* p) {
    uint4 r;
    asm volatile("ld.global.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "l"(p));
    return r;
}

struct DxArgs {
    int T, C, N, k, G;
    int m;                // full-state epilogue: fixed streams 0..m-1 (active on every token)
    int dense;            // full-state epilogue: 0 = sparse-read ablation (no dense-read term)
    int slot;             // active epilogue: slot of the pre-map
    int NH;               // active epilogue: streams of the H_pre rows
    float* dxa;           // active epilogue: dX_act [T][k][C] fp32, updated in place
    int nkb, ksteps;      // k-blocks of 64, MMA k-steps of 16
    int ns;               // operand stages in shared memory (1 or 2)
    int TT, CT;           // token tiles, channel tiles per stream
    long long ntiles;
    int P;
    const uint16_t* X;
    uint16_t* dX;
    const uint16_t* dinput;
    const float* hpre;
    const int* I;
    const float* dxact;
    const float* scal;
    int scal_ld;
    int* err;
    uint64_t wait_ns;     // limit of every bounded wait
    float* dotp;          // active epilogue: [k][ncg][T] dot partials over 32-channel groups
    uint16_t* dcopy;      // active epilogue: [G][T][C] copies of d_input (written by slot-0 tiles)
    int ncg;              // active epilogue: C / 32
};

// ACT = true (the instantiated form): active-state epilogue, "streams" are the k active slots j:
//              dX_act[t][j][c] += acc + H_pre[t][slot][I_j] d_input[t][c] - cx_t x_act[t][j][c]
//              (X = x_act of the slot, scal = the per-token matrices with cx at 112); from the
//              same loads, the dH_pre dot <x_act_j, d_input> of each 32-channel group (dotp) and,
//              in the j = 0 tiles, the workspace copy of d_input (dcopy).
// ACT = false: a full-state epilogue over the N streams; not instantiated (the full-state dX is
// k_dxf_tc, which also adds the dense-read gradient of the non-active rows).
template <bool ACT>
__global__ void __launch_bounds__(DX_THREADS, 1)
k_dx_tc(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, DxArgs a) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);  // stays a shared pointer
    const uint32_t A_BYTES = (uint32_t)a.nkb * BM * BK * 2;
    const uint32_t B_BYTES = (uint32_t)a.nkb * DX_BN * BK * 2;
    const uint32_t STAGE = A_BYTES + B_BYTES;
    const int NS = a.ns;                             // operand stages (1 or 2)
    const int nsh = NS - 1;                          // log2(NS)
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + NS * STAGE);
    // [0,2) operands full, [2,4) operands empty, [4,6) tmem full, [6,8) tmem empty
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 8);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < 2; ++s) {
            mbar_init(smem_u32(&bars[s]), 1);
            mbar_init(smem_u32(&bars[2 + s]), 1);
            mbar_init(smem_u32(&bars[4 + s]), 1);
            mbar_init(smem_u32(&bars[6 + s]), DX_EW / 2);  // one group of epilogue warps per buffer
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)), "r"(256u) : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // 32-bit tile arithmetic (the host keeps ntiles below 2^31): the divisions run per tile
    const int nloc = (a.ntiles > blockIdx.x) ? (int)((a.ntiles - 1 - blockIdx.x) / a.P) + 1 : 0;

    if (warp == 0) {
        if (lane == 0) {
            for (int n = 0; n < nloc; ++n) {
                const int tile = (int)blockIdx.x + n * a.P;
                const int i = tile % a.N;
                const int rest = tile / a.N;
                const int ct = rest % a.CT, tt = rest / a.CT;
                const int s = (int)(n & nsh);
                if (n >= NS && !mbar_wait(smem_u32(&bars[2 + s]), (uint32_t)(((n >> nsh) - 1) & 1), a.wait_ns)) {
                    atomicExch(a.err, 11);
                    break;
                }
                const uint32_t full = smem_u32(&bars[s]);
                mbar_expect_tx(full, STAGE);
                unsigned char* st = smem + (size_t)s * STAGE;
                for (int kb = 0; kb < a.nkb; ++kb) {
                    tma_load_2d(smem_u32(st + kb * BM * BK * 2), &tmA, kb * BK, tt * BM, full);
                    tma_load_2d(smem_u32(st + A_BYTES + kb * DX_BN * BK * 2), &tmB, kb * BK,
                                i * a.C + ct * DX_BN, full);
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(BM, DX_BN);
            for (int n = 0; n < nloc; ++n) {
                const int s = (int)(n & 1);        // TMEM buffer
                const int os = (int)(n & nsh);     // operand stage
                if (!mbar_wait(smem_u32(&bars[os]), (uint32_t)((n >> nsh) & 1), a.wait_ns)) {
                    atomicExch(a.err, 12);
                    break;
                }
                if (n >= 2 && !mbar_wait(smem_u32(&bars[6 + s]), (uint32_t)(((n >> 1) - 1) & 1), a.wait_ns)) {
                    atomicExch(a.err, 13);
                    break;
                }
                tc_fence_after();
                const uint32_t abase = smem_u32(smem + (size_t)os * STAGE);
                const uint32_t bbase = abase + A_BYTES;
                for (int ks = 0; ks < a.ksteps; ++ks) {
                    const int kb = ks >> 2, kk = ks & 3;
                    mma_bf16(tmem + (uint32_t)(s * DX_BN), sw128_desc(abase + kb * BM * BK * 2 + kk * 32),
                             sw128_desc(bbase + kb * DX_BN * BK * 2 + kk * 32), idesc, ks > 0 ? 1u : 0u);
                }
                mma_commit(smem_u32(&bars[2 + os]));  // operands consumed
                mma_commit(smem_u32(&bars[4 + s]));  // accumulator ready
            }
        }
    } else {
        // Two groups of 8 epilogue warps take alternate tiles (group g: tiles n = g mod 2, TMEM
        // buffer g), so one group's global reads overlap the other's arithmetic and stores.  In a
        // group, warp w owns rows [32 (w % 4), +32) and columns [64 (w / 4), +64) of the tile,
        // taken as two halves of 32 columns.  The accumulator is read row-per-lane from TMEM,
        // bounced through a padded shared tile and re-read with 4 lanes per row (8 channels each)
        // so that the global reads and writes are contiguous along the channels.
        const int ew = warp - 2;                   // epilogue warp index
        const int grp = ew >> 3;                   // tile parity of this warp's group
        const int quarter = warp & 3;              // TMEM lane quarter (warp id % 4)
        const int chalf = (ew & 7) >> 2;           // 64-column half of the tile
        float* tileb = reinterpret_cast<float*>(smem + NS * STAGE + 128) + ew * (32 * 33 + 32 * 8);
        float* meta = tileb + 32 * 33;             // per row: j, h0..h3, sa, sb
        for (int n = grp; n < nloc; n += 2) {
            const int tile = (int)blockIdx.x + n * a.P;
            const int i = tile % a.N;
            const int rest = tile / a.N;
            const int ct = rest % a.CT, tt = rest / a.CT;
            const int s = (int)(n & 1);
            {
                // per-row metadata of this lane's row (row-per-lane, matches the TMEM layout)
                const int t = tt * BM + quarter * 32 + lane;
                int j = -1;
                float h[4] = {0.f, 0.f, 0.f, 0.f};
                float sa = 0.f, sb = 0.f;
                if (t < a.T) {
                    if (ACT) {
                        j = i;
                        h[0] = a.hpre[((long long)t * a.G + a.slot) * a.NH + a.I[(long long)t * a.k + i]];
                        h[1] = a.scal[(long long)t * a.scal_ld + 112];  // cx
                    } else {
                        for (int q = 0; q < a.k; ++q)
                            if (a.I[(long long)t * a.k + q] == i) j = q;
                        for (int q = 0; q < a.G; ++q) h[q] = a.hpre[((long long)t * a.G + q) * a.N + i];
                        sa = a.scal[(long long)t * a.scal_ld + 0];
                        sb = a.scal[(long long)t * a.scal_ld + 1];
                    }
                }
                float* m = meta + lane * 8;
                m[0] = __int_as_float(j); m[1] = h[0]; m[2] = h[1]; m[3] = h[2]; m[4] = h[3];
                m[5] = sa; m[6] = sb;
            }
            __syncwarp();
            const uint32_t tl = tmem + (uint32_t)(s * DX_BN) + ((uint32_t)(quarter * 32) << 16);
            bool ok = true;
#pragma unroll 1
            for (int hh = 0; hh < 2; ++hh) {
                const int cg = chalf * 2 + hh;     // column group of 32
                // 4 passes of 8 rows; lane -> row rr = 8 pass + lane / 4, channels 8 (lane % 4)..
                const int cq = (lane & 3) * 8;
                const int c = ct * DX_BN + cg * 32 + cq;
                uint4 xr[4], br[4], br2[4], gr[4];
                auto load_pass = [&](int pass) {
                    const int rr = pass * 8 + (lane >> 2);
                    const int t = tt * BM + quarter * 32 + rr;
                    xr[pass] = make_uint4(0, 0, 0, 0);
                    br[pass] = xr[pass];
                    br2[pass] = xr[pass];
                    gr[pass] = xr[pass];
                    if (t >= a.T) return;
                    if (ACT) {
                        const long long row = ((long long)t * a.k + i) * a.C + c;
                        br[pass] = ld_stream(a.dxa + row);
                        br2[pass] = ld_stream(a.dxa + row + 4);
                        gr[pass] = ld_stream(a.dinput + (long long)t * a.C + c);
                        xr[pass] = ld_stream(a.X + row);
                    } else {
                        const int j = __float_as_int(meta[rr * 8]);
                        const long long off = ((long long)t * a.N + i) * a.C + c;
                        xr[pass] = ld_stream(a.X + off);
                        if (j >= 0) {
                            const float* bp = a.dxact + ((long long)t * a.k + j) * a.C + c;
                            br[pass] = ld_stream(bp);
                            br2[pass] = ld_stream(bp + 4);
                        } else {
                            br[pass] = ld_stream(a.dX + off);
                        }
                    }
                };
                // all four passes' reads are issued before the accumulator is awaited and read
                // out (8 columns at a time, few registers live next to the 64 of the reads)
                load_pass(0);
                load_pass(1);
                load_pass(2);
                load_pass(3);
                if (hh == 0) {
                    // one decision per warp (the TMEM reads and the shuffles below are warp-wide)
                    if (!__all_sync(0xffffffffu, mbar_wait(smem_u32(&bars[4 + s]), (uint32_t)((n >> 1) & 1), a.wait_ns))) {
                        atomicExch(a.err, 14);
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                }
#pragma unroll
                for (int q8 = 0; q8 < 4; ++q8) {
                    float acc[8];
                    tmem_ld8(tl + (uint32_t)(cg * 32 + q8 * 8), acc);
#pragma unroll
                    for (int e = 0; e < 8; ++e) tileb[lane * 33 + q8 * 8 + e] = acc[e];
                }
                if (hh == 1) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(smem_u32(&bars[6 + s]));  // TMEM buffer free
                }
                __syncwarp();
#pragma unroll
                for (int pass = 0; pass < 4; ++pass) {
                    const int rr = pass * 8 + (lane >> 2);
                    const int t = tt * BM + quarter * 32 + rr;
                    const bool live = t < a.T;    // the same for the 4 lanes of a row
                    if (!ACT && !live) continue;
                    const float* m = meta + rr * 8;
                    const float* ac = tileb + rr * 33 + cq;
                    float x[8], v[8];
                    unpack8(xr[pass], x);
                    if (ACT) {
                        // dX_act[t][i][c..c+8) += acc + h din - cx x   (i = active slot here)
                        const float hq = m[1], cx = m[2];
                        float g[8];
                        unpack8(gr[pass], g);
                        v[0] = __uint_as_float(br[pass].x); v[1] = __uint_as_float(br[pass].y);
                        v[2] = __uint_as_float(br[pass].z); v[3] = __uint_as_float(br[pass].w);
                        v[4] = __uint_as_float(br2[pass].x); v[5] = __uint_as_float(br2[pass].y);
                        v[6] = __uint_as_float(br2[pass].z); v[7] = __uint_as_float(br2[pass].w);
                        float4 o0, o1;
                        o0.x = v[0] + ac[0] + (hq * g[0] - cx * x[0]);
                        o0.y = v[1] + ac[1] + (hq * g[1] - cx * x[1]);
                        o0.z = v[2] + ac[2] + (hq * g[2] - cx * x[2]);
                        o0.w = v[3] + ac[3] + (hq * g[3] - cx * x[3]);
                        o1.x = v[4] + ac[4] + (hq * g[4] - cx * x[4]);
                        o1.y = v[5] + ac[5] + (hq * g[5] - cx * x[5]);
                        o1.z = v[6] + ac[6] + (hq * g[6] - cx * x[6]);
                        o1.w = v[7] + ac[7] + (hq * g[7] - cx * x[7]);
                        // dH_pre of stream I_i: <x_act_i, d_input>, this lane's 8 channels, then
                        // the row's 32 (4 lanes); rows past T hold zeros
                        float dp = x[0] * g[0];
#pragma unroll
                        for (int e = 1; e < 8; ++e) dp = fmaf(x[e], g[e], dp);
                        if (live) {
                            float4* dst = reinterpret_cast<float4*>(a.dxa + ((long long)t * a.k + i) * a.C + c);
                            dst[0] = o0;
                            dst[1] = o1;
                            if (i == 0)
                                *reinterpret_cast<uint4*>(a.dcopy + ((long long)a.slot * a.T + t) * a.C + c) = gr[pass];
                        }
                        dp += __shfl_xor_sync(0xffffffffu, dp, 1);
                        dp += __shfl_xor_sync(0xffffffffu, dp, 2);
                        if (live && (lane & 3) == 0)
                            a.dotp[((long long)i * a.ncg + ct * (DX_BN / 32) + cg) * a.T + t] = dp;
                    } else {
                        const int j = __float_as_int(m[0]);
                        const long long off = ((long long)t * a.N + i) * a.C + c;
                        if (j >= 0) {
                            v[0] = __uint_as_float(br[pass].x); v[1] = __uint_as_float(br[pass].y);
                            v[2] = __uint_as_float(br[pass].z); v[3] = __uint_as_float(br[pass].w);
                            v[4] = __uint_as_float(br2[pass].x); v[5] = __uint_as_float(br2[pass].y);
                            v[6] = __uint_as_float(br2[pass].z); v[7] = __uint_as_float(br2[pass].w);
                        } else {
                            unpack8(br[pass], v);
                        }
                        const float sa = m[5], sb = m[6];
                        float o[8];
#pragma unroll
                        for (int e = 0; e < 8; ++e) o[e] = v[e] + ac[e] + sa + sb * x[e];
                        *reinterpret_cast<uint4*>(a.dX + off) = pack8(o);
                    }
                }
                __syncwarp();
            }
            if (!ok) break;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(256u)
                     : "memory");
    }
}

// ---------------------------------------------------------------------------------------------
// TMA store, bulk-group and proxy-fence helpers of the full-state dX kernel below, and a named
// barrier that also ORs a flag over the participating threads.

__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, uint32_t src, int x, int y) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                     (uint64_t)map), "r"(src), "r"(x), "r"(y)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read0() {
    asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait0() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void fence_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// named barrier over `nthreads` threads that also returns, to every one of them, the OR of `p`
__device__ __forceinline__ bool named_bar_or(int id, int nthreads, bool p) {
    uint32_t r;
    asm volatile(
        "{\n .reg .pred a, b;\n setp.ne.u32 a, %3, 0;\n"
        " barrier.red.or.pred b, %1, %2, a;\n selp.u32 %0, 1, 0, b;\n}\n"
        : "=r"(r) : "r"(id), "r"(nthreads), "r"((uint32_t)p) : "memory");
    return r != 0;
}

constexpr int DG_BN = 64;                    // channels of a full-state dX tile
constexpr int DG_TILE = BM * DG_BN * 2;      // one 128 x 64 bf16 box, 16 KB
constexpr int DG_PF = 4;                     // L2 prefetch distance of the X / dX tiles, in tiles

// Full-state dX, grouped by column block: a block is 128 tokens x 64 channels; its N stream tiles
// are processed in turn by one CTA, which stages the G d_input rows of the block in shared memory
// once for all of them (the dense-read gradient of the non-active rows).  Streams m..N-1 come
// first and the fixed (always active, no d_input) streams 0..m-1 last, so the d_input buffer is
// released, and the next block's rows loaded, while the last tiles of a block are finished.
// Per tile: MMA 128 x 64 x nfull (A = the block's dZ rows, B = the stream's W rows), TMA-staged X
// and dX tiles, the result written over the X tile and TMA-stored into dX.
__global__ void __launch_bounds__(DX_THREADS, 1)
k_dxf_tc(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
         const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmD,
         const __grid_constant__ CUtensorMap tmG, DxArgs a) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    // aligned through an integer, so the epilogue's shared-memory accesses are generic ones: measured
    // 1.3 % faster for this kernel than the shared-window pointer the other two kernels use
    unsigned char* smem = (unsigned char*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const uint32_t A_BYTES = (uint32_t)a.nkb * BM * BK * 2;      // dZ rows of the token tile
    const uint32_t B_BYTES = (uint32_t)a.nkb * DG_BN * BK * 2;   // W rows of one stream's block
    unsigned char* sA = smem;
    unsigned char* sB = sA + A_BYTES;                // [2 stages]
    unsigned char* sG = sB + 2 * B_BYTES;            // [G][128 tokens][64 channels]
    unsigned char* sE = sG + (size_t)a.G * DG_TILE;  // [2 groups][X tile | dX tile]
    uint64_t* bars = reinterpret_cast<uint64_t*>(sE + 2 * 2 * DG_TILE);
    // [0] A full [1] A empty [2,4) B full [4,6) B empty [6] G full [7] G empty
    // [8,10) TMEM full [10,12) TMEM empty [12,14) epi full [14,16) epi empty
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 16);
    volatile int* s_abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        *s_abort = 0;
        mbar_init(smem_u32(&bars[0]), 1);
        mbar_init(smem_u32(&bars[1]), 1);
        mbar_init(smem_u32(&bars[6]), 1);
        mbar_init(smem_u32(&bars[7]), 2);
        for (int g = 0; g < 2; ++g) {
            mbar_init(smem_u32(&bars[2 + g]), 1);
            mbar_init(smem_u32(&bars[4 + g]), 1);
            mbar_init(smem_u32(&bars[8 + g]), 1);
            mbar_init(smem_u32(&bars[10 + g]), DX_EW / 2);
            mbar_init(smem_u32(&bars[12 + g]), 1);
            mbar_init(smem_u32(&bars[14 + g]), 1);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)), "r"(128u) : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const int N = a.N;
    const int ndin = N - a.m;   // leading tiles of a block that may read d_input (streams m..N-1)
    const int nblk = (a.ntiles > blockIdx.x) ? (int)((a.ntiles - 1 - blockIdx.x) / a.P) + 1 : 0;
    const int nloc = nblk * N;   // < 2^31: the host checks ntiles * N
    // local tile n: block n / N of this CTA, position p in the block, stream (p + m) mod N
    // (32-bit arithmetic: the divisions run per tile in every role)
    auto decode = [&](int n, int& p, int& tt, int& cb, int& i) {
        const int b = n / N;
        p = n - b * N;
        const int block = (int)blockIdx.x + b * a.P;
        tt = block / a.CT;
        cb = block - tt * a.CT;
        i = p + a.m;
        if (i >= N) i -= N;
    };

    if (warp == 0) {
        if (lane == 0) {
            for (int n = 0; n < nloc; ++n) {
                if (*s_abort) break;
                int p, tt, cb, i;
                if (DG_PF > 0 && n + DG_PF < nloc) {
                    // the tile DG_PF ahead into L2: its X / dX loads, issued once a stage frees,
                    // then wait for L2 rather than HBM
                    decode(n + DG_PF, p, tt, cb, i);
                    tma_prefetch_2d(&tmX, i * a.C + cb * DG_BN, tt * BM);
                    if (p < ndin) tma_prefetch_2d(&tmD, i * a.C + cb * DG_BN, tt * BM);
                    if (p == 0)
                        for (int q = 0; q < a.G; ++q) tma_prefetch_2d(&tmG, cb * DG_BN, q * a.T + tt * BM);
                }
                decode(n, p, tt, cb, i);
                const int blk = n / N;
                if (p == 0) {
                    if (blk >= 1 && !mbar_wait(smem_u32(&bars[1]), (uint32_t)((blk - 1) & 1), a.wait_ns)) {
                        atomicExch(a.err, 31);
                        *s_abort = 1;
                        break;
                    }
                    const uint32_t fa = smem_u32(&bars[0]);
                    mbar_expect_tx(fa, A_BYTES);
                    for (int kb = 0; kb < a.nkb; ++kb)
                        tma_load_2d(smem_u32(sA + kb * BM * BK * 2), &tmA, kb * BK, tt * BM, fa);
                }
                const int s = (int)(n & 1);
                if (n >= 2 && !mbar_wait(smem_u32(&bars[4 + s]), (uint32_t)(((n >> 1) - 1) & 1), a.wait_ns)) {
                    atomicExch(a.err, 32);
                    *s_abort = 1;
                    break;
                }
                const uint32_t fb = smem_u32(&bars[2 + s]);
                mbar_expect_tx(fb, B_BYTES);
                for (int kb = 0; kb < a.nkb; ++kb)
                    tma_load_2d(smem_u32(sB + s * B_BYTES + kb * DG_BN * BK * 2), &tmB, kb * BK,
                                i * a.C + cb * DG_BN, fb);
                if (n >= 2 && !mbar_wait(smem_u32(&bars[14 + s]), (uint32_t)(((n >> 1) - 1) & 1), a.wait_ns)) {
                    atomicExch(a.err, 33);
                    *s_abort = 1;
                    break;
                }
                const bool need_dx = p < ndin;   // a fixed stream's tile: every row takes the fp32 base
                const uint32_t fe = smem_u32(&bars[12 + s]);
                mbar_expect_tx(fe, need_dx ? 2 * DG_TILE : DG_TILE);
                unsigned char* xt = sE + (size_t)s * 2 * DG_TILE;
                tma_load_2d(smem_u32(xt), &tmX, i * a.C + cb * DG_BN, tt * BM, fe);
                if (need_dx) tma_load_2d(smem_u32(xt + DG_TILE), &tmD, i * a.C + cb * DG_BN, tt * BM, fe);
                if (p == 0) {
                    if (blk >= 1 && !mbar_wait(smem_u32(&bars[7]), (uint32_t)((blk - 1) & 1), a.wait_ns)) {
                        atomicExch(a.err, 34);
                        *s_abort = 1;
                        break;
                    }
                    const uint32_t fg = smem_u32(&bars[6]);
                    mbar_expect_tx(fg, (uint32_t)a.G * DG_TILE);
                    for (int q = 0; q < a.G; ++q)
                        tma_load_2d(smem_u32(sG + q * DG_TILE), &tmG, cb * DG_BN, q * a.T + tt * BM, fg);
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(BM, DG_BN);
            for (int n = 0; n < nloc; ++n) {
                const int blk = n / N;
                const int p = n - blk * N;
                const int s = (int)(n & 1);
                bool ok = (p != 0) || mbar_wait(smem_u32(&bars[0]), (uint32_t)(blk & 1), a.wait_ns);
                ok = ok && mbar_wait(smem_u32(&bars[2 + s]), (uint32_t)((n >> 1) & 1), a.wait_ns);
                ok = ok && (n < 2 || mbar_wait(smem_u32(&bars[10 + s]), (uint32_t)(((n >> 1) - 1) & 1), a.wait_ns));
                if (!ok) {
                    atomicExch(a.err, 35);
                    *s_abort = 1;
                    break;
                }
                tc_fence_after();
                const uint32_t abase = smem_u32(sA);
                const uint32_t bbase = smem_u32(sB + s * B_BYTES);
                for (int ks = 0; ks < a.ksteps; ++ks) {
                    const int kb = ks >> 2, kk = ks & 3;
                    mma_bf16(tmem + (uint32_t)(s * DG_BN), sw128_desc(abase + kb * BM * BK * 2 + kk * 32),
                             sw128_desc(bbase + kb * DG_BN * BK * 2 + kk * 32), idesc, ks > 0 ? 1u : 0u);
                }
                mma_commit(smem_u32(&bars[4 + s]));              // B stage consumed
                mma_commit(smem_u32(&bars[8 + s]));              // accumulator ready
                if (p == N - 1) mma_commit(smem_u32(&bars[1]));  // the block's A rows consumed
            }
        }
    } else {
        // group g = tiles n = g mod 2 (TMEM buffer g, epilogue stage g); in the group, warp w owns
        // the TMEM lane quarter warp % 4 (rows) and the 32-channel half (w % 8) / 4
        const int ew = warp - 2;
        const int grp = ew >> 3;
        const int quarter = warp & 3;
        const int half = (ew & 7) >> 2;
        const int r = quarter * 32 + lane;          // tile row
        const bool leader = (ew & 7) == 0 && lane == 0;
        unsigned char* xt = sE + (size_t)grp * 2 * DG_TILE;
        unsigned char* xrow = xt + r * 128;                       // this row of the X tile
        const unsigned char* drow = xt + DG_TILE + r * 128;       // of the dX tile
        const unsigned char* grow = sG + r * 128;                 // of the d_input rows
        const int sw = r & 7;                                     // 128B swizzle
        bool stored = false;
        // this row's token data of the current block (the same for all N stream tiles of the
        // block): its active streams I[t][0..k) as bytes, and the two per-token scalars
        int cur_blk = -1;
        uint32_t ib[2] = {0xffffffffu, 0xffffffffu};
        float sa = 0.f, sb = 0.f;
        for (int n = grp; n < nloc; n += 2) {
            int p, tt, cb, i;
            decode(n, p, tt, cb, i);
            const int blk = n / N;
            const bool usesg = p < ndin;
            const int t = tt * BM + r;
            // the dense-read weights of this tile's rows: loads issued first, used after the waits
            float hq[4];
#pragma unroll
            for (int q = 0; q < 4; ++q)
                hq[q] = (a.dense && usesg && t < a.T && q < a.G) ? a.hpre[((long long)t * a.G + q) * N + i] : 0.f;
            if ((int)blk != cur_blk) {
                cur_blk = (int)blk;
                ib[0] = ib[1] = 0xffffffffu;
                sa = sb = 0.f;
                if (t < a.T) {
#pragma unroll
                    for (int q = 0; q < MAXK; ++q)
                        if (q < a.k) {
                            const uint32_t v = (uint32_t)a.I[(long long)t * a.k + q] & 0xffu;
                            ib[q >> 2] = (ib[q >> 2] & ~(0xffu << (8 * (q & 3)))) | (v << (8 * (q & 3)));
                        }
                    sa = a.scal[(long long)t * a.scal_ld + 0];
                    sb = a.scal[(long long)t * a.scal_ld + 1];
                }
            }
            int j = -1;
#pragma unroll
            for (int q = 0; q < MAXK; ++q)
                if (q < a.k && ((ib[q >> 2] >> (8 * (q & 3))) & 0xffu) == (uint32_t)i) j = q;
            const bool arow = (j >= 0) && (t < a.T);
            // an active row's fp32 base, 8 channels per chunk, read one chunk ahead (the first
            // before the waits)
            const float* brow = a.dxact + ((long long)t * a.k + (j < 0 ? 0 : j)) * a.C + cb * DG_BN + half * 32;
            uint4 pfa[2], pfb[2];
            auto prefetch = [&](int c4, uint4 (&dst)[2]) {
                if (arow) {
                    dst[0] = ld_stream(brow + c4 * 8);
                    dst[1] = ld_stream(brow + c4 * 8 + 4);
                }
            };
            prefetch(0, pfa);
            bool ok = mbar_wait(smem_u32(&bars[12 + grp]), (uint32_t)((n >> 1) & 1), a.wait_ns);
            ok = ok && mbar_wait(smem_u32(&bars[8 + grp]), (uint32_t)((n >> 1) & 1), a.wait_ns);
            ok = ok && (!usesg || mbar_wait(smem_u32(&bars[6]), (uint32_t)(blk & 1), a.wait_ns));
            if (!ok) {
                atomicExch(a.err, 36);
                *s_abort = 1;
            } else {
                tc_fence_after();
                const uint32_t tl = tmem + (uint32_t)(grp * DG_BN + half * 32) + ((uint32_t)(quarter * 32) << 16);
                // channel pairs in packed float2 arithmetic (the same roundings, in the same order,
                // as the per-channel form: one FFMA2 / FADD2 per pair)
                const float2 sa2 = make_float2(sa, sa), sb2 = make_float2(sb, sb);
                auto chunk = [&](int c4, const uint4 (&pf)[2]) {
                    float acc[8];
                    tmem_ld8(tl + (uint32_t)(c4 * 8), acc);
                    const int ph = ((half * 4 + c4) ^ sw) * 16;
                    float2 x[4], v[4];
                    unpack4x2(*reinterpret_cast<const uint4*>(xrow + ph), x);
                    if (arow) {
                        v[0] = make_float2(__uint_as_float(pf[0].x), __uint_as_float(pf[0].y));
                        v[1] = make_float2(__uint_as_float(pf[0].z), __uint_as_float(pf[0].w));
                        v[2] = make_float2(__uint_as_float(pf[1].x), __uint_as_float(pf[1].y));
                        v[3] = make_float2(__uint_as_float(pf[1].z), __uint_as_float(pf[1].w));
                    } else {
                        unpack4x2(*reinterpret_cast<const uint4*>(drow + ph), v);
                        if (usesg) {
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                if (q < a.G) {
                                    float2 g[4];
                                    unpack4x2(*reinterpret_cast<const uint4*>(grow + q * DG_TILE + ph), g);
                                    const float2 h2 = make_float2(hq[q], hq[q]);
#pragma unroll
                                    for (int e = 0; e < 4; ++e) v[e] = __ffma2_rn(h2, g[e], v[e]);
                                }
                            }
                        }
                    }
                    uint4 o;
                    uint32_t* ow = reinterpret_cast<uint32_t*>(&o);
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float2 s = __fadd2_rn(__fadd2_rn(v[e], make_float2(acc[2 * e], acc[2 * e + 1])), sa2);
                        const float2 r2 = __ffma2_rn(sb2, x[e], s);
                        ow[e] = pack2(r2.x, r2.y);
                    }
                    *reinterpret_cast<uint4*>(xrow + ph) = o;
                };
                prefetch(1, pfb);
                chunk(0, pfa);
                prefetch(2, pfa);
                chunk(1, pfb);
                prefetch(3, pfb);
                chunk(2, pfa);
                chunk(3, pfb);
                tc_fence_before();
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&bars[10 + grp]));  // TMEM buffer free
            fence_async_smem();                                      // results visible to TMA
            if (named_bar_or(1 + grp, (DX_EW / 2) * 32, *s_abort != 0)) break;  // same decision in the group
            if (leader) {
                // the group's last reader of this block's d_input rows (or, when it has none of the
                // block's d_input tiles, its first tile of the block) releases them: one arrival
                // per group and block
                if ((usesg && p + 2 >= ndin) || (!usesg && p < 2)) mbar_arrive(smem_u32(&bars[7]));
                tma_store_2d(&tmD, smem_u32(xt), i * a.C + cb * DG_BN, tt * BM);
                bulk_commit();
                bulk_wait_read0();                                   // the stage may be reloaded
                mbar_arrive(smem_u32(&bars[14 + grp]));
                stored = true;
            }
        }
        if (leader && stored) bulk_wait0();
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(128u)
                     : "memory");
    }
}

// bf16 copies with a padded row stride: dst[r][o] = src[r][o] (o < n), 0 for n <= o < ld
__global__ void k_pack_rows(WSegs W, int n, int rows, int ld, uint16_t* __restrict__ dst) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)rows * ld) return;
    const int r = (int)(idx / ld), o = (int)(idx - (long long)r * ld);
    float v = 0.f;
    if (o < n) v = seg_elem(W, r, o);
    dst[idx] = __bfloat16_as_ushort(__float2bfloat16_rn(v));
}

// rows of three bf16 parts along K: A rows [hi | lo | hi] of dz, B rows [hi | hi | lo] of W, so
// that sum_k A B = dz_hi W_hi + dz_lo W_hi + dz_hi W_lo (~2^-16 relative)
__global__ void k_pack3(WSegs W, int n, int rows, int ld, int lo_part, uint16_t* __restrict__ dst) {
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (long long)rows * ld) return;
    const int r = (int)(idx / ld), col = (int)(idx - (long long)r * ld);
    float v = 0.f;
    if (col < 3 * n) {
        const int part = col / n, o = col - part * n;
        const float w = seg_elem(W, r, o);
        const float hi = __bfloat162float(__float2bfloat16_rn(w));
        v = (part == lo_part) ? (w - hi) : hi;
    }
    dst[idx] = __bfloat16_as_ushort(__float2bfloat16_rn(v));
}

}  // namespace

// two operand stages of up to two k-blocks each fit the 227 KB of shared memory
bool dxa_tc_ok(int T, int k, int C, int nact) {
    return T >= BM && C % DX_BN == 0 && 3 * nact <= 2 * BK &&
           (long long)((T + BM - 1) / BM) * (C / DX_BN) * k < (1LL << 31);   // 32-bit tile indices
}

cudaError_t launch_dxa_tc(const Dims& d, int slot, int T, const float* dzs, int nact, const WSegs& W,
                          uint16_t* dz3, uint16_t* w3, const uint16_t* d_input, const float* hpre,
                          const int* I, const uint16_t* xact, const float* tokmat, float* dxact,
                          float* dotp, uint16_t* dcopy, int* err, cudaStream_t st) {
    const int KC = d.k * d.C;
    const int K3 = 3 * nact;
    const int ld = (K3 + 7) / 8 * 8;
    WSegs dzsg;
    memset(&dzsg, 0, sizeof(dzsg));
    dzsg.ptr[0] = dzs; dzsg.width[0] = nact; dzsg.off[0] = 0; dzsg.off[1] = nact; dzsg.n = 1;
    long long tot = (long long)T * ld;
    k_pack3<<<(unsigned)((tot + 255) / 256), 256, 0, st>>>(dzsg, nact, T, ld, 1, dz3); note_launch();
    tot = (long long)KC * ld;
    k_pack3<<<(unsigned)((tot + 255) / 256), 256, 0, st>>>(W, nact, KC, ld, 2, w3); note_launch();
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    CUtensorMap ma, mb;
    if (!make_map_box(&ma, dz3, (uint64_t)K3, (uint64_t)T, BK, BM, (uint64_t)ld * 2)) return cudaErrorInvalidValue;
    if (!make_map_box(&mb, w3, (uint64_t)K3, (uint64_t)KC, BK, DX_BN, (uint64_t)ld * 2)) return cudaErrorInvalidValue;
    DxArgs a;
    memset(&a, 0, sizeof(a));
    a.T = T; a.C = d.C; a.N = d.N; a.k = d.k; a.G = d.G; a.slot = slot;
    a.nkb = (K3 + BK - 1) / BK;
    a.ksteps = (K3 + 15) / 16;
    a.TT = (T + BM - 1) / BM;
    a.CT = d.C / DX_BN;
    a.ntiles = (long long)a.TT * a.CT * d.k;
    a.P = (int)std::min<long long>(num_sms(), a.ntiles);
    a.N = d.k;  // tile "streams" are the active slots
    a.NH = d.N;
    a.dinput = d_input; a.hpre = hpre; a.I = I; a.dxa = dxact; a.err = err;
    a.wait_ns = debug_wait_ns();
    a.X = xact; a.scal = tokmat; a.scal_ld = TOKMAT;
    a.dotp = dotp; a.dcopy = dcopy; a.ncg = d.C / 32;
    // one operand stage (the MMA of a tile is short next to its epilogue): the shared memory
    // left over is L1 for the epilogue's in-flight reads
    a.ns = 1;
    const size_t sm = (size_t)a.ns * a.nkb * (BM + DX_BN) * BK * 2 + 128 +
                      (size_t)DX_EW * (32 * 33 + 32 * 8) * 4 + 1024;
    e = cudaFuncSetAttribute((const void*)k_dx_tc<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    k_dx_tc<true><<<a.P, DX_THREADS, sm, st>>>(ma, mb, a); note_launch();
    return cudaGetLastError();
}

namespace {
// dH_pre[t][slot][I_j] from the dot partials of k_dx_tc<true>: a block per (32 tokens, j); warp w
// sums the groups g = w, w + 8, ... of its lane's token (coalesced 128-byte rows), and the eight
// warp sums are added in warp order (a fixed order: the result does not depend on the schedule)
__global__ void __launch_bounds__(256) k_dots_act(const float* __restrict__ dotp, int T, int k, int ncg,
                                                  int G, int N, int slot, const int* __restrict__ I,
                                                  float* __restrict__ dhpre) {
    __shared__ float part[8][32];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int j = blockIdx.y, t = blockIdx.x * 32 + lane;
    float s = 0.f;
    if (t < T) {
        const float* p = dotp + (long long)j * ncg * T + t;
        for (int g = w; g < ncg; g += 8) s += p[(long long)g * T];
    }
    part[w][lane] = s;
    __syncthreads();
    if (w == 0 && t < T) {
        float v = part[0][lane];
#pragma unroll
        for (int q = 1; q < 8; ++q) v += part[q][lane];
        dhpre[((long long)t * G + slot) * N + I[(long long)t * k + j]] = v;
    }
}
}  // namespace

cudaError_t launch_dots_act(const Dims& d, int slot, int T, const float* dotp, const int* I, float* dhpre,
                            cudaStream_t st) {
    const dim3 grid((unsigned)((T + 31) / 32), (unsigned)d.k);
    k_dots_act<<<grid, 256, 0, st>>>(dotp, T, d.k, d.C / 32, d.G, d.N, slot, I, dhpre);
    note_launch();
    return cudaGetLastError();
}

// shared memory of k_dxf_tc: the token tile's dZ rows and two stages of W rows (nkb k-blocks
// each), the G d_input tiles and two X | dX tile pairs, barriers, alignment slack
static size_t dxf_smem(int nfull, int G) {
    const int nkb = (nfull + BK - 1) / BK;
    return (size_t)nkb * (BM + 2 * DG_BN) * BK * 2 + (size_t)(G + 4) * DG_TILE + 256 + 1024;
}

// up to three k-blocks (nfull <= 192: N = 32 with a router and four pre-maps) fit the 227 KB a
// block may use
bool dx_tc_ok(int T, int N, int C, int nfull, int G) {
    return T >= BM && C % DG_BN == 0 && nfull <= 3 * BK && N >= 2 && G >= 1 && G <= 4 &&
           dxf_smem(nfull, G) <= 232448 &&
           (long long)((T + BM - 1) / BM) * (C / DG_BN) * N < (1LL << 31);   // 32-bit tile indices
}

cudaError_t launch_dx_tc(const Dims& d, int T, const float* dz, const WSegs& W, uint16_t* dz16,
                         uint16_t* w16, const uint16_t* X, const uint16_t* dinput, const float* hpre,
                         const int* I, const float* dxact, const float* scal, int scal_ld,
                         uint16_t* dX, int* err, cudaStream_t st) {
    const int n = d.nfull, NC = d.N * d.C;
    const int ld = (n + 7) / 8 * 8;
    WSegs dzs;
    memset(&dzs, 0, sizeof(dzs));
    dzs.ptr[0] = dz; dzs.width[0] = n; dzs.off[0] = 0; dzs.off[1] = n; dzs.n = 1;
    long long tot = (long long)T * ld;
    k_pack_rows<<<(unsigned)((tot + 255) / 256), 256, 0, st>>>(dzs, n, T, ld, dz16); note_launch();
    tot = (long long)NC * ld;
    k_pack_rows<<<(unsigned)((tot + 255) / 256), 256, 0, st>>>(W, n, NC, ld, w16); note_launch();
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    CUtensorMap ma, mb, mx, md, mg;
    if (!make_map_box(&ma, dz16, (uint64_t)n, (uint64_t)T, BK, BM, (uint64_t)ld * 2)) return cudaErrorInvalidValue;
    if (!make_map_box(&mb, w16, (uint64_t)n, (uint64_t)NC, BK, DG_BN, (uint64_t)ld * 2)) return cudaErrorInvalidValue;
    if (!make_map_box(&mx, X, (uint64_t)NC, (uint64_t)T, DG_BN, BM)) return cudaErrorInvalidValue;
    if (!make_map_box(&md, dX, (uint64_t)NC, (uint64_t)T, DG_BN, BM)) return cudaErrorInvalidValue;
    // the G d_input copies [G][T][C] as one [G T][C] matrix (rows of a token tile past T read the
    // next copy's rows or zeros; those rows are never stored)
    if (!make_map_box(&mg, dinput, (uint64_t)d.C, (uint64_t)d.G * T, DG_BN, BM)) return cudaErrorInvalidValue;
    DxArgs a;
    memset(&a, 0, sizeof(a));
    a.T = T; a.C = d.C; a.N = d.N; a.k = d.k; a.G = d.G; a.m = d.m; a.dense = d.dense;
    a.nkb = (n + BK - 1) / BK;
    a.ksteps = (n + 15) / 16;
    a.TT = (T + BM - 1) / BM;
    a.CT = d.C / DG_BN;
    a.ntiles = (long long)a.TT * a.CT;   // column blocks, N tiles each
    a.P = (int)std::min<long long>(num_sms(), a.ntiles);
    a.X = X; a.dX = dX; a.dinput = dinput; a.hpre = hpre; a.I = I; a.dxact = dxact;
    a.scal = scal; a.scal_ld = scal_ld; a.err = err;
    a.wait_ns = debug_wait_ns();
    const size_t sm = dxf_smem(n, d.G);
    e = cudaFuncSetAttribute((const void*)k_dxf_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    k_dxf_tc<<<a.P, DX_THREADS, sm, st>>>(ma, mb, mx, md, mg, a); note_launch();
    return cudaGetLastError();
}

}  // namespace xhc
