// Write-back kernels of the connection op with the causal conv held in registers.
//
// Every kernel here walks a run of consecutive tokens for one pair of channels per thread.  The
// conv taps of the pair and a ring of the recent values of `out` stay in registers, indexed by
// compile-time positions: wb_gram unrolls the token loop by KW over a KW-slot ring; the forward
// apply and the backward kernels unroll it by 4-token blocks over a ring of KW + 3 slots that
// moves by 4 after each block (a shorter loop body: the 12-token one overflowed the instruction
// cache).  Each out value is loaded once per run instead of once per tap.  Runs never cross a sequence boundary (Sec.
// 3.3.4: the conv restarts with every sequence), so the conv needs no per-tap test.  KS = 1
// specialises the tap counts to the (4, 8, 12) kernels of the MLP sublayers, so no FMA is spent
// on zero taps.  Per-token reductions over the channels use a reduce-scatter butterfly inside
// the warp (about V shuffles for V values instead of 5 V), then shared memory across warps.
//   wb_gram   Gram matrix of u = [out, g_1..g_r] (Eq. aug, Eq. gs), partial per channel slice
//   wb_coef   per token: Gram-Schmidt coefficients (Eq. gs) folded with p and H_post into
//             E[j][a]; keeps the token's Gram matrix for the backward
//   wb_fwd    X_act_new = (H_res) X_act + sum_a E[j][a] u_a (Eq. sparse_write_delta,
//             Eq. sparse_write), scatter into X on the last slot
//   wb_bred   backward reductions <dXn_j, u_a> and, on the last slot, <dXn_j, x_i>
//   wb_bapp   component gradients du_a consumed on the fly: d_out = du_0 + conv^T(du_1..r)
//             (emitted KW - 1 tokens late), conv weight-gradient partials, and on the last slot
//             the mixed active-state gradient H_res^T dXn
//   wb_fwd8, wb_b8   the same for slots without conv (K = 1), 8 channels per thread; wb_b8 does
//             the backward reductions and apply in one pass
#pragma once
#include "xhc_internal.cuh"

namespace xhc {
namespace {

constexpr int WT = 128;        // threads per CTA
constexpr int WSL = 2 * WT;    // channels per CTA slice
constexpr unsigned FULLM = 0xffffffffu;

__device__ __forceinline__ float2 ld2(const uint16_t* p) {
    const uint32_t u = *reinterpret_cast<const uint32_t*>(p);
    return make_float2(__uint_as_float(u << 16), __uint_as_float(u & 0xffff0000u));
}
__device__ __forceinline__ void st2(uint16_t* p, float2 v) {
    *reinterpret_cast<uint32_t*>(p) = pack2(v.x, v.y);
}
__device__ __forceinline__ float dot2(float2 a, float2 b) { return fmaf(a.x, b.x, a.y * b.y); }
__device__ __forceinline__ float2 fma2(float s, float2 a, float2 acc) {
    return __ffma2_rn(make_float2(s, s), a, acc);
}
// the same as two scalar FMAs (measured faster in the backward apply, where the packed form
// lengthens the schedule)
__device__ __forceinline__ float2 fma2s(float s, float2 a, float2 acc) {
    return make_float2(fmaf(s, a.x, acc.x), fmaf(s, a.y, acc.y));
}
__device__ __forceinline__ float2 f2z() { return make_float2(0.f, 0.f); }
// a * b + c on both channels of a pair in one packed instruction (each lane rounded as fmaf)
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) { return __ffma2_rn(a, b, c); }
__device__ __forceinline__ uint32_t s_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

// Per-thread prefetch of the next tokens' values with cp.async into a PD-slot ring in shared
// memory (field-major [slot][field][thread], so a warp's accesses are consecutive words).
constexpr int PD = 4;
__device__ __forceinline__ void cpa4(void* dst, const void* src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(s_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cpa8(void* dst, const void* src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(s_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cpa16(void* dst, const void* src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(s_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cpa_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cpa_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }
__device__ __forceinline__ float2 u2f2(uint32_t u) {
    return make_float2(__uint_as_float(u << 16), __uint_as_float(u & 0xffff0000u));
}

// Runs of tokens: with a conv (KW > 0) every run lies inside one sequence (runs of TB tokens
// from each sequence start, the last one shorter), so a conv window never crosses a run's
// sequence boundary except at the run start; without a conv, runs of TB tokens.
template <int KW>
__device__ __forceinline__ void run_bounds(const Dims& d, int T, int TB, long long& t0, long long& t1,
                                           long long& send, int& pos0) {
    if constexpr (KW == 0) {
        t0 = (long long)blockIdx.y * TB;
        t1 = min((long long)T, t0 + TB);
        send = t1;
        pos0 = 0;
    } else {
        const int rps = (d.S + TB - 1) / TB;
        const long long seq = blockIdx.y / rps;
        const int r = (int)(blockIdx.y - seq * rps);
        const long long s0 = seq * d.S;
        send = min((long long)T, s0 + d.S);
        pos0 = r * TB;
        t0 = s0 + pos0;
        t1 = min(send, t0 + TB);
    }
}

// Kernel variants: KS = 0 generic; KS = 1 the (4, 8, 12) kernel set of the MLP sublayers (taps
// of component j held in registers: 4, 8, 12, else KW each); KS = 2 as KS = 1 (or no conv) with,
// in addition, k equal to the compile-time KM and every thread of a channel slice in range, so
// that the loops over active slots and the range tests fold away.
template <int KW, int KS>
__host__ __device__ constexpr int ntap(int j) {
    return KS >= 1 ? (j == 0 ? 4 : (j == 1 ? 8 : 12)) : KW;
}

template <int KW, int KS>
__device__ __forceinline__ void taps_reg(const Dims& d, const ConvPtrs& cw, int c, bool act,
                                         float2 (&tw)[3][KW]) {
#pragma unroll
    for (int j = 0; j < 3; ++j)
#pragma unroll
        for (int i = 0; i < KW; ++i) {
            float2 v = f2z();
            if (i < ntap<KW, KS>(j) && act && j < d.nconv && i < d.kap[j])
                v = make_float2(cw.w[j][(size_t)i * d.C + c], cw.w[j][(size_t)i * d.C + c + 1]);
            tw[j][i] = v;
        }
}

// ring w[s] = out[t] for t - t0 = s (mod KW); prepares the run starting at t0, whose position in
// its sequence is pos0: values before the sequence start come from the call's halo rows of the
// sequence (the previous chunk's last outputs), or are zero without a halo
template <int KW>
__device__ __forceinline__ void ring_init(const Dims& d, const ConvPtrs& cw, const uint16_t* out, int c,
                                          bool act, long long t0, int pos0, float2 (&w)[KW]) {
    const int C = d.C, R = d.kapmax - 1;
    const long long seq = (t0 - pos0) / d.S;
    w[0] = f2z();
#pragma unroll
    for (int i = 1; i < KW; ++i) {
        float2 v = f2z();
        if (act && i <= pos0) {
            v = ld2(out + (t0 - i) * C + c);
        } else if (act && cw.halo != nullptr) {
            const int r = R + pos0 - i;   // halo row of position pos0 - i < 0
            if (r >= 0) v = ld2(cw.halo + (seq * R + r) * C + c);
        }
        w[KW - i] = v;
    }
}

// g_j = sum_i tw[j][i] out[t - i], with out[t - i] at ring slot (U - i) mod KW
template <int KW, int KS>
__device__ __forceinline__ void conv_ring(const float2 (&tw)[3][KW], const float2 (&w)[KW], int U,
                                          float2 (&g)[3]) {
#pragma unroll
    for (int j = 0; j < 3; ++j) g[j] = f2z();
#pragma unroll
    for (int i = 0; i < KW; ++i) {
        const float2 o = w[(U - i + KW) % KW];
#pragma unroll
        for (int j = 0; j < 3; ++j) {
            if (i >= ntap<KW, KS>(j)) continue;
            g[j] = ffma2(tw[j][i], o, g[j]);
        }
    }
}

// Block ring of the forward write-back, the backward reductions and the backward apply: the
// token loop is unrolled by UB tokens only (a 12-token body does not fit the instruction cache),
// and the ring holds the KW + UB - 1 values a block needs: for the block of tokens tb..tb+UB-1,
// slot KW - 1 + u - i holds out[tb + u - i] (i < KW).  After a block the ring moves by UB slots.
constexpr int UB = 4;

template <int KW>
__device__ __forceinline__ void ring_init_b(const Dims& d, const ConvPtrs& cw, const uint16_t* out, int c,
                                            bool act, long long t0, int pos0, float2 (&w)[KW + UB - 1]) {
    const int C = d.C, R = d.kapmax - 1;
    const long long seq = (t0 - pos0) / d.S;
#pragma unroll
    for (int s = 0; s < KW + UB - 1; ++s) w[s] = f2z();
#pragma unroll
    for (int i = 1; i < KW; ++i) {
        float2 v = f2z();
        if (act && i <= pos0) {
            v = ld2(out + (t0 - i) * C + c);
        } else if (act && cw.halo != nullptr) {
            const int r = R + pos0 - i;   // halo row of position pos0 - i < 0
            if (r >= 0) v = ld2(cw.halo + (seq * R + r) * C + c);
        }
        w[KW - 1 - i] = v;
    }
}

// g_j = sum_i tw[j][i] out[t - i] for token t = tb + u of the block
template <int KW, int KS>
__device__ __forceinline__ void conv_blk(const float2 (&tw)[3][KW], const float2 (&w)[KW + UB - 1], int u,
                                         float2 (&g)[3]) {
#pragma unroll
    for (int j = 0; j < 3; ++j) g[j] = f2z();
#pragma unroll
    for (int i = 0; i < KW; ++i) {
        const float2 o = w[KW - 1 + u - i];
#pragma unroll
        for (int j = 0; j < 3; ++j) {
            if (i >= ntap<KW, KS>(j)) continue;
            g[j] = ffma2(tw[j][i], o, g[j]);
        }
    }
}

// move a block ring on by UB tokens
template <int KW>
__device__ __forceinline__ void ring_shift(float2 (&w)[KW + UB - 1]) {
#pragma unroll
    for (int q = 0; q + 1 < KW; ++q) w[q] = w[q + UB];
}

// Reduce-scatter of V values (power of two, <= 32) over the warp: every lane returns the total
// of value index lane >> (5 - log2 V).
template <int V, int O>
struct WRed {
    static __device__ __forceinline__ float run(float* v, int lane) {
        if constexpr (V > 1) {
            constexpr int H = V / 2;
            const bool up = (lane & O) != 0;
#pragma unroll
            for (int q = 0; q < H; ++q) {
                const float send = up ? v[q] : v[q + H];
                const float keep = up ? v[q + H] : v[q];
                v[q] = keep + __shfl_xor_sync(FULLM, send, O);
            }
            if constexpr (O > 1) return WRed<H, O / 2>::run(v, lane);
            else return v[0];
        } else {
            float x = v[0];
#pragma unroll
            for (int o = O; o >= 1; o >>= 1) x += __shfl_xor_sync(FULLM, x, o);
            return x;
        }
    }
};

// reduce NB blocks of 32 values; lane l receives the totals of values b*32 + l
template <int NB>
__device__ __forceinline__ void wred32(float (&v)[NB * 32], int lane, float (&tot)[NB]) {
#pragma unroll
    for (int b = 0; b < NB; ++b) tot[b] = WRed<32, 16>::run(v + 32 * b, lane);
}

// ---------------------------------------------------------------------------------------------
// wb_gram

template <int KW, int KS>
__global__ void __launch_bounds__(WT) k_wb_gram(Dims d, int slot, int T, int TB,
                                                const uint16_t* __restrict__ out, ConvPtrs cw,
                                                int nslice, float* __restrict__ red) {
    extern __shared__ float wsh[];  // [TB][WT/32][16]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int slice = blockIdx.x, C = d.C;
    const int c = slice * WSL + 2 * threadIdx.x;
    const bool act = (KS == 2) || c < C;
    long long t0, t1, send;
    int pos0;
    run_bounds<KW>(d, T, TB, t0, t1, send, pos0);
    const int n1 = (int)(t1 - t0);
    const int K = d.K[slot];
    const int nq = K * (K + 1) / 2;
    float2 tw[3][KW], w[KW];
    taps_reg<KW, KS>(d, cw, c, act, tw);
    ring_init<KW>(d, cw, out, c, act, t0, pos0, w);
    const uint16_t* po = out + t0 * C + c;
    // the out values of the next block of KW tokens are loaded while this block is processed
    uint32_t ob[KW];
#pragma unroll
    for (int u = 0; u < KW; ++u)
        ob[u] = (act && u < n1) ? *reinterpret_cast<const uint32_t*>(po + (long long)u * C) : 0u;
    for (int tb = 0; tb < n1; tb += KW) {
        uint32_t on[KW];
#pragma unroll
        for (int u = 0; u < KW; ++u) {
            const int tn = tb + KW + u;
            on[u] = (act && tn < n1) ? *reinterpret_cast<const uint32_t*>(po + (long long)tn * C) : 0u;
        }
#pragma unroll
        for (int u = 0; u < KW; ++u) {
            const int tt = tb + u;
            if (tt < n1) {
                const float2 o = u2f2(ob[u]);
                w[u] = o;
                float2 g[3];
                conv_ring<KW, KS>(tw, w, u, g);
                const float2 uu[4] = {o, g[0], g[1], g[2]};
                float v[16];
                int q = 0;
#pragma unroll
                for (int a = 0; a < 4; ++a)
#pragma unroll
                    for (int b = 0; b <= a; ++b) v[q++] = (a < K) ? dot2(uu[a], uu[b]) : 0.f;
#pragma unroll
                for (int r = 10; r < 16; ++r) v[r] = 0.f;
                const float tot = WRed<16, 16>::run(v, lane);
                if ((lane & 1) == 0) wsh[(tt * (WT / 32) + warp) * 16 + (lane >> 1)] = tot;
            }
        }
#pragma unroll
        for (int u = 0; u < KW; ++u) ob[u] = on[u];
    }
    __syncthreads();
    const int ntok = (int)(t1 - t0);
    for (int idx = threadIdx.x; idx < ntok * nq; idx += WT) {
        const int tt = idx / nq, q = idx - tt * nq;
        float s = 0.f;
#pragma unroll
        for (int ww = 0; ww < WT / 32; ++ww) s += wsh[(tt * (WT / 32) + ww) * 16 + q];
        red[((t0 + tt) * nslice + slice) * NRED + q] = s;
    }
}

// The Gram matrix with two channel pairs per thread (4 consecutive channels, WSL2 channels per
// CTA) and the 4-token block ring: a token's warp reduction covers 128 channels.  For the
// (4, 8, 12) tap set and C a multiple of 4 WT.
constexpr int WSL2 = 4 * WT;

__global__ void __launch_bounds__(WT, 2) k_wb_gram2(Dims d, int slot, int T, int TB,
                                                    const uint16_t* __restrict__ out, ConvPtrs cw,
                                                    int nslice, float* __restrict__ red) {
    constexpr int KW = 12, KS = 2;
    extern __shared__ float wsh[];  // [TB][WT/32][16]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int slice = blockIdx.x, C = d.C;
    const int c = slice * WSL2 + 4 * threadIdx.x;
    long long t0, t1, send;
    int pos0;
    run_bounds<KW>(d, T, TB, t0, t1, send, pos0);
    const int n1 = (int)(t1 - t0);
    const int K = d.K[slot];
    const int nq = K * (K + 1) / 2;
    float2 tw[2][3][KW], w[2][KW + UB - 1];
#pragma unroll
    for (int p = 0; p < 2; ++p) {
        taps_reg<KW, KS>(d, cw, c + 2 * p, true, tw[p]);
        ring_init_b<KW>(d, cw, out, c + 2 * p, true, t0, pos0, w[p]);
    }
    const uint16_t* po = out + t0 * C + c;
    // the out values of the next block of UB tokens are loaded while this block is processed
    uint2 ob[UB];
#pragma unroll
    for (int u = 0; u < UB; ++u)
        ob[u] = (u < n1) ? *reinterpret_cast<const uint2*>(po + (long long)u * C) : make_uint2(0u, 0u);
    for (int tb = 0; tb < n1; tb += UB) {
        uint2 on[UB];
#pragma unroll
        for (int u = 0; u < UB; ++u) {
            const int tn = tb + UB + u;
            on[u] = (tn < n1) ? *reinterpret_cast<const uint2*>(po + (long long)tn * C) : make_uint2(0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < UB; ++u) {
            const int tt = tb + u;
            if (tt < n1) {
                float2 uu[2][4];
#pragma unroll
                for (int p = 0; p < 2; ++p) {
                    const float2 o = u2f2(p == 0 ? ob[u].x : ob[u].y);
                    w[p][KW - 1 + u] = o;
                    float2 g[3];
                    conv_blk<KW, KS>(tw[p], w[p], u, g);
                    uu[p][0] = o;
                    uu[p][1] = g[0];
                    uu[p][2] = g[1];
                    uu[p][3] = g[2];
                }
                float v[16];
                int q = 0;
#pragma unroll
                for (int a = 0; a < 4; ++a)
#pragma unroll
                    for (int b = 0; b <= a; ++b)
                        v[q++] = (a < K) ? fmaf(uu[1][a].y, uu[1][b].y,
                                                fmaf(uu[1][a].x, uu[1][b].x, dot2(uu[0][a], uu[0][b])))
                                         : 0.f;
#pragma unroll
                for (int r = 10; r < 16; ++r) v[r] = 0.f;
                const float tot = WRed<16, 16>::run(v, lane);
                if ((lane & 1) == 0) wsh[(tt * (WT / 32) + warp) * 16 + (lane >> 1)] = tot;
            }
        }
#pragma unroll
        for (int p = 0; p < 2; ++p) ring_shift<KW>(w[p]);
#pragma unroll
        for (int u = 0; u < UB; ++u) ob[u] = on[u];
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < n1 * nq; idx += WT) {
        const int tt = idx / nq, q = idx - tt * nq;
        float s = 0.f;
#pragma unroll
        for (int ww = 0; ww < WT / 32; ++ww) s += wsh[(tt * (WT / 32) + ww) * 16 + q];
        red[((t0 + tt) * nslice + slice) * NRED + q] = s;
    }
}

// ---------------------------------------------------------------------------------------------
// wb_fwd: per-token coefficients E[j][a], H_res and I in shared memory; each thread prefetches
// the out value and the k active values of its channel pair PD - 1 tokens ahead with cp.async.

template <int KM>
struct FRing {
    uint32_t o[PD][WT];
    uint32_t x[PD][KM][WT];
};

template <int KM, int KW, int KS>
__global__ void __launch_bounds__(WT) k_wb_fwd(Dims d, int slot, int T, int TB,
                                               const uint16_t* __restrict__ out, ConvPtrs cw,
                                               const float* __restrict__ emat,
                                               const uint16_t* __restrict__ xact,
                                               const int* __restrict__ I,
                                               const float* __restrict__ hres,
                                               uint16_t* __restrict__ xact_next,
                                               uint16_t* __restrict__ X) {
    extern __shared__ __align__(16) unsigned char smu[];
    FRing<KM>& R = *reinterpret_cast<FRing<KM>*>(smu);
    const int k = (KS == 2) ? KM : d.k, C = d.C;
    const bool last = (slot == d.G - 1);
    float* Esh = reinterpret_cast<float*>(smu + sizeof(FRing<KM>));  // [TB][KM][4]
    float* Hsh = Esh + TB * KM * 4;                                 // [TB][KM][KM]
    int* Ish = reinterpret_cast<int*>(Hsh + TB * KM * KM);           // [TB][KM]
    long long t0, t1, send;
    int pos0;
    run_bounds<KW>(d, T, TB, t0, t1, send, pos0);
    const int ntok = (int)(t1 - t0);
    const int c = blockIdx.x * WSL + 2 * threadIdx.x;
    const bool act = (KS == 2) || c < C;
    // running pointers of the next token to prefetch (issue() is called once per token, in order)
    const uint16_t* po = out + t0 * C + c;
    const uint16_t* px = xact + t0 * k * C + c;
    const long long kC = (long long)k * C;
    auto issue = [&](int sl, int tn) {
        if (act && tn < ntok) {
            cpa4(&R.o[sl][threadIdx.x], po);
            const uint16_t* pj = px;
#pragma unroll
            for (int j = 0; j < KM; ++j) {
                if (j < k) cpa4(&R.x[sl][j][threadIdx.x], pj);
                pj += C;
            }
        }
        po += C;
        px += kC;
        cpa_commit();
    };
#pragma unroll
    for (int q = 0; q < PD - 1; ++q) issue(q, q);
    for (int idx = threadIdx.x; idx < ntok * KM * 4; idx += WT) {
        const int tt = idx / (KM * 4), q = idx - tt * (KM * 4);
        Esh[idx] = (q < k * 4) ? emat[(t0 + tt) * TOKMAT + q] : 0.f;
    }
    for (int idx = threadIdx.x; idx < ntok * KM * KM; idx += WT) {
        const int tt = idx / (KM * KM), q = idx - tt * (KM * KM);
        const int j = q / KM, i = q - j * KM;
        Hsh[idx] = (last && j < k && i < k) ? hres[(t0 + tt) * k * k + j * k + i] : 0.f;
    }
    for (int idx = threadIdx.x; idx < ntok * KM; idx += WT) {
        const int tt = idx / KM, j = idx - tt * KM;
        Ish[idx] = (j < k) ? I[(t0 + tt) * k + j] : 0;
    }
    float2 tw[3][KW > 0 ? KW : 1], w[KW > 0 ? KW + UB - 1 : 1];
    if constexpr (KW > 0) {
        taps_reg<KW, KS>(d, cw, c, act, tw);
        ring_init_b<KW>(d, cw, out, c, act, t0, pos0, w);
    }
    uint16_t* pX = X + t0 * d.N * C + c;                              // token rows, advanced per token
    uint16_t* pn = last ? nullptr : xact_next + t0 * k * C + c;
    const long long NC = (long long)d.N * C;
    __syncthreads();
    constexpr int RU = UB;
    for (int tb = 0; tb < ntok; tb += RU) {
#pragma unroll
        for (int u = 0; u < RU; ++u) {
            const int tt = tb + u;
            if (tt < ntok) {
                const int sl = u % PD;
                issue((u + PD - 1) % PD, tt + PD - 1);
                cpa_wait<PD - 1>();
                if (act) {
                    const float2 o = u2f2(R.o[sl][threadIdx.x]);
                    float2 uu[4] = {o, f2z(), f2z(), f2z()};
                    if constexpr (KW > 0) {
                        w[KW - 1 + u] = o;
                        float2 g[3];
                        conv_blk<KW, KS>(tw, w, u, g);
                        uu[1] = g[0];
                        uu[2] = g[1];
                        uu[3] = g[2];
                    }
                    float2 x[KM];
#pragma unroll
                    for (int j = 0; j < KM; ++j) x[j] = (j < k) ? u2f2(R.x[sl][j][threadIdx.x]) : f2z();
                    const float4* E4 = reinterpret_cast<const float4*>(Esh + tt * KM * 4);
                    const float4* H4 = reinterpret_cast<const float4*>(Hsh + tt * KM * KM);
#pragma unroll
                    for (int j = 0; j < KM; ++j) {
                        if (j >= k) continue;
                        float2 v;
                        if (last) {
                            v = f2z();
#pragma unroll
                            for (int q = 0; q < KM / 4; ++q) {
                                const float4 h = H4[j * (KM / 4) + q];
                                v = fma2(h.x, x[4 * q + 0], v);
                                v = fma2(h.y, x[4 * q + 1], v);
                                v = fma2(h.z, x[4 * q + 2], v);
                                v = fma2(h.w, x[4 * q + 3], v);
                            }
                        } else {
                            v = x[j];
                        }
                        const float4 e = E4[j];
                        v = fma2(e.x, uu[0], v);
                        if constexpr (KW > 0) {
                            v = fma2(e.y, uu[1], v);
                            v = fma2(e.z, uu[2], v);
                            v = fma2(e.w, uu[3], v);
                        }
                        if (last)
                            st2(pX + (long long)Ish[tt * KM + j] * C, v);
                        else
                            st2(pn + (long long)j * C, v);
                    }
                }
                if (last) pX += NC;
                else pn += kC;
            }
        }
        if constexpr (KW > 0) ring_shift<KW>(w);
    }
    cpa_wait<0>();
}

// prefetch ring of the backward reductions: per slot, out (bf16 pair), x_j (bf16 pairs), dn_j
// (fp32 pair, or a bf16 pair in .x at the last slot)
template <int KM>
struct BRing {
    uint32_t o[PD][WT];
    uint32_t x[PD][KM][WT];
    uint2 dn[PD][KM][WT];
};

// Per token, NV partial sums over this CTA's channel slice: P[j][a] = <dXn_j, u_a> at j*4 + a
// and, on the last slot, Q[j][i] = <dXn_j, x_i> at KM*4 + j*KM + i.  NV = 16 is reduced to
// lane pairs, larger NV in blocks of 32.
template <int KM, int KW, int NV, int KS>
__global__ void __launch_bounds__(WT) k_wb_bred(Dims d, int slot, int T, int TB,
                                                const uint16_t* __restrict__ out, ConvPtrs cw,
                                                const uint16_t* __restrict__ dX,
                                                const int* __restrict__ I,
                                                const float* __restrict__ dxact,
                                                const uint16_t* __restrict__ xact, int nslice,
                                                float* __restrict__ red) {
    static_assert(NV == 16 || NV % 32 == 0, "reduction width");
    constexpr int NVP = NV < 32 ? 16 : NV;      // values per token and warp in shared memory
    extern __shared__ __align__(16) unsigned char smu[];
    BRing<KM>& R = *reinterpret_cast<BRing<KM>*>(smu);
    int* Ish = reinterpret_cast<int*>(smu + sizeof(BRing<KM>));          // [TB][KM]
    float* wsh = reinterpret_cast<float*>(Ish + TB * KM);                 // [TB][WT/32][NVP]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int slice = blockIdx.x, C = d.C, k = (KS == 2) ? KM : d.k;
    const bool last = (slot == d.G - 1);
    const int nv = last ? KM * 4 + KM * KM : KM * 4;
    const int c = slice * WSL + 2 * threadIdx.x;
    const bool act = (KS == 2) || c < C;
    long long t0, t1, send;
    int pos0;
    run_bounds<KW>(d, T, TB, t0, t1, send, pos0);
    const int ntok = (int)(t1 - t0);
    for (int q = threadIdx.x; q < ntok * KM; q += WT) {
        const int tt = q / KM, j = q - tt * KM;
        Ish[q] = (j < k) ? I[(t0 + tt) * k + j] : 0;
    }
    __syncthreads();
    // running pointers of the next token to prefetch (issue() is called once per token, in order)
    const uint16_t* po = out + t0 * C + c;
    const uint16_t* px = xact + t0 * k * C + c;
    const uint16_t* pX = dX + t0 * d.N * C + c;
    const float* pd = dxact + t0 * k * C + c;
    const long long kC = (long long)k * C, NC = (long long)d.N * C;
    auto issue = [&](int sl, int tn) {
        if (act && tn < ntok) {
            cpa4(&R.o[sl][threadIdx.x], po);
#pragma unroll
            for (int j = 0; j < KM; ++j) {
                if (j >= k) continue;
                if (last) {
                    cpa4(&R.x[sl][j][threadIdx.x], px + (long long)j * C);
                    cpa4(&R.dn[sl][j][threadIdx.x], pX + (long long)Ish[tn * KM + j] * C);
                } else {
                    cpa8(&R.dn[sl][j][threadIdx.x], pd + (long long)j * C);
                }
            }
        }
        po += C;
        if (last) {
            px += kC;
            pX += NC;
        } else {
            pd += kC;
        }
        cpa_commit();
    };
#pragma unroll
    for (int q = 0; q < PD - 1; ++q) issue(q, q);
    float2 tw[3][KW > 0 ? KW : 1], w[KW > 0 ? KW + UB - 1 : 1];
    if constexpr (KW > 0) {
        taps_reg<KW, KS>(d, cw, c, act, tw);
        ring_init_b<KW>(d, cw, out, c, act, t0, pos0, w);
    }
    constexpr int RU = UB;
    for (int tb = 0; tb < ntok; tb += RU) {
#pragma unroll
        for (int u = 0; u < RU; ++u) {
            const int tt = tb + u;
            if (tt < ntok) {
                const int sl = u % PD;                       // == tt % PD (runs start on a multiple of 4)
                issue((u + PD - 1) % PD, tt + PD - 1);
                cpa_wait<PD - 1>();
                float2 uu[4] = {f2z(), f2z(), f2z(), f2z()};
                float2 dn[KM], x[KM];
#pragma unroll
                for (int j = 0; j < KM; ++j) {
                    dn[j] = f2z();
                    x[j] = f2z();
                }
                if (act) {
                    const float2 o = u2f2(R.o[sl][threadIdx.x]);
                    uu[0] = o;
                    if constexpr (KW > 0) {
                        w[KW - 1 + u] = o;
                        float2 g[3];
                        conv_blk<KW, KS>(tw, w, u, g);
                        uu[1] = g[0];
                        uu[2] = g[1];
                        uu[3] = g[2];
                    }
#pragma unroll
                    for (int j = 0; j < KM; ++j) {
                        if (j >= k) continue;
                        const uint2 r = R.dn[sl][j][threadIdx.x];
                        if (last) {
                            dn[j] = u2f2(r.x);
                            x[j] = u2f2(R.x[sl][j][threadIdx.x]);
                        } else {
                            dn[j] = make_float2(__uint_as_float(r.x), __uint_as_float(r.y));
                        }
                    }
                }
                // dn, x and the unused components are zero where a term does not apply
                float v[NVP];
#pragma unroll
                for (int q = 0; q < NVP; ++q) v[q] = 0.f;
#pragma unroll
                for (int j = 0; j < KM; ++j)
#pragma unroll
                    for (int a = 0; a < 4; ++a)
                        if (j * 4 + a < NVP && (KW > 0 || a == 0)) v[j * 4 + a] = dot2(dn[j], uu[a]);
                if constexpr (NVP >= KM * 4 + KM * KM) {
                    if (last) {
#pragma unroll
                        for (int j = 0; j < KM; ++j)
#pragma unroll
                            for (int i = 0; i < KM; ++i) v[KM * 4 + j * KM + i] = dot2(dn[j], x[i]);
                    }
                }
                float* dst = wsh + ((size_t)tt * (WT / 32) + warp) * NVP;
                if constexpr (KW == 0 && NV == 16) {
                    // no conv: only P[j][0] = <dXn_j, out> (slots j * 4) carry terms
                    float v4[KM];
#pragma unroll
                    for (int j = 0; j < KM; ++j) v4[j] = v[j * 4];
                    const float tot = WRed<KM, 16>::run(v4, lane);
                    constexpr int SH = KM == 4 ? 3 : 2;          // lane >> SH = value index
                    if ((lane & ((1 << SH) - 1)) == 0) dst[(lane >> SH) * 4] = tot;
                } else if constexpr (NV == 16) {
                    const float tot = WRed<16, 16>::run(v, lane);
                    if ((lane & 1) == 0) dst[lane >> 1] = tot;
                } else {
                    float tot[NV / 32];
                    wred32<NV / 32>(v, lane, tot);
#pragma unroll
                    for (int bb = 0; bb < NV / 32; ++bb) dst[bb * 32 + lane] = tot[bb];
                }
            }
        }
        if constexpr (KW > 0) ring_shift<KW>(w);
    }
    cpa_wait<0>();
    __syncthreads();
    for (int idx = threadIdx.x; idx < ntok * nv; idx += WT) {
        const int tt = idx / nv, q = idx - tt * nv;
        if (KW == 0 && NV == 16 && (q & 3) != 0) continue;  // entries without terms (K = 1)
        float sm = 0.f;
#pragma unroll
        for (int ww = 0; ww < WT / 32; ++ww) sm += wsh[((size_t)tt * (WT / 32) + ww) * NVP + q];
        red[((t0 + tt) * nslice + slice) * NRED + q] = sm;
    }
}

// The same reductions with two channel pairs per thread (4 consecutive channels, WSL2 channels
// per CTA): a token's warp reduction then covers 128 channels instead of 64, halving its cost
// per channel, and the loads are 8 / 16 bytes wide.  For the (4, 8, 12) tap set with k = KM
// and C a multiple of WSL2 (every thread in range).

template <int KM>
struct BRing2 {
    uint2 o[PD][WT];
    uint2 x[PD][KM][WT];
    uint4 dn[PD][KM][WT];
};

template <int KM, int NV>
__global__ void __launch_bounds__(WT, 2) k_wb_bred2(Dims d, int slot, int T, int TB,
                                                    const uint16_t* __restrict__ out, ConvPtrs cw,
                                                    const uint16_t* __restrict__ dX,
                                                    const int* __restrict__ I,
                                                    const float* __restrict__ dxact,
                                                    const uint16_t* __restrict__ xact, int nslice,
                                                    float* __restrict__ red) {
    constexpr int KW = 12, KS = 2;
    static_assert(NV == 16 || NV % 32 == 0, "reduction width");
    constexpr int NVP = NV < 32 ? 16 : NV;
    extern __shared__ __align__(16) unsigned char smu[];
    BRing2<KM>& R = *reinterpret_cast<BRing2<KM>*>(smu);
    int* Ish = reinterpret_cast<int*>(smu + sizeof(BRing2<KM>));         // [TB][KM]
    float* wsh = reinterpret_cast<float*>(Ish + TB * KM);                 // [TB][WT/32][NVP]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int slice = blockIdx.x, C = d.C, k = KM;
    const bool last = (slot == d.G - 1);
    const int nv = last ? KM * 4 + KM * KM : KM * 4;
    const int c = slice * WSL2 + 4 * threadIdx.x;
    long long t0, t1, send;
    int pos0;
    run_bounds<KW>(d, T, TB, t0, t1, send, pos0);
    const int ntok = (int)(t1 - t0);
    for (int q = threadIdx.x; q < ntok * KM; q += WT) {
        const int tt = q / KM, j = q - tt * KM;
        Ish[q] = I[(t0 + tt) * k + j];
    }
    __syncthreads();
    const uint16_t* po = out + t0 * C + c;
    const uint16_t* px = xact + t0 * k * C + c;
    const uint16_t* pX = dX + t0 * d.N * C + c;
    const float* pd = dxact + t0 * k * C + c;
    const long long kC = (long long)k * C, NC = (long long)d.N * C;
    auto issue = [&](int sl, int tn) {
        if (tn < ntok) {
            cpa8(&R.o[sl][threadIdx.x], po);
#pragma unroll
            for (int j = 0; j < KM; ++j) {
                if (last) {
                    cpa8(&R.x[sl][j][threadIdx.x], px + (long long)j * C);
                    cpa8(&R.dn[sl][j][threadIdx.x], pX + (long long)Ish[tn * KM + j] * C);
                } else {
                    cpa16(&R.dn[sl][j][threadIdx.x], pd + (long long)j * C);
                }
            }
        }
        po += C;
        if (last) {
            px += kC;
            pX += NC;
        } else {
            pd += kC;
        }
        cpa_commit();
    };
#pragma unroll
    for (int q = 0; q < PD - 1; ++q) issue(q, q);
    float2 tw[2][3][KW], w[2][KW + UB - 1];
#pragma unroll
    for (int p = 0; p < 2; ++p) {
        taps_reg<KW, KS>(d, cw, c + 2 * p, true, tw[p]);
        ring_init_b<KW>(d, cw, out, c + 2 * p, true, t0, pos0, w[p]);
    }
    for (int tb = 0; tb < ntok; tb += UB) {
#pragma unroll
        for (int u = 0; u < UB; ++u) {
            const int tt = tb + u;
            if (tt < ntok) {
                const int sl = u % PD;
                issue((u + PD - 1) % PD, tt + PD - 1);
                cpa_wait<PD - 1>();
                float2 uu[2][4], dn[2][KM], x[2][KM];
                const uint2 orow = R.o[sl][threadIdx.x];
#pragma unroll
                for (int p = 0; p < 2; ++p) {
                    const float2 o = u2f2(p == 0 ? orow.x : orow.y);
                    w[p][KW - 1 + u] = o;
                    float2 g[3];
                    conv_blk<KW, KS>(tw[p], w[p], u, g);
                    uu[p][0] = o;
                    uu[p][1] = g[0];
                    uu[p][2] = g[1];
                    uu[p][3] = g[2];
                }
#pragma unroll
                for (int j = 0; j < KM; ++j) {
                    const uint4 r = R.dn[sl][j][threadIdx.x];
                    if (last) {
                        const uint2 rb = *reinterpret_cast<const uint2*>(&r);
                        dn[0][j] = u2f2(rb.x);
                        dn[1][j] = u2f2(rb.y);
                        const uint2 xr = R.x[sl][j][threadIdx.x];
                        x[0][j] = u2f2(xr.x);
                        x[1][j] = u2f2(xr.y);
                    } else {
                        dn[0][j] = make_float2(__uint_as_float(r.x), __uint_as_float(r.y));
                        dn[1][j] = make_float2(__uint_as_float(r.z), __uint_as_float(r.w));
                        x[0][j] = x[1][j] = f2z();
                    }
                }
                float v[NVP];
#pragma unroll
                for (int q = 0; q < NVP; ++q) v[q] = 0.f;
#pragma unroll
                for (int j = 0; j < KM; ++j)
#pragma unroll
                    for (int a = 0; a < 4; ++a)
                        if (j * 4 + a < NVP)
                            v[j * 4 + a] = fmaf(dn[1][j].y, uu[1][a].y,
                                                fmaf(dn[1][j].x, uu[1][a].x, dot2(dn[0][j], uu[0][a])));
                if constexpr (NVP >= KM * 4 + KM * KM) {
                    if (last) {
#pragma unroll
                        for (int j = 0; j < KM; ++j)
#pragma unroll
                            for (int i = 0; i < KM; ++i)
                                v[KM * 4 + j * KM + i] = fmaf(dn[1][j].y, x[1][i].y,
                                                              fmaf(dn[1][j].x, x[1][i].x, dot2(dn[0][j], x[0][i])));
                    }
                }
                float* dst = wsh + ((size_t)tt * (WT / 32) + warp) * NVP;
                if constexpr (NV == 16) {
                    const float tot = WRed<16, 16>::run(v, lane);
                    if ((lane & 1) == 0) dst[lane >> 1] = tot;
                } else {
                    float tot[NV / 32];
                    wred32<NV / 32>(v, lane, tot);
#pragma unroll
                    for (int bb = 0; bb < NV / 32; ++bb) dst[bb * 32 + lane] = tot[bb];
                }
            }
        }
#pragma unroll
        for (int p = 0; p < 2; ++p) ring_shift<KW>(w[p]);
    }
    cpa_wait<0>();
    __syncthreads();
    for (int idx = threadIdx.x; idx < ntok * nv; idx += WT) {
        const int tt = idx / nv, q = idx - tt * nv;
        float sm = 0.f;
#pragma unroll
        for (int ww = 0; ww < WT / 32; ++ww) sm += wsh[((size_t)tt * (WT / 32) + ww) * NVP + q];
        red[((t0 + tt) * nslice + slice) * NRED + q] = sm;
    }
}

// ---------------------------------------------------------------------------------------------
// wb_bapp: du_a = sum_j E[j][a] dXn_j + sum_b D[a][b] u_b (Eq. sparse_write reversed, with the
// Gram-Schmidt Jacobian in D), never stored:
//   d_out[s] = du_0[s] + sum_j sum_{i < kappa_j, s + i in the sequence} w_j[i] du_{1+j}[s + i]
// (the transpose of the causal conv of Eq. aug) is accumulated in a ring of KW pending outputs;
// output s is complete, and stored, once token s + KW - 1 has been seen (du is taken as zero
// past the sequence end).  Each run therefore recomputes du for up to KW - 1 tokens after it.
// The conv weight gradient sum_t du_{1+j}[t] out[t - i] is accumulated per run.  Last slot:
// dX_act_i = sum_j H_res[j][i] dXn_j.  The -cx x_i term of the active-state gradient is added by
// the backward of the slot's pre-map.

template <int KM>
struct ARing {
    uint32_t o[PD][WT];
    uint2 dn[PD][KM][WT];
};

// HALO: the variant for a call on a later chunk of its sequences, which also returns the
// gradient of the halo rows (cw.dhalo); compiled only for the generic tap set (KS = 0), so the
// common variants carry none of its registers
template <int KM, int KW, int KS, bool HALO = false>
__global__ void __launch_bounds__(WT, 2) k_wb_bapp(Dims d, int slot, int T, int TB,
                                                   const uint16_t* __restrict__ out, ConvPtrs cw,
                                                   const uint16_t* __restrict__ dX,
                                                   const int* __restrict__ I,
                                                   const float* dn_in,  // may alias dxact_out
                                                   const float* __restrict__ tokmat,
                                                   float* dxact_out,
                                                   uint16_t* __restrict__ d_out,
                                                   float* __restrict__ cpart) {
    constexpr int HL = KW > 0 ? KW - 1 : 0;   // tokens after the run whose du the run needs
    constexpr int RU = UB;
    constexpr int NR = KW > 0 ? KW + UB - 1 : 1;   // block ring slots
    extern __shared__ __align__(16) unsigned char smu[];
    ARing<KM>& R = *reinterpret_cast<ARing<KM>*>(smu);
    const int k = (KS == 2) ? KM : d.k, C = d.C;
    const bool last = (slot == d.G - 1);
    const int TH = TB + HL;
    float* Esh = reinterpret_cast<float*>(smu + sizeof(ARing<KM>));  // [TH][KM][4]
    float* Dsh = Esh + TH * KM * 4;                                 // [TH][4][4]
    float* Hsh = Dsh + TH * 16;                                     // [TH][KM][KM]
    int* Ish = reinterpret_cast<int*>(Hsh + TH * KM * KM);           // [TH][KM]
    long long t0, t1, send;
    int pos0;
    run_bounds<KW>(d, T, TB, t0, t1, send, pos0);
    const int n1 = (int)(t1 - t0);                                  // tokens of the run
    const int ntok = (int)(min(t1 + HL, send) - t0);                // + the halo inside the sequence
    const int nloop = n1 + HL;                                      // + the emission lag
    for (int idx = threadIdx.x; idx < ntok * KM * 4; idx += WT) {
        const int tt = idx / (KM * 4), q = idx - tt * (KM * 4);
        Esh[idx] = tokmat[(t0 + tt) * TOKMAT + q];
    }
    if constexpr (KW > 0) {
        for (int idx = threadIdx.x; idx < ntok * 16; idx += WT) {
            const int tt = idx >> 4, q = idx & 15;
            Dsh[idx] = tokmat[(t0 + tt) * TOKMAT + 32 + q];
        }
    }
    if (last) {
        for (int idx = threadIdx.x; idx < ntok * KM * KM; idx += WT) {
            const int tt = idx / (KM * KM), q = idx - tt * (KM * KM);
            Hsh[idx] = tokmat[(t0 + tt) * TOKMAT + 48 + (q / KM) * 8 + (q % KM)];
        }
        for (int idx = threadIdx.x; idx < ntok * KM; idx += WT) {
            const int tt = idx / KM, j = idx - tt * KM;
            Ish[idx] = (j < k) ? I[(t0 + tt) * k + j] : 0;
        }
    }
    const int c = blockIdx.x * WSL + 2 * threadIdx.x;
    const bool act = (KS == 2) || c < C;
    __syncthreads();
    // running pointers: next token to prefetch (issue() is called once per token, in order), the
    // token whose active gradient is written (last slot), the next d_out row to store
    const uint16_t* po = out + t0 * C + c;
    const uint16_t* pX = dX + t0 * d.N * C + c;
    const float* pd = dn_in + t0 * k * C + c;
    float* pxo = dxact_out + t0 * k * C + c;
    uint16_t* pdo = d_out + t0 * C + c;
    const long long kC = (long long)k * C, NC = (long long)d.N * C;
    auto issue = [&](int sl, int tn) {
        if (act && tn < ntok) {
            cpa4(&R.o[sl][threadIdx.x], po);
#pragma unroll
            for (int j = 0; j < KM; ++j) {
                if (j >= k) continue;
                if (last)
                    cpa4(&R.dn[sl][j][threadIdx.x], pX + (long long)Ish[tn * KM + j] * C);
                else
                    cpa8(&R.dn[sl][j][threadIdx.x], pd + (long long)j * C);
            }
        }
        po += C;
        if (last) pX += NC;
        else pd += kC;
        cpa_commit();
    };
#pragma unroll
    for (int q = 0; q < PD - 1; ++q) issue(q, q);
    // pend: the block ring of pending outputs, slot KW - 1 + u - i <-> output tb + u - i
    float2 tw[3][KW > 0 ? KW : 1], w[NR], pend[NR];
    float2 acc[3][KW > 0 ? KW : 1];
    if constexpr (KW > 0) {
        taps_reg<KW, KS>(d, cw, c, act, tw);
        ring_init_b<KW>(d, cw, out, c, act, t0, pos0, w);
#pragma unroll
        for (int s = 0; s < NR; ++s) pend[s] = f2z();
#pragma unroll
        for (int j = 0; j < 3; ++j)
#pragma unroll
            for (int i = 0; i < KW; ++i) acc[j][i] = f2z();
    }
    // the halo gradient (a call on a later chunk): rows of this sequence, this channel pair
    float* dhalo_row = (HALO && KW > 0 && cw.dhalo != nullptr && pos0 == 0)
                           ? cw.dhalo + (t0 / d.S) * (d.kapmax - 1) * C + c : nullptr;
    for (int tb = 0; tb < nloop; tb += RU) {
#pragma unroll
        for (int u = 0; u < RU; ++u) {
            const int tt = tb + u;
            if (tt < nloop) {
                const int sl = u % PD;
                issue((u + PD - 1) % PD, tt + PD - 1);
                cpa_wait<PD - 1>();
                if (act) {
                    float2 du[4] = {f2z(), f2z(), f2z(), f2z()};
                    if (tt < ntok) {
                        const float2 o = u2f2(R.o[sl][threadIdx.x]);
                        float2 dn[KM];
#pragma unroll
                        for (int j = 0; j < KM; ++j) {
                            dn[j] = f2z();
                            if (j < k) {
                                const uint2 r = R.dn[sl][j][threadIdx.x];
                                dn[j] = last ? u2f2(r.x) : make_float2(__uint_as_float(r.x), __uint_as_float(r.y));
                            }
                        }
                        const float4* E4 = reinterpret_cast<const float4*>(Esh + tt * KM * 4);
#pragma unroll
                        for (int j = 0; j < KM; ++j) {
                            if (j >= k) continue;
                            const float4 e = E4[j];
                            du[0] = fma2s(e.x, dn[j], du[0]);
                            if constexpr (KW > 0) {
                                du[1] = fma2s(e.y, dn[j], du[1]);
                                du[2] = fma2s(e.z, dn[j], du[2]);
                                du[3] = fma2s(e.w, dn[j], du[3]);
                            }
                        }
                        if constexpr (KW > 0) {
                            w[KW - 1 + u] = o;
                            float2 g[3];
                            conv_blk<KW, KS>(tw, w, u, g);
                            const float2 uu[4] = {o, g[0], g[1], g[2]};
                            const float4* D4 = reinterpret_cast<const float4*>(Dsh + tt * 16);
#pragma unroll
                            for (int a = 0; a < 4; ++a) {
                                const float4 m = D4[a];
                                du[a] = fma2s(m.x, uu[0], du[a]);
                                du[a] = fma2s(m.y, uu[1], du[a]);
                                du[a] = fma2s(m.z, uu[2], du[a]);
                                du[a] = fma2s(m.w, uu[3], du[a]);
                            }
                        }
                        if (last && tt < n1) {
                            const float4* H4 = reinterpret_cast<const float4*>(Hsh + tt * KM * KM);
                            float2 v[KM];
#pragma unroll
                            for (int i = 0; i < KM; ++i) v[i] = f2z();
#pragma unroll
                            for (int j = 0; j < KM; ++j) {
                                if (j >= k) continue;
#pragma unroll
                                for (int q = 0; q < KM / 4; ++q) {
                                    const float4 h = H4[j * (KM / 4) + q];
                                    v[4 * q + 0] = fma2s(h.x, dn[j], v[4 * q + 0]);
                                    v[4 * q + 1] = fma2s(h.y, dn[j], v[4 * q + 1]);
                                    v[4 * q + 2] = fma2s(h.z, dn[j], v[4 * q + 2]);
                                    v[4 * q + 3] = fma2s(h.w, dn[j], v[4 * q + 3]);
                                }
                            }
#pragma unroll
                            for (int i = 0; i < KM; ++i)
                                if (i < k) *reinterpret_cast<float2*>(pxo + (long long)i * C) = v[i];
                            pxo += kC;
                        }
                    } else if constexpr (KW > 0) {
                        w[KW - 1 + u] = f2z();   // past the sequence end
                    }
                    if constexpr (KW == 0) {
                        if (tt < n1) {
                            st2(pdo, du[0]);
                            pdo += C;
                        }
                    } else {
                        // conv weight gradient of the run's tokens
                        if (tt < n1) {
#pragma unroll
                            for (int j = 0; j < 3; ++j)
#pragma unroll
                                for (int i = 0; i < KW; ++i) {
                                    if (i >= ntap<KW, KS>(j)) continue;
                                    const float2 o = w[KW - 1 + u - i];
                                    acc[j][i] = ffma2(du[1 + j], o, acc[j][i]);
                                }
                        }
                        // d_out[t - i] += w_j[i] du_{1+j}[t]
                        pend[KW - 1 + u] = du[0];
#pragma unroll
                        for (int i = 0; i < KW; ++i) {
#pragma unroll
                            for (int j = 0; j < 3; ++j) {
                                if (i >= ntap<KW, KS>(j)) continue;
                                float2& q = pend[KW - 1 + u - i];
                                q = ffma2(tw[j][i], du[1 + j], q);
                            }
                        }
                    }
                }
            }
        }
        if constexpr (KW > 0) {
            // outputs tb + q - (KW - 1), q < UB, have all their terms (du is zero past the
            // sequence end): stored in order; positions before the run start are the halo rows
            // of a call on a later chunk of its sequences
            if (act) {
#pragma unroll
                for (int q = 0; q < UB; ++q) {
                    const int ot = tb + q - (KW - 1);
                    if (ot >= 0) {
                        if (ot < n1) {
                            st2(pdo, pend[q]);
                            pdo += C;
                        }
                    } else if constexpr (HALO) {
                        const int r = d.kapmax - 1 + ot;
                        if (dhalo_row != nullptr && r >= 0)
                            *reinterpret_cast<float2*>(dhalo_row + (long long)r * C) = pend[q];
                    }
                }
            }
            ring_shift<KW>(w);
            ring_shift<KW>(pend);
        }
    }
    cpa_wait<0>();
    if constexpr (KW > 0) {
        if (!act) return;
        int off = 0;
#pragma unroll
        for (int j = 0; j < 3; ++j) {
            if (j < d.nconv) {
#pragma unroll
                for (int i = 0; i < KW; ++i)
                    if (i < d.kap[j])
                        *reinterpret_cast<float2*>(cpart + ((long long)blockIdx.y * d.kapsum + off + i) * C + c) =
                            acc[j][i];
                off += d.kap[j];
            }
        }
    }
}

// ---------------------------------------------------------------------------------------------
// Write-back kernels of the sublayers without temporal conv (K = 1), 8 channels per thread: no
// conv ring to keep, so every thread moves 16-byte rows; the next token's rows are loaded into
// registers while the current one is processed.  A CTA covers W8 channels of a run of tokens.

constexpr int W8 = WT * 8;   // channels per CTA

__device__ __forceinline__ uint4 ld16(const void* p) { return __ldg(reinterpret_cast<const uint4*>(p)); }
__device__ __forceinline__ void l2_prefetch(const void* p) { asm volatile("prefetch.global.L2 [%0];" ::"l"(p)); }
constexpr int B8_PF = 2;   // L2 prefetch distance of the one-pass attention backward, in tokens

// per-token tables shared by the CTA: E[j][0] (write-back coefficient of out), H_res, I
template <int KM>
__device__ __forceinline__ void k1_tables(int ntok, long long t0, int k, bool last, const float* emat,
                                          int estride, const float* hres, const int* I, float* Esh,
                                          float* Hsh, int* Ish) {
    for (int idx = threadIdx.x; idx < ntok * KM; idx += WT) {
        const int tt = idx / KM, j = idx - tt * KM;
        Esh[idx] = (j < k) ? emat[(t0 + tt) * estride + j * 4] : 0.f;
        Ish[idx] = (j < k) ? I[(t0 + tt) * k + j] : 0;
    }
    if (last)
        for (int idx = threadIdx.x; idx < ntok * KM * KM; idx += WT) {
            const int tt = idx / (KM * KM), q = idx - tt * (KM * KM);
            const int j = q / KM, i = q - j * KM;
            Hsh[idx] = (j < k && i < k) ? hres[(t0 + tt) * k * k + j * k + i] : 0.f;
        }
}

// forward: X_act_new_j = (sum_i H_res[j][i] x_i  |  x_j) + E[j][0] out
template <int KM>
__global__ void __launch_bounds__(WT) k_wb_fwd8(Dims d, int slot, int T, int TB,
                                                const uint16_t* __restrict__ out,
                                                const float* __restrict__ emat,
                                                const uint16_t* __restrict__ xact,
                                                const int* __restrict__ I,
                                                const float* __restrict__ hres,
                                                uint16_t* __restrict__ xact_next,
                                                uint16_t* __restrict__ X) {
    extern __shared__ __align__(16) unsigned char smu[];
    float* Esh = reinterpret_cast<float*>(smu);        // [TB][KM]
    float* Hsh = Esh + TB * KM;                        // [TB][KM][KM]
    int* Ish = reinterpret_cast<int*>(Hsh + TB * KM * KM);
    const int k = d.k, C = d.C;
    const bool last = (slot == d.G - 1);
    const long long t0 = (long long)blockIdx.y * TB;
    const int ntok = (int)(min((long long)T, t0 + TB) - t0);
    k1_tables<KM>(ntok, t0, k, last, emat, TOKMAT, hres, I, Esh, Hsh, Ish);
    __syncthreads();
    const int c = blockIdx.x * W8 + threadIdx.x * 8;
    if (c >= C) return;
    const long long kC = (long long)k * C, NC = (long long)d.N * C;
    const uint16_t* po = out + t0 * C + c;
    const uint16_t* px = xact + t0 * kC + c;
    uint4 on = ld16(po), xn[KM];
#pragma unroll
    for (int j = 0; j < KM; ++j) xn[j] = (j < k) ? ld16(px + j * (long long)C) : make_uint4(0, 0, 0, 0);
    for (int tt = 0; tt < ntok; ++tt) {
        const uint4 oc = on;
        uint4 xc[KM];
#pragma unroll
        for (int j = 0; j < KM; ++j) xc[j] = xn[j];
        po += C;
        px += kC;
        if (tt + 1 < ntok) {
            on = ld16(po);
#pragma unroll
            for (int j = 0; j < KM; ++j)
                if (j < k) xn[j] = ld16(px + j * (long long)C);
        }
        const long long t = t0 + tt;
        float o[8], x[KM][8];
        unpack8(oc, o);
#pragma unroll
        for (int j = 0; j < KM; ++j) unpack8(xc[j], x[j]);
#pragma unroll
        for (int j = 0; j < KM; ++j) {
            if (j >= k) continue;
            const float e = Esh[tt * KM + j];
            float v[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                float a = 0.f;
                if (last) {
#pragma unroll
                    for (int i = 0; i < KM; ++i) a = fmaf(Hsh[(tt * KM + j) * KM + i], x[i][q], a);
                } else {
                    a = x[j][q];
                }
                v[q] = fmaf(e, o[q], a);
            }
            uint16_t* dst = last ? X + t * NC + (long long)Ish[tt * KM + j] * C + c
                                 : xact_next + t * kC + (long long)j * C + c;
            *reinterpret_cast<uint4*>(dst) = pack8(v);
        }
    }
}

// Backward of a slot without conv (K = 1) in one pass: the apply coefficients of such a slot
// are forward quantities (E[j][0] = p_j H_post[j], and on the last slot the forward H_res), so
// the reductions P[j][0] = <dXn_j, out> (last slot: Q[j][i] = <dXn_j, x_i>) and the apply
// d_out = sum_j E[j][0] dXn_j (last slot: dX_act_i = sum_j H_res[j][i] dXn_j) read dXn once.
// Partial sums per W8-channel slice: P[j][0] at j*4, Q[j][i] at KM*4 + j*KM + i (the layout
// bwd_coef reads).
template <int KM>
__global__ void __launch_bounds__(WT, 3) k_wb_b8(Dims d, int slot, int T, int TB,
                                              const uint16_t* __restrict__ out,
                                              const uint16_t* __restrict__ dX,
                                              const int* __restrict__ I,
                                              const float* __restrict__ p,
                                              const float* __restrict__ hpost,
                                              const float* __restrict__ hres,
                                              const float* dxact,   // read (earlier slots)
                                              float* dxact_out,     // written (last slot)
                                              const uint16_t* __restrict__ xact, int nslice,
                                              float* __restrict__ red,
                                              uint16_t* __restrict__ d_out) {
    constexpr int NQ = KM + KM * KM;                  // P[j][0], then Q[j][i]
    constexpr int NV = NQ <= 32 ? 32 : 96;            // reduce-scatter width (blocks of 32)
    extern __shared__ __align__(16) unsigned char smu[];
    int* Ish = reinterpret_cast<int*>(smu);                  // [TB][KM]
    float* Esh = reinterpret_cast<float*>(Ish + TB * KM);    // [TB][KM]
    float* Hsh = Esh + TB * KM;                              // [TB][KM][KM] (last slot)
    float* wsh = Hsh + TB * KM * KM;                         // [TB][WT/32][NV]
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int k = d.k, C = d.C;
    const bool last = (slot == d.G - 1);
    const long long t0 = (long long)blockIdx.y * TB;
    const int ntok = (int)(min((long long)T, t0 + TB) - t0);
    for (int idx = threadIdx.x; idx < ntok * KM; idx += WT) {
        const int tt = idx / KM, j = idx - tt * KM;
        const long long tj = (t0 + tt) * k + j;
        Ish[idx] = (j < k) ? I[tj] : 0;
        Esh[idx] = (j < k) ? p[tj] * hpost[tj] : 0.f;
    }
    if (last)
        for (int idx = threadIdx.x; idx < ntok * KM * KM; idx += WT) {
            const int tt = idx / (KM * KM), q = idx - tt * (KM * KM);
            const int j = q / KM, i = q - j * KM;
            Hsh[idx] = (j < k && i < k) ? hres[(t0 + tt) * k * k + j * k + i] : 0.f;
        }
    __syncthreads();
    const int c = blockIdx.x * W8 + threadIdx.x * 8;
    const bool act = c < C;
    const long long kC = (long long)k * C, NC = (long long)d.N * C;
    const uint16_t* po = out + t0 * C + c;
    const uint16_t* px = xact + t0 * kC + c;
    const uint16_t* pX = dX + t0 * NC + c;
    const float* pd = dxact + t0 * kC + c;
    // next token's rows: out, dXn_j (bf16 rows of dX, or fp32 active gradient), x_j (last)
    uint4 on = make_uint4(0, 0, 0, 0), dn0[KM], dn1[KM], xn[KM];
    // an L2 prefetch of the rows B8_PF tokens further on, one request per 128-byte line
    const bool pf32 = (threadIdx.x & 3) == 0, pf16 = (threadIdx.x & 7) == 0;
    auto prefetch = [&](int tt) {
        if (B8_PF == 0 || !act || tt >= ntok) return;
        const long long dt = (long long)B8_PF;
        if (pf16) l2_prefetch(po + dt * C);
#pragma unroll
        for (int j = 0; j < KM; ++j) {
            if (j >= k) continue;
            if (last) {
                if (pf16) {
                    l2_prefetch(pX + dt * NC + (long long)Ish[tt * KM + j] * C);
                    l2_prefetch(px + dt * kC + j * (long long)C);
                }
            } else if (pf32) {
                l2_prefetch(pd + dt * kC + j * (long long)C);
            }
        }
    };
    auto load = [&](int tt) {
        prefetch(tt + B8_PF);
#pragma unroll
        for (int j = 0; j < KM; ++j) {
            dn0[j] = make_uint4(0, 0, 0, 0);
            dn1[j] = dn0[j];
            xn[j] = dn0[j];
        }
        on = dn0[0];
        if (!act || tt >= ntok) return;
        on = ld16(po);
#pragma unroll
        for (int j = 0; j < KM; ++j) {
            if (j >= k) continue;
            if (last) {
                dn0[j] = ld16(pX + (long long)Ish[tt * KM + j] * C);
                xn[j] = ld16(px + j * (long long)C);
            } else {
                dn0[j] = ld16(pd + j * (long long)C);
                dn1[j] = ld16(pd + j * (long long)C + 4);
            }
        }
    };
    load(0);
    for (int tt = 0; tt < ntok; ++tt) {
        const uint4 oc = on;
        uint4 d0[KM], d1[KM], xc[KM];
#pragma unroll
        for (int j = 0; j < KM; ++j) {
            d0[j] = dn0[j];
            d1[j] = dn1[j];
            xc[j] = xn[j];
        }
        po += C;
        if (last) {
            px += kC;
            pX += NC;
        } else {
            pd += kC;
        }
        load(tt + 1);
        const long long t = t0 + tt;
        float o[8], dn[KM][8];
        unpack8(oc, o);
#pragma unroll
        for (int j = 0; j < KM; ++j) {
            if (last) {
                unpack8(d0[j], dn[j]);
            } else {
                dn[j][0] = __uint_as_float(d0[j].x); dn[j][1] = __uint_as_float(d0[j].y);
                dn[j][2] = __uint_as_float(d0[j].z); dn[j][3] = __uint_as_float(d0[j].w);
                dn[j][4] = __uint_as_float(d1[j].x); dn[j][5] = __uint_as_float(d1[j].y);
                dn[j][6] = __uint_as_float(d1[j].z); dn[j][7] = __uint_as_float(d1[j].w);
            }
        }
        float v[NV];
#pragma unroll
        for (int q = 0; q < NV; ++q) v[q] = 0.f;
#pragma unroll
        for (int j = 0; j < KM; ++j)
#pragma unroll
            for (int q = 0; q < 8; ++q) v[j] = fmaf(dn[j][q], o[q], v[j]);
        if (last) {
            float x[KM][8];
#pragma unroll
            for (int i = 0; i < KM; ++i) unpack8(xc[i], x[i]);
#pragma unroll
            for (int j = 0; j < KM; ++j)
#pragma unroll
                for (int i = 0; i < KM; ++i)
#pragma unroll
                    for (int q = 0; q < 8; ++q) v[KM + j * KM + i] = fmaf(dn[j][q], x[i][q], v[KM + j * KM + i]);
        }
        if (act) {
            // apply: d_out = sum_j E[j][0] dXn_j, and the mixed active gradient of the last slot
            float g[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) g[q] = 0.f;
#pragma unroll
            for (int j = 0; j < KM; ++j) {
                const float e = Esh[tt * KM + j];
#pragma unroll
                for (int q = 0; q < 8; ++q) g[q] = fmaf(e, dn[j][q], g[q]);
            }
            *reinterpret_cast<uint4*>(d_out + t * C + c) = pack8(g);
            if (last) {
#pragma unroll
                for (int i = 0; i < KM; ++i) {
                    if (i >= k) continue;
                    float w[8];
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        float a = 0.f;
#pragma unroll
                        for (int j = 0; j < KM; ++j) a = fmaf(Hsh[(tt * KM + j) * KM + i], dn[j][q], a);
                        w[q] = a;
                    }
                    float4* dst = reinterpret_cast<float4*>(dxact_out + t * kC + (long long)i * C + c);
                    dst[0] = make_float4(w[0], w[1], w[2], w[3]);
                    dst[1] = make_float4(w[4], w[5], w[6], w[7]);
                }
            }
        }
        float tot[NV / 32];
        wred32<NV / 32>(v, lane, tot);
        float* dst = wsh + ((size_t)tt * (WT / 32) + warp) * NV;
#pragma unroll
        for (int bb = 0; bb < NV / 32; ++bb) dst[bb * 32 + lane] = tot[bb];
    }
    __syncthreads();
    const int nq = last ? NQ : KM;
    for (int idx = threadIdx.x; idx < ntok * nq; idx += WT) {
        const int tt = idx / nq, q = idx - tt * nq;
        float sm = 0.f;
#pragma unroll
        for (int ww = 0; ww < WT / 32; ++ww) sm += wsh[((size_t)tt * (WT / 32) + ww) * NV + q];
        const int slotq = q < KM ? q * 4 : KM * 4 + (q - KM);
        red[((t0 + tt) * nslice + blockIdx.x) * NRED + slotq] = sm;
    }
}

inline int kw_of(const Dims& d) {
    const int km = d.kapmax;
    return km <= 4 ? 4 : km <= 8 ? 8 : km <= 12 ? 12 : 16;
}

// the (4, 8, 12) kernels of the MLP sublayers
inline bool paper_kaps(const Dims& d) {
    return d.nconv == 3 && d.kap[0] == 4 && d.kap[1] == 8 && d.kap[2] == 12;
}

inline int run_len(int KW, int per) {  // tokens per CTA run: a multiple of KW near `per`
    const int u = KW > 0 ? KW : 4;
    int r = (per / u) * u;
    return r < u ? u : r;
}

// number of runs of TB tokens (with a conv: runs inside each sequence of S tokens)
inline long long n_runs(const Dims& d, int T, int TB, bool conv) {
    if (!conv || d.S <= 0) return ((long long)T + TB - 1) / TB;
    const long long rps = (d.S + TB - 1) / TB;
    const long long rem = T % d.S;
    return (T / d.S) * rps + (rem + TB - 1) / TB;
}

// tokens per run of the backward apply (longer runs amortise the KW - 1 recomputed tokens)
// tokens per run of the backward apply (with a conv: any length works with the block ring; 296
// measured best at S = 4096, C = 4096 among 240 / 256 / 296 — fewer, fuller waves of CTAs)
inline int bapp_run(int KW) { return KW > 0 ? 296 : 64; }

inline cudaError_t smem_attr(const void* fn, size_t bytes) {
    if (bytes <= 48 * 1024) return cudaSuccess;
    return cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

// KWC: conv taps held per component (0: no conv); KSC: the kernel variant (see ntap)
#define XHC_KW_DISPATCH(D, FAST, CALL)                                        \
    switch (kw_of(D)) {                                                       \
        case 4: { constexpr int KWC = 4, KSC = 0; return CALL; }              \
        case 8: { constexpr int KWC = 8, KSC = 0; return CALL; }              \
        case 12:                                                              \
            if (paper_kaps(D) && (FAST)) { constexpr int KWC = 12, KSC = 2; return CALL; } \
            if (paper_kaps(D)) { constexpr int KWC = 12, KSC = 1; return CALL; } \
            { constexpr int KWC = 12, KSC = 0; return CALL; }                 \
        default: { constexpr int KWC = 16, KSC = 0; return CALL; }            \
    }

// the KS = 2 variants: four active slots and whole channel slices
inline bool wb_fast(const Dims& d) { return d.k == 4 && d.C % WSL == 0; }


}  // namespace
}  // namespace xhc
