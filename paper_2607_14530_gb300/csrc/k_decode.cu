// Decode: the write-back of a conv slot for one new token per sequence.
//
// In decoding, token t of the call is the next token of its own sequence b = t, at position
// pos[t] of that sequence.  The causal conv of Eq. aug (Sec. 3.3.4: g_j[s] = sum_{i < kappa_j}
// w_j[i] out[s - i], zero before the sequence start) needs the R = max(kappa) - 1 previous `out`
// rows of the sequence, which no longer exist as a contiguous [T][C] buffer: they are kept in a
// per-sequence ring [B][R][C] bf16 (row (s mod R) holds out[s]).  The kernels below are the
// decode forms of the Gram reduction and of the write-back (Eq. gs, Eq. sparse_write_delta,
// Eq. sparse_write): CTAs over (256-channel slice, 4 tokens), one channel pair per thread, the
// conv read from the ring plus the token's own `out` row.  The write-back stores the token's
// `out` into its ring row afterwards, and the group's last slot advances pos.
#include <algorithm>

#include "xhc_internal.cuh"

namespace xhc {
namespace {

__device__ __forceinline__ float2 ldp(const uint16_t* p) {
    const uint32_t u = *reinterpret_cast<const uint32_t*>(p);
    return make_float2(__uint_as_float(u << 16), __uint_as_float(u & 0xffff0000u));
}

// the write-back components of channels (c, c + 1) of token t: u_0 = out, u_{1+j} = g_j
__device__ __forceinline__ void dec_components(const Dims& d, int slot, int t, int c,
                                               const uint16_t* __restrict__ out, ConvPtrs cw,
                                               const uint16_t* __restrict__ ring, long long pos,
                                               float2 (&u)[4]) {
    const int C = d.C, R = d.kapmax - 1;
    const float2 o = ldp(out + (long long)t * C + c);
    u[0] = o;
    u[1] = u[2] = u[3] = make_float2(0.f, 0.f);
    if (d.K[slot] <= 1) return;
    const int r0 = (int)(pos % R);                             // ring row of position pos
    const uint16_t* rt = ring + (long long)t * R * C + c;
    // the component loop runs to its maximum of 3 with a guard, so that cw.w[j] and d.kap[j]
    // are static indices (a dynamic index copies the parameter structs to local memory)
#pragma unroll
    for (int j = 0; j < 3; ++j) {
        if (j >= d.nconv) break;
        float2 g = make_float2(0.f, 0.f);
        for (int i = 0; i < d.kap[j]; ++i) {
            if (pos - i < 0) break;                            // before the sequence start: zero
            int r = r0 - i;                                    // row of position pos - i
            if (r < 0) r += R;
            const float2 v = (i == 0) ? o : ldp(rt + (long long)r * C);
            const float2 w = make_float2(cw.w[j][(size_t)i * C + c], cw.w[j][(size_t)i * C + c + 1]);
            g.x = fmaf(w.x, v.x, g.x);
            g.y = fmaf(w.y, v.y, g.y);
        }
        u[1 + j] = g;
    }
}

// Both kernels: CTA (slice, block) takes the 256 channels of slice `slice` (one pair per
// thread) for DT consecutive tokens, so the conv taps of its channels are read once per CTA and
// reused from L1 for the following tokens.
constexpr int DT = 4;
constexpr int DTH = 128;

// Gram matrix of the components of each token (lower triangle, the order of the prefill's
// reduction), partial over the CTA's channel slice: red[t][slice][q]
__global__ void __launch_bounds__(DTH) k_dec_gram(Dims d, int slot, int B, const uint16_t* __restrict__ out,
                                                  ConvPtrs cw, const uint16_t* __restrict__ ring,
                                                  const long long* __restrict__ pos, int nslice,
                                                  float* __restrict__ red) {
    __shared__ float sh[DTH / 32][NGRAM];
    const int slice = blockIdx.x, K = d.K[slot];
    const int c = slice * 2 * DTH + 2 * threadIdx.x;
    const bool act = c < d.C;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int tt = 0; tt < DT; ++tt) {
        const int t = blockIdx.y * DT + tt;
        if (t >= B) break;
        float v[NGRAM];
#pragma unroll
        for (int q = 0; q < NGRAM; ++q) v[q] = 0.f;
        if (act) {
            float2 u[4];
            dec_components(d, slot, t, c, out, cw, ring, pos[t], u);
            int q = 0;
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int b = 0; b <= a; ++b, ++q)
                    if (a < K) v[q] = fmaf(u[a].x, u[b].x, u[a].y * u[b].y);
        }
#pragma unroll
        for (int q = 0; q < NGRAM; ++q) {
            float x = v[q];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
            if (lane == 0) sh[warp][q] = x;
        }
        __syncthreads();
        if (threadIdx.x < NGRAM) {
            float s2 = 0.f;
#pragma unroll
            for (int w = 0; w < DTH / 32; ++w) s2 += sh[w][threadIdx.x];
            red[((long long)t * nslice + slice) * NRED + threadIdx.x] = s2;
        }
        __syncthreads();
    }
}

// X_act_new_j = (H_res x_act)_j (last slot) or x_act_j, + sum_a E[j][a] u_a; the last slot
// scatters into the state rows I_j, the others write the next slot's active state.  Then the
// token's out row goes into its ring row (each thread its own channels, after its last read of
// them).
__global__ void __launch_bounds__(DTH) k_dec_fwd(Dims d, int slot, int B, const uint16_t* __restrict__ out,
                                                 ConvPtrs cw, uint16_t* __restrict__ ring,
                                                 const long long* __restrict__ pos,
                                                 const float* __restrict__ emat,
                                                 const uint16_t* __restrict__ xact,
                                                 const int* __restrict__ I,
                                                 const float* __restrict__ hres,
                                                 uint16_t* __restrict__ xact_next,
                                                 uint16_t* __restrict__ X) {
    const int C = d.C, k = d.k, R = d.kapmax - 1;
    const bool last = (slot == d.G - 1);
    const bool conv = d.K[slot] > 1;
    const int c = blockIdx.x * 2 * DTH + 2 * threadIdx.x;
    if (c >= C) return;
    for (int tt = 0; tt < DT; ++tt) {
        const int t = blockIdx.y * DT + tt;
        if (t >= B) break;
        const long long p = pos[t];
        const float* E = emat + (long long)t * TOKMAT;
        float2 u[4];
        dec_components(d, slot, t, c, out, cw, ring, p, u);
        float2 x[MAXK];
#pragma unroll
        for (int j = 0; j < MAXK; ++j)
            x[j] = (j < k) ? ldp(xact + ((long long)t * k + j) * C + c) : make_float2(0.f, 0.f);
#pragma unroll
        for (int j = 0; j < MAXK; ++j) {
            if (j >= k) break;
            float2 v;
            if (last) {
                v = make_float2(0.f, 0.f);
#pragma unroll
                for (int i = 0; i < MAXK; ++i) {
                    if (i >= k) break;
                    const float h = hres[((long long)t * k + j) * k + i];
                    v.x = fmaf(h, x[i].x, v.x);
                    v.y = fmaf(h, x[i].y, v.y);
                }
            } else {
                v = x[j];
            }
#pragma unroll
            for (int a = 0; a < 4; ++a) {
                const float e = E[j * 4 + a];
                v.x = fmaf(e, u[a].x, v.x);
                v.y = fmaf(e, u[a].y, v.y);
            }
            uint16_t* dst = last ? X + ((long long)t * d.N + I[(long long)t * k + j]) * C + c
                                 : xact_next + ((long long)t * k + j) * C + c;
            *reinterpret_cast<uint32_t*>(dst) = pack2(v.x, v.y);
        }
        if (conv && R > 0)
            *reinterpret_cast<uint32_t*>(ring + ((long long)t * R + (int)(p % R)) * C + c) =
                *reinterpret_cast<const uint32_t*>(out + (long long)t * C + c);
    }
}

// the last slot advances every token's position (after every CTA of the write-back is done:
// a separate launch)
__global__ void k_pos_advance(long long* __restrict__ pos, int B) {
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b < B) pos[b] += 1;
}

// ring rows from a prefill: sequence b of S tokens (rows b*S .. b*S + S - 1 of out) leaves its
// last min(S, R) rows in ring rows (s mod R)
__global__ void k_ring_fill(const uint16_t* __restrict__ out, int B, int S, int C, int R,
                            uint16_t* __restrict__ ring) {
    const long long n = (long long)B * R * (C / 8);
    for (long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x; idx < n;
         idx += (long long)gridDim.x * blockDim.x) {
        const int c8 = (int)(idx % (C / 8));
        const long long r = idx / (C / 8);
        const int lag = (int)(r % R) + 1;           // 1..R: token S - lag
        const int b = (int)(r / R);
        const long long s = (long long)S - lag;
        if (s < 0) continue;
        *reinterpret_cast<uint4*>(ring + ((long long)b * R + (int)(s % R)) * C + c8 * 8) =
            *reinterpret_cast<const uint4*>(out + ((long long)b * S + s) * C + c8 * 8);
    }
}

// halo rows for the next chunk of B sequences of S tokens: halo[b][r] = out of position
// S - R + r of sequence b (zero where that position is before the sequence start)
__global__ void k_halo_fill(const uint16_t* __restrict__ out, int B, int S, int C, int R,
                            uint16_t* __restrict__ halo) {
    const long long n = (long long)B * R * (C / 8);
    for (long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x; idx < n;
         idx += (long long)gridDim.x * blockDim.x) {
        const int c8 = (int)(idx % (C / 8));
        const long long br = idx / (C / 8);
        const int r = (int)(br % R);
        const long long b = br / R;
        const long long s = (long long)S - R + r;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (s >= 0) v = *reinterpret_cast<const uint4*>(out + (b * S + s) * C + c8 * 8);
        *reinterpret_cast<uint4*>(halo + br * C + c8 * 8) = v;
    }
}

// the gradient of a chunk's halo rows, returned to the chunk that produced them: d_out of
// position S - R + r of sequence b += d_halo[b][r] (in fp32, one bf16 rounding)
__global__ void k_halo_add(uint16_t* __restrict__ d_out, int B, int S, int C, int R,
                           const float* __restrict__ dhalo) {
    const long long n = (long long)B * R * (C / 2);
    for (long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x; idx < n;
         idx += (long long)gridDim.x * blockDim.x) {
        const int c2 = (int)(idx % (C / 2));
        const long long br = idx / (C / 2);
        const int r = (int)(br % R);
        const long long b = br / R;
        const long long s = (long long)S - R + r;
        if (s < 0) continue;
        uint32_t* p = reinterpret_cast<uint32_t*>(d_out + (b * S + s) * C + c2 * 2);
        const float2 g = *reinterpret_cast<const float2*>(dhalo + br * C + c2 * 2);
        const uint32_t u = *p;
        *p = pack2(__uint_as_float(u << 16) + g.x, __uint_as_float(u & 0xffff0000u) + g.y);
    }
}

int dec_slices(int C) { return (C + 2 * DTH - 1) / (2 * DTH); }

}  // namespace

cudaError_t launch_dec_gram(const Dims& d, int slot, int B, const uint16_t* out, ConvPtrs cw,
                            const uint16_t* ring, const long long* pos, float* red, cudaStream_t st) {
    const dim3 grid(dec_slices(d.C), (B + DT - 1) / DT);
    k_dec_gram<<<grid, DTH, 0, st>>>(d, slot, B, out, cw, ring, pos, dec_slices(d.C), red); note_launch();
    return cudaGetLastError();
}

int dec_nslice(int C) { return dec_slices(C); }

cudaError_t launch_dec_fwd(const Dims& d, int slot, int B, const uint16_t* out, ConvPtrs cw,
                           uint16_t* ring, long long* pos, const float* emat, const uint16_t* xact,
                           const int* I, const float* hres, uint16_t* xact_next, uint16_t* X,
                           cudaStream_t st) {
    const dim3 grid(dec_slices(d.C), (B + DT - 1) / DT);
    k_dec_fwd<<<grid, DTH, 0, st>>>(d, slot, B, out, cw, ring, pos, emat, xact, I, hres, xact_next,
                                    X); note_launch();
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || slot != d.G - 1) return e;
    k_pos_advance<<<(B + 255) / 256, 256, 0, st>>>(pos, B); note_launch();
    return cudaGetLastError();
}

cudaError_t launch_ring_fill(const Dims& d, int B, int S, const uint16_t* out, uint16_t* ring,
                             cudaStream_t st) {
    const int R = d.kapmax - 1;
    if (R <= 0) return cudaSuccess;
    const long long n = (long long)B * R * (d.C / 8);
    const int blocks = (int)std::min<long long>((n + 255) / 256, 4096);
    k_ring_fill<<<blocks, 256, 0, st>>>(out, B, S, d.C, R, ring); note_launch();
    return cudaGetLastError();
}

cudaError_t launch_halo_fill(const Dims& d, int B, int S, const uint16_t* out, uint16_t* halo,
                             cudaStream_t st) {
    const int R = d.kapmax - 1;
    if (R <= 0) return cudaSuccess;
    const long long n = (long long)B * R * (d.C / 8);
    const int blocks = (int)std::min<long long>((n + 255) / 256, 4096);
    k_halo_fill<<<blocks, 256, 0, st>>>(out, B, S, d.C, R, halo); note_launch();
    return cudaGetLastError();
}

cudaError_t launch_halo_add(const Dims& d, int B, int S, uint16_t* d_out, const float* dhalo,
                            cudaStream_t st) {
    const int R = d.kapmax - 1;
    if (R <= 0) return cudaSuccess;
    const long long n = (long long)B * R * (d.C / 2);
    const int blocks = (int)std::min<long long>((n + 255) / 256, 4096);
    k_halo_add<<<blocks, 256, 0, st>>>(d_out, B, S, d.C, R, dhalo); note_launch();
    return cudaGetLastError();
}

}  // namespace xhc
