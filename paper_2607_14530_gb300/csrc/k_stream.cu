// Streaming kernels of the connection op (HBM-bound, fp32 math on bf16 data):
//   read        second full-state pass: dense read of slot 0 (Eq. dense_read), non-active base
//               readouts of the later slots (Eq. app_four_sub_base), gather of the active
//               streams (Alg. 1 Gather)
//   input       input_t = base_t + sum_j H_pre_t[I_j] x_act_j (Eq. app_active_state_correction)
//   aug_gram    Gram matrix of u = [out, g_1..g_r] per token (Eq. aug, conv formula of
//               Sec. 3.3.4), one partial per 256-channel slice
//   post_apply  X_act_new = (H_res) X_act + p (H_post out_aug) (Eq. sparse_write_delta,
//               Eq. sparse_write) with the Gram-Schmidt basis of Eq. gs folded into per-token
//               coefficients on u; the last slot scatters into X
//   restore     put the saved entry rows back into X before the backward
//   bwd_reduce  per-token reductions of the write-back backward
//   bwd_apply   gradients of the write-back components and of the active state
//   bwd_conv    transpose of the causal conv and its weight-gradient partials
//   dinput_act  dense-read backward on the active streams (and dH_pre of the active streams)
//   full_dots   dH_pre of the non-active streams: <x_i, d_input_t>
#include "xhc_internal.cuh"

namespace xhc {

constexpr int ST = 128;        // threads of a channel-sliced block, 2 channels each
constexpr int SLICE = 2 * ST;  // channels per slice
constexpr int TBR = 8;         // tokens per block of the reduction kernels
constexpr int TBA = 16;        // tokens per block of the apply kernels
constexpr int TBC = 128;       // tokens per block of the conv-transpose kernel

__device__ __forceinline__ float2 ld_bf2(const uint16_t* p) {
    const uint32_t u = *reinterpret_cast<const uint32_t*>(p);
    return make_float2(__uint_as_float(u << 16), __uint_as_float(u & 0xffff0000u));
}
__device__ __forceinline__ void st_bf2(uint16_t* p, float2 v) {
    *reinterpret_cast<uint32_t*>(p) = pack2(v.x, v.y);
}
__device__ __forceinline__ float dot2(float2 a, float2 b) { return fmaf(a.x, b.x, a.y * b.y); }
__device__ __forceinline__ float2 fma2(float s, float2 a, float2 acc) {
    return make_float2(fmaf(s, a.x, acc.x), fmaf(s, a.y, acc.y));
}

// Conv taps of the block's slice in shared memory: taps[(off_j + i) * ST + tid] (float2).
__device__ __forceinline__ void load_taps(const Dims& d, const ConvPtrs& cw, int c0,
                                          float2* taps) {
    int off = 0;
    const int c = c0 + 2 * threadIdx.x;
    for (int j = 0; j < d.nconv; ++j) {
        for (int i = 0; i < d.kap[j]; ++i) {
            float2 v = make_float2(0.f, 0.f);
            if (c < d.C) v = make_float2(cw.w[j][i * d.C + c], cw.w[j][i * d.C + c + 1]);
            taps[(off + i) * ST + threadIdx.x] = v;
        }
        off += d.kap[j];
    }
}

// Write-back components of token t at channels c, c+1: u_0 = out, u_{1+j} = g_j where
// g_j[t] = sum_{i < kappa_j} w_j[i] out[t - i], zero before the sequence start.
__device__ __forceinline__ void comp_u(const Dims& d, int K, const uint16_t* out, int64_t t,
                                       int c, const float2* taps, float2 (&u)[MAXCOMP]) {
    u[0] = ld_bf2(out + t * d.C + c);
#pragma unroll
    for (int j = 1; j < MAXCOMP; ++j) u[j] = make_float2(0.f, 0.f);
    if (K == 1) return;
    const int pos = (int)(t % d.S);
    const int imax = min(d.kapmax, pos + 1);
    for (int i = 0; i < imax; ++i) {
        const float2 o = (i == 0) ? u[0] : ld_bf2(out + (t - i) * d.C + c);
        int off = 0;
#pragma unroll
        for (int j = 0; j < 3; ++j) {
            if (j < d.nconv) {
                if (i < d.kap[j]) {
                    const float2 w = taps[(off + i) * ST + threadIdx.x];
                    u[1 + j].x = fmaf(w.x, o.x, u[1 + j].x);
                    u[1 + j].y = fmaf(w.y, o.y, u[1 + j].y);
                }
                off += d.kap[j];
            }
        }
    }
}

static cudaError_t set_smem(const void* fn, size_t bytes) {
    if (bytes <= 48 * 1024) return cudaSuccess;
    return cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

static int chunk_threads(int C) {
    int th = ((C / 8 + 31) / 32) * 32;
    return th > 256 ? 256 : th;
}

// ---------------------------------------------------------------------------------------------
// read: one block per token, threads over 8-channel chunks.

__global__ void __launch_bounds__(256) k_read(Dims d, int T, const uint16_t* __restrict__ X,
                                              const float* __restrict__ hpre,
                                              const int* __restrict__ I,
                                              uint16_t* __restrict__ input0,
                                              float* __restrict__ base,
                                              uint16_t* __restrict__ xact0) {
    __shared__ float sh[4 * MAXN];
    __shared__ int slotmap[MAXN];
    const int t = blockIdx.x;
    const int N = d.N, G = d.G, C = d.C;
    for (int q = threadIdx.x; q < G * N; q += blockDim.x) sh[q] = hpre[(int64_t)t * G * N + q];
    for (int i = threadIdx.x; i < N; i += blockDim.x) {
        int j = -1;
        for (int q = 0; q < d.k; ++q)
            if (I[(int64_t)t * d.k + q] == i) j = q;
        slotmap[i] = j;
    }
    __syncthreads();
    const uint16_t* xt = X + (int64_t)t * N * C;
    for (int c8 = threadIdx.x; c8 < C / 8; c8 += blockDim.x) {
        float acc[4][8];
#pragma unroll
        for (int q = 0; q < 4; ++q)
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[q][e] = 0.f;
#pragma unroll 4
        for (int i = 0; i < N; ++i) {
            const uint4 u = __ldg(reinterpret_cast<const uint4*>(xt + (int64_t)i * C + c8 * 8));
            float x[8];
            unpack8(u, x);
            const int j = slotmap[i];
            const float h0 = sh[i];
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[0][e] = fmaf(h0, x[e], acc[0][e]);
            if (j < 0) {
#pragma unroll
                for (int q = 1; q < 4; ++q) {
                    if (q < G) {
                        const float h = sh[q * N + i];
#pragma unroll
                        for (int e = 0; e < 8; ++e) acc[q][e] = fmaf(h, x[e], acc[q][e]);
                    }
                }
            } else {
                *reinterpret_cast<uint4*>(xact0 + ((int64_t)t * d.k + j) * C + c8 * 8) = u;
            }
        }
        *reinterpret_cast<uint4*>(input0 + (int64_t)t * C + c8 * 8) = pack8(acc[0]);
#pragma unroll
        for (int q = 1; q < 4; ++q) {
            if (q < G) {
                float* bp = base + ((int64_t)(q - 1) * T + t) * C + c8 * 8;
                *reinterpret_cast<float4*>(bp) = make_float4(acc[q][0], acc[q][1], acc[q][2], acc[q][3]);
                *reinterpret_cast<float4*>(bp + 4) = make_float4(acc[q][4], acc[q][5], acc[q][6], acc[q][7]);
            }
        }
    }
}

cudaError_t launch_read(const Dims& d, int T, const uint16_t* X, const float* hpre, const int* I,
                        uint16_t* input0, float* base, uint16_t* xact0, cudaStream_t st) {
    k_read<<<T, chunk_threads(d.C), 0, st>>>(d, T, X, hpre, I, input0, base, xact0); note_launch();
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// input: slots >= 1

__global__ void __launch_bounds__(256) k_input(Dims d, int slot, int T,
                                               const float* __restrict__ base,
                                               const uint16_t* __restrict__ xact,
                                               const float* __restrict__ hpre,
                                               const int* __restrict__ I,
                                               uint16_t* __restrict__ input) {
    __shared__ float hj[MAXK];
    const int t = blockIdx.x, C = d.C;
    if (threadIdx.x < d.k)
        hj[threadIdx.x] = hpre[((int64_t)t * d.G + slot) * d.N + I[(int64_t)t * d.k + threadIdx.x]];
    __syncthreads();
    for (int c8 = threadIdx.x; c8 < C / 8; c8 += blockDim.x) {
        const float* bp = base + ((int64_t)(slot - 1) * T + t) * C + c8 * 8;
        const float4 b0 = *reinterpret_cast<const float4*>(bp);
        const float4 b1 = *reinterpret_cast<const float4*>(bp + 4);
        float acc[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
        for (int j = 0; j < d.k; ++j) {
            const uint4 u = *reinterpret_cast<const uint4*>(xact + ((int64_t)t * d.k + j) * C + c8 * 8);
            float x[8];
            unpack8(u, x);
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[e] = fmaf(hj[j], x[e], acc[e]);
        }
        *reinterpret_cast<uint4*>(input + (int64_t)t * C + c8 * 8) = pack8(acc);
    }
}

cudaError_t launch_input(const Dims& d, int slot, int T, const float* base, const uint16_t* xact,
                         const float* hpre, const int* I, uint16_t* input, cudaStream_t st) {
    k_input<<<T, chunk_threads(d.C), 0, st>>>(d, slot, T, base, xact, hpre, I, input); note_launch();
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// aug_gram: red[t][slice][q] = sum over the slice of u_a u_b, (a, b) with b <= a packed row-wise

__global__ void __launch_bounds__(ST) k_aug_gram(Dims d, int slot, int T,
                                                 const uint16_t* __restrict__ out, ConvPtrs cw,
                                                 int nslice, float* __restrict__ red) {
    extern __shared__ float2 taps[];
    __shared__ float wsh[TBR][4][16];
    const int slice = blockIdx.x, c0 = slice * SLICE, c = c0 + 2 * threadIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int K = d.K[slot];
    const int nq = K * (K + 1) / 2;
    load_taps(d, cw, c0, taps);
    __syncthreads();
    const int t0 = blockIdx.y * TBR;
    for (int tt = 0; tt < TBR; ++tt) {
        const int64_t t = t0 + tt;
        if (t >= T) break;
        float2 u[MAXCOMP];
        if (c < d.C) {
            comp_u(d, K, out, t, c, taps, u);
        } else {
#pragma unroll
            for (int a = 0; a < MAXCOMP; ++a) u[a] = make_float2(0.f, 0.f);
        }
        int q = 0;
#pragma unroll
        for (int a = 0; a < MAXCOMP; ++a)
#pragma unroll
            for (int b = 0; b <= a; ++b) {
                if (a < K) {
                    const float v = warp_sum(dot2(u[a], u[b]));
                    if (lane == 0) wsh[tt][warp][q] = v;
                    ++q;
                }
            }
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < TBR * nq; idx += ST) {
        const int tt = idx / nq, q = idx - tt * nq;
        const int64_t t = t0 + tt;
        if (t < T)
            red[(t * nslice + slice) * NRED + q] = wsh[tt][0][q] + wsh[tt][1][q] + wsh[tt][2][q] + wsh[tt][3][q];
    }
}

cudaError_t launch_aug_gram(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs convw,
                            int nslice, float* red, cudaStream_t st) {
    const size_t sm = (size_t)d.kapsum * ST * sizeof(float2);
    cudaError_t e = set_smem((const void*)k_aug_gram, sm);
    if (e != cudaSuccess) return e;
    dim3 grid(nslice, (T + TBR - 1) / TBR);
    k_aug_gram<<<grid, ST, sm, st>>>(d, slot, T, out, convw, nslice, red); note_launch();
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// post_apply

template <int KM>
__global__ void __launch_bounds__(ST) k_post_apply(Dims d, int slot, int T,
                                                   const uint16_t* __restrict__ out, ConvPtrs cw,
                                                   const float* __restrict__ red, int nslice,
                                                   const uint16_t* __restrict__ xact,
                                                   const int* __restrict__ I,
                                                   const float* __restrict__ p,
                                                   const float* __restrict__ hpost,
                                                   const float* __restrict__ hres,
                                                   uint16_t* __restrict__ xact_next,
                                                   uint16_t* __restrict__ X) {
    extern __shared__ float2 taps[];
    __shared__ float Esh[TBA][KM][MAXCOMP];
    __shared__ float Hsh[TBA][KM][KM];
    __shared__ int Ish[TBA][KM];
    const int k = d.k, K = d.K[slot], C = d.C;
    const bool last = (slot == d.G - 1);
    const bool gs = (K > 1) && d.gs;
    const int t0 = blockIdx.y * TBA;
    if (threadIdx.x < TBA) {
        const int tt = threadIdx.x;
        const int64_t t = t0 + tt;
        if (t < T) {
            double B[MAXCOMP][MAXCOMP];
            for (int a = 0; a < MAXCOMP; ++a)
                for (int b = 0; b < MAXCOMP; ++b) B[a][b] = (a == b) ? 1.0 : 0.0;
            if (gs) {
                double Gm[MAXCOMP][MAXCOMP], cc[MAXCOMP][MAXCOMP], vv[MAXCOMP];
                for (int a = 0; a < MAXCOMP; ++a)
                    for (int b = 0; b < MAXCOMP; ++b) Gm[a][b] = 0.0;
                for (int s = 0; s < nslice; ++s) {
                    const float* rp = red + (t * nslice + s) * NRED;
                    int q = 0;
                    for (int a = 0; a < K; ++a)
                        for (int b = 0; b <= a; ++b) Gm[a][b] += (double)rp[q++];
                }
                for (int a = 0; a < K; ++a)
                    for (int b = a + 1; b < K; ++b) Gm[a][b] = Gm[b][a];
                gs_coef(Gm, K, (double)d.eps_gs, B, cc, vv);
            }
            for (int j = 0; j < KM; ++j) {
                if (j >= k) break;
                const float pj = p[t * k + j];
                for (int a = 0; a < MAXCOMP; ++a) {
                    float e = 0.f;
                    if (a < K)
                        for (int q = 0; q < K; ++q) e += hpost[(t * k + j) * K + q] * (float)B[q][a];
                    Esh[tt][j][a] = pj * e;
                }
                Ish[tt][j] = I[t * k + j];
                if (last)
                    for (int i = 0; i < k; ++i) Hsh[tt][j][i] = hres[t * k * k + j * k + i];
            }
        }
    }
    const int c0 = blockIdx.x * SLICE, c = c0 + 2 * threadIdx.x;
    if (K > 1) load_taps(d, cw, c0, taps);
    __syncthreads();
    if (c >= C) return;
    for (int tt = 0; tt < TBA; ++tt) {
        const int64_t t = t0 + tt;
        if (t >= T) break;
        float2 u[MAXCOMP];
        comp_u(d, K, out, t, c, taps, u);
        float2 x[KM];
#pragma unroll
        for (int j = 0; j < KM; ++j)
            x[j] = (j < k) ? ld_bf2(xact + (t * k + j) * C + c) : make_float2(0.f, 0.f);
#pragma unroll
        for (int j = 0; j < KM; ++j) {
            if (j >= k) continue;
            float2 v;
            if (last) {
                v = make_float2(0.f, 0.f);
#pragma unroll
                for (int i = 0; i < KM; ++i)
                    if (i < k) v = fma2(Hsh[tt][j][i], x[i], v);
            } else {
                v = x[j];
            }
#pragma unroll
            for (int a = 0; a < MAXCOMP; ++a)
                if (a < K) v = fma2(Esh[tt][j][a], u[a], v);
            if (last)
                st_bf2(X + (t * d.N + Ish[tt][j]) * C + c, v);
            else
                st_bf2(xact_next + (t * k + j) * C + c, v);
        }
    }
}

cudaError_t launch_post_apply(const Dims& d, int slot, int T, const uint16_t* out,
                              ConvPtrs convw, const float* red, int nslice, const uint16_t* xact,
                              const int* I, const float* p, const float* hpost, const float* hres,
                              uint16_t* xact_next, uint16_t* X, cudaStream_t st) {
    const size_t sm = (d.K[slot] > 1) ? (size_t)d.kapsum * ST * sizeof(float2) : 0;
    dim3 grid(nslice, (T + TBA - 1) / TBA);
    cudaError_t e;
    if (d.k <= 4) {
        e = set_smem((const void*)k_post_apply<4>, sm);
        if (e != cudaSuccess) return e;
        k_post_apply<4><<<grid, ST, sm, st>>>(d, slot, T, out, convw, red, nslice, xact, I, p, hpost,
                                              hres, xact_next, X); note_launch();
    } else {
        e = set_smem((const void*)k_post_apply<8>, sm);
        if (e != cudaSuccess) return e;
        k_post_apply<8><<<grid, ST, sm, st>>>(d, slot, T, out, convw, red, nslice, xact, I, p, hpost,
                                              hres, xact_next, X); note_launch();
    }
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// restore: X[t][I_j] = X_act^(0)[t][j]

__global__ void __launch_bounds__(256) k_restore(Dims d, int T, const uint16_t* __restrict__ xact0,
                                                 const int* __restrict__ I,
                                                 uint16_t* __restrict__ X) {
    const int t = blockIdx.x, C = d.C;
    const int n8 = C / 8;
    for (int idx = threadIdx.x; idx < d.k * n8; idx += blockDim.x) {
        const int j = idx / n8, c8 = idx - j * n8;
        const int i = I[(int64_t)t * d.k + j];
        *reinterpret_cast<uint4*>(X + ((int64_t)t * d.N + i) * C + c8 * 8) =
            *reinterpret_cast<const uint4*>(xact0 + ((int64_t)t * d.k + j) * C + c8 * 8);
    }
}

cudaError_t launch_restore(const Dims& d, int T, const uint16_t* xact0, const int* I,
                           uint16_t* X, cudaStream_t st) {
    k_restore<<<T, 256, 0, st>>>(d, T, xact0, I, X); note_launch();
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// bwd_reduce: per token and slice
//   P[j][a] = <dXn_j, u_a>  (k*K)      Q[j][i] = <dXn_j, x_act_i>  (k*k, last slot)
//   Gm[a][b] = <u_a, u_b>, b <= a      (Gram-Schmidt on)
// dXn is the gradient w.r.t. the slot's output active state: dX rows I (last slot) or the
// workspace active gradient.

template <int KM>
__global__ void __launch_bounds__(ST) k_bwd_reduce(Dims d, int slot, int T,
                                                   const uint16_t* __restrict__ out, ConvPtrs cw,
                                                   const uint16_t* __restrict__ dX,
                                                   const int* __restrict__ I,
                                                   const float* __restrict__ dxact,
                                                   const uint16_t* __restrict__ xact, int nslice,
                                                   float* __restrict__ red) {
    extern __shared__ float2 taps[];
    __shared__ float wsh[TBR][4][NRED];
    const int slice = blockIdx.x, c0 = slice * SLICE, c = c0 + 2 * threadIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int k = d.k, K = d.K[slot], C = d.C;
    const bool last = (slot == d.G - 1);
    const bool gs = (K > 1) && d.gs;
    const int nv = k * K + (last ? k * k : 0) + (gs ? K * (K + 1) / 2 : 0);
    if (K > 1) load_taps(d, cw, c0, taps);
    __syncthreads();
    const int t0 = blockIdx.y * TBR;
    for (int tt = 0; tt < TBR; ++tt) {
        const int64_t t = t0 + tt;
        if (t >= T) break;
        float2 u[MAXCOMP], dn[KM], x[KM];
#pragma unroll
        for (int j = 0; j < KM; ++j) {
            dn[j] = make_float2(0.f, 0.f);
            x[j] = make_float2(0.f, 0.f);
        }
#pragma unroll
        for (int a = 0; a < MAXCOMP; ++a) u[a] = make_float2(0.f, 0.f);
        if (c < C) {
#pragma unroll
            for (int j = 0; j < KM; ++j) {
                if (j >= k) continue;
                if (last) {
                    dn[j] = ld_bf2(dX + (t * d.N + I[t * k + j]) * C + c);
                    x[j] = ld_bf2(xact + (t * k + j) * C + c);
                } else {
                    dn[j] = *reinterpret_cast<const float2*>(dxact + (t * k + j) * C + c);
                }
            }
            comp_u(d, K, out, t, c, taps, u);
        }
        int q = 0;
#pragma unroll
        for (int j = 0; j < KM; ++j)
#pragma unroll
            for (int a = 0; a < MAXCOMP; ++a)
                if (j < k && a < K) {
                    const float v = warp_sum(dot2(dn[j], u[a]));
                    if (lane == 0) wsh[tt][warp][q] = v;
                    ++q;
                }
        if (last) {
#pragma unroll
            for (int j = 0; j < KM; ++j)
#pragma unroll
                for (int i = 0; i < KM; ++i)
                    if (j < k && i < k) {
                        const float v = warp_sum(dot2(dn[j], x[i]));
                        if (lane == 0) wsh[tt][warp][q] = v;
                        ++q;
                    }
        }
        if (gs) {
#pragma unroll
            for (int a = 0; a < MAXCOMP; ++a)
#pragma unroll
                for (int b = 0; b <= a; ++b)
                    if (a < K) {
                        const float v = warp_sum(dot2(u[a], u[b]));
                        if (lane == 0) wsh[tt][warp][q] = v;
                        ++q;
                    }
        }
    }
    __syncthreads();
    for (int idx = threadIdx.x; idx < TBR * nv; idx += ST) {
        const int tt = idx / nv, q = idx - tt * nv;
        const int64_t t = t0 + tt;
        if (t < T)
            red[(t * nslice + slice) * NRED + q] = wsh[tt][0][q] + wsh[tt][1][q] + wsh[tt][2][q] + wsh[tt][3][q];
    }
}

cudaError_t launch_bwd_reduce(const Dims& d, int slot, int T, const uint16_t* out,
                              ConvPtrs convw, const uint16_t* dX, const int* I, const float* dxact,
                              const uint16_t* xact, int nslice, float* red, cudaStream_t st) {
    const size_t sm = (d.K[slot] > 1) ? (size_t)d.kapsum * ST * sizeof(float2) : 0;
    dim3 grid(nslice, (T + TBR - 1) / TBR);
    cudaError_t e;
    if (d.k <= 4) {
        e = set_smem((const void*)k_bwd_reduce<4>, sm);
        if (e != cudaSuccess) return e;
        k_bwd_reduce<4><<<grid, ST, sm, st>>>(d, slot, T, out, convw, dX, I, dxact, xact, nslice, red); note_launch();
    } else {
        e = set_smem((const void*)k_bwd_reduce<8>, sm);
        if (e != cudaSuccess) return e;
        k_bwd_reduce<8><<<grid, ST, sm, st>>>(d, slot, T, out, convw, dX, I, dxact, xact, nslice, red); note_launch();
    }
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// bwd_apply: per token and channel pair
//   du_a      = sum_j E[j][a] dXn_j + sum_b D[a][b] u_b        (d out, d g_j)
//   dX_act_i  = sum_j H_res[j][i] dXn_j (last slot) or dXn_i, minus cx * x_act_i
// K == 1 writes d_out directly; otherwise du goes to the workspace for bwd_conv.

template <int KM>
__global__ void __launch_bounds__(ST) k_bwd_apply(Dims d, int slot, int T,
                                                  const uint16_t* __restrict__ out, ConvPtrs cw,
                                                  const uint16_t* __restrict__ dX,
                                                  const int* __restrict__ I,
                                                  const uint16_t* __restrict__ xact,
                                                  const float* __restrict__ tokmat,
                                                  float* __restrict__ dxact,
                                                  float* __restrict__ du,
                                                  uint16_t* __restrict__ d_out) {
    extern __shared__ float2 taps[];
    __shared__ float Esh[TBA][KM][MAXCOMP];
    __shared__ float Dsh[TBA][MAXCOMP][MAXCOMP];
    __shared__ float Hsh[TBA][KM][KM];
    __shared__ float cxs[TBA];
    __shared__ int Ish[TBA][KM];
    const int k = d.k, K = d.K[slot], C = d.C;
    const bool last = (slot == d.G - 1);
    const int t0 = blockIdx.y * TBA;
    for (int idx = threadIdx.x; idx < TBA * 128; idx += ST) {
        const int tt = idx >> 7, q = idx & 127;
        const int64_t t = t0 + tt;
        if (t >= T) continue;
        const float v = tokmat[t * TOKMAT + q];
        if (q < 32) {
            const int j = q >> 2, a = q & 3;
            if (j < KM) Esh[tt][j][a] = v;
        } else if (q < 48) {
            Dsh[tt][(q - 32) >> 2][(q - 32) & 3] = v;
        } else if (q < 112) {
            const int a = (q - 48) >> 3, b = (q - 48) & 7;
            if (a < KM && b < KM) Hsh[tt][a][b] = v;
        } else if (q == 112) {
            cxs[tt] = v;
        } else if (q >= 120 && q < 120 + KM) {
            Ish[tt][q - 120] = (q - 120 < k) ? I[t * k + (q - 120)] : 0;
        }
    }
    const int c0 = blockIdx.x * SLICE, c = c0 + 2 * threadIdx.x;
    if (K > 1) load_taps(d, cw, c0, taps);
    __syncthreads();
    if (c >= C) return;
    for (int tt = 0; tt < TBA; ++tt) {
        const int64_t t = t0 + tt;
        if (t >= T) break;
        float2 u[MAXCOMP], dn[KM], x[KM];
#pragma unroll
        for (int j = 0; j < KM; ++j) {
            if (j < k) {
                dn[j] = last ? ld_bf2(dX + (t * d.N + Ish[tt][j]) * C + c)
                             : *reinterpret_cast<const float2*>(dxact + (t * k + j) * C + c);
                x[j] = ld_bf2(xact + (t * k + j) * C + c);
            } else {
                dn[j] = make_float2(0.f, 0.f);
                x[j] = make_float2(0.f, 0.f);
            }
        }
        comp_u(d, K, out, t, c, taps, u);
#pragma unroll
        for (int a = 0; a < MAXCOMP; ++a) {
            if (a >= K) continue;
            float2 g = make_float2(0.f, 0.f);
#pragma unroll
            for (int j = 0; j < KM; ++j)
                if (j < k) g = fma2(Esh[tt][j][a], dn[j], g);
#pragma unroll
            for (int b = 0; b < MAXCOMP; ++b)
                if (b < K) g = fma2(Dsh[tt][a][b], u[b], g);
            if (K == 1)
                st_bf2(d_out + t * C + c, g);
            else
                *reinterpret_cast<float2*>(du + (t * K + a) * C + c) = g;
        }
        const float cx = cxs[tt];
#pragma unroll
        for (int i = 0; i < KM; ++i) {
            if (i >= k) continue;
            float2 v;
            if (last) {
                v = make_float2(0.f, 0.f);
#pragma unroll
                for (int j = 0; j < KM; ++j)
                    if (j < k) v = fma2(Hsh[tt][j][i], dn[j], v);
            } else {
                v = dn[i];
            }
            v = fma2(-cx, x[i], v);
            *reinterpret_cast<float2*>(dxact + (t * k + i) * C + c) = v;
        }
    }
}

cudaError_t launch_bwd_apply(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs convw,
                             const uint16_t* dX, const int* I, const uint16_t* xact,
                             const float* tokmat, float* dxact, float* du, uint16_t* d_out,
                             cudaStream_t st) {
    const size_t sm = (d.K[slot] > 1) ? (size_t)d.kapsum * ST * sizeof(float2) : 0;
    const int nslice = (d.C + SLICE - 1) / SLICE;
    dim3 grid(nslice, (T + TBA - 1) / TBA);
    cudaError_t e;
    if (d.k <= 4) {
        e = set_smem((const void*)k_bwd_apply<4>, sm);
        if (e != cudaSuccess) return e;
        k_bwd_apply<4><<<grid, ST, sm, st>>>(d, slot, T, out, convw, dX, I, xact, tokmat, dxact, du, d_out); note_launch();
    } else {
        e = set_smem((const void*)k_bwd_apply<8>, sm);
        if (e != cudaSuccess) return e;
        k_bwd_apply<8><<<grid, ST, sm, st>>>(d, slot, T, out, convw, dX, I, xact, tokmat, dxact, du, d_out); note_launch();
    }
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// bwd_conv: d_out[t] = du_0[t] + sum_j sum_i w_j[i] du_{1+j}[t + i] (same sequence);
//           cpart[tile][off_j + i][c] = sum_{t in tile, pos(t) >= i} du_{1+j}[t] out[t - i]

__global__ void __launch_bounds__(ST) k_bwd_conv(Dims d, int slot, int T,
                                                 const uint16_t* __restrict__ out, ConvPtrs cw,
                                                 const float* __restrict__ du,
                                                 uint16_t* __restrict__ d_out,
                                                 float* __restrict__ cpart) {
    extern __shared__ float2 sm2[];
    float2* taps = sm2;
    float2* acc = sm2 + d.kapsum * ST;
    const int K = d.K[slot], C = d.C;
    const int c0 = blockIdx.x * SLICE, c = c0 + 2 * threadIdx.x;
    load_taps(d, cw, c0, taps);
    for (int q = 0; q < d.kapsum; ++q) acc[q * ST + threadIdx.x] = make_float2(0.f, 0.f);
    __syncthreads();
    if (c >= C) return;
    const int t0 = blockIdx.y * TBC;
    for (int tt = 0; tt < TBC; ++tt) {
        const int64_t t = t0 + tt;
        if (t >= T) break;
        const int pos = (int)(t % d.S);
        float2 r = *reinterpret_cast<const float2*>(du + (t * K + 0) * C + c);
        int off = 0;
        for (int j = 0; j < d.nconv; ++j) {
            const float2 g = *reinterpret_cast<const float2*>(du + (t * K + 1 + j) * C + c);
            for (int i = 0; i < d.kap[j]; ++i) {
                const float2 w = taps[(off + i) * ST + threadIdx.x];
                if (pos + i < d.S && t + i < T) {
                    const float2 gf = *reinterpret_cast<const float2*>(du + ((t + i) * K + 1 + j) * C + c);
                    r.x = fmaf(w.x, gf.x, r.x);
                    r.y = fmaf(w.y, gf.y, r.y);
                }
                if (pos >= i) {
                    const float2 o = ld_bf2(out + (t - i) * C + c);
                    float2& a = acc[(off + i) * ST + threadIdx.x];
                    a.x = fmaf(g.x, o.x, a.x);
                    a.y = fmaf(g.y, o.y, a.y);
                }
            }
            off += d.kap[j];
        }
        st_bf2(d_out + t * C + c, r);
    }
    for (int q = 0; q < d.kapsum; ++q)
        *reinterpret_cast<float2*>(cpart + ((int64_t)blockIdx.y * d.kapsum + q) * C + c) = acc[q * ST + threadIdx.x];
}

cudaError_t launch_bwd_conv(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs convw,
                            const float* du, uint16_t* d_out, float* cpart, int ntiles,
                            cudaStream_t st) {
    const size_t sm = 2 * (size_t)d.kapsum * ST * sizeof(float2);
    cudaError_t e = set_smem((const void*)k_bwd_conv, sm);
    if (e != cudaSuccess) return e;
    const int nslice = (d.C + SLICE - 1) / SLICE;
    (void)ntiles;
    dim3 grid(nslice, (T + TBC - 1) / TBC);
    k_bwd_conv<<<grid, ST, sm, st>>>(d, slot, T, out, convw, du, d_out, cpart); note_launch();
    return cudaGetLastError();
}

__global__ void k_conv_wgrad_reduce(Dims d, const float* __restrict__ cpart, int ntiles,
                                    ConvGradPtrs g) {
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= d.kapsum * d.C) return;
    const int q = idx / d.C, c = idx - q * d.C;
    float s = 0.f;
    for (int tile = 0; tile < ntiles; ++tile) s += cpart[((int64_t)tile * d.kapsum + q) * d.C + c];
    int j = 0, off = 0;
    while (q >= off + d.kap[j]) {
        off += d.kap[j];
        ++j;
    }
    g.w[j][(q - off) * d.C + c] += s;
}

cudaError_t launch_conv_wgrad_reduce(const Dims& d, int slot, const float* cpart, int ntiles,
                                     ConvGradPtrs gconv, cudaStream_t st) {
    (void)slot;
    const int n = d.kapsum * d.C;
    k_conv_wgrad_reduce<<<(n + 255) / 256, 256, 0, st>>>(d, cpart, ntiles, gconv); note_launch();
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// dinput_act: dX_act[t][j] += H_pre_slot[I_j] d_input;  dH_pre_slot[I_j] = <x_act_j, d_input>;
// d_input is copied to the workspace for the full-state backward of slot 0.

template <int KM>
__global__ void __launch_bounds__(256) k_dinput_act(Dims d, int slot, int T, int add_dx,
                                                    const uint16_t* __restrict__ din,
                                                    const uint16_t* __restrict__ xact,
                                                    const float* __restrict__ hpre,
                                                    const int* __restrict__ I,
                                                    float* __restrict__ dxact,
                                                    float* __restrict__ dhpre,
                                                    uint16_t* __restrict__ dcopy) {
    __shared__ float hj[KM];
    __shared__ float wsh[8][KM];
    const int t = blockIdx.x, C = d.C, k = d.k;
    if (threadIdx.x < k)
        hj[threadIdx.x] = hpre[((int64_t)t * d.G + slot) * d.N + I[(int64_t)t * k + threadIdx.x]];
    __syncthreads();
    float dot[KM];
#pragma unroll
    for (int j = 0; j < KM; ++j) dot[j] = 0.f;
    for (int c8 = threadIdx.x; c8 < C / 8; c8 += blockDim.x) {
        const uint4 du8 = *reinterpret_cast<const uint4*>(din + (int64_t)t * C + c8 * 8);
        *reinterpret_cast<uint4*>(dcopy + ((int64_t)slot * T + t) * C + c8 * 8) = du8;
        float g[8];
        unpack8(du8, g);
#pragma unroll
        for (int j = 0; j < KM; ++j) {
            if (j >= k) continue;
            float x[8];
            unpack8(*reinterpret_cast<const uint4*>(xact + ((int64_t)t * k + j) * C + c8 * 8), x);
#pragma unroll
            for (int e = 0; e < 8; ++e) dot[j] = fmaf(x[e], g[e], dot[j]);
            if (!add_dx) continue;
            float* dp = dxact + ((int64_t)t * k + j) * C + c8 * 8;
            float4 a = *reinterpret_cast<float4*>(dp);
            float4 b = *reinterpret_cast<float4*>(dp + 4);
            const float h = hj[j];
            a.x = fmaf(h, g[0], a.x); a.y = fmaf(h, g[1], a.y); a.z = fmaf(h, g[2], a.z); a.w = fmaf(h, g[3], a.w);
            b.x = fmaf(h, g[4], b.x); b.y = fmaf(h, g[5], b.y); b.z = fmaf(h, g[6], b.z); b.w = fmaf(h, g[7], b.w);
            *reinterpret_cast<float4*>(dp) = a;
            *reinterpret_cast<float4*>(dp + 4) = b;
        }
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int j = 0; j < KM; ++j) {
        const float v = warp_sum(dot[j]);
        if (lane == 0) wsh[warp][j] = v;
    }
    __syncthreads();
    if (threadIdx.x < k) {
        const int nw = (blockDim.x + 31) / 32;
        float s = 0.f;
        for (int w = 0; w < nw; ++w) s += wsh[w][threadIdx.x];
        dhpre[((int64_t)t * d.G + slot) * d.N + I[(int64_t)t * k + threadIdx.x]] = s;
    }
}

cudaError_t launch_dinput_act(const Dims& d, int slot, int T, int add_dx, const uint16_t* d_input,
                              const uint16_t* xact, const float* hpre, const int* I, float* dxact,
                              float* dhpre, uint16_t* dinput_copy, cudaStream_t st) {
    if (d.k <= 4) {
        k_dinput_act<4><<<T, chunk_threads(d.C), 0, st>>>(d, slot, T, add_dx, d_input, xact, hpre, I, dxact,
                                                           dhpre, dinput_copy); note_launch();
    } else {
        k_dinput_act<8><<<T, chunk_threads(d.C), 0, st>>>(d, slot, T, add_dx, d_input, xact, hpre, I, dxact,
                                                           dhpre, dinput_copy); note_launch();
    }
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// full_dots: for the non-active streams i, dH_pre[t][q][i] = <x_i, d_input_q> and the dense-read
// gradient dX[t][i] += sum_q H_pre[t][q][i] d_input_q (Eq. dense_read reversed)

__global__ void __launch_bounds__(256) k_full_dots(Dims d, int T, const uint16_t* __restrict__ X,
                                                   const uint16_t* __restrict__ dinput,
                                                   const int* __restrict__ I,
                                                   const float* __restrict__ hpre,
                                                   uint16_t* __restrict__ dX,
                                                   float* __restrict__ dhpre) {
    __shared__ float wsh[8][4];
    __shared__ int active[MAXN];
    __shared__ float hs[4 * MAXN];
    const int t = blockIdx.x, C = d.C, G = d.G;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nw = (blockDim.x + 31) / 32;
    for (int i = threadIdx.x; i < d.N; i += blockDim.x) {
        int a = 0;
        for (int q = 0; q < d.k; ++q)
            if (I[(int64_t)t * d.k + q] == i) a = 1;
        active[i] = a;
    }
    for (int q = threadIdx.x; q < G * d.N; q += blockDim.x) hs[q] = hpre[(int64_t)t * G * d.N + q];
    __syncthreads();
    for (int i = 0; i < d.N; ++i) {
        if (active[i]) continue;
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
        for (int c8 = threadIdx.x; c8 < C / 8; c8 += blockDim.x) {
            float x[8], dx[8];
            const int64_t off = ((int64_t)t * d.N + i) * C + c8 * 8;
            unpack8(__ldg(reinterpret_cast<const uint4*>(X + off)), x);
            unpack8(*reinterpret_cast<const uint4*>(dX + off), dx);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                if (q >= G) continue;
                float g[8];
                unpack8(*reinterpret_cast<const uint4*>(dinput + ((int64_t)q * T + t) * C + c8 * 8), g);
                const float h = hs[q * d.N + i];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    acc[q] = fmaf(x[e], g[e], acc[q]);
                    dx[e] = fmaf(h, g[e], dx[e]);
                }
            }
            *reinterpret_cast<uint4*>(dX + off) = pack8(dx);
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float v = warp_sum(acc[q]);
            if (lane == 0) wsh[warp][q] = v;
        }
        __syncthreads();
        if (threadIdx.x < G) {
            float s = 0.f;
            for (int w = 0; w < nw; ++w) s += wsh[w][threadIdx.x];
            dhpre[((int64_t)t * G + threadIdx.x) * d.N + i] = s;
        }
        __syncthreads();
    }
}

cudaError_t launch_full_dots(const Dims& d, int T, const uint16_t* X, const uint16_t* dinput,
                             const int* I, const float* hpre, uint16_t* dX, float* dhpre,
                             cudaStream_t st) {
    k_full_dots<<<T, chunk_threads(d.C), 0, st>>>(d, T, X, dinput, I, hpre, dX, dhpre); note_launch();
    return cudaGetLastError();
}

}  // namespace xhc
