// Streaming kernels of the connection op (HBM-bound, fp32 math on bf16 data):
//   read        second full-state pass: dense read of slot 0 (Eq. dense_read), non-active base
//               readouts of the later slots (Eq. app_four_sub_base; stored in bf16, as the
//               paper's traffic model stores them), gather of the active streams (Alg. 1
//               Gather), sum of squares of the gathered rows
//   input       input_t = base_t + sum_j H_pre_t[I_j] x_act_j (Eq. app_active_state_correction),
//               sum of squares of x_act
//   (the sums of squares are the norm statistics of the slot's active-state projection, which
//   then reads its operand only through the tensor-core pipeline)
//   restore     put the saved entry rows back into X before the backward
//   conv_wgrad_reduce  sum of the per-run conv weight-gradient partials
//   dinput_act  dense-read backward on the active streams (and dH_pre of the active streams)
//   full_dots   dH_pre of the non-active streams: <x_i, d_input_t>
#include "xhc_internal.cuh"

namespace xhc {

static int chunk_threads(int C) {
    int th = ((C / 8 + 31) / 32) * 32;
    return th > 256 ? 256 : th;
}

// ---------------------------------------------------------------------------------------------
// the block's warps each store their partial of a per-token sum: slot w of [warps][T][2], entry 1
// (no block barrier, so the block retires as soon as its stores are issued)
__device__ __forceinline__ void warp_partial(float v, float* __restrict__ dst, int T, int t) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if ((threadIdx.x & 31) == 0) dst[((int64_t)(threadIdx.x >> 5) * T + t) * 2 + 1] = v;
}

int stream_warps(int C) { return chunk_threads(C) / 32; }

// ---------------------------------------------------------------------------------------------
// read: one block per token, threads over 8-channel chunks.

__global__ void __launch_bounds__(256, 3) k_read(Dims d, int T, const uint16_t* __restrict__ X,
                                              const float* __restrict__ hpre,
                                              const int* __restrict__ I,
                                              uint16_t* __restrict__ input0,
                                              uint16_t* __restrict__ base,
                                              uint16_t* __restrict__ xact0,
                                              float* __restrict__ astat) {
    __shared__ float sh[4 * MAXN];
    __shared__ int slotmap[MAXN];
    const int t = blockIdx.x;
    const int N = d.N, G = d.G, C = d.C;
    const uint16_t* xt = X + (int64_t)t * N * C;
    // the first 8 streams of this thread's first chunk are read before the coefficient set-up
    uint4 ub[8];
    if (threadIdx.x < C / 8) {
#pragma unroll
        for (int ii = 0; ii < 8; ++ii)
            if (ii < N) ub[ii] = __ldg(reinterpret_cast<const uint4*>(xt + (int64_t)ii * C + threadIdx.x * 8));
    }
    for (int q = threadIdx.x; q < G * N; q += blockDim.x) sh[q] = hpre[(int64_t)t * G * N + q];
    for (int i = threadIdx.x; i < N; i += blockDim.x) {
        int j = -1;
        for (int q = 0; q < d.k; ++q)
            if (I[(int64_t)t * d.k + q] == i) j = q;
        slotmap[i] = j;
    }
    __syncthreads();
    float ss = 0.f;  // sum of squares of the gathered active rows (their projection's norm)
    for (int c8 = threadIdx.x; c8 < C / 8; c8 += blockDim.x) {
        float acc[4][8];
#pragma unroll
        for (int q = 0; q < 4; ++q)
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[q][e] = 0.f;
        // streams in blocks of 8: the block's 8 reads are issued before any is used
        for (int i0 = 0; i0 < N; i0 += 8) {
            if (i0 != 0 || c8 != (int)threadIdx.x) {
#pragma unroll
                for (int ii = 0; ii < 8; ++ii)
                    if (i0 + ii < N) ub[ii] = __ldg(reinterpret_cast<const uint4*>(xt + (int64_t)(i0 + ii) * C + c8 * 8));
            }
#pragma unroll
            for (int ii = 0; ii < 8; ++ii) {
                const int i = i0 + ii;
                if (i >= N) continue;
                float x[8];
                unpack8(ub[ii], x);
                const int j = slotmap[i];
                // sparse-read ablation: the non-active streams are not read
                const float h0 = (j >= 0 || d.dense) ? sh[i] : 0.f;
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[0][e] = fmaf(h0, x[e], acc[0][e]);
                if (j < 0) {
                    if (d.dense) {
#pragma unroll
                        for (int q = 1; q < 4; ++q) {
                            if (q < G) {
                                const float h = sh[q * N + i];
#pragma unroll
                                for (int e = 0; e < 8; ++e) acc[q][e] = fmaf(h, x[e], acc[q][e]);
                            }
                        }
                    }
                } else {
                    *reinterpret_cast<uint4*>(xact0 + ((int64_t)t * d.k + j) * C + c8 * 8) = ub[ii];
#pragma unroll
                    for (int e = 0; e < 8; ++e) ss = fmaf(x[e], x[e], ss);
                }
            }
        }
        *reinterpret_cast<uint4*>(input0 + (int64_t)t * C + c8 * 8) = pack8(acc[0]);
#pragma unroll
        for (int q = 1; q < 4; ++q)
            if (q < G)
                *reinterpret_cast<uint4*>(base + ((int64_t)(q - 1) * T + t) * C + c8 * 8) = pack8(acc[q]);
    }
    warp_partial(ss, astat, T, t);
}

cudaError_t launch_read(const Dims& d, int T, const uint16_t* X, const float* hpre, const int* I,
                        uint16_t* input0, uint16_t* base, uint16_t* xact0, float* astat, cudaStream_t st) {
    k_read<<<T, chunk_threads(d.C), 0, st>>>(d, T, X, hpre, I, input0, base, xact0, astat); note_launch();
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// input: slots >= 1

template <int KM>
__global__ void __launch_bounds__(256) k_input(Dims d, int slot, int T,
                                               const uint16_t* __restrict__ base,
                                               const uint16_t* __restrict__ xact,
                                               const float* __restrict__ hpre,
                                               const int* __restrict__ I,
                                               uint16_t* __restrict__ input,
                                               float* __restrict__ astat) {
    const int t = blockIdx.x, C = d.C, k = d.k;
    const int lane = threadIdx.x & 31;
    // the reads of this thread's first chunk (base row, k active rows) are issued before the
    // coefficients, which every warp fetches for itself (lanes j < k, then broadcast: no block
    // barrier)
    uint4 bb, xx[KM];
    auto load = [&](int c8) {
        bb = *reinterpret_cast<const uint4*>(base + ((int64_t)(slot - 1) * T + t) * C + c8 * 8);
#pragma unroll
        for (int j = 0; j < KM; ++j)
            if (j < k) xx[j] = *reinterpret_cast<const uint4*>(xact + ((int64_t)t * k + j) * C + c8 * 8);
    };
    if ((int)threadIdx.x < C / 8) load(threadIdx.x);
    float hl = 0.f;
    if (lane < k) hl = hpre[((int64_t)t * d.G + slot) * d.N + I[(int64_t)t * k + lane]];
    float hj[KM];
#pragma unroll
    for (int j = 0; j < KM; ++j) hj[j] = __shfl_sync(0xffffffffu, hl, j);
    float ss = 0.f;  // sum of squares of the active state (its projection's norm)
    for (int c8 = threadIdx.x; c8 < C / 8; c8 += blockDim.x) {
        if (c8 != (int)threadIdx.x) load(c8);
        float acc[8];
        unpack8(bb, acc);
#pragma unroll
        for (int j = 0; j < KM; ++j) {
            if (j >= k) break;
            float x[8];
            unpack8(xx[j], x);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                acc[e] = fmaf(hj[j], x[e], acc[e]);
                ss = fmaf(x[e], x[e], ss);
            }
        }
        *reinterpret_cast<uint4*>(input + (int64_t)t * C + c8 * 8) = pack8(acc);
    }
    warp_partial(ss, astat, T, t);
}

cudaError_t launch_input(const Dims& d, int slot, int T, const uint16_t* base, const uint16_t* xact,
                         const float* hpre, const int* I, uint16_t* input, float* astat, cudaStream_t st) {
    if (d.k <= 4) {
        k_input<4><<<T, chunk_threads(d.C), 0, st>>>(d, slot, T, base, xact, hpre, I, input, astat); note_launch();
    } else {
        k_input<8><<<T, chunk_threads(d.C), 0, st>>>(d, slot, T, base, xact, hpre, I, input, astat); note_launch();
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
// conv weight gradient: sum of the per-run partials

__global__ void k_conv_wgrad_reduce(Dims d, const float* __restrict__ cpart, int ntiles,
                                    ConvGradPtrs g) {
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= d.kapsum * d.C) return;
    const int q = idx / d.C, c = idx - q * d.C;
    // four interleaved partial sums over the runs, added in a fixed order
    const float* p = cpart + (int64_t)q * d.C + c;
    const int64_t step = (int64_t)d.kapsum * d.C;
    float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
    int tile = 0;
    for (; tile + 4 <= ntiles; tile += 4) {
        s0 += p[(int64_t)tile * step];
        s1 += p[(int64_t)(tile + 1) * step];
        s2 += p[(int64_t)(tile + 2) * step];
        s3 += p[(int64_t)(tile + 3) * step];
    }
    for (; tile < ntiles; ++tile) s0 += p[(int64_t)tile * step];
    const float s = (s0 + s1) + (s2 + s3);
    // the component of row q, selected with static indices (no local copy of the parameters)
    const int off1 = d.kap[0], off2 = d.kap[0] + d.kap[1];
    const int j = q >= off2 ? 2 : (q >= off1 ? 1 : 0);
    const int off = j == 2 ? off2 : (j == 1 ? off1 : 0);
    float* w = j == 2 ? g.w[2] : (j == 1 ? g.w[1] : g.w[0]);
    w[(q - off) * d.C + c] += s;
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
                                                    uint16_t* __restrict__ dcopy,
                                                    const float* __restrict__ tokmat) {
    __shared__ float hj[KM];
    __shared__ float wsh[8][KM];
    const int t = blockIdx.x, C = d.C, k = d.k;
    const float cx = add_dx ? tokmat[(int64_t)t * TOKMAT + 112] : 0.f;
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
            // + H_pre[I_j] d_input - cx x_j (the write-back's own term on the active state)
            a.x += h * g[0] - cx * x[0]; a.y += h * g[1] - cx * x[1];
            a.z += h * g[2] - cx * x[2]; a.w += h * g[3] - cx * x[3];
            b.x += h * g[4] - cx * x[4]; b.y += h * g[5] - cx * x[5];
            b.z += h * g[6] - cx * x[6]; b.w += h * g[7] - cx * x[7];
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
                              float* dhpre, uint16_t* dinput_copy, const float* tokmat,
                              cudaStream_t st) {
    if (d.k <= 4) {
        k_dinput_act<4><<<T, chunk_threads(d.C), 0, st>>>(d, slot, T, add_dx, d_input, xact, hpre, I, dxact,
                                                           dhpre, dinput_copy, tokmat); note_launch();
    } else {
        k_dinput_act<8><<<T, chunk_threads(d.C), 0, st>>>(d, slot, T, add_dx, d_input, xact, hpre, I, dxact,
                                                           dhpre, dinput_copy, tokmat); note_launch();
    }
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// full_dots: for the non-active streams i, dH_pre[t][q][i] = <x_i, d_input_q> (Eq. dense_read
// reversed; the dense-read gradient itself, dX[t][i] += sum_q H_pre[t][q][i] d_input_q, is added
// by the full-state dX kernel).  One CTA per token with one warp per two non-active streams
// (there are N - k of them on every token: the k active streams are distinct); the token's G
// d_input rows are staged in shared memory while each warp's first X reads are in flight, and
// each chunk read back from shared memory serves the warp's two X rows.

template <int NS>
__global__ void __launch_bounds__(512) k_full_dots(Dims d, int T, const uint16_t* __restrict__ X,
                                                   const uint16_t* __restrict__ dinput,
                                                   const int* __restrict__ I,
                                                   float* __restrict__ dhpre) {
    extern __shared__ __align__(16) uint16_t din[];   // [G][C]
    const int t = blockIdx.x, C = d.C, G = d.G;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    // this warp's streams: the (NS warp + h)-th streams not active on token t, h < NS (each
    // d_input chunk read from shared memory serves NS X rows)
    uint32_t act = 0u;
    for (int q = 0; q < d.k; ++q) act |= 1u << I[(int64_t)t * d.k + q];
    int is[NS];
#pragma unroll
    for (int h = 0; h < NS; ++h) is[h] = -1;
    for (int s = 0, cnt = 0; s < d.N; ++s)
        if (!(act & (1u << s))) {
#pragma unroll
            for (int h = 0; h < NS; ++h)
                if (cnt == NS * warp + h) is[h] = s;
            ++cnt;
        }
    if (!d.dense) {
        // sparse-read ablation: the non-active streams are not read, so their dH_pre is zero
        if (lane == 0)
            for (int h = 0; h < NS; ++h)
                if (is[h] >= 0)
                    for (int q = 0; q < G; ++q) dhpre[((int64_t)t * G + q) * d.N + is[h]] = 0.f;
        return;
    }
    int64_t row[NS];
#pragma unroll
    for (int h = 0; h < NS; ++h) row[h] = ((int64_t)t * d.N + (is[h] < 0 ? 0 : is[h])) * C;
    // the first 4 chunks per lane and stream, read before the staging barrier
    uint4 xr[NS][4];
#pragma unroll
    for (int h = 0; h < NS; ++h)
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int c8 = lane + 32 * u;
            xr[h][u] = make_uint4(0u, 0u, 0u, 0u);
            if (is[h] >= 0 && c8 < C / 8) xr[h][u] = __ldg(reinterpret_cast<const uint4*>(X + row[h] + c8 * 8));
        }
    for (int idx = threadIdx.x; idx < G * C / 8; idx += blockDim.x) {
        const int q = idx / (C / 8), c8 = idx - q * (C / 8);
        reinterpret_cast<uint4*>(din)[idx] =
            *reinterpret_cast<const uint4*>(dinput + ((int64_t)q * T + t) * C + c8 * 8);
    }
    __syncthreads();
    if (is[0] < 0) return;
    float acc[NS][4];
#pragma unroll
    for (int h = 0; h < NS; ++h)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[h][q] = 0.f;
    for (int c0 = lane; c0 < C / 8; c0 += 128) {
        if (c0 != lane) {
#pragma unroll
            for (int h = 0; h < NS; ++h)
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int c8 = c0 + 32 * u;
                    if (is[h] >= 0 && c8 < C / 8) xr[h][u] = __ldg(reinterpret_cast<const uint4*>(X + row[h] + c8 * 8));
                }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int c8 = c0 + 32 * u;
            if (c8 >= C / 8) continue;
            float xs[NS][8];
#pragma unroll
            for (int h = 0; h < NS; ++h) unpack8(xr[h][u], xs[h]);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                if (q >= G) continue;
                float g[8];
                unpack8(reinterpret_cast<const uint4*>(din + q * C)[c8], g);
#pragma unroll
                for (int h = 0; h < NS; ++h)
#pragma unroll
                    for (int e = 0; e < 8; ++e) acc[h][q] = fmaf(xs[h][e], g[e], acc[h][q]);
            }
        }
    }
#pragma unroll
    for (int h = 0; h < NS; ++h)
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float v = warp_sum(acc[h][q]);
            if (lane == 0 && q < G && is[h] >= 0) dhpre[((int64_t)t * G + q) * d.N + is[h]] = v;
        }
}

cudaError_t launch_full_dots(const Dims& d, int T, const uint16_t* X, const uint16_t* dinput,
                             const int* I, float* dhpre, cudaStream_t st) {
    constexpr int NS = 2;                       // non-active streams per warp
    const int nw = (d.N - d.k + NS - 1) / NS;   // warps per token
    if (nw <= 0) return cudaSuccess;
    const size_t sm = (size_t)d.G * d.C * 2;
    if (sm > 48 * 1024) {
        cudaError_t e = cudaFuncSetAttribute((const void*)k_full_dots<NS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)sm);
        if (e != cudaSuccess) return e;
    }
    k_full_dots<NS><<<T, 32 * nw, sm, st>>>(d, T, X, dinput, I, dhpre); note_launch();
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// model glue: stream expansion and the final stream sum, one CTA per token, 16-byte accesses

// X[t][i] = h[t] for every stream i (N copies; also the backward of the stream sum)
__global__ void __launch_bounds__(256) k_stream_bcast(int T, int N, int C, const uint16_t* __restrict__ h,
                                                      uint16_t* __restrict__ X) {
    const long long t = blockIdx.x;
    for (int c8 = threadIdx.x; c8 < C / 8; c8 += blockDim.x) {
        const uint4 v = *reinterpret_cast<const uint4*>(h + t * C + c8 * 8);
        for (int i = 0; i < N; ++i) *reinterpret_cast<uint4*>(X + (t * N + i) * C + c8 * 8) = v;
    }
}

// y[t] = sum_i X[t][i] in fp32, stored bf16 (also the backward of the expansion)
__global__ void __launch_bounds__(256) k_stream_sum(int T, int N, int C, const uint16_t* __restrict__ X,
                                                    uint16_t* __restrict__ y) {
    const long long t = blockIdx.x;
    for (int c8 = threadIdx.x; c8 < C / 8; c8 += blockDim.x) {
        float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        for (int i = 0; i < N; ++i) {
            float x[8];
            unpack8(*reinterpret_cast<const uint4*>(X + (t * N + i) * C + c8 * 8), x);
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[e] += x[e];
        }
        *reinterpret_cast<uint4*>(y + t * C + c8 * 8) = pack8(acc);
    }
}

cudaError_t launch_stream_bcast(int T, int N, int C, const uint16_t* h, uint16_t* X, cudaStream_t st) {
    k_stream_bcast<<<T, chunk_threads(C), 0, st>>>(T, N, C, h, X); note_launch();
    return cudaGetLastError();
}

cudaError_t launch_stream_sum(int T, int N, int C, const uint16_t* X, uint16_t* y, cudaStream_t st) {
    k_stream_sum<<<T, chunk_threads(C), 0, st>>>(T, N, C, X, y); note_launch();
    return cudaGetLastError();
}

}  // namespace xhc
