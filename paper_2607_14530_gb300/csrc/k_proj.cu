// Projection-shaped kernels of the connection op on the CUDA cores (fp32 FMA):
//   rowproj   Z = A W over a row of the state (Eq. fused_normalized_projection, Eq. param_post /
//             param_res), split over the reduction dimension, plus sum / sum of squares of A
//   gemm_dzw  dX_act += dZ W^T (backward of the active projection)
//   full_dx   dX = dX_base + dZ W^T + a + b x (backward of the full-state projection and norms)
//   wgrad     dW += A^T dZ, reduced over tokens in a fixed order
//   colsum    fixed-order column sums (per-token parameter-gradient contributions, W_r sums)
#include "xhc_internal.cuh"

namespace xhc {

// ---------------------------------------------------------------------------------------------
// rowproj: part[split][t][o] = sum_{e in split} A[t][e] * W[e][o];  pstats[split][t] = (sum a, sum a^2)

template <int NT>
__global__ void __launch_bounds__(256) k_rowproj(const uint16_t* __restrict__ A, int64_t lda, int K,
                                                 int T, WSegs W, int n, int kchunk,
                                                 float* __restrict__ part,
                                                 float* __restrict__ pstats) {
    constexpr int BM = 64, BK = 32, NP = 16 * NT;
    __shared__ __align__(16) float As[BK][BM + 4];
    __shared__ __align__(16) float Ws[BK][NP];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int row0 = blockIdx.x * BM;
    const int split = blockIdx.y;
    const int kbeg = split * kchunk;
    const int kend = min(K, kbeg + kchunk);
    float acc[4][NT];
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int j = 0; j < NT; ++j) acc[r][j] = 0.f;
    const int lr = tid >> 2, lseg = tid & 3;
    const int grow = row0 + lr;
    float s1 = 0.f, s2 = 0.f;
    for (int k0 = kbeg; k0 < kend; k0 += BK) {
        float av[8];
        const int kc = k0 + lseg * 8;
        if (grow < T && kc < kend) {
            const uint4 u = __ldg(reinterpret_cast<const uint4*>(A + (int64_t)grow * lda + kc));
            unpack8(u, av);
        } else {
#pragma unroll
            for (int q = 0; q < 8; ++q) av[q] = 0.f;
        }
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            s1 += av[q];
            s2 = fmaf(av[q], av[q], s2);
            As[lseg * 8 + q][lr] = av[q];
        }
        for (int idx = tid; idx < BK * NP; idx += 256) {
            const int kk = idx / NP, o = idx - kk * NP;
            const int kr = k0 + kk;
            float v = 0.f;
            if (o < n && kr < kend) {
                v = seg_elem<true>(W, kr, o);
            }
            Ws[kk][o] = v;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < BK; ++kk) {
            const float4 a = *reinterpret_cast<const float4*>(&As[kk][ty * 4]);
#pragma unroll
            for (int j = 0; j < NT; ++j) {
                const float w = Ws[kk][tx + 16 * j];
                acc[0][j] = fmaf(a.x, w, acc[0][j]);
                acc[1][j] = fmaf(a.y, w, acc[1][j]);
                acc[2][j] = fmaf(a.z, w, acc[2][j]);
                acc[3][j] = fmaf(a.w, w, acc[3][j]);
            }
        }
        __syncthreads();
    }
    s1 += __shfl_xor_sync(0xffffffffu, s1, 1);
    s1 += __shfl_xor_sync(0xffffffffu, s1, 2);
    s2 += __shfl_xor_sync(0xffffffffu, s2, 1);
    s2 += __shfl_xor_sync(0xffffffffu, s2, 2);
    if (lseg == 0 && grow < T) {
        pstats[((int64_t)split * T + grow) * 2 + 0] = s1;
        pstats[((int64_t)split * T + grow) * 2 + 1] = s2;
    }
#pragma unroll
    for (int r = 0; r < 4; ++r) {
        const int row = row0 + ty * 4 + r;
        if (row >= T) continue;
#pragma unroll
        for (int j = 0; j < NT; ++j) {
            const int o = tx + 16 * j;
            if (o < n) part[((int64_t)split * T + row) * n + o] = acc[r][j];
        }
    }
}

template <int NT>
static cudaError_t rowproj_nt(const uint16_t* A, int64_t lda, int K, int T, const WSegs& W, int n,
                              int splits, float* part, float* pstats, cudaStream_t st) {
    const int kchunk = ((K + splits - 1) / splits + 31) / 32 * 32;
    dim3 grid((T + 63) / 64, splits);
    k_rowproj<NT><<<grid, 256, 0, st>>>(A, lda, K, T, W, n, kchunk, part, pstats); note_launch();
    return cudaGetLastError();
}

cudaError_t launch_rowproj(const uint16_t* A, int64_t lda, int K, int T, const WSegs& W, int n,
                           int splits, float* part, float* pstats, cudaStream_t st) {
    const int nt = (n + 15) / 16;
    if (nt <= 1) return rowproj_nt<1>(A, lda, K, T, W, n, splits, part, pstats, st);
    if (nt <= 2) return rowproj_nt<2>(A, lda, K, T, W, n, splits, part, pstats, st);
    if (nt <= 4) return rowproj_nt<4>(A, lda, K, T, W, n, splits, part, pstats, st);
    if (nt <= 6) return rowproj_nt<6>(A, lda, K, T, W, n, splits, part, pstats, st);
    if (nt <= 8) return rowproj_nt<8>(A, lda, K, T, W, n, splits, part, pstats, st);
    if (nt <= 10) return rowproj_nt<10>(A, lda, K, T, W, n, splits, part, pstats, st);
    return cudaErrorInvalidValue;
}

// ---------------------------------------------------------------------------------------------
// colsum: out[o] (+)= sum_r in[r * ld + o], fixed order: each of 8 threads per column sums a
// strided subset of the row chunk, then a fixed tree; long columns go through a second stage.

__global__ void __launch_bounds__(256) k_colsum(const float* __restrict__ in, int rows, int ld, int n,
                                                int rchunk, float* __restrict__ out, int out_ld,
                                                int accumulate) {
    __shared__ float sh[8][33];
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    const int o = blockIdx.x * 32 + tx;
    const int r0 = blockIdx.y * rchunk, r1 = min(rows, r0 + rchunk);
    float s = 0.f;
    if (o < n)
        for (int r = r0 + ty; r < r1; r += 8) s += in[(int64_t)r * ld + o];
    sh[ty][tx] = s;
    __syncthreads();
    if (ty == 0 && o < n) {
        float t = 0.f;
#pragma unroll
        for (int q = 0; q < 8; ++q) t += sh[q][tx];
        float* dst = out + (int64_t)blockIdx.y * out_ld + o;
        *dst = accumulate ? *dst + t : t;
    }
}

// scratch holds up to 64 x 256 floats (n <= 256)
cudaError_t launch_colsum(const float* in, int rows, int ld, int n, float* out, int accumulate,
                          float* scratch, cudaStream_t st) {
    if (n <= 0 || rows <= 0) return cudaSuccess;
    if (rows <= 4096 || scratch == nullptr || n > 256) {
        dim3 grid((n + 31) / 32, 1);
        k_colsum<<<grid, 256, 0, st>>>(in, rows, ld, n, rows, out, n, accumulate); note_launch();
        return cudaGetLastError();
    }
    int rchunk = (rows + 63) / 64;
    const int nch = (rows + rchunk - 1) / rchunk;
    dim3 g1((n + 31) / 32, nch);
    k_colsum<<<g1, 256, 0, st>>>(in, rows, ld, n, rchunk, scratch, n, 0); note_launch();
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    dim3 g2((n + 31) / 32, 1);
    k_colsum<<<g2, 256, 0, st>>>(scratch, nch, n, n, nch, out, n, accumulate); note_launch();
    return cudaGetLastError();
}

// sub_rows: G[e][o] -= v[o] for every row e (the mean term of the router LayerNorm)

__global__ void k_sub_rows(float* __restrict__ G, int rows, int n, const float* __restrict__ v) {
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (int64_t)rows * n) return;
    G[idx] -= v[idx % n];
}

cudaError_t launch_sub_rows(float* G, int rows, int n, const float* v, cudaStream_t st) {
    const int64_t tot = (int64_t)rows * n;
    k_sub_rows<<<(unsigned)((tot + 255) / 256), 256, 0, st>>>(G, rows, n, v); note_launch();
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// gemm_dzw: out[t][e] += sum_o dz[t][o] * W[e][o]   (t < T, e < E, o < n)

__global__ void __launch_bounds__(256) k_gemm_dzw(const float* __restrict__ dz, int ldz, int n,
                                                  WSegs W, int E, int T,
                                                  float* __restrict__ out) {
    constexpr int BT = 64, BE = 64, BO = 32;
    __shared__ __align__(16) float Ds[BO][BT + 4];
    __shared__ __align__(16) float Wt[BO][BE + 4];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int t0 = blockIdx.y * BT, e0 = blockIdx.x * BE;
    float acc[4][4] = {};
    for (int o0 = 0; o0 < n; o0 += BO) {
        for (int idx = tid; idx < BT * BO; idx += 256) {
            const int tt = idx / BO, oo = idx - tt * BO;
            const int t = t0 + tt, o = o0 + oo;
            Ds[oo][tt] = (t < T && o < n) ? dz[(int64_t)t * ldz + o] : 0.f;
        }
        for (int idx = tid; idx < BE * BO; idx += 256) {
            const int ee = idx / BO, oo = idx - ee * BO;
            const int e = e0 + ee, o = o0 + oo;
            float v = 0.f;
            if (e < E && o < n) {
                v = seg_elem<true>(W, e, o);
            }
            Wt[oo][ee] = v;
        }
        __syncthreads();
#pragma unroll 8
        for (int oo = 0; oo < BO; ++oo) {
            const float4 a = *reinterpret_cast<const float4*>(&Ds[oo][ty * 4]);
            const float4 w = *reinterpret_cast<const float4*>(&Wt[oo][tx * 4]);
            const float av[4] = {a.x, a.y, a.z, a.w}, wv[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
            for (int r = 0; r < 4; ++r)
#pragma unroll
                for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(av[r], wv[c], acc[r][c]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int r = 0; r < 4; ++r) {
        const int t = t0 + ty * 4 + r;
        if (t >= T) continue;
        const int e = e0 + tx * 4;
        if (e + 3 < E) {
            float4* dst = reinterpret_cast<float4*>(out + (int64_t)t * E + e);
            float4 v = *dst;
            v.x += acc[r][0]; v.y += acc[r][1]; v.z += acc[r][2]; v.w += acc[r][3];
            *dst = v;
        } else {
            for (int c = 0; c < 4; ++c)
                if (e + c < E) out[(int64_t)t * E + e + c] += acc[r][c];
        }
    }
}

cudaError_t launch_gemm_dzw(const Dims& d, int T, const float* dz, int ldz, int n,
                            const WSegs& W, int E, float* dxact, cudaStream_t st) {
    (void)d;
    dim3 grid((E + 63) / 64, (T + 63) / 64);
    k_gemm_dzw<<<grid, 256, 0, st>>>(dz, ldz, n, W, E, T, dxact); note_launch();
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// full_dx: dX[t][e] = base(t, e) + sum_o dz[t][o] W[e][o] + a_t + b_t * x[t][e], e = i*C + c,
// base = dX_act[t][j][c] if stream i is active slot j, else dX[t][e] plus the dense-read
// gradient sum_q H_pre[t][q][i] d_input_q[t][c] (Eq. dense_read reversed; din holds the G
// d_input copies [G][T][C])

__global__ void __launch_bounds__(256) k_full_dx(Dims d, int T, const float* __restrict__ dz,
                                                 WSegs W, const uint16_t* __restrict__ X,
                                                 const uint16_t* __restrict__ din,
                                                 const float* __restrict__ hpre,
                                                 const int* __restrict__ I,
                                                 const float* __restrict__ dxact,
                                                 const float* __restrict__ scal,
                                                 uint16_t* __restrict__ dX) {
    constexpr int BT = 64, BE = 64, BO = 32;
    __shared__ __align__(16) float Ds[BO][BT + 4];
    __shared__ __align__(16) float Wt[BO][BE + 4];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int t0 = blockIdx.y * BT, e0 = blockIdx.x * BE;
    const int E = d.N * d.C, n = d.nfull;
    float acc[4][4] = {};
    for (int o0 = 0; o0 < n; o0 += BO) {
        for (int idx = tid; idx < BT * BO; idx += 256) {
            const int tt = idx / BO, oo = idx - tt * BO;
            const int t = t0 + tt, o = o0 + oo;
            Ds[oo][tt] = (t < T && o < n) ? dz[(int64_t)t * n + o] : 0.f;
        }
        for (int idx = tid; idx < BE * BO; idx += 256) {
            const int ee = idx / BO, oo = idx - ee * BO;
            const int e = e0 + ee, o = o0 + oo;
            float v = 0.f;
            if (e < E && o < n) {
                v = seg_elem<true>(W, e, o);
            }
            Wt[oo][ee] = v;
        }
        __syncthreads();
#pragma unroll 8
        for (int oo = 0; oo < BO; ++oo) {
            const float4 a = *reinterpret_cast<const float4*>(&Ds[oo][ty * 4]);
            const float4 w = *reinterpret_cast<const float4*>(&Wt[oo][tx * 4]);
            const float av[4] = {a.x, a.y, a.z, a.w}, wv[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
            for (int r = 0; r < 4; ++r)
#pragma unroll
                for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(av[r], wv[c], acc[r][c]);
        }
        __syncthreads();
    }
    const int e = e0 + tx * 4;
    if (e >= E) return;
    const int i = e / d.C, c = e - i * d.C;  // 4 consecutive channels of one stream (C % 8 == 0)
#pragma unroll
    for (int r = 0; r < 4; ++r) {
        const int t = t0 + ty * 4 + r;
        if (t >= T) continue;
        int j = -1;
        for (int q = 0; q < d.k; ++q)
            if (I[(int64_t)t * d.k + q] == i) j = q;
        float v[4];
        if (j >= 0) {
            const float4 b = *reinterpret_cast<const float4*>(dxact + ((int64_t)t * d.k + j) * d.C + c);
            v[0] = b.x; v[1] = b.y; v[2] = b.z; v[3] = b.w;
        } else {
            const uint2 u = *reinterpret_cast<const uint2*>(dX + (int64_t)t * E + e);
            v[0] = __uint_as_float(u.x << 16); v[1] = __uint_as_float(u.x & 0xffff0000u);
            v[2] = __uint_as_float(u.y << 16); v[3] = __uint_as_float(u.y & 0xffff0000u);
            for (int q = 0; q < (d.dense ? d.G : 0); ++q) {   // sparse-read ablation: none
                const float h = hpre[((int64_t)t * d.G + q) * d.N + i];
                const uint2 g = *reinterpret_cast<const uint2*>(din + ((int64_t)q * T + t) * d.C + c);
                v[0] = fmaf(h, __uint_as_float(g.x << 16), v[0]);
                v[1] = fmaf(h, __uint_as_float(g.x & 0xffff0000u), v[1]);
                v[2] = fmaf(h, __uint_as_float(g.y << 16), v[2]);
                v[3] = fmaf(h, __uint_as_float(g.y & 0xffff0000u), v[3]);
            }
        }
        const float a = scal[(int64_t)t * NTG + 0], b = scal[(int64_t)t * NTG + 1];
        const uint2 xu = *reinterpret_cast<const uint2*>(X + (int64_t)t * E + e);
        const float xv[4] = {__uint_as_float(xu.x << 16), __uint_as_float(xu.x & 0xffff0000u),
                             __uint_as_float(xu.y << 16), __uint_as_float(xu.y & 0xffff0000u)};
        float res[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) res[q] = v[q] + acc[r][q] + a + b * xv[q];
        uint2 o;
        o.x = pack2(res[0], res[1]);
        o.y = pack2(res[2], res[3]);
        *reinterpret_cast<uint2*>(dX + (int64_t)t * E + e) = o;
    }
}

cudaError_t launch_full_dx(const Dims& d, int T, const float* dz, const WSegs& W,
                           const uint16_t* X, const uint16_t* dinput, const float* hpre,
                           const int* I, const float* dxact, const float* scal, uint16_t* dX,
                           cudaStream_t st) {
    const int E = d.N * d.C;
    dim3 grid((E + 63) / 64, (T + 63) / 64);
    k_full_dx<<<grid, 256, 0, st>>>(d, T, dz, W, X, dinput, hpre, I, dxact, scal, dX); note_launch();
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// wgrad: wpart[split][e][o] = sum_{t in split} A[t][e] dz[t][o]; then G[e][o] += sum_split

template <int NT>
__global__ void __launch_bounds__(256) k_wgrad(const uint16_t* __restrict__ A, int64_t lda, int E,
                                               int T, const float* __restrict__ dz, int ldz, int n,
                                               int tchunk, float* __restrict__ wpart) {
    constexpr int BE = 64, BT = 32, NP = 16 * NT;
    __shared__ __align__(16) float As[BT][BE + 4];
    __shared__ __align__(16) float Ds[BT][NP];
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const int e0 = blockIdx.x * BE;
    const int split = blockIdx.y;
    const int tbeg = split * tchunk, tend = min(T, tbeg + tchunk);
    float acc[4][NT];
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int j = 0; j < NT; ++j) acc[r][j] = 0.f;
    const int lt = tid >> 3, lseg = tid & 7;  // 32 token rows x 8 segments of 8 columns
    for (int tk = tbeg; tk < tend; tk += BT) {
        {
            const int t = tk + lt, e = e0 + lseg * 8;
            float av[8];
            if (t < tend && e < E) {
                const uint4 u = __ldg(reinterpret_cast<const uint4*>(A + (int64_t)t * lda + e));
                unpack8(u, av);
            } else {
#pragma unroll
                for (int q = 0; q < 8; ++q) av[q] = 0.f;
            }
#pragma unroll
            for (int q = 0; q < 8; ++q) As[lt][lseg * 8 + q] = av[q];
        }
        for (int idx = tid; idx < BT * NP; idx += 256) {
            const int tt = idx / NP, o = idx - tt * NP;
            const int t = tk + tt;
            Ds[tt][o] = (t < tend && o < n) ? dz[(int64_t)t * ldz + o] : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int tt = 0; tt < BT; ++tt) {
            const float4 a = *reinterpret_cast<const float4*>(&As[tt][ty * 4]);
#pragma unroll
            for (int j = 0; j < NT; ++j) {
                const float w = Ds[tt][tx + 16 * j];
                acc[0][j] = fmaf(a.x, w, acc[0][j]);
                acc[1][j] = fmaf(a.y, w, acc[1][j]);
                acc[2][j] = fmaf(a.z, w, acc[2][j]);
                acc[3][j] = fmaf(a.w, w, acc[3][j]);
            }
        }
        __syncthreads();
    }
#pragma unroll
    for (int r = 0; r < 4; ++r) {
        const int e = e0 + ty * 4 + r;
        if (e >= E) continue;
#pragma unroll
        for (int j = 0; j < NT; ++j) {
            const int o = tx + 16 * j;
            if (o < n) wpart[((int64_t)split * E + e) * n + o] = acc[r][j];
        }
    }
}

__global__ void k_wgrad_reduce(const float* __restrict__ wpart, int splits, int E, int n,
                               WSegsOut G) {
    const int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= (int64_t)E * n) return;
    const int e = (int)(idx / n), o = (int)(idx - (int64_t)e * n);
    float s = 0.f;
    for (int q = 0; q < splits; ++q) s += wpart[(int64_t)q * E * n + idx];
    // the segment of column o, selected with static indices (no local copy of the parameter)
    float* p = G.ptr[0];
    int width = G.width[0], off = G.off[0];
#pragma unroll
    for (int q = 1; q < MAXSEG; ++q)
        if (q < G.n && o >= G.off[q]) {
            p = G.ptr[q];
            width = G.width[q];
            off = G.off[q];
        }
    p[(int64_t)e * width + (o - off)] += s;
}

cudaError_t launch_wgrad_reduce(const float* wpart, int splits, int E, int n, const WSegsOut& G,
                                cudaStream_t st) {
    const int64_t tot = (int64_t)E * n;
    k_wgrad_reduce<<<(unsigned)((tot + 255) / 256), 256, 0, st>>>(wpart, splits, E, n, G); note_launch();
    return cudaGetLastError();
}

template <int NT>
static cudaError_t wgrad_nt(const uint16_t* A, int64_t lda, int E, int T, const float* dz, int ldz,
                            int n, int tsplits, float* wpart, const WSegsOut& G, cudaStream_t st) {
    const int tchunk = ((T + tsplits - 1) / tsplits + 31) / 32 * 32;
    const int splits = (T + tchunk - 1) / tchunk;
    dim3 grid((E + 63) / 64, splits);
    k_wgrad<NT><<<grid, 256, 0, st>>>(A, lda, E, T, dz, ldz, n, tchunk, wpart); note_launch();
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int64_t tot = (int64_t)E * n;
    k_wgrad_reduce<<<(unsigned)((tot + 255) / 256), 256, 0, st>>>(wpart, splits, E, n, G); note_launch();
    return cudaGetLastError();
}

cudaError_t launch_wgrad(const uint16_t* A, int64_t lda, int E, int T, const float* dz, int ldz,
                         int n, int tsplits, float* wpart, const WSegsOut& G, cudaStream_t st) {
    const int nt = (n + 15) / 16;
    if (nt <= 1) return wgrad_nt<1>(A, lda, E, T, dz, ldz, n, tsplits, wpart, G, st);
    if (nt <= 2) return wgrad_nt<2>(A, lda, E, T, dz, ldz, n, tsplits, wpart, G, st);
    if (nt <= 4) return wgrad_nt<4>(A, lda, E, T, dz, ldz, n, tsplits, wpart, G, st);
    if (nt <= 6) return wgrad_nt<6>(A, lda, E, T, dz, ldz, n, tsplits, wpart, G, st);
    if (nt <= 8) return wgrad_nt<8>(A, lda, E, T, dz, ldz, n, tsplits, wpart, G, st);
    if (nt <= 10) return wgrad_nt<10>(A, lda, E, T, dz, ldz, n, tsplits, wpart, G, st);
    return cudaErrorInvalidValue;
}

}  // namespace xhc
