// Per-token coefficient kernels (one thread per token, fp32):
//   coef_full  norm statistics -> router scores, TopK routing, pre-maps
//              (Eq. fused_normalized_projection, Eq. router, Eq. router_topk, Eq. param_pre)
//   coef_act   active RMS -> post-map, Sinkhorn residual map + row clamp
//              (Eq. param_post, Eq. param_res, App. A)
//   bwd_coef   reverse of coef_act, of the Gram-Schmidt coefficients (Eq. gs) and of the
//              write-back contraction (Eq. sparse_write_delta)
//   full_coef  reverse of coef_full (norm corrections, pre-map sigmoid, router through the
//              selected routed scores only)
#include <algorithm>

#include "xhc_internal.cuh"

namespace xhc {

// ---------------------------------------------------------------------------------------------
// Sinkhorn of Eq. mhc_sinkhorn on a k x k block (k <= KM), with the App. A row clamp.
// exp(M - rowmax): the first row normalisation removes any per-row scale, so this equals exp(M).

template <int KM>
__device__ __forceinline__ void sk_init(const float (&M)[KM][KM], int k, float (&A)[KM][KM]) {
#pragma unroll
    for (int a = 0; a < KM; ++a) {
        float mx = -INFINITY;
#pragma unroll
        for (int b = 0; b < KM; ++b)
            if (a < k && b < k) mx = fmaxf(mx, M[a][b]);
#pragma unroll
        for (int b = 0; b < KM; ++b) A[a][b] = (a < k && b < k) ? expf(M[a][b] - mx) : 0.f;
    }
}

// one half-step: h even = row normalisation, h odd = column normalisation (one reciprocal per
// row or column, then products)
template <int KM>
__device__ __forceinline__ void sk_half(float (&A)[KM][KM], int k, int h) {
    if ((h & 1) == 0) {
#pragma unroll
        for (int a = 0; a < KM; ++a) {
            if (a >= k) continue;
            float s = 0.f;
#pragma unroll
            for (int b = 0; b < KM; ++b) s += A[a][b];
            const float r = 1.0f / s;
#pragma unroll
            for (int b = 0; b < KM; ++b) A[a][b] = A[a][b] * r;
        }
    } else {
#pragma unroll
        for (int b = 0; b < KM; ++b) {
            if (b >= k) continue;
            float s = 0.f;
#pragma unroll
            for (int a = 0; a < KM; ++a) s += A[a][b];
            const float r = 1.0f / s;
#pragma unroll
            for (int a = 0; a < KM; ++a) A[a][b] = A[a][b] * r;
        }
    }
}

template <int KM>
__device__ __forceinline__ void sinkhorn_fwd(const float (&M)[KM][KM], int k, int iters,
                                             float (&H)[KM][KM]) {
    sk_init<KM>(M, k, H);
    for (int h = 0; h < 2 * iters; ++h) sk_half<KM>(H, k, h);
#pragma unroll
    for (int a = 0; a < KM; ++a) {
        float s = 0.f;
#pragma unroll
        for (int b = 0; b < KM; ++b) s += H[a][b];
        if (s > 1.f) {
#pragma unroll
            for (int b = 0; b < KM; ++b) H[a][b] = H[a][b] / s;
        }
    }
}

// Reverse mode of sinkhorn_fwd: given dH returns dM (and H).  The forward iterates are rebuilt
// from checkpoints: the matrix entering every L-th half-step is kept in shared memory (ck, laid
// out [segment][entry][thread] with stride nth), and the half-steps of a segment are replayed
// from its checkpoint, so the reverse sweep costs O(iters * L) half-steps instead of O(iters^2).
// The replayed values are bit-identical to the forward ones.
template <int KM>
__device__ void sinkhorn_bwd(const float (&M)[KM][KM], int k, int iters, int L, float* ck, int nth,
                             const float (&dH)[KM][KM], float (&H)[KM][KM], float (&dM)[KM][KM]) {
    const int nh = 2 * iters;
    float A[KM][KM], dA[KM][KM];
    sk_init<KM>(M, k, A);
    for (int h = 0; h < nh; ++h) {
        if (h % L == 0) {
            float* c = ck + (size_t)(h / L) * KM * KM * nth;
#pragma unroll
            for (int a = 0; a < KM; ++a)
#pragma unroll
                for (int b = 0; b < KM; ++b) c[(a * KM + b) * nth] = A[a][b];
        }
        sk_half<KM>(A, k, h);
    }
    // clamp
#pragma unroll
    for (int a = 0; a < KM; ++a) {
        float s = 0.f;
#pragma unroll
        for (int b = 0; b < KM; ++b) s += A[a][b];
        if (s > 1.f) {
            float dot = 0.f;
#pragma unroll
            for (int b = 0; b < KM; ++b) {
                H[a][b] = A[a][b] / s;
                dot += dH[a][b] * H[a][b];
            }
#pragma unroll
            for (int b = 0; b < KM; ++b) dA[a][b] = (dH[a][b] - dot) / s;
        } else {
#pragma unroll
            for (int b = 0; b < KM; ++b) {
                H[a][b] = A[a][b];
                dA[a][b] = dH[a][b];
            }
        }
    }
    // half-steps in reverse; the input of step h is replayed from its segment's checkpoint
    for (int h = nh - 1; h >= 0; --h) {
        const int h0 = (h / L) * L;
        float In[KM][KM];
        const float* c = ck + (size_t)(h / L) * KM * KM * nth;
#pragma unroll
        for (int a = 0; a < KM; ++a)
#pragma unroll
            for (int b = 0; b < KM; ++b) In[a][b] = c[(a * KM + b) * nth];
        for (int q = h0; q < h; ++q) sk_half<KM>(In, k, q);
        // output of step h
        float Out[KM][KM];
#pragma unroll
        for (int a = 0; a < KM; ++a)
#pragma unroll
            for (int b = 0; b < KM; ++b) Out[a][b] = In[a][b];
        sk_half<KM>(Out, k, h);
        if ((h & 1) == 0) {
#pragma unroll
            for (int a = 0; a < KM; ++a) {
                if (a >= k) continue;
                float s = 0.f, dot = 0.f;
#pragma unroll
                for (int b = 0; b < KM; ++b) {
                    s += In[a][b];
                    dot += dA[a][b] * Out[a][b];
                }
#pragma unroll
                for (int b = 0; b < KM; ++b) dA[a][b] = (dA[a][b] - dot) * (1.0f / s);
            }
        } else {
#pragma unroll
            for (int b = 0; b < KM; ++b) {
                if (b >= k) continue;
                float s = 0.f, dot = 0.f;
#pragma unroll
                for (int a = 0; a < KM; ++a) {
                    s += In[a][b];
                    dot += dA[a][b] * Out[a][b];
                }
#pragma unroll
                for (int a = 0; a < KM; ++a) dA[a][b] = (dA[a][b] - dot) * (1.0f / s);
            }
        }
    }
    float A0[KM][KM];
    sk_init<KM>(M, k, A0);
#pragma unroll
    for (int a = 0; a < KM; ++a)
#pragma unroll
        for (int b = 0; b < KM; ++b) dM[a][b] = (a < k && b < k) ? dA[a][b] * A0[a][b] : 0.f;
}

// ---------------------------------------------------------------------------------------------
// slot_sum: x[e] = sum_q x[q * n + e] over the split-K partial slots, in slot order (the order
// in which the coefficient kernels sum them, so a summed buffer read as one slot gives the same
// bits), into slot 0.  Used when there are many slots (few tokens): one thread per element
// instead of one thread per token walking every slot.

__global__ void k_slot_sum(float* __restrict__ x, int nslots, long long n) {
    for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < n;
         e += (long long)gridDim.x * blockDim.x) {
        float s = 0.f;
        for (int q = 0; q < nslots; ++q) s += x[(long long)q * n + e];
        x[e] = s;
    }
}

cudaError_t launch_slot_sum(float* x, int nslots, long long n, cudaStream_t st) {
    const int blocks = (int)std::min<long long>((n + 255) / 256, 4096);
    k_slot_sum<<<blocks, 256, 0, st>>>(x, nslots, n); note_launch();
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// coef_full

__global__ void k_coef_full(Dims d, int T, const float* __restrict__ part,
                            const float* __restrict__ pstats, int splits,
                            const float* __restrict__ wsum, const float* __restrict__ alpha_pre,
                            const float* __restrict__ b_pre, float* __restrict__ zfull,
                            float* __restrict__ stats, float* __restrict__ hpre,
                            int* __restrict__ I, float* __restrict__ p) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= T) return;
    const int n = d.nfull;
    const float inv_nc = 1.0f / (float)(d.N * d.C);
    float s1 = 0.f, s2 = 0.f;
    for (int q = 0; q < splits; ++q) {
        s1 += pstats[((int64_t)q * T + t) * 2 + 0];
        s2 += pstats[((int64_t)q * T + t) * 2 + 1];
    }
    const float mu = s1 * inv_nc, nu = s2 * inv_nc;
    stats[(int64_t)t * 2 + 0] = mu;
    stats[(int64_t)t * 2 + 1] = nu;
    const float rstd = 1.0f / sqrtf(nu + d.eps);
    float zr[MAXN];
    for (int o = 0; o < n; ++o) {
        float z = 0.f;
        for (int q = 0; q < splits; ++q) z += part[((int64_t)q * T + t) * n + o];
        zfull[(int64_t)t * n + o] = z;
        if (d.hr && o < d.N) {
            zr[o] = z;
        } else {
            const int qo = o - (d.hr ? d.N : 0);
            const int slot = qo / d.N, i = qo - slot * d.N;
            hpre[((int64_t)t * d.G + slot) * d.N + i] =
                sigm(alpha_pre[slot] * (z * rstd) + b_pre[slot * d.N + i]);
        }
    }
    // Eq. router_topk: fixed streams 0..m-1 (p = 1), then TopK over i >= m by router logit
    // (sigmoid and softmax are both monotone in the logit), descending, ties to the lower
    // stream index.
    for (int j = 0; j < d.m; ++j) {
        I[(int64_t)t * d.k + j] = j;
        p[(int64_t)t * d.k + j] = 1.0f;
    }
    if (d.hr) {
        const float lstd = 1.0f / sqrtf(nu - mu * mu + d.eps);
        float zmax = -INFINITY;
        for (int i = 0; i < d.N; ++i) {
            zr[i] = (zr[i] - mu * wsum[i]) * lstd;
            zmax = fmaxf(zmax, zr[i]);
        }
        // softmax router: s_i = exp(z_i) / sum over all N logits (the fixed streams' included)
        float den = 0.f;
        if (d.softmax)
            for (int i = 0; i < d.N; ++i) den += expf(zr[i] - zmax);
        uint32_t taken = 0u;
        for (int j = d.m; j < d.k; ++j) {
            int best = -1;
            float bv = 0.f;
            for (int i = d.m; i < d.N; ++i) {
                if (taken & (1u << i)) continue;
                if (best < 0 || zr[i] > bv) {
                    best = i;
                    bv = zr[i];
                }
            }
            taken |= 1u << best;
            I[(int64_t)t * d.k + j] = best;
            p[(int64_t)t * d.k + j] = d.softmax ? expf(bv - zmax) / den : sigm(bv);
        }
    }
}

cudaError_t launch_coef_full(const Dims& d, int T, const float* part, const float* pstats,
                             int splits, const float* wsum, const float* alpha_pre,
                             const float* b_pre, float* zfull, float* stats, float* hpre,
                             int* I, float* p, cudaStream_t st) {
    k_coef_full<<<(T + 127) / 128, 128, 0, st>>>(d, T, part, pstats, splits, wsum, alpha_pre,
                                                  b_pre, zfull, stats, hpre, I, p); note_launch();
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// coef_act

template <int KM>
__global__ void k_coef_act(Dims d, int slot, int T, const float* __restrict__ part,
                           const float* __restrict__ pstats, int ssplits, int splits,
                           const float* __restrict__ alpha_post, const float* __restrict__ b_post,
                           const float* __restrict__ alpha_res, const float* __restrict__ b_res,
                           float* __restrict__ zact, float* __restrict__ rs,
                           float* __restrict__ hpost, float* __restrict__ hres) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= T) return;
    const int k = d.k, K = d.K[slot], n = d.nact[slot];
    const bool last = (slot == d.G - 1);
    float s2 = 0.f;
    for (int q = 0; q < ssplits; ++q) s2 += pstats[((int64_t)q * T + t) * 2 + 1];
    const float r = 1.0f / sqrtf(s2 / (float)(k * d.C) + d.eps);
    rs[t] = r;
    const float ap = alpha_post[slot];
    float M[KM][KM];
#pragma unroll
    for (int a = 0; a < KM; ++a)
#pragma unroll
        for (int b = 0; b < KM; ++b) M[a][b] = 0.f;
    const float ar = last ? alpha_res[0] : 0.f;
    for (int o = 0; o < n; ++o) {
        float z = 0.f;
        for (int q = 0; q < splits; ++q) z += part[((int64_t)q * T + t) * n + o];
        zact[(int64_t)t * n + o] = z;
        if (o < k * K) {
            hpost[(int64_t)t * k * K + o] = 2.0f * sigm(ap * (z * r) + b_post[o]);
        } else {
            const int q = o - k * K, a = q / k, b = q - a * k;
#pragma unroll
            for (int aa = 0; aa < KM; ++aa)
#pragma unroll
                for (int bb = 0; bb < KM; ++bb)
                    if (aa == a && bb == b) M[aa][bb] = ar * (z * r) + b_res[q];
        }
    }
    if (last) {
        float H[KM][KM];
        sinkhorn_fwd<KM>(M, k, d.iters, H);
#pragma unroll
        for (int a = 0; a < KM; ++a)
#pragma unroll
            for (int b = 0; b < KM; ++b)
                if (a < k && b < k) hres[(int64_t)t * k * k + a * k + b] = H[a][b];
    }
}

cudaError_t launch_coef_act(const Dims& d, int slot, int T, const float* part,
                            const float* pstats, int ssplits, int splits, const float* alpha_post,
                            const float* b_post, const float* alpha_res, const float* b_res,
                            float* zact, float* rs, float* hpost, float* hres, cudaStream_t st) {
    if (d.k <= 4) {
        k_coef_act<4><<<(T + 127) / 128, 128, 0, st>>>(d, slot, T, part, pstats, ssplits, splits, alpha_post,
                                                        b_post, alpha_res, b_res, zact, rs, hpost, hres); note_launch();
    } else {
        k_coef_act<8><<<(T + 127) / 128, 128, 0, st>>>(d, slot, T, part, pstats, ssplits, splits, alpha_post,
                                                        b_post, alpha_res, b_res, zact, rs, hpost, hres); note_launch();
    }
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// bwd_coef: per token, from the reductions
//   P[j][a] = <dXn_j, u_a>   Q[j][i] = <dXn_j, x_act_i> (last slot)   Gm[a][b] = <u_a, u_b> (GS)
// produce E[j][a] = p_j sum_q Hpost[j][q] B[q][a], D = dG + dG^T, H_res, the scaled projection
// gradient dZs = dz * r, the RMS coefficient cx, dp (+=) and the alpha/b contributions.

template <int KM>
__global__ void k_bwd_coef(Dims d, int slot, int T, const float* __restrict__ red, int nslice,
                           const float* __restrict__ zact, const float* __restrict__ rs,
                           const float* __restrict__ p, const float* __restrict__ hpost,
                           const double* __restrict__ gram, int skL,
                           const float* __restrict__ alpha_post, const float* __restrict__ b_post,
                           const float* __restrict__ alpha_res, const float* __restrict__ b_res,
                           float* __restrict__ tokmat, float* __restrict__ dzs,
                           float* __restrict__ dp, float* __restrict__ tokgrad) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= T) return;
    const int k = d.k, K = d.K[slot], n = d.nact[slot];
    const bool last = (slot == d.G - 1);
    const bool gs = (K > 1) && d.gs;
    // reduction slots per token (see wb_bred): P at j*4 + a, Q at KM*4 + j*KM + i; the Gram
    // matrix of the components comes from the forward (lower triangle packed, fp64)
    const int offQ = KM * 4;
    float Pm[KM][MAXCOMP], Q[KM][KM];
    double Gm[MAXCOMP][MAXCOMP];
#pragma unroll
    for (int j = 0; j < KM; ++j) {
#pragma unroll
        for (int a = 0; a < MAXCOMP; ++a) Pm[j][a] = 0.f;
#pragma unroll
        for (int i = 0; i < KM; ++i) Q[j][i] = 0.f;
    }
    // loops to MAXCOMP / KM with guards on K / k: compile-time indices, registers only
#pragma unroll
    for (int a = 0; a < MAXCOMP; ++a)
#pragma unroll
        for (int b = 0; b < MAXCOMP; ++b) Gm[a][b] = 0.0;
    for (int s = 0; s < nslice; ++s) {
        const float* rp = red + ((int64_t)t * nslice + s) * NRED;
#pragma unroll
        for (int j = 0; j < KM; ++j)
#pragma unroll
            for (int a = 0; a < MAXCOMP; ++a)
                if (j < k && a < K) Pm[j][a] += rp[j * 4 + a];
        if (last) {
#pragma unroll
            for (int j = 0; j < KM; ++j)
#pragma unroll
                for (int i = 0; i < KM; ++i)
                    if (j < k && i < k) Q[j][i] += rp[offQ + j * KM + i];
        }
    }
    if (gs) {
#pragma unroll
        for (int a = 0; a < MAXCOMP; ++a)
#pragma unroll
            for (int b = 0; b <= a; ++b)
                if (a < K) Gm[a][b] = gram[(int64_t)t * NGRAM + a * (a + 1) / 2 + b];
    }
#pragma unroll
    for (int a = 0; a < MAXCOMP; ++a)
#pragma unroll
        for (int b = a + 1; b < MAXCOMP; ++b)
            if (b < K) Gm[a][b] = Gm[b][a];
    double B[MAXCOMP][MAXCOMP], cc[MAXCOMP][MAXCOMP], vv[MAXCOMP];
    if (gs) {
        gs_coef(Gm, K, (double)d.eps_gs, B, cc, vv);
    } else {
#pragma unroll
        for (int a = 0; a < MAXCOMP; ++a)
#pragma unroll
            for (int b = 0; b < MAXCOMP; ++b) B[a][b] = (a == b) ? 1.0 : 0.0;
    }
    float* tm = tokmat + (int64_t)t * TOKMAT;
    float* tg = tokgrad + (int64_t)t * NTG;
    const float r = rs[t];
    const float* za = zact + (int64_t)t * n;
    const float ap = alpha_post[slot];
    // the scaled map-logit gradients go straight to dzs (dz * r); sdz = sum_o dz_o zact_o feeds
    // the RMS coefficient cx
    float* dzr = dzs + (int64_t)t * n;
    float sdz = 0.f;
    double dB[MAXCOMP][MAXCOMP];
#pragma unroll
    for (int a = 0; a < MAXCOMP; ++a)
#pragma unroll
        for (int b = 0; b < MAXCOMP; ++b) dB[a][b] = 0.0;
    float dap = 0.f;
#pragma unroll
    for (int j = 0; j < KM; ++j) {
        if (j >= k) continue;
        const float pj = p[(int64_t)t * k + j];
        float dpj = 0.f;
#pragma unroll
        for (int a = 0; a < 4; ++a) {
            float e = 0.f;
            if (a < K) {
#pragma unroll
                for (int q = 0; q < MAXCOMP; ++q)
                    if (q < K) e += hpost[((int64_t)t * k + j) * K + q] * (float)B[q][a];
            }
            tm[j * 4 + a] = pj * e;
        }
#pragma unroll
        for (int q = 0; q < MAXCOMP; ++q) {
            if (q >= K) continue;
            float pb = 0.f;
#pragma unroll
            for (int a = 0; a < MAXCOMP; ++a)
                if (a < K) pb += Pm[j][a] * (float)B[q][a];
            const float h = hpost[((int64_t)t * k + j) * K + q];
            const float dh = pj * pb;
            dpj += h * pb;
#pragma unroll
            for (int a = 0; a < MAXCOMP; ++a)
                if (a < K) dB[q][a] += (double)(pj * h) * (double)Pm[j][a];
            // H = 2 sigma(y): dy = dH * H * (1 - H / 2)
            const float dy = dh * h * (1.0f - 0.5f * h);
            const int o = j * K + q;
            const float dzo = ap * dy;
            dap += dy * (za[o] * r);
            tg[o] = dy;
            sdz += dzo * za[o];
            dzr[o] = dzo * r;
        }
        dp[(int64_t)t * k + j] += dpj;
    }
    tg[k * K] = dap;
    // D = dG + dG^T (symmetric Gram entries)
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) tm[32 + a * 4 + b] = 0.f;
    if (gs) {
        double dG[MAXCOMP][MAXCOMP];
        gs_coef_bwd(Gm, K, B, cc, vv, dB, dG);
#pragma unroll
        for (int a = 0; a < MAXCOMP; ++a)
#pragma unroll
            for (int b = 0; b < MAXCOMP; ++b)
                if (a < K && b < K) tm[32 + a * 4 + b] = (float)(dG[a][b] + dG[b][a]);
    }
    if (last) {
        float M[KM][KM], dH[KM][KM], H[KM][KM], dM[KM][KM];
        const float ar = alpha_res[0];
#pragma unroll
        for (int a = 0; a < KM; ++a)
#pragma unroll
            for (int b = 0; b < KM; ++b) {
                const bool v = (a < k && b < k);
                M[a][b] = v ? ar * (za[k * K + a * k + b] * r) + b_res[a * k + b] : 0.f;
                dH[a][b] = v ? Q[a][b] : 0.f;
            }
        extern __shared__ float sk_ck[];
        sinkhorn_bwd<KM>(M, k, d.iters, skL, sk_ck + threadIdx.x, blockDim.x, dH, H, dM);
        float dar = 0.f;
#pragma unroll
        for (int a = 0; a < KM; ++a)
#pragma unroll
            for (int b = 0; b < KM; ++b) {
                if (a >= k || b >= k) continue;
                const int o = k * K + a * k + b;
                const float dzo = ar * dM[a][b];
                dar += dM[a][b] * (za[o] * r);
                tg[k * K + 1 + a * k + b] = dM[a][b];
                tm[48 + a * 8 + b] = H[a][b];
                sdz += dzo * za[o];
                dzr[o] = dzo * r;
            }
        tg[k * K + 1 + k * k] = dar;
    }
    // active RMS: z_o = r * zraw_o, r = (sum x^2 / kC + eps)^(-1/2)
    tm[112] = r * r * r / (float)(k * d.C) * sdz;
}

cudaError_t launch_bwd_coef(const Dims& d, int slot, int T, const float* red, int nslice,
                            const float* zact, const float* rs, const float* p,
                            const float* hpost, const double* gram, const float* alpha_post,
                            const float* b_post, const float* alpha_res, const float* b_res,
                            float* tokmat, float* dz, float* dp, float* tokgrad, cudaStream_t st) {
    (void)b_post;
    // Sinkhorn checkpoints (last slot): segments of L half-steps, at most ~96 KB per block
    const int KMv = d.k <= 4 ? 4 : 8, nth = 64;
    const int nh = 2 * d.iters;
    const int segmax = std::max(1, (96 * 1024) / (KMv * KMv * 4 * nth));
    const int L = std::max(8, (nh + segmax - 1) / segmax);
    const int nseg = std::max(1, (nh + L - 1) / L);
    const size_t sm = (slot == d.G - 1) ? (size_t)nseg * KMv * KMv * 4 * nth : 0;
    cudaError_t e;
    if (d.k <= 4) {
        if ((e = cudaFuncSetAttribute((const void*)k_bwd_coef<4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)std::max<size_t>(sm, 1))) != cudaSuccess)
            return e;
        k_bwd_coef<4><<<(T + nth - 1) / nth, nth, sm, st>>>(d, slot, T, red, nslice, zact, rs, p, hpost, gram,
                                                            L, alpha_post, b_post, alpha_res, b_res, tokmat,
                                                            dz, dp, tokgrad); note_launch();
    } else {
        if ((e = cudaFuncSetAttribute((const void*)k_bwd_coef<8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)std::max<size_t>(sm, 1))) != cudaSuccess)
            return e;
        k_bwd_coef<8><<<(T + nth - 1) / nth, nth, sm, st>>>(d, slot, T, red, nslice, zact, rs, p, hpost, gram,
                                                            L, alpha_post, b_post, alpha_res, b_res, tokmat,
                                                            dz, dp, tokgrad); note_launch();
    }
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------------------------
// full_coef: reverse of coef_full for one token.  dz columns follow zfull: [router | pre_0..].
// tokgrad: [0] = d mu / NC, [1] = 2 d nu / NC, [2 + q*N + i] = db_pre, [2 + G*N + q] = dalpha_pre,
// [2 + G*N + G + o] = mu * dZ_r[o]: the router logit subtracts mu * colsum(W_r), so every row of
// dW_r also receives -sum_t mu_t dZ_r[t][o].

__global__ void k_full_coef(Dims d, int T, const float* __restrict__ dhpre,
                            const float* __restrict__ hpre, const float* __restrict__ zfull,
                            const float* __restrict__ stats, const float* __restrict__ wsum,
                            const int* __restrict__ I, const float* __restrict__ dp,
                            const float* __restrict__ alpha_pre, float* __restrict__ dz,
                            float* __restrict__ tokgrad) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= T) return;
    const int N = d.N, G = d.G, n = d.nfull;
    const int roff = d.hr ? N : 0;
    const float mu = stats[(int64_t)t * 2], nu = stats[(int64_t)t * 2 + 1];
    const float rstd = 1.0f / sqrtf(nu + d.eps);
    const float* zf = zfull + (int64_t)t * n;
    float* dzt = dz + (int64_t)t * n;
    float* tg = tokgrad + (int64_t)t * NTG;
    float drstd = 0.f;
    for (int q = 0; q < G; ++q) {
        const float a = alpha_pre[q];
        float da = 0.f;
        for (int i = 0; i < N; ++i) {
            const float h = hpre[((int64_t)t * G + q) * N + i];
            const float dy = dhpre[((int64_t)t * G + q) * N + i] * h * (1.0f - h);
            const float zraw = zf[roff + q * N + i];
            dzt[roff + q * N + i] = a * dy * rstd;
            drstd += a * dy * zraw;
            da += dy * (zraw * rstd);
            tg[2 + q * N + i] = dy;
        }
        tg[2 + G * N + q] = da;
    }
    float dmu = 0.f;
    float dnu = -0.5f * drstd * rstd * rstd * rstd;
    if (d.hr) {
        const float lstd = 1.0f / sqrtf(nu - mu * mu + d.eps);
        float dlstd = 0.f;
        for (int i = 0; i < N; ++i) {
            dzt[i] = 0.f;
            tg[2 + G * N + G + i] = 0.f;
        }
        if (!d.softmax) {
            // sigmoid scores: only the selected routed streams' logits receive a gradient
            for (int j = d.m; j < d.k; ++j) {
                const int i = I[(int64_t)t * d.k + j];
                const float zc = zf[i] - mu * wsum[i];
                const float s = sigm(zc * lstd);
                const float dzr = dp[(int64_t)t * d.k + j] * s * (1.0f - s);
                dzt[i] = dzr * lstd;
                tg[2 + G * N + G + i] = mu * dzr * lstd;
                dmu -= dzr * lstd * wsum[i];
                dlstd += dzr * zc;
            }
        } else {
            // softmax scores s = softmax(z): dz_l = s_l (g_l - sum_j dp_j s_{I_j}), g_l = dp_j
            // where l = I_j is a selected routed stream, 0 elsewhere; every logit receives one
            float zmax = -INFINITY;
            for (int i = 0; i < N; ++i) zmax = fmaxf(zmax, (zf[i] - mu * wsum[i]) * lstd);
            float den = 0.f;
            for (int i = 0; i < N; ++i) den += expf((zf[i] - mu * wsum[i]) * lstd - zmax);
            float gs[MAXN];
            for (int i = 0; i < N; ++i) gs[i] = 0.f;
            float dot = 0.f;
            for (int j = d.m; j < d.k; ++j) {
                const int i = I[(int64_t)t * d.k + j];
                const float s = expf((zf[i] - mu * wsum[i]) * lstd - zmax) / den;
                gs[i] = dp[(int64_t)t * d.k + j];
                dot += gs[i] * s;
            }
            for (int i = 0; i < N; ++i) {
                const float zc = zf[i] - mu * wsum[i];
                const float s = expf(zc * lstd - zmax) / den;
                const float dzr = s * (gs[i] - dot);
                dzt[i] = dzr * lstd;
                tg[2 + G * N + G + i] = mu * dzr * lstd;
                dmu -= dzr * lstd * wsum[i];
                dlstd += dzr * zc;
            }
        }
        const float l3 = lstd * lstd * lstd;
        dnu += -0.5f * dlstd * l3;
        dmu += dlstd * mu * l3;
    }
    const float inv_nc = 1.0f / (float)(N * d.C);
    tg[0] = dmu * inv_nc;
    tg[1] = 2.0f * dnu * inv_nc;
}

cudaError_t launch_full_coef(const Dims& d, int T, const float* dhpre, const float* hpre,
                             const float* zfull, const float* stats, const float* wsum,
                             const int* I, const float* dp, const float* alpha_pre, float* dz,
                             float* tokgrad, cudaStream_t st) {
    k_full_coef<<<(T + 127) / 128, 128, 0, st>>>(d, T, dhpre, hpre, zfull, stats, wsum, I, dp,
                                                  alpha_pre, dz, tokgrad); note_launch();
    return cudaGetLastError();
}

}  // namespace xhc
