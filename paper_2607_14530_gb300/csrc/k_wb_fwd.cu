// Launchers of the forward write-back kernels (wb_gram, wb_coef, wb_fwd).
#include "k_wb.cuh"

namespace xhc {
namespace {

// ---------------------------------------------------------------------------------------------
// wb_coef: one thread per token.  With Gram-Schmidt, the slice partials of the Gram matrix are
// summed in fp64, kept in `gram` for the backward and turned into the coefficients B of Eq. gs
// (orthogonalised component q = sum_a B[q][a] u_a), so that the write-back of active slot j is
// sum_a E[j][a] u_a with E[j][a] = p_j sum_q H_post[j][q] B[q][a]; without it B is the
// identity.  E goes to the per-token matrix buffer (rows j < k, four entries each).

__global__ void __launch_bounds__(64) k_wb_coef(Dims d, int slot, int T, const float* __restrict__ red,
                                                int nslice, const float* __restrict__ p,
                                                const float* __restrict__ hpost,
                                                double* __restrict__ gram, float* __restrict__ emat) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= T) return;
    const int k = d.k, K = d.K[slot];
    const bool gs = (K > 1) && d.gs;
    // loops to MAXCOMP with guards on K: compile-time indices, the arrays stay in registers
    double B[MAXCOMP][MAXCOMP];
#pragma unroll
    for (int a = 0; a < MAXCOMP; ++a)
#pragma unroll
        for (int b = 0; b < MAXCOMP; ++b) B[a][b] = (a == b) ? 1.0 : 0.0;
    if (gs) {
        double Gm[MAXCOMP][MAXCOMP], cc[MAXCOMP][MAXCOMP], vv[MAXCOMP];
#pragma unroll
        for (int a = 0; a < MAXCOMP; ++a)
#pragma unroll
            for (int b = 0; b < MAXCOMP; ++b) Gm[a][b] = 0.0;
        for (int sl = 0; sl < nslice; ++sl) {
            const float* rp = red + ((int64_t)t * nslice + sl) * NRED;
#pragma unroll
            for (int a = 0; a < MAXCOMP; ++a)
#pragma unroll
                for (int b = 0; b <= a; ++b)
                    if (a < K) Gm[a][b] += (double)rp[a * (a + 1) / 2 + b];
        }
#pragma unroll
        for (int a = 0; a < MAXCOMP; ++a)
#pragma unroll
            for (int b = 0; b <= a; ++b)
                if (a < K) gram[(int64_t)t * NGRAM + a * (a + 1) / 2 + b] = Gm[a][b];
#pragma unroll
        for (int a = 0; a < MAXCOMP; ++a)
#pragma unroll
            for (int b = a + 1; b < MAXCOMP; ++b)
                if (b < K) Gm[a][b] = Gm[b][a];
        gs_coef(Gm, K, (double)d.eps_gs, B, cc, vv);
    }
    float* em = emat + (int64_t)t * TOKMAT;
    for (int j = 0; j < k; ++j) {
        const float pj = p[(int64_t)t * k + j];
#pragma unroll
        for (int a = 0; a < 4; ++a) {
            float e = 0.f;
            if (a < K) {
#pragma unroll
                for (int q = 0; q < MAXCOMP; ++q)
                    if (q < K) e += hpost[((int64_t)t * k + j) * K + q] * (float)B[q][a];
            }
            em[j * 4 + a] = pj * e;
        }
    }
}

template <int KW, int KS>
cudaError_t gram_kw(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw, int nslice,
                    float* red, cudaStream_t st) {
    const int TB = run_len(KW, 64);
    const size_t sm = (size_t)TB * (WT / 32) * 16 * sizeof(float);
    cudaError_t e = smem_attr((const void*)k_wb_gram<KW, KS>, sm);
    if (e != cudaSuccess) return e;
    dim3 grid(nslice, (unsigned)n_runs(d, T, TB, true));
    k_wb_gram<KW, KS><<<grid, WT, sm, st>>>(d, slot, T, TB, out, cw, nslice, red); note_launch();
    return cudaGetLastError();
}

template <int KM, int KW, int KS>
cudaError_t fwd_kw(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw, const float* emat,
                   int nslice, const uint16_t* xact, const int* I, const float* hres,
                   uint16_t* xact_next, uint16_t* X, cudaStream_t st) {
    const int TB = KW > 0 ? 128 : run_len(KW, 96);   // 128 measured faster than 96 with the block ring
    const size_t sm = sizeof(FRing<KM>) + (size_t)TB * (KM * 4 + KM * KM + KM) * 4;
    cudaError_t e = smem_attr((const void*)k_wb_fwd<KM, KW, KS>, sm);
    if (e != cudaSuccess) return e;
    dim3 grid(nslice, (unsigned)n_runs(d, T, TB, KW > 0));
    k_wb_fwd<KM, KW, KS><<<grid, WT, sm, st>>>(d, slot, T, TB, out, cw, emat, xact, I, hres, xact_next,
                                               X); note_launch();
    return cudaGetLastError();
}

template <int KM>
cudaError_t fwd8_kw(const Dims& d, int slot, int T, const uint16_t* out, const float* emat,
                    const uint16_t* xact, const int* I, const float* hres, uint16_t* xact_next,
                    uint16_t* X, cudaStream_t st) {
    const int TB = 32;
    const size_t sm = (size_t)TB * (KM + KM * KM + KM) * 4;
    dim3 grid((d.C + W8 - 1) / W8, (T + TB - 1) / TB);
    k_wb_fwd8<KM><<<grid, WT, sm, st>>>(d, slot, T, TB, out, emat, xact, I, hres, xact_next, X); note_launch();
    return cudaGetLastError();
}

}  // namespace

int wb_nslice(int C) { return (C + WSL - 1) / WSL; }
int wb_conv_runs(const Dims& d, int64_t T) {
    const int KW = kw_of(d);
    return (int)n_runs(d, (int)T, bapp_run(KW), true);
}

// the two-pair Gram kernel: the (4, 8, 12) taps and C a multiple of WSL2
static bool gram2_ok(const Dims& d) { return paper_kaps(d) && d.C % WSL2 == 0; }

// partial-sum slices per token of the Gram kernel (read back by wb_coef)
int wb_gram_slices(const Dims& d) { return gram2_ok(d) ? d.C / WSL2 : wb_nslice(d.C); }

cudaError_t launch_wb_gram(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw,
                           int nslice, float* red, cudaStream_t st) {
    if (gram2_ok(d)) {
        const int TB = 64;
        const size_t sm = (size_t)TB * (WT / 32) * 16 * sizeof(float);
        dim3 grid(d.C / WSL2, (unsigned)n_runs(d, T, TB, true));
        k_wb_gram2<<<grid, WT, sm, st>>>(d, slot, T, TB, out, cw, nslice, red); note_launch();
        return cudaGetLastError();
    }
    XHC_KW_DISPATCH(d, d.C % WSL == 0, (gram_kw<KWC, KSC>(d, slot, T, out, cw, nslice, red, st)));
}

cudaError_t launch_wb_coef(const Dims& d, int slot, int T, const float* red, int nslice, const float* p,
                           const float* hpost, double* gram, float* emat, cudaStream_t st) {
    k_wb_coef<<<(T + 63) / 64, 64, 0, st>>>(d, slot, T, red, nslice, p, hpost, gram, emat); note_launch();
    return cudaGetLastError();
}

cudaError_t launch_wb_fwd(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw,
                          const float* emat, int nslice, const uint16_t* xact, const int* I,
                          const float* hres, uint16_t* xact_next, uint16_t* X, cudaStream_t st) {
    const bool conv = d.K[slot] > 1;
    if (d.k <= 4) {
        if (!conv) return fwd8_kw<4>(d, slot, T, out, emat, xact, I, hres, xact_next, X, st);
        XHC_KW_DISPATCH(d, wb_fast(d), (fwd_kw<4, KWC, KSC>(d, slot, T, out, cw, emat, nslice, xact, I, hres, xact_next, X, st)));
    }
    if (!conv) return fwd8_kw<8>(d, slot, T, out, emat, xact, I, hres, xact_next, X, st);
    XHC_KW_DISPATCH(d, false, (fwd_kw<8, KWC, KSC>(d, slot, T, out, cw, emat, nslice, xact, I, hres, xact_next, X, st)));
}

}  // namespace xhc
