// Launcher of the backward write-back apply (wb_bapp).
#include "k_wb.cuh"

namespace xhc {
namespace {

template <int KM, int KW, int KS, bool HALO = false>
cudaError_t bapp_kw(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw, const uint16_t* dX,
                    const int* I, const float* dn_in, const float* tokmat, float* dxact_out,
                    uint16_t* d_out, float* cpart, int nslice, cudaStream_t st) {
    const int TB = bapp_run(KW);
    const int TH = TB + (KW > 0 ? KW - 1 : 0);
    const size_t sm = sizeof(ARing<KM>) + (size_t)TH * (KM * 4 + 16 + KM * KM + KM) * 4;
    cudaError_t e = smem_attr((const void*)k_wb_bapp<KM, KW, KS, HALO>, sm);
    if (e != cudaSuccess) return e;
    dim3 grid(nslice, (unsigned)n_runs(d, T, TB, KW > 0));
    k_wb_bapp<KM, KW, KS, HALO><<<grid, WT, sm, st>>>(d, slot, T, TB, out, cw, dX, I, dn_in, tokmat,
                                                      dxact_out, d_out, cpart); note_launch();
    return cudaGetLastError();
}

// a call that returns a halo gradient: the generic tap variants with the halo code
template <int KM>
cudaError_t bapp_halo(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw, const uint16_t* dX,
                      const int* I, const float* dn_in, const float* tokmat, float* dxact_out,
                      uint16_t* d_out, float* cpart, int nslice, cudaStream_t st) {
    switch (kw_of(d)) {
        case 4: return bapp_kw<KM, 4, 0, true>(d, slot, T, out, cw, dX, I, dn_in, tokmat, dxact_out, d_out, cpart, nslice, st);
        case 8: return bapp_kw<KM, 8, 0, true>(d, slot, T, out, cw, dX, I, dn_in, tokmat, dxact_out, d_out, cpart, nslice, st);
        case 12: return bapp_kw<KM, 12, 0, true>(d, slot, T, out, cw, dX, I, dn_in, tokmat, dxact_out, d_out, cpart, nslice, st);
        default: return bapp_kw<KM, 16, 0, true>(d, slot, T, out, cw, dX, I, dn_in, tokmat, dxact_out, d_out, cpart, nslice, st);
    }
}

}  // namespace

cudaError_t launch_wb_bapp(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw,
                           const uint16_t* dX, const int* I, const float* dn_in,
                           const float* tokmat, float* dxact_out, uint16_t* d_out, float* cpart,
                           cudaStream_t st) {
    const int nslice = wb_nslice(d.C);
    const bool conv = d.K[slot] > 1;
    if (conv && cw.dhalo != nullptr) {
        if (d.k <= 4) return bapp_halo<4>(d, slot, T, out, cw, dX, I, dn_in, tokmat, dxact_out, d_out, cpart, nslice, st);
        return bapp_halo<8>(d, slot, T, out, cw, dX, I, dn_in, tokmat, dxact_out, d_out, cpart, nslice, st);
    }
    // a slot without conv takes the one-pass backward (launch_wb_b8), not this kernel
    if (!conv) return cudaErrorInvalidValue;
    if (d.k <= 4) {
        XHC_KW_DISPATCH(d, wb_fast(d), (bapp_kw<4, KWC, KSC>(d, slot, T, out, cw, dX, I, dn_in, tokmat, dxact_out, d_out, cpart, nslice, st)));
    }
    XHC_KW_DISPATCH(d, false, (bapp_kw<8, KWC, KSC>(d, slot, T, out, cw, dX, I, dn_in, tokmat, dxact_out, d_out, cpart, nslice, st)));
}

}  // namespace xhc
