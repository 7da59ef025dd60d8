// Launcher of the backward write-back reductions (wb_bred).
#include "k_wb.cuh"

namespace xhc {
namespace {

template <int KM, int KW, int NV, int KS>
cudaError_t bred_kw(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw, const uint16_t* dX,
                    const int* I, const float* dxact, const uint16_t* xact, int nslice, float* red,
                    cudaStream_t st) {
    constexpr int NVP = NV < 32 ? 16 : NV;
    int TB = run_len(KW, 48);
    while (TB > (KW > 0 ? KW : 4) && (size_t)TB * (WT / 32) * NVP * 4 > 96 * 1024) TB -= (KW > 0 ? KW : 4);
    const size_t sm = sizeof(BRing<KM>) + (size_t)TB * KM * 4 + (size_t)TB * (WT / 32) * NVP * sizeof(float);
    cudaError_t e = smem_attr((const void*)k_wb_bred<KM, KW, NV, KS>, sm);
    if (e != cudaSuccess) return e;
    dim3 grid(nslice, (unsigned)n_runs(d, T, TB, KW > 0));
    k_wb_bred<KM, KW, NV, KS><<<grid, WT, sm, st>>>(d, slot, T, TB, out, cw, dX, I, dxact, xact, nslice, red); note_launch();
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_wb_bred(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw,
                           const uint16_t* dX, const int* I, const float* dxact,
                           const uint16_t* xact, int nslice, float* red, cudaStream_t st) {
    const bool conv = d.K[slot] > 1;
    const bool last = (slot == d.G - 1);
#define XHC_BRED(KM_, NV_, FAST_)                                                                   \
    do {                                                                                            \
        if (!conv && (FAST_)) return bred_kw<KM_, 0, NV_, 2>(d, slot, T, out, cw, dX, I, dxact, xact, nslice, red, st); \
        if (!conv) return bred_kw<KM_, 0, NV_, 0>(d, slot, T, out, cw, dX, I, dxact, xact, nslice, red, st); \
        XHC_KW_DISPATCH(d, FAST_, (bred_kw<KM_, KWC, NV_, KSC>(d, slot, T, out, cw, dX, I, dxact, xact, nslice, red, st))); \
    } while (0)
    if (d.k <= 4) {
        if (last) XHC_BRED(4, 32, wb_fast(d));
        XHC_BRED(4, 16, wb_fast(d));
    }
    if (last) XHC_BRED(8, 96, false);
    XHC_BRED(8, 32, false);
#undef XHC_BRED
}

}  // namespace xhc
