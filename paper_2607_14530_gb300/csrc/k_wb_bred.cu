// Launcher of the backward write-back reductions (wb_bred).
#include "k_wb.cuh"

namespace xhc {
namespace {

template <int KM, int KW, int NV, int KS>
cudaError_t bred_kw(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw, const uint16_t* dX,
                    const int* I, const float* dxact, const uint16_t* xact, int nslice, float* red,
                    cudaStream_t st) {
    constexpr int NVP = NV < 32 ? 16 : NV;
    int TB = KW > 0 ? 64 : run_len(KW, 48);   // 64 measured faster than 48 with the block ring
    while (TB > 4 && (size_t)TB * (WT / 32) * NVP * 4 > 96 * 1024) TB -= 4;
    const size_t sm = sizeof(BRing<KM>) + (size_t)TB * KM * 4 + (size_t)TB * (WT / 32) * NVP * sizeof(float);
    cudaError_t e = smem_attr((const void*)k_wb_bred<KM, KW, NV, KS>, sm);
    if (e != cudaSuccess) return e;
    dim3 grid(nslice, (unsigned)n_runs(d, T, TB, KW > 0));
    k_wb_bred<KM, KW, NV, KS><<<grid, WT, sm, st>>>(d, slot, T, TB, out, cw, dX, I, dxact, xact, nslice, red); note_launch();
    return cudaGetLastError();
}

template <int KM, int NV>
cudaError_t bred2_kw(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw, const uint16_t* dX,
                     const int* I, const float* dxact, const uint16_t* xact, int nslice, float* red,
                     cudaStream_t st) {
    constexpr int NVP = NV < 32 ? 16 : NV;
    const int TB = 64;
    const size_t sm = sizeof(BRing2<KM>) + (size_t)TB * KM * 4 + (size_t)TB * (WT / 32) * NVP * sizeof(float);
    cudaError_t e = smem_attr((const void*)k_wb_bred2<KM, NV>, sm);
    if (e != cudaSuccess) return e;
    dim3 grid(d.C / WSL2, (unsigned)n_runs(d, T, TB, true));
    k_wb_bred2<KM, NV><<<grid, WT, sm, st>>>(d, slot, T, TB, out, cw, dX, I, dxact, xact, nslice, red); note_launch();
    return cudaGetLastError();
}

// the two-pair reductions: the (4, 8, 12) taps, k = 4, C a multiple of WSL2
bool bred2_ok(const Dims& d) { return paper_kaps(d) && d.k == 4 && d.C % WSL2 == 0; }

template <int KM>
cudaError_t b8_kw(const Dims& d, int slot, int T, const uint16_t* out, const uint16_t* dX, const int* I,
                  const float* p, const float* hpost, const float* hres, const float* dxact,
                  float* dxact_out, const uint16_t* xact, int nslice, float* red, uint16_t* d_out,
                  cudaStream_t st) {
    constexpr int NQ = KM + KM * KM;
    constexpr int NV = NQ <= 32 ? 32 : 96;
    const int TB = 32;
    const size_t sm = (size_t)TB * (2 * KM + KM * KM) * 4 + (size_t)TB * (WT / 32) * NV * 4;
    cudaError_t e = smem_attr((const void*)k_wb_b8<KM>, sm);
    if (e != cudaSuccess) return e;
    dim3 grid((d.C + W8 - 1) / W8, (T + TB - 1) / TB);
    k_wb_b8<KM><<<grid, WT, sm, st>>>(d, slot, T, TB, out, dX, I, p, hpost, hres, dxact, dxact_out, xact,
                                      nslice, red, d_out); note_launch();
    return cudaGetLastError();
}

}  // namespace

// slices (partial sums per token) of the backward reductions of a slot
int wb_bred_slices(const Dims& d, int slot) {
    if (d.K[slot] == 1) return (d.C + W8 - 1) / W8;
    return bred2_ok(d) ? d.C / WSL2 : wb_nslice(d.C);
}

cudaError_t launch_wb_bred(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw,
                           const uint16_t* dX, const int* I, const float* dxact,
                           const uint16_t* xact, int nslice, float* red, cudaStream_t st) {
    const bool conv = d.K[slot] > 1;
    const bool last = (slot == d.G - 1);
    // a slot without conv takes the one-pass backward (launch_wb_b8), not this kernel
    if (!conv) return cudaErrorInvalidValue;
    if (bred2_ok(d)) {
        if (last) return bred2_kw<4, 32>(d, slot, T, out, cw, dX, I, dxact, xact, nslice, red, st);
        return bred2_kw<4, 16>(d, slot, T, out, cw, dX, I, dxact, xact, nslice, red, st);
    }
#define XHC_BRED(KM_, NV_, FAST_)                                                                   \
    do {                                                                                            \
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

// backward reductions and apply of a slot without conv (K = 1), in one pass over dXn
cudaError_t launch_wb_b8(const Dims& d, int slot, int T, const uint16_t* out, const uint16_t* dX,
                         const int* I, const float* p, const float* hpost, const float* hres,
                         const float* dxact, float* dxact_out, const uint16_t* xact, int nslice,
                         float* red, uint16_t* d_out, cudaStream_t st) {
    if (d.K[slot] != 1) return cudaErrorInvalidValue;
    if (d.k <= 4)
        return b8_kw<4>(d, slot, T, out, dX, I, p, hpost, hres, dxact, dxact_out, xact, nslice, red, d_out, st);
    return b8_kw<8>(d, slot, T, out, dX, I, p, hpost, hres, dxact, dxact_out, xact, nslice, red, d_out, st);
}

}  // namespace xhc
