// Routing and pre-maps without any device allocation by the caller or the library.
//
// Some callers cannot allocate device memory for the workspace that xhc_pre_fwd expects: code
// that runs inside another allocator's arena, inference engines that fix every buffer at start-up,
// or plug-ins whose host framework owns all device memory.  xhc_route_noalloc serves them: it
// runs the full-state mapping generation of one group (norm statistics, the projections of
// Eq. fused_normalized_projection, Eq. router_topk, Eq. param_pre) with its split-K partial sums
// in a fixed-size array that is part of this library's device image, so the caller passes only
// inputs and outputs.
#include <string.h>

#include <mutex>

#include "xhc_internal.cuh"

namespace {

// Scratch of xhc_route_noalloc.  Part of the loaded module: every GPU that loads the library
// holds these bytes until the process exits.
static __device__ __align__(256) unsigned char g_route_scratch[XHC_NOALLOC_SCRATCH_BYTES];

std::mutex g_mu;
void* g_ptr[128];
bool g_ready[128];

size_t al256(size_t x) { return (x + 255) & ~(size_t)255; }

}  // namespace

using namespace xhc;

extern "C" xhc_status xhc_route_noalloc(const xhc_handle* hh, int64_t T, const xhc_params* P,
                                        const uint16_t* X, int32_t* I, float* p, float* hpre,
                                        void* stream) {
    if (!hh || !P || !X || !I || !p || !hpre || T <= 0 || T > ((int64_t)1 << 30))
        return XHC_ERR_INVALID_ARG;
    if ((((uintptr_t)X) | ((uintptr_t)I) | ((uintptr_t)p) | ((uintptr_t)hpre)) & 15u)
        return XHC_ERR_ALIGNMENT;
    Dims d = hh->h.d;
    d.S = (int)T;  // no conv here: the sequence length plays no role
    if (d.hr && !P->W_r) return XHC_ERR_INVALID_ARG;
    for (int q = 0; q < d.G; ++q)
        if (!P->W_pre[q]) return XHC_ERR_INVALID_ARG;
    if (!P->alpha_pre || !P->b_pre) return XHC_ERR_INVALID_ARG;

    // scratch layout, same split-K choice as xhc_pre_fwd
    const Layout L = make_layout(d, T);
    const int splits = L.splits_full;
    const size_t t = (size_t)T;
    size_t o = 0;
    const size_t o_part = o;  o = al256(o + (size_t)splits * t * d.nfull * 4);
    const size_t o_pst = o;   o = al256(o + (size_t)splits * t * 2 * 4);
    const size_t o_wsum = o;  o = al256(o + (size_t)d.N * 4);
    const size_t o_scr = o;   o = al256(o + (size_t)64 * 256 * 4);
    const size_t o_zf = o;    o = al256(o + t * d.nfull * 4);
    const size_t o_st = o;    o = al256(o + t * 2 * 4);
    if (o > (size_t)XHC_NOALLOC_SCRATCH_BYTES) return XHC_ERR_UNSUPPORTED;

    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 128) return XHC_ERR_CUDA;
    char* base = nullptr;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        if (!g_ready[dev]) {
            void* ptr = nullptr;
            if (cudaGetSymbolAddress(&ptr, g_route_scratch) != cudaSuccess || ptr == nullptr)
                return XHC_ERR_CUDA;
            g_ptr[dev] = ptr;
            g_ready[dev] = true;
        }
        base = (char*)g_ptr[dev];
    }
    cudaStream_t st = (cudaStream_t)stream;
    float* part = (float*)(base + o_part);
    float* pst = (float*)(base + o_pst);
    float* wsum = (float*)(base + o_wsum);
    float* scr = (float*)(base + o_scr);
    // every scratch word read below is first written by this call (split-K partials, column
    // sums, statistics), so no clearing is needed
    if (d.hr && launch_colsum(P->W_r, d.N * d.C, d.N, d.N, wsum, 0, scr, st) != cudaSuccess)
        return XHC_ERR_CUDA;
    WSegs w;
    memset(&w, 0, sizeof(w));
    int off = 0;
    if (d.hr) {
        w.ptr[w.n] = P->W_r; w.width[w.n] = d.N; w.off[w.n] = off; off += d.N; ++w.n;
    }
    for (int q = 0; q < d.G; ++q) {
        w.ptr[w.n] = P->W_pre[q]; w.width[w.n] = d.N; w.off[w.n] = off; off += d.N; ++w.n;
    }
    w.off[w.n] = off;
    if (launch_rowproj(X, (int64_t)d.N * d.C, d.N * d.C, (int)T, w, d.nfull, splits, part, pst, st) !=
        cudaSuccess)
        return XHC_ERR_CUDA;
    if (launch_coef_full(d, (int)T, part, pst, splits, wsum, P->alpha_pre, P->b_pre,
                         (float*)(base + o_zf), (float*)(base + o_st), hpre, I, p, st) != cudaSuccess)
        return XHC_ERR_CUDA;
    return XHC_OK;
}
