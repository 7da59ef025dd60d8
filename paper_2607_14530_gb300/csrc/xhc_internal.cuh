// Internal declarations of libxhc: dimensions, buffer layout, device helpers, launchers.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>
#include <stddef.h>

#include "../../include/xhc.h"

namespace xhc {

constexpr int MAXN = 32;     // streams
constexpr int MAXK = 8;      // active streams
constexpr int MAXKAP = 16;   // conv kernel size
constexpr int MAXCOMP = 4;   // write-back components (1 + r)
constexpr int MAXSEG = 5;    // weight segments of one projection (router + 4 pre-maps)

// Everything a kernel needs to know about the group's shape (passed by value).
struct Dims {
    int N, k, m, C, G;
    int hr;              // 1 if the group has a router (m < k)
    int nfull;           // columns of the full-state projection: (hr ? N : 0) + G * N
    int S;               // sequence length
    int iters;           // Sinkhorn iterations
    float eps;           // norm epsilon
    float eps_gs;        // Gram-Schmidt epsilon (already resolved)
    int gs;              // Gram-Schmidt on/off
    int nconv;           // conv branches r
    int kap[3];          // kernel sizes
    int kapmax;          // max kernel size
    int kapsum;          // sum of kernel sizes
    int K[4];            // write-back components per slot
    int nact[4];         // active projection width per slot: k*K_t (+ k*k for the last slot)
    int softmax;         // router scores: 0 sigmoid (Eq. router), 1 softmax over the N logits
    int dense;           // 1: dense read of all N streams (Eq. dense_read); 0: active streams only
};

// Column segments of a projection weight: column o of the logical [rows, n] matrix lives in
// segment s with off[s] <= o < off[s+1] at ptr[s][row * width[s] + (o - off[s])].
struct WSegs {
    const float* ptr[MAXSEG];
    int width[MAXSEG];
    int off[MAXSEG + 1];
    int n;  // number of segments
};
struct WSegsOut {
    float* ptr[MAXSEG];
    int width[MAXSEG];
    int off[MAXSEG + 1];
    int n;
};

// Stream-K plan of the tensor-core full-state projection.
struct ProjTcPlan {
    int KB, MT;      // k-blocks per tile, token tiles
    long long W;     // total k-blocks
    int P;           // persistent CTAs
    int nseg;        // partial slots per tile
    int NB;          // B rows (hi + lo + pad)
    int nchunk;      // MMA instructions per k-step
    int kps;         // k-blocks of 64 per stage
    int ctas;        // CTAs per SM
};
ProjTcPlan plan_proj_tc(int T, int K, int nfull, int nsm, bool proj);  // proj: A = X rows (else weight gradient)
int device_sms();

// Byte offsets of the per-group buffers for a given T (all 256-byte aligned).
struct Layout {
    // saved
    size_t xact;            // bf16 [G][T][k][C]: active state entering slot t
    size_t I;               // int32 [T][k]
    size_t p;               // f32 [T][k]
    size_t stats;           // f32 [T][2]: mu, nu of the flattened entry state
    size_t zfull;           // f32 [T][nfull]: raw projections x W
    size_t hpre;            // f32 [T][G][N]
    size_t zact[4];         // f32 [T][nact_t]: raw active projections
    size_t rs[4];           // f32 [T]: active rstd
    size_t hpost[4];        // f32 [T][k*K_t]
    size_t hres;            // f32 [T][k*k]
    size_t gram[4];         // f64 [T][NGRAM]: Gram matrix of the write-back components (lower
                            // triangle), slots with a temporal conv and Gram-Schmidt
    size_t saved_total;
    // workspace
    size_t err;             // int: device error word (first 256 bytes of the workspace)
    size_t wpack;           // bf16 [NB][N*C]: hi / lo rows of the full-state projection weight
    size_t part;            // f32 [splits][T][nmax] projection split-K partials
    size_t pstats;          // f32 [splits][T][2]
    size_t astat;           // f32 [stream_warps(C)][T][2]: per-warp partial sums of squares (at 1;
                            // 0 is not written) of the active state being mapped
    size_t wsum;            // f32 [N]: column sums of W_r
    size_t rsum;            // f32 [N]: sum_t mu_t dZ_r[t] (router mean-term gradient)
    size_t base;            // bf16 [G-1][T][C]: non-active base readouts of slots 1..G-1
    size_t red;             // f32 [T][nslice][NRED]: per-slice reduction partials
    size_t dxact;           // f32 [T][k][C]: active-state gradient
    size_t dinput;          // bf16 [G][T][C]: copies of d_input
    size_t dotp;            // f32 [k][C/32][T]: <x_act_j, d_input> over 32-channel groups
    size_t dp;              // f32 [T][k]: routing-weight gradient accumulated over slots
    size_t dhpre;           // f32 [T][G][N]
    size_t tokmat;          // f32 [T][TOKMAT]: per-token matrices (E, D, H_res, scalars)
    size_t dz;              // f32 [T][max(nfull, nact)]: projection-output gradients
    size_t tokgrad;         // f32 [T][NTG]: per-token alpha / b gradient contributions
    size_t wpart;           // f32 [tsplits][rows * n]: weight-gradient partials
    size_t cpart;           // f32 [ntiles][kapsum][C]: conv weight-gradient partials
    size_t colscr;          // f32 [64][256]: column-sum scratch
    size_t ws_total;
    int splits_full, splits_act, nslice, tsplits, ntiles;
    ProjTcPlan tc;          // full-state projection: rows T, K = N*C
    ProjTcPlan tca;         // active projection: rows T, K = k*C
    ProjTcPlan twf;         // full weight gradient: rows N*C, K = T
    ProjTcPlan twa;         // active weight gradient: rows k*C, K = T
    size_t dzpack;          // bf16 [NB][T]: hi / lo rows of the projection-output gradient
    size_t dz16;            // bf16 [T][ld]: projection-output gradient (full-state dX GEMM)
    size_t w16;             // bf16 [N*C][ld]: full-state projection weight rows
};

constexpr int NGRAM = 10;    // lower triangle of the 4 x 4 component Gram matrix
constexpr int NRED = 112;    // per-token reduction slots (>= k*K + k*k + K*K)
constexpr int TOKMAT = 176;  // E[k][4] + D[4][4] + Hres[k][k] + dX_act mix + scalars (k<=8)
constexpr int NTG = 208;     // per-token alpha/b gradient contributions

// Conv taps of one MLP slot (by value into kernels): w[j] is [kappa_j, C].  For a call on a
// later chunk of its sequences (sequence split), halo [B][R][C] bf16 holds the R = max(kappa) - 1
// sublayer outputs preceding each sequence of the call (null: none, zero padding as at a
// sequence start) and dhalo [B][R][C] fp32 receives their gradient (backward apply only).
struct ConvPtrs {
    const float* w[3];
    const uint16_t* halo;
    float* dhalo;
};
struct ConvGradPtrs {
    float* w[3];
};

struct Handle {
    xhc_config cfg;
    Dims d;
};

}  // namespace xhc

// The opaque handle of the C ABI (include/xhc.h), defined once for every translation unit.
struct xhc_handle {
    xhc::Handle h;
};

namespace xhc {

Layout make_layout(const Dims& d, int64_t T);
Dims make_dims(const xhc_config& c);

// ---------------------------------------------------------------------------------------------
// device helpers

__device__ __forceinline__ float bf2f(uint16_t v) {
    return __uint_as_float(((uint32_t)v) << 16);
}
__device__ __forceinline__ uint16_t f2bf(float f) {
    return __bfloat16_as_ushort(__float2bfloat16_rn(f));
}
__device__ __forceinline__ void unpack8(const uint4& u, float* f) {
    f[0] = __uint_as_float(u.x << 16); f[1] = __uint_as_float(u.x & 0xffff0000u);
    f[2] = __uint_as_float(u.y << 16); f[3] = __uint_as_float(u.y & 0xffff0000u);
    f[4] = __uint_as_float(u.z << 16); f[5] = __uint_as_float(u.z & 0xffff0000u);
    f[6] = __uint_as_float(u.w << 16); f[7] = __uint_as_float(u.w & 0xffff0000u);
}
// two floats to bf16 (round to nearest even) in one conversion: a in the low half, b in the high
__device__ __forceinline__ uint32_t pack2(float a, float b) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    uint32_t r;
    memcpy(&r, &h, sizeof(r));
    return r;
}
// 8 bf16 as 4 channel pairs (low half first)
__device__ __forceinline__ void unpack4x2(const uint4& u, float2* f) {
    f[0] = make_float2(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u));
    f[1] = make_float2(__uint_as_float(u.y << 16), __uint_as_float(u.y & 0xffff0000u));
    f[2] = make_float2(__uint_as_float(u.z << 16), __uint_as_float(u.z & 0xffff0000u));
    f[3] = make_float2(__uint_as_float(u.w << 16), __uint_as_float(u.w & 0xffff0000u));
}
__device__ __forceinline__ uint4 pack8(const float* f) {
    return make_uint4(pack2(f[0], f[1]), pack2(f[2], f[3]), pack2(f[4], f[5]), pack2(f[6], f[7]));
}
__device__ __forceinline__ float sigm(float z) { return 1.0f / (1.0f + expf(-z)); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ int seg_of(const WSegs& w, int o) {
    int s = 0;
#pragma unroll
    for (int q = 1; q < MAXSEG; ++q)
        if (q < w.n && o >= w.off[q]) s = q;
    return s;
}
// W[r][o] of the segmented weight (the segment of column o): the segment's fields are selected
// with static indices, so the kernel parameter is not copied to local memory for a dynamic index
template <bool RO = false>
__device__ __forceinline__ float seg_elem(const WSegs& w, long long r, int o) {
    const float* p = w.ptr[0];
    int width = w.width[0], off = w.off[0];
#pragma unroll
    for (int q = 1; q < MAXSEG; ++q)
        if (q < w.n && o >= w.off[q]) {
            p = w.ptr[q];
            width = w.width[q];
            off = w.off[q];
        }
    return RO ? __ldg(p + r * width + (o - off)) : p[r * width + (o - off)];
}

// ---------------------------------------------------------------------------------------------
// Gram-Schmidt of Eq. gs expressed on the Gram matrix of u = [out, g_1, ..., g_r]:
// v_j = sum_a B[j][a] u_a, B unit lower-triangular.  Denominators <v_i, v_i> + eps.

// The loops run to MAXCOMP with guards on K (the same operations in the same order as loops to
// K), so every array index is a compile-time constant and the arrays stay in registers.
__device__ inline void gs_coef(const double (&G)[MAXCOMP][MAXCOMP], int K, double eps,
                        double (&B)[MAXCOMP][MAXCOMP], double (&c)[MAXCOMP][MAXCOMP],
                        double (&vv)[MAXCOMP]) {
#pragma unroll
    for (int j = 0; j < MAXCOMP; ++j)
#pragma unroll
        for (int a = 0; a < MAXCOMP; ++a) {
            B[j][a] = (j == a) ? 1.0 : 0.0;
            c[j][a] = 0.0;
        }
#pragma unroll
    for (int j = 0; j < MAXCOMP; ++j) {
        if (j >= K) break;
#pragma unroll
        for (int i = 0; i < j; ++i) {
            double num = 0.0;
#pragma unroll
            for (int a = 0; a <= i; ++a) num += B[i][a] * G[j][a];
            c[j][i] = num / vv[i];
        }
#pragma unroll
        for (int i = 0; i < j; ++i)
#pragma unroll
            for (int a = 0; a <= i; ++a) B[j][a] -= c[j][i] * B[i][a];
        double q = 0.0;
#pragma unroll
        for (int a = 0; a <= j; ++a)
#pragma unroll
            for (int b = 0; b <= j; ++b) q += B[j][a] * B[j][b] * G[a][b];
        vv[j] = q + eps;
    }
}

// Reverse of gs_coef: dB (modified in place) -> dG (full, not symmetrised).
__device__ inline void gs_coef_bwd(const double (&G)[MAXCOMP][MAXCOMP], int K,
                            const double (&B)[MAXCOMP][MAXCOMP], const double (&c)[MAXCOMP][MAXCOMP],
                            const double (&vv)[MAXCOMP], double (&dB)[MAXCOMP][MAXCOMP],
                            double (&dG)[MAXCOMP][MAXCOMP]) {
    double dvv[MAXCOMP] = {0.0, 0.0, 0.0, 0.0};
#pragma unroll
    for (int a = 0; a < MAXCOMP; ++a)
#pragma unroll
        for (int b = 0; b < MAXCOMP; ++b) dG[a][b] = 0.0;
#pragma unroll
    for (int j = MAXCOMP - 1; j >= 0; --j) {
        if (j >= K) continue;
        // vv[j] = B[j]^T G B[j] + eps
        if (dvv[j] != 0.0) {
#pragma unroll
            for (int a = 0; a <= j; ++a) {
                double s = 0.0;
#pragma unroll
                for (int b = 0; b <= j; ++b) s += (G[a][b] + G[b][a]) * B[j][b];
                dB[j][a] += dvv[j] * s;
#pragma unroll
                for (int b = 0; b <= j; ++b) dG[a][b] += dvv[j] * B[j][a] * B[j][b];
            }
        }
        // B[j] = e_j - sum_i c[j][i] B[i];  c[j][i] = num / vv[i];  num = sum_a B[i][a] G[j][a]
#pragma unroll
        for (int i = j - 1; i >= 0; --i) {
            double dc = 0.0;
#pragma unroll
            for (int a = 0; a <= i; ++a) {
                dc -= dB[j][a] * B[i][a];
                dB[i][a] -= c[j][i] * dB[j][a];
            }
            const double dnum = dc / vv[i];
            dvv[i] -= dc * c[j][i] / vv[i];
#pragma unroll
            for (int a = 0; a <= i; ++a) {
                dB[i][a] += dnum * G[j][a];
                dG[j][a] += dnum * B[i][a];
            }
        }
    }
}

// ---------------------------------------------------------------------------------------------
// launch accounting and tracing (host side)

void note_launch();  // counts every kernel launch of the library
// test hooks (xhc_debug_set): the limit of the bounded device waits, and a one-shot request that
// the next full-state projection time out before it issues any copy
uint64_t debug_wait_ns();
int debug_take_force_timeout();

// ---------------------------------------------------------------------------------------------
// launchers (each returns cudaGetLastError() after enqueueing)

cudaError_t launch_rowproj(const uint16_t* A, int64_t lda, int K, int T, const WSegs& W, int n,
                           int splits, float* part, float* pstats, cudaStream_t st);
cudaError_t launch_pack_w(const WSegs& W, int nfull, int NB, int K, uint16_t* Wpack, cudaStream_t st);
// pstats null: no row statistics (the caller has them from the kernel that wrote X)
cudaError_t launch_proj_tc(const uint16_t* X, int T, int K, const uint16_t* Wpack, int nfull,
                           const ProjTcPlan& p, float* part, float* pstats, int* err,
                           cudaStream_t st);
cudaError_t launch_wgrad_tc(const uint16_t* A, int T, int E, const float* dz, int ldz, int n,
                            uint16_t* dzpack, const ProjTcPlan& p, float* part, int* err,
                            cudaStream_t st);
bool dx_tc_ok(int T, int N, int C, int nfull, int G);
bool dxa_tc_ok(int T, int k, int C, int nact);
// dX_act += dZ_act W_act^T (three-term bf16 split on the tensor cores) + H_pre[slot][I_j] d_input
//           - cx x_act (the write-back's own term, cx per token in tokmat);
// in the same pass: dotp[j][g][t] = <x_act_j, d_input> over channels 32 g .. 32 g + 31, and the
// copy dcopy[slot][t][:] = d_input[t][:]
cudaError_t launch_dxa_tc(const Dims& d, int slot, int T, const float* dzs, int nact, const WSegs& W,
                          uint16_t* dz3, uint16_t* w3, const uint16_t* d_input, const float* hpre,
                          const int* I, const uint16_t* xact, const float* tokmat, float* dxact,
                          float* dotp, uint16_t* dcopy, int* err, cudaStream_t st);
// dH_pre[t][slot][I_j] = sum over the C/32 groups g of dotp[j][g][t] (g in order)
cudaError_t launch_dots_act(const Dims& d, int slot, int T, const float* dotp, const int* I, float* dhpre,
                            cudaStream_t st);
cudaError_t launch_dx_tc(const Dims& d, int T, const float* dz, const WSegs& W, uint16_t* dz16,
                         uint16_t* w16, const uint16_t* X, const uint16_t* dinput, const float* hpre,
                         const int* I, const float* dxact, const float* scal, int scal_ld,
                         uint16_t* dX, int* err, cudaStream_t st);
int wb_nslice(int C);
int wb_gram_slices(const Dims& d);  // partial-sum slices of wb_gram (and wb_coef)
int wb_conv_runs(const Dims& d, int64_t T);
int wb_bred_slices(const Dims& d, int slot);  // partial-sum slices of wb_bred (and bwd_coef)  // runs (conv weight-gradient partials) of wb_bapp
// decode (one token per sequence, conv history in a per-sequence ring of max(kappa) - 1 rows)
cudaError_t launch_dec_gram(const Dims& d, int slot, int B, const uint16_t* out, ConvPtrs cw,
                            const uint16_t* ring, const long long* pos, float* red, cudaStream_t st);
cudaError_t launch_dec_fwd(const Dims& d, int slot, int B, const uint16_t* out, ConvPtrs cw,
                           uint16_t* ring, long long* pos, const float* emat, const uint16_t* xact,
                           const int* I, const float* hres, uint16_t* xact_next, uint16_t* X,
                           cudaStream_t st);
cudaError_t launch_ring_fill(const Dims& d, int B, int S, const uint16_t* out, uint16_t* ring,
                             cudaStream_t st);
int dec_nslice(int C);  // channel slices (partial Gram slots) of the decode Gram reduction
// model glue: N copies of a hidden vector per token, and the sum of the N streams
cudaError_t launch_stream_bcast(int T, int N, int C, const uint16_t* h, uint16_t* X, cudaStream_t st);
cudaError_t launch_stream_sum(int T, int N, int C, const uint16_t* X, uint16_t* y, cudaStream_t st);
// sequence split: the halo rows a chunk passes to the next, and the return of their gradient
cudaError_t launch_halo_fill(const Dims& d, int B, int S, const uint16_t* out, uint16_t* halo,
                             cudaStream_t st);
cudaError_t launch_halo_add(const Dims& d, int B, int S, uint16_t* d_out, const float* dhalo,
                            cudaStream_t st);
cudaError_t launch_wb_gram(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw,
                           int nslice, float* red, cudaStream_t st);
cudaError_t launch_wb_coef(const Dims& d, int slot, int T, const float* red, int nslice, const float* p,
                           const float* hpost, double* gram, float* emat, cudaStream_t st);
cudaError_t launch_wb_fwd(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw,
                          const float* emat, int nslice, const uint16_t* xact, const int* I,
                          const float* hres, uint16_t* xact_next, uint16_t* X, cudaStream_t st);
cudaError_t launch_wb_bred(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw,
                           const uint16_t* dX, const int* I, const float* dxact,
                           const uint16_t* xact, int nslice, float* red, cudaStream_t st);
cudaError_t launch_wb_b8(const Dims& d, int slot, int T, const uint16_t* out, const uint16_t* dX,
                         const int* I, const float* p, const float* hpost, const float* hres,
                         const float* dxact, float* dxact_out, const uint16_t* xact, int nslice,
                         float* red, uint16_t* d_out, cudaStream_t st);
cudaError_t launch_wb_bapp(const Dims& d, int slot, int T, const uint16_t* out, ConvPtrs cw,
                           const uint16_t* dX, const int* I, const float* dn_in,
                           const float* tokmat, float* dxact_out, uint16_t* d_out, float* cpart,
                           cudaStream_t st);
cudaError_t launch_wgrad_reduce(const float* wpart, int splits, int E, int n, const WSegsOut& G,
                                cudaStream_t st);
cudaError_t launch_colsum(const float* in, int rows, int ld, int n, float* out, int accumulate,
                          float* scratch, cudaStream_t st);
cudaError_t launch_sub_rows(float* G, int rows, int n, const float* v, cudaStream_t st);
// sum of split-K partial slots into slot 0, in slot order ([nslots][n] -> [n])
cudaError_t launch_slot_sum(float* x, int nslots, long long n, cudaStream_t st);
cudaError_t launch_coef_full(const Dims& d, int T, const float* part, const float* pstats,
                             int splits, const float* wsum, const float* alpha_pre,
                             const float* b_pre, float* zfull, float* stats, float* hpre,
                             int* I, float* p, cudaStream_t st);
cudaError_t launch_coef_act(const Dims& d, int slot, int T, const float* part,
                            const float* pstats, int ssplits, int splits, const float* alpha_post,
                            const float* b_post, const float* alpha_res, const float* b_res,
                            float* zact, float* rs, float* hpost, float* hres, cudaStream_t st);
int stream_warps(int C);  // warps per block of the one-block-per-token stream kernels
cudaError_t launch_read(const Dims& d, int T, const uint16_t* X, const float* hpre, const int* I,
                        uint16_t* input0, uint16_t* base, uint16_t* xact0, float* astat, cudaStream_t st);
cudaError_t launch_input(const Dims& d, int slot, int T, const uint16_t* base, const uint16_t* xact,
                         const float* hpre, const int* I, uint16_t* input, float* astat, cudaStream_t st);
cudaError_t launch_restore(const Dims& d, int T, const uint16_t* xact0, const int* I,
                           uint16_t* X, cudaStream_t st);
cudaError_t launch_bwd_coef(const Dims& d, int slot, int T, const float* red, int nslice,
                            const float* zact, const float* rs, const float* p,
                            const float* hpost, const double* gram, const float* alpha_post,
                            const float* b_post, const float* alpha_res, const float* b_res,
                            float* tokmat, float* dz, float* dp, float* tokgrad, cudaStream_t st);
cudaError_t launch_gemm_dzw(const Dims& d, int T, const float* dz, int ldz, int n,
                            const WSegs& W, int E, float* dxact, cudaStream_t st);
cudaError_t launch_conv_wgrad_reduce(const Dims& d, int slot, const float* cpart, int ntiles,
                                     ConvGradPtrs gconv, cudaStream_t st);
cudaError_t launch_wgrad(const uint16_t* A, int64_t lda, int E, int T, const float* dz, int ldz,
                         int n, int tsplits, float* wpart, const WSegsOut& G, cudaStream_t st);
cudaError_t launch_dinput_act(const Dims& d, int slot, int T, int add_dx, const uint16_t* d_input,
                              const uint16_t* xact, const float* hpre, const int* I,
                              float* dxact, float* dhpre, uint16_t* dinput_copy,
                              const float* tokmat, cudaStream_t st);
cudaError_t launch_full_dots(const Dims& d, int T, const uint16_t* X, const uint16_t* dinput,
                             const int* I, float* dhpre, cudaStream_t st);
cudaError_t launch_full_coef(const Dims& d, int T, const float* dhpre, const float* hpre,
                             const float* zfull, const float* stats, const float* wsum,
                             const int* I, const float* dp, const float* alpha_pre, float* dz,
                             float* tokgrad, cudaStream_t st);
cudaError_t launch_full_dx(const Dims& d, int T, const float* dz, const WSegs& W,
                           const uint16_t* X, const uint16_t* dinput, const float* hpre,
                           const int* I, const float* dxact, const float* tokgrad_scal,
                           uint16_t* dX, cudaStream_t st);

}  // namespace xhc
