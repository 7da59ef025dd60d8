/*
 * libxhc -- the expanded-residual connection op of xHC / xHC-Flash / mHC
 * (arXiv 2607.14530, "xHC: Expanded Hyper-Connections") as a C ABI over CUDA kernels for
 * sm_103a (GB300).
 *
 * One "group" is G consecutive sublayers (slots) that share one routing decision and one
 * full-state mapping generation:
 *   G = 1  full xHC sublayer (Alg. 1) or mHC sublayer (Sec. 3.1, k = m = N);
 *   G = 2  xHC-Flash block (Alg. 2, slots Attention, MLP);
 *   G = 4  xHC-Flash-4sub group (Sec. 5.2 and App. E.2, slots A, M, A, M).
 * Per group the caller runs, in order,
 *   forward :  pre_fwd(0) F_0 post_fwd(0)  pre_fwd(1) F_1 post_fwd(1) ... post_fwd(G-1)
 *   backward:  post_bwd(G-1) F_{G-1}' pre_bwd(G-1) ... post_bwd(0) F_0' pre_bwd(0)
 * where F_t is the caller's sublayer (Attention / MLP) and F_t' its backward.
 *
 * Tensor layouts (row-major, contiguous):
 *   X, dX        [T, N, C] bf16 residual state / its gradient; token t = b*S + s
 *                (sequence-major, S = seq_len), stream i, channel c at (t*N + i)*C + c.
 *   input        [T, C] bf16 sublayer input written by pre_fwd (Eq. dense_read).
 *   out          [T, C] bf16 sublayer output read by post_fwd / post_bwd.
 *   d_input      [T, C] bf16 gradient w.r.t. input (read by pre_bwd).
 *   d_out        [T, C] bf16 gradient w.r.t. out (written by post_bwd).
 *   parameters   fp32, shapes in xhc_params; gradients fp32 with the same shapes.
 * bf16 values are passed as their 16-bit patterns (uint16_t).
 *
 * Ownership and execution: every buffer is allocated and owned by the caller (device memory
 * unless stated).  The library allocates no device memory, never synchronises, and enqueues
 * all work asynchronously on the caller's stream (a cudaStream_t passed as void*; NULL = the
 * legacy default stream).  post_bwd and pre_bwd(0) run their weight-gradient and column-sum
 * kernels on an internal stream of the device (created on first use, one per device), forked
 * from the caller's stream with an event after the work they depend on and joined back into
 * it with an event before the call returns: to the caller every call stays ordered on its
 * stream.  `saved` (xhc_saved_bytes) carries the group's forward state to its
 * backward and must not be touched in between; `workspace` (xhc_workspace_bytes) is scratch that
 * must stay the same buffer across the calls of one group's forward and across those of its
 * backward, and may be reused by other groups between those phases.  Two groups in flight on
 * different streams need separate saved and workspace buffers.
 *
 * State is updated in place: post_fwd(G-1) overwrites the k active rows of X (Eq.
 * sparse_write, inactive rows untouched); post_bwd(G-1) restores them from `saved`, so after the
 * backward call sequence X holds the group-entry state again.  dX is updated in place from the
 * gradient w.r.t. the group's output state to the gradient w.r.t. its entry state.  Parameter
 * gradients are ACCUMULATED (+=) in fp32 with a fixed reduction order (run-to-run
 * deterministic, no float atomics).
 *
 * Errors: every entry point validates its arguments on the host before enqueueing anything and
 * returns a status; no exception crosses the ABI.  Requirements: device pointers 16-byte
 * aligned; C % 8 == 0 and 8 <= C <= 16384; 1 <= N <= 32; 1 <= k <= 8; 0 <= m <= k <= N;
 * T % seq_len == 0.  A launch failure returns XHC_ERR_CUDA; xhc_last_error_string() gives the
 * CUDA message of the most recent failure on the calling thread.
 */
#ifndef XHC_H
#define XHC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    XHC_OK = 0,
    XHC_ERR_INVALID_ARG = 1, /* null pointer, bad slot, T or config field out of range     */
    XHC_ERR_UNSUPPORTED = 2, /* valid per the paper but outside the limits listed above     */
    XHC_ERR_ALIGNMENT = 3,   /* a pointer is not 16-byte aligned                            */
    XHC_ERR_CUDA = 4,        /* a CUDA launch or query failed                               */
    XHC_ERR_TIMEOUT = 5      /* a bounded device-side wait gave up (xhc_workspace_error)    */
} xhc_status;

typedef enum {
    XHC_MHC = 0,   /* mHC (Sec. 3.1): k = m = N, no router, G = 1, single write-back signal */
    XHC_FULL = 1,  /* full xHC sublayer (Alg. 1), G = 1                                    */
    XHC_FLASH = 2  /* xHC-Flash group (Alg. 2, App. E.2), G = 2 or 4                        */
} xhc_variant;

#define XHC_MAX_GROUP 4
#define XHC_MAX_CONV 3

/* Immutable after xhc_create.  Hyper-parameters of Sec. 3.3 / App. A. */
typedef struct {
    int variant;               /* xhc_variant                                                */
    int N;                     /* streams (expansion rate)                                   */
    int k;                     /* active streams per sublayer                                */
    int m;                     /* fixed streams (always active, p = 1), Eq. router_topk      */
    int C;                     /* hidden size                                                */
    int group;                 /* G: sublayers sharing the routing decision                  */
    int mlp_mask;              /* bit t set: slot t is an MLP sublayer (temporal augmentation)*/
    int n_conv;                /* r causal depthwise conv branches (0 = none), Eq. aug        */
    int conv_k[XHC_MAX_CONV];  /* kernel sizes kappa_j (paper: 4, 8, 12), each 1..16          */
    int gram_schmidt;          /* 1: Eq. gs on [out, g_1..g_r]; 0: raw components            */
    int sinkhorn_iters;        /* 20 in App. A                                                */
    float eps_norm;            /* LayerNorm / RMSNorm epsilon (1e-5)                          */
    float eps_gs;              /* Gram-Schmidt denominator epsilon; <= 0 means 1e-6 * C        */
    int seq_len;               /* S: the conv never crosses a sequence start; 0 means T       */
    int router;                /* 0: sigmoid scores (Eq. router); 1: softmax over the N       */
                               /*    logits (the softmax-router ablation, Table ablation (11)) */
    int sparse_read;           /* 0: dense read of all N streams (Eq. dense_read); 1: read     */
                               /*    only the k active streams (Table ablation (6), (7))      */
} xhc_config;

/* Device pointers to the fp32 parameters of one group (Sec. 3.3.4, Sec. 5.2).
 *   W_r        [N*C, N]      router projection (Eq. router); NULL when m == k
 *   W_pre[t]   [N*C, N]      pre-map projection of slot t (Eq. param_pre)
 *   alpha_pre  [G]           gating scalars of the pre-maps;  b_pre [G, N] biases
 *   W_post[t]  [k*C, k*K_t]  post-map projection of slot t (Eq. param_post), K_t = 1 + r for
 *                            MLP slots with augmentation, 1 otherwise
 *   alpha_post [G];  b_post[t] [k*K_t]
 *   W_res      [k*C, k*k]    residual-map projection of the last slot (Eq. param_res)
 *   alpha_res  [1];  b_res [k*k]
 *   conv_w[t][j] [kappa_j, C] depthwise taps of branch j of MLP slot t; tap 0 = current token
 * Row index of every W is the flattened (stream-major) state index i*C + c; mat_{a x b} of a
 * projection is row-major (column j*b + r is entry [j][r]). */
typedef struct {
    const float* W_r;
    const float* W_pre[XHC_MAX_GROUP];
    const float* alpha_pre;
    const float* b_pre;
    const float* W_post[XHC_MAX_GROUP];
    const float* alpha_post;
    const float* b_post[XHC_MAX_GROUP];
    const float* W_res;
    const float* alpha_res;
    const float* b_res;
    const float* conv_w[XHC_MAX_GROUP][XHC_MAX_CONV];
} xhc_params;

/* Gradient buffers, same shapes as xhc_params; every field is accumulated (+=).  A NULL field
 * is an error if the parameter exists in the configuration. */
typedef struct {
    float* W_r;
    float* W_pre[XHC_MAX_GROUP];
    float* alpha_pre;
    float* b_pre;
    float* W_post[XHC_MAX_GROUP];
    float* alpha_post;
    float* b_post[XHC_MAX_GROUP];
    float* W_res;
    float* alpha_res;
    float* b_res;
    float* conv_w[XHC_MAX_GROUP][XHC_MAX_CONV];
} xhc_grads;

typedef struct xhc_handle xhc_handle;

/* Validate *cfg and create a handle (host memory only).  XHC_ERR_INVALID_ARG for values the
 * paper's method cannot take (e.g. m > k), XHC_ERR_UNSUPPORTED for values beyond the limits
 * above, or for a variant whose structure does not match (MHC needs k = m = N, G = 1, no MLP
 * augmentation; FULL needs G = 1; FLASH needs G in {2, 4} with slots alternating A, M: the MLP
 * slots' bits set in mlp_mask, the attention slots' bits optional -- set, they give the
 * attention-side temporal augmentation of App. "Additional Ablation Studies"). */
xhc_status xhc_create(const xhc_config* cfg, xhc_handle** out);
void xhc_destroy(xhc_handle* h);

/* Bytes of the caller-allocated `saved` and `workspace` buffers for T tokens. */
xhc_status xhc_saved_bytes(const xhc_handle* h, int64_t T, size_t* bytes);
xhc_status xhc_workspace_bytes(const xhc_handle* h, int64_t T, size_t* bytes);

/* Byte offsets, inside `saved`, of the coefficients a forward pass leaves there (for inspection
 * and tests; the content is defined once pre_fwd(slot) has run for the slot concerned):
 *   I        int32 [T, k]        active stream indices, fixed streams first (Eq. router_topk)
 *   p        fp32  [T, k]        routing weights (1 for fixed streams)
 *   hpre     fp32  [T, G, N]     pre-maps of the G slots (Eq. param_pre)
 *   hpost[t] fp32  [T, k, K_t]   post-map of slot t (Eq. param_post)
 *   hres     fp32  [T, k, k]     clamped Sinkhorn residual map of the last slot (Eq. param_res)
 *   xact     bf16  [G, T, k, C]  active state entering each slot
 *   zfull    fp32  [T, nfull]     raw full-state projections x W, columns [router N | pre-map
 *                                 N of each slot] (router columns only when m < k)
 *   stats    fp32  [T, 2]         mean and mean square of the flattened entry state */
typedef struct {
    size_t I;
    size_t p;
    size_t hpre;
    size_t hpost[XHC_MAX_GROUP];
    size_t hres;
    size_t xact;
    size_t zfull;
    size_t stats;
} xhc_saved_layout;
xhc_status xhc_saved_layout_of(const xhc_handle* h, int64_t T, xhc_saved_layout* out);

/* Forward, before sublayer `slot`: writes input [T, C].
 * slot 0 runs the group's full-state passes: norm statistics, the projections of Eq.
 * fused_normalized_projection (router and the G pre-maps), Eq. router_topk, the dense read of
 * Eq. dense_read, the non-active base readouts of Eq. app_four_sub_base and the gather of the
 * active streams; slot t > 0 forms input = base_t + sum_j H_pre_t[I_j] x_act_j (Eq.
 * app_active_state_correction).  Every slot then generates its post-map (and, for the last
 * slot, the Sinkhorn residual map with the App. A row clamp) from the current active state
 * (Eq. param_post, Eq. param_res). */
xhc_status xhc_pre_fwd(const xhc_handle* h, int slot, int64_t T, const xhc_params* P,
                       const uint16_t* X, uint16_t* input, void* saved, void* workspace,
                       void* stream);

/* Forward, after sublayer `slot`: sparse write-back of out (Eq. sparse_write_delta,
 * Eq. sparse_write; temporal augmentation Eq. aug + Eq. gs on MLP slots).  Slots before the
 * last update the saved active state only (no mixing, Eq. flash_attn_update); the last slot
 * applies H_res and scatters the k active rows into X in place. */
xhc_status xhc_post_fwd(const xhc_handle* h, int slot, int64_t T, const xhc_params* P,
                        uint16_t* X, const uint16_t* out, void* saved, void* workspace,
                        void* stream);

/* Decoding: one new token per sequence.
 *
 * The op is token-parallel except for the causal conv of the MLP slots (Eq. aug, Sec. 3.3.4),
 * which reads the R = max(kappa) - 1 previous `out` rows of the token's sequence.  For decoding
 * those rows live in a per-sequence ring owned by the caller, one per conv slot: ring [B][R][C]
 * bf16, row (s mod R) holding out[s] of position s.  pos [B] int64 (device) is the position of
 * each sequence's current token.  A decode step of a group is, for slot = 0..G-1,
 * xhc_pre_fwd(slot, T = B) then xhc_post_fwd_decode(slot, B); use a handle whose seq_len is 0
 * (or divides B): the conv history comes from the ring, not from the call's tokens.
 *
 * xhc_ring_bytes: size of one conv slot's ring for B sequences (0 without a conv).
 * xhc_ring_fill: after a prefill of B sequences of S tokens each (rows b*S .. b*S+S-1 of `out`,
 *   the slot's sublayer output), stores each sequence's last min(S, R) rows in its ring; the
 *   caller then sets pos[b] = S.  Rows the conv will not read are left as they are.
 * xhc_post_fwd_decode: xhc_post_fwd for B tokens, token b at position pos[b] of sequence b, with
 *   the conv history read from `ring` (null for a slot without a conv); afterwards the token's
 *   out row is stored in its ring row, and the group's last slot advances pos by one.  Same
 *   saved / workspace contract as xhc_post_fwd with T = B.  Errors: XHC_ERR_INVALID_ARG for a
 *   null ring on a conv slot, null pos, B <= 0; XHC_ERR_ALIGNMENT for pointers not 16-byte
 *   aligned. */
xhc_status xhc_ring_bytes(const xhc_handle* h, int64_t B, size_t* bytes);
xhc_status xhc_ring_fill(const xhc_handle* h, int64_t B, int64_t S, const uint16_t* out, void* ring,
                         void* stream);
xhc_status xhc_post_fwd_decode(const xhc_handle* h, int slot, int64_t B, const xhc_params* P,
                               uint16_t* X, const uint16_t* out, void* ring, int64_t* pos,
                               void* saved, void* workspace, void* stream);

/* Backward of post_fwd(slot).  Reads dX (slot G-1: the gradient w.r.t. the group output) or the
 * workspace-held active gradient, leaves the post/res map-logit gradient in the workspace for
 * pre_bwd(slot), writes d_out [T, C] (= dL/d out, including the paths through
 * later sublayer inputs), accumulates the post/res/conv parameter gradients.  slot G-1 also
 * restores the active rows of X to the group-entry state. */
xhc_status xhc_post_bwd(const xhc_handle* h, int slot, int64_t T, const xhc_params* P,
                        uint16_t* X, uint16_t* dX, const uint16_t* out, uint16_t* d_out,
                        const xhc_grads* grads, void* saved, void* workspace, void* stream);

/* Backward of pre_fwd(slot).  Adds the dense-read gradient of d_input and the gradient through
 * the post/res map projections of this slot to the active gradient (the map-logit gradient is
 * left in the workspace by post_bwd(slot), so the calls of one slot run back to back on the same
 * workspace; P needs W_post[slot], and W_res at the last slot, on every slot); slot 0 finishes
 * the group: dX becomes the gradient w.r.t. the entry state (dense reads,
 * norm statistics, router through the selected routed scores only) and the W_r / W_pre /
 * alpha_pre / b_pre gradients are accumulated. */
xhc_status xhc_pre_bwd(const xhc_handle* h, int slot, int64_t T, const xhc_params* P,
                       const uint16_t* X, const uint16_t* d_input, uint16_t* dX,
                       const xhc_grads* grads, void* saved, void* workspace, void* stream);

/* Sequence split (context parallelism, chunked prefill).
 *
 * A sequence may be cut into consecutive chunks that are processed by separate calls (on separate
 * GPUs, or one after the other).  Every step of the op is token-local except the causal conv of
 * the temporal augmentation (conv formula of Sec. 3.3.4), which reads the R = max(kappa) - 1
 * sublayer outputs before each token; for the first tokens of a chunk those belong to the previous
 * chunk.  They travel as a halo: [B][R][C] bf16 per conv slot, row r of sequence b holding `out`
 * at position r - R relative to the chunk's first token (zero rows where that position is before
 * the sequence start; B = T / seq_len sequences in the call, each a chunk).
 *
 * xhc_halo_bytes: bytes of one slot's halo for B sequences (0 without a conv); its gradient
 *   d_halo is the same shape in fp32 (twice the bytes).
 * xhc_halo_fill: from a chunk's sublayer output `out` (B sequences of S tokens), the halo the
 *   next chunk needs: halo[b][r] = out[b*S + S - R + r] (zero where S - R + r < 0).
 * xhc_post_fwd_halo: xhc_post_fwd with the conv history of every sequence's first tokens read
 *   from `halo` (null = a sequence start; ignored on slots without a conv).
 * xhc_post_bwd_halo: xhc_post_bwd of such a call; the conv weight gradient includes the halo's
 *   terms, and d_halo [B][R][C] fp32 (required with a halo on a conv slot, else
 *   XHC_ERR_INVALID_ARG) receives the gradient w.r.t. the halo rows, which belongs to the
 *   previous chunk's d_out.
 * xhc_halo_add: on the previous chunk, d_out[b*S + S - R + r] += d_halo[b][r] (the sum rounded
 *   once to bf16); run after its own xhc_post_bwd(slot), before its sublayer's backward.
 * The parameter gradients of the chunks add up (accumulate into the same buffers, or all-reduce
 * them across the GPUs that hold the chunks).  Same ownership and error rules as above. */
xhc_status xhc_halo_bytes(const xhc_handle* h, int64_t B, size_t* bytes);
xhc_status xhc_halo_fill(const xhc_handle* h, int64_t B, int64_t S, const uint16_t* out, void* halo,
                         void* stream);
xhc_status xhc_post_fwd_halo(const xhc_handle* h, int slot, int64_t T, const xhc_params* P,
                             uint16_t* X, const uint16_t* out, const uint16_t* halo, void* saved,
                             void* workspace, void* stream);
xhc_status xhc_post_bwd_halo(const xhc_handle* h, int slot, int64_t T, const xhc_params* P,
                             uint16_t* X, uint16_t* dX, const uint16_t* out, uint16_t* d_out,
                             const xhc_grads* grads, const uint16_t* halo, float* d_halo,
                             void* saved, void* workspace, void* stream);
xhc_status xhc_halo_add(const xhc_handle* h, int64_t B, int64_t S, uint16_t* d_out,
                        const float* d_halo, void* stream);

/* Model glue around a stack of groups (App. A, "Final Stream Reduction"):
 * xhc_stream_expand: X[t][i] = hidden[t] for the N streams of every token ([T, C] -> [T, N, C]
 *   bf16): the expanded state entering the first group (the paper does not state the
 *   initialisation; N copies of the embedding output is the HC convention).  It is also the
 *   backward of xhc_stream_sum (the gradient of a sum reaches every term).
 * xhc_stream_sum: y[t] = sum_i X[t][i] ([T, N, C] -> [T, C], fp32 sum, bf16 store): the N
 *   streams reduced to one hidden vector before the final RMSNorm and unembedding.  It is also
 *   the backward of xhc_stream_expand.
 * N and C come from the handle; same ownership and error rules as above. */
xhc_status xhc_stream_expand(const xhc_handle* h, int64_t T, const uint16_t* hidden, uint16_t* X,
                             void* stream);
xhc_status xhc_stream_sum(const xhc_handle* h, int64_t T, const uint16_t* X, uint16_t* y, void* stream);

/* Routing and pre-maps for callers that cannot allocate device memory.
 *
 * The paper has no counterpart: this is a deployment convenience.  Some callers cannot provide
 * the `workspace` of xhc_pre_fwd -- code running inside another framework's memory arena,
 * engines that fix every device buffer at start-up, plug-ins whose host owns all allocation.
 * xhc_route_noalloc computes, for T tokens of X, the same routing and pre-maps as the
 * full-state part of xhc_pre_fwd(slot 0): I [T, k] int32, p [T, k] fp32 and hpre [T, G, N]
 * fp32 (caller-owned device outputs; P needs W_r (if m < k), W_pre, alpha_pre and b_pre).  Its
 * split-K partial sums live in a fixed array of XHC_NOALLOC_SCRATCH_BYTES that is part of the
 * library's device image (every GPU that loads the library holds it until the process exits);
 * it calls no allocator.  A T whose partial sums do not fit returns XHC_ERR_UNSUPPORTED
 * (for N = 16, G = 4 and T above ~20K tokens about 1 KB per token, so T up to ~50K).
 * The first call on a device looks up the array's device address (cudaGetSymbolAddress) with
 * that device current; make that first call before any stream capture.  All calls share the one
 * array: calls that overlap on the GPU (several streams or host threads at once) race and give
 * wrong results; serialise them.  Nothing in the array needs to start at zero: each call writes
 * every word it later reads. */
#define XHC_NOALLOC_SCRATCH_BYTES (48u << 20)
xhc_status xhc_route_noalloc(const xhc_handle* h, int64_t T, const xhc_params* P,
                             const uint16_t* X, int32_t* I, float* p, float* hpre, void* stream);

/* Tracing, a host-side profiling aid: while enabled, every kernel launch of the library is
 * bracketed by two CUDA events recorded on the stream it runs on.  xhc_trace_enable(1) drops the
 * previous records and starts recording; xhc_trace_enable(0) stops.  xhc_trace_only restricts
 * the recording to the launches of the named kernels (a comma-separated list of the names the
 * records carry, e.g. "dxa_tc,dinput_act"; NULL or "" records every launch again); it takes
 * effect for later launches and is kept until the next xhc_trace_only.  xhc_trace_record gives
 * record i's name and device duration in ms; xhc_trace_span also gives its start in ms after
 * the start of record 0 (a timeline across the library's streams).  The caller must have
 * synchronised the streams first (otherwise XHC_ERR_CUDA, "not ready"); i out of range or a
 * NULL output pointer is XHC_ERR_INVALID_ARG.  Not for concurrent use from several host
 * threads. */
xhc_status xhc_trace_enable(int on);
xhc_status xhc_trace_only(const char* names);
int xhc_trace_count(void);
xhc_status xhc_trace_record(int i, const char** name, float* ms);
xhc_status xhc_trace_span(int i, const char** name, float* start_ms, float* ms);

/* Device error word of a workspace: kernels with bounded waits (the tensor-core kernels) set it
 * to a nonzero code instead of waiting forever, and return; a launch whose wait gave up leaves
 * its outputs undefined, and the CUDA context stays usable.  Synchronous (a device-to-host copy).
 * *code receives the word (the number of the wait that gave up); returns XHC_ERR_TIMEOUT if it is
 * nonzero; clear != 0 resets it.  A fresh workspace must be zeroed once before first use (e.g.
 * cudaMemset). */
xhc_status xhc_workspace_error(const void* workspace, int* code, int clear);

/* Test hooks for the bounded waits (process-wide, host side; not for production use).
 * XHC_DEBUG_WAIT_LIMIT_NS: the limit of every bounded device wait of later launches, in ns
 *   (0 = the default of about 4 s).
 * XHC_DEBUG_FORCE_TIMEOUT: value != 0 makes the next full-state projection launch (xhc_pre_fwd
 *   of slot 0 on the tensor cores) wait, before it issues any copy or MMA, for a release that
 *   nothing triggers, so that every wait of that launch runs out: it sets the workspace's error
 *   word and returns without touching its outputs.  One-shot.
 * XHC_DEBUG_ONE_STREAM: value != 0 runs the work that later calls put on the library's side
 *   stream (weight gradients, column sums, dH_pre dots) on the caller's stream instead, in the
 *   same order; the results are the same.  0 restores the side stream.
 * Returns XHC_ERR_INVALID_ARG for an unknown `what` or a negative limit. */
#define XHC_DEBUG_WAIT_LIMIT_NS 1
#define XHC_DEBUG_FORCE_TIMEOUT 2
#define XHC_DEBUG_ONE_STREAM 3
xhc_status xhc_debug_set(int what, int64_t value);

/* Number of kernels the library has launched since it was loaded. */
uint64_t xhc_launch_count(void);

/* Short static description of a status; message of the last CUDA failure on this thread. */
const char* xhc_status_string(xhc_status s);
const char* xhc_last_error_string(void);

/* Library version as major*10000 + minor*100 + patch. */
int xhc_version(void);

#ifdef __cplusplus
}
#endif
#endif /* XHC_H */
