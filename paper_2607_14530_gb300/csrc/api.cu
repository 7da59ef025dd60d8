// libxhc C ABI: validation, buffer layout and the launch sequence of each entry point.
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <mutex>
#include <string>
#include <vector>

#include "xhc_internal.cuh"

namespace xhc {

// ---- launch accounting and tracing ----------------------------------------------------------
static std::atomic<unsigned long long> g_launches{0};
void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

// ---- test hooks -----------------------------------------------------------------------------
static std::atomic<unsigned long long> g_wait_ns{0};   // 0: the default limit (~4 s)
static std::atomic<int> g_force_timeout{0};
static std::atomic<int> g_one_stream{0};
uint64_t debug_wait_ns() {
    const unsigned long long v = g_wait_ns.load();
    return v ? (uint64_t)v : 4000000000ull;
}
int debug_take_force_timeout() { return g_force_timeout.exchange(0); }

struct TraceRec {
    const char* name;
    cudaEvent_t a, b;
};
static std::mutex g_tmu;
static bool g_trace_on = false;
static std::vector<TraceRec> g_recs;
static std::vector<cudaEvent_t> g_pool;
static std::vector<std::string> g_only;   // names recorded while tracing (empty: every launch)

static bool traced(const char* n) {
    if (g_only.empty()) return true;
    for (const auto& s : g_only)
        if (s == n) return true;
    return false;
}

static cudaEvent_t take_event() {
    cudaEvent_t e = nullptr;
    if (!g_pool.empty()) {
        e = g_pool.back();
        g_pool.pop_back();
    } else if (cudaEventCreate(&e) != cudaSuccess) {
        e = nullptr;
    }
    return e;
}

struct TraceScope {
    const char* name;
    cudaStream_t st;
    cudaEvent_t a = nullptr;
    TraceScope(const char* n, cudaStream_t s) : name(n), st(s) {
        if (!g_trace_on) return;
        std::lock_guard<std::mutex> lk(g_tmu);
        if (!traced(n)) return;
        a = take_event();
        if (a) cudaEventRecord(a, st);
    }
    void done() {
        if (!a) return;
        std::lock_guard<std::mutex> lk(g_tmu);
        cudaEvent_t b = take_event();
        if (!b) return;
        cudaEventRecord(b, st);
        g_recs.push_back({name, a, b});
    }
};

static thread_local char g_last_error[256] = "";

static xhc_status cuda_fail(cudaError_t e, int line) {
    (void)cudaGetLastError();  // do not leave a launch-configuration error for the caller's next call
    snprintf(g_last_error, sizeof(g_last_error), "api.cu:%d: %s", line, cudaGetErrorString(e));
    return XHC_ERR_CUDA;
}

#define XHC_CUDA(call)                                         \
    do {                                                       \
        cudaError_t e_ = (call);                               \
        if (e_ != cudaSuccess) return cuda_fail(e_, __LINE__); \
    } while (0)

// a library launch, bracketed by trace events when tracing is on
#define XHC_K(name, stream, call)                              \
    do {                                                       \
        TraceScope ts_(name, stream);                          \
        cudaError_t e_ = (call);                               \
        if (e_ != cudaSuccess) return cuda_fail(e_, __LINE__); \
        ts_.done();                                            \
    } while (0)

static size_t al(size_t x) { return (x + 255) & ~(size_t)255; }

Dims make_dims(const xhc_config& c) {
    Dims d;
    memset(&d, 0, sizeof(d));
    d.N = c.N;
    d.k = c.k;
    d.m = c.m;
    d.C = c.C;
    d.G = c.group;
    d.hr = (c.m < c.k) ? 1 : 0;
    d.nfull = (d.hr ? d.N : 0) + d.G * d.N;
    d.S = c.seq_len;
    d.iters = c.sinkhorn_iters;
    d.eps = c.eps_norm;
    d.eps_gs = (c.eps_gs > 0.f) ? c.eps_gs : 1e-6f * (float)c.C;
    d.gs = c.gram_schmidt ? 1 : 0;
    d.nconv = c.n_conv;
    d.kapmax = 0;
    d.kapsum = 0;
    for (int j = 0; j < 3; ++j) {
        d.kap[j] = (j < c.n_conv) ? c.conv_k[j] : 0;
        d.kapmax = std::max(d.kapmax, d.kap[j]);
        d.kapsum += d.kap[j];
    }
    d.softmax = c.router == 1 ? 1 : 0;
    d.dense = c.sparse_read ? 0 : 1;
    for (int t = 0; t < 4; ++t) {
        const bool mlp = (t < d.G) && ((c.mlp_mask >> t) & 1) && c.n_conv > 0;
        d.K[t] = mlp ? 1 + c.n_conv : 1;
        d.nact[t] = (t < d.G) ? d.k * d.K[t] + (t == d.G - 1 ? d.k * d.k : 0) : 0;
    }
    return d;
}

static int pick_splits(int rowblocks, int K) {
    int s = (608 + rowblocks - 1) / rowblocks;
    s = std::min(s, std::max(1, K / 256));
    return std::max(1, s);
}

static int pick_tsplits(int E, int T) {
    const int eb = (E + 63) / 64;
    int s = (608 + eb - 1) / eb;
    s = std::min(s, std::max(1, (T + 63) / 64));
    return std::max(1, s);
}

Layout make_layout(const Dims& d, int64_t T) {
    Layout L;
    memset(&L, 0, sizeof(L));
    const size_t t = (size_t)T;
    int nact_max = 0;
    for (int q = 0; q < d.G; ++q) {
        nact_max = std::max(nact_max, d.nact[q]);
    }
    size_t o = 0;
    L.xact = o; o = al(o + (size_t)d.G * t * d.k * d.C * 2);
    L.I = o; o = al(o + t * d.k * 4);
    L.p = o; o = al(o + t * d.k * 4);
    L.stats = o; o = al(o + t * 2 * 4);
    L.zfull = o; o = al(o + t * d.nfull * 4);
    L.hpre = o; o = al(o + t * d.G * d.N * 4);
    for (int q = 0; q < d.G; ++q) {
        L.zact[q] = o; o = al(o + t * d.nact[q] * 4);
        L.rs[q] = o; o = al(o + t * 4);
        L.hpost[q] = o; o = al(o + t * d.k * d.K[q] * 4);
    }
    L.hres = o; o = al(o + t * d.k * d.k * 4);
    for (int q = 0; q < d.G; ++q)
        if (d.K[q] > 1 && d.gs) { L.gram[q] = o; o = al(o + t * NGRAM * 8); }
    L.saved_total = o;

    const int rowblocks = (int)((T + 63) / 64);
    const int sms = device_sms();
    L.tc = plan_proj_tc((int)T, d.N * d.C, d.nfull, sms, true);
    L.tca = plan_proj_tc((int)T, d.k * d.C, nact_max, sms, true);
    L.twf = plan_proj_tc(d.N * d.C, (int)T, d.nfull, sms, false);
    L.twa = plan_proj_tc(d.k * d.C, (int)T, nact_max, sms, false);
    L.splits_full = std::max(L.tc.nseg, pick_splits(rowblocks, d.N * d.C));
    L.splits_act = std::max(L.tca.nseg, pick_splits(rowblocks, d.k * d.C));
    L.nslice = wb_nslice(d.C);
    const int ts_full = pick_tsplits(d.N * d.C, (int)T);
    const int ts_act = pick_tsplits(d.k * d.C, (int)T);
    L.tsplits = std::max(ts_full, ts_act);
    {
        L.ntiles = d.nconv > 0 ? wb_conv_runs(d, T) : 1;
    }
    o = 0;
    L.err = o; o = al(o + 256);
    L.wpack = o;
    o = al(o + std::max((size_t)L.tc.NB * d.N * d.C, (size_t)L.tca.NB * d.k * d.C) * 2);
    L.dzpack = o; o = al(o + (size_t)std::max(L.twf.NB, L.twa.NB) * ((t + 7) / 8 * 8) * 2);
    {
        // bf16 operands of the tensor-core input gradients: full maps [T][nfull] and [N C][nfull],
        // active maps in three parts [T][3 nact] and [k C][3 nact] (rows padded to 8)
        const size_t ld = (size_t)(d.nfull + 7) / 8 * 8;
        const size_t ld3 = (size_t)(3 * nact_max + 7) / 8 * 8;
        L.dz16 = o; o = al(o + t * std::max(ld, ld3) * 2);
        L.w16 = o; o = al(o + std::max((size_t)d.N * d.C * ld, (size_t)d.k * d.C * ld3) * 2);
    }
    L.part = o;
    o = al(o + std::max((size_t)L.splits_full * d.nfull, (size_t)L.splits_act * nact_max) * t * 4);
    L.pstats = o; o = al(o + (size_t)std::max(L.splits_full, L.splits_act) * t * 2 * 4);
    L.astat = o; o = al(o + (size_t)stream_warps(d.C) * t * 2 * 4);
    L.wsum = o; o = al(o + (size_t)d.N * 4);
    L.rsum = o; o = al(o + (size_t)d.N * 4);
    L.base = o; o = al(o + (size_t)(d.G - 1) * t * d.C * 2);
    L.red = o; o = al(o + t * L.nslice * NRED * 4);
    L.dxact = o; o = al(o + t * d.k * d.C * 4);
    L.dinput = o; o = al(o + (size_t)d.G * t * d.C * 2);
    L.dotp = o; o = al(o + (size_t)d.k * (d.C / 32) * t * 4);
    L.dp = o; o = al(o + t * d.k * 4);
    L.dhpre = o; o = al(o + t * d.G * d.N * 4);
    L.tokmat = o; o = al(o + t * TOKMAT * 4);
    L.dz = o; o = al(o + t * std::max(d.nfull, nact_max) * 4);
    L.tokgrad = o; o = al(o + t * NTG * 4);
    L.wpart = o;
    {
        size_t w1 = std::max((size_t)ts_full * d.N * d.C * d.nfull, (size_t)ts_act * d.k * d.C * nact_max);
        size_t w2 = std::max((size_t)L.twf.nseg * d.N * d.C * d.nfull, (size_t)L.twa.nseg * d.k * d.C * nact_max);
        o = al(o + std::max(w1, w2) * 4);
    }
    L.cpart = o; o = al(o + (size_t)L.ntiles * d.kapsum * d.C * 4);
    L.colscr = o; o = al(o + (size_t)64 * 256 * 4);
    L.ws_total = o;
    return L;
}

}  // namespace xhc

using namespace xhc;

static bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

extern "C" {

int xhc_version(void) { return 200; }

xhc_status xhc_trace_enable(int on) {
    std::lock_guard<std::mutex> lk(g_tmu);
    if (on) {
        for (auto& r : g_recs) {
            g_pool.push_back(r.a);
            g_pool.push_back(r.b);
        }
        g_recs.clear();
    }
    g_trace_on = (on != 0);
    return XHC_OK;
}

xhc_status xhc_trace_only(const char* names) {
    std::lock_guard<std::mutex> lk(g_tmu);
    g_only.clear();
    if (!names) return XHC_OK;
    std::string cur;
    for (const char* c = names;; ++c) {
        if (*c == ',' || *c == 0) {
            if (!cur.empty()) g_only.push_back(cur);
            cur.clear();
            if (*c == 0) break;
        } else if (*c != ' ') {
            cur.push_back(*c);
        }
    }
    return XHC_OK;
}

int xhc_trace_count(void) {
    std::lock_guard<std::mutex> lk(g_tmu);
    return (int)g_recs.size();
}

xhc_status xhc_trace_record(int i, const char** name, float* ms) {
    std::lock_guard<std::mutex> lk(g_tmu);
    if (i < 0 || i >= (int)g_recs.size() || !name || !ms) return XHC_ERR_INVALID_ARG;
    *name = g_recs[i].name;
    cudaError_t e = cudaEventElapsedTime(ms, g_recs[i].a, g_recs[i].b);
    if (e != cudaSuccess) return cuda_fail(e, __LINE__);
    return XHC_OK;
}

xhc_status xhc_trace_span(int i, const char** name, float* start_ms, float* ms) {
    std::lock_guard<std::mutex> lk(g_tmu);
    if (i < 0 || i >= (int)g_recs.size() || !name || !start_ms || !ms) return XHC_ERR_INVALID_ARG;
    *name = g_recs[i].name;
    cudaError_t e = cudaEventElapsedTime(start_ms, g_recs[0].a, g_recs[i].a);
    if (e == cudaSuccess) e = cudaEventElapsedTime(ms, g_recs[i].a, g_recs[i].b);
    if (e != cudaSuccess) return cuda_fail(e, __LINE__);
    return XHC_OK;
}

uint64_t xhc_launch_count(void) { return (uint64_t)g_launches.load(); }

xhc_status xhc_debug_set(int what, int64_t value) {
    switch (what) {
        case XHC_DEBUG_WAIT_LIMIT_NS:
            if (value < 0) return XHC_ERR_INVALID_ARG;
            g_wait_ns.store((unsigned long long)value);
            return XHC_OK;
        case XHC_DEBUG_FORCE_TIMEOUT:
            g_force_timeout.store(value ? 1 : 0);
            return XHC_OK;
        case XHC_DEBUG_ONE_STREAM:
            g_one_stream.store(value ? 1 : 0);
            return XHC_OK;
    }
    return XHC_ERR_INVALID_ARG;
}

xhc_status xhc_workspace_error(const void* workspace, int* code, int clear) {
    if (!workspace || !code) return XHC_ERR_INVALID_ARG;
    cudaError_t e = cudaMemcpy(code, workspace, sizeof(int), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, __LINE__);
    if (clear) {
        e = cudaMemset(const_cast<void*>(workspace), 0, sizeof(int));
        if (e != cudaSuccess) return cuda_fail(e, __LINE__);
    }
    return *code ? XHC_ERR_TIMEOUT : XHC_OK;
}

const char* xhc_status_string(xhc_status s) {
    switch (s) {
        case XHC_OK: return "ok";
        case XHC_ERR_INVALID_ARG: return "invalid argument";
        case XHC_ERR_UNSUPPORTED: return "unsupported configuration";
        case XHC_ERR_ALIGNMENT: return "pointer not 16-byte aligned";
        case XHC_ERR_CUDA: return "CUDA error";
        case XHC_ERR_TIMEOUT: return "device-side wait timed out";
    }
    return "unknown status";
}

const char* xhc_last_error_string(void) { return g_last_error; }

xhc_status xhc_create(const xhc_config* cfg, xhc_handle** out) {
    if (!cfg || !out) return XHC_ERR_INVALID_ARG;
    *out = nullptr;
    const xhc_config& c = *cfg;
    if (c.N < 1 || c.k < 1 || c.m < 0 || c.m > c.k || c.k > c.N || c.C < 1 || c.group < 1 ||
        c.n_conv < 0 || c.n_conv > XHC_MAX_CONV || c.sinkhorn_iters < 0 || !(c.eps_norm > 0.f) ||
        c.seq_len < 0 || c.variant < XHC_MHC || c.variant > XHC_FLASH || c.router < 0 ||
        c.router > 1 || c.sparse_read < 0 || c.sparse_read > 1)
        return XHC_ERR_INVALID_ARG;
    if (c.group > XHC_MAX_GROUP) return XHC_ERR_UNSUPPORTED;
    if (c.mlp_mask & ~((1 << c.group) - 1)) return XHC_ERR_INVALID_ARG;
    for (int j = 0; j < c.n_conv; ++j)
        if (c.conv_k[j] < 1) return XHC_ERR_INVALID_ARG;
    if (c.N > MAXN || c.k > MAXK || c.C % 8 != 0 || c.C < 8 || c.C > 16384 ||
        c.sinkhorn_iters > 64)
        return XHC_ERR_UNSUPPORTED;
    for (int j = 0; j < c.n_conv; ++j)
        if (c.conv_k[j] > MAXKAP) return XHC_ERR_UNSUPPORTED;
    switch (c.variant) {
        case XHC_MHC:
            if (c.k != c.N || c.m != c.N || c.group != 1 || c.mlp_mask != 0)
                return XHC_ERR_INVALID_ARG;
            break;
        case XHC_FULL:
            if (c.group != 1) return XHC_ERR_INVALID_ARG;
            break;
        case XHC_FLASH: {
            if (c.group != 2 && c.group != 4) return XHC_ERR_INVALID_ARG;
            // slots A, M (, A, M): the MLP slots carry the temporal augmentation; the attention
            // slots may carry it too (the attention-side ablation of App. "Additional Ablation
            // Studies")
            const int want = (c.group == 2) ? 0x2 : 0xA;
            if ((c.mlp_mask & want) != want) return XHC_ERR_INVALID_ARG;
            break;
        }
    }
    xhc_handle* h = new (std::nothrow) xhc_handle;
    if (!h) return XHC_ERR_INVALID_ARG;
    h->h.cfg = c;
    h->h.d = make_dims(c);
    *out = h;
    return XHC_OK;
}

void xhc_destroy(xhc_handle* h) { delete h; }

xhc_status xhc_saved_bytes(const xhc_handle* h, int64_t T, size_t* bytes) {
    if (!h || !bytes || T <= 0) return XHC_ERR_INVALID_ARG;
    *bytes = make_layout(h->h.d, T).saved_total;
    return XHC_OK;
}

xhc_status xhc_workspace_bytes(const xhc_handle* h, int64_t T, size_t* bytes) {
    if (!h || !bytes || T <= 0) return XHC_ERR_INVALID_ARG;
    *bytes = make_layout(h->h.d, T).ws_total;
    return XHC_OK;
}

xhc_status xhc_saved_layout_of(const xhc_handle* h, int64_t T, xhc_saved_layout* out) {
    if (!h || !out || T <= 0) return XHC_ERR_INVALID_ARG;
    const Layout L = make_layout(h->h.d, T);
    memset(out, 0, sizeof(*out));
    out->I = L.I;
    out->p = L.p;
    out->hpre = L.hpre;
    for (int q = 0; q < h->h.d.G; ++q) out->hpost[q] = L.hpost[q];
    out->hres = L.hres;
    out->xact = L.xact;
    out->zfull = L.zfull;
    out->stats = L.stats;
    return XHC_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------------------------

namespace {

// Side stream of a device (created on first use, kept for the life of the process): work of a
// call that does not feed the rest of the call (weight gradients, column sums) runs there,
// forked from and joined back into the caller's stream with events, so it overlaps the
// bandwidth- or latency-bound kernels of the main chain.  Without a side stream everything runs
// on the caller's stream.
static std::mutex g_smu;
static cudaStream_t g_side[64];

static cudaStream_t side_stream() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    std::lock_guard<std::mutex> lk(g_smu);
    if (!g_side[dev]) {
        cudaStream_t st = nullptr;
        if (cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking) != cudaSuccess) {
            cudaGetLastError();
            return nullptr;
        }
        g_side[dev] = st;
    }
    return g_side[dev];
}

// `to` waits for the work enqueued so far on `from` (a fresh event per call: concurrent callers
// never wait on each other's record)
static bool stream_after(cudaStream_t to, cudaStream_t from) {
    cudaEvent_t e;
    if (cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess) return false;
    bool ok = cudaEventRecord(e, from) == cudaSuccess && cudaStreamWaitEvent(to, e, 0) == cudaSuccess;
    cudaEventDestroy(e);
    return ok;
}

// a stream forked from `main`: the side stream, or `main` itself
static cudaStream_t fork_from(cudaStream_t main) {
    if (g_one_stream.load()) return main;
    cudaStream_t side = side_stream();
    if (!side || !stream_after(side, main)) return main;
    return side;
}

static xhc_status join_into(cudaStream_t main, cudaStream_t side) {
    if (side == main) return XHC_OK;
    return stream_after(main, side) ? XHC_OK : XHC_ERR_CUDA;
}

struct Ctx {
    Dims d;
    Layout L;
    int T;
    char* sv;
    char* ws;
    cudaStream_t st;
    template <class P>
    P* S(size_t off) const { return reinterpret_cast<P*>(sv + off); }
    template <class P>
    P* W(size_t off) const { return reinterpret_cast<P*>(ws + off); }
    uint16_t* xact(int slot) const {
        return S<uint16_t>(L.xact) + (size_t)slot * T * d.k * d.C;
    }
};

xhc_status common_check(const xhc_handle* h, int slot, int64_t T, const void* saved,
                        const void* ws, Ctx& cx, void* stream) {
    if (!h || !saved || !ws) return XHC_ERR_INVALID_ARG;
    const Dims& d0 = h->h.d;
    if (slot < 0 || slot >= d0.G || T <= 0 || T > (int64_t)1 << 30) return XHC_ERR_INVALID_ARG;
    const int S = h->h.cfg.seq_len > 0 ? h->h.cfg.seq_len : (int)T;
    if (T % S != 0) return XHC_ERR_INVALID_ARG;
    if (!aligned16(saved) || !aligned16(ws)) return XHC_ERR_ALIGNMENT;
    cx.d = d0;
    cx.d.S = S;
    cx.T = (int)T;
    cx.L = make_layout(cx.d, T);
    cx.sv = (char*)saved;
    cx.ws = (char*)ws;
    cx.st = (cudaStream_t)stream;
    return XHC_OK;
}

bool params_ok(const Dims& d, const xhc_params* P, int slot, bool full) {
    if (!P) return false;
    if (full) {
        if (d.hr && !P->W_r) return false;
        for (int q = 0; q < d.G; ++q)
            if (!P->W_pre[q]) return false;
        if (!P->alpha_pre || !P->b_pre) return false;
    }
    if (!P->W_post[slot] || !P->alpha_post || !P->b_post[slot]) return false;
    if (slot == d.G - 1 && (!P->W_res || !P->alpha_res || !P->b_res)) return false;
    if (d.K[slot] > 1)
        for (int j = 0; j < d.nconv; ++j)
            if (!P->conv_w[slot][j]) return false;
    return true;
}

bool grads_ok(const Dims& d, const xhc_grads* g, int slot, bool full) {
    if (!g) return false;
    if (full) {
        if (d.hr && !g->W_r) return false;
        for (int q = 0; q < d.G; ++q)
            if (!g->W_pre[q]) return false;
        if (!g->alpha_pre || !g->b_pre) return false;
        return true;
    }
    if (!g->W_post[slot] || !g->alpha_post || !g->b_post[slot]) return false;
    if (slot == d.G - 1 && (!g->W_res || !g->alpha_res || !g->b_res)) return false;
    if (d.K[slot] > 1)
        for (int j = 0; j < d.nconv; ++j)
            if (!g->conv_w[slot][j]) return false;
    return true;
}

WSegs full_segs(const Dims& d, const xhc_params* P) {
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
    return w;
}

WSegsOut full_segs_g(const Dims& d, const xhc_grads* g) {
    WSegsOut w;
    memset(&w, 0, sizeof(w));
    int off = 0;
    if (d.hr) {
        w.ptr[w.n] = g->W_r; w.width[w.n] = d.N; w.off[w.n] = off; off += d.N; ++w.n;
    }
    for (int q = 0; q < d.G; ++q) {
        w.ptr[w.n] = g->W_pre[q]; w.width[w.n] = d.N; w.off[w.n] = off; off += d.N; ++w.n;
    }
    w.off[w.n] = off;
    return w;
}

WSegs act_segs(const Dims& d, const xhc_params* P, int slot) {
    WSegs w;
    memset(&w, 0, sizeof(w));
    w.ptr[0] = P->W_post[slot]; w.width[0] = d.k * d.K[slot]; w.off[0] = 0; w.n = 1;
    int off = d.k * d.K[slot];
    if (slot == d.G - 1) {
        w.ptr[1] = P->W_res; w.width[1] = d.k * d.k; w.off[1] = off; off += d.k * d.k; w.n = 2;
    }
    w.off[w.n] = off;
    return w;
}

WSegsOut act_segs_g(const Dims& d, const xhc_grads* g, int slot) {
    WSegsOut w;
    memset(&w, 0, sizeof(w));
    w.ptr[0] = g->W_post[slot]; w.width[0] = d.k * d.K[slot]; w.off[0] = 0; w.n = 1;
    int off = d.k * d.K[slot];
    if (slot == d.G - 1) {
        w.ptr[1] = g->W_res; w.width[1] = d.k * d.k; w.off[1] = off; off += d.k * d.k; w.n = 2;
    }
    w.off[w.n] = off;
    return w;
}

ConvPtrs conv_of(const Dims& d, const xhc_params* P, int slot) {
    ConvPtrs c;
    for (int j = 0; j < 3; ++j) c.w[j] = (j < d.nconv && d.K[slot] > 1) ? P->conv_w[slot][j] : nullptr;
    c.halo = nullptr;
    c.dhalo = nullptr;
    return c;
}

// above this many split-K partial slots the coefficient kernels get them pre-summed
constexpr int SLOT_SUM_MIN = 8;

// Active-state mapping generation of one slot (Eq. param_post, Eq. param_res).
xhc_status active_maps(const Ctx& c, int slot, const xhc_params* P) {
    const Dims& d = c.d;
    const WSegs wa = act_segs(d, P, slot);
    int splits = c.L.splits_act, ssplits = c.L.splits_act;
    float* pstats = c.W<float>(c.L.pstats);
    if (c.T < 128 || d.k * d.C < 64) {
        XHC_K("rowproj_active", c.st, launch_rowproj(c.xact(slot), (int64_t)d.k * d.C, d.k * d.C, c.T, wa,
                                                     d.nact[slot], c.L.splits_act, c.W<float>(c.L.part),
                                                     c.W<float>(c.L.pstats), c.st));
    } else {
        ProjTcPlan pl = plan_proj_tc(c.T, d.k * d.C, d.nact[slot], device_sms(), true);
        splits = pl.nseg;
        XHC_K("pack_w", c.st, launch_pack_w(wa, d.nact[slot], pl.NB, d.k * d.C,
                                            c.W<uint16_t>(c.L.wpack), c.st));
        // the norm statistics come from the read / input pass that produced x_act
        XHC_K("proj_tc_active", c.st, launch_proj_tc(c.xact(slot), c.T, d.k * d.C, c.W<uint16_t>(c.L.wpack),
                                                     d.nact[slot], pl, c.W<float>(c.L.part), nullptr,
                                                     c.W<int>(c.L.err), c.st));
        pstats = c.W<float>(c.L.astat);
        ssplits = stream_warps(d.C);
    }
    if (splits > SLOT_SUM_MIN) {
        XHC_K("slot_sum", c.st, launch_slot_sum(c.W<float>(c.L.part), splits, (long long)c.T * d.nact[slot], c.st));
        splits = 1;
    }
    if (ssplits > SLOT_SUM_MIN && pstats == c.W<float>(c.L.pstats)) {
        XHC_K("slot_sum", c.st, launch_slot_sum(pstats, ssplits, (long long)c.T * 2, c.st));
        ssplits = 1;
    }
    XHC_K("coef_act", c.st, launch_coef_act(d, slot, c.T, c.W<float>(c.L.part), pstats, ssplits,
                             splits, P->alpha_post, P->b_post[slot], P->alpha_res, P->b_res,
                             c.S<float>(c.L.zact[slot]), c.S<float>(c.L.rs[slot]),
                             c.S<float>(c.L.hpost[slot]), c.S<float>(c.L.hres), c.st));
    return XHC_OK;
}

}  // namespace

extern "C" {

xhc_status xhc_pre_fwd(const xhc_handle* h, int slot, int64_t T, const xhc_params* P,
                       const uint16_t* X, uint16_t* input, void* saved, void* workspace,
                       void* stream) {
    Ctx c;
    xhc_status s = common_check(h, slot, T, saved, workspace, c, stream);
    if (s != XHC_OK) return s;
    if (!X || !input || !params_ok(c.d, P, slot, slot == 0)) return XHC_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(input)) return XHC_ERR_ALIGNMENT;
    const Dims& d = c.d;
    if (slot == 0) {
        if (d.hr)
            XHC_K("colsum", c.st, launch_colsum(P->W_r, d.N * d.C, d.N, d.N, c.W<float>(c.L.wsum), 0,
                                   c.W<float>(c.L.colscr), c.st));
        const WSegs wf = full_segs(d, P);
        // partial slots written (and summed by coef_full): the split count of the path taken
        int fsplits = c.L.splits_full;
        if (c.T < 128 || d.N * d.C < 64) {
            // smaller than one tensor-core tile: fp32 CUDA-core projection
            XHC_K("rowproj_full", c.st, launch_rowproj(X, (int64_t)d.N * d.C, d.N * d.C, c.T, wf,
                                                       d.nfull, c.L.splits_full, c.W<float>(c.L.part),
                                                       c.W<float>(c.L.pstats), c.st));
        } else {
        fsplits = c.L.tc.nseg;
        XHC_K("pack_w", c.st, launch_pack_w(wf, d.nfull, c.L.tc.NB, d.N * d.C,
                                            c.W<uint16_t>(c.L.wpack), c.st));
        XHC_K("proj_tc", c.st, launch_proj_tc(X, c.T, d.N * d.C, c.W<uint16_t>(c.L.wpack), d.nfull,
                                              c.L.tc, c.W<float>(c.L.part), c.W<float>(c.L.pstats),
                                              c.W<int>(c.L.err), c.st));
        }
        if (fsplits > SLOT_SUM_MIN) {
            // few tokens, many split-K slots: summed in parallel first
            XHC_K("slot_sum", c.st, launch_slot_sum(c.W<float>(c.L.part), fsplits, (long long)c.T * d.nfull, c.st));
            XHC_K("slot_sum", c.st, launch_slot_sum(c.W<float>(c.L.pstats), fsplits, (long long)c.T * 2, c.st));
            fsplits = 1;
        }
        XHC_K("coef_full", c.st, launch_coef_full(d, c.T, c.W<float>(c.L.part), c.W<float>(c.L.pstats),
                                  fsplits, c.W<float>(c.L.wsum), P->alpha_pre, P->b_pre,
                                  c.S<float>(c.L.zfull), c.S<float>(c.L.stats),
                                  c.S<float>(c.L.hpre), c.S<int>(c.L.I), c.S<float>(c.L.p), c.st));
        XHC_K("read", c.st, launch_read(d, c.T, X, c.S<float>(c.L.hpre), c.S<int>(c.L.I), input,
                             c.W<uint16_t>(c.L.base), c.xact(0), c.W<float>(c.L.astat), c.st));
    } else {
        XHC_K("input", c.st, launch_input(d, slot, c.T, c.W<uint16_t>(c.L.base), c.xact(slot),
                              c.S<float>(c.L.hpre), c.S<int>(c.L.I), input, c.W<float>(c.L.astat), c.st));
    }
    return active_maps(c, slot, P);
}

}  // extern "C"

namespace {

xhc_status post_fwd_impl(const xhc_handle* h, int slot, int64_t T, const xhc_params* P,
                         uint16_t* X, const uint16_t* out, const uint16_t* halo, void* saved,
                         void* workspace, void* stream) {
    Ctx c;
    xhc_status s = common_check(h, slot, T, saved, workspace, c, stream);
    if (s != XHC_OK) return s;
    if (!X || !out || !params_ok(c.d, P, slot, false)) return XHC_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(out) || (halo && !aligned16(halo))) return XHC_ERR_ALIGNMENT;
    const Dims& d = c.d;
    ConvPtrs cw = conv_of(d, P, slot);
    if (d.K[slot] > 1) cw.halo = halo;
    const int gsl = wb_gram_slices(d);
    if (d.K[slot] > 1 && d.gs)
        XHC_K("wb_gram", c.st, launch_wb_gram(d, slot, c.T, out, cw, gsl, c.W<float>(c.L.red), c.st));
    const bool last = (slot == d.G - 1);
    XHC_K("wb_coef", c.st, launch_wb_coef(d, slot, c.T, c.W<float>(c.L.red), gsl, c.S<float>(c.L.p),
                                          c.S<float>(c.L.hpost[slot]),
                                          (d.K[slot] > 1 && d.gs) ? c.S<double>(c.L.gram[slot]) : nullptr,
                                          c.W<float>(c.L.tokmat), c.st));
    XHC_K("wb_fwd", c.st, launch_wb_fwd(d, slot, c.T, out, cw, c.W<float>(c.L.tokmat), c.L.nslice,
                                        c.xact(slot), c.S<int>(c.L.I), c.S<float>(c.L.hres),
                                        last ? nullptr : c.xact(slot + 1), X, c.st));
    return XHC_OK;
}

}  // namespace

extern "C" {

xhc_status xhc_post_fwd(const xhc_handle* h, int slot, int64_t T, const xhc_params* P,
                        uint16_t* X, const uint16_t* out, void* saved, void* workspace,
                        void* stream) {
    return post_fwd_impl(h, slot, T, P, X, out, nullptr, saved, workspace, stream);
}

xhc_status xhc_post_fwd_halo(const xhc_handle* h, int slot, int64_t T, const xhc_params* P,
                             uint16_t* X, const uint16_t* out, const uint16_t* halo, void* saved,
                             void* workspace, void* stream) {
    return post_fwd_impl(h, slot, T, P, X, out, halo, saved, workspace, stream);
}

xhc_status xhc_halo_bytes(const xhc_handle* h, int64_t B, size_t* bytes) {
    if (!h || !bytes || B <= 0) return XHC_ERR_INVALID_ARG;
    const Dims& d = h->h.d;
    *bytes = d.nconv > 0 ? (size_t)B * (d.kapmax - 1) * d.C * 2 : 0;
    return XHC_OK;
}

xhc_status xhc_halo_fill(const xhc_handle* h, int64_t B, int64_t S, const uint16_t* out, void* halo,
                         void* stream) {
    if (!h || !out || !halo || B <= 0 || S <= 0 || B * S > ((int64_t)1 << 30)) return XHC_ERR_INVALID_ARG;
    if (!aligned16(out) || !aligned16(halo)) return XHC_ERR_ALIGNMENT;
    const cudaError_t e = launch_halo_fill(h->h.d, (int)B, (int)S, out, (uint16_t*)halo, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, __LINE__);
    return XHC_OK;
}

xhc_status xhc_halo_add(const xhc_handle* h, int64_t B, int64_t S, uint16_t* d_out, const float* d_halo,
                        void* stream) {
    if (!h || !d_out || !d_halo || B <= 0 || S <= 0 || B * S > ((int64_t)1 << 30)) return XHC_ERR_INVALID_ARG;
    if (!aligned16(d_out) || !aligned16(d_halo)) return XHC_ERR_ALIGNMENT;
    const cudaError_t e = launch_halo_add(h->h.d, (int)B, (int)S, d_out, d_halo, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, __LINE__);
    return XHC_OK;
}

xhc_status xhc_stream_expand(const xhc_handle* h, int64_t T, const uint16_t* hidden, uint16_t* X,
                             void* stream) {
    if (!h || !hidden || !X || T <= 0 || T > ((int64_t)1 << 30)) return XHC_ERR_INVALID_ARG;
    if (!aligned16(hidden) || !aligned16(X)) return XHC_ERR_ALIGNMENT;
    const Dims& d = h->h.d;
    const cudaError_t e = launch_stream_bcast((int)T, d.N, d.C, hidden, X, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, __LINE__);
    return XHC_OK;
}

xhc_status xhc_stream_sum(const xhc_handle* h, int64_t T, const uint16_t* X, uint16_t* y, void* stream) {
    if (!h || !X || !y || T <= 0 || T > ((int64_t)1 << 30)) return XHC_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(y)) return XHC_ERR_ALIGNMENT;
    const Dims& d = h->h.d;
    const cudaError_t e = launch_stream_sum((int)T, d.N, d.C, X, y, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(e, __LINE__);
    return XHC_OK;
}

xhc_status xhc_ring_bytes(const xhc_handle* h, int64_t B, size_t* bytes) {
    if (!h || !bytes || B <= 0) return XHC_ERR_INVALID_ARG;
    const Dims& d = h->h.d;
    *bytes = d.nconv > 0 ? (size_t)B * (d.kapmax - 1) * d.C * 2 : 0;
    return XHC_OK;
}

xhc_status xhc_ring_fill(const xhc_handle* h, int64_t B, int64_t S, const uint16_t* out, void* ring,
                         void* stream) {
    if (!h || !out || !ring || B <= 0 || S <= 0 || B * S > ((int64_t)1 << 30)) return XHC_ERR_INVALID_ARG;
    if (!aligned16(out) || !aligned16(ring)) return XHC_ERR_ALIGNMENT;
    const Dims& d = h->h.d;
    if (d.nconv == 0) return XHC_OK;
    if (launch_ring_fill(d, (int)B, (int)S, out, (uint16_t*)ring, (cudaStream_t)stream) != cudaSuccess)
        return XHC_ERR_CUDA;
    return XHC_OK;
}

xhc_status xhc_post_fwd_decode(const xhc_handle* h, int slot, int64_t B, const xhc_params* P,
                               uint16_t* X, const uint16_t* out, void* ring, int64_t* pos,
                               void* saved, void* workspace, void* stream) {
    Ctx c;
    xhc_status s = common_check(h, slot, B, saved, workspace, c, stream);
    if (s != XHC_OK) return s;
    const Dims& d = c.d;
    const bool conv = d.K[slot] > 1;
    if (!X || !out || !pos || (conv && !ring) || !params_ok(d, P, slot, false)) return XHC_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(out) || (ring && !aligned16(ring))) return XHC_ERR_ALIGNMENT;
    const ConvPtrs cw = conv_of(d, P, slot);
    const bool last = (slot == d.G - 1);
    long long* ps = reinterpret_cast<long long*>(pos);
    uint16_t* rg = static_cast<uint16_t*>(ring);
    if (conv && d.gs)
        XHC_K("dec_gram", c.st, launch_dec_gram(d, slot, c.T, out, cw, rg, ps, c.W<float>(c.L.red), c.st));
    XHC_K("wb_coef", c.st, launch_wb_coef(d, slot, c.T, c.W<float>(c.L.red), dec_nslice(d.C), c.S<float>(c.L.p),
                                          c.S<float>(c.L.hpost[slot]),
                                          (conv && d.gs) ? c.S<double>(c.L.gram[slot]) : nullptr,
                                          c.W<float>(c.L.tokmat), c.st));
    XHC_K("dec_fwd", c.st, launch_dec_fwd(d, slot, c.T, out, cw, rg, ps, c.W<float>(c.L.tokmat),
                                          c.xact(slot), c.S<int>(c.L.I), c.S<float>(c.L.hres),
                                          last ? nullptr : c.xact(slot + 1), X, c.st));
    return XHC_OK;
}

}  // extern "C"

namespace {

xhc_status post_bwd_impl(const xhc_handle* h, int slot, int64_t T, const xhc_params* P,
                         uint16_t* X, uint16_t* dX, const uint16_t* out, uint16_t* d_out,
                         const xhc_grads* g, const uint16_t* halo, float* d_halo, void* saved,
                         void* workspace, void* stream) {
    Ctx c;
    xhc_status s = common_check(h, slot, T, saved, workspace, c, stream);
    if (s != XHC_OK) return s;
    if (!X || !dX || !out || !d_out || !params_ok(c.d, P, slot, false) ||
        !grads_ok(c.d, g, slot, false))
        return XHC_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(dX) || !aligned16(out) || !aligned16(d_out) ||
        (halo && !aligned16(halo)) || (d_halo && !aligned16(d_halo)))
        return XHC_ERR_ALIGNMENT;
    const Dims& d = c.d;
    const int T32 = c.T;
    const bool last = (slot == d.G - 1);
    ConvPtrs cw = conv_of(d, P, slot);
    if (d.K[slot] > 1) {
        cw.halo = halo;
        cw.dhalo = d_halo;
    }
    const int K = d.K[slot], n = d.nact[slot];
    float* red = c.W<float>(c.L.red);
    float* dxact = c.W<float>(c.L.dxact);
    if (last) {
        XHC_CUDA(cudaMemsetAsync(c.W<float>(c.L.dp), 0, (size_t)T32 * d.k * 4, c.st));
        XHC_K("restore", c.st, launch_restore(d, T32, c.xact(0), c.S<int>(c.L.I), X, c.st));
    }
    const int bslices = wb_bred_slices(d, slot);
    if (K == 1) {
        // no conv: reductions and apply in one pass (the apply coefficients are forward values)
        XHC_K("wb_b8", c.st, launch_wb_b8(d, slot, T32, out, dX, c.S<int>(c.L.I), c.S<float>(c.L.p),
                                          c.S<float>(c.L.hpost[slot]), c.S<float>(c.L.hres), dxact, dxact,
                                          c.xact(slot), bslices, red, d_out, c.st));
    } else {
        XHC_K("wb_bred", c.st, launch_wb_bred(d, slot, T32, out, cw, dX, c.S<int>(c.L.I), dxact, c.xact(slot),
                                              bslices, red, c.st));
    }
    XHC_K("bwd_coef", c.st, launch_bwd_coef(d, slot, T32, red, bslices, c.S<float>(c.L.zact[slot]),
                             c.S<float>(c.L.rs[slot]), c.S<float>(c.L.p),
                             c.S<float>(c.L.hpost[slot]),
                             (d.K[slot] > 1 && d.gs) ? c.S<double>(c.L.gram[slot]) : nullptr,
                             P->alpha_post, P->b_post[slot],
                             P->alpha_res, P->b_res, c.W<float>(c.L.tokmat), c.W<float>(c.L.dz),
                             c.W<float>(c.L.dp), c.W<float>(c.L.tokgrad), c.st));
    // weight gradient of the post/res projections and the alpha / b column sums need only dZ_act
    // and the per-token contributions: side stream, overlapping the apply kernel
    const cudaStream_t sd = fork_from(c.st);
    if (T32 < 64 || d.k * d.C < 128) {
        const int ts = std::min(c.L.tsplits, pick_tsplits(d.k * d.C, T32));
        XHC_K("wgrad_active", sd, launch_wgrad(c.xact(slot), (int64_t)d.k * d.C, d.k * d.C, T32,
                                               c.W<float>(c.L.dz), n, n, ts, c.W<float>(c.L.wpart),
                                               act_segs_g(d, g, slot), sd));
    } else {
        ProjTcPlan pl = plan_proj_tc(d.k * d.C, T32, n, device_sms(), false);
        XHC_K("wgrad_tc_active", sd, launch_wgrad_tc(c.xact(slot), T32, d.k * d.C, c.W<float>(c.L.dz), n, n,
                                                     c.W<uint16_t>(c.L.dzpack), pl, c.W<float>(c.L.wpart),
                                                     c.W<int>(c.L.err), sd));
        XHC_K("wgrad_reduce", sd, launch_wgrad_reduce(c.W<float>(c.L.wpart), pl.nseg, d.k * d.C, n,
                                                      act_segs_g(d, g, slot), sd));
    }
    float* tg = c.W<float>(c.L.tokgrad);
    float* scr = c.W<float>(c.L.colscr);
    XHC_K("colsum", sd, launch_colsum(tg, T32, NTG, d.k * K, g->b_post[slot], 1, scr, sd));
    XHC_K("colsum", sd, launch_colsum(tg + d.k * K, T32, NTG, 1, g->alpha_post + slot, 1, scr, sd));
    if (last) {
        XHC_K("colsum", sd, launch_colsum(tg + d.k * K + 1, T32, NTG, d.k * d.k, g->b_res, 1, scr, sd));
        XHC_K("colsum", sd, launch_colsum(tg + d.k * K + 1 + d.k * d.k, T32, NTG, 1, g->alpha_res, 1, scr, sd));
    }
    // d_out, conv weight-gradient partials and (last slot) the mixed active gradient; the
    // active gradient of earlier slots is read in place and completed by pre_bwd(slot)
    if (K > 1)
        XHC_K("wb_bapp", c.st, launch_wb_bapp(d, slot, T32, out, cw, dX, c.S<int>(c.L.I), dxact,
                                              c.W<float>(c.L.tokmat), dxact, d_out,
                                              c.W<float>(c.L.cpart), c.st));
    const WSegs wa = act_segs(d, P, slot);
    // dZ_act stays in the workspace: pre_bwd(slot) applies it to dX_act on the tensor cores
    if (!dxa_tc_ok(T32, d.k, d.C, n))
        XHC_K("gemm_dzw", c.st, launch_gemm_dzw(d, T32, c.W<float>(c.L.dz), n, n, wa, d.k * d.C, dxact, c.st));
    if (K > 1) {
        ConvGradPtrs gc;
        for (int j = 0; j < 3; ++j) gc.w[j] = (j < d.nconv) ? g->conv_w[slot][j] : nullptr;
        XHC_K("conv_wgrad_reduce", c.st, launch_conv_wgrad_reduce(d, slot, c.W<float>(c.L.cpart), c.L.ntiles, gc, c.st));
    }
    return join_into(c.st, sd);
}

}  // namespace

extern "C" {

xhc_status xhc_post_bwd(const xhc_handle* h, int slot, int64_t T, const xhc_params* P,
                        uint16_t* X, uint16_t* dX, const uint16_t* out, uint16_t* d_out,
                        const xhc_grads* g, void* saved, void* workspace, void* stream) {
    return post_bwd_impl(h, slot, T, P, X, dX, out, d_out, g, nullptr, nullptr, saved, workspace, stream);
}

xhc_status xhc_post_bwd_halo(const xhc_handle* h, int slot, int64_t T, const xhc_params* P,
                             uint16_t* X, uint16_t* dX, const uint16_t* out, uint16_t* d_out,
                             const xhc_grads* g, const uint16_t* halo, float* d_halo, void* saved,
                             void* workspace, void* stream) {
    // a slot with a conv and a halo must return the halo's gradient
    if (h && slot >= 0 && slot < h->h.d.G && h->h.d.K[slot] > 1 && halo && !d_halo)
        return XHC_ERR_INVALID_ARG;
    return post_bwd_impl(h, slot, T, P, X, dX, out, d_out, g, halo, d_halo, saved, workspace, stream);
}

xhc_status xhc_pre_bwd(const xhc_handle* h, int slot, int64_t T, const xhc_params* P,
                       const uint16_t* X, const uint16_t* d_input, uint16_t* dX,
                       const xhc_grads* g, void* saved, void* workspace, void* stream) {
    Ctx c;
    xhc_status s = common_check(h, slot, T, saved, workspace, c, stream);
    if (s != XHC_OK) return s;
    if (!X || !d_input || !dX || !params_ok(c.d, P, slot, slot == 0) ||
        (slot == 0 && !grads_ok(c.d, g, slot, true)))
        return XHC_ERR_INVALID_ARG;
    if (!aligned16(X) || !aligned16(d_input) || !aligned16(dX)) return XHC_ERR_ALIGNMENT;
    const Dims& d = c.d;
    const int T32 = c.T;
    uint16_t* dinput = c.W<uint16_t>(c.L.dinput);
    const int n = d.nact[slot];
    const bool tc = dxa_tc_ok(T32, d.k, d.C, n);
    if (tc) {
        // post_bwd(slot) left dZ_act of this slot in the workspace; the update also forms the
        // dH_pre dots of the active streams (per 32 channels) and copies d_input
        XHC_K("dxa_tc", c.st, launch_dxa_tc(d, slot, T32, c.W<float>(c.L.dz), n, act_segs(d, P, slot),
                                            c.W<uint16_t>(c.L.dz16), c.W<uint16_t>(c.L.w16), d_input,
                                            c.S<float>(c.L.hpre), c.S<int>(c.L.I), c.xact(slot),
                                            c.W<float>(c.L.tokmat), c.W<float>(c.L.dxact),
                                            c.W<float>(c.L.dotp), dinput, c.W<int>(c.L.err), c.st));
        XHC_K("dots_act", c.st, launch_dots_act(d, slot, T32, c.W<float>(c.L.dotp), c.S<int>(c.L.I),
                                                c.W<float>(c.L.dhpre), c.st));
    } else {
        XHC_K("dinput_act", c.st, launch_dinput_act(d, slot, T32, 1, d_input, c.xact(slot),
                                    c.S<float>(c.L.hpre), c.S<int>(c.L.I), c.W<float>(c.L.dxact),
                                    c.W<float>(c.L.dhpre), dinput, c.W<float>(c.L.tokmat), c.st));
    }
    if (slot != 0) return XHC_OK;
    if (d.hr)
        XHC_K("colsum", c.st, launch_colsum(P->W_r, d.N * d.C, d.N, d.N, c.W<float>(c.L.wsum), 0,
                               c.W<float>(c.L.colscr), c.st));
    XHC_K("full_dots", c.st, launch_full_dots(d, T32, X, dinput, c.S<int>(c.L.I), c.W<float>(c.L.dhpre), c.st));
    XHC_K("full_coef", c.st, launch_full_coef(d, T32, c.W<float>(c.L.dhpre), c.S<float>(c.L.hpre),
                              c.S<float>(c.L.zfull), c.S<float>(c.L.stats), c.W<float>(c.L.wsum),
                              c.S<int>(c.L.I), c.W<float>(c.L.dp), P->alpha_pre,
                              c.W<float>(c.L.dz), c.W<float>(c.L.tokgrad), c.st));
    // the full-state weight gradient and the pre-map / router column sums need only dZ and the
    // per-token contributions: side stream, overlapping the full-state dX
    const cudaStream_t sd = fork_from(c.st);
    if (T32 < 64 || d.N * d.C < 128) {
        const int ts = std::min(c.L.tsplits, pick_tsplits(d.N * d.C, T32));
        XHC_K("wgrad_full", sd, launch_wgrad(X, (int64_t)d.N * d.C, d.N * d.C, T32, c.W<float>(c.L.dz),
                                               d.nfull, d.nfull, ts, c.W<float>(c.L.wpart),
                                               full_segs_g(d, g), sd));
    } else {
        const ProjTcPlan& pl = c.L.twf;
        XHC_K("wgrad_tc_full", sd, launch_wgrad_tc(X, T32, d.N * d.C, c.W<float>(c.L.dz), d.nfull, d.nfull,
                                                     c.W<uint16_t>(c.L.dzpack), pl, c.W<float>(c.L.wpart),
                                                     c.W<int>(c.L.err), sd));
        XHC_K("wgrad_reduce", sd, launch_wgrad_reduce(c.W<float>(c.L.wpart), pl.nseg, d.N * d.C, d.nfull,
                                                        full_segs_g(d, g), sd));
    }
    float* tg = c.W<float>(c.L.tokgrad);
    float* scr = c.W<float>(c.L.colscr);
    XHC_K("colsum", sd, launch_colsum(tg + 2, T32, NTG, d.G * d.N, g->b_pre, 1, scr, sd));
    XHC_K("colsum", sd, launch_colsum(tg + 2 + d.G * d.N, T32, NTG, d.G, g->alpha_pre, 1, scr, sd));
    if (d.hr) {
        float* rsum = c.W<float>(c.L.rsum);
        XHC_K("colsum", sd, launch_colsum(tg + 2 + d.G * d.N + d.G, T32, NTG, d.N, rsum, 0, scr, sd));
        XHC_K("sub_rows", sd, launch_sub_rows(g->W_r, d.N * d.C, d.N, rsum, sd));
    }
    const WSegs wf = full_segs(d, P);
    if (dx_tc_ok(T32, d.N, d.C, d.nfull, d.G)) {
        XHC_K("dx_tc", c.st, launch_dx_tc(d, T32, c.W<float>(c.L.dz), wf, c.W<uint16_t>(c.L.dz16),
                                          c.W<uint16_t>(c.L.w16), X, dinput, c.S<float>(c.L.hpre),
                                          c.S<int>(c.L.I), c.W<float>(c.L.dxact), c.W<float>(c.L.tokgrad),
                                          NTG, dX, c.W<int>(c.L.err), c.st));
    } else {
        XHC_K("full_dx", c.st, launch_full_dx(d, T32, c.W<float>(c.L.dz), wf, X, dinput, c.S<float>(c.L.hpre),
                                              c.S<int>(c.L.I), c.W<float>(c.L.dxact),
                                              c.W<float>(c.L.tokgrad), dX, c.st));
    }
    return join_into(c.st, sd);
}

}  // extern "C"
