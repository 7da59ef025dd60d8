"""Python binding of libxhc: ctypes marshalling of torch tensors into the C ABI of include/xhc.h.

Every step of the connection op runs in the library's CUDA kernels; this module only passes
``data_ptr()`` values, sizes and the current CUDA stream.  Importing it loads
``lib/libxhc.so``; if the library is missing the import fails loudly (there is no fallback).
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass, field

import torch

from . import build as _build

MAX_GROUP = 4
MAX_CONV = 3

MHC, FULL, FLASH = 0, 1, 2
STATUS = {0: "ok", 1: "invalid argument", 2: "unsupported", 3: "alignment", 4: "cuda error", 5: "timeout"}


class _Config(ctypes.Structure):
    _fields_ = [("variant", ctypes.c_int), ("N", ctypes.c_int), ("k", ctypes.c_int),
                ("m", ctypes.c_int), ("C", ctypes.c_int), ("group", ctypes.c_int),
                ("mlp_mask", ctypes.c_int), ("n_conv", ctypes.c_int),
                ("conv_k", ctypes.c_int * MAX_CONV), ("gram_schmidt", ctypes.c_int),
                ("sinkhorn_iters", ctypes.c_int), ("eps_norm", ctypes.c_float),
                ("eps_gs", ctypes.c_float), ("seq_len", ctypes.c_int), ("router", ctypes.c_int),
                ("sparse_read", ctypes.c_int)]


_P = ctypes.c_void_p


class _Params(ctypes.Structure):
    _fields_ = [("W_r", _P), ("W_pre", _P * MAX_GROUP), ("alpha_pre", _P), ("b_pre", _P),
                ("W_post", _P * MAX_GROUP), ("alpha_post", _P), ("b_post", _P * MAX_GROUP),
                ("W_res", _P), ("alpha_res", _P), ("b_res", _P),
                ("conv_w", (_P * MAX_CONV) * MAX_GROUP)]


_Grads = _Params  # same layout (float* instead of const float*)


class _SavedLayout(ctypes.Structure):
    _fields_ = [("I", ctypes.c_size_t), ("p", ctypes.c_size_t), ("hpre", ctypes.c_size_t),
                ("hpost", ctypes.c_size_t * MAX_GROUP), ("hres", ctypes.c_size_t),
                ("xact", ctypes.c_size_t), ("zfull", ctypes.c_size_t), ("stats", ctypes.c_size_t)]


class XhcError(RuntimeError):
    pass


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded libxhc.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        path = _build.LIB
        if not os.path.exists(path):
            raise XhcError(f"libxhc.so not found at {path}: run paper_2607_14530_gb300.build.build()")
        L = ctypes.CDLL(path)
        i64, vp, sz = ctypes.c_int64, ctypes.c_void_p, ctypes.c_size_t
        L.xhc_create.argtypes = [ctypes.POINTER(_Config), ctypes.POINTER(vp)]
        L.xhc_destroy.argtypes = [vp]
        L.xhc_destroy.restype = None
        L.xhc_saved_bytes.argtypes = [vp, i64, ctypes.POINTER(sz)]
        L.xhc_workspace_bytes.argtypes = [vp, i64, ctypes.POINTER(sz)]
        P = ctypes.POINTER(_Params)
        L.xhc_pre_fwd.argtypes = [vp, ctypes.c_int, i64, P, vp, vp, vp, vp, vp]
        L.xhc_post_fwd.argtypes = [vp, ctypes.c_int, i64, P, vp, vp, vp, vp, vp]
        L.xhc_post_bwd.argtypes = [vp, ctypes.c_int, i64, P, vp, vp, vp, vp, P, vp, vp, vp]
        L.xhc_pre_bwd.argtypes = [vp, ctypes.c_int, i64, P, vp, vp, vp, P, vp, vp, vp]
        L.xhc_saved_layout_of.argtypes = [vp, i64, ctypes.POINTER(_SavedLayout)]
        L.xhc_route_noalloc.argtypes = [vp, i64, P, vp, vp, vp, vp, vp]
        L.xhc_ring_bytes.argtypes = [vp, i64, ctypes.POINTER(sz)]
        L.xhc_ring_fill.argtypes = [vp, i64, i64, vp, vp, vp]
        L.xhc_post_fwd_decode.argtypes = [vp, ctypes.c_int, i64, P, vp, vp, vp, vp, vp, vp, vp]
        L.xhc_stream_expand.argtypes = [vp, i64, vp, vp, vp]
        L.xhc_stream_sum.argtypes = [vp, i64, vp, vp, vp]
        L.xhc_halo_bytes.argtypes = [vp, i64, ctypes.POINTER(sz)]
        L.xhc_halo_fill.argtypes = [vp, i64, i64, vp, vp, vp]
        L.xhc_halo_add.argtypes = [vp, i64, i64, vp, vp, vp]
        L.xhc_post_fwd_halo.argtypes = [vp, ctypes.c_int, i64, P, vp, vp, vp, vp, vp, vp]
        L.xhc_post_bwd_halo.argtypes = [vp, ctypes.c_int, i64, P, vp, vp, vp, vp, P, vp, vp, vp, vp, vp]
        L.xhc_workspace_error.argtypes = [vp, ctypes.POINTER(ctypes.c_int), ctypes.c_int]
        L.xhc_debug_set.argtypes = [ctypes.c_int, i64]
        L.xhc_trace_enable.argtypes = [ctypes.c_int]
        L.xhc_trace_count.restype = ctypes.c_int
        L.xhc_trace_record.argtypes = [ctypes.c_int, ctypes.POINTER(ctypes.c_char_p),
                                       ctypes.POINTER(ctypes.c_float)]
        L.xhc_trace_only.argtypes = [ctypes.c_char_p]
        L.xhc_trace_span.argtypes = [ctypes.c_int, ctypes.POINTER(ctypes.c_char_p),
                                     ctypes.POINTER(ctypes.c_float), ctypes.POINTER(ctypes.c_float)]
        L.xhc_launch_count.restype = ctypes.c_uint64
        L.xhc_status_string.argtypes = [ctypes.c_int]
        L.xhc_status_string.restype = ctypes.c_char_p
        L.xhc_last_error_string.restype = ctypes.c_char_p
        L.xhc_version.restype = ctypes.c_int
        _lib = L
    return _lib


def _check(status: int, what: str):
    if status != 0:
        msg = STATUS.get(status, str(status))
        if status == 4:
            msg += ": " + lib().xhc_last_error_string().decode()
        raise XhcError(f"{what} failed: {msg}")


def trace_enable(on: bool) -> None:
    """Start (clearing old records) or stop recording per-launch CUDA events in the library."""
    _check(lib().xhc_trace_enable(1 if on else 0), "xhc_trace_enable")


def trace_only(names=None) -> None:
    """Record only the launches of these kernel names (an iterable of names; None: every launch)."""
    arg = None if not names else ",".join(names).encode()
    _check(lib().xhc_trace_only(arg), "xhc_trace_only")


def trace_spans() -> list:
    """[(kernel name, start ms after the first record's start, device ms)]; synchronise first."""
    L = lib()
    out = []
    for i in range(L.xhc_trace_count()):
        name, t0, ms = ctypes.c_char_p(), ctypes.c_float(), ctypes.c_float()
        _check(L.xhc_trace_span(i, ctypes.byref(name), ctypes.byref(t0), ctypes.byref(ms)), "xhc_trace_span")
        out.append((name.value.decode(), float(t0.value), float(ms.value)))
    return out


def trace_records() -> list:
    """[(kernel name, device ms)] of the recorded launches; synchronise the stream first."""
    L = lib()
    out = []
    for i in range(L.xhc_trace_count()):
        name, ms = ctypes.c_char_p(), ctypes.c_float()
        _check(L.xhc_trace_record(i, ctypes.byref(name), ctypes.byref(ms)), "xhc_trace_record")
        out.append((name.value.decode(), float(ms.value)))
    return out


def debug_wait_limit_ns(ns: int) -> None:
    """Limit of the library's bounded device waits for later launches (0: the default ~4 s).
    A test hook (xhc_debug_set)."""
    _check(lib().xhc_debug_set(1, int(ns)), "xhc_debug_set")


def debug_force_timeout() -> None:
    """Make the next tensor-core full-state projection time out before it issues any work (a
    test hook for the bounded-wait abort path; xhc_debug_set)."""
    _check(lib().xhc_debug_set(2, 1), "xhc_debug_set")


def debug_one_stream(on: bool) -> None:
    """Run the library's side-stream work on the caller's stream (same order, same results)."""
    _check(lib().xhc_debug_set(3, 1 if on else 0), "xhc_debug_set")


def launch_count() -> int:
    """Kernels launched by the library since it was loaded."""
    return int(lib().xhc_launch_count())


@dataclass(frozen=True)
class Config:
    """Mirror of xhc_config (include/xhc.h)."""
    variant: int
    N: int
    k: int
    m: int
    C: int
    G: int = 1
    mlp_mask: int = 0
    conv_k: tuple = (4, 8, 12)
    gram_schmidt: bool = True
    sinkhorn_iters: int = 20
    eps_norm: float = 1e-5
    eps_gs: float = 0.0
    seq_len: int = 0
    router: str = "sigmoid"        # or "softmax" (the softmax-router ablation)
    sparse_read: bool = False      # read only the k active streams (the sparse-read ablation)

    @staticmethod
    def mhc(N, C, **kw):
        return Config(MHC, N, N, N, C, 1, 0, (), **kw)

    @staticmethod
    def full(N, k, m, C, mlp, **kw):
        return Config(FULL, N, k, m, C, 1, 1 if mlp else 0, **kw)

    @staticmethod
    def flash(N, k, m, C, G, attn_tfa=False, **kw):
        """xHC-Flash group, slots A, M (, A, M); attn_tfa also augments the attention slots."""
        mask = (0x2 if G == 2 else 0xA) | ((0x1 if G == 2 else 0x5) if attn_tfa else 0)
        return Config(FLASH, N, k, m, C, G, mask, **kw)

    @property
    def has_router(self):
        return self.m < self.k

    def K(self, t):
        return 1 + len(self.conv_k) if ((self.mlp_mask >> t) & 1 and len(self.conv_k) > 0) else 1

    def param_shapes(self) -> dict:
        """Flat ``{name: shape}`` of every parameter (names used by the binding)."""
        N, k, C, G = self.N, self.k, self.C, self.G
        sh = {}
        if self.has_router:
            sh["W_r"] = (N * C, N)
        for t in range(G):
            sh[f"W_pre.{t}"] = (N * C, N)
            sh[f"W_post.{t}"] = (k * C, k * self.K(t))
            sh[f"b_post.{t}"] = (k * self.K(t),)
            if self.K(t) > 1:
                for j, kap in enumerate(self.conv_k):
                    sh[f"conv_w.{t}.{j}"] = (kap, C)
        sh["alpha_pre"] = (G,)
        sh["b_pre"] = (G, N)
        sh["alpha_post"] = (G,)
        sh["W_res"] = (k * C, k * k)
        sh["alpha_res"] = (1,)
        sh["b_res"] = (k * k,)
        return sh

    def _c(self) -> _Config:
        c = _Config()
        c.variant, c.N, c.k, c.m, c.C, c.group = self.variant, self.N, self.k, self.m, self.C, self.G
        c.mlp_mask = self.mlp_mask
        c.n_conv = len(self.conv_k)
        for j, v in enumerate(self.conv_k):
            c.conv_k[j] = v
        c.gram_schmidt = 1 if self.gram_schmidt else 0
        c.sinkhorn_iters = self.sinkhorn_iters
        c.eps_norm = self.eps_norm
        c.eps_gs = self.eps_gs
        c.seq_len = self.seq_len
        c.router = {"sigmoid": 0, "softmax": 1}[self.router]
        c.sparse_read = 1 if self.sparse_read else 0
        return c


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _fill(struct, d: dict, cfg: Config):
    """Fill a _Params/_Grads from a flat dict of fp32 CUDA tensors."""
    def get(n):
        v = d.get(n)
        if v is None:
            return None
        if v.dtype != torch.float32 or not v.is_cuda or not v.is_contiguous():
            raise XhcError(f"parameter {n} must be a contiguous fp32 CUDA tensor")
        return v.data_ptr()
    struct.W_r = get("W_r")
    for t in range(cfg.G):
        struct.W_pre[t] = get(f"W_pre.{t}")
        struct.W_post[t] = get(f"W_post.{t}")
        struct.b_post[t] = get(f"b_post.{t}")
        for j in range(len(cfg.conv_k)):
            struct.conv_w[t][j] = get(f"conv_w.{t}.{j}")
    struct.alpha_pre = get("alpha_pre")
    struct.b_pre = get("b_pre")
    struct.alpha_post = get("alpha_post")
    struct.W_res = get("W_res")
    struct.alpha_res = get("alpha_res")
    struct.b_res = get("b_res")
    return struct


def _bf16(t, name):
    if t.dtype != torch.bfloat16 or not t.is_cuda or not t.is_contiguous():
        raise XhcError(f"{name} must be a contiguous bf16 CUDA tensor")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


class Group:
    """One connection-op group (G sublayers) bound to a libxhc handle."""

    def __init__(self, cfg: Config):
        self.cfg = cfg
        self._c = cfg._c()
        h = ctypes.c_void_p()
        _check(lib().xhc_create(ctypes.byref(self._c), ctypes.byref(h)), "xhc_create")
        self._h = h

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None and h.value and _lib is not None:
            _lib.xhc_destroy(h)
            self._h = None

    def saved_bytes(self, T: int) -> int:
        n = ctypes.c_size_t()
        _check(lib().xhc_saved_bytes(self._h, T, ctypes.byref(n)), "xhc_saved_bytes")
        return n.value

    def workspace_bytes(self, T: int) -> int:
        n = ctypes.c_size_t()
        _check(lib().xhc_workspace_bytes(self._h, T, ctypes.byref(n)), "xhc_workspace_bytes")
        return n.value

    def coefficients(self, saved, T: int) -> dict:
        """Views into `saved` of the coefficients left by the forward (see xhc_saved_layout)."""
        L = _SavedLayout()
        _check(lib().xhc_saved_layout_of(self._h, T, ctypes.byref(L)), "xhc_saved_layout_of")
        cfg = self.cfg
        k, N, G = cfg.k, cfg.N, cfg.G

        def view(off, n, dtype):
            nb = n * torch.empty(0, dtype=dtype).element_size()
            return saved[off:off + nb].view(dtype)

        out = dict(I=view(L.I, T * k, torch.int32).view(T, k),
                   p=view(L.p, T * k, torch.float32).view(T, k),
                   hpre=view(L.hpre, T * G * N, torch.float32).view(T, G, N),
                   hres=view(L.hres, T * k * k, torch.float32).view(T, k, k),
                   xact=view(L.xact, G * T * k * cfg.C, torch.bfloat16).view(G, T, k, cfg.C))
        nfull = (N if cfg.has_router else 0) + G * N
        out["zfull"] = view(L.zfull, T * nfull, torch.float32).view(T, nfull)
        out["stats"] = view(L.stats, T * 2, torch.float32).view(T, 2)
        out["hpost"] = [view(L.hpost[t], T * k * cfg.K(t), torch.float32).view(T, k, cfg.K(t))
                        for t in range(G)]
        return out

    def alloc_saved(self, T: int, device="cuda"):
        """A `saved` buffer: one per forward whose backward is still to come."""
        return torch.empty(self.saved_bytes(T), dtype=torch.uint8, device=device)

    def alloc_workspace(self, T: int, device="cuda"):
        """A `workspace` buffer (scratch, reusable between the phases of groups), error word zeroed."""
        ws = torch.empty(self.workspace_bytes(T), dtype=torch.uint8, device=device)
        ws[:256].zero_()  # device error word
        return ws

    def alloc(self, T: int, device="cuda"):
        """(saved, workspace) uint8 CUDA tensors of the sizes the library asks for."""
        ws = self.alloc_workspace(T, device)
        return (self.alloc_saved(T, device), ws)

    def device_error(self, ws, clear: bool = False) -> int:
        """The workspace's device error word (nonzero: a bounded wait gave up).  Synchronous."""
        code = ctypes.c_int()
        lib().xhc_workspace_error(_ptr(ws), ctypes.byref(code), 1 if clear else 0)
        return code.value

    def params(self, P: dict) -> _Params:
        return _fill(_Params(), P, self.cfg)

    def route_noalloc(self, P, X, I, p, hpre, stream=None):
        """Routing (I int32 [T, k], p fp32 [T, k]) and pre-maps (hpre fp32 [T, G, N]) of X, for
        callers that cannot allocate a workspace (xhc_route_noalloc)."""
        T = X.shape[0]
        pp = P if isinstance(P, _Params) else self.params(P)
        for t, n, dt in ((I, "I", torch.int32), (p, "p", torch.float32), (hpre, "hpre", torch.float32)):
            if t.dtype != dt or not t.is_cuda or not t.is_contiguous():
                raise XhcError(f"{n} must be a contiguous {dt} CUDA tensor")
        _check(lib().xhc_route_noalloc(self._h, T, ctypes.byref(pp), _bf16(X, "X"), _ptr(I), _ptr(p),
                                       _ptr(hpre), _stream(stream)), "xhc_route_noalloc")

    def pre_fwd(self, slot, P, X, inp, saved, ws, stream=None):
        T = X.shape[0]
        pp = P if isinstance(P, _Params) else self.params(P)
        _check(lib().xhc_pre_fwd(self._h, slot, T, ctypes.byref(pp), _bf16(X, "X"), _bf16(inp, "input"),
                                 _ptr(saved), _ptr(ws), _stream(stream)), f"xhc_pre_fwd({slot})")

    def post_fwd(self, slot, P, X, out, saved, ws, stream=None, halo=None):
        """xhc_post_fwd; with ``halo`` (bf16 [B, R, C], see halo_fill) xhc_post_fwd_halo."""
        T = X.shape[0]
        pp = P if isinstance(P, _Params) else self.params(P)
        if halo is None:
            _check(lib().xhc_post_fwd(self._h, slot, T, ctypes.byref(pp), _bf16(X, "X"), _bf16(out, "out"),
                                      _ptr(saved), _ptr(ws), _stream(stream)), f"xhc_post_fwd({slot})")
        else:
            _check(lib().xhc_post_fwd_halo(self._h, slot, T, ctypes.byref(pp), _bf16(X, "X"),
                                           _bf16(out, "out"), _bf16(halo, "halo"), _ptr(saved), _ptr(ws),
                                           _stream(stream)), f"xhc_post_fwd_halo({slot})")

    def post_bwd(self, slot, P, X, dX, out, d_out, grads, saved, ws, stream=None, halo=None,
                 d_halo=None):
        """xhc_post_bwd; with ``halo`` xhc_post_bwd_halo, writing the halo's gradient into
        ``d_halo`` (fp32 [B, R, C])."""
        T = X.shape[0]
        pp = P if isinstance(P, _Params) else self.params(P)
        gg = grads if isinstance(grads, _Params) else self.params(grads)
        if halo is None:
            _check(lib().xhc_post_bwd(self._h, slot, T, ctypes.byref(pp), _bf16(X, "X"), _bf16(dX, "dX"),
                                      _bf16(out, "out"), _bf16(d_out, "d_out"), ctypes.byref(gg),
                                      _ptr(saved), _ptr(ws), _stream(stream)), f"xhc_post_bwd({slot})")
        else:
            if d_halo is None or d_halo.dtype != torch.float32 or not d_halo.is_cuda or not d_halo.is_contiguous():
                raise XhcError("d_halo must be a contiguous fp32 CUDA tensor")
            _check(lib().xhc_post_bwd_halo(self._h, slot, T, ctypes.byref(pp), _bf16(X, "X"), _bf16(dX, "dX"),
                                           _bf16(out, "out"), _bf16(d_out, "d_out"), ctypes.byref(gg),
                                           _bf16(halo, "halo"), _ptr(d_halo), _ptr(saved), _ptr(ws),
                                           _stream(stream)), f"xhc_post_bwd_halo({slot})")

    # ---- model glue ----

    def stream_expand(self, hidden, X=None, stream=None):
        """[T, C] -> [T, N, C]: N copies of every token's hidden vector (xhc_stream_expand)."""
        T = hidden.shape[0]
        if X is None:
            X = torch.empty(T, self.cfg.N, self.cfg.C, dtype=torch.bfloat16, device=hidden.device)
        _check(lib().xhc_stream_expand(self._h, T, _bf16(hidden, "hidden"), _bf16(X, "X"), _stream(stream)),
               "xhc_stream_expand")
        return X

    def stream_sum(self, X, y=None, stream=None):
        """[T, N, C] -> [T, C]: the sum of the N streams of every token (xhc_stream_sum)."""
        T = X.shape[0]
        if y is None:
            y = torch.empty(T, self.cfg.C, dtype=torch.bfloat16, device=X.device)
        _check(lib().xhc_stream_sum(self._h, T, _bf16(X, "X"), _bf16(y, "y"), _stream(stream)),
               "xhc_stream_sum")
        return y

    # ---- sequence split: halo rows between consecutive chunks of the same sequences ----

    def halo_rows(self) -> int:
        """R = max(kappa) - 1 (0 without a conv)."""
        return max(self.cfg.conv_k) - 1 if self.cfg.conv_k else 0

    def halo_fill(self, B: int, S: int, out, halo=None, stream=None):
        """The halo [B, R, C] bf16 that the next chunk of these B sequences (S tokens each here)
        needs from this chunk's sublayer output ``out``."""
        if halo is None:
            halo = torch.empty(B, self.halo_rows(), self.cfg.C, dtype=torch.bfloat16, device=out.device)
        _check(lib().xhc_halo_fill(self._h, B, S, _bf16(out, "out"), _bf16(halo, "halo"), _stream(stream)),
               "xhc_halo_fill")
        return halo

    def halo_add(self, B: int, S: int, d_out, d_halo, stream=None):
        """d_out of this chunk's last R tokens += the next chunk's d_halo (fp32 [B, R, C])."""
        if d_halo.dtype != torch.float32 or not d_halo.is_cuda or not d_halo.is_contiguous():
            raise XhcError("d_halo must be a contiguous fp32 CUDA tensor")
        _check(lib().xhc_halo_add(self._h, B, S, _bf16(d_out, "d_out"), _ptr(d_halo), _stream(stream)),
               "xhc_halo_add")

    def pre_bwd(self, slot, P, X, d_input, dX, grads, saved, ws, stream=None):
        T = X.shape[0]
        pp = P if isinstance(P, _Params) else self.params(P)
        gg = grads if isinstance(grads, _Params) else self.params(grads)
        _check(lib().xhc_pre_bwd(self._h, slot, T, ctypes.byref(pp), _bf16(X, "X"),
                                 _bf16(d_input, "d_input"), _bf16(dX, "dX"), ctypes.byref(gg),
                                 _ptr(saved), _ptr(ws), _stream(stream)), f"xhc_pre_bwd({slot})")

    # convenience: the whole group with caller-supplied sublayer outputs / gradients

    def forward(self, P, X, outs, saved, ws, inputs=None, stream=None):
        """Runs pre_fwd/post_fwd for every slot; X is updated in place.  Returns the inputs."""
        T, C = X.shape[0], self.cfg.C
        if inputs is None:
            inputs = [torch.empty(T, C, dtype=torch.bfloat16, device=X.device) for _ in range(self.cfg.G)]
        pp = self.params(P)
        for t in range(self.cfg.G):
            self.pre_fwd(t, pp, X, inputs[t], saved, ws, stream)
            self.post_fwd(t, pp, X, outs[t], saved, ws, stream)
        return inputs

    # ---- decoding: one new token per sequence (see xhc_post_fwd_decode) ----

    def ring_bytes(self, B: int) -> int:
        n = ctypes.c_size_t()
        _check(lib().xhc_ring_bytes(self._h, B, ctypes.byref(n)), "xhc_ring_bytes")
        return n.value

    def alloc_rings(self, B: int, device="cuda") -> list:
        """One conv-history ring per slot (None for a slot without a conv)."""
        n = self.ring_bytes(B)
        return [torch.zeros(n, dtype=torch.uint8, device=device) if (n and self.cfg.K(t) > 1) else None
                for t in range(self.cfg.G)]

    def ring_fill(self, B: int, S: int, out, ring, stream=None):
        """After a prefill of B sequences of S tokens: the last rows of each sequence's `out`."""
        _check(lib().xhc_ring_fill(self._h, B, S, _bf16(out, "out"), _ptr(ring), _stream(stream)),
               "xhc_ring_fill")

    def post_fwd_decode(self, slot, P, X, out, ring, pos, saved, ws, stream=None):
        B = X.shape[0]
        pp = P if isinstance(P, _Params) else self.params(P)
        if pos.dtype != torch.int64 or not pos.is_cuda or not pos.is_contiguous():
            raise XhcError("pos must be a contiguous int64 CUDA tensor")
        _check(lib().xhc_post_fwd_decode(self._h, slot, B, ctypes.byref(pp), _bf16(X, "X"), _bf16(out, "out"),
                                         _ptr(ring), _ptr(pos), _ptr(saved), _ptr(ws), _stream(stream)),
               f"xhc_post_fwd_decode({slot})")

    def forward_decode(self, P, X, outs, rings, pos, saved, ws, inputs=None, stream=None):
        """One decode step of the group: X [B, N, C] (token b = next token of sequence b, at
        position pos[b]) updated in place; pos advanced by one.  Returns the inputs."""
        B, C = X.shape[0], self.cfg.C
        if inputs is None:
            inputs = [torch.empty(B, C, dtype=torch.bfloat16, device=X.device) for _ in range(self.cfg.G)]
        pp = self.params(P)
        for t in range(self.cfg.G):
            self.pre_fwd(t, pp, X, inputs[t], saved, ws, stream)
            self.post_fwd_decode(t, pp, X, outs[t], rings[t], pos, saved, ws, stream)
        return inputs

    def backward(self, P, X, dX, outs, d_inputs, grads, saved, ws, d_outs=None, stream=None):
        """Runs post_bwd/pre_bwd for every slot in reverse; X is restored and dX updated in
        place; grads accumulate.  Returns the d_out tensors."""
        T, C = X.shape[0], self.cfg.C
        if d_outs is None:
            d_outs = [torch.empty(T, C, dtype=torch.bfloat16, device=X.device) for _ in range(self.cfg.G)]
        pp, gg = self.params(P), self.params(grads)
        for t in reversed(range(self.cfg.G)):
            self.post_bwd(t, pp, X, dX, outs[t], d_outs[t], gg, saved, ws, stream)
            self.pre_bwd(t, pp, X, d_inputs[t], dX, gg, saved, ws, stream)
        return d_outs
