"""Host-side checks of the libxhc C ABI (no GPU needed, no compute call is made).

The library builds for sm_103a here, loads, exports every function include/xhc.h declares, and
rejects bad configurations and arguments on the host with the documented status codes before
anything is enqueued on a device."""
import ctypes
import os
import re

import pytest

from paper_2607_14530_gb300 import build
from paper_2607_14530_gb300 import xhc as X

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
OK, INVALID, UNSUPPORTED, ALIGN = 0, 1, 2, 3


@pytest.fixture(scope="module")
def L():
    build.build()
    return X.lib()


def test_exports_every_declared_function(L):
    hdr = open(os.path.join(ROOT, "include", "xhc.h")).read()
    names = sorted(set(re.findall(r"^\s*(?:xhc_status|void|int|const char\*)\s+(xhc_\w+)\s*\(", hdr, re.M)))
    assert len(names) >= 10, names
    for n in names:
        assert hasattr(L, n), f"{n} not exported"
    assert L.xhc_version() == 200


def _create(cfg):
    h = ctypes.c_void_p()
    st = X.lib().xhc_create(ctypes.byref(cfg._c()), ctypes.byref(h))
    if st == OK:
        X.lib().xhc_destroy(h)
    return st


def test_create_accepts_paper_configs(L):
    assert _create(X.Config.full(16, 4, 2, 2048, True)) == OK
    assert _create(X.Config.full(16, 4, 2, 2048, False)) == OK
    assert _create(X.Config.mhc(4, 2048)) == OK
    assert _create(X.Config.flash(16, 4, 2, 4096, 4)) == OK
    assert _create(X.Config.flash(16, 4, 2, 4096, 2)) == OK
    assert _create(X.Config.flash(32, 4, 2, 4096, 4)) == OK
    # ablations: softmax router, sparse read, attention-side temporal augmentation
    assert _create(X.Config.full(16, 4, 2, 2048, True, router="softmax")) == OK
    assert _create(X.Config.full(16, 4, 0, 2048, False, sparse_read=True)) == OK
    assert _create(X.Config.flash(16, 4, 2, 4096, 4, attn_tfa=True)) == OK


def test_create_rejects_unknown_ablation_codes(L):
    c = X.Config.full(16, 4, 2, 256, True)._c()
    for field, bad in (("router", 2), ("router", -1), ("sparse_read", 2)):
        cc = X._Config.from_buffer_copy(c)
        setattr(cc, field, bad)
        h = ctypes.c_void_p()
        assert L.xhc_create(ctypes.byref(cc), ctypes.byref(h)) == INVALID, field


@pytest.mark.parametrize("cfg,want", [
    (X.Config(X.FULL, 16, 4, 5, 256), INVALID),                     # m > k
    (X.Config(X.FULL, 4, 5, 2, 256), INVALID),                      # k > N
    (X.Config(X.FULL, 16, 4, 2, 256, G=2), INVALID),                # FULL needs G = 1
    (X.Config(X.MHC, 4, 4, 2, 256), INVALID),                       # MHC needs m = k = N
    (X.Config(X.FLASH, 16, 4, 2, 256, G=3, mlp_mask=0x2), INVALID), # FLASH needs G in {2, 4}
    (X.Config(X.FLASH, 16, 4, 2, 256, G=4, mlp_mask=0x5), INVALID), # slots must be A, M, A, M
    (X.Config(X.FULL, 16, 4, 2, 256, mlp_mask=0x2), INVALID),       # mask beyond G
    (X.Config(X.FULL, 16, 4, 2, 260), UNSUPPORTED),                 # C % 8
    (X.Config(X.FULL, 33, 4, 2, 256), UNSUPPORTED),                 # N > 32
    (X.Config(X.FULL, 16, 9, 2, 256), UNSUPPORTED),                 # k > 8
    (X.Config(X.FULL, 16, 4, 2, 256, mlp_mask=1, conv_k=(4, 8, 17)), UNSUPPORTED),
    (X.Config(X.FULL, 16, 4, 2, 256, eps_norm=0.0), INVALID),
    (X.Config(X.FLASH, 16, 4, 2, 256, G=8, mlp_mask=0xAA), UNSUPPORTED),
])
def test_create_rejects(L, cfg, want):
    assert _create(cfg) == want


def test_sizes_grow_with_T(L):
    g = X.Group(X.Config.flash(16, 4, 2, 4096, 4))
    s1, s2 = g.saved_bytes(512), g.saved_bytes(1024)
    w1, w2 = g.workspace_bytes(512), g.workspace_bytes(1024)
    assert 0 < s1 < s2 and 0 < w1 < w2
    # saved holds at least the G active-state copies: G*T*k*C bf16
    assert s1 >= 4 * 512 * 4 * 4096 * 2


def test_entry_points_validate_on_host(L):
    cfg = X.Config.full(8, 4, 2, 64, True)
    g = X.Group(cfg)
    fake = {n: None for n in cfg.param_shapes()}
    P = X._Params()
    # fake 16-byte aligned device addresses: never dereferenced, validation happens first
    addr = [0x7f0000000000 + 4096 * i for i in range(64)]
    P.W_r = addr[0]
    P.W_pre[0] = addr[1]
    P.alpha_pre = addr[2]
    P.b_pre = addr[3]
    P.W_post[0] = addr[4]
    P.alpha_post = addr[5]
    P.b_post[0] = addr[6]
    P.W_res = addr[7]
    P.alpha_res = addr[8]
    P.b_res = addr[9]
    for j in range(3):
        P.conv_w[0][j] = addr[10 + j]
    sv, ws, Xp, inp = addr[20], addr[21], addr[22], addr[23]
    h = g._h
    assert L.xhc_pre_fwd(None, 0, 64, ctypes.byref(P), Xp, inp, sv, ws, None) == INVALID
    assert L.xhc_pre_fwd(h, 1, 64, ctypes.byref(P), Xp, inp, sv, ws, None) == INVALID  # slot >= G
    assert L.xhc_pre_fwd(h, 0, 0, ctypes.byref(P), Xp, inp, sv, ws, None) == INVALID   # T = 0
    assert L.xhc_pre_fwd(h, 0, 64, ctypes.byref(P), None, inp, sv, ws, None) == INVALID
    assert L.xhc_pre_fwd(h, 0, 64, ctypes.byref(P), Xp + 2, inp, sv, ws, None) == ALIGN
    assert L.xhc_pre_fwd(h, 0, 64, ctypes.byref(P), Xp, inp, sv + 8, ws, None) == ALIGN
    P2 = X._Params()
    ctypes.memmove(ctypes.byref(P2), ctypes.byref(P), ctypes.sizeof(P))
    P2.W_res = None
    assert L.xhc_pre_fwd(h, 0, 64, ctypes.byref(P2), Xp, inp, sv, ws, None) == INVALID
    P2.W_res = addr[7]
    P2.conv_w[0][2] = None
    assert L.xhc_post_fwd(h, 0, 64, ctypes.byref(P2), Xp, inp, sv, ws, None) == INVALID
    # grads struct missing W_post gradient
    Gd = X._Params()
    ctypes.memmove(ctypes.byref(Gd), ctypes.byref(P), ctypes.sizeof(P))
    Gd.W_post[0] = None
    assert L.xhc_post_bwd(h, 0, 64, ctypes.byref(P), Xp, addr[30], inp, addr[31], ctypes.byref(Gd),
                          sv, ws, None) == INVALID
    # decode entry points: sizes, and validation before any launch
    sz = ctypes.c_size_t()
    assert L.xhc_ring_bytes(h, 4, ctypes.byref(sz)) == 0 and sz.value == 4 * 11 * 64 * 2
    assert L.xhc_ring_bytes(h, 0, ctypes.byref(sz)) == INVALID
    ring, pos = addr[33], addr[34]
    assert L.xhc_post_fwd_decode(h, 0, 64, ctypes.byref(P), Xp, inp, None, pos, sv, ws, None) == INVALID
    assert L.xhc_post_fwd_decode(h, 0, 64, ctypes.byref(P), Xp, inp, ring, None, sv, ws, None) == INVALID
    assert L.xhc_post_fwd_decode(h, 0, 64, ctypes.byref(P), Xp, inp, ring + 4, pos, sv, ws, None) == ALIGN
    assert L.xhc_ring_fill(h, 4, 0, inp, ring, None) == INVALID
    assert L.xhc_ring_fill(h, 4, 16, inp + 2, ring, None) == ALIGN
    # sequence length must divide T
    g2 = X.Group(X.Config.full(8, 4, 2, 64, True, seq_len=48))
    assert L.xhc_pre_fwd(g2._h, 0, 64, ctypes.byref(P), Xp, inp, sv, ws, None) == INVALID
    assert L.xhc_status_string(3) == b"pointer not 16-byte aligned"


def test_route_noalloc_rejects_oversized_T(L):
    """xhc_route_noalloc checks T against its fixed scratch array on the host, before any device
    work (the pointers below are never dereferenced)."""
    g = X.Group(X.Config.flash(32, 4, 2, 4096, 4))
    T = 1 << 20
    P = X._Params()
    for i in range(4):
        P.W_pre[i] = 0x7f0000000000 + 4096 * i
    P.W_r, P.alpha_pre, P.b_pre = 0x7f0000100000, 0x7f0000200000, 0x7f0000300000
    addr = 0x7f0001000000
    st = L.xhc_route_noalloc(g._h, T, ctypes.byref(P), addr, addr, addr, addr, None)
    assert st == UNSUPPORTED


def test_debug_hook_argument_checks(L):
    assert L.xhc_debug_set(1, -5) == INVALID
    assert L.xhc_debug_set(99, 0) == INVALID
    assert L.xhc_debug_set(1, 0) == OK
    assert L.xhc_debug_set(2, 0) == OK
    assert L.xhc_debug_set(3, 1) == OK    # side-stream work on the caller's stream
    assert L.xhc_debug_set(3, 0) == OK


def test_trace_filter_and_records_on_host(L):
    """The trace filter parses its name list on the host; with nothing recorded, every record
    index is out of range (no CUDA call is made)."""
    name, ms, t0 = ctypes.c_char_p(), ctypes.c_float(), ctypes.c_float()
    try:
        assert L.xhc_trace_only(b" dxa_tc, read,,dots_act ") == OK
        assert L.xhc_trace_only(b"") == OK
        assert L.xhc_trace_only(None) == OK
        assert L.xhc_trace_enable(1) == OK       # drops the previous records
        assert L.xhc_trace_count() == 0
        assert L.xhc_trace_record(0, ctypes.byref(name), ctypes.byref(ms)) == INVALID
        assert L.xhc_trace_span(0, ctypes.byref(name), ctypes.byref(t0), ctypes.byref(ms)) == INVALID
        assert L.xhc_trace_span(-1, ctypes.byref(name), ctypes.byref(t0), ctypes.byref(ms)) == INVALID
        assert L.xhc_trace_span(0, None, None, None) == INVALID
    finally:
        L.xhc_trace_enable(0)
        L.xhc_trace_only(None)
