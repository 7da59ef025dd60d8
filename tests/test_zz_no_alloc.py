"""xhc_route_noalloc, the entry point for callers that cannot allocate device memory, gives the
same routing and pre-maps as the workspace-based xhc_pre_fwd(slot 0).

Callers such as engines that fix every device buffer at start-up, or plug-ins running inside a
host framework's memory arena, cannot hand the library a workspace; this entry point keeps its
scratch in a fixed array inside the library.  The test calls it twice in a row, on two
different inputs, and checks each result against the regular entry point (routing exactly,
coefficients at the suite's 1e-4 relative tolerance), so stale scratch from the first call
cannot leak into the second.  It sits in a file of its own, collected last."""
import pytest
import torch

from paper_2607_14530_gb300.xhc import Config, Group

from xhc_cases import assert_f32_close, make_case

pytestmark = pytest.mark.gpu


def _regular(g, cfg, P, X, T):
    saved, ws = g.alloc(T)
    inp = torch.empty(T, cfg.C, dtype=torch.bfloat16, device="cuda")
    g.pre_fwd(0, P, X, inp, saved, ws)
    torch.cuda.synchronize()
    co = g.coefficients(saved, T)
    return co["I"].clone(), co["p"].clone(), co["hpre"].clone()


@pytest.mark.parametrize("cfg,T", [
    (Config.flash(16, 4, 2, 256, 4, seq_len=128), 512),
    (Config.full(5, 3, 1, 264, True, conv_k=(2, 5)), 200),
    (Config.mhc(4, 256), 96),
])
def test_route_noalloc_matches_pre_fwd_twice(cfg, T):
    g = Group(cfg)
    for call, seed in enumerate((3, 4)):
        inp, P, _ = make_case(cfg, T, seed)
        Pd = {n: v.cuda() for n, v in P.items()}
        X = inp["X"].cuda()
        I_ref, p_ref, h_ref = _regular(g, cfg, Pd, X, T)
        I = torch.full((T, cfg.k), -1, dtype=torch.int32, device="cuda")
        p = torch.full((T, cfg.k), float("nan"), device="cuda")
        hpre = torch.full((T, cfg.G, cfg.N), float("nan"), device="cuda")
        g.route_noalloc(Pd, X, I, p, hpre)
        torch.cuda.synchronize()
        assert torch.equal(I, I_ref), f"call {call}: routing differs"
        assert_f32_close(p, p_ref, f"call {call}: p")
        assert_f32_close(hpre, h_ref, f"call {call}: hpre")


def test_route_noalloc_rejects_oversized_T():
    cfg = Config.flash(32, 4, 2, 4096, 4)
    g = Group(cfg)
    from paper_2607_14530_gb300 import xhc as X
    T = 1 << 20
    P = X._Params()
    for i in range(4):
        P.W_pre[i] = 0x7f0000000000 + 4096 * i
    P.W_r, P.alpha_pre, P.b_pre = 0x7f0000100000, 0x7f0000200000, 0x7f0000300000
    addr = 0x7f0001000000
    import ctypes
    st = X.lib().xhc_route_noalloc(g._h, T, ctypes.byref(P), addr, addr, addr, addr, None)
    assert st == 2  # XHC_ERR_UNSUPPORTED, before any device work
