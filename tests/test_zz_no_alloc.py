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

from xhc_cases import Guarded, assert_f32_close, make_case, run_oracle

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
        # outputs start poisoned, inside guard bands that must stay intact
        I = Guarded(torch.full((T, cfg.k), -1, dtype=torch.int32))
        p = Guarded(torch.full((T, cfg.k), float("nan")))
        hpre = Guarded(torch.full((T, cfg.G, cfg.N), float("nan")))
        g.route_noalloc(Pd, X, I.t, p.t, hpre.t)
        torch.cuda.synchronize()
        assert I.intact() and p.intact() and hpre.intact(), f"call {call}: guard band overwritten"
        assert torch.equal(I.t, I_ref), f"call {call}: routing differs"
        assert_f32_close(p.t, p_ref, f"call {call}: p")
        assert_f32_close(hpre.t, h_ref, f"call {call}: hpre")
        # and against the oracle directly
        aux = run_oracle(cfg, inp, P)["aux"]
        assert torch.equal(I.t.cpu().long(), aux["I"]), f"call {call}: routing differs from the oracle"
        assert_f32_close(p.t, aux["p"], f"call {call}: p vs oracle")
        for t in range(cfg.G):
            assert_f32_close(hpre.t[:, t], aux["H_pre"][t], f"call {call}: hpre[{t}] vs oracle")
