"""The test helpers' per-term alpha contributions sum to the oracle's scalar alpha gradients."""
import torch

from paper_2607_14530_gb300 import synth
from paper_2607_14530_gb300.xhc import Config
from xhc_cases import make_case, run_oracle

F64 = torch.float64


def test_alpha_terms_sum_to_the_gradient():
    from oracle import xhc_oracle as O
    from xhc_cases import oracle_cfg
    cfg = Config.flash(6, 3, 1, 16, 4, conv_k=(2, 3), seq_len=8)
    T = 16
    inp, P, s = make_case(cfg, T, 0, alpha=0.3, w_std=0.2)
    gi = synth.group_grads(T, cfg.N, cfg.C, cfg.G, s)
    ref = run_oracle(cfg, inp, P, gi)
    ocfg = oracle_cfg(cfg)
    P64 = {n: v.to(F64) for n, v in P.items()}
    a_res = torch.full((1, T, cfg.k, cfg.k), float(P64["alpha_res"][0]), dtype=F64, requires_grad=True)
    a_post = [torch.full((T, cfg.k, cfg.K(t)), float(P64["alpha_post"][t]), dtype=F64, requires_grad=True)
              for t in range(cfg.G)]
    a_pre = [torch.full((T, cfg.N), float(P64["alpha_pre"][t]), dtype=F64, requires_grad=True)
             for t in range(cfg.G)]
    Pp = dict(P64)
    Pp["alpha_res"], Pp["alpha_post"], Pp["alpha_pre"] = a_res, a_post, a_pre
    Xo, ins, _ = O.forward(ocfg, Pp, inp["X"].to(F64), [o.to(F64) for o in inp["outs"]])
    L = (Xo * gi["dX"].to(F64)).sum() + sum((a * d.to(F64)).sum() for a, d in zip(ins, gi["d_inputs"]))
    g = torch.autograd.grad(L, a_pre + a_post + [a_res])
    for t in range(cfg.G):
        assert torch.allclose(g[t].sum(), ref["dP"]["alpha_pre"][t], rtol=1e-10, atol=1e-12)
        assert torch.allclose(g[cfg.G + t].sum(), ref["dP"]["alpha_post"][t], rtol=1e-10, atol=1e-12)
    assert torch.allclose(g[-1].sum(), ref["dP"]["alpha_res"][0], rtol=1e-10, atol=1e-12)
