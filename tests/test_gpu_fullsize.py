"""Parity at the benchmark's full size, in the launch configuration bench.py times.

The xHC-Flash-4sub group N=16 k=4 m=2 C=4096 runs on T=32768 tokens (8 sequences of 4096) with
the inputs bench.py draws (same generators, same seed), through the same Group calls.  The fp64
oracle cannot run the whole step, so it is checked on samples it can compute on its own: the
first TS tokens of two sequences.  Everything of a token depends only on that token and the
earlier tokens of its sequence (the conv is causal and restarts at each sequence start), except
d_out, whose transposed conv reaches max(kappa) - 1 tokens ahead: d_out is compared on the first
TS - (max(kappa) - 1) tokens of each sample.  The parameter gradients sum over all T tokens and
are checked through properties that hold at any size: finite, and bit-identical over two runs."""
import os
import sys

import pytest
import torch

from oracle import xhc_oracle as O
from paper_2607_14530_gb300 import synth
from paper_2607_14530_gb300.xhc import Config, Group

from xhc_cases import F64, TIE_MARGIN, assert_bf16_close, assert_f32_close, oracle_cfg, run_oracle

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
TS = 40          # sampled tokens at the start of a sequence
SEED = 1234      # bench.py's seed on rank 0


def _workload():
    sys.path.insert(0, ROOT)
    import bench
    _, cfg, T = bench.workloads()["flash4"]
    return cfg, T


def _sample_cfg(cfg: Config) -> Config:
    return Config.flash(cfg.N, cfg.k, cfg.m, cfg.C, cfg.G, conv_k=tuple(cfg.conv_k), seq_len=TS)


def test_fullsize_sampled_parity():
    cfg, T = _workload()
    S = cfg.seq_len
    dev = torch.device("cuda", 0)
    # the bench's inputs
    X = synth.normal_bf16_on((T, cfg.N, cfg.C), SEED, dev)
    outs = [synth.normal_bf16_on((T, cfg.C), SEED + 101 + t, dev) for t in range(cfg.G)]
    dX0 = synth.normal_bf16_on((T, cfg.N, cfg.C), SEED + 7, dev)
    dins = [synth.normal_bf16_on((T, cfg.C), SEED + 211 + t, dev) for t in range(cfg.G)]
    P = synth.params(cfg.param_shapes(), SEED)
    Pd = {n: v.to(dev) for n, v in P.items()}

    # samples: the first TS tokens of the first two sequences without a near tie in their routing
    # (the oracle decides; a tie would let either selection be correct)
    scfg = _sample_cfg(cfg)
    ocfg = oracle_cfg(scfg)
    samples = []
    for b in range(T // S):
        rows = torch.arange(b * S, b * S + TS)
        x = X[rows.to(dev)].cpu()
        sc = O.router_scores(ocfg, x.to(F64).reshape(TS, -1), P["W_r"].to(F64))
        if bool((O.routing_margin(ocfg, sc) > TIE_MARGIN).all()):
            samples.append((b, rows, x))
        if len(samples) == 2:
            break
    assert len(samples) == 2, "no tie-free sample"

    refs = []
    for b, rows, x in samples:
        r = rows.to(dev)
        inp = dict(X=x, outs=[o[r].cpu() for o in outs])
        gin = dict(dX=dX0[r].cpu(), d_inputs=[d[r].cpu() for d in dins])
        refs.append(run_oracle(scfg, inp, P, gin))

    g = Group(cfg)
    saved, ws = g.alloc(T, device=dev)
    inputs = [torch.empty(T, cfg.C, dtype=torch.bfloat16, device=dev) for _ in range(cfg.G)]
    d_outs = [torch.empty(T, cfg.C, dtype=torch.bfloat16, device=dev) for _ in range(cfg.G)]

    def step(grads):
        dX = dX0.clone()
        g.forward(Pd, X, outs, saved, ws, inputs=inputs)
        torch.cuda.synchronize()
        fwd = dict(X=[X[rows.to(dev)].cpu() for _, rows, _ in samples],
                   inputs=[[i[rows.to(dev)].cpu() for i in inputs] for _, rows, _ in samples],
                   co=g.coefficients(saved, T))
        fwd["co"] = {n: (v.cpu() if torch.is_tensor(v) else [w.cpu() for w in v])
                     for n, v in fwd["co"].items() if n != "xact"}
        g.backward(Pd, X, dX, outs, dins, grads, saved, ws, d_outs=d_outs)
        torch.cuda.synchronize()
        bwd = dict(dX=[dX[rows.to(dev)].cpu() for _, rows, _ in samples],
                   d_outs=[[d[rows.to(dev)].cpu() for d in d_outs] for _, rows, _ in samples],
                   X=[X[rows.to(dev)].cpu() for _, rows, _ in samples])
        return fwd, bwd

    grads = [{n: torch.zeros_like(v) for n, v in Pd.items()} for _ in range(2)]
    fwd, bwd = step(grads[0])
    assert g.device_error(ws) == 0, "a bounded device wait gave up"

    lag = max(cfg.conv_k) - 1
    errors = []

    def chk(fn, *a):
        try:
            fn(*a)
        except AssertionError as e:
            errors.append(str(e).split("\n")[0])

    for s, ((b, rows, x), ref) in enumerate(zip(samples, refs)):
        aux = ref["aux"]
        tag = f"seq {b}"
        if not torch.equal(fwd["co"]["I"][rows].long(), aux["I"]):
            errors.append(f"{tag}: routing differs")
        chk(assert_f32_close, fwd["co"]["p"][rows], aux["p"], f"{tag} p")
        for t in range(cfg.G):
            chk(assert_f32_close, fwd["co"]["hpre"][rows][:, t], aux["H_pre"][t], f"{tag} H_pre[{t}]")
            chk(assert_f32_close, fwd["co"]["hpost"][t][rows], aux["H_post"][t], f"{tag} H_post[{t}]")
            chk(assert_bf16_close, fwd["inputs"][s][t], ref["inputs"][t], f"{tag} input[{t}]")
        chk(assert_f32_close, fwd["co"]["hres"][rows], aux["H_res"], f"{tag} H_res")
        chk(assert_bf16_close, fwd["X"][s], ref["X"], f"{tag} X_out")
        if not torch.equal(bwd["X"][s], x):
            errors.append(f"{tag}: X not restored to the entry state")
        chk(assert_bf16_close, bwd["dX"][s], ref["dX"], f"{tag} dX")
        for t in range(cfg.G):
            chk(assert_bf16_close, bwd["d_outs"][s][t][:TS - lag], ref["d_outs"][t][:TS - lag],
                f"{tag} d_out[{t}]")
    assert not errors, "\n".join(errors)

    # the parameter gradients: finite, and the same bits on a second run
    step(grads[1])
    for n in grads[0]:
        assert bool(torch.isfinite(grads[0][n]).all()), f"grad {n} not finite"
        assert torch.equal(grads[0][n], grads[1][n]), f"grad {n} not deterministic"
