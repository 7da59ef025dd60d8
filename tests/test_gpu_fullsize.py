"""Parity at the benchmark's full size, in the launch configuration bench.py times.

The xHC-Flash-4sub group N=16 k=4 m=2 C=4096 runs on T=32768 tokens (8 sequences of 4096) with
the inputs bench.py draws (same generators, same seed), through the same Group calls.  The fp64
oracle cannot run the whole step, so it is checked on windows of L tokens it can compute on its
own: at the start of a sequence, in the middle of one (across a 128-token tile boundary), across
the boundaries of the write-back kernels' token runs (32 / 60 / 64 / 128 / 296 tokens), and the last tokens
of the last sequence (the last tile).  In the full-state projection every token tile is cut by a
stream-K segment boundary (about 860 of its 1024 k-blocks per CTA), so every window covers those
too.

A token's forward depends only on its own state and on the sublayer outputs of the previous
max(kappa) - 1 = 11 tokens of its sequence, so the oracle runs each window with 11 tokens of
context before it (fewer at a sequence start), treating the context's start as a sequence start;
only the window's own tokens are compared.  The upstream gradients (dX and every d_input) are
zero outside the windows, on both sides: then every token outside the windows contributes
exactly nothing to the backward, the full-size parameter gradients equal the sum of the
oracle's gradients over the windows (compared element by element), d_out is comparable on the
windows and their context, and dX must be exactly zero everywhere else.

The kernels' own forward is checked first (the intermediate active states of the window tokens
against the oracle's, up to ambiguous roundings); the comparisons downstream of those states use
a forward into which the oracle's intermediate states of the window tokens are injected."""
import os
import sys

import pytest
import torch

from paper_2607_14530_gb300 import synth
from paper_2607_14530_gb300.xhc import Config, Group

from xhc_cases import (alpha_term_scales, ambiguity_masks, assert_alpha_close, assert_bf16_close,
                       assert_f32_close, check_active_states, flash_bases, run_oracle, tie_free)

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
L = 40           # compared tokens per window
SEED = 1234      # bench.py's seed on rank 0
# (sequence, first token inside the sequence): start; middle across a 128-token tile boundary
# (2048); across a boundary of every write-back run length (888 = 3 x 296 for the backward apply,
# 896 = 7 x 128 = 14 x 64 = 28 x 32 for the forward apply, the backward reductions and the
# conv-free kernels, 900 = 15 x 60 for the Gram kernel); the last L tokens of T
WINDOWS = [(0, 0), (2, 2030), (5, 870), (7, 4096 - L)]


def _workload():
    sys.path.insert(0, ROOT)
    import bench
    _, cfg, T = bench.workloads()["flash4"]
    return cfg, T


def _window_cfg(cfg: Config, n: int) -> Config:
    return Config.flash(cfg.N, cfg.k, cfg.m, cfg.C, cfg.G, conv_k=tuple(cfg.conv_k), seq_len=n)


def test_fullsize_windows_parity():
    cfg, T = _workload()
    S = cfg.seq_len
    ctx = max(cfg.conv_k) - 1
    dev = torch.device("cuda", 0)
    # the bench's inputs
    X = synth.normal_bf16_on((T, cfg.N, cfg.C), SEED, dev)
    outs = [synth.normal_bf16_on((T, cfg.C), SEED + 101 + t, dev) for t in range(cfg.G)]
    dX0 = synth.normal_bf16_on((T, cfg.N, cfg.C), SEED + 7, dev)
    dins = [synth.normal_bf16_on((T, cfg.C), SEED + 211 + t, dev) for t in range(cfg.G)]
    P = synth.params(cfg.param_shapes(), SEED)
    Pd = {n: v.to(dev) for n, v in P.items()}

    # windows without a near tie in the routing of their tokens (the oracle decides; a tie would
    # let either selection be correct): shifted forward by a token until there is none
    wins = []
    for b, s0 in WINDOWS:
        for shift in range(64):
            s = min(s0 + shift, S - L) if s0 + L < S else s0 - shift
            a = max(0, s - ctx)
            rows = torch.arange(b * S + a, b * S + s + L)
            x = X[rows.to(dev)].cpu()
            if bool(tie_free(cfg, x[s - a:], P["W_r"]).all()):
                wins.append(dict(b=b, s=s, a=a, rows=rows, own=s - a, x=x))
                break
        else:
            raise AssertionError(f"no tie-free window near sequence {b} token {s0}")

    # upstream gradients zero outside the windows
    keep = torch.zeros(T, dtype=torch.bool)
    for w in wins:
        keep[w["rows"][w["own"]:]] = True
    kd = keep.to(dev)
    dX0 = dX0 * kd[:, None, None].to(dX0.dtype)
    dins = [d * kd[:, None].to(d.dtype) for d in dins]

    refs = []
    for w in wins:
        r = w["rows"].to(dev)
        n = len(w["rows"])
        inp = dict(X=w["x"], outs=[o[r].cpu() for o in outs])
        gin = dict(dX=dX0[r].cpu(), d_inputs=[d[r].cpu() for d in dins])
        wcfg = _window_cfg(cfg, n)
        ref = run_oracle(wcfg, inp, P, gin)
        ref["scales"] = alpha_term_scales(wcfg, inp, P, gin)
        ref["cfg"] = wcfg
        refs.append(ref)

    g = Group(cfg)
    saved, ws = g.alloc(T, device=dev)
    inputs = [torch.empty(T, cfg.C, dtype=torch.bfloat16, device=dev) for _ in range(cfg.G)]
    d_outs = [torch.empty(T, cfg.C, dtype=torch.bfloat16, device=dev) for _ in range(cfg.G)]
    X0 = X.clone()
    errors = []

    def chk(fn, *a):
        try:
            fn(*a)
        except AssertionError as e:
            errors.append(str(e).split("\n")[0])

    def forward(inject):
        X.copy_(X0)
        pp = g.params(Pd)
        xact = g.coefficients(saved, T)["xact"]
        for t in range(cfg.G):
            if inject and t >= 1:
                for w, ref in zip(wins, refs):
                    own = w["rows"][w["own"]:].to(dev)
                    xact[t][own] = ref["aux"]["X_act"][t][w["own"]:].to(torch.bfloat16).to(dev)
            g.pre_fwd(t, pp, X, inputs[t], saved, ws)
            g.post_fwd(t, pp, X, outs[t], saved, ws)
        torch.cuda.synchronize()

    # the kernels' own forward: intermediate active states of the window tokens
    forward(False)
    xact = g.coefficients(saved, T)["xact"]
    for w, ref in zip(wins, refs):
        own = w["rows"][w["own"]:].to(dev)
        aux = {k: v for k, v in ref["aux"].items()}
        aux["X_act"] = [v[w["own"]:] for v in ref["aux"]["X_act"]]
        aux["pre"] = {t: v[w["own"]:] for t, v in ref["aux"]["pre"].items()}
        aux["mag"] = {t: v[w["own"]:] for t, v in ref["aux"]["mag"].items()}
        masks = {t: m[w["own"]:] for t, m in ambiguity_masks(ref["cfg"], ref["aux"]).items()}
        errors += check_active_states([x[own] for x in xact], aux, masks, cfg, f"seq {w['b']}@{w['s']} own: ")

    def step(grads):
        forward(True)
        co = g.coefficients(saved, T)
        fwd = dict(X=[X[w["rows"].to(dev)].cpu() for w in wins],
                   inputs=[[i[w["rows"].to(dev)].cpu() for i in inputs] for w in wins],
                   co={n: (v.cpu() if torch.is_tensor(v) else [u.cpu() for u in v])
                       for n, v in co.items() if n != "xact"})
        dX = dX0.clone()
        g.backward(Pd, X, dX, outs, dins, grads, saved, ws, d_outs=d_outs)
        torch.cuda.synchronize()
        return fwd, dX

    grads = [{n: torch.zeros_like(v) for n, v in Pd.items()} for _ in range(2)]
    fwd, dX = step(grads[0])
    assert g.device_error(ws) == 0, "a bounded device wait gave up"

    near = torch.zeros(T, dtype=torch.bool)
    for w, ref in zip(wins, refs):
        aux = ref["aux"]
        o = w["own"]
        rows = w["rows"]
        own = rows[o:]
        tag = f"seq {w['b']}@{w['s']}"
        near[rows] = True
        bases = flash_bases(cfg, w["x"], aux)
        if not torch.equal(fwd["co"]["I"][own].long(), aux["I"][o:]):
            errors.append(f"{tag}: routing differs")
        chk(assert_f32_close, fwd["co"]["p"][own], aux["p"][o:], f"{tag} p")
        for t in range(cfg.G):
            chk(assert_f32_close, fwd["co"]["hpre"][own][:, t], aux["H_pre"][t][o:], f"{tag} H_pre[{t}]")
            chk(assert_f32_close, fwd["co"]["hpost"][t][own], aux["H_post"][t][o:], f"{tag} H_post[{t}]")
            chk(assert_bf16_close, fwd["inputs"][wins.index(w)][t][o:], ref["inputs"][t][o:], f"{tag} input[{t}]",
                None if bases[t] is None else bases[t][o:])
        chk(assert_f32_close, fwd["co"]["hres"][own], aux["H_res"][o:], f"{tag} H_res")
        chk(assert_bf16_close, fwd["X"][wins.index(w)][o:], ref["X"][o:], f"{tag} X_out")
        r = rows.to(dev)
        if not torch.equal(X[r].cpu(), w["x"]):
            errors.append(f"{tag}: X not restored to the entry state")
        chk(assert_bf16_close, dX[r].cpu()[o:], ref["dX"][o:], f"{tag} dX")
        for t in range(cfg.G):
            # d_out of the context tokens gets the window's conv-transpose terms on both sides
            chk(assert_bf16_close, d_outs[t][r].cpu(), ref["d_outs"][t], f"{tag} d_out[{t}]")
    # nothing outside the windows receives a gradient
    far = (~keep).to(dev)
    if bool((dX[far] != 0).any()):
        errors.append("dX nonzero outside the windows")
    for t in range(cfg.G):
        if bool((d_outs[t][(~near).to(dev)] != 0).any()):
            errors.append(f"d_out[{t}] nonzero outside the windows and their context")

    # the parameter gradients of the whole run are the oracle's sums over the windows
    for n, v in grads[0].items():
        want = sum(ref["dP"][n] for ref in refs)
        if n.startswith("alpha"):
            chk(assert_alpha_close, v, want, sum(ref["scales"][n] for ref in refs), f"grad {n}")
        else:
            chk(assert_f32_close, v, want, f"grad {n}")
    assert not errors, "\n".join(errors)

    # and the same bits on a second run
    step(grads[1])
    for n in grads[0]:
        assert torch.equal(grads[0][n], grads[1][n]), f"grad {n} not deterministic"
