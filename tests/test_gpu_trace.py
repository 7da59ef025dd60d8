"""The library's tracing and stream debugging entry points on the GPU: xhc_trace_only restricts
the recorded launches to the named kernels, xhc_trace_span places every record on one timeline,
and XHC_DEBUG_ONE_STREAM (the side-stream work run on the caller's stream) gives results that are
bit-identical to the two-stream schedule."""
import pytest
import torch

from paper_2607_14530_gb300 import synth, xhc
from paper_2607_14530_gb300.xhc import Config, Group

pytestmark = pytest.mark.gpu

CFG = Config.flash(16, 4, 2, 256, 4, seq_len=128)
T = 256


def _setup(seed=5):
    dev = torch.device("cuda", 0)
    g = Group(CFG)
    X = synth.normal_bf16_on((T, CFG.N, CFG.C), seed, dev)
    outs = [synth.normal_bf16_on((T, CFG.C), seed + 101 + t, dev) for t in range(CFG.G)]
    dX = synth.normal_bf16_on((T, CFG.N, CFG.C), seed + 7, dev)
    dins = [synth.normal_bf16_on((T, CFG.C), seed + 211 + t, dev) for t in range(CFG.G)]
    P = {n: v.to(dev) for n, v in synth.params(CFG.param_shapes(), seed).items()}
    return g, X, outs, dX, dins, P


def _step(g, X, outs, dX, dins, P):
    G_ = {n: torch.zeros_like(v) for n, v in P.items()}
    saved, ws = g.alloc(T)
    inputs = g.forward(P, X, outs, saved, ws)
    d_outs = g.backward(P, X, dX, outs, dins, G_, saved, ws)
    torch.cuda.synchronize()
    return inputs, d_outs, G_


def test_trace_only_and_spans():
    g, X, outs, dX, dins, P = _setup()
    try:
        xhc.trace_only(None)
        xhc.trace_enable(True)
        _step(g, X, outs, dX.clone(), dins, P)
        xhc.trace_enable(False)
        names = [n for n, _ in xhc.trace_records()]
        assert "dxa_tc" in names and "read" in names and len(set(names)) > 5
        spans = xhc.trace_spans()
        assert len(spans) == len(names) and spans[0][1] == 0.0
        assert all(t0 >= 0.0 and ms >= 0.0 for _, t0, ms in spans)

        xhc.trace_only(["dxa_tc", "read"])
        xhc.trace_enable(True)
        _step(g, X, outs, dX.clone(), dins, P)
        xhc.trace_enable(False)
        kept = [n for n, _ in xhc.trace_records()]
        assert sorted(set(kept)) == ["dxa_tc", "read"]
        assert kept.count("dxa_tc") == names.count("dxa_tc") and kept.count("read") == names.count("read")
    finally:
        xhc.trace_enable(False)
        xhc.trace_only(None)


def test_one_stream_matches_two_streams():
    g, X, outs, dX, dins, P = _setup(seed=9)
    X0 = X.clone()
    res = []
    try:
        for one in (False, True):
            xhc.debug_one_stream(one)
            Xr, dXr = X0.clone(), dX.clone()
            inputs, d_outs, G_ = _step(g, Xr, outs, dXr, dins, P)
            res.append((inputs, d_outs, G_, dXr, Xr))
    finally:
        xhc.debug_one_stream(False)
    (i0, o0, g0, d0, x0), (i1, o1, g1, d1, x1) = res
    assert all(torch.equal(a, b) for a, b in zip(i0, i1))
    assert all(torch.equal(a, b) for a, b in zip(o0, o1))
    assert torch.equal(d0, d1) and torch.equal(x0, x1) and torch.equal(x0, X0)
    for n in g0:
        assert torch.equal(g0[n], g1[n]), n
