"""Failure detection of the bounded device waits, without a GPU fault.

The tensor-core kernels wait on mbarriers with a time limit; a wait that runs out sets the
workspace's device error word, the kernel leaves its loops, frees its tensor memory and returns,
and the host reads XHC_ERR_TIMEOUT from xhc_workspace_error.  The test hook
XHC_DEBUG_FORCE_TIMEOUT makes the next full-state projection wait, before it issues any copy or
MMA, for a release that nothing triggers (the first release of its stage 0, which needs an MMA
on a load that was never issued): every role's wait then runs out after the limit (set to
100 ms here), with nothing in flight.  Afterwards the same context runs a whole group, forward
and backward, and matches the oracle."""
import ctypes

import pytest
import torch

from paper_2607_14530_gb300 import synth, xhc
from paper_2607_14530_gb300.xhc import Config, Group

from xhc_cases import assert_bf16_close, assert_f32_close, make_case, run_oracle

pytestmark = pytest.mark.gpu


def test_a_wait_that_runs_out_reports_a_timeout_and_the_context_stays_usable():
    cfg = Config.flash(16, 4, 2, 256, 4, seq_len=128)
    T = 512                      # >= 128 tokens: the tensor-core projection path
    inp, P, seed = make_case(cfg, T, 5)
    gin = synth.group_grads(T, cfg.N, cfg.C, cfg.G, seed)
    g = Group(cfg)
    Pd = {n: v.cuda() for n, v in P.items()}
    saved, ws = g.alloc(T)
    X = inp["X"].cuda()
    first = torch.empty(T, cfg.C, dtype=torch.bfloat16, device="cuda")
    try:
        xhc.debug_wait_limit_ns(100_000_000)
        xhc.debug_force_timeout()
        g.pre_fwd(0, g.params(Pd), X, first, saved, ws)
        torch.cuda.synchronize()
    finally:
        xhc.debug_wait_limit_ns(0)
        xhc.lib().xhc_debug_set(2, 0)
    code = ctypes.c_int()
    st = xhc.lib().xhc_workspace_error(ctypes.c_void_p(ws.data_ptr()), ctypes.byref(code), 1)
    assert st == 5 and code.value != 0, (st, code.value)          # XHC_ERR_TIMEOUT, then cleared
    assert g.device_error(ws) == 0
    assert torch.equal(X.cpu(), inp["X"]), "an aborted pre_fwd must not touch the state"

    # the context is usable: a whole group, forward and backward, on fresh buffers
    ref = run_oracle(cfg, inp, P, gin)
    saved, ws = g.alloc(T)
    X = inp["X"].cuda()
    outs = [o.cuda() for o in inp["outs"]]
    inputs = g.forward(Pd, X, outs, saved, ws)
    dX = gin["dX"].cuda()
    gr = {n: torch.zeros_like(v) for n, v in Pd.items()}
    d_outs = g.backward(Pd, X, dX, outs, [d.cuda() for d in gin["d_inputs"]], gr, saved, ws)
    torch.cuda.synchronize()
    assert g.device_error(ws) == 0
    co = g.coefficients(saved, T)
    assert torch.equal(co["I"].cpu().long(), ref["aux"]["I"])
    assert_f32_close(co["p"], ref["aux"]["p"], "p")
    assert_bf16_close(inputs[0], ref["inputs"][0], "input[0]")
    assert_bf16_close(dX, ref["dX"], "dX")
    for t in range(cfg.G):
        assert_bf16_close(d_outs[t], ref["d_outs"][t], f"d_out[{t}]")
