"""GPU parity of libxhc against the fp64 oracle, element by element, through the C ABI.

Each case runs the whole group forward (pre_fwd / post_fwd for every slot) and backward
(post_bwd / pre_bwd in reverse) on seeded inputs and compares: the sublayer inputs, the new
state, the coefficients (I exactly, p / H_pre / H_post / H_res at 1e-4), dX, every d_out and
every parameter gradient.  Guard bands around the caller buffers must stay intact, inactive
rows must be bit-identical after the forward, and X must hold the entry state again after
the backward.  Shapes span several tiles and ragged tails (T not a multiple of the token tiles,
C not a multiple of the 256-channel slices)."""
import pytest
import torch

from paper_2607_14530_gb300 import synth
from paper_2607_14530_gb300.xhc import Config, Group

from xhc_cases import (Guarded, alpha_term_scales, assert_alpha_close, assert_bf16_close,
                       assert_f32_close, make_case, run_oracle)

pytestmark = pytest.mark.gpu

CASES = {
    # BASELINE config 1 shapes: N=16, k=4, C=256, T=512
    "fullA_N16k4_C256": (Config.full(16, 4, 2, 256, False, seq_len=512), 512, {}),
    "fullM_N16k4_C256": (Config.full(16, 4, 2, 256, True, seq_len=128), 512, {}),
    "flash2_N16k4_C256": (Config.flash(16, 4, 2, 256, 2, seq_len=256), 512, {}),
    "flash4_N16k4_C256": (Config.flash(16, 4, 2, 256, 4, seq_len=128), 512, {}),
    "mhc_N4_C256": (Config.mhc(4, 256), 512, {}),
    # ragged tails, other k / m / N, options
    "fullM_ragged_T200_C264": (Config.full(5, 3, 1, 264, True, conv_k=(2, 5), seq_len=100), 200, {}),
    "fullM_k8": (Config.full(12, 8, 3, 128, True, seq_len=96), 192, {}),
    "flash4_m0": (Config.flash(6, 2, 0, 64, 4, conv_k=(3,)), 72, {}),
    "fullM_no_gs": (Config.full(8, 4, 2, 64, True, gram_schmidt=False), 96, {}),
    "fullM_all_active": (Config.full(4, 4, 2, 64, True, seq_len=16), 48, {}),
    "mhc_N1": (Config.mhc(1, 16), 33, {}),
    "fullM_T1": (Config.full(4, 2, 1, 8, True, conv_k=(2, 3)), 1, {}),
    "fullM_alpha1_stress": (Config.full(16, 4, 2, 256, True, seq_len=256), 256, dict(alpha=1.0)),
}


def _cuda(d):
    return {n: v.cuda().contiguous() for n, v in d.items()}


def run_case(cfg, T, seed=0, alpha=0.01):
    inp, P, seed = make_case(cfg, T, seed, alpha=alpha)
    grads_in = synth.group_grads(T, cfg.N, cfg.C, cfg.G, seed)
    ref = run_oracle(cfg, inp, P, grads_in)

    g = Group(cfg)
    Pd = _cuda(P)
    Xg = Guarded(inp["X"].cuda())
    outs = [Guarded(o.cuda()) for o in inp["outs"]]
    inputs = [Guarded(torch.zeros(T, cfg.C, dtype=torch.bfloat16)) for _ in range(cfg.G)]
    saved, ws = g.alloc(T)
    # saved and workspace start poisoned (0xFF bytes: NaN as fp32 / bf16, -1 as int32), except the
    # workspace's device error word: nothing may be read before this call sequence wrote it
    saved_g = Guarded(torch.full((saved.numel(),), 0xFF, dtype=torch.uint8))
    ws0 = torch.full((ws.numel(),), 0xFF, dtype=torch.uint8)
    ws0[:256] = 0
    ws_g = Guarded(ws0)
    g.forward(Pd, Xg.t, [o.t for o in outs], saved_g.t, ws_g.t, inputs=[i.t for i in inputs])
    torch.cuda.synchronize()
    return g, inp, P, Pd, grads_in, ref, Xg, outs, inputs, saved_g, ws_g


class _Collect:
    """Run every comparison, then fail once with all messages."""

    def __init__(self):
        self.errors = []

    def __call__(self, fn, *a):
        try:
            fn(*a)
        except AssertionError as e:
            self.errors.append(str(e).split("\n")[0])

    def done(self):
        assert not self.errors, "\n".join(self.errors)


@pytest.mark.parametrize("name", list(CASES))
def test_forward_backward_parity(name):
    cfg, T, kw = CASES[name]
    g, inp, P, Pd, grads_in, ref, Xg, outs, inputs, saved_g, ws_g = run_case(cfg, T, **kw)
    aux = ref["aux"]
    chk = _Collect()
    assert_f32 = lambda *a: chk(assert_f32_close, *a)  # noqa: E731
    assert_bf16 = lambda *a: chk(assert_bf16_close, *a)  # noqa: E731

    # coefficients
    co = g.coefficients(saved_g.t, T)
    assert torch.equal(co["I"].cpu().long(), aux["I"]), "routing differs"
    assert_f32(co["p"], aux["p"], "p")
    for t in range(cfg.G):
        assert_f32(co["hpre"][:, t], aux["H_pre"][t], f"H_pre[{t}]")
        assert_f32(co["hpost"][t], aux["H_post"][t], f"H_post[{t}]")
    assert_f32(co["hres"], aux["H_res"], "H_res")

    # forward outputs
    for t in range(cfg.G):
        assert_bf16(inputs[t].t, ref["inputs"][t], f"input[{t}]")
    assert_bf16(Xg.t, ref["X"], "X_out")
    # inactive rows bit-identical
    I = aux["I"]
    mask = torch.ones(T, cfg.N, dtype=torch.bool)
    mask[torch.arange(T)[:, None], I] = False
    assert torch.equal(Xg.t.cpu()[mask], inp["X"][mask]), "inactive rows changed"

    # backward
    dXg = Guarded(grads_in["dX"].cuda())
    d_inputs = [Guarded(d.cuda()) for d in grads_in["d_inputs"]]
    d_outs = [Guarded(torch.zeros(T, cfg.C, dtype=torch.bfloat16)) for _ in range(cfg.G)]
    gr = {n: torch.zeros_like(v) for n, v in Pd.items()}
    g.backward(Pd, Xg.t, dXg.t, [o.t for o in outs], [d.t for d in d_inputs], gr, saved_g.t, ws_g.t,
               d_outs=[d.t for d in d_outs])
    torch.cuda.synchronize()
    assert torch.equal(Xg.t.cpu(), inp["X"]), "X not restored to the entry state"
    assert_bf16(dXg.t, ref["dX"], "dX")
    for t in range(cfg.G):
        assert_bf16(d_outs[t].t, ref["d_outs"][t], f"d_out[{t}]")
    scales = alpha_term_scales(cfg, inp, P, grads_in)
    for n, v in gr.items():
        if n.startswith("alpha"):
            # a gating scalar's gradient sums T x (map size) terms with cancellation: 1e-4 of
            # the summed term magnitudes
            chk(assert_alpha_close, v, ref["dP"][n], scales[n], f"grad {n}")
        else:
            assert_f32(v, ref["dP"][n], f"grad {n}")

    for buf in [Xg, dXg, saved_g, ws_g] + outs + inputs + d_inputs + d_outs:
        assert buf.intact(), "guard band overwritten"
    assert g.device_error(ws_g.t) == 0, "a bounded device wait gave up"
    chk.done()


def test_param_grads_accumulate_and_are_deterministic():
    cfg, T, _ = CASES["flash4_N16k4_C256"]
    g, inp, P, Pd, grads_in, ref, Xg, outs, inputs, saved_g, ws_g = run_case(cfg, T)
    res = []
    for rep in range(2):
        gr = {n: torch.full_like(v, 0.5) for n, v in Pd.items()}
        for _ in range(2):
            X = inp["X"].cuda()
            ins = g.forward(Pd, X, [o.t for o in outs], saved_g.t, ws_g.t)
            dX = grads_in["dX"].cuda()
            g.backward(Pd, X, dX, [o.t for o in outs], [d.cuda() for d in grads_in["d_inputs"]], gr,
                       saved_g.t, ws_g.t)
        torch.cuda.synchronize()
        res.append({n: v.cpu() for n, v in gr.items()})
    scales = alpha_term_scales(cfg, inp, P, grads_in)
    for n in res[0]:
        assert torch.equal(res[0][n], res[1][n]), f"{n} not deterministic"
        if n.startswith("alpha"):
            assert_alpha_close(res[0][n] - 0.5, 2 * ref["dP"][n], 2 * scales[n], f"accumulated {n}")
        else:
            assert_f32_close(res[0][n] - 0.5, 2 * ref["dP"][n], f"accumulated {n}")
