"""GPU parity of libxhc against the fp64 oracle, element by element, through the C ABI.

Each case runs the whole group forward (pre_fwd / post_fwd for every slot) and backward
(post_bwd / pre_bwd in reverse) on seeded inputs and compares: the sublayer inputs, the new
state, the coefficients (I exactly, p / H_pre / H_post / H_res element by element at 1e-4), the
intermediate active states of xHC-Flash groups (bit-identical except where the oracle finds the
bf16 rounding ambiguous), dX, every d_out and every parameter gradient (element by element at
1e-4).  Everything downstream of an intermediate active state is compared on a second run into
which the oracle's intermediate states are injected (xhc_cases.group_forward).
Guard bands around the caller buffers must stay intact, inactive rows must be bit-identical
after the forward, and X must hold the entry state again after the backward.  Shapes span
several tiles and ragged tails (T not a multiple of the token tiles, C not a multiple of the
256-channel slices)."""
import pytest
import torch

from paper_2607_14530_gb300 import synth
from paper_2607_14530_gb300.xhc import Config, Group

from xhc_cases import (Guarded, alpha_term_scales, ambiguity_masks, assert_alpha_close,
                       assert_bf16_close, assert_f32_close, check_active_states, flash_bases,
                       group_forward, make_case, run_oracle)

pytestmark = pytest.mark.gpu

CASES = {
    # the small flash4 shapes: N=16, k=4, C=256, T=512
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
    # N = 32: 160 full-state projection columns (router + 4 pre-maps), above the tensor-core
    # full-state dX's single k-block pair
    "flash4_N32_C256": (Config.flash(32, 4, 2, 256, 4, seq_len=128), 256, {}),
    # C a multiple of 512: the MLP slots' reductions with two channel pairs per thread
    "flash4_N8k4_C512": (Config.flash(8, 4, 2, 512, 4, seq_len=160), 320, {}),
    # attention-side temporal augmentation (App. "Additional Ablation Studies")
    "flash4_attn_tfa": (Config.flash(16, 4, 2, 256, 4, attn_tfa=True, seq_len=128), 512, {}),
    "flash2_attn_tfa": (Config.flash(16, 4, 2, 256, 2, attn_tfa=True, seq_len=128), 256, {}),
    # Table ablation: softmax router (11); no dense read (7); no dense read and no fixed stream (6)
    "fullM_softmax_router": (Config.full(16, 4, 2, 256, True, seq_len=128, router="softmax"), 256, {}),
    "fullM_sparse_read": (Config.full(16, 4, 2, 256, True, seq_len=128, sparse_read=True), 256, {}),
    "fullA_sparse_read_m0": (Config.full(16, 4, 0, 256, False, sparse_read=True), 200, {}),
    "flash4_softmax_sparse": (Config.flash(16, 4, 2, 256, 4, seq_len=128, router="softmax",
                                           sparse_read=True), 256, {}),
    # every active stream fixed (m = k < N): no router
    "fullM_m_eq_k": (Config.full(8, 4, 4, 128, True, seq_len=64), 128, {}),
    "flash4_m_eq_k": (Config.flash(8, 4, 4, 128, 4, seq_len=64), 128, {}),
}


def _cuda(d):
    return {n: v.cuda().contiguous() for n, v in d.items()}


def gpu_forward(g, cfg, inp, Pd, T, inject=None):
    """The group forward on guarded buffers; saved and workspace start poisoned (0xFF bytes: NaN
    as fp32 / bf16, -1 as int32), except the workspace's device error word: nothing may be read
    before the call sequence wrote it."""
    Xg = Guarded(inp["X"].cuda())
    outs = [Guarded(o.cuda()) for o in inp["outs"]]
    inputs = [Guarded(torch.zeros(T, cfg.C, dtype=torch.bfloat16)) for _ in range(cfg.G)]
    saved, ws = g.alloc(T)
    saved_g = Guarded(torch.full((saved.numel(),), 0xFF, dtype=torch.uint8))
    ws0 = torch.full((ws.numel(),), 0xFF, dtype=torch.uint8)
    ws0[:256] = 0
    ws_g = Guarded(ws0)
    group_forward(g, cfg, Pd, Xg.t, [o.t for o in outs], saved_g.t, ws_g.t, [i.t for i in inputs], inject)
    torch.cuda.synchronize()
    return Xg, outs, inputs, saved_g, ws_g


def run_case(cfg, T, seed=0, alpha=0.01, inject=True):
    inp, P, seed = make_case(cfg, T, seed, alpha=alpha)
    grads_in = synth.group_grads(T, cfg.N, cfg.C, cfg.G, seed)
    ref = run_oracle(cfg, inp, P, grads_in)
    g = Group(cfg)
    Pd = _cuda(P)
    Xg, outs, inputs, saved_g, ws_g = gpu_forward(g, cfg, inp, Pd, T, ref["aux"] if inject else None)
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


def _forward_outputs(chk, cfg, T, inp, ref, Xg, inputs, tag):
    bases = flash_bases(cfg, inp["X"], ref["aux"])
    for t in range(cfg.G):
        chk(assert_bf16_close, inputs[t].t, ref["inputs"][t], f"{tag}input[{t}]", bases[t])
    chk(assert_bf16_close, Xg.t, ref["X"], f"{tag}X_out")
    I = ref["aux"]["I"]
    mask = torch.ones(T, cfg.N, dtype=torch.bool)
    mask[torch.arange(T)[:, None], I] = False
    if not torch.equal(Xg.t.cpu()[mask], inp["X"][mask]):
        chk.errors.append(f"{tag}inactive rows changed")


@pytest.mark.parametrize("name", list(CASES))
def test_forward_backward_parity(name):
    cfg, T, kw = CASES[name]
    g, inp, P, Pd, grads_in, ref, Xg, outs, inputs, saved_g, ws_g = run_case(cfg, T, **kw)
    aux = ref["aux"]
    chk = _Collect()
    assert_f32 = lambda *a: chk(assert_f32_close, *a)  # noqa: E731
    assert_bf16 = lambda *a: chk(assert_bf16_close, *a)  # noqa: E731

    if cfg.G > 1:
        # the kernels' own forward: the bf16 roundings of the intermediate active states are the
        # oracle's wherever the oracle finds them unambiguous; the outputs within bf16 tolerance
        Xo, outs_o, inputs_o, saved_o, ws_o = gpu_forward(g, cfg, inp, Pd, T)
        co = g.coefficients(saved_o.t, T)
        if not torch.equal(co["I"].cpu().long(), aux["I"]):
            chk.errors.append("own forward: routing differs")
        chk.errors += check_active_states(co["xact"], aux, ambiguity_masks(cfg, aux), cfg, "own forward: ")
        _forward_outputs(chk, cfg, T, inp, ref, Xo, inputs_o, "own forward: ")
        for buf in [Xo, saved_o, ws_o] + outs_o + inputs_o:
            if not buf.intact():
                chk.errors.append("own forward: guard band overwritten")

    # coefficients
    co = g.coefficients(saved_g.t, T)
    assert torch.equal(co["I"].cpu().long(), aux["I"]), "routing differs"
    assert_f32(co["p"], aux["p"], "p")
    for t in range(cfg.G):
        assert_f32(co["hpre"][:, t], aux["H_pre"][t], f"H_pre[{t}]")
        assert_f32(co["hpost"][t], aux["H_post"][t], f"H_post[{t}]")
    assert_f32(co["hres"], aux["H_res"], "H_res")

    # forward outputs
    _forward_outputs(chk, cfg, T, inp, ref, Xg, inputs, "")

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
            chk(assert_alpha_close, v, ref["dP"][n], scales[n], f"grad {n}")
        else:
            assert_f32(v, ref["dP"][n], f"grad {n}")

    for buf in [Xg, dXg, saved_g, ws_g] + outs + inputs + d_inputs + d_outs:
        assert buf.intact(), "guard band overwritten"
    assert g.device_error(ws_g.t) == 0, "a bounded device wait gave up"
    chk.done()


def test_param_grads_accumulate_and_are_deterministic():
    """Gradients are accumulated (+=): from zero, two forward/backward passes give the second
    pass's increment equal to the oracle's gradient; the same call sequence repeated gives the
    same bits (fixed reduction order)."""
    cfg, T, _ = CASES["flash4_N16k4_C256"]
    g, inp, P, Pd, grads_in, ref, Xg, outs, inputs, saved_g, ws_g = run_case(cfg, T)
    res = []
    for rep in range(2):
        gr = {n: torch.zeros_like(v) for n, v in Pd.items()}
        snaps = []
        for _ in range(2):
            X = inp["X"].cuda()
            ins = [torch.empty(T, cfg.C, dtype=torch.bfloat16, device="cuda") for _ in range(cfg.G)]
            group_forward(g, cfg, Pd, X, [o.t for o in outs], saved_g.t, ws_g.t, ins, ref["aux"])
            dX = grads_in["dX"].cuda()
            g.backward(Pd, X, dX, [o.t for o in outs], [d.cuda() for d in grads_in["d_inputs"]], gr,
                       saved_g.t, ws_g.t)
            torch.cuda.synchronize()
            snaps.append({n: v.cpu().to(torch.float64) for n, v in gr.items()})
        res.append(snaps)
    scales = alpha_term_scales(cfg, inp, P, grads_in)
    for n in res[0][1]:
        assert torch.equal(res[0][1][n], res[1][1][n]), f"{n} not deterministic"
        inc = res[0][1][n] - res[0][0][n]
        if n.startswith("alpha"):
            assert_alpha_close(inc, ref["dP"][n], scales[n], f"accumulated {n}")
        else:
            assert_f32_close(inc, ref["dP"][n], f"accumulated {n}")
