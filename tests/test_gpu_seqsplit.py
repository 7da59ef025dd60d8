"""Sequence split through the C ABI on one GPU: the halo entry points against the unsplit oracle.

B sequences of S1 + S2 tokens are processed as two chunks by separate calls, as two ranks of a
context-parallel job would (here one after the other on one GPU; the exchange between ranks is
tests/test_seqsplit_gloo.py): the first chunk with plain calls, the second with
xhc_post_fwd_halo / xhc_post_bwd_halo and the halo that xhc_halo_fill takes from the first
chunk's sublayer outputs; the second chunk's halo gradient is added to the first chunk's d_out
with xhc_halo_add, and both chunks accumulate into the same parameter gradients.  Everything is
compared with the oracle's forward and backward of the unsplit sequences, element by element.
A first chunk shorter than the halo (S1 < R) checks the zero rows before the sequence start."""
import pytest
import torch

from oracle import xhc_oracle as O
from paper_2607_14530_gb300 import synth
from paper_2607_14530_gb300.xhc import Config, Group

from xhc_cases import (F64, Guarded, alpha_term_scales, assert_alpha_close, assert_bf16_close,
                       assert_f32_close, flash_bases, make_case, oracle_cfg, run_oracle)

pytestmark = pytest.mark.gpu


def _with_seq(cfg: Config, S: int) -> Config:
    d = dict(cfg.__dict__)
    d["seq_len"] = S
    return Config(**d)


@pytest.mark.parametrize("cfg,B,S1,S2", [
    (Config.full(16, 4, 2, 256, True), 3, 5, 7),            # S1 < R = 11: zero halo rows
    (Config.flash(16, 4, 2, 256, 4), 2, 140, 120),         # chunks longer than a token tile
    (Config.flash(8, 4, 2, 512, 4), 2, 70, 66),            # C = 512: two channel pairs per thread
], ids=["fullM_S5+7", "flash4_S140+120", "flash4_C512_S70+66"])
def test_two_chunks_with_halo_equal_the_unsplit_sequences(cfg, B, S1, S2):
    S = S1 + S2
    T = B * S
    full = _with_seq(cfg, S)
    inp, P, seed = make_case(full, T, 3)
    gin = synth.group_grads(T, cfg.N, cfg.C, cfg.G, seed)
    ref = run_oracle(full, inp, P, gin)
    aux = ref["aux"]
    dev = torch.device("cuda", 0)
    Pd = {n: v.to(dev) for n, v in P.items()}

    def rows(lo, hi):
        return torch.cat([torch.arange(b * S + lo, b * S + hi) for b in range(B)])

    chunks = []
    for lo, hi in ((0, S1), (S1, S)):
        r = rows(lo, hi)
        g = Group(_with_seq(cfg, hi - lo))
        saved, ws = g.alloc(B * (hi - lo), device=dev)
        chunks.append(dict(r=r, g=g, saved=saved, ws=ws, n=hi - lo,
                           X=Guarded(inp["X"][r].to(dev)),
                           outs=[Guarded(o[r].to(dev)) for o in inp["outs"]],
                           inputs=[Guarded(torch.zeros(B * (hi - lo), cfg.C, dtype=torch.bfloat16))
                                   for _ in range(cfg.G)]))
    A, C2 = chunks
    R = A["g"].halo_rows()
    halos = [A["g"].halo_fill(B, S1, A["outs"][t].t) if cfg.K(t) > 1 else None for t in range(cfg.G)]

    # forward of both chunks; the oracle's intermediate active states are injected between the
    # slots (as in tests/test_gpu_parity.py), so results downstream compare without ambiguity
    for ch, use_halo in ((A, False), (C2, True)):
        g = ch["g"]
        pp = g.params(Pd)
        xact = g.coefficients(ch["saved"], B * ch["n"])["xact"]
        for t in range(cfg.G):
            if t >= 1:
                xact[t].copy_(aux["X_act"][t][ch["r"]].to(torch.bfloat16))
            g.pre_fwd(t, pp, ch["X"].t, ch["inputs"][t].t, ch["saved"], ch["ws"])
            g.post_fwd(t, pp, ch["X"].t, ch["outs"][t].t, ch["saved"], ch["ws"],
                       halo=halos[t] if use_halo else None)
    torch.cuda.synchronize()
    errors = []

    def chk(fn, *a):
        try:
            fn(*a)
        except AssertionError as e:
            errors.append(str(e).split("\n")[0])

    bases = flash_bases(cfg, inp["X"], aux)
    for name, ch in (("chunk 1", A), ("chunk 2", C2)):
        r = ch["r"]
        co = ch["g"].coefficients(ch["saved"], B * ch["n"])
        if not torch.equal(co["I"].cpu().long(), aux["I"][r]):
            errors.append(f"{name}: routing differs")
        for t in range(cfg.G):
            chk(assert_f32_close, co["hpost"][t], aux["H_post"][t][r], f"{name} H_post[{t}]")
            chk(assert_bf16_close, ch["inputs"][t].t, ref["inputs"][t][r], f"{name} input[{t}]",
                None if bases[t] is None else bases[t][r])
        chk(assert_f32_close, co["hres"], aux["H_res"][r], f"{name} H_res")
        chk(assert_bf16_close, ch["X"].t, ref["X"][r], f"{name} X_out")

    # backward: the second chunk first (it produces the halo gradient), then the first
    grads = {n: torch.zeros_like(v) for n, v in Pd.items()}
    for ch in chunks:
        ch["dX"] = Guarded(gin["dX"][ch["r"]].to(dev))
        ch["d_in"] = [Guarded(d[ch["r"]].to(dev)) for d in gin["d_inputs"]]
        ch["d_outs"] = [Guarded(torch.zeros(B * ch["n"], cfg.C, dtype=torch.bfloat16)) for _ in range(cfg.G)]
    d_halos = [torch.full((B, R, cfg.C), float("nan"), device=dev) if cfg.K(t) > 1 else None
               for t in range(cfg.G)]
    for t in reversed(range(cfg.G)):
        for ch, use_halo in ((C2, True), (A, False)):
            g = ch["g"]
            pp, gg = g.params(Pd), g.params(grads)
            g.post_bwd(t, pp, ch["X"].t, ch["dX"].t, ch["outs"][t].t, ch["d_outs"][t].t, gg, ch["saved"],
                       ch["ws"], halo=halos[t] if use_halo else None,
                       d_halo=d_halos[t] if use_halo else None)
            if not use_halo and halos[t] is not None:
                g.halo_add(B, S1, ch["d_outs"][t].t, d_halos[t])
            g.pre_bwd(t, pp, ch["X"].t, ch["d_in"][t].t, ch["dX"].t, gg, ch["saved"], ch["ws"])
    torch.cuda.synchronize()
    # the first chunk's d_out of its last R tokens is its own bf16 d_out plus the returned halo
    # gradient: it inherits half an ulp of that bf16 partial, whose magnitude the oracle gives
    # (the unsplit d_out minus the oracle's halo gradient of the second chunk)
    c2 = oracle_cfg(_with_seq(cfg, S - S1))
    r2 = C2["r"]
    _, _, _, dh_ref = O.backward(c2, {n: v.to(F64) for n, v in P.items()}, inp["X"][r2].to(F64),
                                 [o[r2].to(F64) for o in inp["outs"]], gin["dX"][r2].to(F64),
                                 [d[r2].to(F64) for d in gin["d_inputs"]],
                                 halos=[None if h is None else h.cpu().to(F64) for h in halos])
    for name, ch in (("chunk 1", A), ("chunk 2", C2)):
        r = ch["r"]
        if not torch.equal(ch["X"].t.cpu(), inp["X"][r]):
            errors.append(f"{name}: X not restored")
        chk(assert_bf16_close, ch["dX"].t, ref["dX"][r], f"{name} dX")
        for t in range(cfg.G):
            scale = None
            if ch is A and dh_ref[t] is not None:
                part = ref["d_outs"][t][r].reshape(B, S1, cfg.C).clone()
                part[:, max(0, S1 - R):] -= dh_ref[t][:, max(0, R - S1):]
                scale = part.reshape(-1, cfg.C).abs()
            chk(assert_bf16_close, ch["d_outs"][t].t, ref["d_outs"][t][r], f"{name} d_out[{t}]", scale)
        for buf in [ch["X"], ch["dX"]] + ch["outs"] + ch["inputs"] + ch["d_in"] + ch["d_outs"]:
            if not buf.intact():
                errors.append(f"{name}: guard band overwritten")
        if ch["g"].device_error(ch["ws"]) != 0:
            errors.append(f"{name}: a bounded device wait gave up")
    scales = alpha_term_scales(full, inp, P, gin)
    for n, v in grads.items():
        if n.startswith("alpha"):
            chk(assert_alpha_close, v, ref["dP"][n], scales[n], f"grad {n}")
        else:
            chk(assert_f32_close, v, ref["dP"][n], f"grad {n}")
    assert not errors, "\n".join(errors)
