"""GPU parity of decoding (one new token per sequence, conv history in per-sequence rings).

B sequences are prefilled with S tokens through the ordinary forward, the rings are filled from
the prefill's sublayer outputs, then ND tokens are decoded one at a time.  The oracle runs the
plain forward on the whole sequences of S + ND tokens: every decoded token must give the oracle's
sublayer inputs, coefficients and new state rows at its position (tokens interact only through
the causal conv, whose history the rings carry).  S below max(kappa) - 1 exercises the zero
padding before the sequence start."""
import pytest
import torch

from paper_2607_14530_gb300 import synth
from paper_2607_14530_gb300.xhc import Config, Group

from xhc_cases import assert_bf16_close, assert_f32_close, flash_bases, run_oracle, tie_free

pytestmark = pytest.mark.gpu

ND = 3


def _cfg(N, k, m, C, G, S, **kw):
    if G == 1:
        return Config.full(N, k, m, C, True, seq_len=S, **kw)
    return Config.flash(N, k, m, C, G, seq_len=S, **kw)


@pytest.mark.parametrize("N,k,m,C,G,B,S", [
    (16, 4, 2, 256, 4, 3, 20),    # Flash-4sub, prefill longer than the ring
    (16, 4, 2, 256, 4, 2, 5),     # prefill shorter than the ring: zero padding
    (8, 4, 2, 128, 1, 4, 13),     # one full-xHC MLP sublayer
])
def test_decode_matches_the_whole_sequence_forward(N, k, m, C, G, B, S):
    L = S + ND
    cfg_o = _cfg(N, k, m, C, G, L)
    # seeded whole sequences without a routing near-tie (the oracle decides)
    for attempt in range(50):
        seed = 7 + 1000 * attempt
        inp = synth.group_inputs(B * L, N, C, G, seed)
        P = synth.params(cfg_o.param_shapes(), seed)
        if bool(tie_free(cfg_o, inp["X"], P["W_r"]).all()):
            break
    else:
        raise RuntimeError("no tie-free draw")
    ref = run_oracle(cfg_o, inp, P)
    aux = ref["aux"]
    bases = flash_bases(cfg_o, inp["X"], aux)

    pre_rows = torch.cat([torch.arange(b * L, b * L + S) for b in range(B)])

    def rows_at(p):
        return torch.tensor([b * L + p for b in range(B)])

    dev = torch.device("cuda", 0)
    Pd = {n: v.to(dev) for n, v in P.items()}
    # prefill: B sequences of S tokens
    gp = Group(_cfg(N, k, m, C, G, S))
    Xp = inp["X"][pre_rows].to(dev).contiguous()
    outs_p = [o[pre_rows].to(dev).contiguous() for o in inp["outs"]]
    saved, ws = gp.alloc(B * S)
    gp.forward(Pd, Xp, outs_p, saved, ws)
    rings = gp.alloc_rings(B)
    for t in range(G):
        if rings[t] is not None:
            gp.ring_fill(B, S, outs_p[t], rings[t])
    pos = torch.full((B,), S, dtype=torch.int64, device=dev)

    # decode ND tokens
    gd = Group(_cfg(N, k, m, C, G, 0))
    saved_d, ws_d = gd.alloc(B)
    errors = []

    def chk(fn, *a):
        try:
            fn(*a)
        except AssertionError as e:
            errors.append(str(e).split("\n")[0])

    for n in range(ND):
        r = rows_at(S + n)
        X = inp["X"][r].to(dev).contiguous()
        outs = [o[r].to(dev).contiguous() for o in inp["outs"]]
        ins = gd.forward_decode(Pd, X, outs, rings, pos, saved_d, ws_d)
        torch.cuda.synchronize()
        co = gd.coefficients(saved_d, B)
        tag = f"token {S + n}"
        if not torch.equal(co["I"].cpu().long(), aux["I"][r]):
            errors.append(f"{tag}: routing differs")
        for t in range(G):
            chk(assert_bf16_close, ins[t], ref["inputs"][t][r], f"{tag} input[{t}]",
                None if bases[t] is None else bases[t][r])
            chk(assert_f32_close, co["hpost"][t].cpu(), aux["H_post"][t][r], f"{tag} H_post[{t}]")
        chk(assert_f32_close, co["hres"].cpu(), aux["H_res"][r], f"{tag} H_res")
        chk(assert_bf16_close, X, ref["X"][r], f"{tag} X_out")
    assert gd.device_error(ws_d) == 0
    assert torch.equal(pos.cpu(), torch.full((B,), S + ND, dtype=torch.int64)), "pos not advanced"
    assert not errors, "\n".join(errors)
