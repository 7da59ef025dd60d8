"""Pins of the fp64 oracle against what the paper and the mathematics fix (no GPU needed).

Each test checks the oracle against something other than itself: a closed form, an invariant,
a special case reducing to a textbook result, brute force on tiny inputs, finite differences,
or numbers printed in the paper (tests/golden/paper_counts.json).
"""
import json
import math
import os

import pytest
import torch

from oracle import brute as B
from oracle import xhc_oracle as O
from paper_2607_14530_gb300 import synth, traffic

F64 = torch.float64
GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_counts.json")


def _params(cfg, seed, alpha=0.5, w_std=0.3):
    return {n: v.to(F64) for n, v in synth.params(O.param_shapes(cfg), seed, alpha=alpha, w_std=w_std).items()}


def _inputs(cfg, T, seed):
    d = synth.group_inputs(T, cfg.N, cfg.C, cfg.G, seed)
    return d["X"].to(F64), [o.to(F64) for o in d["outs"]]


# ---------------------------------------------------------------------------------------------
# special cases with closed forms


def test_n1_reduces_to_plain_residual():
    """N = 1 (k = m = 1), alpha_post = 0, b_post = 0: H_res = [1], H_post = 2 sigma(0) = 1,
    so X_new = x + out (ordinary residual, Sec. 3.1) and input = sigma(b_pre) x."""
    cfg = O.mhc(1, 16)
    P = _params(cfg, 3)
    P["alpha_post"].zero_()
    P["b_post.0"].zero_()
    X, outs = _inputs(cfg, 9, 3)
    Xo, ins, aux = O.forward(cfg, P, X, outs, round_bf16=False)
    assert torch.allclose(aux["H_res"], torch.ones(9, 1, 1, dtype=F64), atol=0, rtol=1e-15)
    assert torch.allclose(Xo[:, 0], X[:, 0] + outs[0], atol=1e-14, rtol=0)
    # pre-map of the single stream: sigma(alpha * z + b) with z the projection
    x = X.reshape(9, 16)
    z = (x / torch.sqrt((x * x).mean(1, keepdim=True) + cfg.eps_norm)) @ P["W_pre.0"]
    h = torch.sigmoid(P["alpha_pre"][0] * z + P["b_pre"][0])
    assert torch.allclose(ins[0], h * X[:, 0], atol=1e-14, rtol=0)
    P["alpha_pre"].zero_()
    _, ins0, _ = O.forward(cfg, P, X, outs, round_bf16=False)
    assert torch.allclose(ins0[0], torch.sigmoid(P["b_pre"][0]) * X[:, 0], atol=1e-14, rtol=0)


def test_identity_mixing_reproduces_per_stream_residual():
    """mHC with alpha = 0, b_res = 40 I, b_pre = 40, b_post = 0: H_res = I, H_pre = 1 and
    H_post = 1 to within e^-40, so every stream gets x_i + out and input = sum_i x_i."""
    cfg = O.mhc(4, 12)
    P = _params(cfg, 5)
    for n in ("alpha_pre", "alpha_post", "alpha_res"):
        P[n].zero_()
    P["b_res"].copy_((40.0 * torch.eye(4, dtype=F64)).reshape(-1))
    P["b_pre"].fill_(40.0)
    P["b_post.0"].zero_()
    X, outs = _inputs(cfg, 7, 5)
    Xo, ins, aux = O.forward(cfg, P, X, outs, round_bf16=False)
    assert torch.allclose(aux["H_res"], torch.eye(4, dtype=F64).expand(7, 4, 4), atol=1e-15)
    assert torch.allclose(Xo, X + outs[0][:, None, :], atol=1e-13, rtol=0)
    assert torch.allclose(ins[0], X.sum(1), atol=1e-13, rtol=0)


def test_mhc_matches_hc_update():
    """With k = N (mHC) the op is Eq. hc: X_new = H_res X + H_post out, input = H_pre X."""
    cfg = O.mhc(4, 8)
    P = _params(cfg, 9)
    X, outs = _inputs(cfg, 5, 9)
    Xo, ins, aux = O.forward(cfg, P, X, outs, round_bf16=False)
    ref = torch.einsum("tij,tjc->tic", aux["H_res"], X) + aux["H_post"][0] * outs[0][:, None, :]
    assert torch.allclose(Xo, ref, atol=1e-13, rtol=0)
    assert torch.allclose(ins[0], torch.einsum("ti,tic->tc", aux["H_pre"][0], X), atol=1e-13)


# ---------------------------------------------------------------------------------------------
# Sinkhorn (Eq. mhc_sinkhorn) and the App. A row clamp


def test_sinkhorn_doubly_stochastic_at_workload_scale():
    """Logits alpha * z + b with alpha = 0.01 and b ~ N(0, 0.02): row and column sums are 1
    within 1e-6 after 20 iterations."""
    g = torch.Generator().manual_seed(0)
    M = 0.01 * torch.randn(2000, 4, 4, generator=g, dtype=F64) * 5 + 0.02 * torch.randn(4, 4, generator=g, dtype=F64)
    H = O.sinkhorn(M, 20)
    assert (H.sum(-1) - 1).abs().max() < 1e-6
    assert (H.sum(-2) - 1).abs().max() < 1e-6
    assert (H > 0).all()


def test_sinkhorn_uniform_gives_one_over_k():
    for k in (2, 3, 4, 8):
        H = O.sinkhorn(torch.full((1, k, k), 0.37, dtype=F64), 20)
        assert torch.allclose(H, torch.full_like(H, 1.0 / k), atol=1e-15)


def test_sinkhorn_permutation_equivariance():
    g = torch.Generator().manual_seed(1)
    M = torch.randn(1, 5, 5, generator=g, dtype=F64)
    pr, pc = torch.randperm(5, generator=g), torch.randperm(5, generator=g)
    H = O.sinkhorn(M, 20)[0]
    Hp = O.sinkhorn(M[:, pr][:, :, pc], 20)[0]
    assert torch.allclose(Hp, H[pr][:, pc], atol=1e-14)


def test_sinkhorn_2x2_closed_form_limit():
    """For a positive 2x2 matrix A the Sinkhorn limit is [[a, 1-a], [1-a, a]] with
    a = sqrt(A11 A22) / (sqrt(A11 A22) + sqrt(A12 A21))."""
    g = torch.Generator().manual_seed(2)
    for _ in range(20):
        M = torch.randn(1, 2, 2, generator=g, dtype=F64)
        A = torch.exp(M)[0]
        d, o = math.sqrt(A[0, 0] * A[1, 1]), math.sqrt(A[0, 1] * A[1, 0])
        a = d / (d + o)
        H = O.sinkhorn(M, 1000)[0]
        ref = torch.tensor([[a, 1 - a], [1 - a, a]], dtype=F64)
        assert torch.allclose(H, ref, atol=1e-12)


def test_row_clamp_never_raises_a_row_sum_above_one():
    g = torch.Generator().manual_seed(3)
    H = torch.rand(500, 4, 4, generator=g, dtype=F64) * 0.6
    Hc = O.row_clamp(H)
    rs, rsc = H.sum(-1), Hc.sum(-1)
    assert (rsc <= 1 + 1e-15).all()
    keep = rs <= 1
    assert torch.equal(Hc[keep], H[keep])
    assert torch.allclose(rsc[~keep], torch.ones_like(rsc[~keep]), atol=1e-15)


# ---------------------------------------------------------------------------------------------
# temporal feature augmentation (Eq. aug, conv formula) and Gram-Schmidt (Eq. gs)


def test_gram_schmidt_hand_example():
    out = torch.tensor([[1.0, 0.0, 0.0]], dtype=F64)
    g1 = torch.tensor([[1.0, 1.0, 0.0]], dtype=F64)
    g2 = torch.tensor([[2.0, 3.0, 5.0]], dtype=F64)
    v = O.gram_schmidt(out, [g1, g2], 0.0)
    assert torch.equal(v[0], out)
    assert torch.allclose(v[1], torch.tensor([[0.0, 1.0, 0.0]], dtype=F64), atol=1e-15)
    assert torch.allclose(v[2], torch.tensor([[0.0, 0.0, 5.0]], dtype=F64), atol=1e-15)


def test_gram_schmidt_orthogonal_span_and_mgs_agreement():
    g = torch.Generator().manual_seed(4)
    C = 64
    out = torch.randn(10, C, generator=g, dtype=F64)
    gs = [0.7 * out + torch.randn(10, C, generator=g, dtype=F64) for _ in range(3)]
    v = O.gram_schmidt(out, gs, 0.0)
    assert torch.equal(v[0], out)
    for a in range(4):
        for b in range(a):
            cos = (v[a] * v[b]).sum(1) / (v[a].norm(dim=1) * v[b].norm(dim=1))
            assert cos.abs().max() < 1e-12
    # span preserved: [out, g1, g2, g3] = V R with R upper-triangular
    U = torch.stack([out] + gs, 2)
    V = torch.stack(v, 2)
    R = torch.linalg.lstsq(V, U).solution
    assert torch.allclose(V @ R, U, atol=1e-10)
    assert torch.allclose(torch.tril(R, -1), torch.zeros_like(R), atol=1e-10)
    # modified Gram-Schmidt (project the running vector) equals Eq. gs in exact arithmetic
    w = [out]
    for gj in gs:
        r = gj
        for wi in w:
            r = r - ((r * wi).sum(1, keepdim=True) / (wi * wi).sum(1, keepdim=True)) * wi
        w.append(r)
    for a in range(4):
        assert torch.allclose(v[a], w[a], atol=1e-10)


def test_conv_delta_shift_causality_and_sequence_reset():
    g = torch.Generator().manual_seed(5)
    T, C, S = 12, 5, 4
    out = torch.randn(T, C, generator=g, dtype=F64)
    delta = torch.zeros(4, C, dtype=F64)
    delta[0] = 1
    assert torch.equal(O.causal_dwconv(out, delta, S), out)
    shift = torch.zeros(3, C, dtype=F64)
    shift[2] = 1
    gsh = O.causal_dwconv(out, shift, S)
    for t in range(T):
        ref = out[t - 2] if t % S >= 2 else torch.zeros(C, dtype=F64)
        assert torch.equal(gsh[t], ref)
    w = torch.randn(8, C, generator=g, dtype=F64)
    base = O.causal_dwconv(out, w, T)
    for tp in range(T):
        pert = out.clone()
        pert[tp] += 1.0
        gp = O.causal_dwconv(pert, w, T)
        assert torch.equal(gp[:tp], base[:tp])          # causal: no future token leaks back
        if tp + 8 < T:
            assert torch.equal(gp[tp + 8:], base[tp + 8:])  # support of a width-8 kernel
    # brute force sum for one token
    t = 7
    ref = sum(w[i] * out[t - i] for i in range(8))
    assert torch.allclose(base[t], ref, atol=1e-14)


@pytest.mark.parametrize("cfg", [O.flash(5, 3, 1, 8, 4, conv_k=(2, 3)), O.full(4, 2, 1, 6, True, conv_k=(3,))],
                         ids=["flash4", "fullM"])
def test_forward_of_a_sequence_prefix_is_the_prefix_of_the_forward(cfg):
    # tokens interact only through the causal conv: the forward of the first L' tokens of a
    # sequence equals the first L' rows of the forward of the whole sequence (what decoding one
    # token at a time relies on); with sequence starts every L, sequences are independent too
    L, Lp, nseq = 9, 5, 2
    P = _params(cfg, 11)
    Xw, outs_w = _inputs(cfg, nseq * L, 12)
    cw = O.Config(**{**cfg.__dict__, "seq_len": L})
    cp = O.Config(**{**cfg.__dict__, "seq_len": Lp})
    Xo_w, ins_w, aux_w = O.forward(cw, P, Xw, outs_w)
    rows = torch.cat([torch.arange(b * L, b * L + Lp) for b in range(nseq)])
    Xo_p, ins_p, aux_p = O.forward(cp, P, Xw[rows], [o[rows] for o in outs_w])
    assert torch.allclose(Xo_p, Xo_w[rows], rtol=0, atol=1e-12)
    for t in range(cfg.G):
        assert torch.allclose(ins_p[t], ins_w[t][rows], rtol=0, atol=1e-12)
    assert torch.equal(aux_p["I"], aux_w["I"][rows])


# ---------------------------------------------------------------------------------------------
# routing, sparse write-back and the whole group against the brute-force oracle

CFGS = [
    O.full(4, 2, 1, 8, False, seq_len=3),
    O.full(4, 2, 1, 8, True, seq_len=3, conv_k=(2, 3)),
    O.full(4, 4, 2, 8, True, seq_len=6, conv_k=(2,)),     # every stream active, routed order matters
    O.full(5, 3, 0, 6, False),                           # m = 0: no fixed stream
    O.mhc(3, 8),
    O.mhc(2, 4),
    O.flash(5, 3, 1, 8, 2, conv_k=(2, 3)),
    O.flash(5, 3, 1, 8, 4, seq_len=3, conv_k=(2, 3)),
    O.flash(4, 2, 1, 6, 4, conv_k=(2, 3), gram_schmidt=False),
    # ablations of Table ablation: softmax router (11), no dense read (7), neither dense read
    # nor fixed streams (6)
    O.full(5, 3, 1, 8, True, seq_len=3, conv_k=(2, 3), router="softmax"),
    O.full(5, 3, 1, 8, False, dense_read=False),
    O.full(5, 3, 0, 6, True, conv_k=(2,), dense_read=False),
    O.flash(5, 3, 1, 8, 4, seq_len=3, conv_k=(2, 3), router="softmax", dense_read=False),
]


def _cid(c):
    tag = f"N{c.N}k{c.k}m{c.m}G{c.G}{''.join('M' if x else 'A' for x in c.mlp)}"
    return tag + ("-softmax" if c.router == "softmax" else "") + ("-sparse" if not c.dense_read else "")


@pytest.mark.parametrize("cfg", CFGS, ids=_cid)
@pytest.mark.parametrize("rounding", [False, True])
def test_group_matches_brute_force(cfg, rounding):
    T = 6
    P = _params(cfg, 11)
    X, outs = _inputs(cfg, T, 11)
    Xo, ins, aux = O.forward(cfg, P, X, outs, round_bf16=rounding)
    Pl = {k: (v.tolist() if v.dim() > 0 else v.item()) for k, v in P.items()}
    Xb, insb, Ib = B.forward(cfg, Pl, X.tolist(), [o.tolist() for o in outs], round_bf16=rounding)
    assert torch.equal(aux["I"], torch.tensor(Ib))
    tol = 0.0 if rounding else 1e-13
    # with rounding on, fp64 summation order can flip a bf16 rounding at a tie: allow one ulp
    if rounding:
        d = (Xo - torch.tensor(Xb, dtype=F64)).abs()
        assert (d <= 2.0 ** -7 * torch.tensor(Xb, dtype=F64).abs().clamp(min=2.0 ** -10)).all()
        assert (d > 0).float().mean() < 0.01
    else:
        assert (Xo - torch.tensor(Xb, dtype=F64)).abs().max() <= tol
        for a, b in zip(ins, insb):
            assert (a - torch.tensor(b, dtype=F64)).abs().max() <= tol


def test_inactive_rows_bitwise_unchanged():
    cfg = O.flash(16, 4, 2, 32, 4, conv_k=(4, 8, 12), seq_len=16)
    T = 32
    P = _params(cfg, 12, alpha=0.01, w_std=0.02)
    X, outs = _inputs(cfg, T, 12)
    Xo, _, aux = O.forward(cfg, P, X, outs)
    I = aux["I"]
    mask = torch.ones(T, 16, dtype=torch.bool)
    mask[torch.arange(T)[:, None], I] = False
    assert torch.equal(Xo[mask], X[mask])
    assert mask.sum() == T * 12
    # fixed streams always active, routed streams distinct and outside the fixed set
    assert torch.equal(I[:, :2], torch.arange(2).expand(T, 2))
    for t in range(T):
        assert len(set(I[t].tolist())) == 4


def test_routed_scores_sorted_and_maximal():
    cfg = O.full(16, 4, 2, 8, False)
    T = 50
    P = _params(cfg, 13, alpha=0.01, w_std=0.2)
    X, outs = _inputs(cfg, T, 13)
    _, _, aux = O.forward(cfg, P, X, outs, round_bf16=False)
    s, I, p = aux["s"], aux["I"], aux["p"]
    for t in range(T):
        routed = I[t, 2:].tolist()
        others = [i for i in range(2, 16) if i not in routed]
        assert min(s[t, routed]) >= max(s[t, others])
        assert s[t, routed[0]] >= s[t, routed[1]]
        assert torch.equal(p[t, 2:], s[t, routed])
        assert torch.equal(p[t, :2], torch.ones(2, dtype=F64))


def test_routing_margin_hand_computed_gaps():
    """routing_margin decides which seeds the parity suite uses (a selection is unique only
    when the routed scores that TopK separates differ): the smallest gap between consecutive
    non-fixed scores among the k - m + 1 largest, computed here by hand."""
    cfg = O.full(5, 3, 1, 8, False)  # m = 1 fixed, k - m = 2 routed out of streams 1..4
    s = torch.tensor([[0.99, 0.10, 0.50, 0.45, 0.20],   # sorted routed: .50 .45 .20 .10 -> gaps .05, .25
                      [0.01, 0.70, 0.30, 0.60, 0.65],   # .70 .65 .60 -> gaps .05, .05
                      [0.50, 0.40, 0.40, 0.90, 0.10],   # .90 .40 .40 -> gaps .50, 0 (a tie)
                      [0.50, 0.80, 0.20, 0.30, 0.10]],  # .80 .30 .20 -> gaps .50, .10
                     dtype=F64)
    got = O.routing_margin(cfg, s)
    want = torch.tensor([0.05, 0.05, 0.0, 0.10], dtype=F64)
    assert torch.allclose(got, want, atol=1e-15, rtol=0), got
    # the fixed stream's score never enters (stream 0 is fixed whatever its score)
    s2 = s.clone()
    s2[:, 0] = 0.475
    assert torch.equal(O.routing_margin(cfg, s2), got)
    # k - m + 1 larger than the routed candidates: every candidate counts (N = 3, m = 1, k = 3)
    cfg3 = O.full(3, 3, 1, 8, False)
    assert torch.allclose(O.routing_margin(cfg3, torch.tensor([[0.3, 0.8, 0.5]], dtype=F64)),
                          torch.tensor([0.3], dtype=F64), atol=1e-15, rtol=0)
    # nothing to choose: no router (k = m), or a single routed candidate
    assert math.isinf(float(O.routing_margin(O.full(4, 2, 2, 8, False), s[:, :4])[0]))
    assert math.isinf(float(O.routing_margin(O.full(2, 2, 1, 8, False), s[:, :2])[0]))


# ---------------------------------------------------------------------------------------------
# xHC-Flash dense-read reuse is exact (App. E.1, E.2, E.3)


@pytest.mark.parametrize("G", [2, 4])
def test_flash_corrected_inputs_equal_full_dense_reads(G):
    cfg = O.flash(16, 4, 2, 16, G, conv_k=(4, 8, 12), seq_len=8)
    T = 16
    P = _params(cfg, 14)
    X, outs = _inputs(cfg, T, 14)
    _, ins, aux = O.forward(cfg, P, X, outs, round_bf16=False)
    I, p = aux["I"], aux["p"]
    inactive = torch.ones(T, 16, dtype=F64)
    inactive[torch.arange(T)[:, None], I] = 0
    for t in range(G):
        Hp = aux["H_pre"][t]
        base = torch.einsum("ti,tic->tc", Hp * inactive, X)            # Eq. app_four_sub_base
        act = torch.einsum("tj,tjc->tc", Hp.gather(1, I), aux["X_act"][t])  # Eq. app_active_read
        assert torch.allclose(base + act, ins[t], atol=1e-12, rtol=0)
    if G == 2:
        # Eq. read_reuse: input_MLP = inp_M + alpha out_Attn, alpha = sum_j Hpre_M[I_j] p_j Hpost_A[j]
        inp_M = torch.einsum("ti,tic->tc", aux["H_pre"][1], X)
        alpha = (aux["H_pre"][1].gather(1, I) * p * aux["H_post"][0][:, :, 0]).sum(1)
        assert torch.allclose(inp_M + alpha[:, None] * outs[0], ins[1], atol=1e-12, rtol=0)


# ---------------------------------------------------------------------------------------------
# backward: central finite differences in fp64 (no rounding)


@pytest.mark.parametrize("cfg", [
    O.full(4, 2, 1, 8, True, seq_len=3, conv_k=(2, 3)),
    O.full(4, 3, 1, 6, False),
    O.mhc(3, 8),
    O.flash(5, 3, 1, 8, 4, seq_len=3, conv_k=(2, 3)),
    O.full(4, 2, 1, 8, True, seq_len=3, conv_k=(2, 3), router="softmax"),
    O.flash(5, 3, 0, 8, 4, seq_len=3, conv_k=(2, 3), dense_read=False),
], ids=["fullM", "fullA", "mhc", "flash4", "fullM-softmax", "flash4-sparse-m0"])
def test_backward_matches_central_differences(cfg):
    T = 6
    P = _params(cfg, 1)
    X, outs = _inputs(cfg, T, 1)
    gr = synth.group_grads(T, cfg.N, cfg.C, cfg.G, 1)
    dXo = gr["dX"].to(F64)
    dins = [d.to(F64) for d in gr["d_inputs"]]
    _, _, aux = O.forward(cfg, P, X, outs, round_bf16=False)
    assert (O.routing_margin(cfg, aux["s"]) > 1e-3).all() if cfg.has_router else True
    dX, douts, dP = O.backward(cfg, P, X, outs, dXo, dins, round_bf16=False)

    def L(P_, X_, outs_):
        Xo, ins, _ = O.forward(cfg, P_, X_, outs_, round_bf16=False)
        return (Xo * dXo).sum().item() + sum((a * b).sum().item() for a, b in zip(ins, dins))

    g = torch.Generator().manual_seed(7)
    h = 1e-6

    def check(fd, an):
        assert abs(fd - an) <= 2e-6 * max(1.0, abs(an)), (fd, an)

    for name in P:
        flat = P[name].view(-1)
        for idx in torch.randint(0, flat.numel(), (3,), generator=g).tolist():
            Pp = {k: v.clone() for k, v in P.items()}
            Pm = {k: v.clone() for k, v in P.items()}
            Pp[name].view(-1)[idx] += h
            Pm[name].view(-1)[idx] -= h
            check((L(Pp, X, outs) - L(Pm, X, outs)) / (2 * h), dP[name].view(-1)[idx].item())
    for idx in torch.randint(0, X.numel(), (12,), generator=g).tolist():
        Xp, Xm = X.clone(), X.clone()
        Xp.view(-1)[idx] += h
        Xm.view(-1)[idx] -= h
        check((L(P, Xp, outs) - L(P, Xm, outs)) / (2 * h), dX.view(-1)[idx].item())
    for t in range(cfg.G):
        for idx in torch.randint(0, outs[t].numel(), (6,), generator=g).tolist():
            op = [o.clone() for o in outs]
            om = [o.clone() for o in outs]
            op[t].view(-1)[idx] += h
            om[t].view(-1)[idx] -= h
            check((L(P, X, op) - L(P, X, om)) / (2 * h), douts[t].view(-1)[idx].item())


# ---------------------------------------------------------------------------------------------
# numbers printed in the paper


def _golden():
    with open(GOLDEN) as f:
        return json.load(f)


def _layer_cfgs(method, N, k=4, C=1):
    if method == "mHC":
        return [O.mhc(N, C), O.mhc(N, C)]
    return [O.full(N, k, min(2, k - 1), C, False), O.full(N, k, min(2, k - 1), C, True)]


def test_parameter_counts_match_paper():
    """Eq. xhc_params / Eq. mhc_params and the values of App. C pin every W shape."""
    gold = _golden()
    for row in gold["param_count_over_C"]:
        cfgs = _layer_cfgs(row["method"], row["N"], row.get("k", 4), C=8)
        assert O.layer_param_count_over_C(cfgs) == row["value"], row
    for row in gold["param_count_per_layer"]:
        cfgs = _layer_cfgs(row["method"], row["N"], row.get("k", 4), C=row["C"])
        n = O.layer_param_count_over_C(cfgs) * row["C"]
        txt = row["printed"]
        scale = 1e6 if txt.endswith("M") else 1e3
        digits = len(txt[:-1].split(".")[1]) if "." in txt else 0
        # the table rounds some entries and truncates others (405,504 -> "405K",
        # 19,464,192 -> "19.5M"): accept anything within one unit of the last printed digit
        assert abs(n / scale - float(txt[:-1])) < 10.0 ** -digits, (row, n)


def test_traffic_model_reproduces_table():
    """Our reading of Table overhead_analysis reproduces its printed totals.  The 4-sublayer
    write column comes out at 13.25C against the printed 13.5C (total 39.75C vs 40C); the
    reconstruction has no row that accounts for the missing C per group."""
    gold = _golden()
    for row in gold["traffic_per_sublayer_over_C"]:
        m = {"mHC": "mhc", "xHC": "xhc", "xHC-Flash": "flash2", "xHC-Flash-4sub": "flash4"}[row["method"]]
        r, w = traffic.paper_model(m, row["N"], row.get("k", 4))
        if m == "flash4":
            assert r == row["read"] and abs(w - row["write"]) <= 0.25 and abs(r + w - row["total"]) <= 0.25
            continue
        assert r + w == row["total"], (row, r, w)
        if "read" in row:
            assert (r, w) == (row["read"], row["write"])


# ---------------------------------------------------------------------------------------------
# bf16 rounding bookkeeping used by the parity tests


def test_bf16_other_neighbor_hand_values():
    """Spacing of bf16 is 2^-7 on [1, 2) and 2^-8 on [1/2, 1); the smallest subnormal is 2^-133."""
    v = torch.tensor([1 + 0.3 * 2 ** -7, 1 - 0.3 * 2 ** -8, -(1 + 0.3 * 2 ** -7), -(1 - 0.3 * 2 ** -8),
                      3e-41, -3e-41, 1.5, 0.0], dtype=F64)
    r = v.to(torch.bfloat16).to(F64)
    want = torch.tensor([1 + 2 ** -7, 1 - 2 ** -8, -(1 + 2 ** -7), -(1 - 2 ** -8),
                         2.0 ** -133, -(2.0 ** -133), 1.5, 0.0], dtype=F64)
    assert torch.equal(r[:4].abs(), torch.ones(4, dtype=F64))
    assert torch.equal(O.bf16_other_neighbor(v, r), want)


def test_bf16_other_neighbor_brackets_random_values():
    g = torch.Generator().manual_seed(7)
    v = torch.randn(20000, generator=g, dtype=F64) * torch.exp2(torch.randint(-20, 20, (20000,), generator=g)).to(F64)
    r = v.to(torch.bfloat16).to(F64)
    o = O.bf16_other_neighbor(v, r)
    assert torch.equal(o.to(torch.bfloat16).to(F64), o)           # representable
    lo, hi = torch.minimum(r, o), torch.maximum(r, o)
    exact = v == r
    assert bool(((lo <= v) & (v <= hi))[~exact].all())              # brackets v
    # adjacent: the midpoint rounds to one of the two (no bf16 value strictly between)
    mid = (0.5 * (r + o)).to(torch.bfloat16).to(F64)
    assert bool(((mid == r) | (mid == o))[~exact].all())
    assert bool(((v - r).abs() <= (v - o).abs())[~exact].all())     # r is the nearer one


def test_prerounding_bookkeeping():
    """pre[t] rounds to the active state entering slot t (Eq. sparse_write, Eq. flash_attn_update)
    and mag[t] bounds |pre[t]| (triangle inequality over the terms it sums)."""
    cfg = O.flash(6, 3, 1, 16, 4, conv_k=(2, 3))
    T = 10
    P = _params(cfg, 21, alpha=0.1, w_std=0.2)
    X, outs = _inputs(cfg, T, 21)
    X = X.to(torch.bfloat16).to(F64)
    outs = [o.to(torch.bfloat16).to(F64) for o in outs]
    _, _, aux = O.forward(cfg, P, X, outs)
    assert sorted(aux["pre"]) == [1, 2, 3]
    for t in range(1, 4):
        assert torch.equal(O.rnd(aux["pre"][t], True), aux["X_act"][t])
        assert bool((aux["mag"][t] >= aux["pre"][t].abs() * (1 - 1e-12)).all())


def test_softmax_router_scores_and_sparse_read_closed_forms():
    """Softmax router (Table ablation row 11): the N scores of a token sum to 1 and order the
    streams like the sigmoid scores (both monotone in the logit).  Sparse read (rows 6-7): the
    sublayer input is the pre-map-weighted sum of the active streams only."""
    cfg = O.full(6, 3, 1, 8, False, router="softmax", dense_read=False)
    T = 7
    P = _params(cfg, 31)
    X, outs = _inputs(cfg, T, 31)
    Xo, ins, aux = O.forward(cfg, P, X, outs, round_bf16=False)
    s = aux["s"]
    assert torch.allclose(s.sum(1), torch.ones(T, dtype=F64), atol=1e-14, rtol=0)
    sig = O.router_scores(O.full(6, 3, 1, 8, False), X.reshape(T, -1), P["W_r"])
    assert torch.equal(torch.argsort(s, dim=1), torch.argsort(sig, dim=1))
    I = aux["I"]
    want = torch.einsum("tj,tjc->tc", aux["H_pre"][0].gather(1, I), X[torch.arange(T)[:, None], I])
    assert torch.allclose(ins[0], want, atol=1e-13, rtol=0)


@pytest.mark.parametrize("cfg", [O.full(5, 3, 1, 8, True, conv_k=(2, 4)),
                                 O.flash(5, 3, 1, 8, 4, conv_k=(2, 3, 4))], ids=["fullM", "flash4"])
def test_sequence_split_with_halo_equals_unsplit(cfg):
    """Cutting each sequence into two chunks: the second chunk's forward with the first chunk's
    last R = max(kappa) - 1 outputs as its halo equals the unsplit forward on those tokens; in the
    backward, the first chunk's d_out plus the second chunk's halo gradient equals the unsplit
    d_out, and the parameter gradients of the chunks add up to the unsplit ones."""
    B, S1, S2 = 2, 5, 4
    S = S1 + S2
    T = B * S
    R = max(cfg.conv_k) - 1
    P = _params(cfg, 41, alpha=0.3)
    X, outs = _inputs(cfg, T, 41)
    g = torch.Generator().manual_seed(42)
    dXo = torch.randn(X.shape, generator=g, dtype=F64)
    dins = [torch.randn(T, cfg.C, generator=g, dtype=F64) for _ in range(cfg.G)]
    full = O.Config(**{**cfg.__dict__, "seq_len": S})
    Xo, ins, _ = O.forward(full, P, X, outs, round_bf16=False)
    dX, dout, dP = O.backward(full, P, X, outs, dXo, dins, round_bf16=False)

    def rows(lo, hi):
        return torch.cat([torch.arange(b * S + lo, b * S + hi) for b in range(B)])

    r1, r2 = rows(0, S1), rows(S1, S)
    c1 = O.Config(**{**cfg.__dict__, "seq_len": S1})
    c2 = O.Config(**{**cfg.__dict__, "seq_len": S2})
    halos = [outs[t].reshape(B, S, cfg.C)[:, S1 - R:S1] for t in range(cfg.G)]
    X2o, ins2, _ = O.forward(c2, P, X[r2], [o[r2] for o in outs], round_bf16=False, halos=halos)
    assert torch.allclose(X2o, Xo[r2], atol=1e-12, rtol=0)
    for t in range(cfg.G):
        assert torch.allclose(ins2[t], ins[t][r2], atol=1e-12, rtol=0)
    dX1, dout1, dP1 = O.backward(c1, P, X[r1], [o[r1] for o in outs], dXo[r1], [d[r1] for d in dins],
                                 round_bf16=False)
    dX2, dout2, dP2, dh = O.backward(c2, P, X[r2], [o[r2] for o in outs], dXo[r2], [d[r2] for d in dins],
                                     round_bf16=False, halos=halos)
    assert torch.allclose(dX1, dX[r1], atol=1e-12, rtol=0) and torch.allclose(dX2, dX[r2], atol=1e-12, rtol=0)
    for t in range(cfg.G):
        d1 = dout1[t].reshape(B, S1, cfg.C).clone()
        d1[:, S1 - R:] += dh[t]
        assert torch.allclose(d1.reshape(-1, cfg.C), dout[t][r1], atol=1e-12, rtol=0)
        assert torch.allclose(dout2[t], dout[t][r2], atol=1e-12, rtol=0)
    for n in dP:
        assert torch.allclose(dP1[n] + dP2[n], dP[n], atol=1e-11, rtol=1e-12), n
