"""Shared helpers of the GPU parity tests: seeded cases, the oracle run, comparisons.

Inputs come from the seeded generators in paper_2607_14530_gb300.synth; expected values come
from oracle/ only.  A case whose routing has a near tie (two routed scores closer than the
rounding of the fp32 kernels can separate) is re-drawn with the next seed before anything runs:
the oracle decides which inputs are used, never the kernels."""
from __future__ import annotations

import torch

from oracle import xhc_oracle as O
from paper_2607_14530_gb300 import synth
from paper_2607_14530_gb300.xhc import Config

F64 = torch.float64

# tolerances: bf16 state/outputs max abs 2e-2 (scaled by max(1, |ref|) for values above unit
# magnitude, where one bf16 ulp alone exceeds 2e-2) and relative L2 5e-3; fp32 coefficients and
# parameter gradients 1e-4 relative, element by element: |g - r| <= 1e-4 (|r| + rms(r)) (the
# tensor's RMS is the floor that keeps the bound defined at r = 0), and relative L2 <= 1e-4.
# Gating scalars alpha: |g - r| <= 1e-4 |r| + 2^-20 sum|terms| -- the sum of T x (map size) terms
# with cancellation, each term known to ~16 fp32 roundoffs (2^-24 each) of its magnitude.
BF16_ABS = 2e-2
BF16_REL_L2 = 5e-3
F32_REL = 1e-4
ALPHA_TERM_REL = 2.0 ** -20
# Routing ties: the kernels rank the routed streams by router logit (the sigmoid is monotone),
# and their logits carry the relative error of the bf16 hi/lo weight split (~1e-5 at worst).
# Two routed logits closer than TIE_LOGIT x max(1, |logit|) may be ordered either way; inputs
# with such a near tie are re-drawn (the oracle decides, never the kernels).
TIE_LOGIT = 1e-4
# An intermediate active state (xHC-Flash slots t >= 1) is stored in bf16; where its exact value
# lies within delta x (the magnitude of its terms) of a bf16 rounding midpoint, an fp32
# evaluation of the same sum may round to either bracketing value.  The kernels' largest error in
# that sum comes from the routing weight p, whose router logit carries the relative error of the
# bf16 hi/lo weight split (~2.5e-6 RMS) and of fp32 accumulation over K = N*C products (up to
# ~2e-6 at K = 65536), times the logit's magnitude (~1.3 RMS at N*C = 4096, ~5 at 65536).
# AMBIG_DELTA = 2^-18 (64 fp32 roundoffs) is four times the largest distance at which the kernels
# were seen to round the other way at K <= 8192 (2^-19.9); at K = 65536 the band is widened to
# AMBIG_DELTA_65536 = 2^-14 for the same reason scaled by the logits' magnitude and accumulation
# length.  These states are checked against the band; everything downstream of them is checked
# on a run whose intermediate states are the oracle's own (group_forward with inject).
AMBIG_DELTA = 2.0 ** -18
AMBIG_DELTA_65536 = 2.0 ** -14


def oracle_cfg(cfg: Config) -> O.Config:
    return O.Config(N=cfg.N, k=cfg.k, m=cfg.m, C=cfg.C, G=cfg.G,
                    mlp=tuple(bool((cfg.mlp_mask >> t) & 1) for t in range(cfg.G)),
                    conv_k=tuple(cfg.conv_k), gram_schmidt=cfg.gram_schmidt,
                    sinkhorn_iters=cfg.sinkhorn_iters, eps_norm=cfg.eps_norm,
                    eps_gs=(cfg.eps_gs if cfg.eps_gs > 0 else None), seq_len=cfg.seq_len,
                    router=cfg.router, dense_read=not cfg.sparse_read)


def tie_free(cfg: Config, X: torch.Tensor, W_r: torch.Tensor) -> torch.Tensor:
    """Per token of X [T, N, C]: no two routed logits TopK separates lie within TIE_LOGIT of
    each other (relative to max(1, the largest logit magnitude of the token))."""
    ocfg = oracle_cfg(cfg)
    T = X.shape[0]
    z = O.router_logits(ocfg, X.to(F64).reshape(T, -1), W_r.to(F64))
    return O.routing_margin(ocfg, z) > TIE_LOGIT * z.abs().amax(dim=1).clamp(min=1.0)


def make_case(cfg: Config, T: int, seed: int, alpha: float = 0.01, w_std: float = 0.02):
    """Seeded inputs and parameters with no near-tie in the routing (checked by the oracle)."""
    for attempt in range(50):
        s = seed + 1000 * attempt
        inp = synth.group_inputs(T, cfg.N, cfg.C, cfg.G, s)
        P = synth.params(cfg.param_shapes(), s, alpha=alpha, w_std=w_std)
        if not cfg.has_router:
            return inp, P, s
        if bool(tie_free(cfg, inp["X"], P["W_r"]).all()):
            return inp, P, s
    raise RuntimeError("no tie-free draw found")


def run_oracle(cfg: Config, inp, P, grads=None):
    ocfg = oracle_cfg(cfg)
    P64 = {n: v.to(F64) for n, v in P.items()}
    X = inp["X"].to(F64)
    outs = [o.to(F64) for o in inp["outs"]]
    Xo, ins, aux = O.forward(ocfg, P64, X, outs)
    res = dict(X=Xo, inputs=ins, aux=aux)
    if grads is not None:
        dX, douts, dP = O.backward(ocfg, P64, X, outs, grads["dX"].to(F64),
                                   [d.to(F64) for d in grads["d_inputs"]])
        res.update(dX=dX, d_outs=douts, dP=dP)
    return res


def ambiguity_delta(cfg: Config) -> float:
    return AMBIG_DELTA if cfg.N * cfg.C <= 8192 else AMBIG_DELTA_65536


def ambiguity_masks(cfg: Config, aux, delta: float | None = None) -> dict:
    """For every slot t >= 1, the elements of the active state entering slot t whose bf16
    rounding an fp32 evaluation may take either way: the exact value lies within AMBIG_DELTA x
    mag of the midpoint between its two bracketing bf16 values, or an earlier slot's state was
    ambiguous at the same (token, slot, channel) (the value is carried forward: Eq.
    flash_attn_update adds to it)."""
    delta = ambiguity_delta(cfg) if delta is None else delta
    masks, prev = {}, None
    for t in range(1, cfg.G):
        v, mag = aux["pre"][t], aux["mag"][t]
        r = v.to(torch.bfloat16).to(F64)
        mid = 0.5 * (r + O.bf16_other_neighbor(v, r))
        A = (v - mid).abs() <= delta * mag
        if prev is not None:
            A = A | prev
        masks[t] = A
        prev = A
    return masks


def check_active_states(gpu_xact, aux, masks, cfg: Config, tag=""):
    """The active state entering every slot t >= 1 (bf16, from the kernels' saved copy): bit-
    identical to the oracle's except at the ambiguous elements, where it must be within the bf16
    tolerance.  Returns the error messages (empty: pass)."""
    errs = []
    for t in range(1, cfg.G):
        g = gpu_xact[t].detach().cpu().to(F64)
        o = aux["X_act"][t].to(F64)
        A = masks[t]
        bad = (g != o) & ~A
        if bool(bad.any()):
            i = int(bad.flatten().nonzero()[0])
            v, mag = aux["pre"][t], aux["mag"][t]
            r = v.to(torch.bfloat16).to(F64)
            d = ((v - 0.5 * (r + O.bf16_other_neighbor(v, r))).abs() / mag)[bad]
            errs.append(f"{tag}x_act[{t}]: {int(bad.sum())} of {g.numel()} elements differ outside the "
                        f"ambiguity band ({int(A.sum())} in it; their distance to the midpoint up to "
                        f"2^{float(torch.log2(d.max())):.1f} of the term magnitude; first: gpu "
                        f"{float(g.flatten()[i])} oracle {float(o.flatten()[i])})")
        far = ((g - o).abs() > BF16_ABS * o.abs().clamp(min=1.0)) & A
        if bool(far.any()):
            errs.append(f"{tag}x_act[{t}]: {int(far.sum())} ambiguous elements beyond the bf16 bound")
    return errs


def alpha_term_scales(cfg: Config, inp, P, grads):
    """For each gating scalar alpha, the sum over tokens and map entries of |d L / d alpha| taken
    term by term (the oracle's forward broadcasts alpha, so passing it per entry gives the
    per-term contributions).  A scalar gradient is a sum of T * (map size) such terms with
    cancellation; its floating-point error scale is this sum of magnitudes, not |sum|."""
    ocfg = oracle_cfg(cfg)
    T = inp["X"].shape[0]
    P64 = {n: v.to(F64) for n, v in P.items()}
    X = inp["X"].to(F64)
    outs = [o.to(F64) for o in inp["outs"]]
    k, N, G = cfg.k, cfg.N, cfg.G
    a_pre = [torch.full((T, N), float(P64["alpha_pre"][t]), dtype=F64, requires_grad=True) for t in range(G)]
    a_post = [torch.full((T, k, cfg.K(t)), float(P64["alpha_post"][t]), dtype=F64, requires_grad=True)
              for t in range(G)]
    a_res = torch.full((1, T, k, k), float(P64["alpha_res"][0]), dtype=F64, requires_grad=True)
    Pp = dict(P64)
    Pp["alpha_pre"], Pp["alpha_post"], Pp["alpha_res"] = a_pre, a_post, a_res
    Xo, ins, _ = O.forward(ocfg, Pp, X, outs)
    L = (Xo * grads["dX"].to(F64)).sum() + sum((a * d.to(F64)).sum() for a, d in zip(ins, grads["d_inputs"]))
    g = torch.autograd.grad(L, a_pre + a_post + [a_res])
    return dict(alpha_pre=torch.stack([x.abs().sum() for x in g[:G]]),
                alpha_post=torch.stack([x.abs().sum() for x in g[G:2 * G]]),
                alpha_res=g[-1].abs().sum().reshape(1))


def assert_alpha_close(gpu, ref, scale, name, tol=F32_REL, allow=None):
    """Gating scalars: |g - r| <= tol |r| + ALPHA_TERM_REL * scale (+ allow)."""
    g = gpu.detach().to("cpu", F64)
    r = ref.detach().to("cpu", F64)
    err = (g - r).abs()
    bound = tol * r.abs() + ALPHA_TERM_REL * scale.to(F64)
    if allow is not None:
        bound = bound + allow
    bad = err > bound
    assert not bool(bad.any()), (f"{name}: error {err.tolist()} vs bound {bound.tolist()} "
                                 f"(|ref| {r.abs().tolist()}, term scale {scale.tolist()})")


def bf16_ulps(x: torch.Tensor) -> torch.Tensor:
    """bf16 spacing at |x| (2^(floor(log2|x|) - 7)), at least the smallest normal's spacing."""
    a = x.abs().clamp(min=2.0 ** -126)
    return torch.exp2(torch.floor(torch.log2(a)) - 7)


def assert_bf16_close(gpu, ref, name, scale=None):
    """|g - r| <= 2e-2 max(1, |r|, scale) element by element (scale: the magnitude of a bf16
    intermediate the result was formed from, whose half-ulp error it inherits) and relative L2
    <= 5e-3.  Reports the worst error in bf16 ulps of max(1, |r|, scale)."""
    g = gpu.detach().to("cpu", F64)
    r = ref.detach().to("cpu", F64)
    assert g.shape == r.shape, (name, g.shape, r.shape)
    err = (g - r).abs()
    mag = r.abs().clamp(min=1.0)
    if scale is not None:
        mag = torch.maximum(mag, scale.detach().to("cpu", F64).abs())
    bound = BF16_ABS * mag
    bad = err > bound
    if bool(bad.any()):
        q = err / bound
        i = int(q.argmax())
        ulps = float((err / bf16_ulps(mag)).max())
        raise AssertionError(
            f"{name}: {int(bad.sum())} elements over bound, worst err {float(err.flatten()[i]):.3e} "
            f"at ref {float(r.flatten()[i]):.4f} (bound {float(bound.flatten()[i]):.3e}; worst "
            f"{ulps:.1f} bf16 ulps of max(1, |ref|))")
    rel = float((g - r).norm() / r.norm().clamp(min=1e-30))
    assert rel <= BF16_REL_L2, f"{name}: relative L2 {rel:.3e}"


def flash_bases(cfg: Config, X: torch.Tensor, aux) -> list:
    """|base^t| per token and channel for the slots t >= 1 of an xHC-Flash group (None for slot
    0): the non-active dense readout sum_{i not in I} H_pre^t_i x_i of Eq. app_four_sub_base,
    which the kernels store in bf16 (as the paper's traffic model counts it) and to which they add
    the active streams' term (Eq. app_active_state_correction)."""
    T = X.shape[0]
    inactive = torch.ones(T, cfg.N, dtype=F64)
    inactive[torch.arange(T)[:, None], aux["I"]] = 0
    Xf = X.to(F64)
    return [None] + [torch.einsum("ti,tic->tc", aux["H_pre"][t].detach() * inactive, Xf).abs()
                     for t in range(1, cfg.G)]


def assert_f32_close(gpu, ref, name, tol=F32_REL, allow=None):
    """Element by element |g - r| <= tol (|r| + rms(r)) + allow, and relative L2 of the error
    beyond the allowance <= tol."""
    g = gpu.detach().to("cpu", F64)
    r = ref.detach().to("cpu", F64)
    assert g.shape == r.shape, (name, g.shape, r.shape)
    err = (g - r).abs()
    if r.numel() == 0:
        return
    rms = float(r.pow(2).mean().sqrt())
    excess = err if allow is None else (err - allow).clamp(min=0.0)
    ratio = excess / (r.abs() + rms).clamp(min=1e-300)
    worst = float(ratio.max())
    assert worst <= tol, (f"{name}: element-wise error {worst:.3e} of (|ref| + rms) at index "
                          f"{int(ratio.argmax())} (ref {float(r.flatten()[int(ratio.argmax())]):.4e})")
    nr = float(r.norm())
    rel = float(excess.norm()) / max(nr, 1e-30)
    assert rel <= tol, f"{name}: relative L2 {rel:.3e} (|ref| {nr:.3e})"


class Guarded:
    """A CUDA tensor with guard bands of a fixed pattern on both sides, to catch stray writes."""
    PAD = 4096

    def __init__(self, t: torch.Tensor):
        n = t.numel()
        self.big = torch.empty(n + 2 * self.PAD, dtype=t.dtype, device="cuda")
        self.big.view(torch.uint8).fill_(0xA5)
        self.t = self.big[self.PAD:self.PAD + n].view(t.shape)
        self.t.copy_(t)

    def intact(self) -> bool:
        lo = self.big[:self.PAD].view(torch.uint8)
        hi = self.big[-self.PAD:].view(torch.uint8)
        return bool((lo == 0xA5).all()) and bool((hi == 0xA5).all())


def group_forward(g, cfg: Config, P, X, outs, saved, ws, inputs, inject=None):
    """pre_fwd / post_fwd of every slot through the C ABI.  With ``inject`` (the oracle's aux),
    the bf16 active state entering every slot t >= 1 is overwritten in ``saved`` with the
    oracle's own value before pre_fwd(t): the kernels then compute every later step from the same
    intermediate states as the oracle (oracle values into the CUDA path, never the reverse), so
    results downstream of those states can be compared without the ambiguity of their
    rounding.  The kernels' own roundings are checked separately (check_active_states)."""
    T = X.shape[0]
    pp = g.params(P)
    xact = g.coefficients(saved, T)["xact"] if inject is not None else None
    for t in range(cfg.G):
        if inject is not None and t >= 1:
            xact[t].copy_(inject["X_act"][t].to(torch.bfloat16))
        g.pre_fwd(t, pp, X, inputs[t], saved, ws)
        g.post_fwd(t, pp, X, outs[t], saved, ws)
