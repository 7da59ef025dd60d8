"""fp64 CPU oracle of the xHC connection op (arXiv 2607.14530, "xHC: Expanded Hyper-Connections").

TEST INFRASTRUCTURE ONLY.  Only tests/, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this module.  The product path (libxhc and its Python binding) never
imports, links or calls anything under ``oracle/``, and this module imports nothing from the
product package.

This is a plain, slow, vectorised-over-tokens restatement of the paper's equations in float64
(PyTorch CPU ops as library primitives: matmul, sort, exp).  No blocking, fusion or reordering
beyond what the equations state: the router uses the literal LayerNorm of the flattened state
(Eq. router), the pre-map the literal RMSNorm (Eq. param_pre), every sublayer input is the literal
dense read of the *current* full state (Eq. dense_read; for xHC-Flash the state after the
preceding sparse write-backs, which App. E.2 shows the base/active correction reproduces), and the
write-back materialises the augmented components, the Gram-Schmidt basis and the scatter.

Backward: exact reverse-mode derivative of this forward, taken by ``torch.autograd`` in float64
(a library primitive computing the plain definition of the gradient).  Storage rounding to bf16
is treated as the identity in the backward (straight-through), as the kernels do.

Sources (section / equation labels of the paper):
  Sec. 3.1     Eq. hc (HC update), Eq. mhc_sinkhorn (Sinkhorn-projected residual mixing)
  Sec. 3.3.1   Eq. aug (temporal feature augmentation), Eq. gs (Gram-Schmidt)
  Sec. 3.3.2   Eq. router, Eq. router_topk, Eq. dense_read, Eq. sparse_hres, Eq. sparse_hpost,
               Eq. sparse_write_delta, Eq. sparse_write
  Sec. 3.3.4   Eq. param_pre, Eq. param_res, Eq. param_post and the causal depthwise conv formula
  Alg. 1       one xHC sublayer;  Alg. 2 / Sec. 5.2  xHC-Flash block;  App. E.2  4-sublayer group
  App. A       20 Sinkhorn iterations, row-sum clamp, alpha initialised to 0.01
  App. C       per-layer parameter counts (Eq. xhc_params, Eq. mhc_params)

Readings where the paper is silent (the same readings are used by the kernels):
  eps_norm = 1e-5 for every LayerNorm / RMSNorm (the backbone RMSNorm epsilon, App. A table);
  no affine weights in those norms; LayerNorm variance is the population variance nu - mu^2;
  FixedIdx = streams 0..m-1; routed streams are taken by score descending, ties to the lower
  stream index; active slot order = fixed ascending, then routed by rank;
  mat_{a x b} is row-major (H[j][r] = z[j*b + r]); row j of H_res is destination slot j;
  one Sinkhorn iteration = row normalisation then column normalisation, no epsilon;
  row-sum clamp divides a row by max(rowsum, 1) and at rowsum == 1 exactly takes the
  un-clamped branch;  Gram-Schmidt is Eq. gs literally (numerator <g_j, v_i>) with denominator
  <v_i, v_i> + eps_gs, eps_gs = 1e-6 * C, no unit normalisation;  the conv has no bias, tap i=0
  is the current token and it restarts (zero padding) at every sequence start, tokens being
  sequence-major (t = b*S + s);  alpha is one scalar per map, b has the map's shape;
  xHC-Flash slots alternate Attention (K=1) and MLP (K=1+r, temporal augmentation), each slot
  has its own post-map weights computed from the current active state, H_res only at the last
  slot of the group;  bf16 rounding is applied exactly where the library stores bf16: the
  sublayer inputs, the active state after every write-back, and the written state rows.
"""
from __future__ import annotations

from dataclasses import dataclass, field
import itertools

import torch

F64 = torch.float64


@dataclass(frozen=True)
class Config:
    """Shape and hyper-parameters of one connection-op group.

    A group is G consecutive sublayers sharing one routing decision and one full-state
    mapping generation (G = 1: full xHC or mHC, Alg. 1; G = 2: xHC-Flash, Alg. 2; G = 4:
    xHC-Flash-4sub, App. E.2).  ``mlp[t]`` marks slot t as an MLP sublayer, which receives the
    temporal feature augmentation (Sec. 3.3.1) when ``conv_k`` is non-empty.
    """
    N: int
    k: int
    m: int
    C: int
    G: int = 1
    mlp: tuple = (False,)
    conv_k: tuple = (4, 8, 12)
    gram_schmidt: bool = True
    sinkhorn_iters: int = 20
    eps_norm: float = 1e-5
    eps_gs: float | None = None
    seq_len: int = 0
    router: str = "sigmoid"     # "softmax": the softmax-router ablation (Table ablation, row 11)
    dense_read: bool = True     # False: read only the active streams (Table ablation, rows 6-7)

    @property
    def has_router(self) -> bool:
        # Eq. router_topk: only the k - m routed streams use the router scores.
        return self.m < self.k

    def K(self, t: int) -> int:
        """Number of write-back components of slot t (K_r = r + 1 for MLP, 1 for Attention)."""
        return 1 + len(self.conv_k) if (self.mlp[t] and len(self.conv_k) > 0) else 1

    def gs_eps(self) -> float:
        return self.eps_gs if self.eps_gs is not None else 1e-6 * self.C

    def S(self, T: int) -> int:
        return self.seq_len if self.seq_len > 0 else T


def mhc(N: int, C: int, **kw) -> Config:
    """mHC (Sec. 3.1): every stream active, no router, single write-back signal."""
    return Config(N=N, k=N, m=N, C=C, G=1, mlp=(False,), conv_k=(), **kw)


def full(N: int, k: int, m: int, C: int, mlp: bool, **kw) -> Config:
    """One full-xHC sublayer (Alg. 1): Attention (mlp=False, K_r = 1) or MLP (K_r = 4)."""
    return Config(N=N, k=k, m=m, C=C, G=1, mlp=(bool(mlp),), **kw)


def flash(N: int, k: int, m: int, C: int, G: int, **kw) -> Config:
    """xHC-Flash group of G sublayers, slots Attention, MLP, Attention, MLP (Sec. 5.2)."""
    return Config(N=N, k=k, m=m, C=C, G=G, mlp=tuple(t % 2 == 1 for t in range(G)), **kw)


# ----------------------------------------------------------------------------------------------
# parameters


def param_shapes(cfg: Config) -> dict:
    """Shapes of every learnable tensor of one group (Sec. 3.3.4, Sec. 5.2).

    W_r: [N*C, N] (Eq. router); W_pre[t]: [N*C, N] (Eq. param_pre); W_res: [k*C, k*k]
    (Eq. param_res); W_post[t]: [k*C, k*K_t] (Eq. param_post); conv_w[t][j]: [kappa_j, C]
    (conv formula, Sec. 3.3.4); alpha_*: one scalar per map; b_*: the map's shape.
    """
    N, k, C, G = cfg.N, cfg.k, cfg.C, cfg.G
    sh = {}
    if cfg.has_router:
        sh["W_r"] = (N * C, N)
    for t in range(G):
        sh[f"W_pre.{t}"] = (N * C, N)
        sh[f"W_post.{t}"] = (k * C, k * cfg.K(t))
        sh[f"b_post.{t}"] = (k * cfg.K(t),)
        if cfg.K(t) > 1:
            for j, kap in enumerate(cfg.conv_k):
                sh[f"conv_w.{t}.{j}"] = (kap, C)
    sh["alpha_pre"] = (G,)
    sh["b_pre"] = (G, N)
    sh["alpha_post"] = (G,)
    sh["W_res"] = (k * C, k * k)
    sh["alpha_res"] = (1,)
    sh["b_res"] = (k * k,)
    return sh


def layer_param_count_over_C(cfgs) -> float:
    """Sum of the C-proportional parameter counts (all W and conv tensors) over the given
    sublayer configs, divided by C: the quantity Eq. xhc_params / Eq. mhc_params report."""
    tot = 0
    for cfg in cfgs:
        for name, shp in param_shapes(cfg).items():
            if name.startswith(("W_", "conv_w")):
                n = 1
                for d in shp:
                    n *= d
                tot += n
    return tot / cfgs[0].C


def to_oracle_params(flat: dict, cfg: Config, requires_grad: bool = False) -> dict:
    """Turn a flat ``{name: tensor}`` dict (names as in :func:`param_shapes`) into float64
    leaves.  Returns the same flat layout."""
    out = {}
    for name in param_shapes(cfg):
        v = flat[name].detach().to(F64).clone()
        if requires_grad:
            v.requires_grad_(True)
        out[name] = v
    return out


# ----------------------------------------------------------------------------------------------
# building blocks


def bf16_other_neighbor(v: torch.Tensor, r: torch.Tensor) -> torch.Tensor:
    """The bf16 value next to r on the side of v, where r is v rounded to bf16 (r itself where
    v == r exactly).  Together r and this value bracket v: they are the two roundings that an
    evaluation of v with an error across the midpoint between them can produce."""
    bits = r.to(torch.bfloat16).view(torch.int16).to(torch.int32) & 0xFFFF
    neg = (bits >> 15) == 1
    mag = bits & 0x7FFF
    up = v > r                                    # the neighbour lies towards +infinity
    away = torch.where(neg, ~up, up)              # ... i.e. away from zero in magnitude
    mag2 = torch.where(away, mag + 1, mag - 1)
    bits2 = torch.where(neg, mag2 | 0x8000, mag2)
    zero = mag == 0                               # r = +-0: smallest subnormal of v's sign
    bits2 = torch.where(zero, torch.where(v < 0, torch.full_like(bits, 0x8001),
                                          torch.full_like(bits, 0x0001)), bits2)
    bits2 = torch.where(v == r, bits, bits2)
    out = (bits2 - ((bits2 >> 15) << 16)).to(torch.int16).view(torch.bfloat16)
    return out.to(v.dtype)


def rnd(x: torch.Tensor, on: bool) -> torch.Tensor:
    """Round to bf16 storage (round-to-nearest-even); identity in the backward."""
    if not on:
        return x
    return x + (x.to(torch.bfloat16).to(x.dtype) - x).detach()


def sinkhorn(M: torch.Tensor, iters: int) -> torch.Tensor:
    """SK(exp(M)) of Eq. mhc_sinkhorn: alternate row and column normalisation of exp(M)."""
    A = torch.exp(M)
    for _ in range(iters):
        A = A / A.sum(dim=-1, keepdim=True)
        A = A / A.sum(dim=-2, keepdim=True)
    return A


def row_clamp(H: torch.Tensor) -> torch.Tensor:
    """App. A: replace each row by row / max(rowsum, 1) (rowsum == 1: un-clamped branch)."""
    s = H.sum(dim=-1, keepdim=True)
    return H / torch.where(s > 1.0, s, torch.ones_like(s))


def causal_dwconv(out: torch.Tensor, w: torch.Tensor, S: int, hist: torch.Tensor | None = None) -> torch.Tensor:
    """g[t] = sum_{i=0}^{kappa-1} w[i] * out[t-i] channel-wise (Sec. 3.3.4), zero before the
    start of each length-S sequence.  out: [T, C], w: [kappa, C].

    ``hist`` [B, R, C] (B = T / S): the R outputs that precede each of the B sequences, when the
    call holds a later chunk of longer sequences (sequence split); out[t - i] before the chunk's
    first token is then hist[b][R + (t - i) - b S] (zero before that)."""
    if hist is not None:
        B, R, C = hist.shape
        ext = torch.cat([hist, out.reshape(B, S, C)], dim=1).reshape(B * (R + S), C)
        return causal_dwconv(ext, w, R + S).reshape(B, R + S, C)[:, R:].reshape(B * S, C)
    T = out.shape[0]
    pos = torch.arange(T) % S
    g = torch.zeros_like(out)
    for i in range(w.shape[0]):
        shifted = torch.zeros_like(out)
        if i < T:
            shifted[i:] = out[: T - i]
        valid = (pos >= i).to(out.dtype)[:, None]
        g = g + w[i][None, :] * shifted * valid
    return g


def gram_schmidt(out: torch.Tensor, gs: list, eps: float) -> list:
    """Eq. gs per token along C: v_1 = out, v_{j+1} = g_j - sum_{i<=j} <g_j,v_i>/<v_i,v_i> v_i."""
    v = [out]
    for g in gs:
        vn = g
        for vi in v:
            coef = (g * vi).sum(dim=1, keepdim=True) / ((vi * vi).sum(dim=1, keepdim=True) + eps)
            vn = vn - coef * vi
        v.append(vn)
    return v


def augment(cfg: Config, out: torch.Tensor, conv_ws: list, T: int, hist: torch.Tensor | None = None) -> list:
    """out_aug of Eq. aug (after Eq. gs when enabled): K_r = r + 1 components, each [T, C].
    ``hist``: the outputs preceding each sequence of a later chunk (see causal_dwconv)."""
    S = cfg.S(T)
    gs = [causal_dwconv(out, w, S, hist) for w in conv_ws]
    if cfg.gram_schmidt:
        return gram_schmidt(out, gs, cfg.gs_eps())
    return [out] + gs


def router_logits(cfg: Config, x: torch.Tensor, W_r: torch.Tensor) -> torch.Tensor:
    """LN(flatten X) W_r, the argument of the sigmoid in Eq. router.  x: [T, N*C]."""
    mu = x.mean(dim=1, keepdim=True)
    nu = (x * x).mean(dim=1, keepdim=True)
    x_ln = (x - mu) / torch.sqrt(nu - mu * mu + cfg.eps_norm)
    return x_ln @ W_r


def router_scores(cfg: Config, x: torch.Tensor, W_r: torch.Tensor) -> torch.Tensor:
    """s = sigmoid(LN(flatten X) W_r) (Eq. router).  x: [T, N*C].  With the softmax-router
    ablation (Sec. 4, Table ablation row 11) the sigmoid is replaced by a softmax over the N
    logits of the token (the fixed streams' logits included, as the projection produces all N)."""
    z = router_logits(cfg, x, W_r)
    if cfg.router == "softmax":
        return torch.softmax(z, dim=1)
    return torch.sigmoid(z)


def route(cfg: Config, s: torch.Tensor | None, T: int):
    """Eq. router_topk: I = FixedIdx u TopK_{i>m}(s, k-m); p_j = 1 (fixed) or s_{I_j}.

    Returns I [T, k] (int64) and p [T, k] (differentiable through s)."""
    m, k = cfg.m, cfg.k
    fixed = torch.arange(m).expand(T, m)
    if k == m:
        return fixed.clone(), torch.ones(T, k, dtype=F64)
    order = torch.sort(s[:, m:].detach(), dim=1, descending=True, stable=True).indices[:, : k - m] + m
    I = torch.cat([fixed, order], dim=1)
    p = torch.cat([torch.ones(T, m, dtype=s.dtype), s.gather(1, order)], dim=1)
    return I, p


def routing_margin(cfg: Config, s: torch.Tensor) -> torch.Tensor:
    """Per token, the smallest gap between consecutive routed scores among the top k-m+1
    (sorted descending).  A small gap means another choice / slot order is equally valid up to
    rounding.  Returns +inf when there is nothing to choose."""
    T = s.shape[0]
    if not cfg.has_router:
        return torch.full((T,), float("inf"), dtype=F64)
    srt = torch.sort(s[:, cfg.m:].detach(), dim=1, descending=True).values
    n = min(cfg.k - cfg.m + 1, srt.shape[1])
    if n < 2:
        return torch.full((T,), float("inf"), dtype=F64)
    return (srt[:, : n - 1] - srt[:, 1:n]).min(dim=1).values


# ----------------------------------------------------------------------------------------------
# forward / backward of one group


def forward(cfg: Config, P: dict, X: torch.Tensor, outs: list, *, round_bf16: bool = True,
            halos: list | None = None):
    """One connection-op group: Alg. 1 (G = 1) or Alg. 2 / App. E.2 (G = 2, 4).

    X: [T, N, C] float64 holding the entry state; outs[t]: [T, C] float64, the caller's
    sublayer output of slot t (out^(t) = F_t(input^(t)) in the paper; here an input of the op),
    or a callable F_t applied to the slot's input (to compose groups with sublayers, Alg. 1).
    Returns (X_out, inputs, aux): the state after the group, the G sublayer inputs, and a dict
    of intermediates (s, H_pre, I, p, H_post, H_res, the active state before every slot).
    ``halos[t]`` ([B, R, C] or None): for a call holding a later chunk of its sequences, the
    sublayer outputs of slot t that precede each sequence (read by the causal conv only).

    For the tests, aux also holds, for every slot t >= 1 of a group, the active state entering
    slot t before its bf16 rounding (``pre[t]``) and the sum of the magnitudes of the terms that
    make it up (``mag[t]``: |X_act| plus p_j sum_r |H_post[j][r]| times the summed magnitudes of
    out and of the raw conv components), which bounds the error of any evaluation of that sum.
    """
    T, N, C = X.shape
    k, G, eps = cfg.k, cfg.G, cfg.eps_norm
    x = X.reshape(T, N * C)                         # flatten(X), stream-major: x[i*C + c]

    # Stream routing (Eq. router, Eq. router_topk), shared by the G sublayers.
    s = router_scores(cfg, x, P["W_r"]) if cfg.has_router else None
    I, p = route(cfg, s, T)

    # Pre-maps from the RMSNorm-normalised entry state (Eq. param_pre), one per sublayer.
    nu = (x * x).mean(dim=1, keepdim=True)
    x_rms = x / torch.sqrt(nu + eps)
    H_pre = [torch.sigmoid(P["alpha_pre"][t] * (x_rms @ P[f"W_pre.{t}"]) + P["b_pre"][t])
             for t in range(G)]

    rows = torch.arange(T)[:, None].expand(T, k)
    X_act = X[rows, I]                              # Gather(X, I): [T, k, C]
    # read mask: every stream (Eq. dense_read), or only the active ones (sparse-read ablation)
    read = torch.ones(T, N, dtype=X.dtype)
    if not cfg.dense_read:
        read = torch.zeros(T, N, dtype=X.dtype)
        read[rows, I] = 1.0
    X_cur = X
    inputs, H_post_all, X_act_all = [], [], []
    pre, mag = {}, {}
    H_res = None
    for t in range(G):
        X_act_all.append(X_act)
        # Dense read of the current full state (Eq. dense_read).
        inputs.append(rnd(torch.einsum("ti,tic->tc", H_pre[t] * read, X_cur), round_bf16))

        # Post- and residual maps from the RMSNorm-normalised current active state
        # (Eq. param_post, Eq. param_res with the App. A row clamp).
        xa = X_act.reshape(T, k * C)
        xt = xa / torch.sqrt((xa * xa).mean(dim=1, keepdim=True) + eps)
        K = cfg.K(t)
        Zp = (xt @ P[f"W_post.{t}"]).reshape(T, k, K)
        H_post = 2.0 * torch.sigmoid(P["alpha_post"][t] * Zp + P[f"b_post.{t}"].reshape(k, K))
        H_post_all.append(H_post)

        # Write-back components (Eq. aug + Eq. gs for MLP slots, out itself otherwise).
        hist = None if halos is None else halos[t]
        o_t = outs[t](inputs[t]) if callable(outs[t]) else outs[t]
        if K > 1:
            comps = augment(cfg, o_t, [P[f"conv_w.{t}.{j}"] for j in range(len(cfg.conv_k))], T, hist)
        else:
            comps = [o_t]
        out_aug = torch.stack(comps, dim=1)                       # [T, K, C]
        delta = p[:, :, None] * torch.einsum("tjr,trc->tjc", H_post, out_aug)  # Eq. sparse_write_delta

        if t == G - 1:
            Zr = (xt @ P["W_res"]).reshape(T, k, k)
            M = P["alpha_res"][0] * Zr + P["b_res"].reshape(k, k)
            H_res = row_clamp(sinkhorn(M, cfg.sinkhorn_iters))
            mixed = torch.einsum("tji,tic->tjc", H_res, X_act)   # H_res X_act
        else:
            mixed = X_act                                         # Eq. flash_attn_update
        new = mixed + delta                                       # Eq. sparse_write
        if t < G - 1:
            # magnitudes of the terms of the next slot's active state (test bookkeeping only)
            raw = [o_t] + ([causal_dwconv(o_t, P[f"conv_w.{t}.{j}"], cfg.S(T), hist)
                                for j in range(len(cfg.conv_k))] if K > 1 else [])
            mu = sum(c.detach().abs() for c in raw)                   # [T, C]
            hp = (p.detach().abs() * H_post.detach().abs().sum(dim=2))  # [T, k]
            pre[t + 1] = new.detach()
            mag[t + 1] = mixed.detach().abs() + hp[:, :, None] * mu[:, None, :]
        X_act = rnd(new, round_bf16)
        X_cur = torch.index_put(X_cur, (rows, I), X_act)          # Scatter: inactive rows unchanged

    aux = dict(s=s, I=I, p=p, H_pre=H_pre, H_post=H_post_all, H_res=H_res, X_act=X_act_all,
               pre=pre, mag=mag)
    return X_cur, inputs, aux


def backward(cfg: Config, P: dict, X: torch.Tensor, outs: list, dX_out: torch.Tensor,
             d_inputs: list, *, round_bf16: bool = True, halos: list | None = None):
    """Reverse mode of :func:`forward` for the loss L = <X_out, dX_out> + sum_t <input_t, d_input_t>.

    Returns (dX, d_outs, dP): the gradient w.r.t. the entry state, each sublayer output and every
    parameter (flat names as in :func:`param_shapes`).  No gradient flows through the TopK
    selection or the fixed p = 1 (Eq. router_topk); routing gradients reach W_r only through the
    selected routed scores p_j.

    With ``halos`` (see :func:`forward`) a fourth value is returned: the gradient w.r.t. every
    halo (None where the slot has none), which belongs to the previous chunk's sublayer outputs."""
    Xl = X.detach().clone().requires_grad_(True)
    outl = [o.detach().clone().requires_grad_(True) for o in outs]
    Pl = {n: v.detach().clone().requires_grad_(True) for n, v in P.items()}
    hl = None if halos is None else [None if h is None else h.detach().clone().requires_grad_(True)
                                     for h in halos]
    Xo, inputs, _ = forward(cfg, Pl, Xl, outl, round_bf16=round_bf16, halos=hl)
    L = (Xo * dX_out).sum()
    for inp, d in zip(inputs, d_inputs):
        L = L + (inp * d).sum()
    names = list(Pl)
    hx = [] if hl is None else [h for h in hl if h is not None]
    grads = torch.autograd.grad(L, [Xl] + outl + [Pl[n] for n in names] + hx, allow_unused=True)
    dX = grads[0]
    d_outs = list(grads[1:1 + len(outl)])
    dP = {}
    nP = 1 + len(outl) + len(names)
    for n, g in zip(names, grads[1 + len(outl):nP]):
        dP[n] = g if g is not None else torch.zeros_like(Pl[n])
    if hl is None:
        return dX, d_outs, dP
    dh, i = [], nP
    for h in hl:
        if h is None:
            dh.append(None)
        else:
            dh.append(grads[i] if grads[i] is not None else torch.zeros_like(h))
            i += 1
    return dX, d_outs, dP, dh
