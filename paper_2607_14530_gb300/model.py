"""Model glue: stacks of connection-op groups under torch.autograd.

A model with expanded residual streams runs, per token: the embedding output expanded to N
streams; for every group, its G sublayers (attention / MLP, the caller's modules) each between a
pre- and a post-call of the connection op; the N streams summed back to one hidden vector before
the final RMSNorm and the unembedding (App. A, "Final Stream Reduction").  This module chains
those steps for autograd; every step of the connection op itself runs in libxhc's kernels
(``Group`` of xhc.py), the sublayers in whatever the caller's modules run.

* ``StreamExpand`` / ``StreamSum``: xhc_stream_expand / xhc_stream_sum, each other's backward.
* ``XhcGroup``: one group's parameters (fp32 ``nn.Parameter``) and sublayers.  Its forward runs
  pre_fwd(t), sublayer t, post_fwd(t) for every slot, recording each sublayer's own autograd
  graph; its backward runs post_bwd(t), the sublayer's backward (autograd on the recorded graph),
  pre_bwd(t) in reverse slot order.  The residual state is updated in place (xhc.h: the library
  writes the k active rows of X and restores them in the backward), so the state tensor flows
  through the groups of a stack without copies; the library's saved / workspace buffers are kept
  per group and per token count.  So does the state gradient: a group's backward updates the
  gradient it receives in place when that tensor is the one the next group or the stream sum
  returned and no hook or retain_grad watches the state; any other incoming gradient is copied
  first.
* ``XhcStack``: expansion, L groups, stream sum.
"""
from __future__ import annotations

import torch
from torch import nn

from . import synth
from .xhc import Config, Group


def _owned(t: torch.Tensor) -> torch.Tensor:
    """Mark a state gradient this module created and hands on to autograd (nothing else keeps it):
    the group whose backward receives it next updates it in place instead of copying it."""
    t._xhc_owned = True
    return t


class StreamExpand(torch.autograd.Function):
    """hidden [T, C] -> X [T, N, C] (N copies); backward: the sum of the N stream gradients."""

    @staticmethod
    def forward(ctx, hidden, g):
        ctx.g = g
        return g.stream_expand(hidden.contiguous())

    @staticmethod
    def backward(ctx, dX):
        return ctx.g.stream_sum(dX.contiguous()), None


class StreamSum(torch.autograd.Function):
    """X [T, N, C] -> y [T, C] (sum of the N streams); backward: the gradient to every stream."""

    @staticmethod
    def forward(ctx, X, g):
        ctx.g = g
        return g.stream_sum(X.contiguous())

    @staticmethod
    def backward(ctx, dy):
        return _owned(ctx.g.stream_expand(dy.contiguous())), None


class _GroupFn(torch.autograd.Function):
    @staticmethod
    def forward(ctx, X, mod, *pvals):
        g, cfg = mod.g, mod.cfg
        T = X.shape[0]
        saved, ws = mod.buffers(T, X.device)
        P = mod.param_dict()
        pp = g.params(P)
        leaves, outs = [], []
        for t in range(cfg.G):
            inp = torch.empty(T, cfg.C, dtype=torch.bfloat16, device=X.device)
            g.pre_fwd(t, pp, X, inp, saved, ws)
            with torch.enable_grad():
                leaf = inp.detach().requires_grad_(True)
                out = mod.sublayers[t](leaf)
            if out.shape != (T, cfg.C):
                raise ValueError(f"sublayer {t} must return [T, C], got {tuple(out.shape)}")
            out_b = out.detach().to(torch.bfloat16).contiguous()
            g.post_fwd(t, pp, X, out_b, saved, ws)
            leaves.append(leaf)
            outs.append((out, out_b))
        ctx.mark_dirty(X)
        # the state is restored in place by the backward of the next group before this group's
        # backward runs, so it is kept as a plain reference (the in-place contract of xhc.h)
        ctx.mod, ctx.X, ctx.io = mod, X, (saved, ws, leaves, outs)
        return X

    @staticmethod
    def backward(ctx, dX_out):
        mod, X = ctx.mod, ctx.X
        saved, ws, leaves, outs = ctx.io
        g, cfg = mod.g, mod.cfg
        T = X.shape[0]
        # the incoming gradient is updated in place only when it is the next group's (or the
        # stream sum's) own result and nothing else can hold it: a hook or retain_grad on the
        # state (they follow the state tensor through the groups' in-place updates) receives
        # that same tensor, so then it is copied first
        state_watched = ctx.X.retains_grad or bool(ctx.X._backward_hooks)
        if (getattr(dX_out, "_xhc_owned", False) and not state_watched and dX_out.dtype == torch.bfloat16
                and dX_out.is_contiguous()):
            dX = dX_out
        else:
            dX = dX_out.to(torch.bfloat16).contiguous().clone()
        P = mod.param_dict()
        grads = {n: torch.zeros_like(v) for n, v in P.items()}
        pp, gg = g.params(P), g.params(grads)
        for t in reversed(range(cfg.G)):
            out, out_b = outs[t]
            d_out = torch.empty(T, cfg.C, dtype=torch.bfloat16, device=X.device)
            g.post_bwd(t, pp, X, dX, out_b, d_out, gg, saved, ws)
            with torch.enable_grad():
                torch.autograd.backward(out, d_out.to(out.dtype))
            d_in = leaves[t].grad
            if d_in is None:
                d_in = torch.zeros(T, cfg.C, dtype=torch.bfloat16, device=X.device)
            g.pre_bwd(t, pp, X, d_in.to(torch.bfloat16).contiguous(), dX, gg, saved, ws)
        ctx.io = None
        return (_owned(dX), None) + tuple(grads[n] for n in mod.names)


class XhcGroup(nn.Module):
    """One connection-op group with its sublayers (G modules mapping [T, C] bf16 to [T, C])."""

    def __init__(self, cfg: Config, sublayers, seed: int = 0, alpha: float = 0.01, w_std: float = 0.02):
        super().__init__()
        if len(sublayers) != cfg.G:
            raise ValueError(f"{cfg.G} sublayers needed")
        self.cfg = cfg
        self.g = Group(cfg)
        self.sublayers = nn.ModuleList(sublayers)
        self.names = list(cfg.param_shapes())
        init = synth.params(cfg.param_shapes(), seed, alpha=alpha, w_std=w_std)
        for n in self.names:
            self.register_parameter(n.replace(".", "_"), nn.Parameter(init[n].clone()))
        self._bufs = {}

    def param_dict(self) -> dict:
        return {n: getattr(self, n.replace(".", "_")).detach().contiguous() for n in self.names}

    def buffers(self, T: int, device):
        """(saved, workspace) for one forward call: a fresh `saved` (it carries this call's
        forward state to its backward, so two forwards in flight, e.g. two micro-batches before
        one backward, must not share it; the caching allocator makes it cheap) and the workspace
        kept per token count (scratch, reusable between the phases of calls)."""
        return self.g.alloc_saved(T, device=device), self.buffers_workspace(T, device)

    def buffers_workspace(self, T: int, device):
        key = (T, str(device))
        if key not in self._bufs:
            self._bufs[key] = self.g.alloc_workspace(T, device=device)
        return self._bufs[key]

    def forward(self, X):
        if not torch.is_grad_enabled():
            return self._forward_inference(X)
        return _GroupFn.apply(X, self, *[getattr(self, n.replace(".", "_")) for n in self.names])

    def _forward_inference(self, X):
        """The forward without autograd (grad mode off: prefill or evaluation): the same calls,
        the sublayers run without recording a graph, and `saved` is scratch kept per token count
        (no backward will read it)."""
        g, cfg = self.g, self.cfg
        T = X.shape[0]
        key = ("scratch", T, str(X.device))
        if key not in self._bufs:
            self._bufs[key] = g.alloc_saved(T, device=X.device)
        saved, ws = self._bufs[key], self.buffers_workspace(T, X.device)
        pp = g.params(self.param_dict())
        for t in range(cfg.G):
            inp = torch.empty(T, cfg.C, dtype=torch.bfloat16, device=X.device)
            g.pre_fwd(t, pp, X, inp, saved, ws)
            out = self.sublayers[t](inp)
            if out.shape != (T, cfg.C):
                raise ValueError(f"sublayer {t} must return [T, C], got {tuple(out.shape)}")
            g.post_fwd(t, pp, X, out.to(torch.bfloat16).contiguous(), saved, ws)
        return X


class XhcStack(nn.Module):
    """Embedding output [T, C] -> N streams -> L groups -> sum of the streams [T, C]."""

    def __init__(self, cfg: Config, n_groups: int, make_sublayer, seed: int = 0, **kw):
        super().__init__()
        self.cfg = cfg
        self.groups = nn.ModuleList(
            XhcGroup(cfg, [make_sublayer(l, t) for t in range(cfg.G)], seed=seed + 97 * l, **kw)
            for l in range(n_groups))

    def forward(self, hidden):
        g = self.groups[0].g
        X = StreamExpand.apply(hidden, g)
        for grp in self.groups:
            X = grp(X)
        return StreamSum.apply(X, g)
