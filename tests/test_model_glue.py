"""Autograd wiring of the model glue (paper_2607_14530_gb300.model) on CPU, with a stand-in for
the library's calls: the slot order of the forward (pre_fwd(t), sublayer t, post_fwd(t)) and of
the backward (post_bwd(t), the sublayer's backward, pre_bwd(t), in reverse slot order and reverse
group order), and the gradients that reach the embedding, the sublayers' parameters and the
group's parameters.  The stand-in's arithmetic is simple and mirrored by a plain-autograd
re-implementation; the library's own arithmetic is checked on the GPU (tests/test_gpu_model.py)."""
import torch
from torch import nn

from paper_2607_14530_gb300 import model as M
from paper_2607_14530_gb300.xhc import Config


class FakeGroup:
    """pre_fwd: input = mean over streams; post_fwd: every stream += a * out (a = W_post.t[0,0]);
    the backward calls are the exact reverses; bf16 storage as in the library."""

    def __init__(self, cfg, log, tag):
        self.cfg, self.log, self.tag = cfg, log, tag

    def params(self, P):
        return P

    def alloc_saved(self, T, device="cpu"):
        return {"T": T}           # a distinct object per forward call

    def alloc_workspace(self, T, device="cpu"):
        return None

    def stream_expand(self, h, X=None):
        return h[:, None, :].expand(h.shape[0], self.cfg.N, h.shape[1]).contiguous()

    def stream_sum(self, X, y=None):
        return X.float().sum(1).to(torch.bfloat16)

    def pre_fwd(self, t, P, X, inp, saved, ws):
        self.log.append((self.tag, "pre_fwd", t))
        inp.copy_(X.float().mean(1).to(torch.bfloat16))

    def post_fwd(self, t, P, X, out, saved, ws):
        self.log.append((self.tag, "post_fwd", t))
        a = P[f"W_post.{t}"][0, 0]
        X.copy_((X.float() + a * out.float()[:, None, :]).to(torch.bfloat16))

    def post_bwd(self, t, P, X, dX, out, d_out, gg, saved, ws):
        self.log.append((self.tag, "post_bwd", t))
        self.log.append((self.tag, "dX_ptr", dX.data_ptr()))
        a = P[f"W_post.{t}"][0, 0]
        X.copy_((X.float() - a * out.float()[:, None, :]).to(torch.bfloat16))   # restore the entry state
        d_out.copy_((a * dX.float().sum(1)).to(torch.bfloat16))
        gg[f"W_post.{t}"][0, 0] += (dX.float().sum(1) * out.float()).sum()

    def pre_bwd(self, t, P, X, d_in, dX, gg, saved, ws):
        self.log.append((self.tag, "pre_bwd", t))
        dX.copy_((dX.float() + d_in.float()[:, None, :] / self.cfg.N).to(torch.bfloat16))


class Scale(nn.Module):
    def __init__(self, v, log, tag):
        super().__init__()
        self.s = nn.Parameter(torch.tensor(float(v)))
        self.log, self.tag = log, tag

    def forward(self, x):
        self.log.append((self.tag, "sublayer", 0))
        y = x.float() * self.s
        if y.requires_grad:
            y.register_hook(lambda g: self.log.append((self.tag, "sublayer_bwd", 0)))
        return y


def test_group_chain_call_order_and_gradients():
    cfg = Config.flash(4, 2, 1, 8, 2, seq_len=3)
    log = []
    stack = M.XhcStack(cfg, 2, lambda l, t: Scale(0.5 if t == 0 else 2.0, log, (l, t)))
    for l, grp in enumerate(stack.groups):
        grp.g = FakeGroup(cfg, log, l)
        with torch.no_grad():
            for t in range(cfg.G):
                getattr(grp, f"W_post_{t}")[0, 0] = 0.25 * (1 + l + t)
    T = 6
    g = torch.Generator().manual_seed(0)
    h = torch.randn(T, cfg.C, generator=g).to(torch.bfloat16).requires_grad_(True)
    dy = torch.randn(T, cfg.C, generator=g)
    y = stack(h)
    (y.float() * dy).sum().backward()

    # order: forward group by group, slot by slot; backward in reverse, sublayer backward between
    fwd = [e for e in log if e[1] in ("pre_fwd", "post_fwd")]
    assert fwd == [(l, k, t) for l in range(2) for t in range(2) for k in ("pre_fwd", "post_fwd")]
    # the state gradient passes from group 1's backward to group 0's without a copy
    ptrs = {e[0]: e[2] for e in log if e[1] == "dX_ptr"}
    assert ptrs[0] == ptrs[1]
    bwd = [e for e in log if e[1] in ("post_bwd", "pre_bwd", "sublayer_bwd")]
    want = []
    for l in (1, 0):
        for t in (1, 0):
            want += [(l, "post_bwd", t), ((l, t), "sublayer_bwd", 0), (l, "pre_bwd", t)]
    assert bwd == want, bwd

    # gradients against the same arithmetic written with plain autograd (fp32, bf16 storage
    # treated as the identity, as the stand-in's backward does)
    h2 = h.detach().float().requires_grad_(True)
    a = [[torch.tensor(0.25 * (1 + l + t), requires_grad=True) for t in range(2)] for l in range(2)]
    s = [[torch.tensor(0.5 if t == 0 else 2.0, requires_grad=True) for t in range(2)] for l in range(2)]
    X = h2[:, None, :].expand(T, cfg.N, cfg.C)
    for l in range(2):
        for t in range(2):
            out = X.mean(1) * s[l][t]
            X = X + a[l][t] * out[:, None, :]
    (X.sum(1) * dy).sum().backward()
    assert torch.allclose(h.grad.float(), h2.grad, rtol=2e-2, atol=2e-2)
    for l, grp in enumerate(stack.groups):
        for t in range(2):
            assert torch.allclose(grp.sublayers[t].s.grad, s[l][t].grad, rtol=2e-2), (l, t)
            assert torch.allclose(getattr(grp, f"W_post_{t}").grad[0, 0], a[l][t].grad, rtol=2e-2), (l, t)


def test_state_gradient_seen_by_a_hook_is_not_overwritten():
    """A hook that keeps the state gradient it is given (no copy), and retain_grad on the state,
    see the gradient as it arrived: the in-place update of the groups' backward works on a copy
    whenever the state is watched."""
    cfg = Config.flash(4, 2, 1, 8, 2, seq_len=3)
    log = []
    stack = M.XhcStack(cfg, 2, lambda l, t: Scale(0.5 if t == 0 else 2.0, log, (l, t)))
    for l, grp in enumerate(stack.groups):
        grp.g = FakeGroup(cfg, log, l)
    T = 6
    g = torch.Generator().manual_seed(1)
    h = torch.randn(T, cfg.C, generator=g).to(torch.bfloat16).requires_grad_(True)
    dy = torch.randn(T, cfg.C, generator=g)
    X = M.StreamExpand.apply(h, stack.groups[0].g)
    for grp in stack.groups:
        X = grp(X)
    kept = []
    X.register_hook(lambda gr: kept.append(gr))
    X.retain_grad()
    y = M.StreamSum.apply(X, stack.groups[0].g)
    (y.float() * dy).sum().backward()
    # the gradient of the final state is the stream sum's backward: dy on every stream
    want = dy.to(torch.bfloat16)[:, None, :].expand(T, cfg.N, cfg.C)
    assert torch.equal(kept[0], want)
    assert torch.equal(X.grad, want)


class FakeGroupSaved(FakeGroup):
    """As FakeGroup, but the backward takes the sublayer output from `saved` (what the forward
    left there), as the library's backward takes its forward state."""

    def post_fwd(self, t, P, X, out, saved, ws):
        saved[("out", t)] = out.clone()
        super().post_fwd(t, P, X, out, saved, ws)

    def post_bwd(self, t, P, X, dX, out, d_out, gg, saved, ws):
        super().post_bwd(t, P, X, dX, saved[("out", t)], d_out, gg, saved, ws)


def _stack_with(cfg, fake, log):
    stack = M.XhcStack(cfg, 2, lambda l, t: Scale(0.5 if t == 0 else 2.0, log, (l, t)))
    for l, grp in enumerate(stack.groups):
        grp.g = fake(cfg, log, l)
        with torch.no_grad():
            for t in range(cfg.G):
                getattr(grp, f"W_post_{t}")[0, 0] = 0.25 * (1 + l + t)
    return stack


def test_two_forwards_before_one_backward():
    """Two micro-batches through the same stack before one backward: each forward has its own
    `saved`, so the gradients equal the sum of the two micro-batches run one at a time."""
    cfg = Config.flash(4, 2, 1, 8, 2, seq_len=3)
    T = 6
    g = torch.Generator().manual_seed(2)
    hs = [torch.randn(T, cfg.C, generator=g).to(torch.bfloat16) for _ in range(2)]
    dys = [torch.randn(T, cfg.C, generator=g) for _ in range(2)]

    both = _stack_with(cfg, FakeGroupSaved, [])
    xs = [h.clone().requires_grad_(True) for h in hs]
    ys = [both(x) for x in xs]
    sum((y.float() * dy).sum() for y, dy in zip(ys, dys)).backward()

    one = _stack_with(cfg, FakeGroupSaved, [])
    for i in range(2):
        x = hs[i].clone().requires_grad_(True)
        (one(x).float() * dys[i]).sum().backward()
        assert torch.allclose(x.grad.float(), xs[i].grad.float())
    for (n1, p1), (n2, p2) in zip(both.named_parameters(), one.named_parameters()):
        assert n1 == n2
        if p1.grad is None:
            assert p2.grad is None, n1
        else:
            assert torch.allclose(p1.grad, p2.grad, rtol=1e-5, atol=1e-6), n1


def test_forward_without_grad_records_nothing():
    """With grad mode off the stack runs the same calls without autograd: the output equals the
    grad-mode forward's, and no sublayer graph is recorded."""
    cfg = Config.flash(4, 2, 1, 8, 2, seq_len=3)
    T = 6
    g = torch.Generator().manual_seed(3)
    h = torch.randn(T, cfg.C, generator=g).to(torch.bfloat16)
    log1, log2 = [], []
    s1 = _stack_with(cfg, FakeGroupSaved, log1)
    s2 = _stack_with(cfg, FakeGroupSaved, log2)
    y1 = s1(h.clone().requires_grad_(True))
    with torch.no_grad():
        y2 = s2(h.clone())
    assert torch.equal(y1.detach(), y2)
    assert y2.grad_fn is None and not y2.requires_grad
    calls = [e for e in log2 if e[1] in ("pre_fwd", "post_fwd", "sublayer")]
    assert calls == [e for e in log1 if e[1] in ("pre_fwd", "post_fwd", "sublayer")]
