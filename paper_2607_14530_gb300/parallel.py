"""Multi-rank host logic of the connection op: sequence split and data parallelism.

The op is token-parallel except for the causal conv of the temporal augmentation (conv formula of
Sec. 3.3.4), which reads the R = max(kappa) - 1 sublayer outputs preceding each token.  When the
sequences of a batch are cut into consecutive chunks held by consecutive ranks (context
parallelism), rank r needs, per conv slot, the last R outputs of every sequence's chunk on rank
r - 1 (the halo), and returns to rank r - 1 the gradient w.r.t. those rows, which belongs to that
rank's d_out.  Parameter gradients are sums over tokens, so the ranks' gradients add up: one
all-reduce, whether the ranks split sequences, split the batch (data parallelism), or both.

These functions only move tensors between ranks (torch.distributed point-to-point and
all-reduce; gloo on CPU tensors, NCCL on CUDA tensors); the halos themselves come from
``Group.halo_fill`` and are consumed by ``Group.post_fwd(..., halo=)`` /
``Group.post_bwd(..., halo=, d_halo=)`` and ``Group.halo_add`` (include/xhc.h, "Sequence split").
``SequenceChunk`` strings them together for one group on one rank.
"""
from __future__ import annotations

import torch
import torch.distributed as dist


def _rank_world(group):
    return dist.get_rank(group), dist.get_world_size(group)


def _peer(group, r):
    """Global rank of the group's r-th member."""
    return r if group is None else dist.get_global_rank(group, r)


def halo_exchange(halo_send: torch.Tensor, group=None) -> torch.Tensor:
    """Send this rank's halo (the last R outputs of its chunk of every sequence) to the next rank
    and receive the previous rank's.  The first rank receives zeros (its chunks start the
    sequences).  Returns the received halo, shaped like ``halo_send``."""
    rank, world = _rank_world(group)
    recv = torch.zeros_like(halo_send)
    ops = []
    if rank + 1 < world:
        ops.append(dist.P2POp(dist.isend, halo_send.contiguous(), _peer(group, rank + 1), group))
    if rank > 0:
        ops.append(dist.P2POp(dist.irecv, recv, _peer(group, rank - 1), group))
    if ops:
        for w in dist.batch_isend_irecv(ops):
            w.wait()
    return recv


def halo_grad_return(d_halo: torch.Tensor, group=None) -> torch.Tensor:
    """Send the gradient of this rank's received halo back to the previous rank and receive the
    next rank's.  The last rank receives zeros.  Returns the received gradient (to be added to
    the d_out of this rank's last R tokens per sequence)."""
    rank, world = _rank_world(group)
    recv = torch.zeros_like(d_halo)
    ops = []
    if rank > 0:
        ops.append(dist.P2POp(dist.isend, d_halo.contiguous(), _peer(group, rank - 1), group))
    if rank + 1 < world:
        ops.append(dist.P2POp(dist.irecv, recv, _peer(group, rank + 1), group))
    if ops:
        for w in dist.batch_isend_irecv(ops):
            w.wait()
    return recv


def allreduce_grads(grads: dict, group=None) -> dict:
    """Sum every parameter gradient over the ranks, in place (the gradients are sums over
    tokens; each rank holds the sum over its own tokens).  One flat buffer per dtype, so a group's
    gradients take one collective."""
    by_dtype = {}
    for n in sorted(grads):
        by_dtype.setdefault(grads[n].dtype, []).append(n)
    for names in by_dtype.values():
        flat = torch.cat([grads[n].reshape(-1) for n in names])
        dist.all_reduce(flat, op=dist.ReduceOp.SUM, group=group)
        off = 0
        for n in names:
            k = grads[n].numel()
            grads[n].copy_(flat[off:off + k].view_as(grads[n]))
            off += k
    return grads


class SequenceChunk:
    """One connection-op group on a rank that holds one chunk of each of B sequences (S tokens
    per chunk; the chunks of a sequence sit on consecutive ranks of ``group``).

    Per slot t the caller runs, as with a plain Group: ``pre_fwd(t)``, its sublayer, then
    ``post_fwd(t)``, which exchanges the slot's halo with the neighbouring ranks first; in the
    backward ``post_bwd(t)``, which returns the halo's gradient to the previous rank and adds the
    next rank's to this rank's d_out, then the sublayer's backward and ``pre_bwd(t)``.
    Parameter gradients are all-reduced by ``finish_backward`` (or by the caller's data-parallel
    framework)."""

    def __init__(self, g, B: int, S: int, group=None):
        self.g, self.B, self.S, self.group = g, B, S, group
        self.halos = {}

    def _conv(self, t):
        return self.g.cfg.K(t) > 1

    def pre_fwd(self, t, P, X, inp, saved, ws, stream=None):
        self.g.pre_fwd(t, P, X, inp, saved, ws, stream)

    def post_fwd(self, t, P, X, out, saved, ws, stream=None):
        halo = None
        if self._conv(t):
            halo = halo_exchange(self.g.halo_fill(self.B, self.S, out, stream=stream), self.group)
            self.halos[t] = halo
        self.g.post_fwd(t, P, X, out, saved, ws, stream, halo=halo)

    def post_bwd(self, t, P, X, dX, out, d_out, grads, saved, ws, stream=None):
        if not self._conv(t):
            self.g.post_bwd(t, P, X, dX, out, d_out, grads, saved, ws, stream)
            return
        halo = self.halos[t]
        d_halo = torch.empty(halo.shape, dtype=torch.float32, device=halo.device)
        self.g.post_bwd(t, P, X, dX, out, d_out, grads, saved, ws, stream, halo=halo, d_halo=d_halo)
        back = halo_grad_return(d_halo, self.group)
        self.g.halo_add(self.B, self.S, d_out, back, stream)

    def pre_bwd(self, t, P, X, d_input, dX, grads, saved, ws, stream=None):
        self.g.pre_bwd(t, P, X, d_input, dX, grads, saved, ws, stream)

    def finish_backward(self, grads: dict):
        return allreduce_grads(grads, self.group)
