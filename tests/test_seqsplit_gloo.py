"""Sequence split and data parallelism across ranks: the host exchange logic on CPU (gloo,
world size 2).

Each rank holds one chunk of every sequence (rank 0 the first S1 tokens, rank 1 the next S2).
The exchange functions of paper_2607_14530_gb300.parallel move the halo (the last R = max(kappa)
- 1 sublayer outputs of rank 0's chunks) forward and its gradient back, and sum the parameter
gradients; the per-rank compute is the fp64 oracle with halos (the CUDA path runs only on a GPU;
its halo entry points are checked in tests/test_gpu_seqsplit.py).  Together they must reproduce
the unsplit single-rank forward and backward.  A second test splits the batch instead (data
parallelism): the all-reduced gradients equal the single-rank ones."""
import os
import socket
import sys

import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
F64 = torch.float64


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _case():
    sys.path.insert(0, ROOT)
    from oracle import xhc_oracle as O
    from paper_2607_14530_gb300 import synth
    cfg = O.flash(6, 3, 1, 8, 4, conv_k=(2, 3, 5))
    B, S1, S2 = 3, 6, 5
    S = S1 + S2
    T = B * S
    P = {n: v.to(F64) for n, v in synth.params(O.param_shapes(cfg), 5, alpha=0.3, w_std=0.2).items()}
    d = synth.group_inputs(T, cfg.N, cfg.C, cfg.G, 5)
    X, outs = d["X"].to(F64), [o.to(F64) for o in d["outs"]]
    gr = synth.group_grads(T, cfg.N, cfg.C, cfg.G, 5)
    dX, dins = gr["dX"].to(F64), [x.to(F64) for x in gr["d_inputs"]]
    return O, cfg, B, S1, S2, P, X, outs, dX, dins


def _rows(B, S, lo, hi):
    return torch.cat([torch.arange(b * S + lo, b * S + hi) for b in range(B)])


def _seq_rank(rank, world, port, out_dir):
    sys.path.insert(0, ROOT)
    from paper_2607_14530_gb300 import parallel
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        O, cfg, B, S1, S2, P, X, outs, dXo, dins = _case()
        S = S1 + S2
        R = max(cfg.conv_k) - 1
        lo, hi = (0, S1) if rank == 0 else (S1, S)
        Sc = hi - lo
        r = _rows(B, S, lo, hi)
        ccfg = O.Config(**{**cfg.__dict__, "seq_len": Sc})
        my_outs = [o[r] for o in outs]
        # forward: per conv slot, this chunk's last R outputs go to the next rank
        halos = []
        for t in range(cfg.G):
            send = my_outs[t].reshape(B, Sc, cfg.C)[:, Sc - R:].contiguous()
            halos.append(parallel.halo_exchange(send))
        Xo, ins, _ = O.forward(ccfg, P, X[r], my_outs, round_bf16=False, halos=halos)
        dX, d_outs, dP, dh = O.backward(ccfg, P, X[r], my_outs, dXo[r], [d[r] for d in dins],
                                        round_bf16=False, halos=halos)
        # backward: the halo's gradient goes back and lands in the previous chunk's d_out
        for t in range(cfg.G):
            back = parallel.halo_grad_return(dh[t])
            v = d_outs[t].reshape(B, Sc, cfg.C)
            v[:, Sc - R:] += back
        parallel.allreduce_grads(dP)
        torch.save(dict(rows=r, Xo=Xo, ins=ins, dX=dX, d_outs=d_outs, dP=dP),
                   os.path.join(out_dir, f"seq{rank}.pt"))
    finally:
        dist.destroy_process_group()


def test_sequence_split_across_two_ranks_equals_one_rank(tmp_path):
    world = 2
    mp.start_processes(_seq_rank, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True,
                       start_method="spawn")
    O, cfg, B, S1, S2, P, X, outs, dXo, dins = _case()
    full = O.Config(**{**cfg.__dict__, "seq_len": S1 + S2})
    Xo, ins, _ = O.forward(full, P, X, outs, round_bf16=False)
    dX, d_outs, dP = O.backward(full, P, X, outs, dXo, dins, round_bf16=False)
    for rank in range(world):
        res = torch.load(os.path.join(tmp_path, f"seq{rank}.pt"))
        r = res["rows"]
        assert torch.allclose(res["Xo"], Xo[r], atol=1e-12, rtol=0)
        assert torch.allclose(res["dX"], dX[r], atol=1e-12, rtol=0)
        for t in range(cfg.G):
            assert torch.allclose(res["ins"][t], ins[t][r], atol=1e-12, rtol=0)
            assert torch.allclose(res["d_outs"][t], d_outs[t][r], atol=1e-12, rtol=0), (rank, t)
        for n in dP:
            assert torch.allclose(res["dP"][n], dP[n], atol=1e-11, rtol=1e-12), (rank, n)


def _dp_rank(rank, world, port, out_dir):
    sys.path.insert(0, ROOT)
    from paper_2607_14530_gb300 import parallel
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        O, cfg, B, S1, S2, P, X, outs, dXo, dins = _case()
        S = S1 + S2
        # rank r takes whole sequences r, r + world, ...: no halo
        r = torch.cat([torch.arange(b * S, (b + 1) * S) for b in range(rank, B, world)])
        ccfg = O.Config(**{**cfg.__dict__, "seq_len": S})
        _, _, dP = O.backward(ccfg, P, X[r], [o[r] for o in outs], dXo[r], [d[r] for d in dins],
                              round_bf16=False)
        parallel.allreduce_grads(dP)
        torch.save(dP, os.path.join(out_dir, f"dp{rank}.pt"))
    finally:
        dist.destroy_process_group()


def test_data_parallel_gradient_allreduce_equals_one_rank(tmp_path):
    world = 2
    mp.start_processes(_dp_rank, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True,
                       start_method="spawn")
    O, cfg, B, S1, S2, P, X, outs, dXo, dins = _case()
    full = O.Config(**{**cfg.__dict__, "seq_len": S1 + S2})
    _, _, dP = O.backward(full, P, X, outs, dXo, dins, round_bf16=False)
    for rank in range(world):
        res = torch.load(os.path.join(tmp_path, f"dp{rank}.pt"))
        for n in dP:
            assert torch.allclose(res[n], dP[n], atol=1e-11, rtol=1e-12), (rank, n)


def _mixed_rank(rank, world, port, out_dir):
    sys.path.insert(0, ROOT)
    from paper_2607_14530_gb300 import parallel
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        g = {"a": torch.full((3,), 1.0 + rank, dtype=torch.float32),
             "b": torch.full((2, 2), 0.5 * (rank + 1), dtype=F64),
             "c": torch.arange(4, dtype=torch.float32) * (rank + 1)}
        parallel.allreduce_grads(g)
        torch.save(g, os.path.join(out_dir, f"mx{rank}.pt"))
    finally:
        dist.destroy_process_group()


def test_gradient_allreduce_keeps_each_dtype(tmp_path):
    """Gradients of different dtypes are summed in one collective per dtype and keep their dtype
    (one concatenated buffer would promote them)."""
    world = 2
    mp.start_processes(_mixed_rank, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True,
                       start_method="spawn")
    for rank in range(world):
        g = torch.load(os.path.join(tmp_path, f"mx{rank}.pt"))
        assert g["a"].dtype == torch.float32 and torch.equal(g["a"], torch.full((3,), 3.0))
        assert g["b"].dtype == F64 and torch.equal(g["b"], torch.full((2, 2), 1.5, dtype=F64))
        assert torch.equal(g["c"], torch.arange(4, dtype=torch.float32) * 3)
