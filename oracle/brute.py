"""Brute-force per-token forward of the xHC connection op (test infrastructure only).

A second, independent restatement of Alg. 1 / Alg. 2 / App. E.2 in plain Python floats with
explicit loops over tokens, streams and channels: no gather or scatter (every stream is
visited and either updated or copied), TopK by enumerating every (k-m)-subset of the routed
streams (Eq. router_topk), Sinkhorn and Gram-Schmidt written out element by element.  It is
used only on tiny shapes to pin the vectorised oracle.  Imports nothing from the product.
"""
from __future__ import annotations

import itertools
import math


def _sig(z):
    return 1.0 / (1.0 + math.exp(-z))


def _bf16(v):
    import struct
    b = struct.unpack("<I", struct.pack("<f", v))[0]
    # round-to-nearest-even on the upper 16 bits of the float32 pattern
    lsb = (b >> 16) & 1
    b = (b + 0x7FFF + lsb) & 0xFFFF0000
    return struct.unpack("<f", struct.pack("<I", b))[0]


def _round(v, on):
    # float64 -> float32 -> bf16 is the same as float64 -> bf16 except at double-rounding
    # ties, which never occur for the values used here; kept explicit for readability.
    return _bf16(v) if on else v


def forward(cfg, P, X, outs, round_bf16=True):
    """X: nested lists [T][N][C]; outs: [G][T][C]; P: flat dict of nested lists / floats.
    Returns (X_out, inputs, I) with the same nesting."""
    N, k, m, C, G = cfg.N, cfg.k, cfg.m, cfg.C, cfg.G
    T = len(X)
    S = cfg.seq_len if cfg.seq_len > 0 else T
    eps = cfg.eps_norm
    Xo = [[[X[t][i][c] for c in range(C)] for i in range(N)] for t in range(T)]
    inputs = [[[0.0] * C for _ in range(T)] for _ in range(G)]
    I_all = []
    # augmented components need the sublayer outputs of earlier tokens of the same sequence
    for t in range(T):
        x = [X[t][i][c] for i in range(N) for c in range(C)]
        n = N * C
        mu = sum(x) / n
        nu = sum(v * v for v in x) / n
        # router
        if m < k:
            sd = math.sqrt(nu - mu * mu + eps)
            zs = []
            for o in range(N):
                z = 0.0
                for e in range(n):
                    z += (x[e] - mu) / sd * P["W_r"][e][o]
                zs.append(z)
            if getattr(cfg, "router", "sigmoid") == "softmax":
                den = sum(math.exp(z) for z in zs)
                s = [math.exp(z) / den for z in zs]
            else:
                s = [_sig(z) for z in zs]
            best, best_sum = None, None
            for sub in itertools.combinations(range(m, N), k - m):
                tot = sum(s[i] for i in sub)
                if best is None or tot > best_sum:
                    best, best_sum = sub, tot
            routed = sorted(best, key=lambda i: (-s[i], i))
            I = list(range(m)) + routed
            p = [1.0] * m + [s[i] for i in routed]
        else:
            I = list(range(k))
            p = [1.0] * k
        I_all.append(I)
        rms = math.sqrt(nu + eps)
        Hpre = []
        for q in range(G):
            h = []
            for o in range(N):
                z = 0.0
                for e in range(n):
                    z += x[e] / rms * P[f"W_pre.{q}"][e][o]
                h.append(_sig(P["alpha_pre"][q] * z + P["b_pre"][q][o]))
            Hpre.append(h)
        state = [[X[t][i][c] for c in range(C)] for i in range(N)]
        for q in range(G):
            # dense read over every stream of the current state (only the active ones in the
            # sparse-read ablation)
            dense = getattr(cfg, "dense_read", True)
            for c in range(C):
                acc = 0.0
                for i in range(N):
                    if dense or i in I:
                        acc += Hpre[q][i] * state[i][c]
                inputs[q][t][c] = _round(acc, round_bf16)
            act = [state[I[j]] for j in range(k)]
            xa = [act[j][c] for j in range(k) for c in range(C)]
            r = math.sqrt(sum(v * v for v in xa) / (k * C) + eps)
            K = cfg.K(q)
            Hpost = [[0.0] * K for _ in range(k)]
            for j in range(k):
                for rr in range(K):
                    z = 0.0
                    for e in range(k * C):
                        z += xa[e] / r * P[f"W_post.{q}"][e][j * K + rr]
                    Hpost[j][rr] = 2.0 * _sig(P["alpha_post"][q] * z + P[f"b_post.{q}"][j * K + rr])
            # write-back components for this token
            o_t = outs[q][t]
            comps = [list(o_t)]
            if K > 1:
                pos = t % S
                gs = []
                for jj, kap in enumerate(cfg.conv_k):
                    w = P[f"conv_w.{q}.{jj}"]
                    g = [0.0] * C
                    for c in range(C):
                        for i in range(kap):
                            if pos - i >= 0:
                                g[c] += w[i][c] * outs[q][t - i][c]
                    gs.append(g)
                if cfg.gram_schmidt:
                    epsg = cfg.eps_gs if cfg.eps_gs is not None else 1e-6 * C
                    for g in gs:
                        vn = list(g)
                        for vi in comps:
                            num = sum(g[c] * vi[c] for c in range(C))
                            den = sum(vi[c] * vi[c] for c in range(C)) + epsg
                            for c in range(C):
                                vn[c] -= num / den * vi[c]
                        comps.append(vn)
                else:
                    comps.extend(gs)
            if q == G - 1:
                M = [[0.0] * k for _ in range(k)]
                for a in range(k):
                    for b in range(k):
                        z = 0.0
                        for e in range(k * C):
                            z += xa[e] / r * P["W_res"][e][a * k + b]
                        M[a][b] = math.exp(P["alpha_res"][0] * z + P["b_res"][a * k + b])
                for _ in range(cfg.sinkhorn_iters):
                    for a in range(k):
                        rs = sum(M[a])
                        M[a] = [v / rs for v in M[a]]
                    for b in range(k):
                        cs = sum(M[a][b] for a in range(k))
                        for a in range(k):
                            M[a][b] /= cs
                for a in range(k):
                    rs = sum(M[a])
                    if rs > 1.0:
                        M[a] = [v / rs for v in M[a]]
            new_act = []
            for j in range(k):
                row = []
                for c in range(C):
                    if q == G - 1:
                        v = sum(M[j][i] * act[i][c] for i in range(k))
                    else:
                        v = act[j][c]
                    v += p[j] * sum(Hpost[j][rr] * comps[rr][c] for rr in range(K))
                    row.append(_round(v, round_bf16))
                new_act.append(row)
            # visit every stream: active ones take their new row, the rest are copied
            new_state = []
            for i in range(N):
                if i in I:
                    new_state.append(new_act[I.index(i)])
                else:
                    new_state.append(list(state[i]))
            state = new_state
        Xo[t] = state
    return Xo, inputs, I_all
