"""Seeded synthetic inputs shared by the tests, the benchmark and the smoke check.

Holds no arithmetic of the connection op: only random draws with the shapes and value
distributions of the workloads (state and sublayer outputs ~ N(0, 1) rounded to bf16,
projection weights and biases ~ N(0, 0.02) in fp32, gating scalars alpha = 0.01 as initialised
in App. A, causal-conv taps ~ N(0, 1/kappa) so that every conv branch is O(1)).
"""
from __future__ import annotations

import torch


def _gen(seed: int) -> torch.Generator:
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    return g


def normal_bf16(shape, seed: int, std: float = 1.0) -> torch.Tensor:
    """~N(0, std^2) drawn in fp32 on the CPU, rounded to bf16."""
    return (torch.randn(*shape, generator=_gen(seed), dtype=torch.float32) * std).to(torch.bfloat16)


def normal_bf16_on(shape, seed: int, device, std: float = 1.0) -> torch.Tensor:
    """~N(0, std^2) drawn in fp32 by a seeded generator on `device` (large inputs), as bf16."""
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    out = torch.empty(*shape, dtype=torch.bfloat16, device=device)
    flat = out.view(-1)
    step = 1 << 26
    for i in range(0, flat.numel(), step):
        n = min(step, flat.numel() - i)
        flat[i:i + n] = (torch.randn(n, generator=g, dtype=torch.float32, device=device) * std).to(torch.bfloat16)
    return out


def params(shapes: dict, seed: int, alpha: float = 0.01, w_std: float = 0.02) -> dict:
    """fp32 CPU parameters for the given ``{name: shape}`` layout.

    Names starting with ``alpha`` get the constant ``alpha``; ``conv_w`` taps ~ N(0, 1/kappa)
    (kappa = first dimension); everything else ~ N(0, w_std^2).  Each tensor has its own
    stream derived from (seed, position in the layout) so that adding a tensor never shifts
    the draws of another."""
    out = {}
    for i, (name, shp) in enumerate(shapes.items()):
        g = _gen(seed * 1000003 + 7919 * (i + 1))
        if name.startswith("alpha"):
            out[name] = torch.full(shp, float(alpha), dtype=torch.float32)
        elif name.startswith("conv_w"):
            kap = shp[0]
            out[name] = torch.randn(*shp, generator=g, dtype=torch.float32) / float(kap) ** 0.5
        else:
            out[name] = torch.randn(*shp, generator=g, dtype=torch.float32) * w_std
    return out


def group_inputs(T: int, N: int, C: int, G: int, seed: int) -> dict:
    """Entry state X [T, N, C] and the G sublayer outputs [T, C] (all bf16, CPU)."""
    return dict(X=normal_bf16((T, N, C), seed),
                outs=[normal_bf16((T, C), seed + 101 + t) for t in range(G)])


def group_grads(T: int, N: int, C: int, G: int, seed: int) -> dict:
    """Upstream gradients: dX_out [T, N, C] and the G d_input [T, C] (bf16, CPU)."""
    return dict(dX=normal_bf16((T, N, C), seed + 7),
                d_inputs=[normal_bf16((T, C), seed + 211 + t) for t in range(G)])
