"""The Python binding's marshalling checks, on CPU: every argument is validated before the
library is called, and wrong tensors raise XhcError instead of reaching a kernel."""
import pytest
import torch

from paper_2607_14530_gb300 import xhc as X


def test_ring_sizes_follow_the_conv_history():
    g = X.Group(X.Config.flash(16, 4, 2, 256, 4))
    # max(kappa) - 1 = 11 rows of C bf16 per sequence, one ring per conv (MLP) slot
    assert g.ring_bytes(8) == 8 * 11 * 256 * 2
    rings = g.alloc_rings(8, device="cpu")
    assert [r is not None for r in rings] == [False, True, False, True]
    assert all(r.numel() == 8 * 11 * 256 * 2 for r in rings if r is not None)
    ga = X.Group(X.Config.full(8, 4, 2, 64, False))           # attention sublayer: no conv slot
    assert ga.alloc_rings(8, device="cpu") == [None]
    gn = X.Group(X.Config.full(8, 4, 2, 64, True, conv_k=()))  # MLP sublayer without the conv
    assert gn.ring_bytes(8) == 0
    assert gn.alloc_rings(8, device="cpu") == [None]


def test_parameters_must_be_fp32_device_tensors():
    cfg = X.Config.full(8, 4, 2, 64, True)
    g = X.Group(cfg)
    P = {n: torch.zeros(s) for n, s in cfg.param_shapes().items()}   # CPU tensors
    Xs = torch.zeros(4, 8, 64, dtype=torch.bfloat16)
    with pytest.raises(X.XhcError, match="fp32 CUDA tensor"):
        g.forward(P, Xs, [torch.zeros(4, 64, dtype=torch.bfloat16)], None, None)


def test_decode_checks_pos():
    cfg = X.Config.full(8, 4, 2, 64, True)
    g = X.Group(cfg)
    pp = X._Params()
    Xs = torch.zeros(4, 8, 64, dtype=torch.bfloat16)
    out = torch.zeros(4, 64, dtype=torch.bfloat16)
    for pos in (torch.zeros(4, dtype=torch.int32), torch.zeros(4, dtype=torch.int64)):  # wrong type / host
        with pytest.raises(X.XhcError, match="int64 CUDA tensor"):
            g.post_fwd_decode(0, pp, Xs, out, None, pos, None, None)
