"""Per-token memory-traffic models.

``paper_model`` restates the paper's accounting (Table overhead_analysis, Sec. 5.1): per-token
element counts of the residual-stream operations, sublayer function I/O excluded, coefficient
traffic (O(N), O(k^2) elements) excluded, averaged per sublayer.  It is a byte-count check for
the kernels, not their blueprint.  Units: multiples of C elements (bf16: 2 bytes each).
"""
from __future__ import annotations


def paper_model(method: str, N: int, k: int = 4, K_r: int = 4, n_conv: int = 3):
    """(reads, writes) per sublayer in units of C, following Table overhead_analysis.

    method: "mhc", "xhc" (Attention + MLP pair averaged), "flash2" (one block), "flash4"
    (two blocks).  The MLP sublayer adds the separate conv kernel (C read, n_conv*C written) and
    xHC-Flash adds the read-reuse / input correction (2C read, C written) per corrected sublayer.
    """
    if method == "mhc":
        # mapping gen NC | dense read NC, C | mixing NC, NC | write-back C, NC | merge 2NC, NC
        R = N + N + N + 1 + 2 * N
        W = 1 + N + N + N
        return float(R), float(W)
    if method == "xhc":
        def one(Kr, conv):
            R = N + N + k + k + k + Kr + 2 * k + (1 if conv else 0)
            W = 1 + k + k + k + k + (n_conv if conv else 0)
            return R, W
        ra, wa = one(1, False)
        rm, wm = one(K_r, True)
        return (ra + rm) / 2.0, (wa + wm) / 2.0
    if method == "flash2":
        # once per block: mapping gen NC; joint dense read NC (2C written); gather kC/kC;
        # mixing kC/kC.  Per sublayer: active maps kC; write-back K C / kC; merge 2kC / kC.
        R = N + N + k + 2 * k + k + (1 + K_r) + 2 * 2 * k + 1 + 2
        W = 2 + k + k + 2 * k + 2 * k + n_conv + 1
        return R / 2.0, W / 2.0
    if method == "flash4":
        # once per group: mapping gen NC; joint read NC (4 bases written); gather kC/kC;
        # mixing kC/kC.  Per sublayer (x4): active maps kC; write-back K C / kC; merge 2kC / kC.
        # Two MLP convs (C read, n_conv C written each); three input corrections (2C / C each).
        R = N + N + k + 4 * k + k + (1 + K_r + 1 + K_r) + 4 * 2 * k + 2 * 1 + 3 * 2
        W = 4 + k + k + 4 * k + 4 * k + 2 * n_conv + 3
        return R / 4.0, W / 4.0
    raise ValueError(method)


def backward_model(N: int, k: int, G: int) -> float:
    """Elements (units of C) a group's backward must move at least, per token; the paper gives no
    backward count, so this is the build's own model, counted the way the paper counts the
    forward (bf16 state, every stored tensor read or written once, coefficients excluded):
      3N       the entry state X read once, dX read (gradient of the group output) and written
      (G-1)k   the active state entering each slot t >= 1, read back from the forward
      2(G-1)k  the gradient of that state handed from slot t to slot t-1 (bf16 write + read)
      3G       per slot: d_input read, the sublayer output read (write-back components), d_out
               written
    An fp32 active gradient, partial sums or any other intermediate an implementation chooses
    counts as overhead against this model, not as algorithmic traffic."""
    return float(3 * N + (G - 1) * k + 2 * (G - 1) * k + 3 * G)


def forward_model(variant: str, N: int, k: int, G: int) -> float:
    """The paper's forward accounting for one group, units of C per token (Table
    overhead_analysis; per-sublayer averages times the group's sublayers)."""
    if variant == "mhc":
        r, w = paper_model("mhc", N)
        return r + w
    if G == 4:
        r, w = paper_model("flash4", N, k)
    elif G == 2:
        r, w = paper_model("flash2", N, k)
    else:
        r, w = paper_model("xhc", N, k)
    return G * (r + w)
