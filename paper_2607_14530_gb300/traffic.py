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
