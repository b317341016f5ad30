"""Segmented multi-adapter LoRA projection (Sec. 5.6: one base model serves
several LoRA adapters, and a mixed request runs as per-adapter batches) --
test infrastructure only: the tests call it; the library never does.

For token t of a batch with input row x_t (d_in values) and adapter a_t:

    y_t = W x_t + s_a * B_a (A_a x_t)          (a_t >= 0)
    y_t = W x_t                                (a_t = -1: base model only)

W is the base projection [d_out][d_in]; A_a [r][d_in] and B_a [d_out][r] are
adapter a's low-rank factors and s_a its scale (alpha / r in the usual
convention).  The paper names LoRA adapters but prints no formula; this is
the standard low-rank update.  Tokens come in segments (the batches of the
dispatch, each with one adapter), given as CSR offsets seg_start[S + 1] and
seg_adapter[S].

Computed in fp64 from the bf16 inputs, one segment at a time, with plain
matrix products in the order written above.

Parity pinned: the tests check B = 0 (base only), a rank-1 closed form,
segment invariance (any cut of a segment gives the same rows) and equality
with the merged weights W + s_a B_a A_a (the merge-and-save strategy of the
Case C1 table), which takes the products in a different order.
"""

import numpy as np


def lora_segments(x, w, a, b, scale, seg_start, seg_adapter):
    """y [T][d_out] for x [T][d_in], w [d_out][d_in], a [n][r][d_in],
    b [n][d_out][r], scale [n], segments (seg_start [S+1], seg_adapter [S])."""
    x = np.asarray(x, np.float64)
    w = np.asarray(w, np.float64)
    T = x.shape[0]
    seg_start = [int(v) for v in seg_start]
    if seg_start[0] != 0 or seg_start[-1] != T or any(e < s for s, e in zip(seg_start, seg_start[1:])):
        raise ValueError("segments must cover the rows in order")
    y = np.zeros((T, w.shape[0]), np.float64)
    for k, ad in enumerate(seg_adapter):
        s, e = seg_start[k], seg_start[k + 1]
        xs = x[s:e]
        ys = xs @ w.T                                          # W x_t
        if ad >= 0:
            shrink = xs @ np.asarray(a[ad], np.float64).T      # A_a x_t   [rows][r]
            ys = ys + float(scale[ad]) * (shrink @ np.asarray(b[ad], np.float64).T)
        y[s:e] = ys
    return y


def merged_weights(w, a, b, scale, ad):
    """W + s_a B_a A_a (the adapter merged into the base weights)."""
    w = np.asarray(w, np.float64)
    return w + float(scale[ad]) * (np.asarray(b[ad], np.float64) @ np.asarray(a[ad], np.float64))
