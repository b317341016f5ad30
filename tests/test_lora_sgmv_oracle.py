"""The segmented multi-adapter LoRA projection of oracle/lora_sgmv.py pinned
by closed forms and identities (CPU)."""
import numpy as np
import pytest

from oracle import lora_sgmv as L


def _inputs(seed, T=37, d_in=48, d_out=40, r=8, n=3):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((T, d_in))
    w = rng.standard_normal((d_out, d_in)) / np.sqrt(d_in)
    a = rng.standard_normal((n, r, d_in)) / np.sqrt(d_in)
    b = rng.standard_normal((n, d_out, r)) / np.sqrt(r)
    scale = rng.uniform(0.5, 2.0, n)
    return x, w, a, b, scale


def test_zero_b_gives_the_base_projection():
    x, w, a, b, scale = _inputs(0)
    y = L.lora_segments(x, w, a, np.zeros_like(b), scale, [0, 10, 37], [0, 2])
    assert np.allclose(y, x @ w.T, rtol=0, atol=1e-12)
    # adapter -1 on a segment: base only, whatever the factors hold
    y2 = L.lora_segments(x, w, a, b, scale, [0, 37], [-1])
    assert np.array_equal(y2, x @ w.T)


def test_rank_one_closed_form():
    rng = np.random.default_rng(1)
    T, d_in, d_out = 5, 6, 4
    x = rng.integers(-3, 4, (T, d_in)).astype(float)
    w = rng.integers(-2, 3, (d_out, d_in)).astype(float)
    u = rng.integers(-2, 3, d_in).astype(float)
    v = rng.integers(-2, 3, d_out).astype(float)
    a = u[None, None, :]            # A_0 = u^T (one row)
    b = v[None, :, None]            # B_0 = v (one column)
    y = L.lora_segments(x, w, a, b, [0.5], [0, T], [0])
    for t in range(T):
        want = [sum(w[o, c] * x[t, c] for c in range(d_in)) + 0.5 * v[o] * sum(u[c] * x[t, c] for c in range(d_in))
                for o in range(d_out)]
        assert np.array_equal(y[t], np.array(want))     # small integers: exact in fp64


@pytest.mark.parametrize("seed", range(5))
def test_equals_merged_weights_per_segment(seed):
    x, w, a, b, scale = _inputs(seed)
    starts, adapters = [0, 7, 8, 20, 37], [1, 0, -1, 2]
    y = L.lora_segments(x, w, a, b, scale, starts, adapters)
    for k, ad in enumerate(adapters):
        s, e = starts[k], starts[k + 1]
        wm = w if ad < 0 else L.merged_weights(w, a, b, scale, ad)
        assert np.allclose(y[s:e], x[s:e] @ wm.T, rtol=1e-12, atol=1e-12)


def test_segment_cuts_do_not_change_rows():
    x, w, a, b, scale = _inputs(7)
    y = L.lora_segments(x, w, a, b, scale, [0, 37], [1])
    y_cut = L.lora_segments(x, w, a, b, scale, [0, 1, 2, 19, 19, 37], [1, 1, 1, 1, 1])
    # equal up to the summation order the matrix library picks per shape
    assert np.allclose(y, y_cut, rtol=0, atol=1e-12)
    # an empty request and empty segments
    assert L.lora_segments(x[:0], w, a, b, scale, [0], []).shape == (0, w.shape[0])


def test_rejects_segments_that_do_not_cover_the_rows():
    x, w, a, b, scale = _inputs(3)
    for starts in ([0, 30], [1, 37], [0, 20, 10, 37]):
        with pytest.raises(ValueError):
            L.lora_segments(x, w, a, b, scale, starts, [0] * (len(starts) - 1))
