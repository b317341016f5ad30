"""Prefill and decode against the fp64 oracle on score patterns that stress
the online softmax (GPU).

The random workloads of the other tests keep every score within a few units
of the first key tile's maximum, so a kernel's running-max update (the O and l
rescale when a later key tile holds a larger score) is rarely or never taken.
Here keys carry a position-dependent offset along a fixed direction, so that
q . k / sqrt(d) is close to a chosen function of the key position:

  ascending   slope * position: the maximum grows in every key tile, by
              slope * 128 nats per 128-key tile (0.02: never by more than
              2^15 in the running sum; 0.05: just below it; 0.15: above it
              in every tile; 1.0: far above, exp overflows before the
              rescale);
  descending  the first key tile holds the maximum, later tiles underflow;
  spikes      random scores plus a few keys 60 nats above the rest, placed
              in late tiles.

Softmax is the definition (Sec. 2, scaled dot-product attention); the oracle
subtracts the exact maximum in fp64.  Tolerances are those of the other
parity tests: max abs 1e-2, mean abs 1e-3, LSE within 1e-3.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2605_11232_gb300 import batch as B
from paper_2605_11232_gb300 import pkv
from paper_2605_11232_gb300.workloads import make_workload

from _lib import need_gpu

pytestmark = pytest.mark.gpu

MAX_ABS, MEAN_ABS, LSE_ABS = 1e-2, 1e-3, 1e-3
PREFIX = 512


def _f64(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def _score_offset(kind, slope, pos, rng, spikes):
    """Target score (nats) of the key at each absolute position."""
    pos = np.asarray(pos, np.float64)
    if kind == "ascending":
        return slope * pos
    if kind == "descending":
        return slope * (2048.0 - pos)
    out = np.zeros_like(pos)
    out[np.isin(pos, spikes)] = 60.0
    return out


def _shape(w, kind, slope, seed):
    """Overwrite q, K and V of a workload with the chosen score pattern."""
    g = torch.Generator().manual_seed(seed)
    rng = np.random.default_rng(seed)
    d, Hkv = w.head_dim, w.num_kv_heads
    spikes = np.array([600, 601, 777, 930, 1130])

    def keys(positions):
        n = len(positions)
        a = _score_offset(kind, slope, positions, rng, spikes) / math.sqrt(d)
        k = torch.from_numpy(a).float()[:, None, None] * torch.ones(n, Hkv, d)
        k += 0.25 * torch.randn((n, Hkv, d), generator=g)
        v = 0.5 * torch.randn((n, Hkv, d), generator=g)
        return k.to(torch.bfloat16), v.to(torch.bfloat16)

    for i, p in enumerate(w.prefix_lens):
        w.prefix_k[i], w.prefix_v[i] = keys(np.arange(p))
    for r in range(w.num_requests):
        P = w.prefix_len_of(r)
        a, b = int(w.priv_off[r]), int(w.priv_off[r + 1])
        w.priv_k[a:b], w.priv_v[a:b] = keys(np.arange(P, P + b - a))
        c = int(w.cached_lens[r])
        a, b = int(w.cu_new[r]), int(w.cu_new[r + 1])
        w.new_k[a:b], w.new_v[a:b] = keys(np.arange(c, c + b - a))
    q = 1.0 + 0.25 * torch.randn(tuple(w.q.shape), generator=g)
    w.q = q.to(torch.bfloat16)
    return w


def _check(errs, lerrs):
    e = np.concatenate([x.ravel() for x in errs])
    assert np.isfinite(e).all()
    assert e.max() <= MAX_ABS and e.mean() <= MEAN_ABS, (e.max(), e.mean())
    le = np.concatenate([x.ravel() for x in lerrs])
    assert np.isfinite(le).all() and le.max() <= LSE_ABS, le.max()


PATTERNS = [("ascending", 0.02), ("ascending", 0.05), ("ascending", 0.15),
            ("ascending", 1.0), ("descending", 0.15), ("spikes", 0.0)]


@pytest.mark.parametrize("kind,slope", PATTERNS)
def test_prefill_score_patterns(kind, slope):
    """Suffix prefill over a shared 512-token prefix (whole tiles), private
    cached tokens and a ragged causal part; d = 128, g = 8."""
    need_gpu()
    w = make_workload("custom", custom=dict(
        Hq=16, Hkv=2, d=128, prefix_lens=[PREFIX], group=[0, 0, -1],
        cached=[PREFIX + 37, PREFIX, 300], new=[700, 129, 70], decode=[False] * 3))
    w = _shape(w, kind, slope, seed=11)
    b = B.build_batch(w, poison=True)
    B.run_write(b)
    n = w.num_new_tokens
    out = torch.full((n, w.num_q_heads, w.head_dim), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full((n, w.num_q_heads), float("nan"), dtype=torch.float32, device="cuda")
    B.run_prefill(b, out, lse)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    errs, lerrs = [], []
    for r in range(w.num_requests):
        ref_o, ref_l = oracle.request_attention(w, r, threads=16)
        a, e = int(w.cu_new[r]), int(w.cu_new[r + 1])
        errs.append(np.abs(_f64(out[a:e]) - ref_o))
        lerrs.append(np.abs(_f64(lse[a:e]) - ref_l))
    _check(errs, lerrs)
    b.close()


@pytest.mark.parametrize("groups", [False, True])
@pytest.mark.parametrize("kind,slope", PATTERNS)
def test_decode_score_patterns(kind, slope, groups):
    """Decode queries over a shared 512-token prefix plus private tokens;
    groups=True runs the grouped prefix pass, the split pass and the
    combine."""
    need_gpu()
    w = make_workload("custom", custom=dict(
        Hq=16, Hkv=2, d=128, prefix_lens=[PREFIX], group=[0, 0, 0, -1],
        cached=[PREFIX + 700, PREFIX + 3, PREFIX + 250, 1200], new=[1] * 4,
        decode=[True] * 4))
    w = _shape(w, kind, slope, seed=12)
    b = B.build_batch(w, poison=True)
    B.run_write(b)
    R = w.num_requests
    out = torch.full((R, w.num_q_heads, w.head_dim), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full((R, w.num_q_heads), float("nan"), dtype=torch.float32, device="cuda")
    ws = B.decode_workspace(b, groups)
    B.run_decode(b, out, lse, ws, groups)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    errs, lerrs = [], []
    for r in range(R):
        ref_o, ref_l = oracle.request_attention(w, r, threads=16)
        errs.append(np.abs(_f64(out[r]) - ref_o[0]))
        lerrs.append(np.abs(_f64(lse[r]) - ref_l[0]))
    _check(errs, lerrs)
    b.close()
