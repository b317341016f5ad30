"""The segmented multi-adapter LoRA projection on the GPU (pkv_lora_sgmv,
Sec. 5.6) against the fp64 definition of oracle/lora_sgmv.py.

Tolerance, from the arithmetic (bf16 operands, fp32 accumulation): the kernel
rounds U = s_a A_a x to bf16 before its product with B_a, and rounds y to
bf16; each rounding is at most half a bf16 ulp, 2^-8 relative.  So per
element |y - y_ref| <= 2^-8 |y_ref| + 2^-8 sum_j |B_a[o][j]| |U_j| + 1e-4
(the last term covers the fp32 accumulation), and the mean error is at most
half the mean bound (round-to-nearest errors spread over +-half an ulp: a
systematic bias would exceed it).
"""
import numpy as np
import pytest
import torch

from oracle import lora_sgmv as L
from paper_2605_11232_gb300 import pkv

from _lib import built_lib, need_gpu

pytestmark = pytest.mark.gpu


def _bf16(a):
    return torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16)


def _inputs(seed, T, d_in, d_out, rank, n_ad):
    g = torch.Generator().manual_seed(seed)
    x = torch.randn((T, d_in), generator=g).to(torch.bfloat16)
    w = (torch.randn((d_out, d_in), generator=g) / d_in ** 0.5).to(torch.bfloat16)
    a = (torch.randn((n_ad, rank, d_in), generator=g) / d_in ** 0.5).to(torch.bfloat16)
    b = (torch.randn((n_ad, d_out, rank), generator=g) / rank ** 0.5).to(torch.bfloat16)
    scale = np.linspace(0.5, 2.0, n_ad).astype(np.float32)
    return x, w, a, b, scale


def _bound(x, a, b, scale, adapter, ref):
    """Per-element error bound of rows x (fp64) under one adapter."""
    bound = 2.0 ** -8 * np.abs(ref) + 1e-4
    if adapter >= 0:
        u = np.abs(float(scale[adapter]) * (x @ a[adapter].T))          # |U_j| [rows][r]
        bound = bound + 2.0 ** -8 * (u @ np.abs(b[adapter]).T)
    return bound


def _check(got, ref, bound):
    got = got.float().cpu().numpy().astype(np.float64)
    err = np.abs(got - ref)
    assert np.isfinite(got).all()
    assert (err <= bound).all(), float((err - bound).max())
    assert err.mean() <= 0.5 * bound.mean(), (err.mean(), bound.mean())


def _run(x, w, a, b, scale, starts, adapters):
    need_gpu()
    dev = [t.cuda() for t in (x, w, a, b)]
    y = torch.full((x.shape[0], w.shape[0]), float("nan"), dtype=torch.bfloat16, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    pkv.pkv_lora_sgmv(*dev, scale, starts, adapters, y, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    return y


@pytest.mark.parametrize("rank", [16, 32, 48, 64])
def test_segments_match_oracle(rank):
    """Five segments (adapters 2, base, 0, 1, 2) of ragged lengths, some
    shorter than a 128-row tile and one spanning three: every output."""
    x, w, a, b, scale = _inputs(rank, 300, 256, 512, rank, 3)
    starts, adapters = [0, 37, 100, 101, 229, 300], [2, -1, 0, 1, 2]
    y = _run(x, w, a, b, scale, starts, adapters)
    f = lambda t: t.float().numpy().astype(np.float64)
    ref = L.lora_segments(f(x), f(w), f(a), f(b), scale, starts, adapters)
    bound = np.concatenate([_bound(f(x[s0:e0]), f(a), f(b), scale, ad, ref[s0:e0])
                            for s0, e0, ad in zip(starts, starts[1:], adapters)])
    _check(y, ref, bound)


def test_case_c1_shapes_sampled():
    """Llama-3-8B projection shape (4096 x 4096), four adapters of rank 16,
    the 12-prompt 4/3/3/2 request of Case C1 as pkv_lora_dispatch batches it:
    rows of every segment against the oracle."""
    built_lib()
    lens = [412, 1830, 2650, 977, 1210, 2205, 388, 1499, 2800, 640, 1750, 2120]
    ad = [0, 0, 0, 0, 1, 1, 1, 2, 2, 2, 3, 3]
    order, batches = pkv.pkv_lora_dispatch(np.array(ad, np.int32), np.array(lens, np.int32),
                                           np.array([1024, 2048], np.int32), 0)
    T = sum(lens)
    starts, badapter = [0], []
    for adapter, _bucket, b0, b1 in batches:   # the rows of a batch: its prompts' tokens
        starts.append(starts[-1] + sum(lens[order[i]] for i in range(b0, b1)))
        badapter.append(adapter)
    assert starts[-1] == T
    x, w, a, b, scale = _inputs(7, T, 4096, 4096, 16, 4)
    y = _run(x, w, a, b, scale, starts, list(badapter))
    rng = np.random.default_rng(0)
    f = lambda t: t.float().numpy().astype(np.float64)
    for k in range(len(badapter)):
        s0, e0 = starts[k], starts[k + 1]
        rows = sorted({s0, e0 - 1, *rng.integers(s0, e0, 6).tolist()})
        ref = L.lora_segments(f(x[rows]), f(w), f(a), f(b), scale, [0, len(rows)], [int(badapter[k])])
        _check(y[rows], ref, _bound(f(x[rows]), f(a), f(b), scale, int(badapter[k]), ref))


def test_argument_checks():
    built_lib()
    need_gpu()
    x, w, a, b, scale = _inputs(1, 16, 64, 256, 16, 2)
    dev = [t.cuda() for t in (x, w, a, b)]
    y = torch.empty((16, 256), dtype=torch.bfloat16, device="cuda")
    for starts, adapters, code in (([0, 16], [2], pkv.PKV_ERR_INVALID_ARG),     # no adapter 2
                                   ([0, 8], [0], pkv.PKV_ERR_INVALID_ARG),      # rows not covered
                                   ([0, 9, 8, 16], [0, 0, 0], pkv.PKV_ERR_INVALID_ARG)):
        with pytest.raises(pkv.PkvError) as e:
            pkv.pkv_lora_sgmv(*dev, scale, starts, adapters, y)
        assert e.value.code == code
    a8 = torch.zeros((2, 8, 64), dtype=torch.bfloat16, device="cuda")
    b8 = torch.zeros((2, 256, 8), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(pkv.PkvError) as e:
        pkv.pkv_lora_sgmv(dev[0], dev[1], a8, b8, scale, [0, 16], [0], y)
    assert e.value.code == pkv.PKV_ERR_UNSUPPORTED
