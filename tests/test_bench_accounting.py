"""bench.py's byte and FLOP accounting (CPU): algorithmic decode bytes count a
shared prefix once, logical bytes once per request; the summary carries both."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2605_11232_gb300.workloads import make_workload  # noqa: E402


def test_shared_prefix_counts_once_algorithmically_and_per_request_logically():
    w = make_workload("l8b_decode", values=False)
    dec = slice(0, w.num_requests)
    row = bench.kv_row_bytes(w)
    qo = 2 * w.num_requests * w.num_q_heads * w.head_dim * 2
    P = w.prefix_lens[0]
    ctx = sum(int(L) for L in w.context_lens)
    assert bench.decode_logical_bytes(w, dec) == ctx * row + qo
    assert bench.decode_bytes(w, dec) == (ctx - (w.num_requests - 1) * P) * row + qo


def test_without_sharing_the_two_counts_agree():
    R = 5
    w = make_workload("custom", values=False, custom=dict(
        Hq=8, Hkv=2, d=64, prefix_lens=[], group=[-1] * R, cached=[10, 20, 30, 40, 50],
        new=[1] * R, decode=[True] * R))
    dec = slice(0, R)
    assert bench.decode_bytes(w, dec) == bench.decode_logical_bytes(w, dec)


def test_summary_reports_algorithmic_and_logical_rates():
    w = make_workload("l8b_decode", values=False)
    dec = slice(0, w.num_requests)
    res = dict(step_ms=[0.05] * 3, warm_ms=[0.05] * 3, trace={"decode_split": (3, 0.12)}, Rd=64, Rp=0,
               dec_bytes=bench.decode_bytes(w, dec), dec_logical=bench.decode_logical_bytes(w, dec),
               wr_bytes=bench.write_bytes(w, 64), groups=True)
    out = bench.summarize(res, (6774.6, 1934.6, 1725.0, "measured"))
    assert out["decode_logical_gbs"] > out["decode_hbm_gbs"] > 0
    assert abs(out["decode_hbm_gbs"] - (res["dec_bytes"] + res["wr_bytes"]) / 0.05e-3 / 1e9) < 1e-6


def test_mixed_step_rates_use_the_decode_subsets_own_time():
    """A step with prefill and decode requests: the decode bytes are set
    against the decode subset timed alone (its kernels overlapping), not the
    whole step nor the sum of traced kernel times; prefill TFLOP/s against
    the traced prefill kernel."""
    w = make_workload("qwen_mixed", values=False)
    trace = {"decode_split": (3, 0.180), "decode_prefix": (3, 0.105), "decode_combine": (3, 0.030),
             "prefill": (3, 0.750)}
    res = dict(step_ms=[0.35] * 3, warm_ms=[0.35] * 3, dec_ms=[0.09, 0.09, 0.09], trace=trace, Rd=256, Rp=8,
               dec_bytes=3.6e8, dec_logical=2.4e9, wr_bytes=1.0e6, pre_flops=2.6e11, groups=True)
    out = bench.summarize(res, (6774.6, 1934.6, 1725.0, "measured"))
    assert abs(out["decode_us_per_step"] - 90.0) < 1e-9
    assert abs(out["decode_hbm_gbs"] - 3.6e8 / 90e-6 / 1e9) < 1e-6
    assert abs(out["decode_kernels_sum_us"] - 1e3 * (0.180 + 0.105 + 0.030) / 3) < 1e-9
    assert abs(out["prefill_tflops"] - 2.6e11 / 0.250e-3 / 1e12) < 1e-9
    assert "alone" in out["decode_basis"]
