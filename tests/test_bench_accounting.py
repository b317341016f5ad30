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
