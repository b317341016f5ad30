"""Failure detection on the GPU without a fault.

A bounded device wait is made to run out (pkv_selftest_wait_timeout: one
thread waits, with the kernels' bounded mbarrier wait, on a phase that nothing
completes).  The kernel latches DEVICE_TIMEOUT and returns; the host reads it
through pkv_check_device_errors (which clears it); a decode on the same pool
afterwards is still correct, so the context stayed usable.
"""
import time

import numpy as np
import pytest
import torch

import oracle
from paper_2605_11232_gb300 import batch as B
from paper_2605_11232_gb300 import pkv
from paper_2605_11232_gb300.workloads import make_workload

from _lib import need_gpu

pytestmark = pytest.mark.gpu


def test_bounded_wait_runs_out_and_the_context_stays_usable():
    need_gpu()
    w = make_workload("tiny_decode")
    b = B.build_batch(w, poison=True)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    t0 = time.perf_counter()
    pkv.pkv_selftest_wait_timeout(b.pool, 2000)            # 2 ms
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_ERR_DEVICE_TIMEOUT
    assert time.perf_counter() - t0 < 5.0
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK   # read and cleared
    # the same pool and context still decode correctly
    B.run_write(b)
    Rd = b.dec.stop - b.dec.start
    out = torch.empty((Rd, w.num_q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
    ws = B.decode_workspace(b, False)
    B.run_decode(b, out, None, ws, False)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    for i, r in enumerate(range(b.dec.start, b.dec.stop)):
        o_ref, _ = oracle.request_attention(w, r, threads=4)
        e = np.abs(out[i].float().cpu().numpy().astype(np.float64) - o_ref[0])
        assert e.max() <= 1e-2 and e.mean() <= 1e-3
    b.close()


def test_selftest_rejects_bad_limits():
    need_gpu()
    w = make_workload("tiny_decode", values=False)
    kc = torch.zeros((8, w.num_kv_heads, 16, w.head_dim), dtype=torch.bfloat16, device="cuda")
    pool = pkv.kv_pool_create(8, w.num_kv_heads, w.head_dim, kc, kc.clone())
    with pytest.raises(pkv.PkvError) as e:
        pkv.pkv_selftest_wait_timeout(pool, -1)
    assert e.value.code == pkv.PKV_ERR_INVALID_ARG
    pkv.kv_pool_destroy(pool)
