"""paged_attn_decode_noalloc: decode for callers that cannot allocate.

Code recorded into a CUDA graph, inference plugins whose framework owns all
device buffers, and processes with a fixed up-front memory budget cannot call
cudaMalloc when they decode.  This entry point runs the same decode kernels
with the library's static 64 MiB scratch array instead of a caller workspace.
Its outputs must match paged_attn_decode's (same tolerance as the decode
parity tests) on two calls in a row, with and without shared-prefix groups;
shapes that need more scratch than the array holds are refused.

This file is named so that pytest collects it last.
"""
import numpy as np
import pytest
import torch

from paper_2605_11232_gb300 import batch as B
from paper_2605_11232_gb300 import pkv
from paper_2605_11232_gb300.workloads import make_workload

from _lib import need_gpu

pytestmark = pytest.mark.gpu

MAX_ABS, MEAN_ABS = 1e-2, 1e-3


def _within(a, b):
    d = (a.float() - b.float()).abs()
    return d.max().item() <= MAX_ABS and d.mean().item() <= MEAN_ABS


@pytest.mark.parametrize("use_groups", [False, True])
def test_noalloc_matches_workspace_decode_twice(use_groups):
    need_gpu()
    w = make_workload("l8b_decode", scale_requests=0.25)
    b = B.build_batch(w, poison=True)
    B.run_write(b)
    Rd = b.dec.stop - b.dec.start
    shape = (Rd, w.num_q_heads, w.head_dim)
    ref = torch.empty(shape, dtype=torch.bfloat16, device="cuda")
    ref_lse = torch.empty(shape[:2], dtype=torch.float32, device="cuda")
    ws = B.decode_workspace(b, use_groups)
    B.run_decode(b, ref, ref_lse, ws, use_groups)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    groups = b.groups if use_groups else None
    rows = B.new_token_rows(w, b.dec)
    for _ in range(2):
        out = torch.full(shape, float("nan"), dtype=torch.bfloat16, device="cuda")
        lse = torch.full(shape[:2], float("nan"), dtype=torch.float32, device="cuda")
        pkv.paged_attn_decode_noalloc(b.pool, b.q[rows], out, lse, b.context_lens[b.dec],
                                      b.table[b.dec], w.scale, groups)
        assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
        assert torch.isfinite(out.float()).all()
        assert _within(out, ref)
        assert (lse - ref_lse).abs().max().item() <= 1e-3
    b.close()


def test_noalloc_refuses_shapes_beyond_the_static_scratch():
    need_gpu()
    w = make_workload("l70b_decode", scale_requests=1.0, values=False)
    kc = torch.zeros((8, w.num_kv_heads, 16, w.head_dim), dtype=torch.bfloat16, device="cuda")
    pool = pkv.kv_pool_create(8, w.num_kv_heads, w.head_dim, kc, kc.clone())
    R = w.num_requests
    need = pkv.paged_attn_decode_workspace_size(pool, R, w.num_q_heads, 600)
    assert need > 64 << 20
    q = torch.zeros((R, w.num_q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
    out = torch.empty_like(q)
    ctx = torch.ones(R, dtype=torch.int32, device="cuda")
    table = torch.zeros((R, 600), dtype=torch.int32, device="cuda")
    with pytest.raises(pkv.PkvError) as e:
        pkv.paged_attn_decode_noalloc(pool, q, out, None, ctx, table, w.scale, None)
    assert e.value.code == pkv.PKV_ERR_WORKSPACE
    assert "static scratch" in pkv.pkv_last_error()
    pkv.kv_pool_destroy(pool)
