"""The binding refuses tensors whose dtype or shape differs from the layout a
C entry point reads, before it takes any device pointer (CPU: the tensors
here are CPU tensors, so a call whose arguments all pass the checks stops at
the device check instead)."""
import re

import pytest
import torch

from paper_2605_11232_gb300 import pkv

from _lib import built_lib

NB, HKV, D, HQ = 32, 2, 64, 8
BF = torch.bfloat16


@pytest.fixture
def pool():
    built_lib()
    p = pkv.kv_pool_create(NB, HKV, D)        # metadata-only pool
    yield p
    pkv.kv_pool_destroy(p)


def refused(match, fn, *args):
    with pytest.raises(ValueError, match=match):
        fn(*args)


def reaches_device_check(fn, *args):
    refused("expected a CUDA tensor", fn, *args)


def test_pool_geometry_is_recorded_and_dropped():
    built_lib()
    p = pkv.kv_pool_create(NB, HKV, D)
    assert pkv._pool_geometry(p) == (NB, HKV, D)
    pkv.kv_pool_destroy(p)
    assert pkv._pool_geometry(p) is None


def test_pool_create_checks_cache_shape_and_dtype():
    built_lib()
    good = torch.zeros((NB, HKV, 16, D), dtype=BF)
    refused(re.escape("k_cache must have shape [32, 2, 16, 64]"), pkv.kv_pool_create, NB, HKV, D,
            torch.zeros((NB - 1, HKV, 16, D), dtype=BF), good)
    refused("v_cache must be torch.bfloat16", pkv.kv_pool_create, NB, HKV, D, good,
            torch.zeros((NB, HKV, 16, D), dtype=torch.float16))
    refused("v_cache is required", pkv.kv_pool_create, NB, HKV, D, good, None)
    reaches_device_check(pkv.kv_pool_create, NB, HKV, D, good, good.clone())


def test_cache_write_checks(pool):
    T = 10
    k = torch.zeros((T, HKV, D), dtype=BF)
    slots = torch.zeros(T, dtype=torch.int64)
    w = pkv.kv_cache_write
    refused("slot_mapping must be torch.int64", w, pool, k, k, slots.to(torch.int32))
    refused("k_new has 9 rows for 10 slots", w, pool, k[:9], k, slots)
    refused("v_new must be torch.bfloat16", w, pool, k, k.float(), slots)
    refused(re.escape("v_new rows must be [num_kv_heads][head_dim] = [2, 64]"), w, pool, k,
            torch.zeros((T, HKV, 2 * D), dtype=BF), slots)
    refused("k_new must have 3 dimensions", w, pool, k.reshape(T, HKV * D), k, slots)
    reaches_device_check(w, pool, k, k, slots)
    reaches_device_check(w, pool, torch.zeros((T + 5, HKV, D), dtype=BF), k, slots)   # extra rows unread


@pytest.mark.parametrize("fn", ["paged_attn_decode", "paged_attn_decode_noalloc"])
def test_decode_checks(pool, fn):
    R = 4
    q = torch.zeros((R, HQ, D), dtype=BF)
    out = torch.zeros_like(q)
    lse = torch.zeros((R, HQ), dtype=torch.float32)
    ctx = torch.ones(R, dtype=torch.int32)
    table = torch.zeros((R, 3), dtype=torch.int32)
    ws = torch.zeros(1024, dtype=torch.uint8)

    def call(q=q, out=out, lse=lse, ctx=ctx, table=table):
        if fn == "paged_attn_decode":
            return pkv.paged_attn_decode(pool, q, out, lse, ctx, table, 0.125, None, ws)
        return pkv.paged_attn_decode_noalloc(pool, q, out, lse, ctx, table, 0.125, None)

    refused("context_lens must be torch.int32", lambda: call(ctx=ctx.long()))
    refused("block_table must have 2 dimensions", lambda: call(table=table.reshape(-1)))
    refused("block_table has 3 rows for 4 requests", lambda: call(table=table[:3]))
    refused("q has 3 rows, 4 needed", lambda: call(q=q[:3]))
    refused("q head dim 128 != the pool's 64", lambda: call(q=torch.zeros((R, HQ, 128), dtype=BF)))
    refused("3 query heads are not a multiple of the pool's 2 kv heads",
            lambda: call(q=torch.zeros((R, 3, D), dtype=BF), out=torch.zeros((R, 3, D), dtype=BF)))
    refused("out has 3 rows, 4 needed", lambda: call(out=out[:3]))
    refused("out must be torch.bfloat16", lambda: call(out=out.float()))
    refused(re.escape("out rows must be [8, 64]"), lambda: call(out=torch.zeros((R, HQ // 2, D), dtype=BF)))
    refused("lse must have 8 columns, got 4", lambda: call(lse=lse[:, :4]))
    refused("lse has 3 rows, 4 needed", lambda: call(lse=lse[:3]))
    refused("lse must be torch.float32", lambda: call(lse=lse.double()))
    reaches_device_check(call)
    reaches_device_check(lambda: call(lse=None))


def test_prefill_checks(pool):
    T, R = 12, 2
    q = torch.zeros((T, HQ, D), dtype=BF)
    out = torch.zeros_like(q)
    lse = torch.zeros((T, HQ), dtype=torch.float32)
    cu = torch.tensor([0, 5, 12], dtype=torch.int32)
    ctx = torch.tensor([40, 12], dtype=torch.int32)
    table = torch.zeros((R, 3), dtype=torch.int32)

    def call(q=q, out=out, lse=lse, cu=cu, ctx=ctx, table=table):
        return pkv.paged_attn_prefill(pool, q, out, lse, cu, ctx, table, 7, 0.125)

    refused("out must have q's shape", lambda: call(out=torch.zeros((T + 1, HQ, D), dtype=BF)))
    refused("lse must have 12 rows", lambda: call(lse=torch.zeros((T + 1, HQ), dtype=torch.float32)))
    refused("cu_seqlens_q must have 3 entries", lambda: call(cu=cu[:2]))
    refused("cu_seqlens_q must be torch.int32", lambda: call(cu=cu.long()))
    refused("block_table has 1 rows for 2 requests", lambda: call(table=table[:1]))
    refused("q must be torch.bfloat16", lambda: call(q=q.half(), out=out.half()))
    reaches_device_check(call)
    reaches_device_check(lambda: call(lse=None))


def test_prefix_group_checks():
    G = 2
    gs = torch.tensor([0, 2, 4], dtype=torch.int32)
    mr = torch.arange(4, dtype=torch.int32)
    gb = torch.tensor([3, 5], dtype=torch.int32)
    gor = torch.tensor([0, 0, 1, 1], dtype=torch.int32)
    mk = pkv.make_prefix_groups
    refused("group_start has 2 entries, 3 needed", mk, G, 5, 2, gs[:2], mr, gb, gor)
    refused("group_blocks has 1 entries, 2 needed", mk, G, 5, 2, gs, mr, gb[:1], gor)
    refused("member_req must be torch.int32", mk, G, 5, 2, gs, mr.long(), gb, gor)
    refused("group_of_req is required", mk, G, 5, 2, gs, mr, gb, None)
    reaches_device_check(mk, G, 5, 2, gs, mr, gb, gor)
    # no groups: an empty descriptor needs no tensors
    assert mk().num_groups == 0


def test_decode_step_checks(pool):
    R, T = 4, 4
    layout = pkv.StepLayout(q=0, k_new=1024, v_new=2048, slot_mapping=3072, context_lens=3328,
                            bytes=3456)
    host = torch.zeros(layout.bytes, dtype=torch.uint8)
    dev = torch.zeros(layout.bytes, dtype=torch.uint8)
    table = torch.zeros((R, 3), dtype=torch.int32)
    out = torch.zeros((R, HQ, D), dtype=BF)
    lse = torch.zeros((R, HQ), dtype=torch.float32)
    ws = torch.zeros(1024, dtype=torch.uint8)

    def call(**kw):
        a = dict(host_in=host, dev_in=dev, block_table=table, num_q_heads=HQ, out=out, lse=lse,
                 host_out=None, host_lse=None)
        a.update(kw)
        return pkv.paged_attn_decode_step(pool, a["host_in"], a["dev_in"], layout, T, a["block_table"],
                                          a["num_q_heads"], 0.125, None, ws, a["out"], a["lse"],
                                          a["host_out"], a["host_lse"])

    refused("host_in holds 3440 bytes, the layout needs 3456", lambda: call(host_in=host[:-16]))
    refused("dev_in holds 3440 bytes", lambda: call(dev_in=dev[:-16]))
    refused("block_table must be torch.int32", lambda: call(block_table=table.long()))
    refused(re.escape("out must be [>= 4][8][head_dim]"), lambda: call(out=out[:3]))
    refused(re.escape("out must be [>= 4][9][head_dim]"), lambda: call(num_q_heads=HQ + 1))
    refused("out head dim 128 != the pool's 64", lambda: call(out=torch.zeros((R, HQ, 128), dtype=BF)))
    refused(re.escape("lse must be [>= 4][8]"), lambda: call(lse=lse[:, :4].contiguous()))
    refused("host_out must match", lambda: call(host_out=torch.zeros((R - 1, HQ, D), dtype=BF)))
    refused("host_lse needs its device tensor",
            lambda: call(lse=None, host_lse=torch.zeros((R, HQ), dtype=torch.float32)))
    # a host buffer passes the checks and stops at the device check of dev_in
    reaches_device_check(lambda: call(host_out=torch.zeros_like(out), host_lse=torch.zeros_like(lse)))
