"""Host pool, reference counts, block tables and slot mapping (CPU, via the C ABI)."""
import json
import os

import numpy as np
import pytest

import oracle
from paper_2605_11232_gb300 import pkv
from paper_2605_11232_gb300.workloads import make_workload

from _lib import built_lib

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


@pytest.fixture
def pool():
    built_lib()
    p = pkv.kv_pool_create(32, 2, 64)        # metadata-only pool
    yield p
    pkv.kv_pool_destroy(p)


def test_identity_order_and_refcounts(pool):
    ids = pkv.kv_pool_alloc(pool, 5)
    assert list(ids) == [0, 1, 2, 3, 4]
    assert pkv.kv_pool_num_free(pool) == 27
    assert all(pkv.kv_pool_refcount(pool, i) == 1 for i in ids)
    pkv.kv_pool_retain(pool, ids[:2])
    assert pkv.kv_pool_refcount(pool, 0) == 2
    pkv.kv_pool_release(pool, ids)
    assert pkv.kv_pool_refcount(pool, 0) == 1 and pkv.kv_pool_refcount(pool, 4) == 0
    assert pkv.kv_pool_num_free(pool) == 30


def test_out_of_blocks_is_all_or_nothing(pool):
    pkv.kv_pool_alloc(pool, 30)
    with pytest.raises(pkv.PkvError) as e:
        pkv.kv_pool_alloc(pool, 3)
    assert e.value.code == pkv.PKV_ERR_OUT_OF_BLOCKS
    assert pkv.kv_pool_num_free(pool) == 2


def test_release_errors_leave_pool_unchanged(pool):
    ids = pkv.kv_pool_alloc(pool, 2)
    with pytest.raises(pkv.PkvError) as e:
        pkv.kv_pool_release(pool, [ids[0], ids[0]])       # one reference only
    assert e.value.code == pkv.PKV_ERR_REFCOUNT
    assert pkv.kv_pool_refcount(pool, int(ids[0])) == 1
    with pytest.raises(pkv.PkvError):
        pkv.kv_pool_release(pool, [17])                   # a free block
    with pytest.raises(pkv.PkvError):
        pkv.kv_pool_retain(pool, [99])                    # out of range
    with pytest.raises(pkv.PkvError):
        pkv.kv_pool_retain(pool, [20])                    # free, cannot be shared


def test_seeded_placement_is_a_permutation():
    built_lib()
    a = pkv.kv_pool_create(64, 2, 64, placement_seed=12345)
    b = pkv.kv_pool_create(64, 2, 64, placement_seed=12345)
    c = pkv.kv_pool_create(64, 2, 64, placement_seed=999)
    ia, ib, ic = (pkv.kv_pool_alloc(x, 64) for x in (a, b, c))
    assert sorted(ia) == list(range(64))
    assert list(ia) == list(ib) and list(ia) != list(ic) and list(ia) != list(range(64))
    for x in (a, b, c):
        pkv.kv_pool_destroy(x)


def test_alloc_sequence_shares_prefix(pool):
    pre = pkv.kv_pool_alloc(pool, 3)
    row1 = pkv.kv_pool_alloc_sequence(pool, pre, 5)
    row2 = pkv.kv_pool_alloc_sequence(pool, pre, 4)
    assert list(row1[:3]) == list(pre) == list(row2[:3])
    assert len(set(row1[3:]) | set(row2[3:])) == 3
    assert all(pkv.kv_pool_refcount(pool, int(i)) == 3 for i in pre)
    with pytest.raises(pkv.PkvError):
        pkv.kv_pool_alloc_sequence(pool, pre, 100)
    assert all(pkv.kv_pool_refcount(pool, int(i)) == 3 for i in pre)


def test_slot_mapping_matches_oracle_and_rejects_shared_writes(pool):
    pre = pkv.kv_pool_alloc(pool, 2)
    rows = [pkv.kv_pool_alloc_sequence(pool, pre, n) for n in (3, 4, 5)]
    width = 6
    table = np.full((3, width), -1, np.int32)
    for r, row in enumerate(rows):
        table[r, : len(row)] = row
    ctx = np.array([40, 50, 70], np.int32)
    new = np.array([1, 10, 38], np.int32)
    got = pkv.kv_slot_mapping(pool, table, ctx, new)
    want = oracle.slot_mapping(table, ctx, new, 16)
    assert np.array_equal(got, want)
    # a new token inside the shared prefix blocks is refused
    with pytest.raises(pkv.PkvError) as e:
        pkv.kv_slot_mapping(pool, table, ctx, np.array([1, 10, 60], np.int32))
    assert e.value.code == pkv.PKV_ERR_SHARED_BLOCK_WRITE
    # without a pool there is no ownership check
    got2 = pkv.kv_slot_mapping(None, table, ctx, np.array([1, 10, 60], np.int32))
    assert np.array_equal(got2, oracle.slot_mapping(table, ctx, [1, 10, 60], 16))


def test_slot_mapping_rejects_contexts_wider_than_the_table():
    """A context longer than 16 x the table width is refused before any table
    entry is read, up to the largest int32 length (no overflow in the width
    test)."""
    built_lib()
    table = np.arange(4, dtype=np.int32)[None, :]
    for L in (65, 2**31 - 16, 2**31 - 8, 2**31 - 1):
        with pytest.raises(pkv.PkvError) as e:
            pkv.kv_slot_mapping(None, table, [L], [1])
        assert e.value.code == pkv.PKV_ERR_INVALID_ARG
    assert list(pkv.kv_slot_mapping(None, table, [64], [1])) == [63]


def test_kernel_calls_need_device_caches(pool):
    with pytest.raises(pkv.PkvError) as e:
        pkv._check(pkv.load().kv_cache_write(pool, None, None, None, 1, None))
    assert e.value.code == pkv.PKV_ERR_INVALID_ARG


def test_unsupported_shapes_rejected():
    built_lib()
    for kw in (dict(block_size=32), dict(head_dim=96)):
        args = dict(num_blocks=8, num_kv_heads=1, head_dim=64)
        args.update(kw)
        with pytest.raises(pkv.PkvError) as e:
            pkv.kv_pool_create(**args)
        assert e.value.code == pkv.PKV_ERR_UNSUPPORTED


def _paged_waste(w):
    """Allocate every request of a workload in a metadata-only pool, return the
    fraction of allocated slots that hold no token (shared blocks once)."""
    p = pkv.kv_pool_create(w.num_blocks, w.num_kv_heads, w.head_dim, placement_seed=w.placement_seed)
    pre = [pkv.kv_pool_alloc(p, P // 16) for P in w.prefix_lens]
    for r in range(w.num_requests):
        g = int(w.group_of_req[r])
        nblk = (int(w.context_lens[r]) + 15) // 16
        pkv.kv_pool_alloc_sequence(p, pre[g] if g >= 0 else None, nblk)
    used = w.num_blocks - pkv.kv_pool_num_free(p)
    pkv.kv_pool_destroy(p)
    tokens = sum(w.prefix_lens) + sum(int(w.context_lens[r]) - w.prefix_len_of(r)
                                      for r in range(w.num_requests))
    return 1.0 - tokens / (16.0 * used)


@pytest.mark.parametrize("name", ["tiny", "l8b_decode", "l8b_prefill", "qwen_mixed", "l70b_decode"])
def test_paged_waste_below_paper_bound(name):
    """Sec. 5.4 reports paged KV waste under 4% (from ~60% contiguous)."""
    built_lib()
    fig = json.load(open(os.path.join(GOLDEN, "paper_figures.json")))
    w = make_workload(name, values=False)
    assert _paged_waste(w) < fig["paged_kv_waste_upper_bound"]["value"]


def test_check_block_table_on_the_host():
    """Every entry a kernel reads (the first ceil(L / 16) of a row) must name
    an allocated block; later entries are not read and not checked."""
    built_lib()
    p = pkv.kv_pool_create(32, 2, 64)
    pre = pkv.kv_pool_alloc(p, 2)
    rows = [pkv.kv_pool_alloc_sequence(p, pre, n) for n in (3, 4)]
    table = np.full((2, 6), -1, np.int32)
    for r, row in enumerate(rows):
        table[r, : len(row)] = row
    ctx = np.array([40, 64], np.int32)                  # 3 and 4 blocks
    # both rows hold the two prefix blocks: reference count 3 (two rows + the
    # allocation), which the check accepts
    assert [pkv.kv_pool_refcount(p, int(b)) for b in pre] == [3, 3]
    pkv.pkv_check_block_table(p, table, ctx)            # valid; -1 padding past the context
    table[1, 5] = 999                                   # past request 1's context: not read
    pkv.pkv_check_block_table(p, table, ctx)
    for r, j, v, code in ((1, 3, 999, pkv.PKV_ERR_INVALID_ARG), (0, 2, -1, pkv.PKV_ERR_INVALID_ARG),
                          (1, 0, 31, pkv.PKV_ERR_REFCOUNT)):     # block 31 is free
        bad = table.copy()
        bad[r, j] = v
        with pytest.raises(pkv.PkvError) as e:
            pkv.pkv_check_block_table(p, bad, ctx)
        assert e.value.code == code and e.value.bad_request == r
    for c, code in (([40, 97], pkv.PKV_ERR_INVALID_ARG), ([-1, 64], pkv.PKV_ERR_INVALID_ARG)):
        with pytest.raises(pkv.PkvError) as e:
            pkv.pkv_check_block_table(p, table, np.array(c, np.int32))
        assert e.value.code == code
    # a released row's private blocks are free again: the stale row is refused
    pkv.kv_pool_release(p, rows[1])
    with pytest.raises(pkv.PkvError) as e:
        pkv.pkv_check_block_table(p, table, ctx)
    assert e.value.bad_request == 1
    pkv.kv_pool_destroy(p)
