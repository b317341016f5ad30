"""KV-block transfer between pools (prefill/decode disaggregation, Sec. 2 and
Sec. 7): pkv_blocks_gather / pkv_blocks_scatter through a staging buffer.

Checked bit for bit: the staging buffer holds the source blocks' bytes, the
destination pool holds them in its newly allocated blocks and nothing else
changed, every request read back through its new block-table row (the
oracle's gather) equals its logical K/V, and decode over the destination
pool gives the source pool's output bits.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2605_11232_gb300 import batch as B
from paper_2605_11232_gb300 import pkv
from paper_2605_11232_gb300.workloads import make_workload

from _lib import built_lib, need_gpu


def _bits(t):
    return t.view(torch.int16)


def test_staging_size_and_argument_checks():
    built_lib()
    p = pkv.kv_pool_create(32, 8, 128)
    assert pkv.pkv_blocks_staging_size(p, 3) == 3 * 2 * 8 * 16 * 128 * 2
    assert pkv.pkv_blocks_staging_size(p, 0) == 0
    with pytest.raises(pkv.PkvError) as e:
        pkv.pkv_blocks_staging_size(p, -1)
    assert e.value.code == pkv.PKV_ERR_INVALID_ARG
    pkv.kv_pool_destroy(p)


@pytest.mark.gpu
@pytest.mark.parametrize("name,scale", [("l8b_decode", 0.125), ("tiny_decode", 1.0), ("qwen_mixed", 0.0625)])
def test_transfer_requests_bit_exact(name, scale):
    need_gpu()
    w = make_workload(name, scale_requests=scale)
    src = B.build_batch(w, poison=True)
    B.run_write(src)
    Rd = src.dec.stop - src.dec.start
    ref = torch.empty((Rd, w.num_q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
    ref_lse = torch.empty((Rd, w.num_q_heads), dtype=torch.float32, device="cuda")
    ws = B.decode_workspace(src, False)
    B.run_decode(src, ref, ref_lse, ws, False)
    assert pkv.pkv_check_device_errors(src.pool) == pkv.PKV_OK

    # every decode request's whole row moves; a shared prefix block once
    rows = range(src.dec.start, src.dec.stop)
    nblk = [(int(w.context_lens[r]) + 15) // 16 for r in rows]
    all_ids = np.concatenate([src.table_host[r, :n] for r, n in zip(rows, nblk)]).astype(np.int32)
    src_ids, first, uses = np.unique(all_ids, return_index=True, return_counts=True)
    order = np.argsort(first)                       # in the order the rows name them
    src_ids, uses = src_ids[order].astype(np.int32), uses[order]
    n = len(src_ids)

    # destination: same geometry, its own placement, NaN-poisoned
    nb = n + 5
    shape = (nb,) + tuple(src.k_cache.shape[1:])
    dk = torch.full(shape, float("nan"), dtype=torch.bfloat16, device="cuda")
    dv = torch.full(shape, float("nan"), dtype=torch.bfloat16, device="cuda")
    dst = pkv.kv_pool_create(nb, w.num_kv_heads, w.head_dim, dk, dv, placement_seed=77)
    before_k, before_v = _bits(dk).clone(), _bits(dv).clone()
    dst_ids = pkv.kv_pool_alloc(dst, n)
    for x, k in zip(dst_ids, uses):                 # one reference per row that names it
        if k > 1:
            pkv.kv_pool_retain(dst, np.full(k - 1, x, np.int32))
    to_dst = dict(zip(src_ids.tolist(), dst_ids.tolist()))
    staging = torch.full((pkv.pkv_blocks_staging_size(src.pool, n) // 2,), float("nan"),
                         dtype=torch.bfloat16, device="cuda")
    sid, did = torch.from_numpy(src_ids).cuda(), torch.from_numpy(np.asarray(dst_ids, np.int32)).cuda()
    pkv.pkv_blocks_gather(src.pool, sid, staging)
    pkv.pkv_blocks_scatter(dst, did, staging)
    assert pkv.pkv_check_device_errors(src.pool) == pkv.PKV_OK
    assert pkv.pkv_check_device_errors(dst) == pkv.PKV_OK

    # staging: block i's K tile then its V tile
    st = staging.view(n, 2, *src.k_cache.shape[1:])
    assert torch.equal(_bits(st[:, 0]), _bits(src.k_cache[sid.long()]))
    assert torch.equal(_bits(st[:, 1]), _bits(src.v_cache[sid.long()]))
    # destination: the moved blocks, and every other block untouched
    moved = torch.zeros(nb, dtype=torch.bool, device="cuda")
    moved[did.long()] = True
    assert torch.equal(_bits(dk[did.long()]), _bits(src.k_cache[sid.long()]))
    assert torch.equal(_bits(dv[did.long()]), _bits(src.v_cache[sid.long()]))
    assert torch.equal(_bits(dk[~moved]), before_k[~moved]) and torch.equal(_bits(dv[~moved]), before_v[~moved])

    # each request read back through its new table row is its logical K/V
    width = src.table.shape[1]
    table = np.full((Rd, width), -1, np.int32)
    for i, (r, k) in enumerate(zip(rows, nblk)):
        table[i, :k] = [to_dst[int(x)] for x in src.table_host[r, :k]]
    kp, vp = _bits(dk).cpu().numpy().view(np.uint16), _bits(dv).cpu().numpy().view(np.uint16)
    for i, r in enumerate(rows):
        k_log, v_log = w.request_kv(r)
        L = int(w.context_lens[r])
        assert np.array_equal(oracle.gather(kp, table[i], L), k_log.view(torch.int16).numpy().view(np.uint16))
        assert np.array_equal(oracle.gather(vp, table[i], L), v_log.view(torch.int16).numpy().view(np.uint16))

    # decode over the destination pool: the source pool's bits
    out = torch.empty_like(ref)
    lse = torch.empty_like(ref_lse)
    rows_q = B.new_token_rows(w, src.dec)
    pkv.paged_attn_decode(dst, src.q[rows_q], out, lse, src.context_lens[src.dec], torch.from_numpy(table).cuda(),
                          w.scale, None, ws)
    assert pkv.pkv_check_device_errors(dst) == pkv.PKV_OK
    assert torch.equal(out, ref) and torch.equal(lse, ref_lse)

    # the references move: the source releases the rows, the destination
    # holds one per row
    for r, k in zip(rows, nblk):
        pkv.kv_pool_release(src.pool, src.table_host[r, :k])
    assert [pkv.kv_pool_refcount(dst, int(x)) for x in dst_ids] == uses.tolist()
    pkv.kv_pool_destroy(dst)
    src.close()


@pytest.mark.gpu
def test_transfer_bad_block_id_latches_bounds():
    """An id outside the pool is skipped and latches DEVICE_BOUNDS; the other
    blocks still move."""
    need_gpu()
    k = torch.randn((8, 2, 16, 64), device="cuda").to(torch.bfloat16)
    v = torch.randn((8, 2, 16, 64), device="cuda").to(torch.bfloat16)
    p = pkv.kv_pool_create(8, 2, 64, k, v)
    ids = torch.tensor([3, 99, 5], dtype=torch.int32, device="cuda")
    staging = torch.zeros((pkv.pkv_blocks_staging_size(p, 3) // 2,), dtype=torch.bfloat16, device="cuda")
    pkv.pkv_blocks_gather(p, ids, staging)
    assert pkv.pkv_check_device_errors(p) == pkv.PKV_ERR_DEVICE_BOUNDS
    st = staging.view(3, 2, 2, 16, 64)
    assert torch.equal(_bits(st[0, 0]), _bits(k[3])) and torch.equal(_bits(st[2, 1]), _bits(v[5]))
    assert bool((st[1] == 0).all())
    pkv.kv_pool_destroy(p)
