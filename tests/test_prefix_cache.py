"""Automatic prefix caching index (pkv_prefix_cache_*, host C ABI).

First the plain definition in ``oracle/prefix_cache.py`` is pinned on hand-
worked cases (longest cached run of whole blocks, a changed token cutting the
run at its block, eviction order of least recently used leaves that no
request holds, reference counts).  Then the library is run against it on
random request traffic over shared policy prefixes, with full 64-bit keys and
with keys cut to 4 bits (every lookup meets colliding keys, so sharing must
come from the token-by-token check).  CPU only: a pool without caches.
"""
import numpy as np
import pytest

from oracle.prefix_cache import BS, PoolModel, PrefixCacheModel
from paper_2605_11232_gb300 import pkv


# ---- pins of the definition ------------------------------------------------

def test_definition_hand_example():
    pool = PoolModel(16)
    c = PrefixCacheModel(pool)
    A = list(range(100, 148)) + [7] * 5          # 3 full blocks + a partial one
    pool.alloc([0, 1, 2, 3])
    assert c.insert(A, [0, 1, 2, 3]) == 3        # the partial block is not cached
    assert pool.ref[:4] == [2, 2, 2, 1]
    assert c.match(A) == [0, 1, 2]
    assert pool.ref[:3] == [3, 3, 3]
    B = A[:16] + [5] * 40                        # shares block 0 only
    assert c.match(B) == [0]
    C = list(A)
    C[20] += 1                                   # a change inside block 1 cuts the run there
    assert c.match(C) == [0]
    assert c.match(A[:47]) == [0, 1]             # 47 tokens: two full blocks
    assert c.match(A, max_ids=1) == [0]
    assert c.match([1, 2, 3]) == []


def test_definition_eviction_order():
    pool = PoolModel(16)
    c = PrefixCacheModel(pool)
    A = list(range(0, 48))
    B = list(range(0, 16)) + list(range(500, 532))
    pool.alloc([0, 1, 2])
    c.insert(A, [0, 1, 2])                        # tick 1: A0 A1 A2
    pool.alloc([3, 4])
    c.insert(B, [0, 3, 4])                        # tick 2: A0 (shared) B1 B2
    # requests end: only the index holds the blocks
    pool.release([0, 1, 2])
    pool.release([3, 4])
    assert c.match(A) == [0, 1, 2]               # tick 3: A's path is now the most recent
    pool.release([0, 1, 2])
    # B2 (tick 2, depth 2) goes first; then B1 (now a leaf, tick 2); then A2,
    # A1; A0 (the root of both paths) last
    assert c.evict(2) == [4, 3]
    assert c.evict(10) == [2, 1, 0]
    assert c.size() == 0 and pool.num_free() == 16


def test_definition_held_blocks_are_not_evicted():
    pool = PoolModel(8)
    c = PrefixCacheModel(pool)
    A = list(range(32))
    pool.alloc([5, 6])
    c.insert(A, [5, 6])
    assert c.evict(4) == []                      # the request still holds both
    pool.release([6])
    assert c.evict(4) == [6]                     # only the index holds block 6; 5 is still held
    assert pool.ref[5] == 2 and pool.ref[6] == 0
    pool.release([5])
    assert c.evict(4) == [5]


# ---- the library against the definition -----------------------------------

def _refcounts(pool, n):
    return [pkv.kv_pool_refcount(pool, i) for i in range(n)]


def test_library_hand_example():
    pool = pkv.kv_pool_create(16, 2, 64)
    cache = pkv.pkv_prefix_cache_create(pool)
    A = np.arange(100, 153, dtype=np.int32)
    ids = pkv.kv_pool_alloc(pool, 4)
    assert pkv.pkv_prefix_cache_insert(cache, A, ids) == 3
    assert _refcounts(pool, 16)[ids[0]] == 2 and pkv.kv_pool_refcount(pool, int(ids[3])) == 1
    assert list(pkv.pkv_prefix_cache_match(cache, A)) == list(ids[:3])
    C = A.copy()
    C[20] += 1
    assert list(pkv.pkv_prefix_cache_match(cache, C)) == [ids[0]]
    assert pkv.pkv_prefix_cache_size(cache) == 3
    pkv.pkv_prefix_cache_destroy(cache)          # drops the index's references
    assert pkv.kv_pool_refcount(pool, int(ids[0])) == 3   # the request + the two matches
    pkv.kv_pool_destroy(pool)


def test_library_rejects_free_blocks():
    pool = pkv.kv_pool_create(8, 2, 64)
    cache = pkv.pkv_prefix_cache_create(pool)
    with pytest.raises(pkv.PkvError) as e:
        pkv.pkv_prefix_cache_insert(cache, np.arange(16, dtype=np.int32), [3])
    assert e.value.code == pkv.PKV_ERR_REFCOUNT
    pkv.pkv_prefix_cache_destroy(cache)
    pkv.kv_pool_destroy(pool)


@pytest.mark.parametrize("weak", [False, True])
@pytest.mark.parametrize("seed", [0, 1, 2])
def test_library_matches_definition_on_random_traffic(weak, seed):
    rng = np.random.default_rng(seed)
    NB = 300
    pool = pkv.kv_pool_create(NB, 2, 64, placement_seed=seed + 1)
    cache = pkv.pkv_prefix_cache_create(pool, weak_hash=weak)
    pm = PoolModel(NB)
    cm = PrefixCacheModel(pm)
    # a few policy prefixes (some not a whole number of blocks), a small
    # token alphabet so that different requests often agree on blocks
    prefixes = [rng.integers(0, 40, int(rng.integers(1, 10)) * BS + int(rng.integers(0, BS))).astype(np.int32)
                for _ in range(4)]
    live = []
    for step in range(400):
        op = rng.random()
        if op < 0.5:
            p = prefixes[int(rng.integers(len(prefixes)))]
            t = np.concatenate([p, rng.integers(0, 40, int(rng.integers(0, 70))).astype(np.int32)])
            if rng.random() < 0.25 and len(t):
                t[int(rng.integers(len(t)))] += 1
            got = pkv.pkv_prefix_cache_match(cache, t)
            assert list(got) == cm.match(t.tolist())
            n_new = (len(t) + BS - 1) // BS - len(got)
            short = n_new - pkv.kv_pool_num_free(pool)
            if short > 0:
                ev = pkv.pkv_prefix_cache_evict(cache, short)
                assert list(ev) == cm.evict(short)
            if n_new > pkv.kv_pool_num_free(pool):   # still no room: give the match back
                pkv.kv_pool_release(pool, got)
                pm.release(got.tolist())
                continue
            new = pkv.kv_pool_alloc(pool, n_new)
            pm.alloc(new.tolist())
            row = np.concatenate([got, new]).astype(np.int32)
            assert pkv.pkv_prefix_cache_insert(cache, t, row) == cm.insert(t.tolist(), row.tolist())
            live.append(row)
        elif op < 0.85 and live:
            row = live.pop(int(rng.integers(len(live))))
            pkv.kv_pool_release(pool, row)
            pm.release(row.tolist())
        else:
            k = int(rng.integers(0, 25))
            assert list(pkv.pkv_prefix_cache_evict(cache, k)) == cm.evict(k)
        assert _refcounts(pool, NB) == pm.ref
        assert pkv.pkv_prefix_cache_size(cache) == cm.size()
    for row in live:
        pkv.kv_pool_release(pool, row)
    pkv.pkv_prefix_cache_destroy(cache)
    assert pkv.kv_pool_num_free(pool) == NB
    pkv.kv_pool_destroy(pool)


@pytest.mark.gpu
def test_matched_blocks_feed_decode():
    """Request 1 writes its K/V through the cache and registers its blocks;
    request 2, sharing its first 96 tokens, takes those 6 blocks from the
    index, writes only its own suffix and decodes: both outputs against the
    fp64 oracle over the logical K/V (the shared positions hold request 1's
    values, as a model's cache would)."""
    import torch

    import oracle
    from _lib import need_gpu
    need_gpu()
    g = torch.Generator().manual_seed(31)
    Hkv, Hq, d, NB = 2, 8, 128, 64
    kc = torch.zeros((NB, Hkv, 16, d), dtype=torch.bfloat16, device="cuda")
    vc = torch.zeros_like(kc)
    pool = pkv.kv_pool_create(NB, Hkv, d, kc, vc, placement_seed=5)
    cache = pkv.pkv_prefix_cache_create(pool)
    rng = np.random.default_rng(31)
    t1 = rng.integers(0, 1000, 130).astype(np.int32)
    t2 = np.concatenate([t1[:96], rng.integers(0, 1000, 75).astype(np.int32)])
    k1 = torch.randn((130, Hkv, d), generator=g).to(torch.bfloat16)
    v1 = torch.randn((130, Hkv, d), generator=g).to(torch.bfloat16)
    k2 = torch.cat([k1[:96], torch.randn((75, Hkv, d), generator=g).to(torch.bfloat16)])
    v2 = torch.cat([v1[:96], torch.randn((75, Hkv, d), generator=g).to(torch.bfloat16)])

    def write(row, L, n_new, k, v):
        table = np.full((1, 16), -1, np.int32)
        table[0, :len(row)] = row
        slots = pkv.kv_slot_mapping(pool, table, [L], [n_new])
        pkv.kv_cache_write(pool, k[L - n_new:].cuda(), v[L - n_new:].cuda(),
                           torch.from_numpy(slots).cuda(), None)
        return table

    row1 = pkv.kv_pool_alloc(pool, 9)                       # 130 tokens: 9 blocks
    tab1 = write(row1, 130, 130, k1, v1)
    assert pkv.pkv_prefix_cache_insert(cache, t1, row1) == 8
    got = pkv.pkv_prefix_cache_match(cache, t2)
    assert list(got) == list(row1[:6])                      # 96 shared tokens = 6 blocks
    row2 = np.concatenate([got, pkv.kv_pool_alloc(pool, 11 - 6)]).astype(np.int32)   # 171 tokens
    tab2 = write(row2, 171, 171 - 96, k2, v2)
    q = torch.randn((2, Hq, d), generator=g).to(torch.bfloat16)
    table = torch.from_numpy(np.concatenate([tab1, tab2])).cuda()
    ctx = torch.tensor([130, 171], dtype=torch.int32, device="cuda")
    out = torch.empty((2, Hq, d), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((2, Hq), dtype=torch.float32, device="cuda")
    ws = torch.empty(pkv.paged_attn_decode_workspace_size(pool, 2, Hq, 16), dtype=torch.uint8,
                     device="cuda")
    pkv.paged_attn_decode(pool, q.cuda(), out, lse, ctx, table, d ** -0.5, None, ws)
    assert pkv.pkv_check_device_errors(pool) == pkv.PKV_OK
    bits = lambda t: t.contiguous().view(torch.int16).numpy().view(np.uint16)
    for r, (k, v) in enumerate([(k1, v1), (k2, v2)]):
        o_ref, l_ref = oracle.attention(bits(q[r:r + 1]), bits(k), bits(v), d ** -0.5)
        e = np.abs(out[r].float().cpu().numpy().astype(np.float64) - o_ref[0])
        assert e.max() <= 1e-2 and e.mean() <= 1e-3, (e.max(), e.mean())
        assert np.abs(lse[r].cpu().numpy() - l_ref[0]).max() <= 1e-3
    pkv.pkv_prefix_cache_destroy(cache)
    pkv.kv_pool_destroy(pool)


# ---- prefix groups of a decode batch ----------------------------------------

from oracle.prefix_cache import prefix_groups  # noqa: E402


def test_groups_definition_hand_example():
    pad = [-1] * 3
    table = [[5, 6, 7, 8, 9] + pad,
             [5, 6, 7, 20, 21] + pad,
             [5, 6, 30, 31, 32] + pad,
             [9, 10, 11, 12, 13] + pad,
             [5, 6, 7, 8, 9] + pad]
    L = [80, 80, 80, 80, 33]          # the last one: (33 - 1) // 16 = 2 shareable blocks
    gor, groups = prefix_groups(table, L)
    assert gor == [0, 0, 0, -1, 0] and groups == [([0, 1, 2, 4], 2)]
    gor, groups = prefix_groups(table, L, min_shared_blocks=3)
    assert gor == [0, 0, -1, -1, -1] and groups == [([0, 1], 3)]
    gor, groups = prefix_groups(table, [16] * 5)       # one block each: nothing to share
    assert gor == [-1] * 5 and groups == []


def _check_groups(table, L, m):
    got = pkv.pkv_prefix_groups_build(table, L, m)
    gor, groups = prefix_groups(table.tolist(), list(L), m)
    assert got["group_of_req"].tolist() == gor
    assert got["num_groups"] == len(groups)
    for g, (members, shared) in enumerate(groups):
        a, b = got["group_start"][g], got["group_start"][g + 1]
        assert got["member_req"][a:b].tolist() == members
        assert int(got["group_blocks"][g]) == shared
        for r in members:   # the shared blocks head every member's row, and leave it a private one
            assert (table[r, :shared] == table[members[0], :shared]).all()
            assert shared <= (L[r] - 1) // 16
    if groups:
        assert got["max_group_blocks"] == max(s for _, s in groups)
        assert got["max_group_members"] == max(len(mm) for mm, _ in groups)


@pytest.mark.parametrize("seed", [0, 1, 2, 3])
def test_groups_library_matches_definition(seed):
    rng = np.random.default_rng(seed)
    R, MB = 60, 40
    runs = [rng.permutation(1000)[: int(rng.integers(1, 30))] for _ in range(5)]
    table = np.full((R, MB), -1, np.int32)
    L = np.zeros(R, np.int32)
    nxt = 1000
    for r in range(R):
        k = int(rng.integers(0, 6))
        head = runs[k][: int(rng.integers(0, len(runs[k]) + 1))] if k < 5 else np.zeros(0, np.int32)
        nb = int(rng.integers(len(head) + 1, MB + 1))
        own = np.arange(nxt, nxt + nb - len(head), dtype=np.int32)
        nxt += nb - len(head)
        table[r, :nb] = np.concatenate([head, own])
        L[r] = 16 * (nb - 1) + int(rng.integers(1, 17))
    for m in (1, 2, 5):
        _check_groups(table, L, m)


@pytest.mark.gpu
def test_groups_from_tables_reproduce_the_workload_groups():
    """On l8b_decode (scaled), groups derived from the block tables equal the
    workload's own descriptor, and decode with them gives the same bits."""
    import torch

    from _lib import need_gpu
    from paper_2605_11232_gb300 import batch as B
    from paper_2605_11232_gb300.workloads import make_workload
    need_gpu()
    w = make_workload("l8b_decode", scale_requests=0.25)
    b = B.build_batch(w, poison=True)
    g = pkv.pkv_prefix_groups_build(b.table_host, w.context_lens)
    assert g["num_groups"] == 1 and g["group_blocks"].tolist() == [w.prefix_lens[0] // 16]
    assert (g["group_of_req"] == 0).all()
    dev = {k: torch.from_numpy(g[k]).cuda() for k in ("group_start", "member_req", "group_blocks",
                                                      "group_of_req")}
    groups = pkv.make_prefix_groups(g["num_groups"], g["max_group_blocks"], g["max_group_members"], **dev)
    B.run_write(b)
    Rd = b.dec.stop - b.dec.start
    outs = []
    for grp in (b.groups, groups):
        out = torch.empty((Rd, w.num_q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
        ws = torch.empty(pkv.paged_attn_decode_workspace_size(b.pool, Rd, w.num_q_heads, b.table.shape[1], grp),
                         dtype=torch.uint8, device="cuda")
        pkv.paged_attn_decode(b.pool, b.q, out, None, b.context_lens, b.table, w.scale, grp, ws)
        outs.append(out.cpu())
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    assert torch.equal(outs[0], outs[1])
    b.close()
