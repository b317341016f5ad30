"""Verification of tree-shaped draft tokens (Sec. 5.3): the host masks
against the definition (CPU), and paged_attn_verify_tree against the fp64
tree oracle (GPU)."""
import numpy as np
import pytest
import torch

from oracle import tree_verify as TV
from paper_2605_11232_gb300 import pkv

from _lib import built_lib, need_gpu

MAX_ABS, MEAN_ABS, LSE_ABS = 1e-2, 1e-3, 1e-3


def _random_parents(rng, k):
    return [int(rng.integers(-1, i)) if i else -1 for i in range(k)]


def test_tree_masks_match_the_definition():
    built_lib()
    rng = np.random.default_rng(0)
    ks = [1, 5, 64, 0, 17, 3]
    parents = [_random_parents(rng, k) for k in ks]
    cu = np.concatenate([[0], np.cumsum(ks)]).astype(np.int32)
    masks = pkv.pkv_tree_masks(np.concatenate(parents).astype(np.int32), cu).view(np.uint64)
    for r, par in enumerate(parents):
        for i, path in enumerate(TV.ancestors(par)):
            assert int(masks[cu[r] + i]) == sum(1 << j for j in path)
    # a chain is the causal mask: bits 0..i
    chain = pkv.pkv_tree_masks(np.array([-1, 0, 1, 2], np.int32), np.array([0, 4], np.int32))
    assert chain.view(np.uint64).tolist() == [1, 3, 7, 15]


def test_tree_masks_reject_bad_trees():
    built_lib()
    for parent, cu in (([0], [0, 1]), ([-1, 1], [0, 2]), ([-2], [0, 1]), ([-1] * 65, [0, 65]),
                       ([-1], [1, 1])):
        with pytest.raises(pkv.PkvError) as e:
            pkv.pkv_tree_masks(np.array(parent, np.int32), np.array(cu, np.int32))
        assert e.value.code == pkv.PKV_ERR_INVALID_ARG


def _bits(t):
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


@pytest.mark.gpu
@pytest.mark.parametrize("d,hq,hkv", [(128, 32, 8), (64, 8, 2)])
def test_verify_tree_matches_oracle(d, hq, hkv):
    """12 requests, 9 of them over one shared 512-token prefix, ragged private
    contexts, 1 to 64 drafts each in random trees (chains, stars and mixed):
    every draft row against the fp64 tree oracle."""
    from paper_2605_11232_gb300 import batch as B
    from paper_2605_11232_gb300.workloads import make_workload
    need_gpu()
    rng = np.random.default_rng(d)
    R = 12
    ks = [1, 2, 8, 64, 5, 33, 7, 16, 3, 64, 9, 20]
    grp = [0 if i % 4 else -1 for i in range(R)]
    cached = [int(rng.integers(1, 30 * 16)) + (512 if g0 == 0 else 0) for g0 in grp]
    w = make_workload("custom", seed=21, custom=dict(
        Hq=hq, Hkv=hkv, d=d, prefix_lens=[512], group=grp, cached=cached, new=ks,
        decode=[False] * R))
    parents = []
    for r, k in enumerate(ks):
        if r % 3 == 0:
            parents.append([-1] + list(range(k - 1)))          # chain
        elif r % 3 == 1:
            parents.append([-1] * k)                           # star
        else:
            parents.append(_random_parents(rng, k))
    cu = np.concatenate([[0], np.cumsum(ks)]).astype(np.int32)
    masks = pkv.pkv_tree_masks(np.concatenate(parents).astype(np.int32), cu)
    b = B.build_batch(w, poison=True)
    B.run_write(b)
    T = int(cu[-1])
    out = torch.full((T, hq, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full((T, hq), float("nan"), dtype=torch.float32, device="cuda")
    pkv.paged_attn_verify_tree(b.pool, b.q, out, lse, b.cu_pre, b.context_lens, b.table, max(ks),
                               w.scale, torch.from_numpy(masks).cuda())
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    errs, lerrs = [], []
    for r in range(R):
        kr, vr = w.request_kv(r)
        o_ref, l_ref = TV.tree_verify_attention(_bits(w.request_q(r)), _bits(kr), _bits(vr),
                                                parents[r], w.scale)
        a, e = int(cu[r]), int(cu[r + 1])
        errs.append(np.abs(out[a:e].float().cpu().numpy().astype(np.float64) - o_ref).ravel())
        lerrs.append(np.abs(lse[a:e].cpu().numpy().astype(np.float64) - l_ref).ravel())
    err, lerr = np.concatenate(errs), np.concatenate(lerrs)
    assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS and lerr.max() <= LSE_ABS
    # a chain mask is the causal suffix prefill: same bits as paged_attn_prefill
    chain_rows = np.concatenate([np.arange(cu[r], cu[r + 1]) for r in range(0, R, 3)])
    ref = torch.full_like(out, float("nan"))
    pkv.paged_attn_prefill(b.pool, b.q, ref, None, b.cu_pre, b.context_lens, b.table, max(ks), w.scale)
    torch.cuda.synchronize()
    idx = torch.from_numpy(chain_rows).cuda()
    assert torch.equal(out[idx], ref[idx])
    b.close()


# ---- grouped verification: each group's shared prefix read once ----------

def test_verify_groups_build_matches_definition():
    """Token groups against a direct construction: group g lists the draft
    rows of its requests in request order; group_row is its first request."""
    built_lib()
    rng = np.random.default_rng(5)
    for R, G in ((1, 1), (7, 3), (40, 5), (5, 0)):
        ks = rng.integers(0, 9, R)
        cu = np.concatenate([[0], np.cumsum(ks)]).astype(np.int32)
        rg = rng.integers(-1, G, R).astype(np.int32) if G else np.full(R, -1, np.int32)
        tg = pkv.pkv_verify_groups_build(cu, rg, G)
        start, members, rows = [0], [], []
        for g in range(G):
            mine = [r for r in range(R) if rg[r] == g]
            members += [t for r in mine for t in range(cu[r], cu[r + 1])]
            start.append(len(members))
            rows.append(mine[0] if mine else -1)
        assert tg["group_start"].tolist() == start
        assert tg["member_token"].tolist() == members
        assert tg["group_row"].tolist() == rows
        assert tg["max_group_tokens"] == max([start[g + 1] - start[g] for g in range(G)], default=0)


def test_verify_groups_build_rejects_bad_input():
    built_lib()
    for cu, rg, G in (([0, 2], [1], 1), ([0, 2], [-2], 1), ([1, 2], [0], 1), ([0, 3, 2], [0, 0], 1)):
        with pytest.raises(pkv.PkvError) as e:
            pkv.pkv_verify_groups_build(np.array(cu, np.int32), np.array(rg, np.int32), G)
        assert e.value.code == pkv.PKV_ERR_INVALID_ARG


def test_verify_workspace_size_grows_with_prefix_parts():
    """One private slot per (token, q head) plus the prefix partials: the
    workspace without groups holds exactly T x Hq x 1 partial rows."""
    built_lib()
    p = pkv.kv_pool_create(64, 8, 128)
    T, Hq = 512, 32
    plain = pkv.paged_attn_verify_tree_workspace_size(p, T, Hq, 300)
    up = lambda x: (x + 255) & ~255
    assert plain == up(T * Hq * 128 * 4) + up(T * Hq * 8) + up(T * 8 * 4)
    vg = pkv.VerifyGroups(1, 256, T, 0, None, None, None, None, None)
    assert pkv.paged_attn_verify_tree_workspace_size(p, T, Hq, 300, vg) > plain
    pkv.kv_pool_destroy(p)


def _tree_batch(d, hq, hkv, seed):
    from paper_2605_11232_gb300 import batch as B
    from paper_2605_11232_gb300.workloads import make_workload
    rng = np.random.default_rng(seed)
    R = 12
    ks = [1, 2, 8, 64, 5, 33, 7, 16, 3, 64, 9, 20]
    grp = [0 if i % 4 else -1 for i in range(R)]
    cached = [int(rng.integers(1, 30 * 16)) + (512 if g0 == 0 else 0) for g0 in grp]
    w = make_workload("custom", seed=21, custom=dict(
        Hq=hq, Hkv=hkv, d=d, prefix_lens=[512], group=grp, cached=cached, new=ks,
        decode=[False] * R))
    parents = []
    for r, k in enumerate(ks):
        if r % 3 == 0:
            parents.append([-1] + list(range(k - 1)))
        elif r % 3 == 1:
            parents.append([-1] * k)
        else:
            parents.append(_random_parents(rng, k))
    cu = np.concatenate([[0], np.cumsum(ks)]).astype(np.int32)
    masks = pkv.pkv_tree_masks(np.concatenate(parents).astype(np.int32), cu)
    b = B.build_batch(w, poison=True)
    B.run_write(b)
    return w, b, parents, cu, masks, ks


@pytest.mark.gpu
@pytest.mark.parametrize("d,hq,hkv", [(128, 32, 8), (64, 8, 2), (128, 64, 8)])
@pytest.mark.parametrize("use_groups", [True, False])
def test_verify_grouped_matches_oracle(d, hq, hkv, use_groups):
    """paged_attn_verify_tree_grouped on the 12-request tree batch (9 requests
    over one shared 512-token prefix, 1 to 64 drafts, ragged private
    contexts): every draft row against the fp64 tree oracle, and against the
    ungrouped verification within the merge's rounding."""
    from paper_2605_11232_gb300 import batch as B
    need_gpu()
    w, b, parents, cu, masks, ks = _tree_batch(d, hq, hkv, d + hq)
    T = int(cu[-1])
    vg, keep = B.verify_groups(b) if use_groups else (None, None)
    ws = B.verify_workspace(b, vg)
    ws.fill_(0xFF)                          # NaN partials wherever a pass misses a slot
    m = torch.from_numpy(masks).cuda()
    out = torch.full((T, hq, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full((T, hq), float("nan"), dtype=torch.float32, device="cuda")
    B.run_verify_grouped(b, out, lse, m, vg, ws, max(ks))
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    errs, lerrs = [], []
    for r in range(len(ks)):
        kr, vr = w.request_kv(r)
        o_ref, l_ref = TV.tree_verify_attention(_bits(w.request_q(r)), _bits(kr), _bits(vr),
                                                parents[r], w.scale)
        a, e = int(cu[r]), int(cu[r + 1])
        errs.append(np.abs(out[a:e].float().cpu().numpy().astype(np.float64) - o_ref).ravel())
        lerrs.append(np.abs(lse[a:e].cpu().numpy().astype(np.float64) - l_ref).ravel())
    err, lerr = np.concatenate(errs), np.concatenate(lerrs)
    assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS and lerr.max() <= LSE_ABS
    ref = torch.full_like(out, float("nan"))
    ref_lse = torch.full_like(lse, float("nan"))
    pkv.paged_attn_verify_tree(b.pool, b.q, ref, ref_lse, b.cu_pre, b.context_lens, b.table, max(ks),
                               w.scale, m)
    torch.cuda.synchronize()
    assert (out.float() - ref.float()).abs().max().item() <= MAX_ABS
    assert (lse - ref_lse).abs().max().item() <= LSE_ABS
    b.close()


@pytest.mark.gpu
def test_verify_grouped_full_size():
    """The 64-request Llama-3-8B-shaped batch with 8 drafts per request over
    its shared 4096-token prefix (the benchmark's verification workload):
    every row against the ungrouped verification, and sampled rows against
    the fp64 oracle."""
    from paper_2605_11232_gb300 import batch as B
    from paper_2605_11232_gb300.workloads import make_workload
    need_gpu()
    w0 = make_workload("l8b_decode", values=False)
    R, k = w0.num_requests, 8
    w = make_workload("custom", seed=31, custom=dict(
        Hq=w0.num_q_heads, Hkv=w0.num_kv_heads, d=w0.head_dim, prefix_lens=list(w0.prefix_lens),
        group=[int(x) for x in w0.group_of_req], cached=[int(c) for c in w0.cached_lens], new=[k] * R,
        decode=[False] * R))
    rng = np.random.default_rng(31)
    parents = [_random_parents(rng, k) if r % 2 else [-1] + list(range(k - 1)) for r in range(R)]
    cu = np.arange(0, R * k + 1, k, dtype=np.int32)
    masks = torch.from_numpy(pkv.pkv_tree_masks(np.concatenate(parents).astype(np.int32), cu)).cuda()
    b = B.build_batch(w, poison=True)
    B.run_write(b)
    T = R * k
    vg, keep = B.verify_groups(b)
    ws = B.verify_workspace(b, vg)
    out = torch.full((T, w.num_q_heads, w.head_dim), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full((T, w.num_q_heads), float("nan"), dtype=torch.float32, device="cuda")
    B.run_verify_grouped(b, out, lse, masks, vg, ws, k)
    ref, ref_lse = torch.empty_like(out), torch.empty_like(lse)
    pkv.paged_attn_verify_tree(b.pool, b.q, ref, ref_lse, b.cu_pre, b.context_lens, b.table, k, w.scale, masks)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    diff = (out.float() - ref.float()).abs()
    assert diff.max().item() <= MAX_ABS and diff.mean().item() <= MEAN_ABS
    assert (lse - ref_lse).abs().max().item() <= LSE_ABS
    for r in (0, 1, R // 2, R - 1):
        kr, vr = w.request_kv(r)
        o_ref, l_ref = TV.tree_verify_attention(_bits(w.request_q(r)), _bits(kr), _bits(vr), parents[r], w.scale)
        a, e = int(cu[r]), int(cu[r + 1])
        err = np.abs(out[a:e].float().cpu().numpy().astype(np.float64) - o_ref)
        assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS
        assert np.abs(lse[a:e].cpu().numpy().astype(np.float64) - l_ref).max() <= LSE_ABS
    b.close()


@pytest.mark.gpu
def test_verify_grouped_short_cache_latches_bounds():
    """A grouped request whose cached part does not cover its group's blocks
    latches DEVICE_BOUNDS (its rows are undefined; nothing is read outside)."""
    from paper_2605_11232_gb300 import batch as B
    need_gpu()
    w, b, parents, cu, masks, ks = _tree_batch(128, 32, 8, 3)
    vg, keep = B.verify_groups(b)
    keep["group_blocks"].fill_(64)          # 1024 tokens > every member's cached part
    ws = B.verify_workspace(b, vg)
    T = int(cu[-1])
    out = torch.empty((T, 32, 128), dtype=torch.bfloat16, device="cuda")
    B.run_verify_grouped(b, out, None, torch.from_numpy(masks).cuda(), vg, ws, max(ks))
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_ERR_DEVICE_BOUNDS
    b.close()


@pytest.mark.gpu
def test_verify_grouped_two_groups():
    """Two groups over prefixes of different lengths (512 and 256 tokens) and
    ungrouped requests: every draft row against the fp64 tree oracle."""
    from paper_2605_11232_gb300 import batch as B
    from paper_2605_11232_gb300.workloads import make_workload
    need_gpu()
    rng = np.random.default_rng(9)
    R = 10
    ks = [3, 8, 1, 16, 5, 64, 2, 9, 12, 4]
    grp = [0, 1, -1, 0, 1, 0, 1, -1, 0, 1]
    plen = [512, 256]
    cached = [int(rng.integers(1, 20 * 16)) + (plen[g0] if g0 >= 0 else 0) for g0 in grp]
    w = make_workload("custom", seed=9, custom=dict(
        Hq=32, Hkv=8, d=128, prefix_lens=plen, group=grp, cached=cached, new=ks, decode=[False] * R))
    parents = [_random_parents(rng, k) for k in ks]
    cu = np.concatenate([[0], np.cumsum(ks)]).astype(np.int32)
    masks = pkv.pkv_tree_masks(np.concatenate(parents).astype(np.int32), cu)
    b = B.build_batch(w, poison=True)
    B.run_write(b)
    T = int(cu[-1])
    vg, keep = B.verify_groups(b)
    ws = B.verify_workspace(b, vg)
    out = torch.full((T, 32, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full((T, 32), float("nan"), dtype=torch.float32, device="cuda")
    B.run_verify_grouped(b, out, lse, torch.from_numpy(masks).cuda(), vg, ws, max(ks))
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    errs, lerrs = [], []
    for r in range(R):
        kr, vr = w.request_kv(r)
        o_ref, l_ref = TV.tree_verify_attention(_bits(w.request_q(r)), _bits(kr), _bits(vr), parents[r], w.scale)
        a, e = int(cu[r]), int(cu[r + 1])
        errs.append(np.abs(out[a:e].float().cpu().numpy().astype(np.float64) - o_ref).ravel())
        lerrs.append(np.abs(lse[a:e].cpu().numpy().astype(np.float64) - l_ref).ravel())
    err, lerr = np.concatenate(errs), np.concatenate(lerrs)
    assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS and lerr.max() <= LSE_ABS
    b.close()


@pytest.mark.gpu
def test_verify_grouped_token_count_below_cu_seqlens_stays_in_workspace():
    """A num_tokens smaller than cu_seqlens_q[R] (the workspace sized for it):
    the rows past it latch DEVICE_BOUNDS and nothing is written past the
    workspace (a canary after it keeps its bytes)."""
    from paper_2605_11232_gb300 import batch as B
    need_gpu()
    w, b, parents, cu, masks, ks = _tree_batch(128, 32, 8, 4)
    vg, keep = B.verify_groups(b)
    T = int(cu[-1])
    T_small = int(cu[len(ks) // 2])          # half the requests' tokens
    need = pkv.paged_attn_verify_tree_workspace_size(b.pool, T_small, 32, b.table.shape[1], vg)
    buf = torch.full((need + (1 << 20),), 0x5A, dtype=torch.uint8, device="cuda")
    out = torch.empty((T, 32, 128), dtype=torch.bfloat16, device="cuda")
    m = torch.from_numpy(masks).cuda()
    pkv.paged_attn_verify_tree_grouped(b.pool, b.q[:T_small], out[:T_small], None, b.cu_pre, b.context_lens,
                                       b.table, max(ks), w.scale, m, vg, buf[:need])
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_ERR_DEVICE_BOUNDS
    assert bool((buf[need:] == 0x5A).all())
    b.close()
