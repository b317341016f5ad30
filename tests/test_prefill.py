"""paged_attn_prefill against the fp64 oracle (GPU).

Suffix (or chunk) tokens attend to the whole cached context (shared prefix
included) and causally to the new tokens.  Tolerance as for decode: max abs
1e-2, mean abs 1e-3 over the compared elements; LSE within 1e-3.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2605_11232_gb300 import batch as B
from paper_2605_11232_gb300 import pkv
from paper_2605_11232_gb300.workloads import make_workload

from _lib import need_gpu

pytestmark = pytest.mark.gpu

MAX_ABS, MEAN_ABS, LSE_ABS = 1e-2, 1e-3, 1e-3


def _f64(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def run_prefill(b, with_lse=True):
    w = b.w
    rows = B.new_token_rows(w, b.pre)
    n = rows.stop - rows.start
    B.run_write(b)
    out = torch.full((n, w.num_q_heads, w.head_dim), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full((n, w.num_q_heads), float("nan"), dtype=torch.float32, device="cuda") if with_lse else None
    B.run_prefill(b, out, lse)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    return out, lse


def run_prefill_append(b, with_lse=True):
    """The prefill subset's write and attention in one call; the decode
    subset's new tokens (if any) by kv_cache_write, so the pool ends as after
    run_prefill."""
    w = b.w
    rows = B.new_token_rows(w, b.pre)
    rows_d = B.new_token_rows(w, b.dec)
    if rows_d.stop > rows_d.start:
        pkv.kv_cache_write(b.pool, b.k_new[rows_d], b.v_new[rows_d], b.slots[rows_d])
    n = rows.stop - rows.start
    out = torch.full((n, w.num_q_heads, w.head_dim), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full((n, w.num_q_heads), float("nan"), dtype=torch.float32, device="cuda") if with_lse else None
    B.run_prefill_append(b, out, lse)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    return out, lse


def _bits(t):
    return t.view(torch.int16)


def compare(b, out, lse, reqs, rows_per_req=None, threads=16, seed=0):
    """Compare every (or a sample of) query rows of the given requests."""
    w = b.w
    rng = np.random.default_rng(seed)
    base = int(w.cu_new[b.pre.start])
    errs, lerrs = [], []
    for r in reqs:
        S = int(w.new_lens[r])
        if rows_per_req is None or rows_per_req >= S:
            sel = list(range(S))
            ref_o, ref_l = oracle.request_attention(w, r, threads=threads)
        else:
            sel = sorted({0, S - 1, *rng.choice(S, rows_per_req - 2, replace=False).tolist()})
            ref_o, ref_l = oracle.request_attention(w, r, threads=threads, rows=sel)
        off = int(w.cu_new[r]) - base
        got = _f64(out[[off + i for i in sel]])
        errs.append(np.abs(got - ref_o).ravel())
        if lse is not None:
            lerrs.append(np.abs(_f64(lse[[off + i for i in sel]]) - ref_l).ravel())
    e = np.concatenate(errs)
    assert np.isfinite(e).all()
    assert e.max() <= MAX_ABS and e.mean() <= MEAN_ABS, (e.max(), e.mean())
    if lerrs:
        le = np.concatenate(lerrs)
        assert le.max() <= LSE_ABS, le.max()


def test_tiny_prefill_all_rows():
    """d = 64, g = 4: 4 suffixes (32/48/64/96) over a shared 256-token prefix."""
    need_gpu()
    w = make_workload("tiny")
    b = B.build_batch(w, poison=True)
    out, lse = run_prefill(b)
    compare(b, out, lse, range(w.num_requests))
    b.close()


@pytest.mark.parametrize("Hq,Hkv,d,ctx,new", [
    (8, 2, 128, [1, 17, 130, 300], [1, 17, 130, 100]),      # no prefix, causal from 0
    (7, 1, 128, [40, 257], [40, 129]),                        # g = 7: 18 tokens per tile
    (64, 8, 128, [200, 33], [50, 33]),                        # g = 8: 16 tokens per tile
    (4, 4, 64, [70, 500], [3, 250]),                          # g = 1 (MHA), d = 64
    (16, 1, 128, [129, 128], [129, 1]),                       # g = 16
])
def test_prefill_shapes_all_rows(Hq, Hkv, d, ctx, new):
    need_gpu()
    R = len(ctx)
    w = make_workload("custom", custom=dict(Hq=Hq, Hkv=Hkv, d=d, prefix_lens=[], group=[-1] * R,
                                          cached=[c - n for c, n in zip(ctx, new)], new=new,
                                          decode=[False] * R))
    b = B.build_batch(w, poison=True)
    out, lse = run_prefill(b)
    compare(b, out, lse, range(R))
    b.close()


def test_l8b_prefill_scaled_sampled_rows():
    """4 requests of the Llama-3-8B suffix-prefill workload (full 4096 prefix)."""
    need_gpu()
    w = make_workload("l8b_prefill", scale_requests=0.125)
    b = B.build_batch(w, poison=True)
    out, lse = run_prefill(b)
    compare(b, out, lse, range(w.num_requests), rows_per_req=24)
    b.close()


@pytest.mark.parametrize("name", ["l8b_prefill", "qwen_mixed"])
def test_prefill_full_size_every_row(name):
    """Full-size batch (the benchmark's call): every query row of 8 requests
    (the first, the last, the middle, the longest cached context and random
    ones; qwen_mixed has exactly 8) against the oracle, and no NaN anywhere in
    the output."""
    need_gpu()
    w = make_workload(name)
    b = B.build_batch(w, poison=True)
    out, lse = run_prefill_append(b)   # the benchmark's call: write fused into the prefill
    assert torch.isfinite(out.float()).all() and torch.isfinite(lse).all()
    reqs = list(range(b.pre.start, b.pre.stop))
    pick = {reqs[0], reqs[-1], reqs[len(reqs) // 2], reqs[int(np.argmax(w.cached_lens[b.pre]))]}
    rng = np.random.default_rng(5)
    while len(pick) < min(8, len(reqs)):
        pick.add(int(rng.choice(reqs)))
    compare(b, out, lse, sorted(pick))
    b.close()


@pytest.mark.parametrize("name,scale", [("tiny", 1.0), ("l8b_prefill", 0.125), ("qwen_mixed", 0.125)])
def test_prefill_append_equals_write_then_prefill(name, scale):
    """paged_attn_prefill_append reads the new keys from k_new / v_new and
    stores them from inside the prefill kernel: its outputs and LSE have the
    bits of kv_cache_write + paged_attn_prefill, and the whole pool afterwards
    (NaN-poisoned unused slots included) is bit-identical to theirs."""
    need_gpu()
    w = make_workload(name, scale_requests=scale)
    b1 = B.build_batch(w, poison=True)
    o1, l1 = run_prefill(b1)
    k1, v1 = b1.k_cache.clone(), b1.v_cache.clone()
    b1.close()
    b2 = B.build_batch(w, poison=True)
    o2, l2 = run_prefill_append(b2)
    assert torch.equal(o1, o2) and torch.equal(l1, l2)
    assert torch.equal(_bits(k1), _bits(b2.k_cache)) and torch.equal(_bits(v1), _bits(b2.v_cache))
    compare(b2, o2, l2, range(b2.pre.start, b2.pre.stop), rows_per_req=16)
    b2.close()


def test_prefill_append_needs_block_aligned_cache():
    """A request whose cached part is not whole blocks is skipped (output
    untouched) and latches DEVICE_BOUNDS; the aligned one beside it is
    computed and stored."""
    need_gpu()
    w = make_workload("custom", seed=41, custom=dict(Hq=8, Hkv=2, d=128, prefix_lens=[], group=[-1, -1],
                                                   cached=[64, 100], new=[40, 30], decode=[False, False]))
    b = B.build_batch(w, poison=True)
    n = w.num_new_tokens
    out = torch.full((n, 8, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
    B.run_prefill_append(b, out, None)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_ERR_DEVICE_BOUNDS
    assert bool(torch.isnan(out[40:].float()).all())
    compare(b, out, None, [0])
    b.close()


def test_prefill_context_shorter_than_its_new_tokens_latches_bounds():
    """A request whose context length (a device array) is below its own
    new-token count is refused on the device.  In the longest-first order of
    a short grid its items are still given CTAs, so the error is latched
    rather than the rows skipped unnoticed; the other requests are computed."""
    need_gpu()
    w = make_workload("custom", seed=43, custom=dict(Hq=8, Hkv=2, d=128, prefix_lens=[], group=[-1] * 3,
                                                   cached=[64, 80, 96], new=[40, 30, 20], decode=[False] * 3))
    b = B.build_batch(w, poison=True)
    B.run_write(b)
    out = torch.full((w.num_new_tokens, 8, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
    b.context_lens[1] = 0                               # request 1: no context for its 30 new tokens
    B.run_prefill(b, out, None)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_ERR_DEVICE_BOUNDS
    assert bool(torch.isnan(out[40:70].float()).all())
    compare(b, out, None, [0, 2])
    b.close()


def test_prefill_refuses_tables_wider_than_its_limit():
    """A work item's block ids are staged in shared memory, 2048 of them at
    most: a table wider than that is refused on the host (UNSUPPORTED) before
    any launch."""
    need_gpu()
    w = make_workload("tiny")
    b = B.build_batch(w, poison=True)
    rows = B.new_token_rows(w, b.pre)
    wide = torch.full((b.pre.stop - b.pre.start, 2049), -1, dtype=torch.int32, device="cuda")
    wide[:, : b.table.shape[1]] = b.table[b.pre]
    out = torch.empty((rows.stop - rows.start, w.num_q_heads, w.head_dim), dtype=torch.bfloat16,
                      device="cuda")
    with pytest.raises(pkv.PkvError) as e:
        pkv.paged_attn_prefill(b.pool, b.q[rows], out, None, b.cu_pre, b.context_lens[b.pre], wide,
                               b.max_seqlen_pre, w.scale)
    assert e.value.code == pkv.PKV_ERR_UNSUPPORTED
    # 2048 columns are accepted
    pkv.paged_attn_prefill(b.pool, b.q[rows], out, None, b.cu_pre, b.context_lens[b.pre],
                           wide[:, :2048].contiguous(), b.max_seqlen_pre, w.scale)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    b.close()


def test_prefill_last_row_equals_decode():
    """The last prefill row of a request attends to exactly what a decode query
    at that position attends to: the two kernels agree within tolerance."""
    need_gpu()
    w = make_workload("tiny")
    b = B.build_batch(w, poison=True)
    out, lse = run_prefill(b)
    wd = make_workload("custom", seed=w.seed, custom=dict(
        Hq=8, Hkv=2, d=64, prefix_lens=[256], group=[0] * 4,
        cached=list(w.cached_lens + w.new_lens - 1), new=[1] * 4, decode=[True] * 4, num_blocks=64))
    # same K/V and query rows as the prefill batch's last tokens
    wd.prefix_k, wd.prefix_v = w.prefix_k, w.prefix_v
    parts_k, parts_v, q = [], [], []
    for r in range(4):
        a, e = int(w.cu_new[r]), int(w.cu_new[r + 1])
        parts_k.append(torch.cat([w.priv_k[w.priv_off[r]:w.priv_off[r + 1]], w.new_k[a:e - 1]]))
        parts_v.append(torch.cat([w.priv_v[w.priv_off[r]:w.priv_off[r + 1]], w.new_v[a:e - 1]]))
        q.append(w.q[e - 1:e])
    wd.priv_k, wd.priv_v = torch.cat(parts_k), torch.cat(parts_v)
    wd.priv_off = np.concatenate([[0], np.cumsum([len(x) for x in parts_k])])
    wd.new_k = torch.cat([w.new_k[int(w.cu_new[r + 1]) - 1:int(w.cu_new[r + 1])] for r in range(4)])
    wd.new_v = torch.cat([w.new_v[int(w.cu_new[r + 1]) - 1:int(w.cu_new[r + 1])] for r in range(4)])
    wd.q = torch.cat(q)
    bd = B.build_batch(wd, poison=True)
    B.run_write(bd)
    od = torch.empty((4, 8, 64), dtype=torch.bfloat16, device="cuda")
    ws = B.decode_workspace(bd, False)
    B.run_decode(bd, od, None, ws, False)
    last = [int(w.cu_new[r + 1]) - 1 for r in range(4)]
    diff = (out[last].float() - od.float()).abs()
    assert diff.max().item() <= 2e-2
    b.close(); bd.close()


def test_prefill_placement_invariance_bit_exact():
    need_gpu()
    w = make_workload("l8b_prefill", scale_requests=0.0625)
    outs = []
    for seed in (0, 99):
        b = B.build_batch(w, poison=True, placement_seed=seed)
        o, l = run_prefill(b)
        outs.append((o.cpu(), l.cpu()))
        b.close()
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])


def test_prefill_causality_future_keys_ignored():
    """Changing the K/V of the last new token changes no earlier row."""
    need_gpu()
    w = make_workload("tiny")
    b = B.build_batch(w, poison=True)
    o1, l1 = run_prefill(b)
    for r in range(w.num_requests):
        t = int(w.cu_new[r + 1]) - 1
        b.k_new[t] = 50.0
        b.v_new[t] = -7.0
    o2, l2 = run_prefill(b)
    for r in range(w.num_requests):
        a, e = int(w.cu_new[r]), int(w.cu_new[r + 1])
        assert torch.equal(o1[a:e - 1], o2[a:e - 1]) and torch.equal(l1[a:e - 1], l2[a:e - 1])
        assert not torch.equal(o1[e - 1], o2[e - 1])
    b.close()


def test_speculative_verify_chain_drafts():
    """Verification of k = 2..8 chain draft tokens per request (each draft
    attends to the whole context and to the drafts before it) is a suffix
    prefill with S = k: 16 requests, 12 of them over one shared 512-token
    prefix, ragged private contexts; every row against the oracle."""
    need_gpu()
    rng = np.random.default_rng(8)
    R = 16
    k = [2 + (i % 7) for i in range(R)]
    grp = [0 if i % 4 else -1 for i in range(R)]
    cached = [int(rng.integers(1, 40 * 16)) + (512 if g0 == 0 else 0) for g0 in grp]
    w = make_workload("custom", seed=9, custom=dict(
        Hq=32, Hkv=8, d=128, prefix_lens=[512], group=grp, cached=cached, new=k,
        decode=[False] * R))
    b = B.build_batch(w, poison=True)
    out, lse = run_prefill(b)
    compare(b, out, lse, range(R))
    b.close()


def test_prefill_longest_item_and_empty_request():
    """A work item at the longest key range one item may span (32,760 cached
    tokens + 4 queries: 2048 blocks), beside a request with no new tokens (it
    reads and writes nothing) and a short one: every row of the two against
    the oracle."""
    need_gpu()
    w = make_workload("custom", seed=3, custom=dict(
        Hq=8, Hkv=1, d=128, prefix_lens=[], group=[-1] * 3, cached=[32760, 10, 500],
        new=[4, 0, 7], decode=[False] * 3))
    b = B.build_batch(w, poison=True)
    out, lse = run_prefill(b)
    compare(b, out, lse, [0, 2])
    b.close()


@pytest.mark.parametrize("R", [32, 33, 70])
def test_prefill_many_requests_longest_first(R):
    """A short grid (a few waves) takes its items longest first over all
    requests; with more than 32 requests the selection walks them in chunks
    of 32.  Ragged suffixes (some empty), ragged cached contexts: every row
    against the oracle."""
    need_gpu()
    rng = np.random.default_rng(R)
    new = [int(x) for x in rng.choice([0, 1, 7, 33, 64, 65, 130, 200], R)]
    cached = [int(x) for x in rng.integers(1, 600, R)]
    w = make_workload("custom", seed=R, custom=dict(Hq=8, Hkv=2, d=64, prefix_lens=[], group=[-1] * R,
                                                   cached=cached, new=new, decode=[False] * R))
    b = B.build_batch(w, poison=True)
    out, lse = run_prefill(b)
    compare(b, out, lse, [r for r in range(R) if new[r] > 0])
    b.close()
