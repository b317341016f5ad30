"""paged_attn_decode against the fp64 oracle (GPU).

Tolerance: max |out - oracle| <= 1e-2 and mean <= 1e-3 over all elements of a
run (bf16 inputs, fp32 accumulation, bf16 output); LSE within 1e-3.
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


def run_decode(b, use_groups=False, with_lse=True):
    w = b.w
    Rd = b.dec.stop - b.dec.start
    B.run_write(b)
    out = torch.empty((Rd, w.num_q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((Rd, w.num_q_heads), dtype=torch.float32, device="cuda") if with_lse else None
    ws = B.decode_workspace(b, use_groups)
    B.run_decode(b, out, lse, ws, use_groups)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    return out, lse


def run_decode_append(b, use_groups=False, with_lse=True):
    """The decode subset's cache write and attention in one call
    (paged_attn_decode_append); the prefill subset's new tokens, if any, by
    kv_cache_write, so the pool ends as after run_decode."""
    w = b.w
    Rd = b.dec.stop - b.dec.start
    rows_p = B.new_token_rows(w, b.pre)
    if rows_p.stop > rows_p.start:
        pkv.kv_cache_write(b.pool, b.k_new[rows_p], b.v_new[rows_p], b.slots[rows_p])
    out = torch.empty((Rd, w.num_q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((Rd, w.num_q_heads), dtype=torch.float32, device="cuda") if with_lse else None
    ws = B.decode_workspace(b, use_groups)
    B.run_decode_append(b, out, lse, ws, use_groups)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    return out, lse


def _bits(t):
    return t.view(torch.int16)


def compare(b, out, lse, reqs, threads=8):
    w = b.w
    errs, lerrs = [], []
    for r in reqs:
        o_ref, l_ref = oracle.request_attention(w, int(r), threads=threads)
        i = int(r) - b.dec.start
        errs.append(np.abs(_f64(out[i]) - o_ref[0]))
        if lse is not None:
            lerrs.append(np.abs(_f64(lse[i]) - l_ref[0]))
    e = np.concatenate([x.ravel() for x in errs])
    assert np.isfinite(e).all()
    assert e.max() <= MAX_ABS and e.mean() <= MEAN_ABS, (e.max(), e.mean())
    if lerrs:
        le = np.concatenate(lerrs)
        assert le.max() <= LSE_ABS, le.max()
    return e.max(), e.mean()


@pytest.mark.parametrize("groups", [False, True])
@pytest.mark.parametrize("name,scale", [
    ("tiny_decode", 1.0),
    ("l8b_decode", 0.25),     # 16 requests of full length
    ("qwen_mixed", 0.125),    # 32 decode requests over three prefixes, g = 7
    ("l70b_decode", 1 / 32),  # 16 requests, log-uniform suffixes, g = 8
])
def test_decode_matches_oracle(name, scale, groups):
    """groups=True: shared prefix blocks through the grouped prefix pass
    (tcgen05) + private split pass + combine; False: split pass over all."""
    need_gpu()
    w = make_workload(name, scale_requests=scale)
    b = B.build_batch(w, poison=True)
    out, lse = run_decode(b, use_groups=groups)
    compare(b, out, lse, range(b.dec.start, b.dec.stop))
    b.close()


@pytest.mark.parametrize("groups", [True, False])
@pytest.mark.parametrize("name", ["l8b_decode", "qwen_mixed", "l70b_decode"])
def test_decode_full_size_every_request(name, groups):
    """Full-size batch in the benchmark's launch configuration (the fused
    cache write + decode call; groups=True: with the shared-prefix pass):
    every request's outputs and LSE against the oracle, no NaN anywhere."""
    need_gpu()
    w = make_workload(name)
    b = B.build_batch(w, poison=True)
    out, lse = run_decode_append(b, use_groups=groups)
    assert torch.isfinite(out.float()).all()
    compare(b, out, lse, range(b.dec.start, b.dec.stop), threads=16)
    b.close()


@pytest.mark.parametrize("groups", [False, True])
@pytest.mark.parametrize("name,scale", [
    ("tiny_decode", 1.0),
    ("l8b_decode", 0.25),
    ("qwen_mixed", 0.125),
    ("l70b_decode", 1 / 32),
])
def test_decode_append_equals_write_then_decode(name, scale, groups):
    """paged_attn_decode_append stores each query token's K/V from inside the
    decode kernels: its outputs and LSE have the bits of kv_cache_write +
    paged_attn_decode, and the whole pool afterwards is bit-identical to
    theirs (NaN-poisoned unused slots included)."""
    need_gpu()
    w = make_workload(name, scale_requests=scale)
    b1 = B.build_batch(w, poison=True)
    o1, l1 = run_decode(b1, use_groups=groups)
    k1, v1 = b1.k_cache.clone(), b1.v_cache.clone()
    b1.close()
    b2 = B.build_batch(w, poison=True)
    before = _bits(b2.k_cache).clone()
    o2, l2 = run_decode_append(b2, use_groups=groups)
    assert torch.equal(o1, o2) and torch.equal(l1, l2)
    assert torch.equal(_bits(k1), _bits(b2.k_cache)) and torch.equal(_bits(v1), _bits(b2.v_cache))
    assert not torch.equal(before, _bits(b2.k_cache))   # the call did write the new rows
    compare(b2, o2, l2, range(b2.dec.start, b2.dec.stop))
    b2.close()


def test_two_pools_two_threads_concurrently():
    """Two pools on one GPU, each decoded from its own host thread on its own
    stream, ten times each, concurrently: every output has the bits of the
    same decode run alone (launch attributes and pool state are per device and
    per pool, and safe to set up from several threads)."""
    need_gpu()
    import threading
    ws_, refs, bs = [], [], []
    for name, scale in (("l8b_decode", 0.125), ("qwen_mixed", 0.0625)):
        w = make_workload(name, scale_requests=scale)
        b = B.build_batch(w, poison=True)
        ref, _ = run_decode(b, use_groups=True)
        bs.append(b)
        refs.append(ref)
        ws_.append(B.decode_workspace(b, True))
    outs = [[torch.empty_like(r) for _ in range(10)] for r in refs]
    errors = []

    def worker(i):
        try:
            s = torch.cuda.Stream()
            with torch.cuda.stream(s):
                for k in range(10):
                    B.run_decode(bs[i], outs[i][k], None, ws_[i], True, stream=s)
            s.synchronize()
        except Exception as e:   # reported below
            errors.append(e)

    threads = [threading.Thread(target=worker, args=(i,)) for i in range(2)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    torch.cuda.synchronize()
    assert not errors, errors
    for i in range(2):
        assert pkv.pkv_check_device_errors(bs[i].pool) == pkv.PKV_OK
        for o in outs[i]:
            assert torch.equal(o, refs[i])
        bs[i].close()


def test_checked_table_then_decode_without_device_errors():
    """A batch whose rows share refcounted prefix blocks passes the host check
    of its block tables, and its decode then latches no device error."""
    need_gpu()
    w = make_workload("l8b_decode", scale_requests=0.125)
    b = B.build_batch(w, poison=True)
    rows = b.table_host[b.dec]
    assert max(pkv.kv_pool_refcount(b.pool, int(x)) for x in rows[0, :16]) > 1
    pkv.pkv_check_block_table(b.pool, rows, w.context_lens[b.dec].astype(np.int32))
    out, lse = run_decode(b, use_groups=True)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    b.close()


@pytest.mark.parametrize("groups", [False, True])
def test_placement_invariance_bit_exact(groups):
    """Different physical placements of the same logical cache give
    bit-identical outputs (the reduction order depends on positions only)."""
    need_gpu()
    w = make_workload("l8b_decode", scale_requests=0.125)
    outs = []
    for seed in (0, 7, 123456789):
        b = B.build_batch(w, poison=True, placement_seed=seed)
        o, l = run_decode(b, use_groups=groups)
        outs.append((o.cpu(), l.cpu()))
        b.close()
    for o, l in outs[1:]:
        assert torch.equal(o, outs[0][0]) and torch.equal(l, outs[0][1])


def test_shared_prefix_equals_private_copies():
    """Reading the prefix through shared refcounted blocks or through private
    copies gives the same outputs (without the grouped prefix pass: bit-exact)."""
    need_gpu()
    w = make_workload("qwen_mixed", scale_requests=0.0625)
    b1 = B.build_batch(w, poison=True)
    o1, l1 = run_decode(b1)
    b2 = B.build_batch(w, poison=True, share_prefix=False)
    o2, l2 = run_decode(b2)
    assert torch.equal(o1, o2) and torch.equal(l1, l2)
    # the grouped prefix pass reads the shared blocks once per group: same
    # result up to summation order
    o3, l3 = run_decode(b1, use_groups=True)
    assert (o3.float() - o2.float()).abs().max().item() <= 2 * MAX_ABS / 2
    assert (l3 - l2).abs().max().item() <= LSE_ABS
    b1.close(); b2.close()


def test_grouped_members_need_not_be_contiguous():
    """Group membership is a list: interleaved members of two groups."""
    need_gpu()
    R = 12
    group = [i % 2 for i in range(R)]
    w = make_workload("custom", custom=dict(Hq=16, Hkv=2, d=128, prefix_lens=[512, 1024],
                                          group=group, cached=[(512 if g == 0 else 1024) + 40 + 7 * i
                                                               for i, g in enumerate(group)],
                                          new=[1] * R, decode=[True] * R))
    b = B.build_batch(w, poison=True)
    out, lse = run_decode(b, use_groups=True)
    compare(b, out, lse, range(R))
    b.close()


@pytest.mark.parametrize("append,d", [(False, 128), (True, 128), (False, 64)])
def test_prefix_pass_larger_than_the_device(append, d):
    """40 groups of 3 members over 8 kv heads: 320 shared-prefix CTAs (one key
    split each), three waves on a 152-SM device, so the split pass (launched
    once every prefix CTA has started, on all SMs) takes SMs only as
    last-wave prefix CTAs exit.  Ragged prefixes (768-1024 tokens) and 8 requests outside any
    group; every request against the oracle."""
    need_gpu()
    G, M = 40, 3
    prefix_lens = [1024 - 64 * (g % 5) for g in range(G)]
    group = [g for g in range(G) for _ in range(M)] + [-1] * 8
    cached = [(prefix_lens[g] if g >= 0 else 0) + 1 + (37 * i) % 300 for i, g in enumerate(group)]
    R = len(group)
    w = make_workload("custom", custom=dict(Hq=32, Hkv=8, d=d, prefix_lens=prefix_lens, group=group,
                                          cached=cached, new=[1] * R, decode=[True] * R))
    b = B.build_batch(w, poison=True)
    out, lse = (run_decode_append if append else run_decode)(b, use_groups=True)
    assert torch.isfinite(out.float()).all()
    compare(b, out, lse, range(R), threads=16)
    b.close()


@pytest.mark.parametrize("groups", [False, True])
@pytest.mark.parametrize("g,d", [(1, 128), (2, 64), (3, 128), (5, 64), (6, 128)])
def test_decode_uncommon_head_ratios(g, d, groups):
    """GQA ratios the benchmark's models do not use (MHA included): the split
    pass's 4- and 8-row Q areas and the combine's head groups with columns
    left unused.  Two shared prefixes, ragged private tails, requests outside
    any group; every request against the oracle."""
    need_gpu()
    Hkv = 2
    R = 14
    group = [0, 0, 0, 0, 1, 1, 1, 1, 1, -1, -1, 0, 1, -1]
    prefix_lens = [256, 512]
    cached = [(prefix_lens[gi] if gi >= 0 else 0) + 1 + (53 * i) % 400 for i, gi in enumerate(group)]
    w = make_workload("custom", seed=7 + g, custom=dict(Hq=g * Hkv, Hkv=Hkv, d=d, prefix_lens=prefix_lens,
                                                      group=group, cached=cached, new=[1] * R,
                                                      decode=[True] * R))
    b = B.build_batch(w, poison=True)
    out, lse = run_decode(b, use_groups=groups)
    compare(b, out, lse, range(R))
    b.close()


def test_single_key_returns_value():
    """A context of one token returns that token's V (weight exactly 1)."""
    need_gpu()
    w = make_workload("custom", custom=dict(Hq=8, Hkv=2, d=128, prefix_lens=[], group=[-1, -1, -1],
                                          cached=[0, 0, 0], new=[1, 1, 1], decode=[True] * 3,
                                          num_blocks=8))
    b = B.build_batch(w, poison=True)
    out, lse = run_decode(b)
    v = w.new_v.float()
    for r in range(3):
        for h in range(8):
            assert torch.equal(out[r, h].cpu().float(), v[r, h // 4])
    b.close()


def test_causality_future_slots_ignored():
    """Keys past the context (rest of the last block) never matter: the result
    is identical whatever those slots hold."""
    need_gpu()
    w = make_workload("l8b_decode", scale_requests=0.0625)
    b = B.build_batch(w, poison=False)
    o1, l1 = run_decode(b)
    # overwrite every slot past each request's context inside its last block
    for r in range(w.num_requests):
        L = int(w.context_lens[r])
        blk = int(b.table_host[r, (L - 1) // 16])
        b.k_cache[blk, :, L % 16 or 16:, :] = 1000.0
        b.v_cache[blk, :, L % 16 or 16:, :] = float("inf")
    ws = B.decode_workspace(b, False)
    o2 = torch.empty_like(o1)
    l2 = torch.empty_like(l1)
    B.run_decode(b, o2, l2, ws, False)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    assert torch.equal(o1, o2) and torch.equal(l1, l2)
    b.close()


def test_bad_arguments_rejected_before_launch():
    need_gpu()
    w = make_workload("tiny_decode")
    b = B.build_batch(w)
    out = torch.empty((4, 8, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(pkv.PkvError) as e:
        B.run_decode(b, out, None, torch.empty(16, dtype=torch.uint8, device="cuda"), False)
    assert e.value.code == pkv.PKV_ERR_WORKSPACE
    b.close()


@pytest.mark.parametrize("groups", [False, True])
def test_decode_short_and_ragged_segments(groups):
    """96 requests whose private parts are 1 to 40 blocks (many chunks far
    shorter than the streaming warps of a CTA, and ragged last blocks), over
    one shared 256-token prefix and without one: every output against the
    oracle, no device error."""
    need_gpu()
    rng = np.random.default_rng(3)
    R = 96
    priv = rng.integers(1, 41 * 16, R)
    grp = [0 if i % 3 else -1 for i in range(R)]
    cached = [int(p) - 1 + (256 if g0 == 0 else 0) for p, g0 in zip(priv, grp)]
    w = make_workload("custom", seed=17, custom=dict(
        Hq=16, Hkv=2, d=128, prefix_lens=[256], group=grp, cached=cached, new=[1] * R,
        decode=[True] * R))
    b = B.build_batch(w, poison=True)
    out, lse = run_decode(b, use_groups=groups)
    compare(b, out, lse, range(b.dec.start, b.dec.stop), threads=16)
    b.close()


@pytest.mark.parametrize("fused", [False, True])
@pytest.mark.parametrize("groups", [False, True])
def test_decode_step_from_host_buffers_bit_exact(groups, fused):
    """paged_attn_decode_step (one H2D copy of the packed inputs, cache write,
    decode, D2H copy of the output; fused: the decode kernels store the new
    tokens) gives the bits of kv_cache_write + paged_attn_decode on device
    inputs, on two steps in a row."""
    need_gpu()
    w = make_workload("l8b_decode", scale_requests=0.25)
    b = B.build_batch(w, poison=True)
    ref, ref_lse = run_decode(b, use_groups=groups)
    layout, hosts, dev = B.step_buffers(b, copies=1, fused=fused)
    R = b.dec.stop - b.dec.start
    ws = B.decode_workspace(b, groups)
    out = torch.empty_like(ref)
    lse = torch.empty_like(ref_lse)
    host_out = torch.full(tuple(ref.shape), float("nan"), dtype=torch.bfloat16).pin_memory()
    host_lse = torch.full((R, w.num_q_heads), float("nan"), dtype=torch.float32).pin_memory()
    step = pkv.DecodeStep(b.pool, hosts[0], dev, layout, w.num_new_tokens, b.table[b.dec],
                          w.num_q_heads, w.scale, b.groups if groups else None, ws, out, lse,
                          host_out, host_lse)
    for _ in range(2):
        host_out.fill_(float("nan"))
        step()
        torch.cuda.synchronize()
        assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
        assert torch.equal(host_out, ref.cpu()) and torch.equal(host_lse, ref_lse.cpu())
    # a misaligned region, or a decode argument error, is refused before
    # anything is enqueued: the device input buffer keeps its contents
    dev.fill_(0xAB)
    torch.cuda.synchronize()
    bad = pkv.StepLayout(q=layout.q, k_new=layout.k_new + 8, v_new=layout.v_new,
                         slot_mapping=layout.slot_mapping, context_lens=layout.context_lens,
                         bytes=layout.bytes, flags=layout.flags)
    with pytest.raises(pkv.PkvError) as e:
        pkv.paged_attn_decode_step(b.pool, hosts[0], dev, bad, w.num_new_tokens, b.table[b.dec],
                                   w.num_q_heads, w.scale, None, ws, out)
    assert e.value.code == pkv.PKV_ERR_INVALID_ARG
    out_more_heads = torch.empty((R, w.num_q_heads + 1, w.head_dim), dtype=torch.bfloat16,
                                 device="cuda")
    with pytest.raises(pkv.PkvError) as e:
        pkv.paged_attn_decode_step(b.pool, hosts[0], dev, layout, w.num_new_tokens, b.table[b.dec],
                                   w.num_q_heads + 1, w.scale, None, ws, out_more_heads)
    assert e.value.code == pkv.PKV_ERR_INVALID_ARG
    torch.cuda.synchronize()
    assert bool((dev == 0xAB).all())
    b.close()


def test_decode_step_two_streams_alternating():
    """Alternate steps on two streams, each with its own device input and
    output buffers, each step's kernels waiting for the previous step's
    done_event: every step's host output has the device path's bits."""
    need_gpu()
    w = make_workload("l8b_decode", scale_requests=0.25)
    b = B.build_batch(w, poison=True)
    ref, _ = run_decode(b, use_groups=True)
    layout, hosts, _ = B.step_buffers(b, copies=2)
    ws = B.decode_workspace(b, True)
    devs = [torch.empty(layout.bytes, dtype=torch.uint8, device="cuda") for _ in range(2)]
    outs = [torch.empty_like(ref) for _ in range(2)]
    streams = [torch.cuda.Stream() for _ in range(2)]
    done = [torch.cuda.Event() for _ in range(2)]
    host_outs = [torch.empty(tuple(ref.shape), dtype=torch.bfloat16).pin_memory() for _ in range(4)]
    for i in range(4):
        k = i & 1
        pkv.paged_attn_decode_step(b.pool, hosts[k], devs[k], layout, w.num_new_tokens,
                                   b.table[b.dec], w.num_q_heads, w.scale, b.groups, ws, outs[k],
                                   host_out=host_outs[i], wait_event=done[1 - k],
                                   done_event=done[k], stream=streams[k])
    torch.cuda.synchronize()
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    for h in host_outs:
        assert torch.equal(h, ref.cpu())
    b.close()


def test_decode_largest_batch():
    """The largest decode batch the entry point takes (16384 requests), with
    short ragged contexts (1 to 40 tokens), d = 64, g = 4: every output
    against the oracle.  With so few keys an output is an average of a few
    N(0, 1) rows and reaches |o| of 3 to 4 over 8.4M outputs, where half an
    ulp of the bf16 output alone is up to 1.6e-2: the bound per element is
    1e-2 + 2^-8 |o| (bf16 rounding of the output and of the weights, 2^-9
    relative each); the mean bound stays 1e-3."""
    need_gpu()
    rng = np.random.default_rng(4)
    R = 16384
    w = make_workload("custom", seed=4, custom=dict(
        Hq=8, Hkv=2, d=64, prefix_lens=[], group=[-1] * R, cached=rng.integers(0, 40, R).tolist(),
        new=[1] * R, decode=[True] * R))
    b = B.build_batch(w, poison=True)
    out, lse = run_decode(b)
    got, lgot = _f64(out), _f64(lse)
    errs, excess, lerrs = [], [], []
    for r in range(R):
        o_ref, l_ref = oracle.request_attention(w, r, threads=16)
        e = np.abs(got[r] - o_ref[0])
        errs.append(e.ravel())
        excess.append((e - (MAX_ABS + 2.0 ** -8 * np.abs(o_ref[0]))).max())
        lerrs.append(np.abs(lgot[r] - l_ref[0]).max())
    e = np.concatenate(errs)
    assert np.isfinite(e).all() and e.mean() <= MEAN_ABS, e.mean()
    assert max(excess) <= 0, max(excess)
    assert max(lerrs) <= LSE_ABS, max(lerrs)
    b.close()
