"""Pins of the fp64 oracle against things other than itself (CPU only).

The paper prints no kernel-level worked example (it reports serving-level
numbers only), so the oracle is pinned by: a library routine that computes the
same special case (torch's fp64 scaled-dot-product attention with an explicit
mask), closed forms (single key, zero query, constant values, two keys,
a dominant key), invariances (key shift, key order, block placement) and
brute-force enumeration of the paged layout.  Each check is chosen so that a
plausible slip in the oracle -- a wrong causal offset, a q-head to kv-head
mapping of h % Hkv instead of h / g, a missing scale, a transposed pool layout
-- fails at least one of them.
"""

import math

import numpy as np
import pytest
import torch

import oracle


def _bits(x: np.ndarray) -> np.ndarray:
    """bf16 bit patterns of float values (exactly representable ones)."""
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def _rand_bits(rng, shape):
    return _bits(rng.standard_normal(shape).astype(np.float32))


def _sdpa_reference(qb, kb, vb, scale):
    """torch fp64 SDPA with GQA expanded by repeat_interleave and the causal
    mask of a suffix written out as a boolean matrix."""
    q = torch.from_numpy(oracle.bf16_to_f64(qb))            # [S][Hq][d]
    k = torch.from_numpy(oracle.bf16_to_f64(kb))            # [L][Hkv][d]
    v = torch.from_numpy(oracle.bf16_to_f64(vb))
    S, Hq, d = q.shape
    L, Hkv, _ = k.shape
    g = Hq // Hkv
    k = k.repeat_interleave(g, dim=1)
    v = v.repeat_interleave(g, dim=1)
    mask = torch.zeros((S, L), dtype=torch.bool)
    for i in range(S):
        mask[i, : L - S + i + 1] = True
    out = torch.nn.functional.scaled_dot_product_attention(
        q.permute(1, 0, 2), k.permute(1, 0, 2), v.permute(1, 0, 2),
        attn_mask=mask, scale=scale)
    return out.permute(1, 0, 2).numpy()


@pytest.mark.parametrize("S,L,Hq,Hkv,d", [
    (1, 1, 4, 2, 16),      # single key
    (1, 37, 8, 2, 64),     # decode, g = 4
    (5, 37, 6, 2, 16),     # suffix over a cached prefix
    (16, 16, 7, 1, 32),    # full causal self-attention, g = 7
    (9, 40, 28, 4, 128),   # Qwen-shaped heads, d = 128
    (3, 20, 3, 3, 8),      # MHA, g = 1
])
def test_matches_torch_sdpa(S, L, Hq, Hkv, d):
    rng = np.random.default_rng(S * 1000 + L)
    qb = _rand_bits(rng, (S, Hq, d))
    kb = _rand_bits(rng, (L, Hkv, d))
    vb = _rand_bits(rng, (L, Hkv, d))
    scale = 1.0 / math.sqrt(d)
    out, lse = oracle.attention(qb, kb, vb, scale, threads=2)
    ref = _sdpa_reference(qb, kb, vb, scale)
    assert np.max(np.abs(out - ref)) < 1e-12
    # LSE from its definition via torch's logsumexp on the masked scores
    q = oracle.bf16_to_f64(qb)
    k = np.repeat(oracle.bf16_to_f64(kb), Hq // Hkv, axis=1)
    for i in range(S):
        pos = L - S + i
        s = np.einsum("hd,jhd->hj", q[i], k[: pos + 1]) * scale
        ref_lse = torch.logsumexp(torch.from_numpy(s), dim=1).numpy()
        assert np.max(np.abs(lse[i] - ref_lse)) < 1e-12


def test_single_key_returns_value_exactly():
    rng = np.random.default_rng(1)
    qb = _rand_bits(rng, (1, 4, 64))
    kb = _rand_bits(rng, (1, 2, 64))
    vb = _rand_bits(rng, (1, 2, 64))
    out, lse = oracle.attention(qb, kb, vb, 0.125)
    v = oracle.bf16_to_f64(vb)
    for h in range(4):
        assert np.array_equal(out[0, h], v[0, h // 2])      # weight 1, exactly V
        s = 0.125 * float(oracle.bf16_to_f64(qb)[0, h] @ oracle.bf16_to_f64(kb)[0, h // 2])
        assert lse[0, h] == pytest.approx(s, abs=1e-12)


def test_zero_query_is_mean_of_visible_values():
    """q = 0 gives uniform weights over exactly the visible keys: with
    V[j][0] = j the output is pos / 2 and LSE = ln(pos + 1).  An off-by-one in
    the causal limit or in the suffix offset changes both."""
    S, L, Hq, Hkv, d = 6, 50, 4, 2, 8
    qb = _bits(np.zeros((S, Hq, d)))
    rng = np.random.default_rng(2)
    kb = _rand_bits(rng, (L, Hkv, d))
    v = np.zeros((L, Hkv, d), np.float32)
    v[:, :, 0] = np.arange(L)[:, None]
    v[:, :, 1] = 3.0
    out, lse = oracle.attention(qb, kb, _bits(v), 0.3)
    for i in range(S):
        pos = L - S + i
        assert np.allclose(out[i, :, 0], pos / 2.0, atol=1e-12)
        assert np.allclose(out[i, :, 1], 3.0, atol=1e-12)
        assert np.allclose(lse[i], math.log(pos + 1), atol=1e-12)


def test_gqa_head_mapping_constant_values():
    """V constant per kv head: output of q head h equals the constant of kv head
    h // g (contiguous grouping), not h % Hkv."""
    S, L, Hq, Hkv, d = 2, 9, 8, 2, 16
    rng = np.random.default_rng(3)
    v = np.zeros((L, Hkv, d), np.float32)
    v[:, 0, :] = 1.5
    v[:, 1, :] = -2.25
    out, _ = oracle.attention(_rand_bits(rng, (S, Hq, d)), _rand_bits(rng, (L, Hkv, d)),
                              _bits(v), 0.25)
    for h in range(Hq):
        assert np.allclose(out[:, h, :], 1.5 if h < 4 else -2.25, atol=1e-12)


def test_two_key_closed_form():
    """d = 4 (scale 1/2), q = (2,0,0,0), K0 = 0, K1 = (1,0,0,0): scores 0 and 1,
    so O = (V0 + e V1) / (1 + e) and LSE = ln(1 + e)."""
    q = np.array([[[2, 0, 0, 0]]], np.float32)
    k = np.array([[[0, 0, 0, 0]], [[1, 0, 0, 0]]], np.float32)
    v = np.array([[[1, 2, 3, 4]], [[5, 6, 7, 8]]], np.float32)
    out, lse = oracle.attention(_bits(q), _bits(k), _bits(v), 1.0 / math.sqrt(4))
    e = math.e
    want = (np.array([1, 2, 3, 4]) + e * np.array([5, 6, 7, 8])) / (1 + e)
    assert np.allclose(out[0, 0], want, atol=1e-14)
    assert lse[0, 0] == pytest.approx(math.log(1 + e), abs=1e-14)


def test_dominant_key():
    """One key scoring 50 above all others carries weight 1 - O(e^-50)."""
    L, d = 12, 8
    q = np.zeros((1, 1, d), np.float32)
    q[0, 0, 0] = 10.0
    k = np.zeros((L, 1, d), np.float32)
    k[7, 0, 0] = 20.0                      # score 10*20*scale = 50 with scale 0.25
    rng = np.random.default_rng(4)
    vb = _rand_bits(rng, (L, 1, d))
    out, lse = oracle.attention(_bits(q), _bits(k), vb, 0.25)
    assert np.max(np.abs(out[0, 0] - oracle.bf16_to_f64(vb)[7, 0])) < 1e-15
    assert lse[0, 0] == pytest.approx(50.0 + math.log1p((L - 1) * math.exp(-50.0)), abs=1e-12)


def test_key_shift_invariance():
    """Adding the same vector c to every key shifts each score of a query by
    scale*<q, c>, which the softmax removes.  Integer-valued inputs keep K + c
    exact in bf16."""
    rng = np.random.default_rng(5)
    S, L, Hq, Hkv, d = 3, 21, 4, 2, 16
    q = rng.integers(-3, 4, (S, Hq, d)).astype(np.float32)
    k = rng.integers(-4, 5, (L, Hkv, d)).astype(np.float32)
    c = rng.integers(-4, 5, (1, Hkv, d)).astype(np.float32)
    vb = _rand_bits(rng, (L, Hkv, d))
    o1, l1 = oracle.attention(_bits(q), _bits(k), vb, 0.05)
    o2, l2 = oracle.attention(_bits(q), _bits(k + c), vb, 0.05)
    assert np.max(np.abs(o1 - o2)) < 1e-12
    qf = q.astype(np.float64)
    shift = 0.05 * np.einsum("shd,hd->sh", qf, np.repeat(c[0], Hq // Hkv, axis=0))
    assert np.max(np.abs((l2 - l1) - shift)) < 1e-10


def test_decode_key_order_invariance():
    """A decode query sees every key, so permuting (K, V) rows together leaves
    the output unchanged up to summation order."""
    rng = np.random.default_rng(6)
    L, Hq, Hkv, d = 33, 8, 2, 32
    qb = _rand_bits(rng, (1, Hq, d))
    kb = _rand_bits(rng, (L, Hkv, d))
    vb = _rand_bits(rng, (L, Hkv, d))
    perm = rng.permutation(L)
    o1, l1 = oracle.attention(qb, kb, vb, 0.2)
    o2, l2 = oracle.attention(qb, kb[perm], vb[perm], 0.2)
    assert np.max(np.abs(o1 - o2)) < 1e-13 and np.max(np.abs(l1 - l2)) < 1e-13


def test_threads_do_not_change_results():
    rng = np.random.default_rng(7)
    qb, kb, vb = (_rand_bits(rng, (7, 8, 32)), _rand_bits(rng, (40, 2, 32)),
                  _rand_bits(rng, (40, 2, 32)))
    a = oracle.attention(qb, kb, vb, 0.3, threads=1)
    b = oracle.attention(qb, kb, vb, 0.3, threads=5)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


def test_rows_selection_equals_full_request():
    """Query row i of a request equals a single query over keys 0..cached+i."""
    from paper_2605_11232_gb300.workloads import make_workload
    w = make_workload("tiny")
    full_o, full_l = oracle.request_attention(w, 2)
    rows = [0, 17, int(w.new_lens[2]) - 1]
    o, l = oracle.request_attention(w, 2, rows=rows)
    assert np.array_equal(o, full_o[rows]) and np.array_equal(l, full_l[rows])


# ----------------------------------------------------------------------------
# cache write, slot mapping and gather: the paged layout


def test_cache_write_layout_single_token():
    """Pool layout [num_blocks][Hkv][B][d]: a token written to slot s lands at
    block s // B, offset s % B of every head, and nowhere else."""
    nb, hkv, bs, d = 5, 3, 16, 8
    kp = np.zeros((nb, hkv, bs, d), np.uint16)
    vp = np.zeros_like(kp)
    kn = (np.arange(hkv * d, dtype=np.uint16) + 1).reshape(1, hkv, d)
    vn = kn + 1000
    slot = 3 * bs + 11
    assert oracle.cache_write(kp, vp, kn, vn, np.array([slot])) == 1
    flat = kp.reshape(-1)
    for h in range(hkv):
        start = ((3 * hkv + h) * bs + 11) * d
        assert np.array_equal(flat[start:start + d], kn[0, h])
    assert np.count_nonzero(flat) == hkv * d
    assert np.array_equal(vp[3, :, 11, :], vn[0])


def test_cache_write_skips_negative_slots_and_rejects_out_of_pool():
    kp = np.zeros((2, 1, 16, 8), np.uint16)
    vp = np.zeros_like(kp)
    kn = np.ones((2, 1, 8), np.uint16)
    assert oracle.cache_write(kp, vp, kn, kn, np.array([-1, 5])) == 1
    assert np.count_nonzero(kp) == 8
    with pytest.raises(ValueError):
        oracle.cache_write(kp, vp, kn, kn, np.array([0, 32]))


def _random_tables(rng, ctx, nb, bs):
    """Block tables over a random placement of a pool (brute-force helper)."""
    perm = rng.permutation(nb).astype(np.int32)
    need = [(c + bs - 1) // bs for c in ctx]
    width = max(need)
    table = np.full((len(ctx), width), -1, np.int32)
    k = 0
    for r, n in enumerate(need):
        table[r, :n] = perm[k:k + n]
        k += n
    return table


def test_slot_mapping_against_block_walk():
    """Slots from the division formula equal slots found by walking each table
    row block by block and offset by offset."""
    rng = np.random.default_rng(8)
    bs = 16
    ctx = np.array([1, 16, 17, 50, 33], np.int32)
    new = np.array([1, 16, 2, 20, 33], np.int32)
    table = _random_tables(rng, ctx, 64, bs)
    got = oracle.slot_mapping(table, ctx, new, bs)
    want = []
    for r in range(len(ctx)):
        walk = [int(table[r, b]) * bs + o for b in range(table.shape[1]) for o in range(bs)]
        want += walk[ctx[r] - new[r]: ctx[r]]
    assert np.array_equal(got, np.array(want, np.int64))


def test_write_then_gather_roundtrip():
    """Writing every token of every request through its slots, then gathering
    through the table, returns the logical K/V; slots are all distinct."""
    rng = np.random.default_rng(9)
    bs, hkv, d, nb = 16, 2, 16, 40
    ctx = np.array([5, 40, 64, 100], np.int32)
    table = _random_tables(rng, ctx, nb, bs)
    slots = oracle.slot_mapping(table, ctx, ctx, bs)
    assert len(np.unique(slots)) == len(slots)
    kn = _rand_bits(rng, (int(ctx.sum()), hkv, d))
    vn = _rand_bits(rng, (int(ctx.sum()), hkv, d))
    kp = np.zeros((nb, hkv, bs, d), np.uint16)
    vp = np.zeros_like(kp)
    oracle.cache_write(kp, vp, kn, vn, slots)
    off = 0
    for r, L in enumerate(ctx):
        assert np.array_equal(oracle.gather(kp, table[r], int(L)), kn[off:off + L])
        assert np.array_equal(oracle.gather(vp, table[r], int(L)), vn[off:off + L])
        off += L


def test_placement_invariance_and_shared_prefix_equals_private_copies():
    """Paged attention is independent of where blocks live: two different
    placements, and a shared prefix versus private copies of it, give
    bit-identical oracle outputs."""
    rng = np.random.default_rng(10)
    bs, hkv, hq, d = 16, 2, 8, 32
    P, S = 48, 20
    pre_k = _rand_bits(rng, (P, hkv, d))
    pre_v = _rand_bits(rng, (P, hkv, d))
    outs = []
    for trial in range(3):
        nb = 30
        kp = np.zeros((nb, hkv, bs, d), np.uint16)
        vp = np.zeros_like(kp)
        perm = np.random.default_rng(100 + trial).permutation(nb).astype(np.int32)
        pre_blocks = perm[:P // bs]
        row = np.concatenate([pre_blocks, perm[P // bs: P // bs + 2]])
        if trial == 2:   # private copy of the prefix in other blocks
            row = np.concatenate([perm[10:13], perm[13:15]])
        oracle.cache_write(kp, vp, pre_k, pre_v, oracle.slot_mapping(
            row[None], np.array([P]), np.array([P]), bs))
        suf_k = _rand_bits(np.random.default_rng(11), (S, hkv, d))
        suf_v = _rand_bits(np.random.default_rng(12), (S, hkv, d))
        oracle.cache_write(kp, vp, suf_k, suf_v, oracle.slot_mapping(
            row[None], np.array([P + S]), np.array([S]), bs))
        qb = _rand_bits(np.random.default_rng(13), (S, hq, d))
        outs.append(oracle.paged_request_attention(kp, vp, row, P + S, qb, 0.17))
    for o, l in outs[1:]:
        assert np.array_equal(o, outs[0][0]) and np.array_equal(l, outs[0][1])


def test_gather_rejects_bad_table_entry():
    kp = np.zeros((2, 1, 16, 8), np.uint16)
    with pytest.raises(ValueError):
        oracle.gather(kp, np.array([0, 7], np.int32), 20)
