"""Tree-shaped speculative-decode verification attention of
oracle/tree_verify.py pinned by reductions to the causal prefill and
one-token decode oracles and by relabelling / path invariants (CPU)."""
import numpy as np
import pytest
import torch

import oracle
from oracle import tree_verify as TV


def _bits(shape, gen):
    t = torch.randn(shape, generator=gen).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16).copy()


def _case(seed, P=45, k=7, Hq=8, Hkv=2, d=32):
    g = torch.Generator().manual_seed(seed)
    return _bits((k, Hq, d), g), _bits((P + k, Hkv, d), g), _bits((P + k, Hkv, d), g), d ** -0.5


def test_chain_is_the_causal_suffix_prefill():
    q, kb, vb, scale = _case(1)
    k = q.shape[0]
    o, l = TV.tree_verify_attention(q, kb, vb, [-1] + list(range(k - 1)), scale)
    o_ref, l_ref = oracle.attention(q, kb, vb, scale)
    assert np.allclose(o, o_ref, rtol=0, atol=1e-12) and np.allclose(l, l_ref, rtol=0, atol=1e-12)


def test_star_is_independent_one_token_decodes():
    q, kb, vb, scale = _case(2)
    k = q.shape[0]
    P = kb.shape[0] - k
    o, l = TV.tree_verify_attention(q, kb, vb, [-1] * k, scale)
    for i in range(k):
        keys = np.concatenate([kb[:P], kb[P + i:P + i + 1]])
        vals = np.concatenate([vb[:P], vb[P + i:P + i + 1]])
        o_ref, l_ref = oracle.attention(q[i:i + 1], keys, vals, scale)
        assert np.allclose(o[i], o_ref[0], rtol=0, atol=1e-12)
        assert np.allclose(l[i], l_ref[0], rtol=0, atol=1e-12)


PARENT = [-1, 0, 0, 1, -1, 4, 2, 3]      # two roots; branches of depth up to 3


def test_relabelling_in_another_parents_first_order_permutes_outputs():
    q, kb, vb, scale = _case(3, k=len(PARENT))
    P = kb.shape[0] - len(PARENT)
    o, l = TV.tree_verify_attention(q, kb, vb, PARENT, scale)
    # new order: the second root's subtree first, then the first root's
    new_of_old = {4: 0, 5: 1, 0: 2, 2: 3, 1: 4, 6: 5, 3: 6, 7: 7}
    old_of_new = {v: u for u, v in new_of_old.items()}
    n = len(PARENT)
    parent2 = [new_of_old[PARENT[old_of_new[j]]] if PARENT[old_of_new[j]] >= 0 else -1 for j in range(n)]
    assert all(p < j for j, p in enumerate(parent2))
    perm = [old_of_new[j] for j in range(n)]
    q2 = q[perm]
    kb2 = np.concatenate([kb[:P], kb[P:][perm]])
    vb2 = np.concatenate([vb[:P], vb[P:][perm]])
    o2, l2 = TV.tree_verify_attention(q2, kb2, vb2, parent2, scale)
    assert np.array_equal(o2, o[perm]) and np.array_equal(l2, l[perm])


def test_drafts_off_the_path_are_ignored():
    q, kb, vb, scale = _case(4, k=len(PARENT))
    P = kb.shape[0] - len(PARENT)
    o, _ = TV.tree_verify_attention(q, kb, vb, PARENT, scale)
    paths = TV.ancestors(PARENT)
    assert paths[7] == {0, 1, 3, 7} and paths[5] == {4, 5}
    for i, path in enumerate(paths):
        kb2, vb2 = kb.copy(), vb.copy()
        for j in set(range(len(PARENT))) - path:
            kb2[P + j] ^= 0x1234          # other values at every off-path draft
            vb2[P + j] ^= 0x0F0F
        o2, _ = TV.tree_verify_attention(q, kb2, vb2, PARENT, scale)
        assert np.array_equal(o2[i], o[i])
        if len(path) < len(PARENT):
            assert not np.array_equal(o2, o)   # the perturbation reached some draft


def test_rejects_parents_that_are_not_earlier_drafts():
    q, kb, vb, scale = _case(5, k=3)
    for parent in ([-1, 1, 0], [-1, 0, 3], [-2, 0, 1]):
        with pytest.raises(ValueError):
            TV.tree_verify_attention(q, kb, vb, parent, scale)
