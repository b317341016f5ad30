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
