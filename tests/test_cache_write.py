"""kv_cache_write is a bit-exact scatter: the whole GPU pool must equal the
oracle's pool after the same writes (untouched slots included)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2605_11232_gb300 import batch as B
from paper_2605_11232_gb300 import pkv
from paper_2605_11232_gb300.workloads import make_workload

from _lib import need_gpu

pytestmark = pytest.mark.gpu


def _bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


@pytest.mark.parametrize("name,scale", [("tiny", 1.0), ("l8b_prefill", 1.0), ("qwen_mixed", 1.0)])
def test_workload_step_write_bit_exact(name, scale):
    need_gpu()
    w = make_workload(name, scale_requests=scale)
    b = B.build_batch(w, poison=True)
    k0, v0 = _bits(b.k_cache), _bits(b.v_cache)
    B.run_write(b)
    assert pkv.pkv_check_device_errors(b.pool) == pkv.PKV_OK
    k1, v1 = _bits(b.k_cache), _bits(b.v_cache)
    slots = oracle.slot_mapping(b.table_host, w.context_lens, w.new_lens, 16)
    assert np.array_equal(slots, b.slots_host)
    n = oracle.cache_write(k0, v0, _bits(b.k_new), _bits(b.v_new), slots)
    assert n == w.num_new_tokens
    assert np.array_equal(k0, k1) and np.array_equal(v0, v1)
    b.close()


@pytest.mark.parametrize("d", [64, 128])
def test_random_slots_skip_and_bounds(d):
    need_gpu()
    rng = np.random.default_rng(d)
    nb, hkv, T = 50, 3, 300
    kc = torch.full((nb, hkv, 16, d), float("nan"), dtype=torch.bfloat16, device="cuda")
    vc = torch.full_like(kc, float("nan"))
    pool = pkv.kv_pool_create(nb, hkv, d, kc, vc)
    slots = rng.permutation(nb * 16)[:T].astype(np.int64)
    slots[::7] = -1                       # skipped tokens
    kn = torch.randn((T, hkv, d), dtype=torch.float32).to(torch.bfloat16)
    vn = torch.randn((T, hkv, d), dtype=torch.float32).to(torch.bfloat16)
    k0, v0 = _bits(kc), _bits(vc)
    pkv.kv_cache_write(pool, kn.cuda(), vn.cuda(), torch.from_numpy(slots).cuda())
    assert pkv.pkv_check_device_errors(pool) == pkv.PKV_OK
    oracle.cache_write(k0, v0, _bits(kn), _bits(vn), slots)
    assert np.array_equal(k0, _bits(kc)) and np.array_equal(v0, _bits(vc))
    # a slot past the pool is skipped and latched, the others still land
    bad = slots.copy()
    bad[3] = nb * 16 + 5
    k0, v0 = _bits(kc), _bits(vc)
    kn2 = torch.randn((T, hkv, d)).to(torch.bfloat16)
    pkv.kv_cache_write(pool, kn2.cuda(), vn.cuda(), torch.from_numpy(bad).cuda())
    assert pkv.pkv_check_device_errors(pool) == pkv.PKV_ERR_DEVICE_BOUNDS
    assert pkv.pkv_check_device_errors(pool) == pkv.PKV_OK      # cleared on read
    bad_o = bad.copy()
    bad_o[3] = -1
    oracle.cache_write(k0, v0, _bits(kn2), _bits(vn), bad_o)
    assert np.array_equal(k0, _bits(kc))
    pkv.kv_pool_destroy(pool)


def test_zero_tokens_is_noop():
    need_gpu()
    kc = torch.zeros((4, 1, 16, 64), dtype=torch.bfloat16, device="cuda")
    pool = pkv.kv_pool_create(4, 1, 64, kc, kc.clone())
    e = torch.empty((0, 1, 64), dtype=torch.bfloat16, device="cuda")
    pkv.kv_cache_write(pool, e, e, torch.empty(0, dtype=torch.int64, device="cuda"))
    assert pkv.pkv_check_device_errors(pool) == pkv.PKV_OK
    pkv.kv_pool_destroy(pool)
