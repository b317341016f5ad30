"""Adapter-first, length-bucketed dispatch of a multi-adapter request
(Sec. 5.6): the definition in oracle/lora_dispatch.py pinned by hand-worked
cases and invariants, then the library's pkv_lora_dispatch against it (CPU)."""
import numpy as np
import pytest

from oracle import lora_dispatch as D

# A 12-prompt request over four adapters split 4/3/3/2 (the split of the
# Case C1 table in Sec. 5.6), lengths on both sides of each bucket edge.
ADAPTER = [22, 11, 33, 11, 44, 22, 11, 33, 22, 44, 11, 33]
LENGTH = [3000, 400, 800, 2500, 120, 450, 380, 700, 2048, 511, 512, 2047]
EDGES = [512, 2048]          # short < 512 <= medium < 2048 <= long
# worked by hand: adapters in order of first item (22, 11, 33, 44), buckets
# shortest first, request order inside a bucket
HAND_BATCHES = [(22, 0, [5]), (22, 2, [0, 8]), (11, 0, [1, 6]), (11, 1, [10]), (11, 2, [3]),
                (33, 1, [2, 7, 11]), (44, 0, [4, 9])]


def _as_lists(order, batches):
    return [(a, b, order[s:e]) for a, b, s, e in batches]


def test_definition_hand_example():
    order, batches = D.dispatch(ADAPTER, LENGTH, EDGES)
    assert _as_lists(order, batches) == HAND_BATCHES
    assert order == [5, 0, 8, 1, 6, 10, 3, 2, 7, 11, 4, 9]
    assert sorted(ADAPTER.count(a) for a in set(ADAPTER)) == [2, 3, 3, 4]
    # padded prefill tokens: 450 + 2*3000 + 2*400 + 512 + 2500 + 3*2047 + 2*511,
    # against one batch per adapter: 3*3000 + 4*2500 + 3*2047 + 2*511
    assert D.padded_tokens(LENGTH, order, batches) == 17425
    o1, b1 = D.dispatch(ADAPTER, LENGTH)
    assert D.padded_tokens(LENGTH, o1, b1) == 26163
    assert sum(LENGTH) == 13468
    # step 5: results computed in execution order come back in request order
    assert D.restore([f"r{i}" for i in order], order) == [f"r{i}" for i in range(12)]


def test_definition_max_batch_splits_in_request_order():
    order, batches = D.dispatch(ADAPTER, LENGTH, EDGES, max_batch=2)
    got = _as_lists(order, batches)
    assert got == HAND_BATCHES[:5] + [(33, 1, [2, 7]), (33, 1, [11])] + HAND_BATCHES[6:]
    order1, batches1 = D.dispatch(ADAPTER, LENGTH, EDGES, max_batch=1)
    assert order1 == order and len(batches1) == 12


def test_definition_degenerate_cases():
    assert D.dispatch([], []) == ([], [])
    # one adapter, no edges: one batch in request order
    assert D.dispatch([7, 7, 7], [5, 1, 9]) == ([0, 1, 2], [(7, 0, 0, 3)])
    # every item its own adapter
    order, batches = D.dispatch([3, 2, 1], [10, 20, 30], [15])
    assert _as_lists(order, batches) == [(3, 0, [0]), (2, 1, [1]), (1, 1, [2])]
    with pytest.raises(ValueError):
        D.dispatch([1], [5], [10, 10])
    with pytest.raises(ValueError):
        D.dispatch([1], [-5])


def _check_invariants(adapter, length, edges, max_batch, order, batches):
    n = len(adapter)
    assert sorted(order) == list(range(n))
    assert batches[0][2] == 0 if n else batches == []
    first_seen = list(dict.fromkeys(adapter))
    seen_adapters = []
    prev_stop = 0
    for a, b, s, e in batches:
        assert s == prev_stop and e > s
        prev_stop = e
        idx = order[s:e]
        assert all(adapter[i] == a for i in idx)
        assert all(sum(length[i] >= x for x in edges) == b for i in idx)
        assert idx == sorted(idx)
        if max_batch:
            assert len(idx) <= max_batch
        if not seen_adapters or seen_adapters[-1][0] != a:
            seen_adapters.append((a, b))
        else:
            assert b >= seen_adapters[-1][1]
            seen_adapters[-1] = (a, b)
    assert prev_stop == n
    assert [a for a, _ in seen_adapters] == first_seen


@pytest.mark.parametrize("seed", range(20))
def test_definition_invariants_and_padding(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(0, 60))
    adapter = rng.integers(0, 6, n).tolist()
    length = rng.integers(0, 4000, n).tolist()
    edges = sorted(set(rng.integers(1, 4000, int(rng.integers(0, 4))).tolist()))
    max_batch = int(rng.integers(0, 5))
    order, batches = D.dispatch(adapter, length, edges, max_batch)
    _check_invariants(adapter, length, edges, max_batch, order, batches)
    # bucketing by length never adds padded tokens to an adapter's batches
    if not max_batch:
        o0, b0 = D.dispatch(adapter, length)
        assert D.padded_tokens(length, order, batches) <= D.padded_tokens(length, o0, b0)


# ---- the library (CPU: host code of libpkv.so) ------------------------------

def _lib():
    from _lib import built_lib
    from paper_2605_11232_gb300 import pkv
    built_lib()
    return pkv


def test_library_hand_example():
    pkv = _lib()
    for mb in (0, 1, 2, 3, 100):
        assert pkv.pkv_lora_dispatch(ADAPTER, LENGTH, EDGES, mb) == D.dispatch(ADAPTER, LENGTH, EDGES, mb)
    order, batches = pkv.pkv_lora_dispatch(ADAPTER, LENGTH, EDGES)
    assert _as_lists(order, batches) == HAND_BATCHES


@pytest.mark.parametrize("seed", range(30))
def test_library_matches_definition(seed):
    pkv = _lib()
    rng = np.random.default_rng(100 + seed)
    n = int(rng.integers(0, 300))
    adapter = rng.integers(0, int(rng.integers(1, 40)), n).tolist()
    # a mix of short classification, medium summary and long extraction prompts
    length = np.where(rng.random(n) < 0.5, rng.integers(16, 512, n),
                      np.where(rng.random(n) < 0.6, rng.integers(512, 2048, n),
                               rng.integers(2048, 8192, n))).tolist()
    edges = sorted(set(rng.integers(1, 8192, int(rng.integers(0, 6))).tolist()))
    max_batch = int(rng.integers(0, 9))
    got = pkv.pkv_lora_dispatch(adapter, length, edges, max_batch)
    assert got == D.dispatch(adapter, length, edges, max_batch)
    _check_invariants(adapter, length, edges, max_batch, *got)


def test_library_degenerate_and_errors():
    pkv = _lib()
    assert pkv.pkv_lora_dispatch([], []) == ([], [])
    assert pkv.pkv_lora_dispatch([5], [0], [1]) == ([0], [(5, 0, 0, 1)])
    assert pkv.pkv_lora_dispatch([5, 6], [2**31 - 1, 0], [1, 2**31 - 1]) == \
        D.dispatch([5, 6], [2**31 - 1, 0], [1, 2**31 - 1])
    for args in (([1], [5], [10, 10]), ([1], [-5], []), ([-1], [5], []), ([1], [5], [3, 2])):
        with pytest.raises(pkv.PkvError) as e:
            pkv.pkv_lora_dispatch(*args)
        assert e.value.code == pkv.PKV_ERR_INVALID_ARG
    with pytest.raises(pkv.PkvError):
        pkv.pkv_lora_dispatch([1, 2], [3, 4], [], -1)
