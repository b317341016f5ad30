"""Adapter-first, length-bucketed dispatch of a mixed multi-adapter request
(Sec. 5.6, multi-adapter and length-aware batching) -- test infrastructure
only: the tests call it; the library never does.

The paper's procedure, step by step:
  1. parse each item into (adapter_id, prompt_len, original_index);
  2. group the items by adapter_id;
  3. within each adapter group, sub-bucket the items by length range
     (short / medium / long ...);
  4. execute each bucket as one batch call;
  5. restore the original order before returning the response.

Readings where the paper is silent (the library follows the same ones):
  * adapter groups run in the order of each adapter's first item in the
    request; buckets of a group run shortest range first;
  * the length ranges are given by ascending edges e_1 < ... < e_k: an item of
    length n goes to bucket #{j : n >= e_j} (edges [512, 2048]: short below
    512, medium below 2048, long from 2048);
  * inside a bucket items keep their request order; a bucket larger than
    max_batch (when max_batch > 0) runs as consecutive batches of max_batch
    items, the last one shorter.

Parity pinned: the tests check a hand-worked 12-prompt request split 4/3/3/2
over four adapters (the split of the Case C1 table in Sec. 5.6), the invariants of the
output, and that bucketing never adds padded tokens to a group's batches.
"""

from bisect import bisect_right


def dispatch(adapter_id, prompt_len, bucket_edges=(), max_batch=0):
    """Batches of a request, in execution order.

    Returns (order, batches): order[k] is the original index of the k-th item
    executed; batches is a list of (adapter_id, bucket, start, stop) with
    order[start:stop] the batch's items.
    """
    edges = list(bucket_edges)
    if any(b <= a for a, b in zip(edges, edges[1:])):
        raise ValueError("bucket edges must be strictly ascending")
    if len(adapter_id) != len(prompt_len):
        raise ValueError("one adapter id and one length per item")
    # 1. parse
    items = [(int(a), int(n), i) for i, (a, n) in enumerate(zip(adapter_id, prompt_len))]
    for a, n, i in items:
        if a < 0 or n < 0:
            raise ValueError(f"item {i}: negative adapter id or length")
    # 2. group by adapter (a dict keeps the order of first appearance)
    groups = {}
    for a, n, i in items:
        groups.setdefault(a, []).append((a, n, i))
    order, batches = [], []
    for a, members in groups.items():
        # 3. sub-bucket by length range
        buckets = {}
        for _, n, i in members:
            buckets.setdefault(bisect_right(edges, n), []).append(i)
        # 4. one batch call per bucket (split at max_batch)
        for b in sorted(buckets):
            idx = buckets[b]
            step = max_batch if max_batch > 0 else len(idx)
            for s in range(0, len(idx), step):
                start = len(order)
                order.extend(idx[s:s + step])
                batches.append((a, b, start, len(order)))
    return order, batches


def restore(results, order):
    """Step 5: results[k] belongs to item order[k]; return them in request order."""
    out = [None] * len(order)
    for k, i in enumerate(order):
        out[i] = results[k]
    return out


def padded_tokens(prompt_len, order, batches):
    """Tokens a padded prefill of these batches processes: each batch pads
    its items to its longest one."""
    total = 0
    for _, _, start, stop in batches:
        lens = [int(prompt_len[i]) for i in order[start:stop]]
        total += max(lens) * len(lens)
    return total
