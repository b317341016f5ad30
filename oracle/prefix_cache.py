"""Plain definition of the prefix-caching index, for tests.

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, never by the library, and
sharing no code with it.  Automatic Prefix Caching (Sec. 5.4) reuses the KV
blocks of a shared leading token run.  Written out plainly:

* a full block j of a token sequence (tokens [16j, 16j + 16)) is identified by
  the whole token prefix ``tuple(tokens[:16 (j + 1)])``;
* ``match``: the longest j0 such that the prefixes of blocks 0 .. j0-1 are all
  cached; their blocks are handed to the caller (one more reference each);
* ``insert``: every full block whose prefix is not cached yet is cached with
  the caller's block id (the index takes one reference); a cached prefix keeps
  its block;
* every call takes the next tick; matched or inserted prefixes record it;
* ``evict``: repeatedly remove the cached prefix that (a) has no cached prefix
  one block longer, (b) whose block only the index holds (reference count 1),
  and (c) is the least recently used, then the longest, then the oldest;
  its reference is dropped.

The pool is modelled by a reference count per block id (ids are inputs: the
test passes the ids that it allocated).
"""

from __future__ import annotations

BS = 16


class PoolModel:
    """Reference counts of block ids; a block with count 0 is free."""

    def __init__(self, num_blocks: int):
        self.ref = [0] * num_blocks

    def alloc(self, ids):
        for i in ids:
            assert self.ref[i] == 0, f"block {i} handed out while in use"
            self.ref[i] = 1

    def retain(self, ids):
        for i in ids:
            assert self.ref[i] > 0
            self.ref[i] += 1

    def release(self, ids):
        for i in ids:
            assert self.ref[i] > 0
            self.ref[i] -= 1

    def num_free(self) -> int:
        return sum(1 for r in self.ref if r == 0)


class PrefixCacheModel:
    def __init__(self, pool: PoolModel):
        self.pool = pool
        self.entries = {}   # prefix tuple -> [block, last_use, serial]
        self.tick = 0
        self.serial = 0

    def match(self, tokens, max_ids=None):
        self.tick += 1
        full = len(tokens) // BS if max_ids is None else min(len(tokens) // BS, max_ids)
        out = []
        for j in range(full):
            key = tuple(tokens[:BS * (j + 1)])
            if key not in self.entries:
                break
            self.entries[key][1] = self.tick
            out.append(self.entries[key][0])
        self.pool.retain(out)
        return out

    def insert(self, tokens, ids):
        self.tick += 1
        added = 0
        for j in range(min(len(tokens) // BS, len(ids))):
            key = tuple(tokens[:BS * (j + 1)])
            if key not in self.entries:
                self.pool.retain([ids[j]])
                self.entries[key] = [ids[j], self.tick, self.serial]
                self.serial += 1
                added += 1
            else:
                self.entries[key][1] = self.tick
        return added

    def _evictable(self):
        longer = {k[:-BS] for k in self.entries if len(k) > BS}
        return [k for k, e in self.entries.items()
                if k not in longer and self.pool.ref[e[0]] == 1]

    def evict(self, n_wanted):
        out = []
        while len(out) < n_wanted:
            cand = self._evictable()
            if not cand:
                break
            k = min(cand, key=lambda k: (self.entries[k][1], -len(k), self.entries[k][2]))
            block = self.entries.pop(k)[0]
            self.pool.release([block])
            out.append(block)
        return out

    def size(self):
        return len(self.entries)


def prefix_groups(table, context_lens, min_shared_blocks=1):
    """Prefix groups of a decode batch, written out: candidates (requests with
    at least min_shared_blocks shareable blocks, i.e. (L - 1) // 16 full
    blocks before the one holding the query) grouped by their first block id
    in order of first appearance; a member's run is its run of equal leading
    ids with the group's first candidate, within its cap; candidates below
    min_shared_blocks stay out; a group of at least two shares the shortest
    run.  Returns (group_of_req, [(members, shared_blocks), ...])."""
    R, mb = len(table), len(table[0]) if len(table) else 0
    cap = [min((int(L) - 1) // BS, mb) if L >= 1 else 0 for L in context_lens]
    order, cand = [], {}
    for r in range(R):
        if cap[r] < min_shared_blocks or table[r][0] < 0:
            continue
        f = int(table[r][0])
        if f not in cand:
            cand[f] = []
            order.append(f)
        cand[f].append(r)
    group_of_req = [-1] * R
    groups = []
    for f in order:
        c = cand[f]
        if len(c) < 2:
            continue
        ref = table[c[0]]
        runs = []
        for r in c:
            k = 0
            while k < cap[r] and table[r][k] == ref[k] and table[r][k] >= 0:
                k += 1
            if k >= min_shared_blocks:
                runs.append((r, k))
        if len(runs) < 2:
            continue
        for r, _ in runs:
            group_of_req[r] = len(groups)
        groups.append(([r for r, _ in runs], min(k for _, k in runs)))
    return group_of_req, groups
