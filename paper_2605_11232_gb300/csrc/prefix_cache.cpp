// prefix_cache.cpp -- automatic prefix caching: a host index of cached full
// blocks of the paged pool (Sec. 5.4, the prefix reuse that Automatic Prefix
// Caching gives; Sec. 2 for the block-table addressing it feeds).
//
// A request's tokens are cut into blocks of 16.  Every full block that a
// request has written can be registered: the index keys it by its whole token
// prefix (the block's own tokens and every token before it) and keeps one
// reference on the physical block, so that a later request with the same
// leading tokens reuses the block instead of recomputing it.  Only full blocks
// are cached, so a shared block is never written again.
//
// Keys are chained 64-bit hashes (key_j = mix(key_{j-1}, tokens of block j));
// a lookup compares the parent entry and the 16 tokens exactly, so a hash
// collision never shares a block.  Blocks that no request holds (the index's
// reference is the only one) are evicted least recently used first; an entry
// is evicted only once its cached children are gone.
//
// The index talks to the pool only through its public calls (retain, release,
// refcount).  A handle is not thread-safe, like the pool.
#include "../../include/pkv.h"

#include <algorithm>
#include <cstdint>
#include <cstring>
#include <string>
#include <unordered_map>
#include <vector>

#include "pkv_internal.h"

namespace {

constexpr int kBlock = 16;

uint64_t mix64(uint64_t x) {   // splitmix64 finaliser
    x += 0x9e3779b97f4a7c15ull;
    x = (x ^ (x >> 30)) * 0xbf58476d1ce4e5b9ull;
    x = (x ^ (x >> 27)) * 0x94d049bb133111ebull;
    return x ^ (x >> 31);
}

uint64_t chain_key(uint64_t parent_key, const int32_t *tokens) {
    uint64_t h = parent_key;
    for (int i = 0; i < kBlock; ++i) h = mix64(h ^ (uint32_t)tokens[i]);
    return h;
}

constexpr uint64_t kRootKey = 0x243f6a8885a308d3ull;

struct Entry {
    int32_t parent = -1;       // entry of the previous block (-1: the sequence's first block)
    int32_t block = -1;        // physical block (the index holds one reference)
    int32_t children = 0;      // live entries whose parent this is
    int32_t depth = 0;         // block index in the sequence
    uint64_t key = 0;          // chained hash of the whole prefix
    uint64_t last_use = 0;     // tick of the last match / insert through this entry
    uint64_t serial = 0;       // creation order
    bool live = false;
    int32_t tokens[kBlock];
};

}  // namespace

struct pkv_prefix_cache {
    pkv_pool_t pool = nullptr;
    uint64_t key_mask = ~0ull;   // all bits; a test flag keeps 4 (forced collisions)
    std::vector<Entry> entries;
    std::vector<int32_t> free_entries;
    std::unordered_multimap<uint64_t, int32_t> by_key;
    uint64_t tick = 0, serial = 0;
    int32_t live = 0;

    // the live entry for this block under `parent`, or -1
    int32_t find(uint64_t key, int32_t parent, const int32_t *tokens) const {
        auto range = by_key.equal_range(key & key_mask);
        for (auto it = range.first; it != range.second; ++it) {
            const Entry &e = entries[it->second];
            if (e.parent == parent && std::memcmp(e.tokens, tokens, sizeof(e.tokens)) == 0)
                return it->second;
        }
        return -1;
    }
};

namespace {

int fail(int code, const std::string &msg) { return pkv::set_last_error(code, msg.c_str()); }

}  // namespace

extern "C" {

int pkv_prefix_cache_create(pkv_pool_t pool, int32_t flags, pkv_prefix_cache_t *out) {
    if (!pool || !out) return fail(PKV_ERR_INVALID_ARG, "pool and out must be non-NULL");
    if (flags & ~PKV_PREFIX_CACHE_WEAK_HASH) return fail(PKV_ERR_INVALID_ARG, "unknown flags");
    auto *c = new pkv_prefix_cache();
    c->pool = pool;
    if (flags & PKV_PREFIX_CACHE_WEAK_HASH) c->key_mask = 0xF;
    *out = c;
    return PKV_OK;
}

int pkv_prefix_cache_destroy(pkv_prefix_cache_t cache) {
    if (!cache) return PKV_OK;
    std::vector<int32_t> held;
    for (const Entry &e : cache->entries)
        if (e.live) held.push_back(e.block);
    int rc = held.empty() ? PKV_OK : kv_pool_release(cache->pool, held.data(), (int32_t)held.size());
    delete cache;
    return rc;
}

int pkv_prefix_cache_match(pkv_prefix_cache_t cache, const int32_t *tokens, int32_t n_tokens,
                           int32_t *ids_out, int32_t max_ids, int32_t *n_ids_out) {
    if (!cache || !n_ids_out || n_tokens < 0 || max_ids < 0 || (n_tokens > 0 && !tokens) ||
        (max_ids > 0 && !ids_out))
        return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    *n_ids_out = 0;
    const uint64_t tick = ++cache->tick;
    const int32_t full = std::min(n_tokens / kBlock, max_ids);
    std::vector<int32_t> path;
    int32_t parent = -1;
    uint64_t key = kRootKey;
    for (int32_t j = 0; j < full; ++j) {
        const int32_t *t = tokens + (size_t)j * kBlock;
        key = chain_key(key, t);
        const int32_t e = cache->find(key, parent, t);
        if (e < 0) break;
        path.push_back(e);
        parent = e;
    }
    for (size_t i = 0; i < path.size(); ++i) ids_out[i] = cache->entries[path[i]].block;
    if (!path.empty()) {
        // the caller's request now holds each matched block
        const int rc = kv_pool_retain(cache->pool, ids_out, (int32_t)path.size());
        if (rc != PKV_OK) return rc;
        for (int32_t e : path) cache->entries[e].last_use = tick;
    }
    *n_ids_out = (int32_t)path.size();
    return PKV_OK;
}

int pkv_prefix_cache_insert(pkv_prefix_cache_t cache, const int32_t *tokens, int32_t n_tokens,
                            const int32_t *ids, int32_t n_ids, int32_t *n_added_out) {
    if (!cache || n_tokens < 0 || n_ids < 0 || (n_tokens > 0 && !tokens) || (n_ids > 0 && !ids))
        return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    if (n_added_out) *n_added_out = 0;
    const int32_t full = std::min(n_tokens / kBlock, n_ids);
    // every block to be registered must be allocated (held by the caller)
    for (int32_t j = 0; j < full; ++j) {
        int32_t rc_count = 0;
        const int rc = kv_pool_refcount(cache->pool, ids[j], &rc_count);
        if (rc != PKV_OK) return rc;
        if (rc_count <= 0) return fail(PKV_ERR_REFCOUNT, "block " + std::to_string(ids[j]) + " is free");
    }
    const uint64_t tick = ++cache->tick;
    int32_t parent = -1, added = 0;
    uint64_t key = kRootKey;
    for (int32_t j = 0; j < full; ++j) {
        const int32_t *t = tokens + (size_t)j * kBlock;
        key = chain_key(key, t);
        int32_t e = cache->find(key, parent, t);
        if (e < 0) {
            // a new entry: the index takes its own reference on the block
            const int rc = kv_pool_retain(cache->pool, ids + j, 1);
            if (rc != PKV_OK) return rc;
            if (!cache->free_entries.empty()) {
                e = cache->free_entries.back();
                cache->free_entries.pop_back();
            } else {
                e = (int32_t)cache->entries.size();
                cache->entries.emplace_back();
            }
            Entry &n = cache->entries[e];
            n.parent = parent;
            n.block = ids[j];
            n.children = 0;
            n.depth = j;
            n.key = key;
            n.serial = cache->serial++;
            n.live = true;
            std::memcpy(n.tokens, t, sizeof(n.tokens));
            if (parent >= 0) ++cache->entries[parent].children;
            cache->by_key.emplace(key & cache->key_mask, e);
            ++cache->live;
            ++added;
        }
        // an existing entry keeps its block; the caller's copy stays its own
        cache->entries[e].last_use = tick;
        parent = e;
    }
    if (n_added_out) *n_added_out = added;
    return PKV_OK;
}

int pkv_prefix_cache_evict(pkv_prefix_cache_t cache, int32_t n_wanted, int32_t *ids_out,
                           int32_t *n_evicted_out) {
    if (!cache || n_wanted < 0 || !n_evicted_out || (n_wanted > 0 && !ids_out))
        return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    *n_evicted_out = 0;
    // Least recently used first; among equals the deeper block, then the
    // older entry.  A parent is used whenever a child is, so one pass in this
    // order reaches each parent after its children.
    std::vector<int32_t> order;
    for (int32_t i = 0; i < (int32_t)cache->entries.size(); ++i)
        if (cache->entries[i].live) order.push_back(i);
    std::sort(order.begin(), order.end(), [&](int32_t a, int32_t b) {
        const Entry &x = cache->entries[a], &y = cache->entries[b];
        if (x.last_use != y.last_use) return x.last_use < y.last_use;
        if (x.depth != y.depth) return x.depth > y.depth;
        return x.serial < y.serial;
    });
    int32_t n = 0;
    for (int32_t i : order) {
        if (n >= n_wanted) break;
        Entry &e = cache->entries[i];
        if (e.children > 0) continue;
        int32_t count = 0;
        int rc = kv_pool_refcount(cache->pool, e.block, &count);
        if (rc != PKV_OK) return rc;
        if (count != 1) continue;   // a request still holds it
        rc = kv_pool_release(cache->pool, &e.block, 1);
        if (rc != PKV_OK) return rc;
        auto range = cache->by_key.equal_range(e.key & cache->key_mask);
        for (auto it = range.first; it != range.second; ++it)
            if (it->second == i) {
                cache->by_key.erase(it);
                break;
            }
        if (e.parent >= 0) --cache->entries[e.parent].children;
        ids_out[n++] = e.block;
        e.live = false;
        --cache->live;
        cache->free_entries.push_back(i);
    }
    *n_evicted_out = n;
    return PKV_OK;
}

int pkv_prefix_cache_size(pkv_prefix_cache_t cache, int32_t *n_cached_out) {
    if (!cache || !n_cached_out) return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    *n_cached_out = cache->live;
    return PKV_OK;
}

}  // extern "C"

// ---- prefix groups of a decode batch ----------------------------------------

extern "C" int pkv_prefix_groups_build(const int32_t *block_table, int32_t max_blocks,
                                       int32_t num_requests, const int32_t *context_lens,
                                       int32_t min_shared_blocks, int32_t *group_of_req_out,
                                       int32_t *group_start_out, int32_t *member_req_out,
                                       int32_t *group_blocks_out, int32_t *num_groups_out,
                                       int32_t *max_group_blocks_out,
                                       int32_t *max_group_members_out) {
    if (num_requests < 0 || max_blocks <= 0 || min_shared_blocks < 1 || !num_groups_out ||
        !max_group_blocks_out || !max_group_members_out ||
        (num_requests > 0 && (!block_table || !context_lens || !group_of_req_out || !group_start_out ||
                              !member_req_out || !group_blocks_out)))
        return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    *num_groups_out = *max_group_blocks_out = *max_group_members_out = 0;
    if (num_requests == 0) return PKV_OK;
    group_start_out[0] = 0;
    const int32_t R = num_requests;
    auto row = [&](int32_t r) { return block_table + (size_t)r * max_blocks; };
    // blocks of request r that may be shared: full blocks before the one that
    // holds its query token (a decode request keeps at least one private block)
    auto cap = [&](int32_t r) {
        const int32_t L = context_lens[r];
        return L < 1 ? 0 : std::min((L - 1) / kBlock, max_blocks);
    };
    // candidates by first block id, in request order
    std::unordered_map<int32_t, std::vector<int32_t>> by_first;
    std::vector<int32_t> firsts;   // first ids in order of their first request
    for (int32_t r = 0; r < R; ++r) {
        group_of_req_out[r] = -1;
        if (cap(r) < min_shared_blocks || row(r)[0] < 0) continue;
        auto &v = by_first[row(r)[0]];
        if (v.empty()) firsts.push_back(row(r)[0]);
        v.push_back(r);
    }
    int32_t G = 0, nm = 0;
    for (int32_t first : firsts) {
        const std::vector<int32_t> &cand = by_first[first];
        if (cand.size() < 2) continue;
        const int32_t *ref = row(cand[0]);
        // each member's shared run with the first candidate, within its cap
        std::vector<int32_t> members;
        int32_t shared = max_blocks;
        for (int32_t r : cand) {
            const int32_t c = cap(r), *rr = row(r);
            int32_t k = 0;
            while (k < c && rr[k] == ref[k] && rr[k] >= 0) ++k;
            if (k < min_shared_blocks) continue;
            members.push_back(r);
            shared = std::min(shared, k);
        }
        if (members.size() < 2) continue;
        for (int32_t r : members) {
            group_of_req_out[r] = G;
            member_req_out[nm++] = r;
        }
        group_blocks_out[G] = shared;
        group_start_out[G + 1] = nm;
        *max_group_blocks_out = std::max(*max_group_blocks_out, shared);
        *max_group_members_out = std::max(*max_group_members_out, (int32_t)members.size());
        ++G;
    }
    *num_groups_out = G;
    return PKV_OK;
}
