/* A plain C11 client of the library's host-side calls (no GPU): a pool
 * without device caches, block allocation, slot mapping, the prefix-caching
 * index, the prefix-group builder and the multi-adapter dispatch.  Prints
 * "ok" on success; any failure prints the call and its message and exits
 * non-zero. */
#include <stdio.h>
#include <stdlib.h>

#include "pkv.h"

#define CHECK(call)                                                              \
    do {                                                                         \
        int rc_ = (call);                                                        \
        if (rc_ != PKV_OK) {                                                     \
            fprintf(stderr, "%s -> %d: %s\n", #call, rc_, pkv_last_error());     \
            return 1;                                                            \
        }                                                                        \
    } while (0)
#define EXPECT(cond)                                                             \
    do {                                                                         \
        if (!(cond)) {                                                           \
            fprintf(stderr, "expectation failed: %s\n", #cond);                  \
            return 1;                                                            \
        }                                                                        \
    } while (0)

int main(void) {
    pkv_pool_desc desc = {64, 16, 2, 128, PKV_DTYPE_BF16, 0, 0};
    pkv_pool_t pool = NULL;
    CHECK(kv_pool_create(&desc, NULL, NULL, &pool));

    /* request A: 40 tokens (3 blocks); register its 2 full blocks */
    int32_t tokens_a[40], tokens_b[40], row_a[3], row_b[3], n = 0, added = 0, nfree = 0;
    for (int i = 0; i < 40; ++i) tokens_a[i] = tokens_b[i] = 1000 + i;
    tokens_b[35] = 7;   /* B shares A's first two blocks only */
    CHECK(kv_pool_alloc(pool, 3, row_a));
    pkv_prefix_cache_t cache = NULL;
    CHECK(pkv_prefix_cache_create(pool, 0, &cache));
    CHECK(pkv_prefix_cache_insert(cache, tokens_a, 40, row_a, 3, &added));
    EXPECT(added == 2);

    /* request B reuses them and allocates its own last block */
    CHECK(pkv_prefix_cache_match(cache, tokens_b, 40, row_b, 3, &n));
    EXPECT(n == 2 && row_b[0] == row_a[0] && row_b[1] == row_a[1]);
    CHECK(kv_pool_alloc(pool, 1, row_b + 2));
    int32_t rc_count = 0;
    CHECK(kv_pool_refcount(pool, row_a[0], &rc_count));
    EXPECT(rc_count == 3);   /* request A, the index, request B */

    /* slots of both requests' last token, and their prefix groups */
    int32_t table[2][3] = {{row_a[0], row_a[1], row_a[2]}, {row_b[0], row_b[1], row_b[2]}};
    int32_t ctx[2] = {40, 40}, newl[2] = {1, 1};
    int64_t slots[2];
    CHECK(kv_slot_mapping(pool, &table[0][0], 3, ctx, newl, 2, slots));
    EXPECT(slots[0] == (int64_t)row_a[2] * 16 + 7 && slots[1] == (int64_t)row_b[2] * 16 + 7);
    int32_t gor[2], gstart[3], members[2], gblocks[2], G = 0, mgb = 0, mgm = 0;
    CHECK(pkv_prefix_groups_build(&table[0][0], 3, 2, ctx, 1, gor, gstart, members, gblocks, &G, &mgb,
                                  &mgm));
    EXPECT(G == 1 && gblocks[0] == 2 && gor[0] == 0 && gor[1] == 0 && mgm == 2);
    int32_t bad_req = 0;
    CHECK(pkv_check_block_table(pool, &table[0][0], 3, 2, ctx, &bad_req));
    EXPECT(bad_req == -1);

    /* requests end; the index keeps the shared blocks until they are evicted */
    CHECK(kv_pool_release(pool, row_a, 3));
    CHECK(kv_pool_release(pool, row_b, 3));
    int32_t evicted[4];
    CHECK(pkv_prefix_cache_evict(cache, 4, evicted, &n));
    EXPECT(n == 2);
    CHECK(kv_pool_num_free(pool, &nfree));
    EXPECT(nfree == 64);
    CHECK(pkv_prefix_cache_destroy(cache));
    CHECK(kv_pool_destroy(pool));

    /* a 12-prompt request over four adapters (4/3/3/2), short / medium / long */
    {
        const int32_t adapter[12] = {22, 11, 33, 11, 44, 22, 11, 33, 22, 44, 11, 33};
        const int32_t len[12] = {3000, 400, 800, 2500, 120, 450, 380, 700, 2048, 511, 512, 2047};
        const int32_t edges[2] = {512, 2048};
        const int32_t want_order[12] = {5, 0, 8, 1, 6, 10, 3, 2, 7, 11, 4, 9};
        const int32_t want_start[8] = {0, 1, 3, 5, 6, 7, 10, 12};
        int32_t order[12], start[13], badp[12], bbkt[12], nb = 0;
        CHECK(pkv_lora_dispatch(adapter, len, 12, edges, 2, 0, order, start, badp, bbkt, &nb));
        EXPECT(nb == 7);
        for (int k = 0; k < 12; ++k) EXPECT(order[k] == want_order[k]);
        for (int b = 0; b <= 7; ++b) EXPECT(start[b] == want_start[b]);
        EXPECT(badp[0] == 22 && bbkt[0] == 0 && badp[1] == 22 && bbkt[1] == 2 && badp[6] == 44);
    }

    /* every declared entry point resolves */
    void *entries[] = {(void *)kv_cache_write, (void *)paged_attn_prefill, (void *)paged_attn_decode,
                       (void *)paged_attn_decode_workspace_size, (void *)paged_attn_decode_noalloc,
                       (void *)paged_attn_decode_step, (void *)pkv_trace_enable, (void *)pkv_trace_read,
                       (void *)pkv_check_device_errors, (void *)pkv_selftest_wait_timeout,
                       (void *)kv_pool_alloc_sequence, (void *)pkv_prefix_cache_size};
    for (size_t i = 0; i < sizeof entries / sizeof entries[0]; ++i) EXPECT(entries[i] != NULL);
    puts("ok");
    return 0;
}
