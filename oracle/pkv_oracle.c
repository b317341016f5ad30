/*
 * pkv_oracle.c -- plain fp64 CPU oracle for prefix-cached paged attention.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the CPU
 * baseline leg of the benchmark may load this library.  It shares no code,
 * header, table or helper with the CUDA library; both read the same seeded
 * inputs and nothing else.
 *
 * What the paper fixes (arXiv 2605.11232): the serving stack keeps the KV
 * cache in fixed-size physical blocks addressed through a per-request block
 * table (PagedAttention, Sec. 2 and Sec. 5.4) and reuses the blocks of a
 * shared policy/schema prefix across requests instead of recomputing them
 * (Automatic Prefix Caching, Sec. 2, Sec. 5.4, Fig. 1 "Reuse plane", and the
 * design principle at the end of Sec. 3).  Paging and prefix reuse change
 * where keys and values live, not what attention computes, so the oracle is
 * the plain definition written out:
 *
 *   cache write   copy each new token's K/V rows into the slot it is mapped to
 *   slot mapping  slot(p) = table[p / B] * B + p % B
 *   gather        K_r[p] = pool[table_r[p / B]][head][p % B]
 *   attention     query at absolute position pos, q-head h, kv-head h / g:
 *                 s_j = scale * <q, K_j>  for keys j <= pos
 *                 O   = sum_j exp(s_j - m) V_j / sum_j exp(s_j - m),  m = max s_j
 *                 LSE = m + ln sum_j exp(s_j - m)
 *
 * Everything is computed in double precision from the exact bf16 inputs.
 * Pool layout (the library's ABI): pool[num_blocks][Hkv][B][d], bf16 bits.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* A bf16 value is the high half of an IEEE fp32 value. */
static double bf16_to_double(uint16_t bits) {
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

double oracle_bf16_to_double(uint16_t bits) { return bf16_to_double(bits); }

/*
 * Cache write: for each new token t with slot[t] >= 0, block = slot / B,
 * offset = slot % B, copy the d-element rows of every kv head.  Returns the
 * number of tokens written, or -1 if a slot lies outside the pool.
 */
int64_t oracle_cache_write(uint16_t *k_pool, uint16_t *v_pool, int64_t num_blocks,
                           int32_t num_kv_heads, int32_t block_size, int32_t head_dim,
                           const uint16_t *k_new, const uint16_t *v_new,
                           const int64_t *slot, int64_t num_tokens) {
    int64_t written = 0;
    for (int64_t t = 0; t < num_tokens; ++t) {
        int64_t s = slot[t];
        if (s < 0) continue;
        int64_t blk = s / block_size, off = s % block_size;
        if (blk >= num_blocks) return -1;
        for (int32_t h = 0; h < num_kv_heads; ++h) {
            int64_t dst = ((blk * num_kv_heads + h) * block_size + off) * head_dim;
            int64_t src = (t * num_kv_heads + h) * (int64_t)head_dim;
            memcpy(k_pool + dst, k_new + src, sizeof(uint16_t) * (size_t)head_dim);
            memcpy(v_pool + dst, v_new + src, sizeof(uint16_t) * (size_t)head_dim);
        }
        ++written;
    }
    return written;
}

/*
 * Slot mapping: new token i of request r sits at position
 * p = context_len[r] - new_len[r] + i; its slot is table[r][p/B]*B + p%B.
 * Tokens are laid out request after request.  Returns tokens mapped, or -1
 * if a needed table entry is negative.
 */
int64_t oracle_slot_mapping(const int32_t *table, int32_t max_blocks,
                            const int32_t *context_lens, const int32_t *new_lens,
                            int32_t num_requests, int32_t block_size, int64_t *slot_out) {
    int64_t t = 0;
    for (int32_t r = 0; r < num_requests; ++r) {
        for (int32_t i = 0; i < new_lens[r]; ++i) {
            int64_t p = (int64_t)context_lens[r] - new_lens[r] + i;
            int32_t phys = table[(int64_t)r * max_blocks + p / block_size];
            if (phys < 0) return -1;
            slot_out[t++] = (int64_t)phys * block_size + p % block_size;
        }
    }
    return t;
}

/*
 * Gather: contiguous [L][Hkv][d] copy of one request's keys (or values) read
 * through its block-table row.  Returns 0, or -1 on a bad table entry.
 */
int oracle_gather(const uint16_t *pool, int64_t num_blocks, int32_t num_kv_heads,
                  int32_t block_size, int32_t head_dim, const int32_t *table_row,
                  int32_t context_len, uint16_t *out) {
    for (int32_t p = 0; p < context_len; ++p) {
        int32_t phys = table_row[p / block_size];
        if (phys < 0 || phys >= num_blocks) return -1;
        for (int32_t h = 0; h < num_kv_heads; ++h) {
            int64_t src = (((int64_t)phys * num_kv_heads + h) * block_size + p % block_size) * head_dim;
            int64_t dst = ((int64_t)p * num_kv_heads + h) * head_dim;
            memcpy(out + dst, pool + src, sizeof(uint16_t) * (size_t)head_dim);
        }
    }
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Attention of one request: S queries at positions L-S .. L-1 over L keys. */

typedef struct {
    const uint16_t *q, *k, *v;       /* [S][Hq][d], [L][Hkv][d], [L][Hkv][d] */
    int32_t S, L, Hq, Hkv, d;
    double scale;
    double *out, *lse;               /* [S][Hq][d], [S][Hq] */
    int64_t next_item;               /* work counter (under the mutex) */
    pthread_mutex_t mu;
} attn_job;

/* One (query i, q-head h) output, straight from the definition. */
static void attend_one(const attn_job *J, int32_t i, int32_t h, double *scores) {
    const int32_t g = J->Hq / J->Hkv;
    const int32_t kh = h / g;                  /* kv head serving q head h */
    const int32_t pos = J->L - J->S + i;       /* absolute position of the query */
    const uint16_t *qrow = J->q + ((int64_t)i * J->Hq + h) * J->d;
    double m = -INFINITY;
    for (int32_t j = 0; j <= pos; ++j) {       /* causal: keys 0..pos */
        const uint16_t *krow = J->k + ((int64_t)j * J->Hkv + kh) * J->d;
        double dot = 0.0;
        for (int32_t c = 0; c < J->d; ++c)
            dot += bf16_to_double(qrow[c]) * bf16_to_double(krow[c]);
        scores[j] = J->scale * dot;
        if (scores[j] > m) m = scores[j];
    }
    double denom = 0.0;
    for (int32_t j = 0; j <= pos; ++j) {
        scores[j] = exp(scores[j] - m);        /* unnormalised weight */
        denom += scores[j];
    }
    double *o = J->out + ((int64_t)i * J->Hq + h) * J->d;
    for (int32_t c = 0; c < J->d; ++c) o[c] = 0.0;
    for (int32_t j = 0; j <= pos; ++j) {
        const uint16_t *vrow = J->v + ((int64_t)j * J->Hkv + kh) * J->d;
        for (int32_t c = 0; c < J->d; ++c) o[c] += scores[j] * bf16_to_double(vrow[c]);
    }
    for (int32_t c = 0; c < J->d; ++c) o[c] /= denom;
    if (J->lse) J->lse[(int64_t)i * J->Hq + h] = m + log(denom);
}

static void *attn_worker(void *arg) {
    attn_job *J = (attn_job *)arg;
    double *scores = (double *)malloc(sizeof(double) * (size_t)(J->L > 0 ? J->L : 1));
    const int64_t total = (int64_t)J->S * J->Hq;
    for (;;) {
        pthread_mutex_lock(&J->mu);
        int64_t it = J->next_item++;
        pthread_mutex_unlock(&J->mu);
        if (it >= total) break;
        attend_one(J, (int32_t)(it / J->Hq), (int32_t)(it % J->Hq), scores);
    }
    free(scores);
    return NULL;
}

/*
 * Attention for one request with contiguous K/V.  Query i (0 <= i < S) sits at
 * absolute position L - S + i and sees keys 0 .. L - S + i.  Returns 0, or -1
 * on bad shapes (S > L, Hq not a multiple of Hkv).
 */
int oracle_attention(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                     int32_t S, int32_t L, int32_t Hq, int32_t Hkv, int32_t d,
                     double scale, double *out, double *lse, int32_t num_threads) {
    if (S < 0 || S > L || Hkv <= 0 || Hq % Hkv != 0 || d <= 0) return -1;
    if (S == 0) return 0;
    attn_job J;
    J.q = q; J.k = k; J.v = v; J.S = S; J.L = L; J.Hq = Hq; J.Hkv = Hkv; J.d = d;
    J.scale = scale; J.out = out; J.lse = lse; J.next_item = 0;
    pthread_mutex_init(&J.mu, NULL);
    if (num_threads < 1) num_threads = 1;
    if (num_threads > 256) num_threads = 256;
    pthread_t th[256];
    for (int32_t i = 1; i < num_threads; ++i) pthread_create(&th[i], NULL, attn_worker, &J);
    attn_worker(&J);
    for (int32_t i = 1; i < num_threads; ++i) pthread_join(th[i], NULL);
    pthread_mutex_destroy(&J.mu);
    return 0;
}
