// lora_dispatch.cpp -- adapter-first, length-bucketed dispatch of a mixed
// multi-adapter request (Sec. 5.6): the request's items are grouped by LoRA
// adapter, each group is cut into length buckets, each bucket runs as one
// batch (or several, at most max_batch items each), and the caller restores
// request order from the returned permutation.
//
// Order of the batches: adapters in the order of their first item, buckets of
// one adapter from the shortest range up, items of one bucket in request
// order.  Implemented as one stable sort of the item indices by the key
// (adapter rank, bucket) followed by a walk that cuts batches where the key
// changes or a batch is full.  Host only, no state.
#include "../../include/pkv.h"

#include <algorithm>
#include <cstdint>
#include <string>
#include <unordered_map>
#include <vector>

#include "pkv_internal.h"

namespace {

int fail(int code, const std::string &msg) { return pkv::set_last_error(code, msg.c_str()); }

}  // namespace

extern "C" int pkv_lora_dispatch(const int32_t *adapter_id, const int32_t *prompt_len, int32_t n,
                                 const int32_t *bucket_edges, int32_t n_edges, int32_t max_batch,
                                 int32_t *order_out, int32_t *batch_start_out,
                                 int32_t *batch_adapter_out, int32_t *batch_bucket_out,
                                 int32_t *n_batches_out) {
    if (n < 0 || n_edges < 0 || max_batch < 0 || !n_batches_out || !batch_start_out ||
        (n > 0 && (!adapter_id || !prompt_len || !order_out || !batch_adapter_out ||
                   !batch_bucket_out)) ||
        (n_edges > 0 && !bucket_edges))
        return fail(PKV_ERR_INVALID_ARG, "bad arguments");
    for (int32_t j = 1; j < n_edges; ++j)
        if (bucket_edges[j] <= bucket_edges[j - 1])
            return fail(PKV_ERR_INVALID_ARG, "bucket edges must be strictly ascending");
    // rank of each adapter = position of its first item among the adapters
    std::unordered_map<int32_t, int32_t> rank_of;
    std::vector<int64_t> key(n);
    for (int32_t i = 0; i < n; ++i) {
        if (adapter_id[i] < 0 || prompt_len[i] < 0)
            return fail(PKV_ERR_INVALID_ARG, "item " + std::to_string(i) +
                                                  ": negative adapter id or prompt length");
        const int32_t rank = rank_of.emplace(adapter_id[i], (int32_t)rank_of.size()).first->second;
        // bucket = number of edges at or below the length
        const int32_t bucket =
            (int32_t)(std::upper_bound(bucket_edges, bucket_edges + n_edges, prompt_len[i]) - bucket_edges);
        key[i] = (int64_t)rank * ((int64_t)n_edges + 1) + bucket;
    }
    std::vector<int32_t> idx(n);
    for (int32_t i = 0; i < n; ++i) idx[i] = i;
    std::stable_sort(idx.begin(), idx.end(), [&](int32_t a, int32_t b) { return key[a] < key[b]; });
    int32_t nb = 0;
    batch_start_out[0] = 0;
    for (int32_t k = 0; k < n; ++k) {
        const int32_t i = idx[k];
        order_out[k] = i;
        const bool new_batch = k == 0 || key[i] != key[idx[k - 1]] ||
                               (max_batch > 0 && k - batch_start_out[nb - 1] == max_batch);
        if (new_batch) {
            if (nb > 0) batch_start_out[nb] = k;
            batch_adapter_out[nb] = adapter_id[i];
            batch_bucket_out[nb] = (int32_t)(key[i] % ((int64_t)n_edges + 1));
            ++nb;
        }
    }
    batch_start_out[nb] = n;
    *n_batches_out = nb;
    return PKV_OK;
}
