// Host planner: cuts a ragged list of tensors into fixed-size chunks.
//
// Every tensor k of d_k elements becomes ceil(d_k / C) chunks (tensor k,
// offset j*C, length min(C, d_k - j*C)), in tensor order.  A chunk is the
// unit of work of one CTA iteration and owns one partial-sum slot, so the
// per-tensor norms of Algorithm 2 (||x^(i)||, ||r^(i) + lambda x^(i)||) are a
// segmented reduction over the chunks of each tensor.  Chunks are handed out
// dynamically on the device, so a 31M-element embedding and hundreds of
// 1024-element LayerNorm vectors share one launch without a tail.
#include <cstdio>
#include <cstring>

#include "lamb_internal.h"

namespace lamb {

int plan_chunks(const int64_t* sizes, int32_t n, int32_t chunk_elems,
                ChunkDesc* chunks, int64_t capacity, int64_t* n_chunks,
                TensorDesc* tensors, const uint8_t* decay_mask, char* err,
                int errlen) {
  if (n < 1) {
    snprintf(err, errlen, "n_tensors must be >= 1 (got %d)", n);
    return 1;
  }
  if (sizes == nullptr) {
    snprintf(err, errlen, "sizes is NULL");
    return 1;
  }
  if (chunk_elems < 1024 || chunk_elems > (1 << 24) || chunk_elems % 1024) {
    snprintf(err, errlen,
             "chunk_elems must be a multiple of 1024 in [1024, 2^24] (got %d)",
             chunk_elems);
    return 1;
  }
  const int64_t kMaxTotal = int64_t(1) << 62;
  int64_t total = 0, count = 0;
  for (int32_t k = 0; k < n; ++k) {
    const int64_t d = sizes[k];
    if (d < 0) {
      snprintf(err, errlen, "sizes[%d] = %lld is negative", k, (long long)d);
      return 1;
    }
    if (d > kMaxTotal - total) {
      snprintf(err, errlen, "total element count exceeds 2^62");
      return 1;
    }
    total += d;
    const int64_t nk = (d + chunk_elems - 1) / chunk_elems;
    if (nk > kMaxChunks - count) {
      snprintf(err, errlen, "more than 2^30 chunks; raise chunk_elems");
      return 1;
    }
    if (tensors) {
      tensors[k].numel = d;
      tensors[k].first_chunk = (int32_t)count;
      tensors[k].n_chunks = (int32_t)nk;
      tensors[k].decay = (decay_mask == nullptr || decay_mask[k]) ? 1.0f : 0.0f;
      std::memset(tensors[k].pad, 0, sizeof(tensors[k].pad));
    }
    for (int64_t j = 0; j < nk; ++j, ++count) {
      if (chunks && count < capacity) {
        const int64_t off = j * chunk_elems;
        const int64_t rem = d - off;
        chunks[count].offset = off;
        chunks[count].tensor = k;
        chunks[count].len = (int32_t)(rem < chunk_elems ? rem : chunk_elems);
      }
    }
  }
  *n_chunks = count;
  if (chunks && count > capacity) {
    snprintf(err, errlen, "capacity %lld < %lld chunks", (long long)capacity,
             (long long)count);
    return 1;
  }
  return 0;
}

}  // namespace lamb
