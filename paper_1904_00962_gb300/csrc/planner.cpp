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
#include <utility>
#include <vector>

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

// ---------------------------------------------------------------------------
// Schedule of the single-touch step.
//
// Every tensor k of d_k elements becomes ceil(d_k / kFusedChunk) fused
// chunks.  Work items are emitted in this order:
// the pass-1 items of tensor 0, 1, 2, ... in turn; the pass-2 items of a
// tensor whose state fits the L2 budget ("resident") are emitted as one block
// once `lag` further pass-1 items have been emitted after its last pass-1
// item (about one wave of workers, so its norms are usually final when the
// block is reached, while its m, v, w are still in L2); the pass-2 blocks of
// tensors too large for L2 come last.  Every pass-2 item therefore follows
// all pass-1 items of its tensor, which is what makes the kernel
// deadlock-free.
// ---------------------------------------------------------------------------
namespace lamb {

int plan_fused(const int64_t* sizes, int32_t n, const uint8_t* decay_mask,
               int64_t bytes_per_param, int64_t l2_budget, int64_t lag,
               std::vector<FusedChunk>* fchunks,
               std::vector<FusedTensor>* ftensors,
               std::vector<uint32_t>* items, char* err, int errlen) {
  ftensors->assign((size_t)n, FusedTensor{});
  int64_t nf = 0;
  for (int32_t k = 0; k < n; ++k) {
    const int64_t d = sizes[k];
    const int64_t nk = (d + kFusedChunk - 1) / kFusedChunk;
    FusedTensor& t = (*ftensors)[(size_t)k];
    t.numel = d;
    t.first_chunk = (int32_t)nf;
    t.n_chunks = (int32_t)nk;
    t.decay = (decay_mask == nullptr || decay_mask[k]) ? 1.0f : 0.0f;
    t.resident = (d <= l2_budget / bytes_per_param) ? 1u : 0u;
    nf += nk;
    if (nf > (int64_t(1) << 30)) {
      snprintf(err, errlen, "more than 2^30 fused chunks");
      return 1;
    }
  }
  fchunks->resize((size_t)nf);
  for (int32_t k = 0; k < n; ++k) {
    const FusedTensor& t = (*ftensors)[(size_t)k];
    for (int32_t j = 0; j < t.n_chunks; ++j)
      (*fchunks)[(size_t)t.first_chunk + j] = FusedChunk{k, j};
  }
  items->clear();
  items->reserve((size_t)(2 * nf));
  auto emit_pass2 = [&](int32_t k) {
    const FusedTensor& t = (*ftensors)[(size_t)k];
    for (int32_t j = 0; j < t.n_chunks; ++j)
      items->push_back(((uint32_t)(t.first_chunk + j) << 1) | 1u);
  };
  std::vector<std::pair<int64_t, int32_t>> pending;  // (release point, k)
  size_t head = 0;
  std::vector<int32_t> tail;
  int64_t p1 = 0;
  for (int32_t k = 0; k < n; ++k) {
    const FusedTensor& t = (*ftensors)[(size_t)k];
    for (int32_t j = 0; j < t.n_chunks; ++j) {
      items->push_back((uint32_t)(t.first_chunk + j) << 1);
      ++p1;
      while (head < pending.size() && pending[head].first <= p1)
        emit_pass2(pending[head++].second);
    }
    if (t.n_chunks == 0) continue;
    if (t.resident)
      pending.emplace_back(p1 + lag, k);
    else
      tail.push_back(k);
  }
  while (head < pending.size()) emit_pass2(pending[head++].second);
  for (int32_t k : tail) emit_pass2(k);
  return 0;
}

}  // namespace lamb
