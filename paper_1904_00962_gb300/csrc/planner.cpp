// Host planner: cuts a ragged list of tensors into chunks.
//
// Every tensor k of d_k elements becomes chunks of C elements (the last one
// ragged), in tensor order; within tail_elems of either end of the layout
// (the tensors laid end to end) the chunks are tail_chunk elements instead,
// so the last chunks a pass draws are short and the grid finishes together.  A chunk is the
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
#include "lamb_onchip.h"

namespace lamb {

int plan_chunks(const int64_t* sizes, int32_t n, int32_t chunk_elems,
                ChunkDesc* chunks, int64_t capacity, int64_t* n_chunks,
                TensorDesc* tensors, const uint8_t* decay_mask, char* err,
                int errlen, int64_t tail_elems, int32_t tail_chunk) {
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
  if (tail_elems < 0 || (tail_elems > 0 &&
                         (tail_chunk < 1024 || tail_chunk > chunk_elems ||
                          tail_chunk % 1024))) {
    snprintf(err, errlen, "bad tail: %lld elements in chunks of %d",
             (long long)tail_elems, tail_chunk);
    return 1;
  }
  const int64_t kMaxTotal = int64_t(1) << 62;
  int64_t total = 0;
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
  }
  int64_t count = 0, pos = 0;   // pos: first element of tensor k in the layout
  for (int32_t k = 0; k < n; ++k) {
    const int64_t d = sizes[k];
    const int64_t first = count;
    for (int64_t j = 0; j < d;) {
      // small chunks where the layout starts and ends: the last chunks pass 1
      // draws and (in reverse) pass 2 draws
      const int64_t g = pos + j;
      const int64_t size = (tail_elems > 0 &&
                            (g < tail_elems ||
                             g + chunk_elems > total - tail_elems))
                               ? tail_chunk : chunk_elems;
      const int64_t len = d - j < size ? d - j : size;
      if (count >= kMaxChunks) {
        snprintf(err, errlen, "more than 2^30 chunks; raise chunk_elems");
        return 1;
      }
      if (chunks && count < capacity) {
        chunks[count].offset = j;
        chunks[count].tensor = k;
        chunks[count].len = (int32_t)len;
      }
      ++count;
      j += len;
    }
    if (tensors) {
      tensors[k].numel = d;
      tensors[k].first_chunk = (int32_t)first;
      tensors[k].n_chunks = (int32_t)(count - first);
      tensors[k].decay = (decay_mask == nullptr || decay_mask[k]) ? 1.0f : 0.0f;
      std::memset(tensors[k].pad, 0, sizeof(tensors[k].pad));
    }
    pos += d;
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
// Rounds of the on-chip single-touch step.
//
// A tensor of d elements takes ceil(d / kOcRow) rows.  Tensors are taken in
// order; a run of consecutive tensors forms a round as long as its rows can be
// dealt to the grid's CTAs with at most rows_per_cta rows and kOcMaxPieces
// pieces per CTA.  A tensor with more rows than the whole grid holds is
// "streamed" (the two-pass kernels take it) and belongs to no round.
//
// A round is dealt in order: CTA 0 takes rows until it holds S rows or
// kOcMaxPieces pieces, then CTA 1, and so on, cutting a tensor only at a row
// boundary, so every piece starts at a multiple of kOcRow elements inside its
// tensor.  S is the smallest per-CTA row count (at least the even share) with
// which the round fits the grid.  The pieces of a tensor are therefore
// consecutive, and so are their partial-sum slots.
// ---------------------------------------------------------------------------
namespace lamb {
namespace {

// Greedy deal of `rows` (one entry per tensor of the round) with S rows and
// kOcMaxPieces pieces per CTA; returns the CTAs used.
int64_t deal_ctas(const std::vector<int64_t>& rows, int64_t S) {
  int64_t cta = 0, used = 0, np = 0;
  for (int64_t r : rows) {
    while (r > 0) {
      if (used == S || np == kOcMaxPieces) {
        ++cta;
        used = 0;
        np = 0;
      }
      const int64_t take = r < S - used ? r : S - used;
      used += take;
      ++np;
      r -= take;
    }
  }
  return used || np ? cta + 1 : cta;
}

}  // namespace

int32_t onchip_grid(int64_t total_rows, int32_t num_sms) {
  int64_t g = (total_rows + 31) / 32;
  if (g > num_sms) g = num_sms;
  if (g < 1) g = 1;
  return (int32_t)g;
}

int plan_onchip(const int64_t* sizes, int32_t n, const uint8_t* decay_mask,
                int32_t grid, int32_t rows_per_cta, int32_t* n_rounds,
                std::vector<OcSlice>* slices, std::vector<OcPiece>* pieces,
                std::vector<int32_t>* streamed, int64_t* n_slots, char* err,
                int errlen) {
  if (grid < 1 || rows_per_cta < 1 || rows_per_cta > kOcMaxRows) {
    snprintf(err, errlen, "on-chip plan: bad grid %d or rows per CTA %d",
             grid, rows_per_cta);
    return 1;
  }
  slices->clear();
  pieces->clear();
  streamed->clear();
  *n_rounds = 0;
  const int64_t cap = (int64_t)grid * rows_per_cta;
  auto decay_of = [&](int32_t k) {
    return (decay_mask == nullptr || decay_mask[k]) ? 1.0f : 0.0f;
  };
  auto rows_of = [&](int32_t k) { return (sizes[k] + kOcRow - 1) / kOcRow; };

  // one round over the given tensors (in order)
  auto emit_round = [&](const std::vector<int32_t>& members) {
    std::vector<int64_t> rows;
    int64_t total = 0;
    for (int32_t k : members) {
      rows.push_back(rows_of(k));
      total += rows.back();
    }
    // smallest S >= the even share with which the round fits the grid
    int64_t lo = (total + grid - 1) / grid, hi = rows_per_cta;
    if (lo > hi) lo = hi;
    while (lo < hi) {
      const int64_t mid = (lo + hi) / 2;
      if (deal_ctas(rows, mid) <= grid) hi = mid;
      else lo = mid + 1;
    }
    // the full deal (S = rows_per_cta) is known to fit; keep it if the search
    // found nothing smaller that does
    const int64_t S = deal_ctas(rows, lo) <= grid ? lo : rows_per_cta;
    ++*n_rounds;
    const size_t base = slices->size();
    slices->resize(base + (size_t)grid, OcSlice{0, 0, 0});
    int64_t cta = 0, used = 0, np = 0;
    (*slices)[base].piece_begin = (int32_t)pieces->size();
    for (int32_t k : members) {
      int64_t left = rows_of(k), row_in_tensor = 0;
      const size_t first_piece = pieces->size();
      while (left > 0) {
        if (used == S || np == kOcMaxPieces) {
          ++cta;
          used = 0;
          np = 0;
          (*slices)[base + (size_t)cta].piece_begin = (int32_t)pieces->size();
        }
        const int64_t take = left < S - used ? left : S - used;
        OcPiece pc{};
        pc.offset = row_in_tensor * kOcRow;
        const int64_t len = sizes[k] - pc.offset;
        pc.len = (int32_t)(len < take * kOcRow ? len : take * kOcRow);
        pc.tensor = k;
        pc.slot = (int32_t)pieces->size();
        pc.first_row = (int16_t)used;
        pc.n_rows = (int16_t)take;
        pc.decay = decay_of(k);
        pc.flags = pieces->size() == first_piece ? kOcExport : 0u;
        pieces->push_back(pc);
        OcSlice& sl = (*slices)[base + (size_t)cta];
        sl.n_pieces = (int16_t)(sl.n_pieces + 1);
        sl.n_rows = (int16_t)(sl.n_rows + take);
        used += take;
        ++np;
        left -= take;
        row_in_tensor += take;
      }
      for (size_t i = first_piece; i < pieces->size(); ++i) {
        (*pieces)[i].t_slot = (int32_t)first_piece;
        (*pieces)[i].t_nslots = (int32_t)(pieces->size() - first_piece);
      }
    }
    for (int64_t c = cta + 1; c < grid; ++c)
      (*slices)[base + (size_t)c].piece_begin = (int32_t)pieces->size();
  };

  std::vector<int32_t> open;           // tensors of the open round
  int64_t cta = 0, used = 0, np = 0;   // incremental deal, S = rows_per_cta
  auto close = [&]() {
    if (!open.empty()) emit_round(open);
    open.clear();
    cta = used = np = 0;
  };
  // adds r rows to the incremental deal; false if they do not fit
  auto try_add = [&](int64_t r) {
    int64_t c = cta, u = used, p = np;
    while (r > 0) {
      if (u == rows_per_cta || p == kOcMaxPieces) {
        ++c;
        u = 0;
        p = 0;
      }
      if (c >= grid) return false;
      const int64_t take = r < rows_per_cta - u ? r : rows_per_cta - u;
      u += take;
      ++p;
      r -= take;
    }
    cta = c;
    used = u;
    np = p;
    return true;
  };
  for (int32_t k = 0; k < n; ++k) {
    const int64_t r = rows_of(k);
    if (r == 0) continue;         // 0-element tensor: ratio 1, no work
    if (r > cap || r > kOcMaxTensorRows) {   // streamed: the two-pass
                                             // kernels take it
      streamed->push_back(k);
      continue;
    }
    if (!try_add(r)) {
      close();
      try_add(r);
    }
    open.push_back(k);
    if (pieces->size() > (size_t(1) << 30)) {
      snprintf(err, errlen, "on-chip plan: more than 2^30 pieces");
      return 1;
    }
  }
  close();
  *n_slots = (int64_t)pieces->size();
  return 0;
}

}  // namespace lamb

// ---------------------------------------------------------------------------
// Shards of a chunk table (the data-parallel split of the step): rank r of W
// takes the chunks whose first element, counted over the layout, lies in
// [floor(total r / W), floor(total (r + 1) / W)).  Every rank computes the
// same split.
// ---------------------------------------------------------------------------
namespace lamb {

void shard_range(const ChunkDesc* chunks, int64_t n_chunks, int32_t world,
                 int32_t rank, int64_t* begin, int64_t* end) {
  int64_t total = 0;
  for (int64_t c = 0; c < n_chunks; ++c) total += chunks[c].len;
  // split points in elements, rounded to chunk starts
  auto cut = [&](int32_t r) -> int64_t {
    if (r <= 0) return 0;
    if (r >= world) return n_chunks;
    const __int128 target = (__int128)total * r / world;
    int64_t pos = 0;
    for (int64_t c = 0; c < n_chunks; ++c) {
      if (pos >= target) return c;
      pos += chunks[c].len;
    }
    return n_chunks;
  };
  *begin = cut(rank);
  *end = cut(rank + 1);
}

}  // namespace lamb
