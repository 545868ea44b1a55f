// Sanitizer harness of the host planner (test infrastructure, built by
// tests/test_planner_sanitized.py with -fsanitize=address,undefined): random
// ragged layouts through plan_chunks, shard_range, onchip_grid and
// plan_onchip.  Each result is checked against the rule its declaration
// states; the sanitizers abort on any out-of-bounds access, leak or
// undefined behaviour.  Exit status 0: every layout passed.
#include <cstdio>
#include <cstdlib>
#include <vector>

#include "lamb_internal.h"
#include "lamb_onchip.h"

using namespace lamb;

namespace {

uint64_t g_state = 0x2545F4914F6CDD1Dull;

uint64_t next_u64() {   // splitmix64
  uint64_t z = (g_state += 0x9E3779B97F4A7C15ull);
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

int64_t below(int64_t n) { return (int64_t)(next_u64() % (uint64_t)n); }

// empty, tiny, around a row boundary, medium, large, near the row limit of
// a resident tensor
int64_t pick_size() {
  switch (below(7)) {
    case 0: return below(5);
    case 1: return below(300);
    case 2: { const int64_t r = kOcRow * (1 + below(400)) + below(3) - 1;
              return r < 0 ? 0 : r; }
    case 3: return 1000 + below(70000);
    case 4: return below(400000);
    case 5: return kOcRow * (kOcMaxTensorRows - 50 + below(100)) + below(2);
    default: return kOcRow * (1 + below(2000));
  }
}

// A layout in one of three regimes: sizes drawn from every class above;
// mostly tiny tensors (bias and norm vectors) with a few large ones, as in a
// convolutional network; or large matrices alternating with short vectors,
// as in a transformer.
std::vector<int64_t> pick_layout() {
  const int64_t n = 1 + below(120);
  std::vector<int64_t> sizes((size_t)n);
  const int64_t regime = below(3);
  for (int64_t k = 0; k < n; ++k) {
    if (regime == 0)
      sizes[(size_t)k] = pick_size();
    else if (regime == 1)
      sizes[(size_t)k] = below(10) ? 1 + below(3 * kOcRow) : pick_size();
    else
      sizes[(size_t)k] = k % 3 == 2 ? kOcRow * (8 + below(64)) * 8
                                    : 1 + below(8 * kOcRow);
  }
  return sizes;
}

int g_iter = 0;

#define CHECK(c)                                                        \
  do {                                                                  \
    if (!(c)) {                                                         \
      std::fprintf(stderr, "layout %d: check failed: %s (line %d)\n",   \
                   g_iter, #c, __LINE__);                               \
      return false;                                                     \
    }                                                                   \
  } while (0)

bool check_chunks(const std::vector<int64_t>& sizes,
                  const std::vector<uint8_t>& mask) {
  const int32_t n = (int32_t)sizes.size();
  const int32_t chunk = 1024 << below(5);   // 1024 .. 16384
  const int64_t tail =
      chunk >= kTailChunk && below(2) ? below(100000) : 0;
  const int32_t tail_chunk = tail ? kTailChunk : 0;
  char err[256];
  int64_t count = -1;
  CHECK(plan_chunks(sizes.data(), n, chunk, nullptr, 0, &count, nullptr,
                    mask.data(), err, sizeof err, tail, tail_chunk) == 0);
  std::vector<ChunkDesc> chunks((size_t)count + 1);
  std::vector<TensorDesc> td((size_t)n);
  int64_t count2 = -1;
  CHECK(plan_chunks(sizes.data(), n, chunk, chunks.data(), count, &count2,
                    td.data(), mask.data(), err, sizeof err, tail,
                    tail_chunk) == 0);
  CHECK(count2 == count);
  if (count > 0) {   // one short of the count is refused
    CHECK(plan_chunks(sizes.data(), n, chunk, chunks.data(), count - 1,
                      &count2, nullptr, nullptr, err, sizeof err, tail,
                      tail_chunk) != 0);
    CHECK(count2 == count);
    CHECK(plan_chunks(sizes.data(), n, chunk, chunks.data(), count, &count2,
                      td.data(), mask.data(), err, sizeof err, tail,
                      tail_chunk) == 0);
  }
  int64_t c = 0, total = 0;
  for (int32_t k = 0; k < n; ++k) {
    CHECK(td[k].numel == sizes[k]);
    CHECK(td[k].first_chunk == c);
    CHECK(td[k].decay == (mask[k] ? 1.0f : 0.0f));
    int64_t off = 0;
    for (int32_t j = 0; j < td[k].n_chunks; ++j, ++c) {
      const ChunkDesc& d = chunks[(size_t)c];
      CHECK(d.tensor == k && d.offset == off);
      CHECK(d.len >= 1 && d.len <= chunk && d.offset % 1024 == 0);
      off += d.len;
    }
    CHECK(off == sizes[k]);
    total += sizes[k];
  }
  CHECK(c == count);

  // shard ranges: contiguous, covering, split at floor(total r / W)
  const int32_t world = 1 + (int32_t)below(9);
  int64_t prev_end = 0;
  for (int32_t r = 0; r < world; ++r) {
    int64_t b = -1, e = -1;
    shard_range(chunks.data(), count, world, r, &b, &e);
    CHECK(b == prev_end && b <= e && e <= count);
    prev_end = e;
    const int64_t lo = (int64_t)((__int128)total * r / world);
    const int64_t hi = (int64_t)((__int128)total * (r + 1) / world);
    int64_t pos = 0;
    for (int64_t i = 0; i < count; ++i) {
      const bool in = pos >= lo && pos < hi;
      CHECK(in == (i >= b && i < e));
      pos += chunks[(size_t)i].len;
    }
  }
  CHECK(prev_end == count);
  return true;
}

bool check_rounds(const std::vector<int64_t>& sizes,
                  const std::vector<uint8_t>& mask) {
  const int32_t n = (int32_t)sizes.size();
  const int32_t grid = 1 + (int32_t)below(below(4) ? 160 : 600);
  const int32_t rpc = 1 + (int32_t)below(kOcMaxRows);
  int64_t rows_total = 0;
  for (int64_t s : sizes) rows_total += (s + kOcRow - 1) / kOcRow;
  const int32_t sms = 1 + (int32_t)below(200);
  const int32_t g2 = onchip_grid(rows_total, sms);
  CHECK(g2 >= 1 && g2 <= sms);

  char err[256];
  int32_t n_rounds = -1;
  int64_t n_slots = -1;
  std::vector<OcSlice> slices;
  std::vector<OcPiece> pieces;
  std::vector<int32_t> streamed;
  CHECK(plan_onchip(sizes.data(), n, mask.data(), grid, rpc, &n_rounds,
                    &slices, &pieces, &streamed, &n_slots, err,
                    sizeof err) == 0);
  CHECK(n_slots == (int64_t)pieces.size());
  CHECK(slices.size() == (size_t)n_rounds * (size_t)grid);
  const int64_t cap = (int64_t)grid * rpc;
  // streamed: exactly the tensors too large for a round, in order
  size_t si = 0;
  std::vector<int64_t> covered((size_t)n, 0);
  std::vector<int32_t> round_of((size_t)n, -1);
  for (int32_t k = 0; k < n; ++k) {
    const int64_t r = (sizes[k] + kOcRow - 1) / kOcRow;
    const bool big = r > cap || r > kOcMaxTensorRows;
    if (big) {
      CHECK(si < streamed.size() && streamed[si] == k);
      ++si;
    }
  }
  CHECK(si == streamed.size());
  for (int32_t rd = 0; rd < n_rounds; ++rd) {
    for (int32_t c = 0; c < grid; ++c) {
      const OcSlice& sl = slices[(size_t)rd * grid + c];
      CHECK(sl.n_pieces >= 0 && sl.n_pieces <= kOcMaxPieces);
      CHECK(sl.n_rows >= 0 && sl.n_rows <= rpc);
      CHECK(sl.piece_begin >= 0 &&
            (size_t)sl.piece_begin + sl.n_pieces <= pieces.size());
      if (c + 1 < grid)
        CHECK(slices[(size_t)rd * grid + c + 1].piece_begin ==
              sl.piece_begin + sl.n_pieces);
      int32_t row = 0;
      for (int32_t j = 0; j < sl.n_pieces; ++j) {
        const OcPiece& p = pieces[(size_t)sl.piece_begin + j];
        CHECK(p.tensor >= 0 && p.tensor < n);
        CHECK(p.first_row == row && p.n_rows >= 1);
        row += p.n_rows;
        CHECK(p.offset % kOcRow == 0 && p.offset == covered[p.tensor]);
        // the kernel's row record holds a row's index inside its tensor in
        // 16 bits, its element count in 8 and its piece in 4
        CHECK(p.offset / kOcRow + p.n_rows <= 65536);
        CHECK(j < 16 && kOcRow < 256);
        CHECK(p.len >= 1 && p.len <= (int64_t)p.n_rows * kOcRow &&
              p.len > (int64_t)(p.n_rows - 1) * kOcRow);
        covered[p.tensor] += p.len;
        CHECK(round_of[p.tensor] == -1 || round_of[p.tensor] == rd);
        round_of[p.tensor] = rd;
        CHECK(p.slot == sl.piece_begin + j);
        CHECK(p.t_slot <= p.slot && p.slot < p.t_slot + p.t_nslots);
        CHECK(((p.flags & kOcExport) != 0) == (p.slot == p.t_slot));
        CHECK(p.decay == (mask[p.tensor] ? 1.0f : 0.0f));
      }
      CHECK(row == sl.n_rows);
    }
  }
  for (int32_t k = 0; k < n; ++k) {
    const int64_t r = (sizes[k] + kOcRow - 1) / kOcRow;
    const bool big = r > cap || r > kOcMaxTensorRows;
    CHECK(covered[k] == (big ? 0 : sizes[k]));
  }
  return true;
}

}  // namespace

int main(int argc, char** argv) {
  const int layouts = argc > 1 ? std::atoi(argv[1]) : 2000;
  for (g_iter = 0; g_iter < layouts; ++g_iter) {
    const std::vector<int64_t> sizes = pick_layout();
    std::vector<uint8_t> mask(sizes.size());
    for (auto& b : mask) b = (uint8_t)(next_u64() & 1u);
    if (!check_chunks(sizes, mask) || !check_rounds(sizes, mask)) return 1;
  }
  std::printf("%d layouts\n", layouts);
  return 0;
}
