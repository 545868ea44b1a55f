// Plan tables and launcher of the on-chip step (lamb_onchip.cu, planned by
// planner.cpp).  Kept apart from lamb_internal.h so that the two-pass
// kernels do not depend on it.
//
// HBM layout added to a plan with LAMB_ALGO_ON_CHIP (same arena, after the
// two-pass tables, each piece 256-byte aligned):
//   ChunkDesc  oc_chunks[]    the streamed tensors' chunk table (two-pass)
//   TensorDesc oc_tensors[]   their tensor table
//   OcSlice    slices[n_rounds][grid]   8 B  one CTA's part of a round
//   OcPiece    pieces[]                80 B  rows of one tensor in one CTA
//   uint64     slots[n_pieces][2]      16 B  per piece: two-float sums of
//                                             w^2 and u^2, tagged by launch
//   uint32     bar[kBarWords]                launch epoch, finish ticket,
//                                             abort word
#pragma once
#include <stdint.h>

#include <vector>

#include "lamb_internal.h"

namespace lamb {

// ---------------------------------------------------------------------------
// On-chip single-touch step: one cooperative launch per step,
// one CTA per SM.  The tensors are cut into rounds: runs of whole tensors whose
// elements fit the grid's shared memory.  Every CTA owns a fixed slice of a
// round's rows (kOcRow elements each), keeps w and the update direction of its
// rows in shared memory while the CTAs exchange their partial sums, and writes
// the new w from there.  A tensor too large for one round is "streamed": the two-pass kernels
// take it, over a chunk table of such tensors only, before the on-chip launch.
// ---------------------------------------------------------------------------
constexpr int kOcThreads = 768;
constexpr int kOcWarps = kOcThreads / 32;
constexpr int kOcRow = 128;          // elements per row: one float4 per lane
constexpr int kOcMaxPieces = 16;     // pieces per CTA and round
constexpr int kOcMaxRows = 224;      // rows per CTA (the plan may use fewer)
constexpr int kOcMaxTensorRows = 65535;   // rows of a resident tensor (the
                                          // kernel's row records hold 16 bits)
constexpr int kOcRowBytes = 2 * kOcRow * 4;   // w and u of a row, fp32

enum : uint32_t { kOcVec = 1u,       // arrays aligned for 4-element access
                  kOcExport = 2u };  // this piece's CTA writes rho_k, norms

// A piece: the rows of one tensor inside one CTA's slice of a round.  Pointers
// are filled in by bind.
struct __align__(16) OcPiece {
  float* w;
  const void* g;
  float* m;
  float* v;
  void* copy;
  int64_t offset;     // element of the tensor at the piece's first row
  int32_t len;        // elements of the piece
  int32_t tensor;
  int32_t slot;       // this piece's partial-sum slot
  int32_t t_slot;     // the tensor's first slot
  int32_t t_nslots;   // the tensor's slots, combined in this order
  int16_t first_row;  // CTA-local row where the piece starts
  int16_t n_rows;
  float decay;        // 1.0f: weight decay applies
  uint32_t flags;     // kOcVec | kOcExport
};
static_assert(sizeof(OcPiece) == 80, "OcPiece layout");

struct __align__(8) OcSlice {   // one CTA's part of a resident round
  int32_t piece_begin;
  int16_t n_pieces;
  int16_t n_rows;
};

// Words of the plan's launch block (uint32 indices; each on its own 128-byte
// line)
constexpr int kBarEpoch = 0;     // launches of the plan that finished
constexpr int kBarTicket = 32;   // CTAs of the current launch that finished
constexpr int kBarAbort = 64;    // a wait gave up: the plan is unusable
constexpr int kBarWords = 96;

struct OcParams {
  const OcSlice* slices;  // [n_rounds][grid]
  const OcPiece* pieces;
  uint64_t* slots;        // per piece, 2 words: sum w^2 and sum u^2, each
                          // a two-float value with the launch's tag
  uint32_t* bar;          // kBarWords words, see kBar*
  int32_t n_rounds;
  int32_t extra_arrivals; // > 0 only in tests of the give-up path: the
                          // CTAs wait for a launch tag nobody writes
  int64_t wait_limit_ns;  // a wait for partial sums gives up after this long
};

// Host planner of the on-chip step (planner.cpp).  grid CTAs, rows_per_cta
// rows of shared memory each.  Pieces come back without pointers; streamed
// receives the tensors too large for a round, in order.
int plan_onchip(const int64_t* sizes, int32_t n, const uint8_t* decay_mask,
                int32_t grid, int32_t rows_per_cta, int32_t* n_rounds,
                std::vector<OcSlice>* slices, std::vector<OcPiece>* pieces,
                std::vector<int32_t>* streamed, int64_t* n_slots, char* err,
                int errlen);
// CTAs of the on-chip grid for a layout of total_rows rows (at least 32 rows
// per CTA, at most num_sms).
int32_t onchip_grid(int64_t total_rows, int32_t num_sms);

// Launcher (lamb_onchip.cu): opt 0 LAMB, 1 N-LAMB, 2 NN-LAMB, 3 LARS.
int launch_onchip(const StepParams& p, const OcParams& q, int opt,
                  int grad_bf16, int copy_bf16, int grid, int rows_per_cta,
                  void* stream);
// Rows of shared memory a CTA can hold on `device`, after the kernels' static
// shared memory; also raises the kernels' dynamic shared-memory limit.
int onchip_prepare(int device, int* rows_per_cta);

}  // namespace lamb
