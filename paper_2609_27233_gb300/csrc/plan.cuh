// Span metadata shared by rollback and prompt compaction (step "a1"):
// per span its compressed index and the removed-position count, per sequence
// its compressed length, and prefix sums over sequences.
//
// For sorted, non-overlapping spans (s_i, k_i) of one sequence,
//   R_i   = sum_{i' < i} (k_i' - 1)        removed before span i
//   n_i   = s_i - R_i                      compressed index of span i's unit
//   r_i   = R_i + (k_i - 1)                removed up to the end of span i
// and a kept position t after span i moves to t - r_i (App. J.4:
// pi(t) = t - r(t)).  A compressed index j with largest n_i <= j is span i's
// unit when j == n_i, otherwise the kept position j + r_i.
#pragma once

#include "common.cuh"

namespace umim {

struct PlanHeader {
  int32_t status;       // status word used when the caller passes no dev_status
  int32_t epoch;        // call counter
  int32_t ticket;       // rollback: set when a mover gave up waiting
  int32_t done_ctas;    // rollback CTAs that finished
  int32_t total_units;  // rollback units this call (0 when skipped)
  int32_t blocks_done;  // plan blocks that finished
  int32_t error;        // OR of plan errors this call
  int32_t skip;         // 1: the call found invalid input, write nothing
  int32_t total_rows;   // sum of compressed lengths
  int32_t max_dest;     // largest number of compacted pages of one sequence
  int32_t n_active;     // sequences with compacted pages to write (rollback)
  int32_t pad[53];      // header is 256 bytes
};
static_assert(sizeof(PlanHeader) == 256, "header size");

struct PlanArrays {
  PlanHeader *hdr;
  int32_t *new_idx;     // [S]   n_i
  int32_t *r_incl;      // [S]   r_i
  int32_t *seq_L;       // [B]
  int32_t *seq_Lp;      // [B]
  int32_t *first_page;  // [B]   first compacted page (rollback)
  int32_t *n_dest;      // [B]   compacted pages written per lane (rollback)
  int32_t *active;      // [B]   the sequences with n_dest > 0, in order (rollback)
  int32_t *unit_base;   // [B+1] rollback units, prefix
  int32_t *row_base;    // [B+1] compressed rows, prefix (cu_seqlens)
  int32_t *freed_base;  // [B+1] released pages, prefix
  int32_t *flags;       // end of the plan: the caller's own data follows
};

// Bytes of the plan part of a workspace, 256-B aligned pieces.
inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

inline size_t plan_bytes(int B, int S) {
  size_t b = align256(sizeof(PlanHeader));
  b += 2 * align256(sizeof(int32_t) * (size_t)(S > 0 ? S : 1));
  b += 5 * align256(sizeof(int32_t) * (size_t)(B > 0 ? B : 1));
  b += 3 * align256(sizeof(int32_t) * (size_t)(B + 1));
  return b;
}

inline PlanArrays plan_carve(void *ws, int B, int S) {
  char *p = static_cast<char *>(ws);
  PlanArrays a;
  auto take = [&](size_t n) {
    char *r = p;
    p += align256(n);
    return r;
  };
  a.hdr = reinterpret_cast<PlanHeader *>(take(sizeof(PlanHeader)));
  const size_t s4 = sizeof(int32_t) * (size_t)(S > 0 ? S : 1);
  const size_t b4 = sizeof(int32_t) * (size_t)(B > 0 ? B : 1);
  const size_t b14 = sizeof(int32_t) * (size_t)(B + 1);
  a.new_idx = reinterpret_cast<int32_t *>(take(s4));
  a.r_incl = reinterpret_cast<int32_t *>(take(s4));
  a.seq_L = reinterpret_cast<int32_t *>(take(b4));
  a.seq_Lp = reinterpret_cast<int32_t *>(take(b4));
  a.first_page = reinterpret_cast<int32_t *>(take(b4));
  a.n_dest = reinterpret_cast<int32_t *>(take(b4));
  a.active = reinterpret_cast<int32_t *>(take(b4));
  a.unit_base = reinterpret_cast<int32_t *>(take(b14));
  a.row_base = reinterpret_cast<int32_t *>(take(b14));
  a.freed_base = reinterpret_cast<int32_t *>(take(b14));
  a.flags = reinterpret_cast<int32_t *>(p);
  return a;
}

struct PlanArgs {
  const int32_t *seq_lens;   // [B] or nullptr: every sequence has fixed_len
  int32_t fixed_len;
  const int32_t *span_offsets;
  const int32_t *span_start;
  const int32_t *span_len;
  int32_t B, S;
  int32_t max_span_len;      // 0: unbounded
  // rollback only (block_table == nullptr for compaction)
  const int32_t *block_table;
  int32_t max_pages, n_pages;
  int32_t n_lanes;           // units per compacted page (layers x head groups)
  int32_t *status;           // resolved status word
  int32_t *cu_seqlens_out;   // compaction: [B+1] or nullptr
};

// Launches the plan kernel (B blocks; the last block to finish does the
// prefix sums over sequences and resets the per-call counters).
cudaError_t launch_span_plan(const PlanArgs &args, const PlanArrays &arr, cudaStream_t stream);

}  // namespace umim
