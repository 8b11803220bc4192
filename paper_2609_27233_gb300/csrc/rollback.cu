// KV-cache rollback and in-place compaction of a paged bf16 cache
// (App. E "Decoding-Time Merging and KV-Cache Update", Fig. 2): each span's
// k stored entries become one surrogate entry and later entries move left.
//
// Work unit = one (layer, K|V, kv-head) 16 x D tile of one compacted page of
// one sequence: its 16 entries j come from kept entries t = j + r >= j or
// from surrogate rows, and it is written to the same physical page that held
// old page j / 16.  Units are numbered row by row (row = compacted page
// index, over the sequences that have pages to write) and dealt round-robin
// to the mover warps of a cooperative grid; each warp loads two units ahead
// of its stores (through shared memory with the copy engine when keys move
// verbatim, through registers when they are re-rotated).  A unit may overwrite its page once every unit that reads
// that old page has its loads landed.  Because j <= t, the readers of old
// page p are the units of the same sequence at compacted rows whose entries
// come from p: at most two rows, both at or before p's own row (a unit reads
// and writes only its own (layer, K|V, head) column, so within p's row the
// reader is the unit itself).  So every unit counts itself into its row's
// "landed" counter when its loads have arrived (release), and waits (acquire,
// bounded) for the counters of its page's reader rows before it stores.
// Every wait is for units numbered before the waiting one, each warp takes
// its units in increasing order and all warps are resident, so the earliest
// unstored unit can always proceed: no deadlock, and no grid-wide barrier.
// One pass: each moved byte is read once and written once.
#include <algorithm>

#include "plan.cuh"

namespace umim {
namespace {

constexpr int kMoveThreads = 256;   // 8 mover warps
constexpr int kMovers = kMoveThreads / 32;
constexpr int64_t kNoWrite = INT64_MIN;

struct MoveArgs {
  uint16_t *pool;
  int32_t n_lanes;
  int32_t n_layers, n_pages, n_kv_heads, head_dim;
  int32_t *block_table;
  int32_t max_pages;
  int32_t *seq_lens;
  const int32_t *span_offsets, *span_start, *span_len;
  const uint16_t *sur_k, *sur_v;
  int32_t *freed_pages;
  int32_t freed_capacity;
  int32_t B;
  int32_t *status;
  const float *rope_inv_freq;   // [rotary_dim / 2] or nullptr: keys move verbatim
  int32_t rotary_dim;
  uint32_t zero;                // always 0 (see red_add_after)
};

// largest i in [lo, hi) with key(i) <= x, or lo - 1
__device__ __forceinline__ int upper_index(const int32_t *key, int lo, int hi, int x) {
  int l = lo, h = hi;
  while (l < h) {
    const int m = (l + h) >> 1;
    if (key[m] <= x) l = m + 1;
    else h = m;
  }
  return l - 1;
}

__device__ __forceinline__ uint4 ld_v4(const uint16_t *p) {
  uint4 v;
  asm volatile("ld.global.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ void st_v4(uint16_t *p, uint4 v) {
  asm volatile("st.global.v4.u32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}

// Adds 1 + (dep & zero) to *p, zero being 0 at run time (a kernel argument,
// so the compiler cannot drop the term): the add depends on `dep`, a fold of
// the unit's loaded data, so it cannot issue before those loads have returned
// their values, and a load that has returned cannot be changed by a store that
// follows the add -- which is all the page's writer relies on.  No release
// fence: this thread's earlier stores (of another unit) need not be visible to
// the waiter, and a fence would stall the warp until they are.
__device__ __forceinline__ void red_add_after(int32_t *p, uint32_t dep, uint32_t zero) {
  const int32_t v = 1 + (int32_t)(dep & zero);
  asm volatile("red.relaxed.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ int32_t ld_relaxed(const int32_t *p) {
  int32_t v;
  asm volatile("ld.relaxed.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Per compacted row (global row index over the active sequences).
struct RowDep {
  int32_t lo, hi;   // reader rows of this row's old page that precede it (lo > hi: none)
  int32_t landed;   // units of this row whose loads have arrived (n_lanes: all)
  int32_t pad;
};

struct PageDesc {
  int64_t *src;    // [rows][16] source row offset within a layer (no head offset), -(i+1) for span i, kNoWrite
  RowDep *dep;     // [rows]
  int32_t *shift;  // [rows][16] r of a moved kept entry (positions removed before it), else 0
};

// Sixteen threads per (sequence, compacted page): where each of its 16
// entries comes from (kNoWrite: the entry does not move), and which
// compacted rows read the old entries of the page.
__global__ void __launch_bounds__(256) rollback_map_kernel(MoveArgs a, PlanArrays arr, PageDesc pd, int D) {
  griddep_wait();
  if (arr.hdr->skip) return;
  const int b = blockIdx.y;
  const int k = blockIdx.x * 16 + (threadIdx.x >> 4);
  const int slot = threadIdx.x & 15;
  const int nd = arr.n_dest[b];
  const bool row_ok = k < nd;
  int64_t src = kNoWrite;
  int32_t shift = 0;
  int rd_lo = INT32_MAX, rd_hi = -1;
  int idx = 0;
  if (row_ok) {
    const int fp = arr.first_page[b];
    const int p = fp + k;
    idx = arr.unit_base[b] / a.n_lanes + k;
    const int lo = a.span_offsets[b], hi = a.span_offsets[b + 1];
    const int32_t *bt = a.block_table + (int64_t)b * a.max_pages;
    const int64_t page_stride = (int64_t)kPageSize * D * a.n_kv_heads * 2;
    const int j = p * kPageSize + slot;
    if (j < arr.seq_Lp[b] && j >= a.span_start[lo]) {
      const int i = upper_index(arr.new_idx, lo, hi, j);
      if (i >= lo) {
        if (arr.new_idx[i] == j) {
          src = -(int64_t)i - 1;
        } else {
          const int t = j + arr.r_incl[i];
          if (t != j && in_bounds(t / kPageSize, a.max_pages, a.status, kSiteRollbackMapTable)) {
            src = (int64_t)bt[t / kPageSize] * page_stride + (t % kPageSize) * D;
            shift = t - j;
          }
        }
      }
    }
    // the old entry t in this slot of page p: the compacted row that reads it
    const int t = j;
    if (t < arr.seq_L[b]) {
      const int i = upper_index(a.span_start, lo, hi, t);
      if (i >= lo && t >= a.span_start[i] + a.span_len[i] && arr.r_incl[i] > 0) {
        rd_lo = rd_hi = (t - arr.r_incl[i]) / kPageSize - fp;
      }
    }
  }
  for (int o = 8; o > 0; o >>= 1) {   // over the row's 16 slots
    rd_lo = min(rd_lo, __shfl_xor_sync(0xffffffffu, rd_lo, o, 16));
    rd_hi = max(rd_hi, __shfl_xor_sync(0xffffffffu, rd_hi, o, 16));
  }
  if (!row_ok) return;
  pd.src[(int64_t)idx * kPageSize + slot] = src;
  pd.shift[(int64_t)idx * kPageSize + slot] = shift;
  if (slot == 0) {
    rd_hi = min(rd_hi, k - 1);   // the row itself reads only its own units' columns
    RowDep d;
    d.lo = rd_lo <= rd_hi ? idx - k + rd_lo : 1;
    d.hi = rd_lo <= rd_hi ? idx - k + rd_hi : 0;
    d.landed = 0;
    d.pad = 0;
    pd.dep[idx] = d;
  }
}

// The last CTA of the move kernel to finish truncates the block tables,
// reports the freed pages and writes the new lengths (every CTA calls this
// once, after its movers are done).
__device__ void finish_rollback(const MoveArgs &a, const PlanArrays &arr, int &s_last) {
  const int tid = threadIdx.x;
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    const int done = atomicAdd(&arr.hdr->done_ctas, 1);
    s_last = (done == (int)gridDim.x - 1);
  }
  __syncthreads();
  if (!s_last || arr.hdr->skip) return;
  __threadfence();
  for (int b = 0; b < a.B; ++b) {
    if (a.span_offsets[b + 1] == a.span_offsets[b]) continue;
    const int L = arr.seq_L[b], Lp = arr.seq_Lp[b];
    const int keep = ceil_div(Lp, kPageSize), had = ceil_div(L, kPageSize);
    const int fb = arr.freed_base[b];
    for (int q = keep + tid; q < had; q += blockDim.x) {
      int32_t *e = a.block_table + (int64_t)b * a.max_pages + q;
      const int idx = fb + (q - keep);
      if (a.freed_pages && idx < a.freed_capacity) a.freed_pages[idx] = *e;
      *e = -1;
    }
    if (tid == 0) a.seq_lens[b] = Lp;
  }
  if (tid == 0 && a.freed_pages) {
    const int n = arr.freed_base[a.B];
    if (n < a.freed_capacity) a.freed_pages[n] = -1;
  }
}

constexpr int kSmemSeqs = 1024;   // active sequences whose plan values a CTA keeps in shared memory
constexpr int kSmemLanes = 1024;  // tile lanes (layer, K|V, head) whose offsets a CTA keeps in shared memory

// Waits until *cnt >= target; false when it gave up (time limit, or another
// warp gave up: *abort != 0).
__device__ __forceinline__ bool wait_landed(const int32_t *cnt, int target, const int32_t *abort) {
  return wait_count_for(cnt, target, abort, kWaitLimitNs);
}

// Mover warps: lane l moves 16-byte chunks c = l + 32 it of a unit, row
// (slot) c / CPR, column c % CPR.  Step: the next unit's loads land and it is
// counted in; this unit waits for its page's readers and is stored; the unit
// after next is loaded into its registers.
template <int D, bool ROPE>
__global__ void __launch_bounds__(kMoveThreads, 2) rollback_move_kernel(MoveArgs a, PlanArrays arr, PageDesc pd) {
  constexpr int CPR = D / 8;                       // 16-byte chunks per row
  constexpr int PER_LANE = kPageSize * CPR / 32;   // 8 (D=128) or 4 (D=64)
  constexpr int SLOT_STEP = 32 / CPR;              // rows advanced per it
  constexpr int kHead = kPageSize * D;             // elements of one (K|V, head) tile
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int nm = gridDim.x * kMovers;
  const int my_col = lane % CPR;
  const int my_slot0 = lane / CPR;
  __shared__ int s_last;
  __shared__ int s_sq[kSmemSeqs], s_nd[kSmemSeqs], s_ub[kSmemSeqs], s_fp[kSmemSeqs];
  // per tile lane tl: its offset within a page (layer, K|V and head), and layer * Hkv + head | K|V << 31
  __shared__ int64_t s_toff[kSmemLanes];
  __shared__ int32_t s_tlh[kSmemLanes];
  __shared__ float s_w[ROPE ? D / 2 : 1];   // RoPE angular frequencies

  if (ROPE)
    for (int i = threadIdx.x; i < a.rotary_dim / 2; i += blockDim.x) s_w[i] = a.rope_inv_freq[i];
  griddep_wait();
  const PlanHeader *hdr = arr.hdr;
  int32_t *abort_flag = &arr.hdr->ticket;
  const int total = hdr->total_units;
  const int Hkv = a.n_kv_heads;
  const int64_t layer_stride = (int64_t)2 * kHead * Hkv * a.n_pages;
  const int kv_stride32 = kHead * Hkv, page_stride32 = 2 * kHead * Hkv;
  // a row holds the units of the sequences that have pages to write
  const int n_active = total > 0 ? hdr->n_active : 0;
  const int row_size = max(1, n_active * a.n_lanes);
  // unit indices fit in 32 bits: batch x max_pages x tile lanes < 2^30 is checked on the host
  const int max_dest = total > 0 ? hdr->max_dest : 0;
  const int n_slots = max_dest * row_size;
  const int n_rows = total / a.n_lanes;   // compacted rows of all sequences (debug checks)

  // plan values of the active sequences (row position order), from shared
  // memory when there are few enough of them
  const bool seq_in_smem = n_active <= kSmemSeqs;
  if (seq_in_smem) {
    for (int j = threadIdx.x; j < n_active; j += blockDim.x) {
      const int b = arr.active[j];
      s_sq[j] = b;
      s_nd[j] = arr.n_dest[b];
      s_ub[j] = arr.unit_base[b] / a.n_lanes;   // the sequence's first row
      s_fp[j] = arr.first_page[b];
    }
  }
  const bool lanes_in_smem = a.n_lanes <= kSmemLanes;
  if (lanes_in_smem) {
    for (int tl = threadIdx.x; tl < a.n_lanes; tl += blockDim.x) {
      const int layer = tl / (2 * Hkv), kv = (tl / Hkv) & 1, h = tl % Hkv;
      s_toff[tl] = layer * layer_stride + (int)(kv * kv_stride32 + h * kHead);
      s_tlh[tl] = (int32_t)((uint32_t)(layer * Hkv + h) | ((uint32_t)kv << 31));
    }
  }
  __syncthreads();
  auto seq_of = [&](int j) { return seq_in_smem ? s_sq[j] : arr.active[j]; };
  auto nd_of = [&](int j) { return seq_in_smem ? s_nd[j] : arr.n_dest[arr.active[j]]; };
  auto row0_of = [&](int j) { return seq_in_smem ? s_ub[j] : arr.unit_base[arr.active[j]] / a.n_lanes; };
  auto fp_of = [&](int j) { return seq_in_smem ? s_fp[j] : arr.first_page[arr.active[j]]; };

  // a unit in registers, with where it goes and what it waits for
  struct Tile {
    uint4 v[PER_LANE];
    uint32_t mask;
    int valid, rot;     // rot: a K tile whose moved entries get re-rotated
    int64_t dst;
    int32_t row, dlo, dhi;
    int32_t seen;       // the reader rows' smallest landed count when the unit was loaded
    int32_t shift;      // lanes < 16: the shift of slot `lane`
  };
  // A unit's descriptors (its 16 sources, its page, its reader rows), read
  // one unit ahead of its data loads so that the two round trips overlap.
  struct Meta {
    int64_t my_src;   // lanes < 16: the source of slot `lane`
    int32_t valid, idx, page, tl;
    int32_t shift;
    RowDep dep;
  };
  // slot i = kk * row_size + j * n_lanes + tl: kk the compacted page row, j the
  // active sequence, tl the tile lane
  auto fetch = [&](int kk, int j, int tl, Meta &m) {
    m.valid = 0;
    if (kk >= max_dest) return;
    if (kk >= nd_of(j)) return;
    const int b = seq_of(j);
    m.valid = 1;
    m.tl = tl;
    m.idx = row0_of(j) + kk;
    if (!in_bounds(m.idx, n_rows, a.status, kSiteRollbackReaderRow)) {
      m.valid = 0;
      return;
    }
    m.my_src = lane < kPageSize ? pd.src[(int64_t)m.idx * kPageSize + lane] : kNoWrite;
    m.page = a.block_table[(int64_t)b * a.max_pages + fp_of(j) + kk];
    m.shift = (ROPE && lane < kPageSize) ? pd.shift[(int64_t)m.idx * kPageSize + lane] : 0;
    m.dep = pd.dep[m.idx];
  };
  auto load = [&](const Meta &m, Tile &t) {
    t.mask = 0;
    t.valid = 0;
    t.rot = 0;
    t.shift = 0;
    t.dst = 0;
    t.row = 0;
    t.dlo = 1;
    t.dhi = 0;
    t.seen = a.n_lanes;
#pragma unroll
    for (int it = 0; it < PER_LANE; ++it) t.v[it] = make_uint4(0, 0, 0, 0);
    if (!m.valid) return;
    const int tl = m.tl;
    int64_t tile;
    int kv, lh;   // lh = layer * Hkv + head
    if (lanes_in_smem) {
      tile = s_toff[tl] + my_col * 8;
      const int32_t e = s_tlh[tl];
      kv = (int)((uint32_t)e >> 31);
      lh = e & 0x7fffffff;
    } else {
      const int layer = tl / (2 * Hkv), h = tl % Hkv;
      kv = (tl / Hkv) & 1;
      lh = layer * Hkv + h;
      tile = layer * layer_stride + (int)(kv * kv_stride32 + h * kHead + my_col * 8);
    }
    const uint16_t *sur = kv ? a.sur_v : a.sur_k;
    t.valid = 1;
    t.row = m.idx;
    t.dst = tile + (int64_t)m.page * page_stride32;
    if (ROPE) {
      t.rot = kv == 0;
      t.shift = m.shift;
    }
#pragma unroll
    for (int it = 0; it < PER_LANE; ++it) {
      const int slot = my_slot0 + it * SLOT_STEP;
      const int64_t src = __shfl_sync(0xffffffffu, m.my_src, slot);
      if (src != kNoWrite) t.mask |= 1u << it;
      if (src >= 0) {
        if (in_bounds(src, (int64_t)a.n_pages * page_stride32, a.status, kSiteRollbackSrc))
          t.v[it] = ld_v4(a.pool + tile + src);
      } else if (src != kNoWrite) {
        const int64_t si = -src - 1;
        if (in_bounds(si, kDebugChecks ? a.span_offsets[a.B] : 0, a.status, kSiteRollbackSurrogate))
          t.v[it] = ld_v4(sur + (si * a.n_layers * Hkv + lh) * D + my_col * 8);
      }
    }
    t.dlo = m.dep.lo;
    t.dhi = m.dep.hi;
    if (!in_bounds(m.page, a.n_pages, a.status, kSiteRollbackDstPage)) t.mask = 0;
    if (t.dlo <= t.dhi && !(in_bounds(t.dlo, n_rows, a.status, kSiteRollbackReaderRow) &&
                            in_bounds(t.dhi, n_rows, a.status, kSiteRollbackReaderRow))) {
      t.dlo = 1;   // no reader row to wait for, so nothing may be stored either
      t.dhi = 0;
      t.mask = 0;
    }
  };
  auto store = [&](const Tile &t) {
#pragma unroll
    for (int it = 0; it < PER_LANE; ++it) {
      const int slot = my_slot0 + it * SLOT_STEP;
      if (t.mask & (1u << it)) st_v4(a.pool + t.dst + slot * D, t.v[it]);
    }
  };
  // the unit's loads have arrived; count it into its row
  auto land_and_count = [&](Tile &t) {
    uint32_t fold = 0;
#pragma unroll
    for (int it = 0; it < PER_LANE; ++it) fold ^= t.v[it].x ^ t.v[it].y ^ t.v[it].z ^ t.v[it].w;
    // every lane's loads have returned once lane 0 holds the fold of all of them
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) fold ^= __shfl_xor_sync(0xffffffffu, fold, o);
    if (t.valid && lane == 0) red_add_after(&pd.dep[t.row].landed, fold, a.zero);
    // the reader rows' counts, read a step before the store so that their
    // latency overlaps this step; a complete count then needs no further wait
    t.seen = a.n_lanes;
    for (int rw = t.dlo; rw <= t.dhi; ++rw) t.seen = min(t.seen, ld_relaxed(&pd.dep[rw].landed));
  };
  // RoPE: a moved key (shift r) is rotated by -r w_m on the pairs (m, m + rotary_dim/2):
  // x' = x cos + y sin, y' = y cos - x sin.  The lane holding chunk c of a slot's
  // row takes its partner chunk from the lane holding c +- rotary_dim/16.  The
  // angle is r w rounded plus its exact rounding error (an fma), the error
  // folded into the sine and cosine to first order; the rounded angle is
  // reduced to [-pi, pi] (Cody and Waite's three-part reduction) for the
  // hardware sine and cosine, whose error there (about 2^-21) is far below
  // the bf16 result's resolution.
  auto rotate = [&](Tile &t) {
    if (!ROPE || !t.rot) return;
    const int hc = a.rotary_dim / 16;   // 16-byte chunks in each half of the rotated columns
    const bool in_x = my_col < hc, in_y = my_col >= hc && my_col < 2 * hc;
    const int partner = lane - my_col + (in_x ? my_col + hc : (in_y ? my_col - hc : my_col));
    const int m0 = (in_x || in_y) ? 8 * (in_x ? my_col : my_col - hc) : 0;   // lanes past rotary_dim: unused
    const int mine = in_y ? 1 : 0;   // of each element pair (2q, 2q+1) this lane evaluates element 2q + mine
#pragma unroll
    for (int it = 0; it < PER_LANE; ++it) {
      const int slot = my_slot0 + it * SLOT_STEP;
      const float rf = (float)__shfl_sync(0xffffffffu, t.shift, slot);   // 0: the identity (same bytes)
      uint4 pv;
      pv.x = __shfl_sync(0xffffffffu, t.v[it].x, partner);
      pv.y = __shfl_sync(0xffffffffu, t.v[it].y, partner);
      pv.z = __shfl_sync(0xffffffffu, t.v[it].z, partner);
      pv.w = __shfl_sync(0xffffffffu, t.v[it].w, partner);
      // the x and y lanes of a pair need the same angles: each evaluates half and they swap
      float sn_m[4], cs_m[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float w = s_w[m0 + 2 * q + mine];
        const float ang = rf * w;
        const float err = fmaf(rf, w, -ang);
        const float kq = rintf(ang * 0.15915493667125702f);
        float red = fmaf(-kq, 6.28125f, ang);
        red = fmaf(-kq, 0.0019354820251464844f, red);
        red = fmaf(-kq, -1.7484555314695172e-07f, red);
        const float sn = __sinf(red), cs = __cosf(red);
        sn_m[q] = fmaf(err, cs, sn);
        cs_m[q] = fmaf(-err, sn, cs);
      }
      const uint32_t own[4] = {t.v[it].x, t.v[it].y, t.v[it].z, t.v[it].w};
      const uint32_t oth[4] = {pv.x, pv.y, pv.z, pv.w};
      uint32_t out[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const float sn_o = __shfl_sync(0xffffffffu, sn_m[q], partner);
        const float cs_o = __shfl_sync(0xffffffffu, cs_m[q], partner);
        float res[2];
#pragma unroll
        for (int hlf = 0; hlf < 2; ++hlf) {
          const float sn = hlf == mine ? sn_m[q] : sn_o, cs = hlf == mine ? cs_m[q] : cs_o;
          const float x = __uint_as_float(hlf ? (own[q] & 0xFFFF0000u) : (own[q] << 16));
          const float y = __uint_as_float(hlf ? (oth[q] & 0xFFFF0000u) : (oth[q] << 16));
          res[hlf] = in_x ? fmaf(x, cs, y * sn) : fmaf(x, cs, -(y * sn));
        }
        const __nv_bfloat162 b2 = __floats2bfloat162_rn(res[0], res[1]);
        out[q] = *reinterpret_cast<const uint32_t *>(&b2);
      }
      if (in_x || in_y) t.v[it] = make_uint4(out[0], out[1], out[2], out[3]);
    }
  };
  // every reader of the unit's old page has its loads landed
  auto readers_done = [&](const Tile &t) -> bool {
    // counts only grow: if every reader had landed when the unit was loaded,
    // the store may go ahead (it is issued only after that read returned)
    if (t.seen >= a.n_lanes) return true;
    for (int rw = t.dlo; rw <= t.dhi; ++rw)
      if (!wait_landed(&pd.dep[rw].landed, a.n_lanes, abort_flag)) return false;
    return true;
  };

  const int mover = blockIdx.x * kMovers + wid;
  const int my_units = mover < n_slots ? (n_slots - 1 - mover) / nm + 1 : 0;
  // the unit's (kk, j, tl) advance by nm slots without a division
  const int step_kk = nm / row_size, step_pos = nm - step_kk * row_size;
  const int step_j = step_pos / a.n_lanes, step_tl = step_pos - step_j * a.n_lanes;
  int kk = mover / row_size, pos = mover - kk * row_size;
  int j = pos / a.n_lanes, tl = pos - j * a.n_lanes;
  auto advance = [&]() {
    kk += step_kk;
    j += step_j;
    tl += step_tl;
    if (tl >= a.n_lanes) {
      tl -= a.n_lanes;
      ++j;
    }
    if (j >= n_active) {
      j -= n_active;
      ++kk;
    }
  };
  Tile A, B;
  Meta M;   // the descriptors of the next unit to load
  if (my_units > 0) {
    fetch(kk, j, tl, M);
    advance();
    load(M, A);
    fetch(kk, j, tl, M);
    advance();
    load(M, B);
    fetch(kk, j, tl, M);
    advance();
    land_and_count(A);
    rotate(A);
    // unit u in `cur` (landed, counted, rotated), unit u + 1 in flight in `next`:
    // u is stored and u + 2's loads are issued before waiting for u + 1's, so
    // two units' loads are in flight during that wait.  Every unit is still
    // counted before it is stored, so the lowest-numbered unstored unit can
    // always proceed.
    auto step = [&](Tile &cur, Tile &next) -> bool {
      if (!readers_done(cur)) return false;
      store(cur);
      load(M, cur);   // unit u + 2
      fetch(kk, j, tl, M);
      advance();
      land_and_count(next);
      rotate(next);
      return true;
    };
    for (int u = 0; u < my_units; u += 2) {
      bool ok = step(A, B);
      if (ok && u + 1 < my_units) ok = step(B, A);
      if (!ok) {
        if (lane == 0) {
          set_error(a.status, UMIM_ERR_TIMEOUT);
          atomicExch(abort_flag, 1);
        }
        break;
      }
    }
  }

  finish_rollback(a, arr, s_last);
}


// ---------------------------------------------------------------------------
// The move with TMA bulk copies (keys moved verbatim).  Same units, plan,
// landed counters and ordering argument as rollback_move_kernel; a unit's 16
// rows go through shared memory instead of registers.  Each slot's source is
// a moved entry, a surrogate row, or -- for a slot inside the written range
// that keeps its entry -- the row itself; slots whose sources are consecutive
// rows of one old page form a run that its first lane copies with one
// cp.async.bulk into the unit's stage.  The stage's mbarrier completes, the
// unit is counted into its row, and once its page's reader rows have landed
// one bulk store writes the unit's written slot range [ra, rb) back (a
// contiguous part of the 16 x D tile).  Each warp keeps three units in its
// ring.  The copy engine's reads and writes of the same pages keep their full
// rate, where 16-byte loads and stores of a 4 KB tile written back in place a
// few tiles behind its reads lose about a seventh.
// ---------------------------------------------------------------------------
constexpr int kBulkThreads = 512;   // 16 mover warps, one CTA per SM
constexpr int kBulkMovers = kBulkThreads / 32;
constexpr int kBulkStages = 3;      // units in flight per warp

__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(src), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

// The compacted entries are stored with the L2 evict-last priority: the decode
// attention that follows reads them, and finds the most recent ones in L2.
__device__ __forceinline__ void bulk_s2g(void *dst, const void *src, uint32_t bytes, uint64_t policy) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group.L2::cache_hint [%0], [%1], %2, %3;" ::"l"(dst),
               "r"(smem_u32(src)), "r"(bytes), "l"(policy)
               : "memory");
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}

// the smem reads of every bulk store this thread committed are done
__device__ __forceinline__ void bulk_wait_read_all() {
  asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}

__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// earlier generic-proxy accesses of global memory ordered before later async-proxy ones
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

template <int D>
__global__ void __launch_bounds__(kBulkThreads, 1) rollback_bulk_kernel(MoveArgs a, PlanArrays arr, PageDesc pd) {
  constexpr int ROW = D * 2;                 // bytes of one entry of one (K|V, head)
  constexpr int TILE = kPageSize * ROW;      // bytes of a unit
  constexpr int kHead = kPageSize * D;       // elements of one (K|V, head) tile
  extern __shared__ __align__(128) uint8_t bulk_smem[];
  __shared__ uint64_t bars[kBulkMovers][kBulkStages];
  __shared__ int s_last;
  __shared__ int s_sq[kSmemSeqs], s_nd[kSmemSeqs], s_ub[kSmemSeqs], s_fp[kSmemSeqs];
  __shared__ int64_t s_toff[kSmemLanes];
  __shared__ int32_t s_tlh[kSmemLanes];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int nm = gridDim.x * kBulkMovers;
  uint8_t *ring = bulk_smem + (size_t)wid * kBulkStages * TILE;

  if (lane == 0) {
    for (int st = 0; st < kBulkStages; ++st) mbar_init(&bars[wid][st], 1);
    fence_mbar_init();
  }
  griddep_wait();
  const PlanHeader *hdr = arr.hdr;
  int32_t *abort_flag = &arr.hdr->ticket;
  const int total = hdr->total_units;
  const int Hkv = a.n_kv_heads;
  const int64_t layer_stride = (int64_t)2 * kHead * Hkv * a.n_pages;
  const int kv_stride32 = kHead * Hkv, page_stride32 = 2 * kHead * Hkv;
  const int n_active = total > 0 ? hdr->n_active : 0;
  const int row_size = max(1, n_active * a.n_lanes);
  const int max_dest = total > 0 ? hdr->max_dest : 0;
  const int n_slots = max_dest * row_size;
  const int n_rows = total / a.n_lanes;   // compacted rows of all sequences (debug checks)

  const bool seq_in_smem = n_active <= kSmemSeqs;
  if (seq_in_smem) {
    for (int q = threadIdx.x; q < n_active; q += blockDim.x) {
      const int b = arr.active[q];
      s_sq[q] = b;
      s_nd[q] = arr.n_dest[b];
      s_ub[q] = arr.unit_base[b] / a.n_lanes;
      s_fp[q] = arr.first_page[b];
    }
  }
  const bool lanes_in_smem = a.n_lanes <= kSmemLanes;
  if (lanes_in_smem) {
    for (int q = threadIdx.x; q < a.n_lanes; q += blockDim.x) {
      const int layer = q / (2 * Hkv), kv = (q / Hkv) & 1, h = q % Hkv;
      s_toff[q] = layer * layer_stride + (int)(kv * kv_stride32 + h * kHead);
      s_tlh[q] = (int32_t)((uint32_t)(layer * Hkv + h) | ((uint32_t)kv << 31));
    }
  }
  __syncthreads();
  auto seq_of = [&](int q) { return seq_in_smem ? s_sq[q] : arr.active[q]; };
  auto nd_of = [&](int q) { return seq_in_smem ? s_nd[q] : arr.n_dest[arr.active[q]]; };
  auto row0_of = [&](int q) { return seq_in_smem ? s_ub[q] : arr.unit_base[arr.active[q]] / a.n_lanes; };
  auto fp_of = [&](int q) { return seq_in_smem ? s_fp[q] : arr.first_page[arr.active[q]]; };

  // a unit: where its rows come from and go, and which rows read its page.
  // Its descriptors are read a step before its copies are issued, and its
  // reader rows' counts when the copies are issued (a step before its store),
  // so that those round trips overlap the copies in flight.
  struct Unit {
    int64_t my_src;   // lanes < 16: the source of slot `lane` (kNoWrite: the slot keeps its entry)
    int64_t tile;     // offset of its (layer, K|V, head) tile in page 0 of the layer
    int32_t valid, idx, page, lh, kv, ra, rb, dlo, dhi, seen;
  };
  auto fetch = [&](int kk, int j, int tl, Unit &m) {
    m.valid = 0;
    m.ra = m.rb = 0;
    m.dlo = 1;
    m.dhi = 0;
    if (kk >= max_dest || kk >= nd_of(j)) return;
    const int b = seq_of(j);
    m.idx = row0_of(j) + kk;
    if (!in_bounds(m.idx, n_rows, a.status, kSiteRollbackReaderRow)) return;
    m.valid = 1;
    if (lanes_in_smem) {
      m.tile = s_toff[tl];
      const int32_t e = s_tlh[tl];
      m.kv = (int)((uint32_t)e >> 31);
      m.lh = e & 0x7fffffff;
    } else {
      const int layer = tl / (2 * Hkv), h = tl % Hkv;
      m.kv = (tl / Hkv) & 1;
      m.lh = layer * Hkv + h;
      m.tile = layer * layer_stride + (int)(m.kv * kv_stride32 + h * kHead);
    }
    m.my_src = lane < kPageSize ? pd.src[(int64_t)m.idx * kPageSize + lane] : kNoWrite;
    m.page = a.block_table[(int64_t)b * a.max_pages + fp_of(j) + kk];
    const RowDep dep = pd.dep[m.idx];
    m.dlo = dep.lo;
    m.dhi = dep.hi;
  };
  // the unit's rows into stage st (the stage's previous store has read it)
  auto issue = [&](Unit &m, int st) {
    // the slots this unit writes: from its first to its last moved entry
    const uint32_t w = __ballot_sync(0xffffffffu, m.valid && lane < kPageSize && m.my_src != kNoWrite);
    m.ra = w ? __ffs(w) - 1 : 0;
    m.rb = w ? 32 - __clz(w) : 0;
    if (m.valid && !in_bounds(m.page, a.n_pages, a.status, kSiteRollbackDstPage)) m.ra = m.rb = 0;
    if (m.valid && m.dlo <= m.dhi &&
        !(in_bounds(m.dlo, n_rows, a.status, kSiteRollbackReaderRow) &&
          in_bounds(m.dhi, n_rows, a.status, kSiteRollbackReaderRow))) {
      m.dlo = 1;
      m.dhi = 0;
      m.ra = m.rb = 0;
    }
    uint64_t *bar = &bars[wid][st];
    if (lane == 0) mbar_arrive_expect_tx(bar, (uint32_t)((m.rb - m.ra) * ROW));
    __syncwarp();
    // slots whose sources are consecutive rows of one old page form a run,
    // copied by the run's first lane in one piece
    const int64_t prev = __shfl_up_sync(0xffffffffu, m.my_src, 1);
    const bool mine = lane >= m.ra && lane < m.rb;
    const bool cont = mine && lane > m.ra && m.my_src >= 0 && prev >= 0 && m.my_src == prev + D;
    const uint32_t heads = __ballot_sync(0xffffffffu, mine && !cont);
    if (mine && !cont) {
      int rows = 1;
      if (m.my_src >= 0) {
        const uint32_t later = heads & ~((2u << lane) - 1u);   // run heads after this lane
        rows = (later ? __ffs(later) - 1 : m.rb) - lane;
      }
      const uint16_t *src;
      if (m.my_src >= 0) {
        src = a.pool + m.tile + m.my_src;
        if (!in_bounds(m.my_src, (int64_t)a.n_pages * page_stride32, a.status, kSiteRollbackSrc)) src = a.pool;
      } else if (m.my_src != kNoWrite) {
        const int64_t si = -m.my_src - 1;
        src = (m.kv ? a.sur_v : a.sur_k) + (si * a.n_layers * Hkv + m.lh) * D;
        if (!in_bounds(si, kDebugChecks ? a.span_offsets[a.B] : 0, a.status, kSiteRollbackSurrogate))
          src = a.sur_k;
      } else {
        src = a.pool + m.tile + (int64_t)m.page * page_stride32 + lane * D;   // the slot keeps its entry
      }
      bulk_g2s(ring + st * TILE + lane * ROW, src, (uint32_t)(rows * ROW), bar);
    }
    // the reader rows' counts as they are now (counts only grow)
    m.seen = a.n_lanes;
    if (lane == 0)
      for (int rw = m.dlo; rw <= m.dhi; ++rw) m.seen = min(m.seen, ld_relaxed(&pd.dep[rw].landed));
  };
  // every reader row of the unit's old page has its loads landed
  auto readers_done = [&](const Unit &m) -> bool {
    if (m.seen >= a.n_lanes) return true;   // read after this unit's copies were issued
    for (int rw = m.dlo; rw <= m.dhi; ++rw)
      if (!wait_landed(&pd.dep[rw].landed, a.n_lanes, abort_flag)) return false;
    return true;
  };

  const int mover = blockIdx.x * kBulkMovers + wid;
  const int my_units = mover < n_slots ? (n_slots - 1 - mover) / nm + 1 : 0;
  const int step_kk = nm / row_size, step_pos = nm - step_kk * row_size;
  const int step_j = step_pos / a.n_lanes, step_tl = step_pos - step_j * a.n_lanes;
  int kk = mover / row_size, pos = mover - kk * row_size;
  int j = pos / a.n_lanes, tl = pos - j * a.n_lanes;
  const uint64_t pol_store = policy_evict_last();
  auto next_unit = [&](Unit &m) {
    fetch(kk, j, tl, m);
    kk += step_kk;
    j += step_j;
    tl += step_tl;
    if (tl >= a.n_lanes) {
      tl -= a.n_lanes;
      ++j;
    }
    if (j >= n_active) {
      j -= n_active;
      ++kk;
    }
  };
  constexpr int S = kBulkStages;
  Unit U[S];     // unit u's descriptors in U[u % S] (stage u % S); indexed by unrolled constants only
  Unit Nx;       // the descriptors of the next unit to issue
  int issued = 0;   // units whose copies were issued
#pragma unroll
  for (int i = 0; i < S - 1; ++i)
    if (i < my_units) next_unit(U[i]);
  if (S - 1 < my_units) next_unit(Nx);
#pragma unroll
  for (int i = 0; i < S - 1; ++i)
    if (i < my_units) {
      issue(U[i], i);
      ++issued;
    }
  // unit k in stage k % S: refill the stage that unit k - 1 used with unit
  // k + S - 1 (descriptors read a step ago), read the next descriptors, wait
  // for unit k's rows, count it, wait for its readers, store it
  auto step = [&](int k, Unit &cur, int st, Unit &nxt, int st_nxt) -> bool {
    if (k + S - 1 < my_units) {
      nxt = Nx;
      if (lane == 0) bulk_wait_read_all();   // unit k - 1's store has read stage st_nxt
      __syncwarp();
      issue(nxt, st_nxt);
      ++issued;
      if (k + S < my_units) next_unit(Nx);
    }
    if (!__all_sync(0xffffffffu, mbar_wait(&bars[wid][st], (uint32_t)(k / S) & 1u))) return false;
    bool ok = true;
    if (lane == 0 && cur.valid) {
      // the unit's rows are in shared memory, so its reads of the old pages are done: count it
      // (relaxed: a release would also wait for this thread's earlier bulk stores to reach memory)
      asm volatile("red.relaxed.gpu.global.add.s32 [%0], 1;" ::"l"(&pd.dep[cur.idx].landed) : "memory");
      ok = readers_done(cur);
      if (ok && cur.rb > cur.ra) {
        fence_proxy_async_global();
        bulk_s2g(a.pool + cur.tile + (int64_t)cur.page * page_stride32 + cur.ra * D, ring + st * TILE + cur.ra * ROW,
                 (uint32_t)((cur.rb - cur.ra) * ROW), pol_store);
      }
    }
    return __shfl_sync(0xffffffffu, ok, 0);
  };
  int done = 0;   // units whose rows landed
  bool ok = true;
  for (int k = 0; k < my_units && ok; k += S) {
#pragma unroll
    for (int i = 0; i < S; ++i)
      if (ok && k + i < my_units) {
        ok = step(k + i, U[i], i, U[(i + S - 1) % S], (i + S - 1) % S);
        if (ok) ++done;
      }
  }
  if (!ok) {
    if (lane == 0) {
      set_error(a.status, UMIM_ERR_TIMEOUT);
      atomicExch(abort_flag, 1);
    }
    // the copies still in flight land (each wait bounded) before the CTA's shared memory goes away
    for (int u = done; u < issued; ++u)
      mbar_wait(&bars[wid][u % kBulkStages], (uint32_t)(u / kBulkStages) & 1u);
  }
  if (lane == 0) bulk_wait_all();
  __syncwarp();
  finish_rollback(a, arr, s_last);
}

}  // namespace

size_t kv_rollback_workspace_bytes(int B, int S, int max_pages, int n_layers, int n_kv_heads, int head_dim) {
  (void)head_dim;
  (void)n_layers;
  (void)n_kv_heads;
  const size_t pages = (size_t)B * max_pages > 0 ? (size_t)B * max_pages : 1;
  return plan_bytes(B, S) + align256(sizeof(int64_t) * kPageSize * pages) + align256(sizeof(RowDep) * pages) +
         align256(sizeof(int32_t) * kPageSize * pages);
}

umim_status kv_rollback(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages, int32_t *seq_lens,
                        int32_t B, const int32_t *span_offsets, const int32_t *span_start,
                        const int32_t *span_len, int32_t S, const void *sur_k, const void *sur_v,
                        int32_t *freed_pages, void *ws, size_t ws_bytes, int32_t *dev_status,
                        cudaStream_t stream, int num_sms, const float *rope_inv_freq, int rotary_dim) {
  const int D = kv->head_dim;
  const int lanes = kv->n_layers * 2 * kv->n_kv_heads;   // one unit per (layer, K|V, head) tile
  PlanArrays arr = plan_carve(ws, B, S);
  int32_t *status = dev_status ? dev_status : &arr.hdr->status;
  PageDesc pd;
  pd.src = reinterpret_cast<int64_t *>(arr.flags);   // the page descriptions follow the plan
  const size_t pages = (size_t)B * max_pages > 0 ? (size_t)B * max_pages : 1;
  pd.dep = reinterpret_cast<RowDep *>(reinterpret_cast<char *>(pd.src) + align256(sizeof(int64_t) * kPageSize * pages));
  pd.shift = reinterpret_cast<int32_t *>(reinterpret_cast<char *>(pd.dep) + align256(sizeof(RowDep) * pages));

  PlanArgs pa{};
  pa.seq_lens = seq_lens;
  pa.fixed_len = 0;
  pa.span_offsets = span_offsets;
  pa.span_start = span_start;
  pa.span_len = span_len;
  pa.B = B;
  pa.S = S;
  pa.max_span_len = 0;
  pa.block_table = block_table;
  pa.max_pages = max_pages;
  pa.n_pages = kv->n_pages;
  pa.n_lanes = lanes;
  pa.status = status;
  pa.cu_seqlens_out = nullptr;
  trace_mark(stream, "rollback.plan");
  if (launch_span_plan(pa, arr, stream) != cudaSuccess) return UMIM_ERR_CUDA;

  MoveArgs ma{};
  ma.pool = static_cast<uint16_t *>(kv->base);
  ma.n_lanes = lanes;
  ma.n_layers = kv->n_layers;
  ma.n_pages = kv->n_pages;
  ma.n_kv_heads = kv->n_kv_heads;
  ma.head_dim = D;
  ma.block_table = block_table;
  ma.max_pages = max_pages;
  ma.seq_lens = seq_lens;
  ma.span_offsets = span_offsets;
  ma.span_start = span_start;
  ma.span_len = span_len;
  ma.sur_k = static_cast<const uint16_t *>(sur_k);
  ma.sur_v = static_cast<const uint16_t *>(sur_v);
  ma.freed_pages = freed_pages;
  ma.freed_capacity = (int32_t)std::min<int64_t>((int64_t)B * max_pages, INT32_MAX);
  ma.B = B;
  ma.status = status;
  ma.rope_inv_freq = rope_inv_freq;
  ma.rotary_dim = rope_inv_freq ? rotary_dim : 0;
  ma.zero = 0;
  const bool rope = rope_inv_freq != nullptr;
  // verbatim moves go through the copy engine; re-rotated keys through registers
  auto kern = rope ? (D == 128 ? rollback_move_kernel<128, true> : rollback_move_kernel<64, true>)
                   : (D == 128 ? rollback_bulk_kernel<128> : rollback_bulk_kernel<64>);
  const int threads = rope ? kMoveThreads : kBulkThreads;
  const int smem = rope ? 0 : kBulkMovers * kBulkStages * kPageSize * D * 2;
  // set on every call: the attribute belongs to the current device
  if (!rope && cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return UMIM_ERR_CUDA;
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, threads, smem) != cudaSuccess || per_sm < 1)
    per_sm = 1;
  const int grid = std::max(1, num_sms) * per_sm;   // every CTA resident (cooperative launch)
  trace_mark(stream, "rollback.map");
  if (launch_pdl(rollback_map_kernel, dim3((unsigned)std::max(1, ceil_div(max_pages, 16)), (unsigned)B), dim3(256), 0,
                 stream, ma, arr, pd, (int)D) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, "rollback.move");
  // cooperative (every CTA resident), and allowed to launch while the map
  // kernel finishes (the kernel waits for it before reading the plan)
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if (cudaLaunchKernelEx(&cfg, kern, ma, arr, pd) != cudaSuccess) return UMIM_ERR_CUDA;
  trace_mark(stream, nullptr);
  return cudaGetLastError() == cudaSuccess ? UMIM_OK : UMIM_ERR_CUDA;
}

}  // namespace umim
