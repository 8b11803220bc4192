// KV-cache rollback and in-place compaction of a paged bf16 cache
// (App. E "Decoding-Time Merging and KV-Cache Update", Fig. 2): each span's
// k stored entries become one surrogate entry and later entries move left.
//
// Work unit = one (layer, K|V, kv-head) 16 x D tile of one compacted page of
// one sequence: its 16 entries j come from kept entries t = j + r >= j or
// from surrogate rows, and it is written to the same physical page that held
// old page j / 16.  Units are numbered row by row (row = compacted page
// index, over the sequences that have pages to write) and dealt round-robin
// to the mover warps of a cooperative grid; each warp copies two units ahead
// of its stores, through shared memory with the copy engine.  A unit may overwrite its page once every unit that reads
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

// ---------------------------------------------------------------------------
// The move, with TMA bulk copies.  A unit's 16 rows go through shared memory.
// Each slot's source is a moved entry, a surrogate row, or -- for a slot inside
// the written range that keeps its entry -- the row itself; slots whose sources
// are consecutive rows of one old page form a run that its first lane copies
// with one cp.async.bulk into the unit's stage.  The stage's mbarrier
// completes, the unit is counted into its row, and once its page's reader rows
// have landed one bulk store writes the unit's written slot range [ra, rb) back
// (a contiguous part of the 16 x D tile).  With RoPE, the moved keys are
// re-rotated in shared memory between the copies and the store.  Each warp
// keeps three units in its ring.  The copy engine's reads and writes of the
// same pages keep their full rate, where 16-byte loads and stores of a 4 KB
// tile written back in place a few tiles behind its reads lose about a seventh.
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

template <int D, bool ROPE>
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
  __shared__ float s_w[ROPE ? D / 2 : 1];   // RoPE angular frequencies
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int nm = gridDim.x * kBulkMovers;
  uint8_t *ring = bulk_smem + (size_t)wid * kBulkStages * TILE;

  if (ROPE)
    for (int i = threadIdx.x; i < a.rotary_dim / 2; i += blockDim.x) s_w[i] = a.rope_inv_freq[i];
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
    int32_t shift;    // lanes < 16: positions removed before slot `lane`'s moved entry (re-rotated keys)
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
    m.shift = (ROPE && lane < kPageSize) ? pd.shift[(int64_t)m.idx * kPageSize + lane] : 0;
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
  // RoPE: a moved key (shift r > 0) is rotated in shared memory by -r w_m on the
  // pairs (m, m + rotary_dim/2): x' = x cos + y sin, y' = y cos - x sin, with the
  // angle r w rounded plus its exact rounding error (an fma) folded into the sine
  // and cosine to first order, and the rounded angle reduced to [-pi, pi] (Cody
  // and Waite's three-part reduction) for the hardware sine and cosine.  Lane l
  // takes the pairs m = l and l + 32 of every row; consecutive rows with the same
  // shift (a run of moved entries between two spans) reuse the lane's angles.
  static_assert(D / 2 <= 64, "two pairs per lane");
  auto rotate_rows = [&](const Unit &m, uint8_t *stage) {
    const int half = a.rotary_dim / 2;
    float prev = 0.f, snc[2] = {0.f, 0.f}, csc[2] = {1.f, 1.f};
    for (int r = m.ra; r < m.rb; ++r) {
      const float rf = (float)__shfl_sync(0xffffffffu, m.shift, r);
      if (rf == 0.f) continue;   // a surrogate or an entry that keeps its position
      if (rf != prev) {
#pragma unroll
        for (int i = 0; i < 2; ++i) {
          const int q = lane + 32 * i;
          if (q < half) {
            const float w = s_w[q];
            const float ang = rf * w;
            const float err = fmaf(rf, w, -ang);
            const float kq = rintf(ang * 0.15915493667125702f);
            float red = fmaf(-kq, 6.28125f, ang);
            red = fmaf(-kq, 0.0019354820251464844f, red);
            red = fmaf(-kq, -1.7484555314695172e-07f, red);
            const float sn0 = __sinf(red), cs0 = __cosf(red);
            snc[i] = fmaf(err, cs0, sn0);
            csc[i] = fmaf(-err, sn0, cs0);
          }
        }
        prev = rf;
      }
      __nv_bfloat16 *row = reinterpret_cast<__nv_bfloat16 *>(stage + r * ROW);
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        const int q = lane + 32 * i;
        if (q < half) {
          const float x = __bfloat162float(row[q]), y = __bfloat162float(row[q + half]);
          row[q] = __float2bfloat16_rn(fmaf(x, csc[i], y * snc[i]));
          row[q + half] = __float2bfloat16_rn(fmaf(y, csc[i], -(x * snc[i])));
        }
      }
    }
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
    if (ROPE && cur.valid && cur.kv == 0) {
      rotate_rows(cur, ring + st * TILE);
      fence_proxy_async_smem();   // the rotated rows, written by the lanes, are what the bulk store reads
      __syncwarp();
    }
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
  const bool rope = rope_inv_freq != nullptr;
  auto kern = rope ? (D == 128 ? rollback_bulk_kernel<128, true> : rollback_bulk_kernel<64, true>)
                   : (D == 128 ? rollback_bulk_kernel<128, false> : rollback_bulk_kernel<64, false>);
  const int threads = kBulkThreads;
  const int smem = kBulkMovers * kBulkStages * kPageSize * D * 2;
  // set on every call: the attribute belongs to the current device
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
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
