// KV-cache rollback and in-place compaction of a paged bf16 cache
// (App. E "Decoding-Time Merging and KV-Cache Update", Fig. 2): each span's
// k stored entries become one surrogate entry and later entries move left.
//
// Work unit = one (layer, K|V, kv-head) 16 x D tile of one compacted page of
// one sequence: its 16 entries j come from kept entries t = j + r >= j or
// from surrogate rows, and it is written to the same physical page that held
// old page j / 16.  Units are visited row by row (row = compacted page index,
// over the sequences that have pages to write) in rounds: round r gives every
// mover warp of the cooperative grid one unit, its loads land, a grid-wide
// barrier follows, then its stores.  Because j <= t, the units that read a
// unit's destination tile sit in the same column at the same or a lower row,
// i.e. in the same or an earlier round, so every read of a location precedes
// its write; and a round's loads read only tiles at or beyond their own rows,
// which no earlier round writes, so round r + 1's loads are in flight while
// round r waits at the barrier and stores.  One pass: each moved byte is read
// once and written once.  The barrier wait is bounded (UMIM_ERR_TIMEOUT).
#include <algorithm>

#include "plan.cuh"

namespace umim {
namespace {

constexpr int kMoveThreads = 256;   // 7 mover warps + 1 warp that runs the grid barrier
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

struct PageDesc {
  int64_t *src;    // [pages][16] source row offset within a layer (no head offset), -(i+1) for span i, kNoWrite
};

// Sixteen threads per (sequence, compacted page): where each of its 16
// entries comes from (kNoWrite: the entry does not move).
__global__ void __launch_bounds__(256) rollback_map_kernel(MoveArgs a, PlanArrays arr, PageDesc pd, int D) {
  griddep_wait();
  if (arr.hdr->skip) return;
  const int b = blockIdx.y;
  const int k = blockIdx.x * 16 + (threadIdx.x >> 4);
  const int slot = threadIdx.x & 15;
  const int nd = arr.n_dest[b];
  if (k >= nd) return;
  const int p = arr.first_page[b] + k;
  const int idx = arr.unit_base[b] / a.n_lanes + k;
  const int lo = a.span_offsets[b], hi = a.span_offsets[b + 1];
  const int32_t *bt = a.block_table + (int64_t)b * a.max_pages;
  const int64_t page_stride = (int64_t)kPageSize * D * a.n_kv_heads * 2;
  const int L = arr.seq_Lp[b];
  const int j = p * kPageSize + slot;
  int64_t src = kNoWrite;
  if (j < L && j >= a.span_start[lo]) {
    const int i = upper_index(arr.new_idx, lo, hi, j);
    if (i >= lo) {
      if (arr.new_idx[i] == j) {
        src = -(int64_t)i - 1;
      } else {
        const int t = j + arr.r_incl[i];
        if (t != j) src = (int64_t)bt[t / kPageSize] * page_stride + (t % kPageSize) * D;
      }
    }
  }
  pd.src[(int64_t)idx * kPageSize + slot] = src;
}

constexpr int kMovers = kMoveThreads / 32 - 1;
constexpr int kSmemSeqs = 1024;   // active sequences whose plan values a CTA keeps in shared memory

// Grid barrier in two halves, run by lane 0 of the CTA's barrier warp (which
// has no loads of its own in flight, so its fence does not wait for them).
// arrive: after a __syncthreads that follows every load of the round, count
// this CTA in; wait: until every CTA has counted itself in for the round.
__device__ __forceinline__ void grid_arrive(int32_t *count) {
  __threadfence();   // the CTA's completed loads before the arrival
  atomicAdd(count, 1);
}
__device__ __forceinline__ bool grid_wait(const int32_t *count, int target) {
  if (ld_acquire(count) >= target) return true;
  const uint64_t t0 = globaltimer();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 64; ++i)
      if (ld_acquire(count) >= target) return true;
    if (globaltimer() - t0 > kWaitLimitNs) return false;
  }
}

// Mover warps: lane l moves 16-byte chunks c = l + 32 it of a tile, row
// (slot) c / CPR, column c % CPR.  Step r: round r + 1's loads land and the
// CTA arrives at barrier r + 1; then, while that barrier fills up, round r's
// tile (barrier r has passed) is stored and round r + 2's loads are issued
// into the registers it held; then barrier r + 1 is waited for.  A CTA
// arrives at barrier r + 1 only after passing barrier r, so one counter of
// arrivals serves every round: barrier r has passed once it reaches
// (r + 1) x grid.
template <int D>
__global__ void __launch_bounds__(kMoveThreads, 2) rollback_move_kernel(MoveArgs a, PlanArrays arr, PageDesc pd) {
  constexpr int CPR = D / 8;                       // 16-byte chunks per row
  constexpr int PER_LANE = kPageSize * CPR / 32;   // 8 (D=128) or 4 (D=64)
  constexpr int SLOT_STEP = 32 / CPR;              // rows advanced per it
  constexpr int kHead = kPageSize * D;             // elements of one (K|V, head) tile
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int nm = gridDim.x * kMovers;
  const int my_col = lane % CPR;
  const int my_slot0 = lane / CPR;
  __shared__ int s_last, s_abort;
  __shared__ int s_sq[kSmemSeqs], s_nd[kSmemSeqs], s_ub[kSmemSeqs], s_fp[kSmemSeqs];

  const PlanHeader *hdr = arr.hdr;
  const int total = hdr->total_units;
  const int Hkv = a.n_kv_heads;
  const int64_t layer_stride = (int64_t)2 * kHead * Hkv * a.n_pages;
  const int kv_stride32 = kHead * Hkv, page_stride32 = 2 * kHead * Hkv;
  // a row holds the tiles of the sequences that have pages to write
  const int n_active = total > 0 ? hdr->n_active : 0;
  const int row_size = max(1, n_active * a.n_lanes);
  // slot indices fit in 32 bits: batch x max_pages x tile lanes < 2^30 is checked on the host
  const int max_dest = total > 0 ? hdr->max_dest : 0;
  const int n_slots = max_dest * row_size;
  const int rounds = (n_slots + nm - 1) / nm;

  if (threadIdx.x == 0) s_abort = 0;
  // plan values of the active sequences (row position order), from shared
  // memory when there are few enough of them
  const bool seq_in_smem = n_active <= kSmemSeqs;
  if (seq_in_smem) {
    for (int j = threadIdx.x; j < n_active; j += blockDim.x) {
      const int b = arr.active[j];
      s_sq[j] = b;
      s_nd[j] = arr.n_dest[b];
      s_ub[j] = arr.unit_base[b];
      s_fp[j] = arr.first_page[b];
    }
  }
  __syncthreads();
  auto seq_of = [&](int j) { return seq_in_smem ? s_sq[j] : arr.active[j]; };
  auto nd_of = [&](int j) { return seq_in_smem ? s_nd[j] : arr.n_dest[arr.active[j]]; };
  auto ub_of = [&](int j) { return seq_in_smem ? s_ub[j] : arr.unit_base[arr.active[j]]; };
  auto fp_of = [&](int j) { return seq_in_smem ? s_fp[j] : arr.first_page[arr.active[j]]; };

  // slot i = kk * row_size + pos, kk the compacted page row
  struct Desc {
    int valid, tl;
    int64_t src;    // this lane's row source (lanes < 16)
    int32_t page;   // destination physical page
  };
  auto describe = [&](int kk, int pos) {
    Desc x{0, 0, kNoWrite, 0};
    if (kk >= max_dest) return x;
    const int j = pos / a.n_lanes, tl = pos - j * a.n_lanes;
    if (kk >= nd_of(j)) return x;
    const int b = seq_of(j);
    const int idx = ub_of(j) / a.n_lanes + kk;
    x.valid = 1;
    x.tl = tl;
    x.src = lane < kPageSize ? pd.src[(int64_t)idx * kPageSize + lane] : kNoWrite;
    x.page = a.block_table[(int64_t)b * a.max_pages + fp_of(j) + kk];
    return x;
  };
  const int step_kk = nm / row_size, step_pos = nm - step_kk * row_size;
  auto advance = [&](int &kk, int &pos) {
    kk += step_kk;
    pos += step_pos;
    if (pos >= row_size) {
      pos -= row_size;
      ++kk;
    }
  };
  // a tile in registers, with where it goes
  struct Tile {
    uint4 v[PER_LANE];
    uint32_t mask;
    int64_t dst;
  };
  auto load = [&](const Desc &x, Tile &t) {
    t.mask = 0;
    t.dst = 0;
#pragma unroll
    for (int it = 0; it < PER_LANE; ++it) t.v[it] = make_uint4(0, 0, 0, 0);
    if (!x.valid) return;
    const int layer = x.tl / (2 * Hkv), kv = (x.tl / Hkv) & 1, h = x.tl % Hkv;
    const int64_t tile = layer * layer_stride + (int)(kv * kv_stride32 + h * kHead + my_col * 8);
    const uint16_t *sur = kv ? a.sur_v : a.sur_k;
    t.dst = tile + (int64_t)x.page * page_stride32;
#pragma unroll
    for (int it = 0; it < PER_LANE; ++it) {
      const int slot = my_slot0 + it * SLOT_STEP;
      const int64_t src = __shfl_sync(0xffffffffu, x.src, slot);
      if (src != kNoWrite) t.mask |= 1u << it;
      if (src >= 0) {
        t.v[it] = ld_v4(a.pool + tile + src);
      } else if (src != kNoWrite) {
        const int64_t si = -src - 1;
        t.v[it] = ld_v4(sur + ((si * a.n_layers + layer) * Hkv + h) * D + my_col * 8);
      }
    }
  };
  auto store = [&](const Tile &t) {
#pragma unroll
    for (int it = 0; it < PER_LANE; ++it) {
      const int slot = my_slot0 + it * SLOT_STEP;
      if (t.mask & (1u << it)) st_v4(a.pool + t.dst + slot * D, t.v[it]);
    }
  };
  auto landed = [&](const Tile &t) {
    uint32_t fold = 0;
#pragma unroll
    for (int it = 0; it < PER_LANE; ++it) fold ^= t.v[it].x ^ t.v[it].y ^ t.v[it].z ^ t.v[it].w;
    asm volatile("" ::"r"(fold) : "memory");   // every loaded value of the tile has arrived
  };
  // barrier halves, CTA-wide: arrive after this CTA's loads of the round landed
  auto arrive = [&]() {
    __syncthreads();
    if (wid == kMovers && lane == 0) grid_arrive(&arr.hdr->ticket);
  };
  auto wait = [&](int r) -> bool {
    if (wid == kMovers && lane == 0 && !grid_wait(&arr.hdr->ticket, (r + 1) * (int)gridDim.x)) {
      set_error(a.status, UMIM_ERR_TIMEOUT);
      s_abort = 1;
    }
    __syncthreads();
    return !s_abort;
  };
  // step r (tile r in `cur`, round r + 1's loads in flight in `next`, barrier r passed)
  auto step = [&](int r, Tile &cur, Tile &next, Desc &d_next2, int &kk2, int &pos2) -> bool {
    landed(next);                 // round r + 1's loads
    arrive();                     // barrier r + 1
    store(cur);                   // round r
    load(d_next2, cur);           // round r + 2 into the registers just stored
    d_next2 = describe(kk2, pos2);
    advance(kk2, pos2);
    return wait(r + 1);
  };

  // the barrier warp takes a slot past the end: it describes, loads and stores nothing
  const int mover = wid < kMovers ? blockIdx.x * kMovers + wid : n_slots + nm;
  int kk = mover / row_size, pos = mover - kk * row_size;   // round 0
  Tile A, B;
  load(describe(kk, pos), A);                                // round 0
  advance(kk, pos);
  load(describe(kk, pos), B);                                // round 1
  advance(kk, pos);
  Desc d_next2 = describe(kk, pos);                          // round 2
  advance(kk, pos);
  if (rounds > 0) {
    landed(A);
    arrive();
    if (wait(0)) {
      for (int r = 0; r < rounds; r += 2) {
        if (!step(r, A, B, d_next2, kk, pos)) break;
        if (r + 1 < rounds && !step(r + 1, B, A, d_next2, kk, pos)) break;
      }
    }
  }

  // ---- the last CTA to finish truncates block tables and updates lengths ----
  const int tid = threadIdx.x;
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    const int done = atomicAdd(&arr.hdr->done_ctas, 1);
    s_last = (done == (int)gridDim.x - 1);
  }
  __syncthreads();
  if (!s_last || hdr->skip) return;
  __threadfence();
  for (int b = 0; b < a.B; ++b) {
    if (a.span_offsets[b + 1] == a.span_offsets[b]) continue;
    const int L = arr.seq_L[b], Lp = arr.seq_Lp[b];
    const int keep = ceil_div(Lp, kPageSize), had = ceil_div(L, kPageSize);
    const int fb = arr.freed_base[b];
    for (int q = keep + tid; q < had; q += kMoveThreads) {
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

}  // namespace

size_t kv_rollback_workspace_bytes(int B, int S, int max_pages, int n_layers, int n_kv_heads, int head_dim) {
  (void)head_dim;
  (void)n_layers;
  (void)n_kv_heads;
  const size_t pages = (size_t)B * max_pages;
  return plan_bytes(B, S) + align256(sizeof(int64_t) * kPageSize * (pages > 0 ? pages : 1));
}

umim_status kv_rollback(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages, int32_t *seq_lens,
                        int32_t B, const int32_t *span_offsets, const int32_t *span_start,
                        const int32_t *span_len, int32_t S, const void *sur_k, const void *sur_v,
                        int32_t *freed_pages, void *ws, size_t ws_bytes, int32_t *dev_status,
                        cudaStream_t stream, int num_sms) {
  const int D = kv->head_dim;
  const int lanes = kv->n_layers * 2 * kv->n_kv_heads;   // one unit per (layer, K|V, head) tile
  PlanArrays arr = plan_carve(ws, B, S);
  int32_t *status = dev_status ? dev_status : &arr.hdr->status;
  PageDesc pd;
  pd.src = reinterpret_cast<int64_t *>(arr.flags);   // the page descriptions follow the plan

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
  auto kern = (D == 128) ? rollback_move_kernel<128> : rollback_move_kernel<64>;
  const int smem = 0;
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kMoveThreads, smem) != cudaSuccess || per_sm < 1)
    per_sm = 1;
  const int grid = std::max(1, num_sms) * per_sm;   // every CTA resident (cooperative launch)
  trace_mark(stream, "rollback.map");
  if (launch_pdl(rollback_map_kernel, dim3((unsigned)std::max(1, ceil_div(max_pages, 16)), (unsigned)B), dim3(256), 0,
                 stream, ma, arr, pd, (int)D) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, "rollback.move");
  void *args[] = {&ma, &arr, &pd};
  if (cudaLaunchCooperativeKernel(reinterpret_cast<const void *>(kern), dim3(grid), dim3(kMoveThreads), args,
                                  (size_t)smem, stream) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, nullptr);
  return cudaGetLastError() == cudaSuccess ? UMIM_OK : UMIM_ERR_CUDA;
}

}  // namespace umim
