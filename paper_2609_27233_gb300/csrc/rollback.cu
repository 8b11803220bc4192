// KV-cache rollback and in-place compaction of a paged bf16 cache
// (App. E "Decoding-Time Merging and KV-Cache Update", Fig. 2): each span's
// k stored entries become one surrogate entry and later entries move left.
//
// Work unit = (sequence b, lane = layer x head group, compacted page p): the
// 16 compacted entries j in [16p, 16p+16) of one layer and a group of KV
// heads.  A unit copies its sources (kept entries t = j + r >= j, or the
// surrogate rows) into shared memory, publishes "read done", waits until
// every unit that reads old page p has published, then writes page p.
// Because j <= t, the units that read old page p are unit p itself and lower
// pages of the same (b, lane), i.e. smaller unit indices.  The launch is
// cooperative (every CTA resident) and CTA c handles units c, c + grid,
// c + 2 grid, ... in increasing order, publishing each as soon as its copies
// land, so the smallest unpublished unit always makes progress: no deadlock,
// no second pass, each moved byte read once and written once.  Every wait is
// bounded (UMIM_ERR_TIMEOUT).
#include <algorithm>

#include "plan.cuh"

namespace umim {
namespace {

constexpr int kMoveThreads = 256;
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

__device__ __forceinline__ int find_seq(const int32_t *base, int B, int u) {
  int l = 0, h = B;   // largest b with base[b] <= u
  while (l < h) {
    const int m = (l + h) >> 1;
    if (base[m] <= u) l = m + 1;
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
  int2 *dep;       // [pages] range of compacted pages that read this old page
};

// One warp per (sequence, compacted page): where each of its 16 entries comes
// from, and which compacted pages read the same page of the old layout.
__global__ void __launch_bounds__(256) rollback_map_kernel(MoveArgs a, PlanArrays arr, PageDesc pd, int D) {
  griddep_wait();
  if (arr.hdr->skip) return;
  const int b = blockIdx.y;
  const int k = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  const int nd = arr.n_dest[b];
  if (k >= nd) return;
  const int p = arr.first_page[b] + k;
  const int idx = arr.unit_base[b] / a.n_lanes + k;
  const int lo = a.span_offsets[b], hi = a.span_offsets[b + 1];
  const int32_t *bt = a.block_table + (int64_t)b * a.max_pages;
  const int64_t page_stride = (int64_t)kPageSize * D * a.n_kv_heads * 2;
  int dpage = -1;
  if (lane < kPageSize) {
    const int L = arr.seq_Lp[b];
    const int j = p * kPageSize + lane;
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
    pd.src[(int64_t)idx * kPageSize + lane] = src;
  } else {
    const int L = arr.seq_L[b];
    const int t = p * kPageSize + (lane - kPageSize);
    if (t < L) {
      const int i = upper_index(a.span_start, lo, hi, t);
      if (i >= lo && t >= a.span_start[i] + a.span_len[i]) {
        const int r = arr.r_incl[i];
        if (r > 0) dpage = (t - r) / kPageSize;
      }
    }
  }
  int mn = dpage < 0 ? 0x7fffffff : dpage, mx = dpage;
#pragma unroll
  for (int o = 8; o >= 1; o >>= 1) {
    mn = min(mn, __shfl_xor_sync(0xffffffffu, mn, o));
    mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  }
  if (lane == kPageSize) pd.dep[idx] = make_int2(mn, mx);
}

constexpr int kMovers = kMoveThreads / 32 - 1;   // mover warps per CTA; the last warp publishes

__device__ __forceinline__ void st_release_cta_shared(int *p, int v) {
  asm volatile("st.release.cta.shared.b32 [%0], %1;" ::"r"(smem_u32(p)), "r"(v) : "memory");
}
__device__ __forceinline__ int ld_acquire_cta_shared(const int *p) {
  int v;
  asm volatile("ld.acquire.cta.shared.b32 %0, [%1];" : "=r"(v) : "r"(smem_u32(p)) : "memory");
  return v;
}
__device__ __forceinline__ void fence_acq_rel_gpu() { asm volatile("fence.acq_rel.gpu;" ::: "memory"); }
__device__ __forceinline__ void st_relaxed_gpu(int32_t *p, int32_t v) {
  asm volatile("st.relaxed.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// One mover warp per unit = one (layer, K|V, head) 16 x D tile of a compacted
// page.  Lane l moves 16-byte chunks c = l + 32 it of the tile: row c / CPR
// (the slot), column c % CPR.  Units are visited page-row by page-row:
// processing slot i covers compacted page k = i / (B * tiles) of sequence b
// and tile t, (b, t) = divmod(i mod (B * tiles), tiles); slots with k beyond
// the sequence's pages do nothing.  A unit waits only for units of earlier
// rows, which were picked up at least a whole row of slots before it.  Mover m
// of the grid handles slots m, m + M, m + 2M, ... (M movers).  When a unit's loads have returned, the mover
// reports it in its shared-memory mailbox (CTA-scope release) and goes on to
// wait for the units that read its destination page and to write it.  The
// CTA's publisher warp collects reported units, issues one GPU-scope fence
// for the whole batch and then marks their read-done flags: the fence orders
// every reported load before every flag store that follows it, and movers
// never pay for a GPU-scope fence themselves.
template <int D>
__global__ void __launch_bounds__(kMoveThreads, 4) rollback_move_kernel(MoveArgs a, PlanArrays arr, PageDesc pd) {
  constexpr int CPR = D / 8;                       // 16-byte chunks per row
  constexpr int PER_LANE = kPageSize * CPR / 32;   // 8 (D=128) or 4 (D=64)
  constexpr int SLOT_STEP = 32 / CPR;              // slots advanced per it
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int nm = gridDim.x * kMovers;
  const int my_col = lane % CPR;
  const int my_slot0 = lane / CPR;
  __shared__ int s_last;
  __shared__ int s_mail[kMovers];   // units reported loaded by each mover (a count)
  __shared__ int s_finished;        // movers that left their loop

  const PlanHeader *hdr = arr.hdr;
  const int total = hdr->total_units;
  const int epoch = hdr->epoch;
  const int Hkv = a.n_kv_heads;
  const int64_t head_stride = (int64_t)kPageSize * D;
  const int64_t kv_stride = head_stride * Hkv;
  const int64_t page_stride = kv_stride * 2;
  const int64_t layer_stride = page_stride * a.n_pages;
  const int row_size = a.B * a.n_lanes;
  const int64_t n_slots = total > 0 ? (int64_t)hdr->max_dest * row_size : 0;

  if (threadIdx.x < kMovers) s_mail[threadIdx.x] = 0;
  if (threadIdx.x == 0) s_finished = 0;
  __syncthreads();

  if (wid == kMovers) {
    // ---- publisher ----
    int published[kMovers];
#pragma unroll
    for (int m = 0; m < kMovers; ++m) published[m] = 0;
    uint64_t t_idle = globaltimer();
    while (true) {
      int mail[kMovers];
      bool any = false;
      // finished before the mailboxes: a mover's last report precedes its exit
      const int fin = ld_acquire_cta_shared(&s_finished);
#pragma unroll
      for (int m = 0; m < kMovers; ++m) {
        mail[m] = ld_acquire_cta_shared(&s_mail[m]);
        any |= mail[m] > published[m];
      }
      if (any) {
        fence_acq_rel_gpu();   // every reported load happens before the flags below
#pragma unroll
        for (int m = 0; m < kMovers; ++m) {
          const int mover = blockIdx.x * kMovers + m;
          for (int k = published[m] + lane; k < mail[m]; k += 32) {
            const int64_t i = mover + (int64_t)k * nm;
            const int kk = (int)(i / row_size);
            const int pos = (int)(i - (int64_t)kk * row_size);
            const int b = pos / a.n_lanes, tl = pos % a.n_lanes;
            const int nd = arr.n_dest[b];
            if (kk < nd) st_relaxed_gpu(&arr.flags[arr.unit_base[b] + tl * nd + kk], epoch);
          }
          published[m] = mail[m];
        }
        t_idle = globaltimer();
      } else if (fin == kMovers) {
        break;
      } else if (globaltimer() - t_idle > kWaitLimitNs) {
        set_error(a.status, UMIM_ERR_TIMEOUT);
        break;
      } else {
        __nanosleep(32);
      }
    }
  } else {
    // ---- mover ----
    const int mover = blockIdx.x * kMovers + wid;
    int k = 0;
    for (int64_t i = mover; i < n_slots; i += nm, ++k) {
      // slot -> (compacted page row kk, sequence, tile lane)
      const int kk = (int)(i / row_size);
      const int pos = (int)(i - (int64_t)kk * row_size);
      const int b = pos / a.n_lanes, tl = pos % a.n_lanes;
      const int nd = arr.n_dest[b];
      if (kk >= nd) {
        if (lane == 0) st_release_cta_shared(&s_mail[wid], k + 1);
        continue;
      }
      const int u = arr.unit_base[b] + tl * nd + kk;
      const int layer = tl / (2 * Hkv);
      const int kv = (tl / Hkv) & 1;
      const int h = tl % Hkv;
      const int idx = arr.unit_base[b] / a.n_lanes + kk;
      const int p = arr.first_page[b] + kk;
      const int64_t my_src = lane < kPageSize ? pd.src[(int64_t)idx * kPageSize + lane] : kNoWrite;
      const int2 dep = pd.dep[idx];
      const int64_t tile = layer * layer_stride + kv * kv_stride + h * head_stride + my_col * 8;
      const uint16_t *sur = kv ? a.sur_v : a.sur_k;

      uint4 v[PER_LANE];
      uint32_t write_mask = 0;
      uint32_t fold = 0;
#pragma unroll
      for (int it = 0; it < PER_LANE; ++it) {
        const int slot = my_slot0 + it * SLOT_STEP;
        const int64_t src = __shfl_sync(0xffffffffu, my_src, slot);
        if (src != kNoWrite) write_mask |= 1u << it;
        v[it] = make_uint4(0, 0, 0, 0);
        if (src >= 0) {
          v[it] = ld_v4(a.pool + tile + src);
        } else if (src != kNoWrite) {
          const int64_t i = -src - 1;
          v[it] = ld_v4(sur + ((i * a.n_layers + layer) * Hkv + h) * D + my_col * 8);
        }
        fold ^= v[it].x ^ v[it].y ^ v[it].z ^ v[it].w;
      }
      // every loaded value of this lane has arrived before the warp barrier
      asm volatile("" ::"r"(fold) : "memory");
      __syncwarp();
      int ok = 1;
      if (lane == 0) {
        // report: units 0 .. k of this mover have been read
        st_release_cta_shared(&s_mail[wid], k + 1);
        // wait for the units that read this tile of old page p (smaller indices)
        for (int q = dep.x; q <= dep.y && q >= 0 && q < p; ++q) {
          const int uq = u - (p - q);
          if (ld_acquire(&arr.flags[uq]) == epoch) continue;
          const uint64_t t0 = globaltimer();
          bool got = false;
          while (!got) {
#pragma unroll 1
            for (int i = 0; i < 64 && !got; ++i) got = (ld_acquire(&arr.flags[uq]) == epoch);
            if (!got && globaltimer() - t0 > kWaitLimitNs) break;
          }
          if (!got) {
            set_error(a.status, UMIM_ERR_TIMEOUT);
            ok = 0;
            break;
          }
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      const int64_t dst = tile + (int64_t)a.block_table[(int64_t)b * a.max_pages + p] * page_stride;
#pragma unroll
      for (int it = 0; it < PER_LANE; ++it) {
        const int slot = my_slot0 + it * SLOT_STEP;
        if (write_mask & (1u << it)) st_v4(a.pool + dst + slot * D, v[it]);
      }
    }
    __syncwarp();
    if (lane == 0) {
      __threadfence_block();   // the last report is visible before the exit count
      atomicAdd(&s_finished, 1);
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
  const size_t units = (size_t)B * n_layers * 2 * n_kv_heads * (size_t)max_pages;
  const size_t pages = (size_t)B * max_pages;
  return plan_bytes(B, S) + align256(sizeof(int32_t) * (units > 0 ? units : 1)) +
         align256(sizeof(int64_t) * kPageSize * (pages > 0 ? pages : 1)) + align256(sizeof(int2) * (pages > 0 ? pages : 1));
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
  const size_t units = (size_t)B * lanes * (size_t)max_pages;
  const size_t pages = (size_t)B * max_pages;
  PageDesc pd;
  pd.src = reinterpret_cast<int64_t *>(reinterpret_cast<char *>(arr.flags) +
                                       align256(sizeof(int32_t) * (units > 0 ? units : 1)));
  pd.dep = reinterpret_cast<int2 *>(reinterpret_cast<char *>(pd.src) +
                                    align256(sizeof(int64_t) * kPageSize * (pages > 0 ? pages : 1)));

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
  if (launch_pdl(rollback_map_kernel, dim3((unsigned)std::max(1, ceil_div(max_pages, 8)), (unsigned)B), dim3(256), 0,
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
