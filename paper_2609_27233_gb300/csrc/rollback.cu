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
constexpr int kUnitBytes = 32768;                     // data moved per unit
constexpr int kChunksPerThread = kUnitBytes / 16 / kMoveThreads;   // 8 x 16 B
constexpr int64_t kNoWrite = INT64_MIN;

struct MoveArgs {
  uint16_t *pool;
  int32_t n_lanes;
  int32_t n_layers, n_pages, n_kv_heads, head_dim;
  int32_t heads_per_unit, n_head_groups;
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

__device__ __forceinline__ void cp_async_16(void *smem, const void *gmem) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(smem)), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

constexpr int kRing = 3;   // units in flight per CTA
constexpr int kMeta = kRing + 2;

struct PageDesc {
  int64_t *src;    // [pages][16] source row offset within a layer (no head offset), -(i+1) for span i, kNoWrite
  int2 *dep;       // [pages] range of compacted pages that read this old page
};

// One warp per (sequence, compacted page): where each of its 16 entries comes
// from, and which compacted pages read the same page of the old layout.
__global__ void __launch_bounds__(256) rollback_map_kernel(MoveArgs a, PlanArrays arr, PageDesc pd, int D) {
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

struct UnitMeta {
  int unit, b, layer, p, nh, h0, dep_lo, dep_hi;
  int64_t src[kPageSize];
};

template <int D>
__global__ void __launch_bounds__(kMoveThreads) rollback_move_kernel(MoveArgs a, PlanArrays arr, PageDesc pd) {
  constexpr int CPR = D / 8;                                   // 16-byte chunks per (kv, head) row
  constexpr int NH = kUnitBytes / (2 * kPageSize * D * 2);     // KV heads per unit
  constexpr int CHUNKS = 2 * NH * kPageSize * CPR;
  static_assert(CHUNKS == kChunksPerThread * kMoveThreads, "unit size");
  // Chunk c = tid + it * 256 of a unit is 16-byte column c % CPR of row
  // c / CPR = ((kv * NH + h) * 16 + slot).  256 is a multiple of 16 * CPR, so
  // a thread's column and slot are the same for every it; only (kv, h) vary.
  const int tid = threadIdx.x, lane_id = tid & 31, warp = tid >> 5;
  const int my_col = tid % CPR;
  const int my_slot = (tid / CPR) % kPageSize;
  const int my_kvh0 = tid / (CPR * kPageSize);
  constexpr int KVH_STEP = kMoveThreads / (CPR * kPageSize);

  extern __shared__ __align__(16) uint8_t ring[];              // kRing x 32 KB of unit data
  __shared__ UnitMeta meta[kMeta];
  __shared__ int s_last, s_abort, s_done;

  const PlanHeader *hdr = arr.hdr;
  const int total = hdr->total_units;
  const int epoch = hdr->epoch;
  const int Hkv = a.n_kv_heads;
  const int64_t head_stride = (int64_t)kPageSize * D;
  const int64_t kv_stride = head_stride * Hkv;
  const int64_t layer_stride = kv_stride * 2 * a.n_pages;

  // warp 1: describe this CTA's next unit (units blockIdx.x, blockIdx.x +
  // gridDim.x, ... in increasing order) from its precomputed description
  int next_unit = blockIdx.x;
  auto describe = [&](int m) {
    int u = 0, b = 0, ln = 0, k = 0;
    if (lane_id == 0) {
      u = next_unit;
      if (u < total) {
        b = find_seq(arr.unit_base, a.B, u);
        const int rem = u - arr.unit_base[b];
        const int nd = arr.n_dest[b];
        ln = rem / nd;
        k = rem % nd;
      }
    }
    next_unit += gridDim.x;
    u = __shfl_sync(0xffffffffu, u, 0);
    UnitMeta &M = meta[m];
    if (u >= total) {
      if (lane_id == 0) M.unit = u;
      return;
    }
    b = __shfl_sync(0xffffffffu, b, 0);
    ln = __shfl_sync(0xffffffffu, ln, 0);
    k = __shfl_sync(0xffffffffu, k, 0);
    const int idx = arr.unit_base[b] / a.n_lanes + k;
    if (lane_id < kPageSize) M.src[lane_id] = pd.src[(int64_t)idx * kPageSize + lane_id];
    if (lane_id == 0) {
      const int2 dep = pd.dep[idx];
      const int h0 = (ln % a.n_head_groups) * NH;
      M.unit = u;
      M.b = b;
      M.layer = ln / a.n_head_groups;
      M.p = arr.first_page[b] + k;
      M.h0 = h0;
      M.nh = min(NH, Hkv - h0);
      M.dep_lo = dep.x;
      M.dep_hi = dep.y;
    }
  };

  // every thread: start the copies of the unit in meta[m] into ring stage st
  auto issue = [&](int m, int st) {
    const UnitMeta &M = meta[m];
    if (M.unit < total) {
      const int64_t src = M.src[my_slot];
      uint8_t *dst = ring + st * kUnitBytes;
      const int64_t base = M.layer * layer_stride + M.h0 * head_stride + my_col * 8;
#pragma unroll
      for (int it = 0; it < kChunksPerThread; ++it) {
        const int kvh = my_kvh0 + it * KVH_STEP;
        const int h = kvh % NH, kv = kvh / NH;
        if (h < M.nh && src != kNoWrite) {
          const uint16_t *g;
          if (src >= 0) {
            g = a.pool + base + src + kv * kv_stride + h * head_stride;
          } else {
            const int64_t i = -src - 1;
            g = (kv ? a.sur_v : a.sur_k) + ((i * a.n_layers + M.layer) * Hkv + M.h0 + h) * D + my_col * 8;
          }
          cp_async_16(dst + (tid + it * kMoveThreads) * 16, g);
        }
      }
    }
    cp_async_commit();   // one group per ring slot, empty or not
  };

  if (tid == 0) s_abort = 0;
  // prologue: units 0 .. kRing-2 in flight, unit kRing-1 described
  if (warp == 1) describe(0);
  __syncthreads();
  for (int k = 0; k < kRing - 1; ++k) {
    issue(k % kMeta, k % kRing);
    if (warp == 1) describe((k + 1) % kMeta);
    __syncthreads();
  }
  for (int cur = 0;; ++cur) {
    const int head = cur + kRing - 1;
    issue(head % kMeta, head % kRing);
    cp_async_wait<kRing - 1>();          // this thread's copies of unit `cur` have landed
    __syncthreads();
    const UnitMeta &M = meta[cur % kMeta];
    if (tid == 0) {
      const int u = M.unit;
      s_done = u >= total;    // this CTA's units increase: nothing younger is valid either
      if (u < total) {
        const int p = M.p;
        // release: every copy of this unit has landed (wait_group + barrier)
        st_release(&arr.flags[u], epoch);
        // wait for the units that read old page p (all have smaller indices)
        for (int q = M.dep_lo; q <= M.dep_hi && q >= 0 && q < p; ++q) {
          const int uq = u - (p - q);
          if (ld_acquire(&arr.flags[uq]) == epoch) continue;
          const uint64_t t0 = globaltimer();
          bool ok = false;
          while (!ok) {
#pragma unroll 1
            for (int i = 0; i < 64 && !ok; ++i) ok = (ld_acquire(&arr.flags[uq]) == epoch);
            if (!ok && globaltimer() - t0 > kWaitLimitNs) break;
          }
          if (!ok) {
            set_error(a.status, UMIM_ERR_TIMEOUT);
            s_abort = 1;
            break;
          }
        }
      }
    }
    if (warp == 1) describe((head + 1) % kMeta);
    __syncthreads();
    if (s_done) break;
    const int64_t src = M.src[my_slot];
    if (!s_abort && src != kNoWrite) {
      const int32_t *bt = a.block_table + (int64_t)M.b * a.max_pages;
      const int64_t dst = M.layer * layer_stride + M.h0 * head_stride +
                          (int64_t)bt[M.p] * (kv_stride * 2) + my_slot * D + my_col * 8;
      const uint8_t *stage = ring + (cur % kRing) * kUnitBytes;
#pragma unroll
      for (int it = 0; it < kChunksPerThread; ++it) {
        const int kvh = my_kvh0 + it * KVH_STEP;
        const int h = kvh % NH, kv = kvh / NH;
        if (h < M.nh) {
          const uint4 v = *reinterpret_cast<const uint4 *>(stage + (tid + it * kMoveThreads) * 16);
          st_v4(a.pool + dst + kv * kv_stride + h * head_stride, v);
        }
      }
    }
    __syncthreads();   // stage cur % kRing is refilled by the next issue
  }
  cp_async_wait<0>();

  // ---- the last CTA to finish truncates block tables and updates lengths ----
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
  const int hpu = std::max(1, kUnitBytes / (2 * kPageSize * head_dim * 2));
  const int groups = (n_kv_heads + hpu - 1) / hpu;
  const size_t units = (size_t)B * n_layers * groups * (size_t)max_pages;
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
  const int hp = kUnitBytes / (2 * kPageSize * D * 2);     // heads per unit (the kernel's NH)
  const int groups = (kv->n_kv_heads + hp - 1) / hp;
  PlanArrays arr = plan_carve(ws, B, S);
  int32_t *status = dev_status ? dev_status : &arr.hdr->status;
  const size_t units = (size_t)B * kv->n_layers * groups * (size_t)max_pages;
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
  pa.n_lanes = kv->n_layers * groups;
  pa.status = status;
  pa.cu_seqlens_out = nullptr;
  trace_mark(stream, "rollback.plan");
  if (launch_span_plan(pa, arr, stream) != cudaSuccess) return UMIM_ERR_CUDA;

  MoveArgs ma{};
  ma.pool = static_cast<uint16_t *>(kv->base);
  ma.n_lanes = kv->n_layers * groups;
  ma.n_layers = kv->n_layers;
  ma.n_pages = kv->n_pages;
  ma.n_kv_heads = kv->n_kv_heads;
  ma.head_dim = D;
  ma.heads_per_unit = hp;
  ma.n_head_groups = groups;
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
  const int smem = kRing * kUnitBytes;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return UMIM_ERR_CUDA;
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kMoveThreads, smem) != cudaSuccess || per_sm < 1)
    per_sm = 1;
  const int grid = std::max(1, num_sms) * per_sm;   // every CTA resident (cooperative launch)
  trace_mark(stream, "rollback.map");
  rollback_map_kernel<<<dim3((unsigned)std::max(1, ceil_div(max_pages, 8)), (unsigned)B), 256, 0, stream>>>(ma, arr,
                                                                                                         pd, D);
  trace_mark(stream, "rollback.move");
  void *args[] = {&ma, &arr, &pd};
  if (cudaLaunchCooperativeKernel(reinterpret_cast<const void *>(kern), dim3(grid), dim3(kMoveThreads), args,
                                  (size_t)smem, stream) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, nullptr);
  return cudaGetLastError() == cudaSuccess ? UMIM_OK : UMIM_ERR_CUDA;
}

}  // namespace umim
