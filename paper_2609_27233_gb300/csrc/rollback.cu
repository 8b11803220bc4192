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

__device__ __forceinline__ void cp_async_16(uint32_t smem, const void *gmem) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_1() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_0() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

constexpr int kMoveWarps = kMoveThreads / 32;

// One warp per unit = one (layer, K|V, head) 16 x D tile of a compacted page.
// Lane l moves 16-byte chunks c = l + 32 it of the tile: row c / CPR (the
// slot), column c % CPR.  Each warp runs a two-deep pipeline over its units
// (gw, gw + warps, ...): the copies of unit i+1 into one half of the warp's
// shared buffer are in flight while unit i is published, its dependencies
// are checked and it is written out from the other half.  The release that
// publishes unit i therefore only orders stores issued one iteration ago.
template <int D>
__global__ void __launch_bounds__(kMoveThreads) rollback_move_kernel(MoveArgs a, PlanArrays arr, PageDesc pd) {
  constexpr int CPR = D / 8;                       // 16-byte chunks per row
  constexpr int PER_LANE = kPageSize * CPR / 32;   // 8 (D=128) or 4 (D=64)
  constexpr int SLOT_STEP = 32 / CPR;              // slots advanced per it
  constexpr int TILE_BYTES = kPageSize * D * 2;
  extern __shared__ __align__(16) uint8_t move_smem[];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int gw = blockIdx.x * kMoveWarps + wid;
  const int nw = gridDim.x * kMoveWarps;
  const int my_col = lane % CPR;
  const int my_slot0 = lane / CPR;
  const uint32_t wbuf = smem_u32(move_smem + wid * 2 * TILE_BYTES);
  __shared__ int s_last;

  const PlanHeader *hdr = arr.hdr;
  const int total = hdr->total_units;
  const int epoch = hdr->epoch;
  const int Hkv = a.n_kv_heads;
  const int64_t head_stride = (int64_t)kPageSize * D;
  const int64_t kv_stride = head_stride * Hkv;
  const int64_t page_stride = kv_stride * 2;
  const int64_t layer_stride = page_stride * a.n_pages;

  struct Unit {
    int u, b, p;
    int2 dep;
    int64_t tile;       // element offset of the tile (layer, kv, head) within a page, plus this lane's column
    uint32_t mask;      // which of this lane's chunks are written
  };
  // describe unit u and start its copies into buffer half `half`
  auto start = [&](int u, int half) {
    Unit U;
    U.u = u;
    U.mask = 0;
    if (u >= total) {
      cp_async_commit();
      return U;
    }
    const int b = find_seq(arr.unit_base, a.B, u);
    const int rem = u - arr.unit_base[b];
    const int nd = arr.n_dest[b];
    const int tl = rem / nd, k = rem % nd;
    const int layer = tl / (2 * Hkv);
    const int kv = (tl / Hkv) & 1;
    const int h = tl % Hkv;
    const int64_t idx = (int64_t)b * a.max_pages + k;
    U.b = b;
    U.p = arr.first_page[b] + k;
    U.dep = pd.dep[idx];
    U.tile = layer * layer_stride + kv * kv_stride + h * head_stride + my_col * 8;
    const int64_t my_src = lane < kPageSize ? pd.src[idx * kPageSize + lane] : kNoWrite;
    const uint16_t *sur = kv ? a.sur_v : a.sur_k;
    const uint32_t dst = wbuf + half * TILE_BYTES;
#pragma unroll
    for (int it = 0; it < PER_LANE; ++it) {
      const int slot = my_slot0 + it * SLOT_STEP;
      const int64_t src = __shfl_sync(0xffffffffu, my_src, slot);
      if (src == kNoWrite) continue;
      U.mask |= 1u << it;
      const uint16_t *g;
      if (src >= 0) {
        g = a.pool + U.tile + src;
      } else {
        const int64_t i = -src - 1;
        g = sur + ((i * a.n_layers + layer) * Hkv + h) * D + my_col * 8;
      }
      cp_async_16(dst + (lane + it * 32) * 16, g);
    }
    cp_async_commit();
    return U;
  };

  bool abort = false;
  int half = 0;
  Unit cur = start(gw, 0);
  while (cur.u < total) {
    const Unit nxt = start(cur.u + nw, half ^ 1);
    cp_async_wait_1();     // this lane's copies of `cur` have landed
    __syncwarp();          // ... and every other lane's
    int ok = 1;
    if (lane == 0) {
      // release: the copies of this unit are complete and ordered before it
      st_release(&arr.flags[cur.u], epoch);
      // wait for the units that read this tile of old page p (smaller indices)
      for (int q = cur.dep.x; q <= cur.dep.y && q >= 0 && q < cur.p; ++q) {
        const int uq = cur.u - (cur.p - q);
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
    if (!ok) {
      abort = true;
      break;
    }
    const int64_t dst = cur.tile + (int64_t)a.block_table[(int64_t)cur.b * a.max_pages + cur.p] * page_stride;
    const uint32_t src_s = wbuf + half * TILE_BYTES;
#pragma unroll
    for (int it = 0; it < PER_LANE; ++it) {
      if (cur.mask & (1u << it)) {
        uint4 v;
        asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                     : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                     : "r"(src_s + (lane + it * 32) * 16));
        st_v4(a.pool + dst + (my_slot0 + it * SLOT_STEP) * D, v);
      }
    }
    __syncwarp();          // the buffer half is refilled two units later
    cur = nxt;
    half ^= 1;
  }
  (void)abort;
  cp_async_wait_0();

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
  pa.page_src = pd.src;
  pa.page_dep = pd.dep;
  pa.page_stride = (int64_t)kPageSize * D * kv->n_kv_heads * 2;
  pa.head_dim = D;
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
  const int smem = kMoveWarps * 2 * kPageSize * D * 2;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return UMIM_ERR_CUDA;
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kMoveThreads, smem) != cudaSuccess || per_sm < 1)
    per_sm = 1;
  const int grid = std::max(1, num_sms) * per_sm;   // every CTA resident (cooperative launch)
  trace_mark(stream, "rollback.move");
  void *args[] = {&ma, &arr, &pd};
  if (cudaLaunchCooperativeKernel(reinterpret_cast<const void *>(kern), dim3(grid), dim3(kMoveThreads), args,
                                  (size_t)smem, stream) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, nullptr);
  return cudaGetLastError() == cudaSuccess ? UMIM_OK : UMIM_ERR_CUDA;
}

}  // namespace umim
