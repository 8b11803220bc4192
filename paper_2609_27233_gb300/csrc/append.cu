// Decode-step cache update (App. E "Decoding-Time Merging and KV-Cache
// Update", Fig. 2 steps (2) and (3)).
//
// Append: a generated token that completes no merge is forwarded normally
// and its K and V rows are appended, one entry per layer, at slot
// L = seq_lens[b] of the sequence's paged cache.
//
// Append with a suffix merge: after each generated token the recent suffix
// is checked against the merge rules; when an n-gram matches, its stored
// entries are cropped and one surrogate KV entry takes their place.  Per
// sequence b with L = seq_lens[b] and k = merge_k[b]:
//   k == 0  the new entry is appended at slot L;
//   k >= 1  the new entry and the k - 1 entries before it form the merged
//           span: surrogate row merge_row[b] goes to slot s = L + 1 - k, the
//           length becomes s + 1, and a page the append opened or that no
//           longer holds an entry is released (at most one for k <= 16).
// The result equals the append followed by a rollback of the suffix span
// (s, k); the appended entry of a merging sequence is never written since
// the merge replaces it.  No entry moves: a suffix has nothing after it.
//
// One thread-block cluster per sequence.  Every CTA of the cluster reads L,
// k and the destination page and takes the same decision; after a cluster
// barrier (every CTA has read them) the CTAs copy their share of the 16-byte
// chunks of the (layer, K|V, head) rows, and rank 0 records the page in the
// block table, the released page and the new length.  Only this cluster
// touches sequence b, so the reads and the updates cannot race.
#include "common.cuh"

namespace umim {
namespace {

constexpr int kAppendThreads = 256;
constexpr int kUnroll = 4;        // independent 16-byte loads in flight per thread
constexpr int kMaxCluster = 8;    // CTAs per sequence (portable cluster size)

struct AppendArgs {
  uint16_t *pool;
  int32_t n_layers, n_pages, n_kv_heads;
  int32_t *block_table;
  int32_t max_pages;
  int32_t *seq_lens;
  const uint16_t *new_k, *new_v;   // [B][n_layers][Hkv][D]
  const int32_t *new_pages;        // [B] or nullptr
  int32_t *status;
  const int32_t *merge_k;          // [B] or nullptr (append only)
  const int32_t *merge_row;        // [B]
  int32_t n_rows;                  // rows of the surrogate arrays
  const uint16_t *sur_k, *sur_v;   // [n_rows][n_layers][Hkv][D]
  int32_t *released;               // [B] or nullptr
};

__device__ __forceinline__ uint4 ld_nc_v4(const uint16_t *p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

template <int D>
__global__ void __launch_bounds__(kAppendThreads) decode_update_kernel(AppendArgs a, int C) {
  griddep_wait();
  const int b = blockIdx.x / C, rank = blockIdx.x % C;
  __shared__ int s_page, s_slot, s_row, s_L, s_k;
  if (threadIdx.x == 0) {
    const int L = a.seq_lens[b];
    const int k = a.merge_k ? a.merge_k[b] : 0;
    bool ok = L >= 0 && (int64_t)L < (int64_t)a.max_pages * kPageSize && k >= 0 && k <= 16 && k <= L + 1;
    int page_L = -1;
    if (ok) {
      if (L % kPageSize == 0) page_L = a.new_pages ? a.new_pages[b] : -1;
      else page_L = a.block_table[(int64_t)b * a.max_pages + L / kPageSize];
      ok = page_L >= 0 && page_L < a.n_pages;
    }
    int slot = L, page = page_L, row = -1;
    if (ok && k > 0) {
      row = a.merge_row ? a.merge_row[b] : -1;
      slot = L + 1 - k;
      page = slot / kPageSize == L / kPageSize ? page_L : a.block_table[(int64_t)b * a.max_pages + slot / kPageSize];
      ok = row >= 0 && row < a.n_rows && page >= 0 && page < a.n_pages;
    }
    if (!ok) {
      if (rank == 0) set_error(a.status, UMIM_ERR_INVALID_ARG);
      page = -1;
    }
    s_page = page;
    s_slot = slot;
    s_row = row;
    s_L = L;
    s_k = k;
  }
  __syncthreads();
  cluster_sync();   // every CTA of this sequence has read L, k and the pages
  const int page = s_page, slot = s_slot, row = s_row, L = s_L, k = s_k;
  if (page < 0) return;   // this sequence is left unchanged

  constexpr int CPR = D / 8;   // 16-byte chunks per row
  const int Hkv = a.n_kv_heads;
  const int total = a.n_layers * 2 * Hkv * CPR;   // chunks, ordered [layer][K|V][head][chunk]
  const int64_t head_stride = (int64_t)kPageSize * D;
  const int64_t kv_stride = head_stride * Hkv;
  const int64_t page_stride = kv_stride * 2;
  const int64_t layer_stride = page_stride * a.n_pages;
  uint16_t *dst_base = a.pool + (int64_t)page * page_stride + (int64_t)(slot % kPageSize) * D;
  const uint16_t *src_k = k > 0 ? a.sur_k : a.new_k;
  const uint16_t *src_v = k > 0 ? a.sur_v : a.new_v;
  const int src_row = k > 0 ? row : b;
  if (!in_bounds(src_row, k > 0 ? a.n_rows : (int)gridDim.x / C, rank == 0 ? a.status : nullptr,
                 kSiteAppendSrcRow))
    return;
  const int64_t pool_elems = layer_stride * a.n_layers;   // debug checks
  const int stride = kAppendThreads * C;
  for (int c0 = rank * kAppendThreads + threadIdx.x; c0 < total; c0 += stride * kUnroll) {
    uint4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int c = c0 + u * stride;
      if (c < total) {
        const int r = c / CPR, col = c % CPR;
        const int layer = r / (2 * Hkv), kv = (r / Hkv) & 1, h = r % Hkv;
        const uint16_t *src = (kv ? src_v : src_k) + (((int64_t)src_row * a.n_layers + layer) * Hkv + h) * D;
        v[u] = ld_nc_v4(src + col * 8);
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int c = c0 + u * stride;
      if (c < total) {
        const int r = c / CPR, col = c % CPR;
        const int layer = r / (2 * Hkv), kv = (r / Hkv) & 1, h = r % Hkv;
        const int64_t off = layer * layer_stride + kv * kv_stride + h * head_stride + col * 8;
        if (in_bounds((dst_base - a.pool) + off, pool_elems - 7, a.status, kSiteAppendDst))
          *reinterpret_cast<uint4 *>(dst_base + off) = v[u];
      }
    }
  }
  if (rank == 0 && threadIdx.x == 0) {
    int32_t *bt = a.block_table + (int64_t)b * a.max_pages;
    if (L % kPageSize == 0) bt[L / kPageSize] = a.new_pages[b];   // the append opened this page
    const int Ln = k > 0 ? slot + 1 : L + 1;
    const int had = (L + 1 + kPageSize - 1) / kPageSize, keep = (Ln + kPageSize - 1) / kPageSize;
    int rel = -1;
    if (keep < had) {   // k <= 16: at most one page
      rel = bt[keep];
      bt[keep] = -1;
    }
    if (a.released) a.released[b] = rel;
    a.seq_lens[b] = Ln;
  }
}

umim_status launch_update(const AppendArgs &a, int head_dim, int32_t B, cudaStream_t stream, const char *label) {
  // CTAs per sequence: enough that each thread has about kUnroll chunks
  const int total = a.n_layers * 2 * a.n_kv_heads * (head_dim / 8);
  int C = (total + kAppendThreads * kUnroll - 1) / (kAppendThreads * kUnroll);
  C = C < 1 ? 1 : (C > kMaxCluster ? kMaxCluster : C);
  auto kern = head_dim == 128 ? decode_update_kernel<128> : decode_update_kernel<64>;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(B * C));
  cfg.blockDim = dim3(kAppendThreads);
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = (unsigned)C;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  trace_mark(stream, label);
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kern, a, C);
  trace_mark(stream, nullptr);
  return e == cudaSuccess ? UMIM_OK : UMIM_ERR_CUDA;
}

AppendArgs base_args(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages, int32_t *seq_lens,
                     const void *new_k, const void *new_v, const int32_t *new_pages, int32_t *dev_status) {
  AppendArgs a{};
  a.pool = static_cast<uint16_t *>(kv->base);
  a.n_layers = kv->n_layers;
  a.n_pages = kv->n_pages;
  a.n_kv_heads = kv->n_kv_heads;
  a.block_table = block_table;
  a.max_pages = max_pages;
  a.seq_lens = seq_lens;
  a.new_k = static_cast<const uint16_t *>(new_k);
  a.new_v = static_cast<const uint16_t *>(new_v);
  a.new_pages = new_pages;
  a.status = dev_status;
  return a;
}

}  // namespace

umim_status kv_append(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages, int32_t *seq_lens,
                      int32_t B, const void *new_k, const void *new_v, const int32_t *new_pages,
                      int32_t *dev_status, cudaStream_t stream) {
  const AppendArgs a = base_args(kv, block_table, max_pages, seq_lens, new_k, new_v, new_pages, dev_status);
  return launch_update(a, kv->head_dim, B, stream, "append");
}

umim_status decode_append_merge(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages, int32_t *seq_lens,
                                int32_t B, const void *new_k, const void *new_v, const int32_t *new_pages,
                                const int32_t *merge_k, const int32_t *merge_row, int32_t n_rows, const void *sur_k,
                                const void *sur_v, int32_t *released, int32_t *dev_status, cudaStream_t stream) {
  AppendArgs a = base_args(kv, block_table, max_pages, seq_lens, new_k, new_v, new_pages, dev_status);
  a.merge_k = merge_k;
  a.merge_row = merge_row;
  a.n_rows = n_rows;
  a.sur_k = static_cast<const uint16_t *>(sur_k);
  a.sur_v = static_cast<const uint16_t *>(sur_v);
  a.released = released;
  return launch_update(a, kv->head_dim, B, stream, "append_merge");
}

}  // namespace umim
