// Decode-step KV append (App. E "Decoding-Time Merging and KV-Cache Update",
// Fig. 2 step (2)): a generated token that completes no merge is forwarded
// normally and its K and V rows are appended, one entry per layer, at slot
// L = seq_lens[b] of the sequence's paged cache.
//
// One CTA per sequence: thread 0 reads L and the destination page (the
// caller's new page when L opens one), every thread moves 16-byte chunks of
// the (layer, K|V, head) rows, and thread 0 then records the page in the
// block table and the new length.  Only this CTA touches sequence b, so the
// read of L and the update of seq_lens[b] cannot race.
#include "common.cuh"

namespace umim {
namespace {

constexpr int kAppendThreads = 256;
constexpr int kUnroll = 4;   // independent 16-byte loads in flight per thread

struct AppendArgs {
  uint16_t *pool;
  int32_t n_layers, n_pages, n_kv_heads;
  int32_t *block_table;
  int32_t max_pages;
  int32_t *seq_lens;
  const uint16_t *new_k, *new_v;   // [B][n_layers][Hkv][D]
  const int32_t *new_pages;        // [B] or nullptr
  int32_t *status;
};

__device__ __forceinline__ uint4 ld_nc_v4(const uint16_t *p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

template <int D>
__global__ void __launch_bounds__(kAppendThreads) kv_append_kernel(AppendArgs a) {
  griddep_wait();
  const int b = blockIdx.x;
  __shared__ int s_page, s_L;
  if (threadIdx.x == 0) {
    const int L = a.seq_lens[b];
    int page = -1;
    if (L >= 0 && (int64_t)L < (int64_t)a.max_pages * kPageSize) {
      if (L % kPageSize == 0) page = a.new_pages ? a.new_pages[b] : -1;
      else page = a.block_table[(int64_t)b * a.max_pages + L / kPageSize];
      if (page >= a.n_pages) page = -1;
    }
    if (page < 0) set_error(a.status, UMIM_ERR_INVALID_ARG);
    s_page = page;
    s_L = L;
  }
  __syncthreads();
  const int page = s_page, L = s_L;
  if (page < 0) return;   // this sequence is left unchanged

  constexpr int CPR = D / 8;   // 16-byte chunks per row
  const int Hkv = a.n_kv_heads;
  const int total = a.n_layers * 2 * Hkv * CPR;   // chunks, ordered [layer][K|V][head][chunk]
  const int64_t head_stride = (int64_t)kPageSize * D;
  const int64_t kv_stride = head_stride * Hkv;
  const int64_t page_stride = kv_stride * 2;
  const int64_t layer_stride = page_stride * a.n_pages;
  uint16_t *dst_base = a.pool + (int64_t)page * page_stride + (int64_t)(L % kPageSize) * D;
  for (int c0 = threadIdx.x; c0 < total; c0 += kAppendThreads * kUnroll) {
    uint4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int c = c0 + u * kAppendThreads;
      if (c < total) {
        const int row = c / CPR, col = c % CPR;
        const int layer = row / (2 * Hkv), kv = (row / Hkv) & 1, h = row % Hkv;
        const uint16_t *src = (kv ? a.new_v : a.new_k) + (((int64_t)b * a.n_layers + layer) * Hkv + h) * D;
        v[u] = ld_nc_v4(src + col * 8);
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int c = c0 + u * kAppendThreads;
      if (c < total) {
        const int row = c / CPR, col = c % CPR;
        const int layer = row / (2 * Hkv), kv = (row / Hkv) & 1, h = row % Hkv;
        *reinterpret_cast<uint4 *>(dst_base + layer * layer_stride + kv * kv_stride + h * head_stride + col * 8) =
            v[u];
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (L % kPageSize == 0) a.block_table[(int64_t)b * a.max_pages + L / kPageSize] = page;
    a.seq_lens[b] = L + 1;
  }
}

}  // namespace

umim_status kv_append(const umim_paged_kv *kv, int32_t *block_table, int32_t max_pages, int32_t *seq_lens,
                      int32_t B, const void *new_k, const void *new_v, const int32_t *new_pages,
                      int32_t *dev_status, cudaStream_t stream) {
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
  auto kern = kv->head_dim == 128 ? kv_append_kernel<128> : kv_append_kernel<64>;
  trace_mark(stream, "append");
  const cudaError_t e = launch_pdl(kern, dim3((unsigned)B), dim3(kAppendThreads), 0, stream, a);
  trace_mark(stream, nullptr);
  return e == cudaSuccess ? UMIM_OK : UMIM_ERR_CUDA;
}

}  // namespace umim
