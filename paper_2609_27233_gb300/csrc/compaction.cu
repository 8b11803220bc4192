// Packed compressed prompt embeddings with contiguous positions
// (App. E "Prompt Merging", App. C.5, App. J.4): row j of prompt b is the
// surrogate of span i when j is that span's compressed index, otherwise the
// static embedding of the kept token t = j + r_i (span i = last span whose
// compressed index is below j).  One warp per output row, 16-byte moves.
#include <algorithm>

#include "plan.cuh"

namespace umim {
namespace {

struct CompactArgs {
  const uint4 *table;
  int64_t vocab;
  int d;
  const int32_t *token_ids;
  int L;
  int B;
  const int32_t *span_offsets;
  const float *surrogates;
  uint4 *out;
  int64_t capacity;
  int32_t *position_ids;
  int32_t *status;
};

__device__ __forceinline__ int last_le(const int32_t *key, int lo, int hi, int x) {
  int l = lo, h = hi;
  while (l < h) {
    const int m = (l + h) >> 1;
    if (key[m] <= x) l = m + 1;
    else h = m;
  }
  return l - 1;
}

__global__ void __launch_bounds__(256) compact_kernel(CompactArgs a, PlanArrays arr) {
  griddep_wait();
  const PlanHeader *hdr = arr.hdr;
  if (hdr->skip) return;
  const int total = hdr->total_rows;
  if (total > a.capacity) {
    if (blockIdx.x == 0 && threadIdx.x == 0) set_error(a.status, UMIM_ERR_INVALID_ARG);
    return;
  }
  const int lane = threadIdx.x & 31;
  const int vec = a.d / 8;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t r = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < total; r += nwarps) {
    const int b = last_le(arr.row_base, 0, a.B, (int)r);
    const int j = (int)r - arr.row_base[b];
    const int lo = a.span_offsets[b], hi = a.span_offsets[b + 1];
    const int i = last_le(arr.new_idx, lo, hi, j);
    uint4 *dst = a.out + r * vec;
    if (i >= lo && arr.new_idx[i] == j) {
      const float4 *z = reinterpret_cast<const float4 *>(a.surrogates + (int64_t)i * a.d);
      for (int v = lane; v < vec; v += 32) {
        const float4 x = z[2 * v], y = z[2 * v + 1];
        __nv_bfloat162 p0 = __floats2bfloat162_rn(x.x, x.y), p1 = __floats2bfloat162_rn(x.z, x.w);
        __nv_bfloat162 p2 = __floats2bfloat162_rn(y.x, y.y), p3 = __floats2bfloat162_rn(y.z, y.w);
        uint4 o;
        o.x = *reinterpret_cast<uint32_t *>(&p0);
        o.y = *reinterpret_cast<uint32_t *>(&p1);
        o.z = *reinterpret_cast<uint32_t *>(&p2);
        o.w = *reinterpret_cast<uint32_t *>(&p3);
        dst[v] = o;
      }
    } else {
      const int t = (i >= lo) ? j + arr.r_incl[i] : j;
      const bool t_ok = in_bounds(t, a.L, lane == 0 ? a.status : nullptr, kSiteCompactToken);
      const int id = t_ok ? a.token_ids[(int64_t)b * a.L + t] : 0;
      const bool ok = id >= 0 && id < a.vocab && t_ok;
      if (!ok && lane == 0) set_error(a.status, UMIM_ERR_INVALID_ARG);
      const uint4 *src = a.table + (int64_t)(ok ? id : 0) * vec;
      for (int v = lane; v < vec; v += 32) dst[v] = ok ? __ldg(src + v) : make_uint4(0, 0, 0, 0);
    }
    if (lane == 0) a.position_ids[r] = j;
  }
}

}  // namespace

size_t build_compressed_workspace_bytes(int B, int S) { return plan_bytes(B, S); }

umim_status build_compressed(const void *embeddings, int64_t vocab, int d, const int32_t *token_ids, int B, int L,
                             const int32_t *span_offsets, const int32_t *span_start, const int32_t *span_len,
                             int S, const float *surrogates, void *out_embeds, int64_t capacity,
                             int32_t *position_ids, int32_t *cu_seqlens, void *ws, int32_t *dev_status,
                             cudaStream_t stream, int num_sms) {
  PlanArrays arr = plan_carve(ws, B, S);
  int32_t *status = dev_status ? dev_status : &arr.hdr->status;
  PlanArgs pa{};
  pa.seq_lens = nullptr;
  pa.fixed_len = L;
  pa.span_offsets = span_offsets;
  pa.span_start = span_start;
  pa.span_len = span_len;
  pa.B = B;
  pa.S = S;
  pa.max_span_len = 0;
  pa.block_table = nullptr;
  pa.n_lanes = 0;
  pa.status = status;
  pa.cu_seqlens_out = cu_seqlens;
  trace_mark(stream, "compact.plan");
  if (launch_span_plan(pa, arr, stream) != cudaSuccess) return UMIM_ERR_CUDA;
  CompactArgs a;
  a.table = static_cast<const uint4 *>(embeddings);
  a.vocab = vocab;
  a.d = d;
  a.token_ids = token_ids;
  a.L = L;
  a.B = B;
  a.span_offsets = span_offsets;
  a.surrogates = surrogates;
  a.out = static_cast<uint4 *>(out_embeds);
  a.capacity = capacity;
  a.position_ids = position_ids;
  a.status = status;
  const int64_t rows = (int64_t)B * L;
  const int blocks = (int)std::max<int64_t>(1, std::min<int64_t>((rows + 7) / 8, (int64_t)num_sms * 16));
  trace_mark(stream, "compact.rows");
  if (launch_pdl(compact_kernel, dim3(blocks), dim3(256), 0, stream, a, arr) != cudaSuccess) return UMIM_ERR_CUDA;
  trace_mark(stream, nullptr);
  return UMIM_OK;
}

}  // namespace umim
