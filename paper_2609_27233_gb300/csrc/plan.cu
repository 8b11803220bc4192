// Span metadata kernel: one block per sequence validates its spans and scans
// (k_i - 1); the last block to finish builds the prefix sums over sequences.
#include "plan.cuh"

namespace umim {
namespace {

constexpr int kPlanThreads = 1024;

// Inclusive block-wide scan; every thread gets the block total.
__device__ int block_scan_incl(int v, int &total) {
  __shared__ int warp_sums[kPlanThreads / 32];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[w] = x;
  __syncthreads();
  if (w == 0) {
    int s = (lane < kPlanThreads / 32) ? warp_sums[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    if (lane < kPlanThreads / 32) warp_sums[lane] = s;
  }
  __syncthreads();
  const int add = (w > 0) ? warp_sums[w - 1] : 0;
  total = warp_sums[kPlanThreads / 32 - 1];
  __syncthreads();
  return x + add;
}

__global__ void __launch_bounds__(kPlanThreads) span_plan_kernel(PlanArgs a, PlanArrays arr) {
  griddep_wait();
  const int b = blockIdx.x;
  __shared__ int s_err, s_carry, s_last;
  if (threadIdx.x == 0) {
    s_err = 0;
    s_carry = 0;
    s_last = 0;
  }
  __syncthreads();
  const int L = a.seq_lens ? a.seq_lens[b] : a.fixed_len;
  const int lo = a.span_offsets[b], hi = a.span_offsets[b + 1];
  bool bad = (lo < 0) || (hi < lo) || (hi > a.S) || (L < 0);
  if (a.block_table && (int64_t)L > (int64_t)a.max_pages * kPageSize) bad = true;
  if (bad && threadIdx.x == 0) s_err = 1;
  __syncthreads();
  if (!s_err) {
    for (int base = lo; base < hi; base += kPlanThreads) {
      const int i = base + threadIdx.x;
      int v = 0, s = 0;
      if (i < hi) {
        s = a.span_start[i];
        const int k = a.span_len[i];
        bool ok = (k >= 1) && (s >= 0) && ((int64_t)s + k <= L);
        if (a.max_span_len > 0 && k > a.max_span_len) ok = false;
        if (i > lo) {
          const int ps = a.span_start[i - 1], pk = a.span_len[i - 1];
          if ((int64_t)ps + pk > s) ok = false;
        }
        if (!ok) s_err = 1;
        v = ok ? k - 1 : 0;
      }
      int tot;
      const int incl = block_scan_incl(v, tot);
      if (i < hi) {
        const int r = s_carry + incl;
        arr.r_incl[i] = r;
        arr.new_idx[i] = s - (r - v);
      }
      __syncthreads();
      if (threadIdx.x == 0) s_carry += tot;
      __syncthreads();
    }
    if (a.block_table) {
      const int np = ceil_div(L, kPageSize);
      for (int p = threadIdx.x; p < np; p += kPlanThreads) {
        const int pg = a.block_table[(int64_t)b * a.max_pages + p];
        if (pg < 0 || pg >= a.n_pages) s_err = 1;
      }
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const int err = s_err;
    const int Lp = err ? L : L - s_carry;
    arr.seq_L[b] = L;
    arr.seq_Lp[b] = Lp;
    int fp = 0, nd = 0;
    if (!err && hi > lo) {
      fp = a.span_start[lo] / kPageSize;
      nd = ceil_div(Lp, kPageSize) - fp;
    }
    arr.first_page[b] = fp;
    arr.n_dest[b] = nd;
    if (err) atomicOr(&arr.hdr->error, 1);
    __threadfence();
    const int done = atomicAdd(&arr.hdr->blocks_done, 1);
    s_last = (done == (int)gridDim.x - 1);
  }
  __syncthreads();
  if (!s_last) return;

  // ---- last block: prefix sums over sequences, per-call header reset ----
  __threadfence();
  const int err = atomicOr(&arr.hdr->error, 0);
  int cu_units = 0, cu_rows = 0, cu_freed = 0, cu_active = 0;
  __shared__ int s_max_dest;
  if (threadIdx.x == 0) s_max_dest = 0;
  __syncthreads();
  for (int j = threadIdx.x; j < a.B; j += kPlanThreads) atomicMax(&s_max_dest, arr.n_dest[j]);
  for (int base = 0; base < a.B; base += kPlanThreads) {
    const int j = base + threadIdx.x;
    int u = 0, r = 0, f = 0;
    if (j < a.B) {
      const int L = arr.seq_L[j], Lp = arr.seq_Lp[j];
      u = a.n_lanes * arr.n_dest[j];
      r = Lp;
      f = ceil_div(L, kPageSize) - ceil_div(Lp, kPageSize);
    }
    const int act = (j < a.B && arr.n_dest[j] > 0) ? 1 : 0;
    int tu, tr, tf, ta;
    const int iu = block_scan_incl(u, tu);
    const int ir = block_scan_incl(r, tr);
    const int iff = block_scan_incl(f, tf);
    const int ia = block_scan_incl(act, ta);
    if (j < a.B) {
      arr.unit_base[j] = cu_units + iu - u;
      arr.row_base[j] = cu_rows + ir - r;
      arr.freed_base[j] = cu_freed + iff - f;
      if (act) arr.active[cu_active + ia - 1] = j;
      if (a.cu_seqlens_out && !err) a.cu_seqlens_out[j] = cu_rows + ir - r;
    }
    cu_units += tu;
    cu_rows += tr;
    cu_freed += tf;
    cu_active += ta;
  }
  if (threadIdx.x == 0) {
    arr.unit_base[a.B] = cu_units;
    arr.row_base[a.B] = cu_rows;
    arr.freed_base[a.B] = cu_freed;
    if (a.cu_seqlens_out && !err) a.cu_seqlens_out[a.B] = cu_rows;
    PlanHeader *h = arr.hdr;
    h->total_units = err ? 0 : cu_units;
    h->total_rows = cu_rows;
    h->max_dest = err ? 0 : s_max_dest;
    h->n_active = err ? 0 : cu_active;
    h->skip = err ? 1 : 0;
    h->epoch = h->epoch + 1;
    h->ticket = 0;
    h->done_ctas = 0;
    h->blocks_done = 0;
    h->error = 0;
    if (err) set_error(a.status, UMIM_ERR_INVALID_ARG);
    __threadfence();
  }
}

}  // namespace

cudaError_t launch_span_plan(const PlanArgs &args, const PlanArrays &arr, cudaStream_t stream) {
  return launch_pdl(span_plan_kernel, dim3(args.B), dim3(kPlanThreads), 0, stream, args, arr);
}

}  // namespace umim
