// Aligned predictive distillation, the training-side step of the method
// (App. F "Predictive Distillation Loss and Alignment Metrics", Algorithm 1,
// the masked distillation loss):
//
//  * alignment: per sample, the teacher keeps every retained token and the
//    last position of each merged span (the surrogate's anchor) from the
//    first span's start s_b on; the student keeps the last N_b positions of
//    its compressed sequence; Pack pairs them in order.  A kept position t
//    pairs with the compressed index pi(t) = t - r(t) (App. J.4), so the k-th
//    pair of sample b is (teacher row t_cu[b] + t, student row s_cu[b] + pi(t))
//    with k = pi(t) - s_b.  Two kernels: a per-sample plan (validation, the
//    removed-placeholder scan, prefix sums in the last block) and a row writer.
//
//  * soft-target cross-entropy over the full vocabulary and its gradient with
//    respect to the student logits:
//      L = -(1/N) sum_pairs sum_v P^T(v) log(P^S(v) + eps)
//      dL/ds_v = -(1/N) (a_v - P^S(v) sum_u a_u),  a_u = P^T(u) P^S(u) / (P^S(u) + eps)
//    One thread-block cluster of C CTAs per student row (9 at the Llama-3
//    vocabulary): each CTA holds 1/C of the vocabulary of the teacher and
//    student rows in registers (fp32), so every logit byte is read once and
//    every gradient byte written once.  Rows arrive by 1-D TMA bulk copies
//    into a ring of shared-memory stages that a copy warp refills; the
//    softmax statistics and the two sums are exchanged between the cluster's
//    CTAs through distributed shared memory, and each warp keeps two rows in
//    flight (the finished one in tensor memory) so that every exchange is
//    waited for one compute phase after it was pushed.  Student rows that are
//    in no pair get a zero gradient.  The loss is summed from the per-pair
//    losses, in pair order, by the last CTA to finish.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <mutex>
#include <type_traits>

#include <cuda_fp16.h>

#include "common.cuh"

namespace umim {
namespace {

// ===========================================================================
// alignment
// ===========================================================================
constexpr int kAlignThreads = 1024;

struct AlignHeader {
  int32_t status;       // status word when the caller passes none
  int32_t blocks_done;  // plan blocks that finished (reset by the last one)
  int32_t error;        // OR of per-sample errors this call
  int32_t skip;         // 1: invalid input or too many pairs, nothing written
  int32_t pad[60];
};
static_assert(sizeof(AlignHeader) == 256, "align header size");

struct AlignArrays {
  AlignHeader *hdr;
  int32_t *r_before;  // [S] placeholders removed before span i, within its sample
  int32_t *L;         // [B] original length
  int32_t *first;     // [B] first span start (the compressed length when no span)
  int32_t *t_cu;      // [B+1] teacher rows
  int32_t *s_cu;      // [B+1] student rows
  int32_t *p_cu;      // [B+1] pairs
  int32_t *Lc;        // [B] compressed length
};

inline size_t a256(size_t x) { return (x + 255) & ~size_t(255); }

size_t align_ws_bytes(int B, int S) {
  const size_t s4 = sizeof(int32_t) * (size_t)std::max(S, 1), b4 = sizeof(int32_t) * (size_t)std::max(B, 1);
  const size_t b14 = sizeof(int32_t) * (size_t)(B + 1);
  return a256(sizeof(AlignHeader)) + a256(s4) + 3 * a256(b4) + 3 * a256(b14);
}

AlignArrays align_carve(void *ws, int B, int S) {
  char *p = static_cast<char *>(ws);
  auto take = [&](size_t n) {
    char *r = p;
    p += a256(n);
    return r;
  };
  const size_t s4 = sizeof(int32_t) * (size_t)std::max(S, 1), b4 = sizeof(int32_t) * (size_t)std::max(B, 1);
  const size_t b14 = sizeof(int32_t) * (size_t)(B + 1);
  AlignArrays a;
  a.hdr = reinterpret_cast<AlignHeader *>(take(sizeof(AlignHeader)));
  a.r_before = reinterpret_cast<int32_t *>(take(s4));
  a.L = reinterpret_cast<int32_t *>(take(b4));
  a.first = reinterpret_cast<int32_t *>(take(b4));
  a.Lc = reinterpret_cast<int32_t *>(take(b4));
  a.t_cu = reinterpret_cast<int32_t *>(take(b14));
  a.s_cu = reinterpret_cast<int32_t *>(take(b14));
  a.p_cu = reinterpret_cast<int32_t *>(take(b14));
  return a;
}

struct AlignArgs {
  const int32_t *seq_lens;
  const int32_t *span_offsets, *span_start, *span_len;
  int32_t B, S;
  int32_t capacity;
  int32_t *pair_offsets;   // [B+1] out
  int32_t *teacher_rows;   // [capacity] out
  int32_t *student_rows;   // [capacity] out
  int32_t *student_cu;     // [B+1] out or nullptr
  int32_t *status;
};

// Inclusive block-wide scan of 64-bit values; every thread gets the total.
__device__ long long scan_incl_ll(long long v, long long &total) {
  __shared__ long long warp_sums[kAlignThreads / 32];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  long long x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const long long y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[w] = x;
  __syncthreads();
  if (w == 0) {
    long long s = warp_sums[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    warp_sums[lane] = s;
  }
  __syncthreads();
  const long long add = (w > 0) ? warp_sums[w - 1] : 0;
  total = warp_sums[kAlignThreads / 32 - 1];
  __syncthreads();
  return x + add;
}

// One block per sample: validate its spans, scan (n_i - 1), record L, the
// compressed length and the first span start.  The last block to finish
// builds the prefix sums and decides whether the call writes anything.
__global__ void __launch_bounds__(kAlignThreads) align_plan_kernel(AlignArgs a, AlignArrays arr) {
  griddep_wait();
  const int b = blockIdx.x;
  __shared__ int s_err, s_last;
  __shared__ long long s_carry;
  if (threadIdx.x == 0) {
    s_err = 0;
    s_last = 0;
    s_carry = 0;
  }
  __syncthreads();
  const int L = a.seq_lens[b];
  const int lo = a.span_offsets[b], hi = a.span_offsets[b + 1];
  if (threadIdx.x == 0 && (L < 0 || lo < 0 || hi < lo || hi > a.S)) s_err = 1;
  __syncthreads();
  if (!s_err) {
    for (int base = lo; base < hi; base += kAlignThreads) {
      const int i = base + threadIdx.x;
      long long v = 0;
      if (i < hi) {
        const int s = a.span_start[i], n = a.span_len[i];
        bool ok = n >= 1 && s >= 0 && (long long)s + n <= L;
        if (i > lo && (long long)a.span_start[i - 1] + a.span_len[i - 1] > s) ok = false;
        if (!ok) s_err = 1;
        v = ok ? n - 1 : 0;
      }
      long long tot;
      const long long incl = scan_incl_ll(v, tot);
      if (i < hi) arr.r_before[i] = (int)(s_carry + incl - v);
      __syncthreads();
      if (threadIdx.x == 0) s_carry += tot;
      __syncthreads();
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const int err = s_err;
    const int Lc = err ? 0 : L - (int)s_carry;
    arr.L[b] = err ? 0 : L;
    arr.Lc[b] = Lc;
    arr.first[b] = (!err && hi > lo) ? a.span_start[lo] : Lc;
    if (err) atomicOr(&arr.hdr->error, 1);
    __threadfence();
    s_last = atomicAdd(&arr.hdr->blocks_done, 1) == (int)gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;

  __threadfence();
  int err = atomicOr(&arr.hdr->error, 0);
  long long ct = 0, cs = 0, cp = 0;
  for (int base = 0; base < a.B; base += kAlignThreads) {
    const int j = base + threadIdx.x;
    long long t = 0, s = 0, p = 0;
    if (j < a.B) {
      t = arr.L[j];
      s = arr.Lc[j];
      p = arr.Lc[j] - arr.first[j];
    }
    long long tt, ts, tp;
    const long long it = scan_incl_ll(t, tt), is = scan_incl_ll(s, ts), ip = scan_incl_ll(p, tp);
    if (j < a.B) {
      arr.t_cu[j] = (int)(ct + it - t);
      arr.s_cu[j] = (int)(cs + is - s);
      arr.p_cu[j] = (int)(cp + ip - p);
    }
    ct += tt;
    cs += ts;
    cp += tp;
  }
  // rows and pairs are int32 indices; too many pairs for the outputs is an error
  if (ct > INT32_MAX || cp > a.capacity) err = 1;
  if (!err && a.student_cu)
    for (int j = threadIdx.x; j < a.B; j += kAlignThreads) a.student_cu[j] = arr.s_cu[j];
  if (!err)
    for (int j = threadIdx.x; j < a.B; j += kAlignThreads) a.pair_offsets[j] = arr.p_cu[j];
  if (threadIdx.x == 0) {
    arr.t_cu[a.B] = (int)ct;
    arr.s_cu[a.B] = (int)cs;
    arr.p_cu[a.B] = (int)cp;
    if (!err) {
      a.pair_offsets[a.B] = (int)cp;
      if (a.student_cu) a.student_cu[a.B] = (int)cs;
    }
    AlignHeader *h = arr.hdr;
    h->skip = err ? 1 : 0;
    h->blocks_done = 0;
    h->error = 0;
    if (err) set_error(a.status, UMIM_ERR_INVALID_ARG);
    __threadfence();
  }
}

// last index i in [lo, hi) with key[i] <= x (lo - 1 if none)
__device__ __forceinline__ int last_le(const int32_t *key, int lo, int hi, int x) {
  int l = lo, h = hi;
  while (l < h) {
    const int m = (l + h) >> 1;
    if (key[m] <= x) l = m + 1;
    else h = m;
  }
  return l - 1;
}

// One block per sample: every position t >= s_b that is not a placeholder
// becomes pair pi(t) - s_b.
__global__ void __launch_bounds__(256) align_rows_kernel(AlignArgs a, AlignArrays arr) {
  griddep_wait();
  if (arr.hdr->skip) return;
  const int b = blockIdx.x;
  const int lo = a.span_offsets[b], hi = a.span_offsets[b + 1];
  if (hi <= lo) return;
  const int L = arr.L[b], first = arr.first[b];
  const int t0 = arr.t_cu[b], s0 = arr.s_cu[b], p0 = arr.p_cu[b];
  for (int t = first + threadIdx.x; t < L; t += blockDim.x) {
    const int i = last_le(a.span_start, lo, hi, t);   // exists: t >= span_start[lo]
    const int n = a.span_len[i], s = a.span_start[i];
    if (t < s + n - 1) continue;                      // placeholder inside span i
    const int pi = t - (arr.r_before[i] + n - 1);
    const int k = pi - first;
    a.teacher_rows[p0 + k] = t0 + t;
    a.student_rows[p0 + k] = s0 + pi;
  }
}

// ===========================================================================
// soft-target cross-entropy
// ===========================================================================
constexpr int kCeMaxCluster = 16;  // CTAs per student row, at most (16 is a non-portable cluster size)
constexpr int kCeMaxVecs = 5;      // 16-byte vectors per thread per row
constexpr int kCeMaxStages = 3;
constexpr size_t kCeSmemLimit = 200 * 1024;   // dynamic shared memory per SM: room left for the static part
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

struct CeHeader {
  int32_t status;     // status word when the caller passes none
  int32_t error;      // set by the prep kernel: write nothing
  int32_t n_pairs;    // N
  int32_t ctas_done;  // CTAs of the main kernel that finished
  int32_t pad[60];
};
static_assert(sizeof(CeHeader) == 256, "ce header size");

size_t ce_ws_bytes(int R_S, int max_pairs) {
  return a256(sizeof(CeHeader)) + 2 * a256(sizeof(int32_t) * (size_t)std::max(R_S, 1)) +
         a256(sizeof(float) * (size_t)std::max(max_pairs, 1));
}

struct CeArgs {
  const uint16_t *teacher, *student;   // bf16 [R_T][ld], [R_S][ld]
  int64_t ld;
  int32_t V, R_T, R_S;
  const int32_t *teacher_rows, *student_rows;
  int32_t max_pairs;
  const int32_t *n_dev;
  float eps;
  float *loss;
  float *pair_loss;
  uint16_t *grad;                      // bf16 [R_S][ld] or nullptr
  int32_t *row_pair;                   // [R_S] pair of each student row, -1 if none
  int32_t *row_teacher;                // [R_S] teacher row paired with each student row, -1 if none
  CeHeader *hdr;
  int32_t *status;
  int32_t chunk_vecs;                  // 16-byte vectors of a row per CTA
  int32_t stage_vecs;                  // vectors per row in a stage: chunk_vecs, padded with -inf to KV x T
  int32_t stages;
};

// Validate the pairs and record, for every student row, the pair it is in.
__global__ void ce_prep_kernel(CeArgs a) {
  const int N = a.n_dev ? *a.n_dev : a.max_pairs;
  if (N < 0 || N > a.max_pairs) {
    if (blockIdx.x == 0 && threadIdx.x == 0) {
      atomicOr(&a.hdr->error, 1);
      set_error(a.status, UMIM_ERR_INVALID_ARG);
    }
    return;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) a.hdr->n_pairs = N;
  for (int p = blockIdx.x * blockDim.x + threadIdx.x; p < N; p += gridDim.x * blockDim.x) {
    const int t = a.teacher_rows[p], s = a.student_rows[p];
    bool ok = t >= 0 && t < a.R_T && s >= 0 && s < a.R_S;
    if (ok && atomicCAS(&a.row_pair[s], -1, p) != -1) ok = false;   // a student row in two pairs
    if (ok) a.row_teacher[s] = t;
    if (!ok) {
      atomicOr(&a.hdr->error, 1);
      set_error(a.status, UMIM_ERR_INVALID_ARG);
    }
  }
}

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_idx() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_count() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar,
                                          uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

__device__ __forceinline__ uint32_t cluster_size() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}

// The hardware's approximate base-2 exponential, logarithm and reciprocal
// (PTX ex2/lg2/rcp.approx.ftz: relative errors of about 2^-22; subnormal
// results flush to zero).
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float lg2_approx(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float rcp_approx(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// 32 lanes x 16 consecutive 32-bit columns of tensor memory from / to 16
// registers of each thread of the warp (thread i: lane base + i)
__device__ __forceinline__ void tmem_st_x16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
      "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}
__device__ __forceinline__ void tmem_ld_x16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// bf16x2 -inf, and the packed maximum of two bf16 pairs
constexpr uint32_t kNegInfBf16x2 = 0xff80ff80u;
__device__ __forceinline__ uint32_t max_bf16x2(uint32_t x, uint32_t y) {
  uint32_t d;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(x), "r"(y));
  return d;
}
// a bf16 pair (element 0 in the low half) as two floats
__device__ __forceinline__ float2 bf16x2_to_float2(uint32_t w) {
  return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}
// the maximum over the warp, one instruction
__device__ __forceinline__ float redux_max_f32(float x) {
  float r;
  asm volatile("redux.sync.max.f32 %0, %1, 0xffffffff;" : "=f"(r) : "f"(x));
  return r;
}
// sum over the warp of a pair of floats: xor butterflies, so every lane gets
// the same bits
__device__ __forceinline__ float2 warp_sum2(float2 v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1)
    v = __fadd2_rn(v, make_float2(__shfl_xor_sync(0xffffffffu, v.x, o), __shfl_xor_sync(0xffffffffu, v.y, o)));
  return v;
}

// mbarrier wait that sleeps instead of spinning: try_wait with a suspend-time
// hint (the thread is woken when the phase completes, or after 1 ms), so a
// warp waiting for the cluster takes no issue slots from warps still
// computing; bounded by kWaitLimitNs like every wait of the library
__device__ __forceinline__ bool mbar_try_wait_sleep(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(1000000u)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_test_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_wait_sleep(uint64_t *bar, uint32_t parity) {
  const uint32_t a = smem_u32(bar);
  if (mbar_test_wait(a, parity)) return true;   // a phase already complete costs no suspension
  if (mbar_try_wait_sleep(a, parity)) return true;
  const uint64_t t0 = globaltimer();
  while (true) {
    if (mbar_try_wait_sleep(a, parity)) return true;
    if (globaltimer() - t0 > kWaitLimitNs) return false;
  }
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 p = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&p);
}

// Store 8 gradient values at element offset e of a row (only elements < V).
__device__ __forceinline__ void store8(uint16_t *row, int64_t e, int V, const float *g) {
  if (e + 8 <= V) {
    uint4 o;
    o.x = pack_bf16x2(g[0], g[1]);
    o.y = pack_bf16x2(g[2], g[3]);
    o.z = pack_bf16x2(g[4], g[5]);
    o.w = pack_bf16x2(g[6], g[7]);
    *reinterpret_cast<uint4 *>(row + e) = o;
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j)
      if (e + j < V) {
        __nv_bfloat16 h = __float2bfloat16_rn(g[j]);
        row[e + j] = *reinterpret_cast<uint16_t *>(&h);
      }
  }
}

// The exchange between the CTAs of a row's cluster: every warp pushes its
// partial (a float4) into slot [rank][warp] of buffer (kind, b) in every CTA
// of the cluster with st.async, which counts its bytes on that CTA's mbarrier
// (kind, b); a CTA's warps wait on their own mbarrier and then read all C x NW
// partials locally.  No fence and no CTA- or cluster-wide barrier is needed
// per row.  Buffers alternate with the row's parity; each mbarrier phase is
// armed (arrive + expected bytes) by thread 0 one row ahead, right after the
// previous phase of that buffer completed, so its byte count never runs
// negative.
__device__ __forceinline__ uint32_t peer_addr(const void *local, uint32_t rank) {
  uint32_t ra;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(smem_u32(local)), "r"(rank));
  return ra;
}
__device__ __forceinline__ void st_async_f4(uint32_t raddr, float4 v, uint32_t rbar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(
                   raddr),
               "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(rbar)
               : "memory");
}

// One cluster of C CTAs per student row; CTA `rank` owns vectors
// [rank * chunk_vecs, ...) of the row.  T compute threads (NW warps) hold
// KV vectors of the teacher and student row each, and one more warp issues
// the copies: lane 0 walks the CTA's paired rows, waits for a stage of the
// ring to be released by every compute warp, and loads the teacher and
// student chunk into it with two bulk copies.
//
// The compute warps run two rows at once.  For row c they take the logits
// from the stage, the thread's max, exp(x - max) and the sums (pass 1) and
// push the warp's softmax statistics to every CTA of the cluster; then they
// wait for the loss sums of row c - 1 and write its gradient; then they wait
// for row c's statistics, form P^T and P^S, the loss terms and
// a_v = P^T P^S / (P^S + eps) (pass 2) and push the warp's sums.  Each
// exchange is thus waited for one compute phase after it was pushed.
// Between the phases a row is held in registers as fp32 exp(x - max)
// (pass 1 -> 2), then in tensor memory (which this kernel has no other use
// for) as fp32 P^S and -a_v / N (pass 2 -> gradient): each warp owns 16 x KV
// columns of its lane quarter, 16 per vector.
template <int KV, int T, bool TAIL>   // TAIL: V is not a multiple of 8 (a vector is cut by V)
__global__ void __launch_bounds__(T + 32, 1) ce_kernel(CeArgs a) {
  constexpr int NW = T / 32;               // compute warps; warp NW issues the copies
  constexpr int NX = kCeMaxCluster * NW;   // partial slots per buffer
  constexpr int NP = 4 * KV;               // element pairs (one 32-bit word of each row) per thread
  // tensor-memory columns: 16 per vector for each warp of a lane quarter
  constexpr uint32_t kTmemNeed = (uint32_t)((NW + 3) / 4) * 16u * KV;
  constexpr uint32_t kTmemCols = kTmemNeed <= 32 ? 32 : kTmemNeed <= 64 ? 64 : kTmemNeed <= 128 ? 128 : 256;
  static_assert(kTmemNeed <= 256, "tensor memory");
  extern __shared__ __align__(128) uint8_t ce_smem[];
  __shared__ __align__(8) uint64_t full_bar[kCeMaxStages], empty_bar[kCeMaxStages];
  __shared__ __align__(8) uint64_t xbar[2][2];        // [stats | sums][row parity]
  __shared__ __align__(16) float4 xbuf[2][2][NX];     // [stats | sums][row parity][rank * NW + warp]
  __shared__ uint32_t s_tmem;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t rank = cluster_ctarank();
  const int C = (int)cluster_size();
  const int cid = (int)cluster_idx(), ncl = (int)cluster_count();
  const int nvec = (a.V + 7) >> 3;
  const int vbeg = (int)rank * a.chunk_vecs;
  const int vcnt = max(0, min(a.chunk_vecs, nvec - vbeg));
  // vectors of the chunk that lie wholly below V; a vector cut by V is stored element-wise
  const int vfull = TAIL ? max(0, min(vcnt, a.V / 8 - vbeg)) : vcnt;
  const int S = a.stages;
  uint4 *stage_base = reinterpret_cast<uint4 *>(ce_smem);   // [S][2][stage_vecs]
  const int SV = a.stage_vecs;
  const uint32_t tx_bytes = 2u * (uint32_t)vcnt * 16u;
  const uint32_t x_bytes = (uint32_t)(C * NW * 16);

  if (a.hdr->error) return;   // the prep kernel rejected the pairs: write nothing (every CTA alike)
  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], NW);
    }
    for (int k = 0; k < 2; ++k)
      for (int b = 0; b < 2; ++b) mbar_init(&xbar[k][b], 1);
    fence_mbar_init();
    for (int k = 0; k < 2; ++k)
      for (int b = 0; b < 2; ++b) mbar_arrive_expect_tx(&xbar[k][b], x_bytes);   // rows 0 and 1
  }
  // vectors [vcnt, stage_vecs) of every stage hold -inf (no copy writes them), so every
  // thread reads its KV vectors of a row without a bounds check
  for (int i = tid; i < S * 2 * (SV - vcnt); i += T + 32) {
    const int h = i / (SV - vcnt);
    stage_base[(size_t)h * SV + vcnt + i % (SV - vcnt)] =
        make_uint4(kNegInfBf16x2, kNegInfBf16x2, kNegInfBf16x2, kNegInfBf16x2);
  }
  if (warp == 0) {
    tmem_alloc(&s_tmem, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  cluster_sync_all();   // every CTA's mbarriers exist before anyone pushes to them
  tc_fence_after();
  // this warp's columns in its lane quarter
  const uint32_t t_hold = s_tmem + ((uint32_t)((warp & 3) * 32) << 16) + (uint32_t)(warp >> 2) * 16u * KV;
  const int N = a.hdr->n_pairs;
  const float invN = N > 0 ? 1.0f / (float)N : 0.f;
  const float eps = a.eps;
  const float2 kL2 = make_float2(kLog2e, kLog2e);
  bool failed = false;
  // wait for phase `parity` of mbarrier m; a wait that gives up marks the thread failed
  auto xwait = [&](uint64_t *m, uint32_t parity) {
    if (!failed && !mbar_wait_sleep(m, parity)) {
      failed = true;
      set_error(a.status, UMIM_ERR_TIMEOUT);
    }
  };

  if (warp == NW) {
    // ---- the copies ----
    if (lane == 0) {
      const uint64_t pol = policy_evict_first();
      int issued = 0, s = 0;
      uint32_t phase = 0;   // of stage s's full barrier for the copy about to be issued
      int w = cid, t = cid < a.R_S ? a.row_teacher[cid] : -1;
      while (w < a.R_S && !failed) {
        const int cw = w, ct = t;
        w += ncl;
        t = w < a.R_S ? a.row_teacher[w] : -1;   // the next row's teacher, loaded ahead
        if (ct < 0) continue;                     // a student row in no pair
        if (issued >= S) xwait(&empty_bar[s], phase ^ 1u);   // the stage's previous row is consumed
        if (failed) break;
        mbar_arrive_expect_tx(&full_bar[s], tx_bytes);
        if (vcnt > 0) {
          uint4 *dst = stage_base + (size_t)s * 2 * SV;
          const int ctl = in_bounds(ct, a.R_T, a.status, kSiteDistillTeacherRow) ? ct : 0;
          bulk_load(dst, a.teacher + (int64_t)ctl * a.ld + (int64_t)vbeg * 8, (uint32_t)vcnt * 16u, &full_bar[s],
                    pol);
          bulk_load(dst + SV, a.student + (int64_t)cw * a.ld + (int64_t)vbeg * 8, (uint32_t)vcnt * 16u, &full_bar[s],
                    pol);
        }
        ++issued;
        if (++s == S) {
          s = 0;
          phase ^= 1u;
        }
      }
      // every copy has landed before the CTA's shared memory goes away (bounded)
      for (int s = 0; s < S && s < issued; ++s) {
        const int last = ((issued - 1 - s) / S) * S + s;   // the last copy issued to stage s
        mbar_wait_for(&full_bar[s], (uint32_t)(last / S) & 1u, kWaitLimitNs);
      }
    }
  } else {
    // ---- the compute warps ----
    int prev_c = -1, prev_p = -1;
    const int64_t goff = (int64_t)(vbeg + tid) * 8;   // this thread's first gradient element of a row
    uint16_t *prev_grow = nullptr;

    // loss sums of row prev_c, then its gradient -(1/N) (a_v - P^S(v) A) = P^S(v) (A/N) - a_v/N
    auto finish_prev = [&]() {
      const int xb = prev_c & 1;
      xwait(&xbar[1][xb], (uint32_t)(prev_c >> 1) & 1u);
      if (tid == 0 && !failed) mbar_arrive_expect_tx(&xbar[1][xb], x_bytes);   // row prev_c + 2
      const int nx = C * NW;
      float2 LA = make_float2(0.f, 0.f);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int j = lane + 32 * i;
        if (j < nx) LA = __fadd2_rn(LA, *reinterpret_cast<const float2 *>(&xbuf[1][xb][j]));
      }
      for (int j = lane + 128; j < nx; j += 32) LA = __fadd2_rn(LA, *reinterpret_cast<const float2 *>(&xbuf[1][xb][j]));
      LA = warp_sum2(LA);   // (-sum P^T log2(P^S + eps), -A), both / N
      if (rank == 0 && tid == 0 && in_bounds(prev_p, N, a.status, kSiteDistillPair))
        a.pair_loss[prev_p] = LA.x * kLn2 * (float)N;
      if (prev_grow) {
        const float2 A2 = make_float2(-LA.y, -LA.y);
        tmem_wait_st();
#pragma unroll
        for (int k = 0; k < KV; ++k) {
          const int vi = tid + k * T;
          uint32_t hold[16];
          tmem_ld_x16(t_hold + 16u * k, hold);   // P^S (8 values), then -a_v / N (8 values)
          if (vi < vcnt) {
            uint32_t g[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const float2 pS = make_float2(__uint_as_float(hold[2 * j]), __uint_as_float(hold[2 * j + 1]));
              const float2 nav = make_float2(__uint_as_float(hold[8 + 2 * j]), __uint_as_float(hold[9 + 2 * j]));
              const float2 gr = __ffma2_rn(pS, A2, nav);
              g[j] = pack_bf16x2(gr.x, gr.y);
            }
            const int64_t e0 = goff + (int64_t)k * T * 8;
            if (!TAIL || vi < vfull) {
              *reinterpret_cast<uint4 *>(prev_grow + e0) = make_uint4(g[0], g[1], g[2], g[3]);
            } else {   // the vector cut by V: only the elements below V
#pragma unroll
              for (int j = 0; j < 8; ++j)
                if (e0 + j < a.V) prev_grow[e0 + j] = (uint16_t)((j & 1) ? (g[j / 2] >> 16) : (g[j / 2] & 0xffffu));
            }
          }
        }
      }
    };

    int consumed = 0, stage = 0;
    uint32_t sphase = 0;   // of the stage's full barrier for the row about to be consumed
    int p_next = cid < a.R_S ? a.row_pair[cid] : -1;
    for (int w = cid; w < a.R_S; w += ncl) {
      const int p = p_next;
      if (w + ncl < a.R_S) p_next = a.row_pair[w + ncl];
      uint16_t *grow = a.grad ? a.grad + (int64_t)w * a.ld : nullptr;
      if (p < 0) {   // a student row in no pair: zero gradient
        if (grow) {
          float z[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
          for (int vi = tid; vi < vcnt; vi += T) store8(grow, (int64_t)(vbeg + vi) * 8, a.V, z);
        }
        continue;
      }
      const int c = consumed++;
      const int s = stage;
      const uint32_t fpar = sphase;
      if (++stage == S) {
        stage = 0;
        sphase ^= 1u;
      }
      const int xb = c & 1;
      const uint32_t xpar = (uint32_t)(c >> 1) & 1u;

      // ---- pass 1: the logits as bf16 pairs, this thread's max over the
      // packed pairs, then exp(x - max) and its sum, two elements per instruction ----
      xwait(&full_bar[s], fpar);
      const uint4 *st = stage_base + (size_t)s * 2 * SV;
      uint32_t wt[NP], ws[NP];
#pragma unroll
      for (int k = 0; k < KV; ++k) {
        const int vi = tid + k * T;
        const uint4 ut = st[vi], us = st[SV + vi];
        wt[4 * k] = ut.x, wt[4 * k + 1] = ut.y, wt[4 * k + 2] = ut.z, wt[4 * k + 3] = ut.w;
        ws[4 * k] = us.x, ws[4 * k + 1] = us.y, ws[4 * k + 2] = us.z, ws[4 * k + 3] = us.w;
        const int e0 = (vbeg + vi) * 8;
        if (TAIL && vi < vcnt && e0 + 8 > a.V) {   // the row's last vector: elements past V become -inf
#pragma unroll
          for (int j = 0; j < 8; ++j)
            if (e0 + j >= a.V) {
              const uint32_t keep = (j & 1) ? 0x0000ffffu : 0xffff0000u;
              wt[4 * k + j / 2] = (wt[4 * k + j / 2] & keep) | (kNegInfBf16x2 & ~keep);
              ws[4 * k + j / 2] = (ws[4 * k + j / 2] & keep) | (kNegInfBf16x2 & ~keep);
            }
        }
      }
      float mt, ms;
      {
        uint32_t m2t = wt[0], m2s = ws[0];
#pragma unroll
        for (int i = 1; i < NP; ++i) {
          m2t = max_bf16x2(m2t, wt[i]);
          m2s = max_bf16x2(m2s, ws[i]);
        }
        const float2 ft = bf16x2_to_float2(m2t), fs = bf16x2_to_float2(m2s);
        mt = fmaxf(ft.x, ft.y);
        ms = fmaxf(fs.x, fs.y);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_bar[s]);   // this warp is done with the stage
      const float bt = (mt == -INFINITY) ? 0.f : -mt * kLog2e;
      const float bs = (ms == -INFINITY) ? 0.f : -ms * kLog2e;
      const float2 bt2 = make_float2(bt, bt), bs2 = make_float2(bs, bs);
      float2 zt0 = make_float2(0.f, 0.f), zt1 = zt0, zs0 = zt0, zs1 = zt0;
      float2 et[NP], es[NP];
#pragma unroll
      for (int i = 0; i < NP; ++i) {
        const float2 at = __ffma2_rn(bf16x2_to_float2(wt[i]), kL2, bt2);   // -inf -> exp 0
        const float2 as = __ffma2_rn(bf16x2_to_float2(ws[i]), kL2, bs2);
        et[i] = make_float2(ex2_approx(at.x), ex2_approx(at.y));
        es[i] = make_float2(ex2_approx(as.x), ex2_approx(as.y));
        if (i & 1) {
          zt1 = __fadd2_rn(zt1, et[i]);
          zs1 = __fadd2_rn(zs1, es[i]);
        } else {
          zt0 = __fadd2_rn(zt0, et[i]);
          zs0 = __fadd2_rn(zs0, es[i]);
        }
      }
      // ---- softmax statistics of this thread's warp, to every CTA of the cluster ----
      {
        const float2 zt2 = __fadd2_rn(zt0, zt1), zs2 = __fadd2_rn(zs0, zs1);
        const float Mwt = redux_max_f32(mt), Mws = redux_max_f32(ms);
        float2 z = make_float2((mt == -INFINITY) ? 0.f : (zt2.x + zt2.y) * ex2_approx((mt - Mwt) * kLog2e),
                               (ms == -INFINITY) ? 0.f : (zs2.x + zs2.y) * ex2_approx((ms - Mws) * kLog2e));
        z = warp_sum2(z);
        if (lane < C)
          st_async_f4(peer_addr(&xbuf[0][xb][rank * NW + warp], (uint32_t)lane), make_float4(Mwt, Mws, z.x, z.y),
                      peer_addr(&xbar[0][xb], (uint32_t)lane));
      }

      // ---- the previous row, while this row's statistics travel ----
      if (prev_c >= 0) finish_prev();

      // ---- the row's max over the C x NW partials, then one rescale per partial ----
      xwait(&xbar[0][xb], xpar);
      if (tid == 0 && !failed) mbar_arrive_expect_tx(&xbar[0][xb], x_bytes);   // row c + 2
      const int nx = C * NW;
      float Mt = -INFINITY, Ms = -INFINITY;
      auto max_part = [&](int j) {
        const float2 m = *reinterpret_cast<const float2 *>(&xbuf[0][xb][j]);
        Mt = fmaxf(Mt, m.x);
        Ms = fmaxf(Ms, m.y);
      };
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (lane + 32 * i < nx) max_part(lane + 32 * i);
      for (int j = lane + 128; j < nx; j += 32) max_part(j);
      Mt = redux_max_f32(Mt);
      Ms = redux_max_f32(Ms);
      const float nMt = (Mt == -INFINITY) ? 0.f : -Mt * kLog2e, nMs = (Ms == -INFINITY) ? 0.f : -Ms * kLog2e;
      const float2 nM2 = make_float2(nMt, nMs);
      float2 Z = make_float2(0.f, 0.f);
      auto sum_part = [&](int j) {
        const float4 v = xbuf[0][xb][j];
        const float2 x = __ffma2_rn(make_float2(v.x, v.y), kL2, nM2);   // empty partials: z = 0
        Z = __ffma2_rn(make_float2(v.z, v.w), make_float2(ex2_approx(x.x), ex2_approx(x.y)), Z);
      };
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (lane + 32 * i < nx) sum_part(lane + 32 * i);
      for (int j = lane + 128; j < nx; j += 32) sum_part(j);
      Z = warp_sum2(Z);
      // P(v) = exp(x - m_thread) * exp(m_thread - M) / Z.  The teacher's
      // factor carries -1/N: the loss terms, a and A come out as -(.)/N and
      // the gradient P^S(v) (A/N) - a_v/N is one FMA per element.
      const float nct = (mt == -INFINITY) ? 0.f : -ex2_approx(fmaf(mt, kLog2e, nMt)) * rcp_approx(Z.x) * invN;
      const float cs = (ms == -INFINITY) ? 0.f : ex2_approx(fmaf(ms, kLog2e, nMs)) * rcp_approx(Z.y);
      const float2 nct2 = make_float2(nct, nct), cs2 = make_float2(cs, cs);

      // ---- pass 2: -P^T / N, P^S, -(loss terms) / N and -a / N; P^S and -a / N to tensor memory ----
      float2 l0 = make_float2(0.f, 0.f), l1 = l0, s0 = l0, s1 = l0;
      auto pass2 = [&](auto clamp) {
        const float2 eps2 = make_float2(eps, eps);
        uint32_t hold[16];
#pragma unroll
        for (int i = 0; i < NP; ++i) {
          const float2 pt = __fmul2_rn(et[i], nct2);
          const float2 pS = __fmul2_rn(es[i], cs2);
          float2 q = __fadd2_rn(pS, eps2);
          if constexpr (decltype(clamp)::value)   // eps = 0: log2 stays finite
            q = make_float2(fmaxf(q.x, 1.17549435e-38f), fmaxf(q.y, 1.17549435e-38f));
          const float2 lg = make_float2(lg2_approx(q.x), lg2_approx(q.y));
          const float2 rq = make_float2(ex2_approx(-lg.x), ex2_approx(-lg.y));   // 1 / q
          const float2 av = __fmul2_rn(pt, __fmul2_rn(pS, rq));
          if (i & 1) {
            l1 = __ffma2_rn(pt, lg, l1);
            s1 = __fadd2_rn(s1, av);
          } else {
            l0 = __ffma2_rn(pt, lg, l0);
            s0 = __fadd2_rn(s0, av);
          }
          const int j = i & 3;
          hold[2 * j] = __float_as_uint(pS.x);
          hold[2 * j + 1] = __float_as_uint(pS.y);
          hold[8 + 2 * j] = __float_as_uint(av.x);
          hold[9 + 2 * j] = __float_as_uint(av.y);
          if (j == 3) tmem_st_x16(t_hold + 16u * (i / 4), hold);
        }
      };
      if (eps > 0.f)
        pass2(std::false_type{});
      else
        pass2(std::true_type{});
      {
        const float2 l2 = __fadd2_rn(l0, l1), s2 = __fadd2_rn(s0, s1);
        const float2 r = warp_sum2(make_float2(l2.x + l2.y, s2.x + s2.y));
        if (lane < C)
          st_async_f4(peer_addr(&xbuf[1][xb][rank * NW + warp], (uint32_t)lane), make_float4(r.x, r.y, 0.f, 0.f),
                      peer_addr(&xbar[1][xb], (uint32_t)lane));
      }
      prev_c = c;
      prev_p = p;
      prev_grow = grow;
    }
    if (prev_c >= 0) finish_prev();
    tmem_wait_st();   // the last row's stores, when no gradient read them back
  }

  // no CTA leaves while a peer may still push to or read its shared memory
  tc_fence_before();
  cluster_sync_all();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(s_tmem, kTmemCols);
  }

  // ---- the loss: the last CTA sums the per-pair losses in pair order ----
  constexpr int NT = T + 32;
  __shared__ int s_last;
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    s_last = atomicAdd(&a.hdr->ctas_done, 1) == (int)gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  __shared__ double dpart[NW + 1];
  const int per = (N + NT - 1) / NT;
  double acc = 0.0;
  for (int i = 0; i < per; ++i) {
    const int q = tid * per + i;
    if (q < N) acc += (double)*reinterpret_cast<volatile float *>(a.pair_loss + q);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) dpart[warp] = acc;
  __syncthreads();
  if (tid == 0) {
    double t = 0.0;
    for (int w2 = 0; w2 <= NW; ++w2) t += dpart[w2];
    a.loss[0] = N > 0 ? (float)(t / (double)N) : 0.f;
  }
}

using CeKernel = void (*)(CeArgs);

CeKernel ce_kernel_for(int kv, int T, bool tail) {
  static const CeKernel k256[2][kCeMaxVecs] = {
      {ce_kernel<1, 256, false>, ce_kernel<2, 256, false>, ce_kernel<3, 256, false>, ce_kernel<4, 256, false>,
       ce_kernel<5, 256, false>},
      {ce_kernel<1, 256, true>, ce_kernel<2, 256, true>, ce_kernel<3, 256, true>, ce_kernel<4, 256, true>,
       ce_kernel<5, 256, true>}};
  static const CeKernel k448[2][4] = {
      {ce_kernel<1, 448, false>, ce_kernel<2, 448, false>, ce_kernel<3, 448, false>, ce_kernel<4, 448, false>},
      {ce_kernel<1, 448, true>, ce_kernel<2, 448, true>, ce_kernel<3, 448, true>, ce_kernel<4, 448, true>}};
  return T == 256 ? k256[tail][kv - 1] : k448[tail][kv - 1];
}

// 16-byte vectors per thread per row with T compute threads per CTA and C CTAs per row
int ce_vecs(int64_t V, int T, int C) {
  const int64_t nvec = (V + 7) / 8;
  const int64_t chunk = (nvec + C - 1) / C;
  return (int)std::max<int64_t>(1, (chunk + T - 1) / T);
}

// How a call runs: T compute threads (plus the copy warp) per CTA, C CTAs
// (one cluster) per student row, KV vectors of each row per thread.
struct CeLayout {
  int T, C, kv, chunk_vecs, stage_vecs, stages;
  size_t smem;
  int resident;   // clusters that can be resident at once
};

// Clusters of a layout that can be resident at once (0: it cannot launch);
// cached per device and layout.
int ce_resident_clusters(int kv, int T, int C, size_t smem, int num_sms, bool tail) {
  struct Entry {
    int dev, kv, T, C, tail;
    size_t smem;
    int n;
  };
  static Entry cache[64];
  static int n_cache = 0;
  static std::mutex mu;
  int dev = 0;
  cudaGetDevice(&dev);
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < n_cache; ++i) {
    const Entry &e = cache[i];
    if (e.dev == dev && e.kv == kv && e.T == T && e.C == C && e.tail == (int)tail && e.smem == smem) return e.n;
  }
  const CeKernel fn = ce_kernel_for(kv, T, tail);
  // the largest size any call may request, so that no later call finds a smaller limit
  cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kCeSmemLimit);
  if (C > 8) cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(C * std::max(1, num_sms / C)));
  cfg.blockDim = dim3((unsigned)(T + 32));
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess) {
    cudaGetLastError();
    n = 0;
  }
  if (n_cache < 64) cache[n_cache++] = Entry{dev, kv, T, C, (int)tail, smem, n};
  return n;
}

bool ce_try_layout(int64_t V, int T, int C, int num_sms, CeLayout &L) {
  const int kv = ce_vecs(V, T, C);
  if (kv > kCeMaxVecs) return false;
  const int nvec = (int)((V + 7) / 8);
  L.T = T;
  L.C = C;
  L.kv = kv;
  L.chunk_vecs = (nvec + C - 1) / C;
  L.stage_vecs = std::max(L.chunk_vecs, kv * T);
  const size_t stage_bytes = (size_t)2 * L.stage_vecs * 16;
  L.stages = (int)std::min<size_t>(kCeMaxStages, kCeSmemLimit / stage_bytes);
  if (L.stages < 2) return false;
  L.smem = stage_bytes * L.stages;
  L.resident = ce_resident_clusters(kv, T, C, L.smem, num_sms, V % 8 != 0);
  return L.resident > 0;
}

// Candidates: 256 and 448 compute threads per CTA (one CTA per SM), each
// with the three smallest cluster sizes whose threads hold at most 4 vectors
// of a row (5 at 256 threads and the largest cluster).  The score is the SMs
// the resident clusters occupy times the share of the threads' vector slots
// that hold data: cluster placement within a GPC can leave SMs idle (on a
// GB300 at the Llama-3 vocabulary, 15 clusters of 9 x 448 threads occupy
// 135 SMs, 7 clusters of 16 x 256 threads 112).
bool ce_layout(int64_t V, int num_sms, CeLayout &L) {
  const int64_t nvec = (V + 7) / 8;
  CeLayout best{};
  double best_score = -1.0;
  for (const int T : {256, 448}) {
    const int Cmax = kCeMaxCluster;
    const int kv_max = T == 256 ? kCeMaxVecs : 4;
    int tried = 0;
    for (int C = 1; C <= Cmax && tried < 3; ++C) {   // the three smallest admissible cluster sizes
      const int kv = ce_vecs(V, T, C);
      if (kv > 4 && !(C == Cmax && kv <= kv_max)) continue;
      ++tried;
      CeLayout cand;
      if (!ce_try_layout(V, T, C, num_sms, cand)) continue;
      const double sms_used = (double)cand.resident * C;
      const double fill = (double)nvec / ((double)C * T * kv);
      const double score = sms_used * fill;
      if (score > best_score * 1.001) {   // ties: the smaller cluster, found first
        best = cand;
        best_score = score;
      }
      if (kv == 1) break;   // more CTAs per row only adds empty slots
    }
  }
  if (best_score < 0) return false;
  L = best;
  return true;
}

}  // namespace

// ---------------------------------------------------------------------------
// host entry points
// ---------------------------------------------------------------------------
size_t distill_align_workspace_bytes(int B, int S) { return align_ws_bytes(B, S); }

umim_status distill_align(const int32_t *seq_lens, int32_t B, const int32_t *span_offsets, const int32_t *span_start,
                          const int32_t *span_len, int32_t S, int32_t *pair_offsets, int32_t *teacher_rows,
                          int32_t *student_rows, int32_t capacity, int32_t *student_cu, void *ws,
                          int32_t *dev_status, cudaStream_t stream) {
  AlignArrays arr = align_carve(ws, B, S);
  AlignArgs a;
  a.seq_lens = seq_lens;
  a.span_offsets = span_offsets;
  a.span_start = span_start;
  a.span_len = span_len;
  a.B = B;
  a.S = S;
  a.capacity = capacity;
  a.pair_offsets = pair_offsets;
  a.teacher_rows = teacher_rows;
  a.student_rows = student_rows;
  a.student_cu = student_cu;
  a.status = dev_status ? dev_status : &arr.hdr->status;
  trace_mark(stream, "distill.align_plan");
  if (launch_pdl(align_plan_kernel, dim3(B), dim3(kAlignThreads), 0, stream, a, arr) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, "distill.align_rows");
  if (launch_pdl(align_rows_kernel, dim3(B), dim3(256), 0, stream, a, arr) != cudaSuccess) return UMIM_ERR_CUDA;
  trace_mark(stream, nullptr);
  return UMIM_OK;
}

size_t distill_soft_ce_workspace_bytes(int R_S, int max_pairs) { return ce_ws_bytes(R_S, max_pairs); }

// nonzero when the vocabulary is supported (at most 16 CTAs x 256 threads x 5 vectors x 8 values;
// the 448-thread layouts cover the same range with at most 4 vectors)
int distill_soft_ce_vecs(int64_t V) { return (V >= 1 && ce_vecs(V, 256, kCeMaxCluster) <= kCeMaxVecs) ? 1 : 0; }

umim_status distill_soft_ce(const void *teacher, int32_t R_T, const void *student, int32_t R_S, int32_t V, int64_t ld,
                            const int32_t *teacher_rows, const int32_t *student_rows, int32_t max_pairs,
                            const int32_t *n_dev, float eps, float *loss, float *pair_loss, void *grad, void *ws,
                            int32_t *dev_status, cudaStream_t stream, int num_sms) {
  if (!distill_soft_ce_vecs(V)) return UMIM_ERR_UNSUPPORTED;
  CeLayout lay;
  if (!ce_layout(V, num_sms, lay)) return UMIM_ERR_UNSUPPORTED;
  char *p = static_cast<char *>(ws);
  CeHeader *hdr = reinterpret_cast<CeHeader *>(p);
  p += a256(sizeof(CeHeader));
  int32_t *row_pair = reinterpret_cast<int32_t *>(p);
  p += a256(sizeof(int32_t) * (size_t)std::max(R_S, 1));
  int32_t *row_teacher = reinterpret_cast<int32_t *>(p);
  p += a256(sizeof(int32_t) * (size_t)std::max(R_S, 1));
  float *ws_pair_loss = reinterpret_cast<float *>(p);

  CeArgs a;
  a.teacher = static_cast<const uint16_t *>(teacher);
  a.student = static_cast<const uint16_t *>(student);
  a.ld = ld;
  a.V = V;
  a.R_T = R_T;
  a.R_S = R_S;
  a.teacher_rows = teacher_rows;
  a.student_rows = student_rows;
  a.max_pairs = max_pairs;
  a.n_dev = n_dev;
  a.eps = eps;
  a.loss = loss;
  a.pair_loss = pair_loss ? pair_loss : ws_pair_loss;
  a.grad = static_cast<uint16_t *>(grad);
  a.row_pair = row_pair;
  a.row_teacher = row_teacher;
  a.hdr = hdr;
  a.status = dev_status ? dev_status : &hdr->status;
  a.chunk_vecs = lay.chunk_vecs;
  a.stage_vecs = lay.stage_vecs;
  a.stages = lay.stages;

  if (cudaMemsetAsync(hdr, 0, sizeof(CeHeader), stream) != cudaSuccess) return UMIM_ERR_CUDA;
  if (R_S > 0 && cudaMemsetAsync(row_pair, 0xFF, sizeof(int32_t) * (size_t)R_S, stream) != cudaSuccess)
    return UMIM_ERR_CUDA;
  if (R_S > 0 && cudaMemsetAsync(row_teacher, 0xFF, sizeof(int32_t) * (size_t)R_S, stream) != cudaSuccess)
    return UMIM_ERR_CUDA;
  const int prep_blocks = std::max(1, std::min((max_pairs + 255) / 256, num_sms * 4));
  trace_mark(stream, "distill.ce_prep");
  ce_prep_kernel<<<prep_blocks, 256, 0, stream>>>(a);
  if (cudaGetLastError() != cudaSuccess) return UMIM_ERR_CUDA;

  const int n_cl = std::max(1, std::min(R_S, lay.resident));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(n_cl * lay.C));
  cfg.blockDim = dim3((unsigned)(lay.T + 32));
  cfg.dynamicSmemBytes = lay.smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)lay.C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  trace_mark(stream, "distill.soft_ce");
  const cudaError_t e = cudaLaunchKernelEx(&cfg, ce_kernel_for(lay.kv, lay.T, V % 8 != 0), a);
  trace_mark(stream, nullptr);
  return e == cudaSuccess ? UMIM_OK : UMIM_ERR_CUDA;
}

}  // namespace umim
