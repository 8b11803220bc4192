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
//    One thread-block cluster of 8 CTAs per student row: each CTA holds one
//    eighth of the vocabulary of the teacher and student rows in registers
//    (fp32), so every logit byte is read once and every gradient byte written
//    once.  Rows arrive by 1-D TMA bulk copies into a ring of shared-memory
//    stages (the next rows load while the current one is computed); the
//    softmax statistics and the two sums are exchanged between the cluster's
//    CTAs through distributed shared memory.  Student rows that are in no
//    pair get a zero gradient.  The loss is summed from the per-pair losses,
//    in pair order, by the last CTA to finish.
#include <algorithm>
#include <cmath>
#include <mutex>

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
constexpr int kCeCluster = 8;     // CTAs per student row (portable cluster size)
constexpr int kCeThreads = 512;
constexpr int kCeWarps = kCeThreads / 32;
constexpr int kCeMaxVecs = 5;     // 16-byte vectors per thread per row
constexpr int kCeMaxStages = 3;
constexpr size_t kCeSmemLimit = 227 * 1024 - 2048;   // dynamic shared memory: room left for the static part
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
  return a256(sizeof(CeHeader)) + a256(sizeof(int32_t) * (size_t)std::max(R_S, 1)) +
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
  CeHeader *hdr;
  int32_t *status;
  int32_t chunk_vecs;                  // 16-byte vectors of a row per CTA
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
// float4 at the same shared-memory offset in CTA `rank` of this cluster
__device__ __forceinline__ float4 ld_peer_f4(const float4 *local, uint32_t rank) {
  uint32_t ra;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(smem_u32(local)), "r"(rank));
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(ra)
               : "memory");
  return v;
}

__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar,
                                          uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

// (max, sum of exp2(x - max)) of two sets merged; an empty set is (-inf, 0)
__device__ __forceinline__ void lse_merge(float &m, float &z, float m2, float z2) {
  const float M = fmaxf(m, m2);
  if (M == -INFINITY) return;
  z = z * exp2f(m - M) + z2 * exp2f(m2 - M);
  m = M;
}

__device__ __forceinline__ void unpack8(const uint4 u, float *f) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    f[2 * j] = __uint_as_float(w[j] << 16) * kLog2e;
    f[2 * j + 1] = __uint_as_float(w[j] & 0xffff0000u) * kLog2e;
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
    for (int j = 0; j < 8 && e + j < V; ++j) {
      __nv_bfloat16 h = __float2bfloat16_rn(g[j]);
      row[e + j] = *reinterpret_cast<uint16_t *>(&h);
    }
  }
}

template <int KV>
__global__ void __launch_bounds__(kCeThreads, 1) ce_kernel(CeArgs a) {
  extern __shared__ __align__(128) uint8_t ce_smem[];
  __shared__ __align__(8) uint64_t full_bar[kCeMaxStages];
  __shared__ float4 slot_stats;          // this CTA's (m_T, z_T, m_S, z_S), read by the cluster
  __shared__ float4 slot_sums;           // this CTA's (sum P^T log2 q, sum a, -, -)
  __shared__ float4 warp_part[kCeWarps];
  __shared__ float4 bcast;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t rank = cluster_ctarank();
  const int cid = (int)cluster_idx(), ncl = (int)cluster_count();
  const int nvec = (a.V + 7) >> 3;
  const int vbeg = (int)rank * a.chunk_vecs;
  const int vcnt = max(0, min(a.chunk_vecs, nvec - vbeg));
  const int S = a.stages;
  uint4 *stage_base = reinterpret_cast<uint4 *>(ce_smem);   // [S][2][chunk_vecs]
  const uint32_t tx_bytes = 2u * (uint32_t)vcnt * 16u;

  if (tid == 0) {
    for (int s = 0; s < S; ++s) mbar_init(&full_bar[s], 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (a.hdr->error) return;   // the prep kernel rejected the pairs: write nothing
  const int N = a.hdr->n_pairs;
  const float invN = N > 0 ? 1.0f / (float)N : 0.f;

  // producer state (thread 0): next item to consider, copies issued
  int issue_w = cid, issued = 0;
  uint32_t pending = 0;     // stages with a copy in flight that thread 0 has not seen land
  bool failed = false;
  const uint64_t pol = policy_evict_first();
  auto issue_next = [&]() {
    while (issue_w < a.R_S) {
      const int w = issue_w;
      issue_w += ncl;
      const int p = a.row_pair[w];
      if (p < 0) continue;
      const int s = issued % S;
      ++issued;
      uint4 *dst = stage_base + (size_t)s * 2 * a.chunk_vecs;
      mbar_arrive_expect_tx(&full_bar[s], tx_bytes);
      pending |= 1u << s;
      if (vcnt > 0) {
        const int t = a.teacher_rows[p];
        const uint16_t *src_t = a.teacher + (int64_t)t * a.ld + (int64_t)vbeg * 8;
        const uint16_t *src_s = a.student + (int64_t)w * a.ld + (int64_t)vbeg * 8;
        bulk_load(dst, src_t, (uint32_t)vcnt * 16u, &full_bar[s], pol);
        bulk_load(dst + a.chunk_vecs, src_s, (uint32_t)vcnt * 16u, &full_bar[s], pol);
      }
      return;
    }
  };
  if (tid == 0)
    for (int s = 0; s < S; ++s) issue_next();

  int consumed = 0;
  for (int w = cid; w < a.R_S; w += ncl) {
    const int p = a.row_pair[w];
    uint16_t *grow = a.grad ? a.grad + (int64_t)w * a.ld : nullptr;
    if (p < 0) {   // a student row in no pair: zero gradient
      if (grow) {
        float z[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        for (int vi = tid; vi < vcnt; vi += kCeThreads) store8(grow, (int64_t)(vbeg + vi) * 8, a.V, z);
      }
      continue;
    }
    const int s = consumed % S;
    const uint32_t parity = (uint32_t)(consumed / S) & 1u;
    ++consumed;
    if (!failed && !mbar_wait(&full_bar[s], parity)) {
      failed = true;
      set_error(a.status, UMIM_ERR_TIMEOUT);
    }
    if (tid == 0 && !failed) pending &= ~(1u << s);
    const uint4 *st = stage_base + (size_t)s * 2 * a.chunk_vecs;

    // ---- pass 1: logits (scaled by log2 e) into registers, local max and sum ----
    float xt[KV * 8], xs[KV * 8];
    float mt = -INFINITY, ms = -INFINITY;
#pragma unroll
    for (int k = 0; k < KV; ++k) {
      const int vi = tid + k * kCeThreads;
      if (vi < vcnt) {
        unpack8(st[vi], xt + 8 * k);
        unpack8(st[a.chunk_vecs + vi], xs + 8 * k);
        const int e0 = (vbeg + vi) * 8;
        if (e0 + 8 > a.V) {
#pragma unroll
          for (int j = 0; j < 8; ++j)
            if (e0 + j >= a.V) {
              xt[8 * k + j] = -INFINITY;
              xs[8 * k + j] = -INFINITY;
            }
        }
      } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          xt[8 * k + j] = -INFINITY;
          xs[8 * k + j] = -INFINITY;
        }
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        mt = fmaxf(mt, xt[8 * k + j]);
        ms = fmaxf(ms, xs[8 * k + j]);
      }
    }
    __syncthreads();   // stage s is in registers: it may be refilled
    if (tid == 0 && !failed) issue_next();
    float zt = 0.f, zs = 0.f;
#pragma unroll
    for (int i = 0; i < KV * 8; ++i) {
      xt[i] = (mt == -INFINITY) ? 0.f : exp2f(xt[i] - mt);
      xs[i] = (ms == -INFINITY) ? 0.f : exp2f(xs[i] - ms);
      zt += xt[i];
      zs += xs[i];
    }
    // ---- softmax statistics over the cluster ----
    {
      float m1 = mt, z1 = zt, m2 = ms, z2 = zs;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        lse_merge(m1, z1, __shfl_xor_sync(0xffffffffu, m1, o), __shfl_xor_sync(0xffffffffu, z1, o));
        lse_merge(m2, z2, __shfl_xor_sync(0xffffffffu, m2, o), __shfl_xor_sync(0xffffffffu, z2, o));
      }
      if (lane == 0) warp_part[warp] = make_float4(m1, z1, m2, z2);
      __syncthreads();
      if (warp == 0) {
        float4 v = lane < kCeWarps ? warp_part[lane] : make_float4(-INFINITY, 0.f, -INFINITY, 0.f);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          lse_merge(v.x, v.y, __shfl_xor_sync(0xffffffffu, v.x, o), __shfl_xor_sync(0xffffffffu, v.y, o));
          lse_merge(v.z, v.w, __shfl_xor_sync(0xffffffffu, v.z, o), __shfl_xor_sync(0xffffffffu, v.w, o));
        }
        if (lane == 0) slot_stats = v;
      }
      cluster_sync_all();
      if (tid == 0) {
        float4 r[kCeCluster];
#pragma unroll
        for (int c = 0; c < kCeCluster; ++c) r[c] = ld_peer_f4(&slot_stats, (uint32_t)c);
        float4 g = r[0];
#pragma unroll
        for (int c = 1; c < kCeCluster; ++c) {
          lse_merge(g.x, g.y, r[c].x, r[c].y);
          lse_merge(g.z, g.w, r[c].z, r[c].w);
        }
        bcast = g;
      }
      __syncthreads();
    }
    const float4 gs = bcast;
    // P(v) = exp2(x - m_local) * exp2(m_local - M) / Z
    const float ct = (mt == -INFINITY) ? 0.f : exp2f(mt - gs.x) / gs.y;
    const float cs = (ms == -INFINITY) ? 0.f : exp2f(ms - gs.z) / gs.w;

    // ---- pass 2: P^T, P^S, the loss terms and a ----
    float lsum = 0.f, asum = 0.f;
#pragma unroll
    for (int i = 0; i < KV * 8; ++i) {
      const float pt = xt[i] * ct, ps = xs[i] * cs;
      const float q = ps + a.eps;
      const float r = q > 0.f ? __fdividef(ps, q) : 0.f;
      lsum += pt > 0.f ? pt * __log2f(q) : 0.f;
      const float av = pt * r;
      asum += av;
      xt[i] = av;
      xs[i] = ps;
    }
    {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        lsum += __shfl_xor_sync(0xffffffffu, lsum, o);
        asum += __shfl_xor_sync(0xffffffffu, asum, o);
      }
      if (lane == 0) warp_part[warp] = make_float4(lsum, asum, 0.f, 0.f);
      __syncthreads();
      if (warp == 0) {
        float4 v = lane < kCeWarps ? warp_part[lane] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          v.x += __shfl_xor_sync(0xffffffffu, v.x, o);
          v.y += __shfl_xor_sync(0xffffffffu, v.y, o);
        }
        if (lane == 0) slot_sums = v;
      }
      cluster_sync_all();
      if (tid == 0) {
        float4 r[kCeCluster];
#pragma unroll
        for (int c = 0; c < kCeCluster; ++c) r[c] = ld_peer_f4(&slot_sums, (uint32_t)c);
        float l = 0.f, A = 0.f;
#pragma unroll
        for (int c = 0; c < kCeCluster; ++c) {
          l += r[c].x;
          A += r[c].y;
        }
        bcast = make_float4(l, A, 0.f, 0.f);
        if (rank == 0) a.pair_loss[p] = -l * kLn2;
      }
      __syncthreads();
    }
    const float A = bcast.y;

    // ---- pass 3: gradient -(1/N) (a_v - P^S(v) A) ----
    if (grow) {
#pragma unroll
      for (int k = 0; k < KV; ++k) {
        const int vi = tid + k * kCeThreads;
        if (vi < vcnt) {
          float g[8];
#pragma unroll
          for (int j = 0; j < 8; ++j) g[j] = (xs[8 * k + j] * A - xt[8 * k + j]) * invN;
          store8(grow, (int64_t)(vbeg + vi) * 8, a.V, g);
        }
      }
    }
  }

  // no CTA leaves while a peer may still read its shared memory
  cluster_sync_all();

  // a copy whose wait gave up may still be in flight: wait for it, bounded
  if (tid == 0 && failed) {
    for (int s = 0; s < S; ++s)
      if (pending & (1u << s)) {
        // the outstanding phase of stage s is the last one issued there
        const int last = ((issued - 1 - s) / S) * S + s;
        if (last >= 0) mbar_wait_for(&full_bar[s], (uint32_t)(last / S) & 1u, kWaitLimitNs);
      }
  }

  // ---- the loss: the last CTA sums the per-pair losses in pair order ----
  __shared__ int s_last;
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    s_last = atomicAdd(&a.hdr->ctas_done, 1) == (int)gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  __shared__ double dpart[kCeWarps];
  const int per = (N + kCeThreads - 1) / kCeThreads;
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
    for (int w2 = 0; w2 < kCeWarps; ++w2) t += dpart[w2];
    a.loss[0] = N > 0 ? (float)(t / (double)N) : 0.f;
  }
}

template <int KV>
struct CeLaunch {
  static void *fn() { return reinterpret_cast<void *>(ce_kernel<KV>); }
};

void *ce_kernel_ptr(int kv) {
  switch (kv) {
    case 1: return CeLaunch<1>::fn();
    case 2: return CeLaunch<2>::fn();
    case 3: return CeLaunch<3>::fn();
    case 4: return CeLaunch<4>::fn();
    default: return CeLaunch<5>::fn();
  }
}

// Clusters of the main kernel that can be resident at once (cached per
// device, vectors per thread and shared-memory size).
int ce_max_clusters(int kv, size_t smem, int num_sms) {
  struct Entry {
    int dev, kv;
    size_t smem;
    int n;
  };
  static Entry cache[16];
  static int n_cache = 0;
  static std::mutex mu;
  int dev = 0;
  cudaGetDevice(&dev);
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < n_cache; ++i)
    if (cache[i].dev == dev && cache[i].kv == kv && cache[i].smem == smem) return cache[i].n;
  void *fn = ce_kernel_ptr(kv);
  // the largest size any call may request, so that no later call finds a smaller limit
  cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kCeSmemLimit);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kCeCluster * std::max(1, num_sms / kCeCluster));
  cfg.blockDim = dim3(kCeThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kCeCluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    n = std::max(1, num_sms / kCeCluster);
  }
  if (n_cache < 16) cache[n_cache++] = Entry{dev, kv, smem, n};
  return n;
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

// vectors per thread per row for a vocabulary (0: unsupported)
int distill_soft_ce_vecs(int64_t V) {
  const int64_t nvec = (V + 7) / 8;
  const int64_t chunk = (nvec + kCeCluster - 1) / kCeCluster;
  const int64_t kv = (chunk + kCeThreads - 1) / kCeThreads;
  return (V >= 1 && kv <= kCeMaxVecs) ? (int)std::max<int64_t>(kv, 1) : 0;
}

umim_status distill_soft_ce(const void *teacher, int32_t R_T, const void *student, int32_t R_S, int32_t V, int64_t ld,
                            const int32_t *teacher_rows, const int32_t *student_rows, int32_t max_pairs,
                            const int32_t *n_dev, float eps, float *loss, float *pair_loss, void *grad, void *ws,
                            int32_t *dev_status, cudaStream_t stream, int num_sms) {
  const int kv = distill_soft_ce_vecs(V);
  if (kv == 0) return UMIM_ERR_UNSUPPORTED;
  char *p = static_cast<char *>(ws);
  CeHeader *hdr = reinterpret_cast<CeHeader *>(p);
  p += a256(sizeof(CeHeader));
  int32_t *row_pair = reinterpret_cast<int32_t *>(p);
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
  a.hdr = hdr;
  a.status = dev_status ? dev_status : &hdr->status;
  const int nvec = (V + 7) / 8;
  a.chunk_vecs = (nvec + kCeCluster - 1) / kCeCluster;
  const size_t stage_bytes = (size_t)2 * a.chunk_vecs * 16;
  a.stages = (int)std::min<size_t>(kCeMaxStages, kCeSmemLimit / stage_bytes);
  if (a.stages < 2) return UMIM_ERR_UNSUPPORTED;
  const size_t smem = stage_bytes * a.stages;

  if (cudaMemsetAsync(hdr, 0, sizeof(CeHeader), stream) != cudaSuccess) return UMIM_ERR_CUDA;
  if (R_S > 0 && cudaMemsetAsync(row_pair, 0xFF, sizeof(int32_t) * (size_t)R_S, stream) != cudaSuccess)
    return UMIM_ERR_CUDA;
  const int prep_blocks = std::max(1, std::min((max_pairs + 255) / 256, num_sms * 4));
  trace_mark(stream, "distill.ce_prep");
  ce_prep_kernel<<<prep_blocks, 256, 0, stream>>>(a);
  if (cudaGetLastError() != cudaSuccess) return UMIM_ERR_CUDA;

  const int max_cl = ce_max_clusters(kv, smem, num_sms);
  const int n_cl = std::max(1, std::min(R_S, max_cl));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(n_cl * kCeCluster));
  cfg.blockDim = dim3(kCeThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kCeCluster;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  trace_mark(stream, "distill.soft_ce");
  cudaError_t e;
  switch (kv) {
    case 1: e = cudaLaunchKernelEx(&cfg, ce_kernel<1>, a); break;
    case 2: e = cudaLaunchKernelEx(&cfg, ce_kernel<2>, a); break;
    case 3: e = cudaLaunchKernelEx(&cfg, ce_kernel<3>, a); break;
    case 4: e = cudaLaunchKernelEx(&cfg, ce_kernel<4>, a); break;
    default: e = cudaLaunchKernelEx(&cfg, ce_kernel<5>, a); break;
  }
  trace_mark(stream, nullptr);
  return e == cudaSuccess ? UMIM_OK : UMIM_ERR_CUDA;
}

}  // namespace umim
