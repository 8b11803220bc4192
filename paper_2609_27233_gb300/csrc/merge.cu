// Merge module M_phi forward (App. C.1; Sec. 3.2 Eq. 1) for a batch of spans:
//   gather     E   = rows of the embedding table for every span token
//   GEMM1      H   = GELU(E W_kv^T + b_kv)        tcgen05, fp16 out + row stats of the fp32 values
//   pool       P   = LN_kv(H);  a_i = softmax(P_i q_i / sqrt(d_h));  o_i = a_i^T P_i
//   GEMM2      Z   = GELU(o W_o^T + b_o)          tcgen05 on fp16 operands, fp16 out + row stats
//                                                 of the fp32 values
//   LN_o       z   = LN_o(Z)                      fp32 into the output
//
// The two d x d projections are the only dense contractions of the module
// and run on the 5th-generation tensor cores: operands staged by TMA in
// 128-byte-swizzled shared memory, accumulator in tensor memory, one thread
// issuing tcgen05.mma, four epilogue warps reading the accumulator with
// tcgen05.ld.  A LayerNorm needs the statistics of a whole d-wide row, which
// spans d/256 output tiles, so each tile's epilogue writes the (mean, M2) of
// its 256 columns per row and the next kernel merges them (Chan et al.).
#include <algorithm>

#include <cuda_fp16.h>

#include "common.cuh"

namespace umim {
namespace {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int kGemmThreads = 224;   // warp 0: TMA, warp 1: MMA + TMEM owner, warps 2-5: epilogue, warp 6: side job
constexpr int kStageBytes = (BM + BN) * BK * 2;
constexpr int kGemmSmem = STAGES * kStageBytes + 1024;

__device__ __forceinline__ void bf16x8_to_float(uint4 u, float *f) {
  const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&u);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 x = __bfloat1622float2(h[i]);
    f[2 * i] = x.x;
    f[2 * i + 1] = x.y;
  }
}

template <typename OutT>
struct GemmArgs {
  int M, N, K;                 // A is [M][K], B is [N][K]
  uint32_t idesc;              // tcgen05 instruction descriptor (operand types)
  const __nv_bfloat16 *bias;   // [N]
  OutT *out;                   // [M][N]
  float2 *stats;               // [M][N / BN]
  // side job of warp 6: bf16 -> fp16 of cvt_n 16-byte vectors (0: none)
  const uint4 *cvt_in;
  uint4 *cvt_out;
  int64_t cvt_n;
  int32_t *status;
};

// Persistent: each CTA walks tiles blockIdx.x, blockIdx.x + gridDim.x, ...
// (n fastest, so CTAs running at the same time share the A block in L2).
// The accumulator is double-buffered in tensor memory (2 x 256 columns):
// while the epilogue warps drain tile i, the MMA thread accumulates tile i+1.
__device__ __forceinline__ void store32(__half *dst, const float (&v)[32]) {
  uint4 *d4 = reinterpret_cast<uint4 *>(dst);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    uint4 u;
    __half2 *h = reinterpret_cast<__half2 *>(&u);
#pragma unroll
    for (int e = 0; e < 4; ++e) h[e] = __floats2half2_rn(v[8 * i + 2 * e], v[8 * i + 2 * e + 1]);
    d4[i] = u;
  }
}

template <typename OutT>
__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_bias_gelu_kernel(const __grid_constant__ CUtensorMap a_map, const __grid_constant__ CUtensorMap b_map,
                          GemmArgs<OutT> g) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ uint64_t full_bar[STAGES], empty_bar[STAGES], acc_full[2], acc_empty[2];
  __shared__ uint32_t tmem_base;
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int num_kb = g.K / BK;
  const int tiles_n = g.N / BN;
  const int tiles = tiles_n * ((g.M + BM - 1) / BM);

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 4);     // one arrival per epilogue warp
    }
    fence_mbar_init();
    prefetch_tensormap(&a_map);
    prefetch_tensormap(&b_map);
  }
  if (warp == 1) {
    tmem_alloc(&tmem_base, 2 * BN);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;
  griddep_wait();

  if (warp == 0) {
    if (lane == 0) {
      const uint64_t pol_a = policy_evict_first();
      const uint64_t pol_b = policy_evict_last();
      uint32_t it = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < tiles && ok; tile += gridDim.x) {
        const int m0 = (tile / tiles_n) * BM, n0 = (tile % tiles_n) * BN;
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1;
          if (!mbar_wait(&empty_bar[s], ph ^ 1)) {
            set_error(g.status, UMIM_ERR_TIMEOUT);
            ok = false;
            break;
          }
          uint8_t *sa = smem + s * kStageBytes;
          uint8_t *sb = sa + BM * BK * 2;
          mbar_arrive_expect_tx(&full_bar[s], kStageBytes);
          tma_load_2d(sa, &a_map, &full_bar[s], kb * BK, m0, pol_a);
          tma_load_2d(sb, &b_map, &full_bar[s], kb * BK, n0, pol_b);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = g.idesc;
      uint32_t it = 0, local = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < tiles && ok; tile += gridDim.x, ++local) {
        const uint32_t buf = local & 1, aph = (local >> 1) & 1;
        if (!mbar_wait(&acc_empty[buf], aph ^ 1)) {
          set_error(g.status, UMIM_ERR_TIMEOUT);
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem + buf * BN;
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1;
          if (!mbar_wait(&full_bar[s], ph)) {
            set_error(g.status, UMIM_ERR_TIMEOUT);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_base = smem_u32(smem + s * kStageBytes);
          const uint32_t b_base = a_base + BM * BK * 2;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint64_t ad = sw128_kmajor_desc(a_base + k * 32);
            const uint64_t bd = sw128_kmajor_desc(b_base + k * 32);
            tc_mma_bf16(d_tmem, ad, bd, idesc, (kb | k) != 0 ? 1u : 0u);
          }
          tc_commit(&empty_bar[s]);
        }
        tc_commit(&acc_full[buf]);
      }
    }
  } else if (warp == 6) {
    // side job, converted while the tensor cores work (the memory traffic is
    // small next to the tile loads), 8 loads in flight per lane
    const int64_t step = (int64_t)gridDim.x * 32;
    for (int64_t i0 = (int64_t)blockIdx.x * 32 + lane; i0 < g.cvt_n; i0 += 8 * step) {
      uint4 u[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int64_t i = i0 + k * step;
        if (i < g.cvt_n) u[k] = __ldg(g.cvt_in + i);
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int64_t i = i0 + k * step;
        if (i < g.cvt_n) {
          float f[8];
          bf16x8_to_float(u[k], f);
          uint4 o;
          __half2 *hh = reinterpret_cast<__half2 *>(&o);
#pragma unroll
          for (int e = 0; e < 4; ++e) hh[e] = __floats2half2_rn(f[2 * e], f[2 * e + 1]);
          g.cvt_out[i] = o;
        }
      }
    }
  } else {
    const int q = warp & 3;   // TMEM lane quadrant this warp may read
    uint32_t local = 0;
    for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x, ++local) {
      const int m0 = (tile / tiles_n) * BM, n0 = (tile % tiles_n) * BN;
      const uint32_t buf = local & 1, aph = (local >> 1) & 1;
      const int row = m0 + q * 32 + lane;
      if (!mbar_wait(&acc_full[buf], aph)) {
        set_error(g.status, UMIM_ERR_TIMEOUT);
        break;
      }
      tc_fence_after();
      float mean = 0.f, m2 = 0.f, cnt = 0.f;
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        float v[32];
        tmem_ld_32x32b_x32(tmem + buf * BN + (static_cast<uint32_t>(q * 32) << 16) + c * 32, v);
        const uint4 *bp = reinterpret_cast<const uint4 *>(g.bias + n0 + c * 32);
        float sum = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          float bb[8];
          bf16x8_to_float(__ldg(bp + i), bb);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            v[8 * i + e] = gelu_erf(v[8 * i + e] + bb[e]);
            sum += v[8 * i + e];
          }
        }
        const float cm = sum * (1.f / 32.f);
        float cm2 = 0.f;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float dlt = v[i] - cm;
          cm2 += dlt * dlt;
        }
        const float nt = cnt + 32.f;
        const float delta = cm - mean;
        mean += delta * (32.f / nt);
        m2 += cm2 + delta * delta * (cnt * 32.f / nt);
        cnt = nt;
        if (row < g.M) store32(g.out + (int64_t)row * g.N + n0 + c * 32, v);
      }
      if (row < g.M) g.stats[(int64_t)row * tiles_n + n0 / BN] = make_float2(mean, m2);
      // this warp's quarter of the accumulator has been read
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[buf]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * BN);
  }
}

// ---------------------------------------------------------------------------
// gather the static embeddings of the span tokens
// ---------------------------------------------------------------------------
__global__ void gather_rows_kernel(const uint4 *table, int64_t vocab, const int32_t *ids, int64_t T, int d,
                                   uint4 *out, int32_t *status) {
  griddep_wait();
  const int vec = d / 8;   // 16-byte vectors per row
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  const int lane = threadIdx.x & 31;
  for (int64_t t = warp; t < T; t += nwarps) {
    const int id = ids[t];
    const bool ok = id >= 0 && id < vocab;
    if (!ok && lane == 0) set_error(status, UMIM_ERR_INVALID_ARG);
    const uint4 *src = table + (int64_t)(ok ? id : 0) * vec;
    uint4 *dst = out + t * vec;
    for (int i = lane; i < vec; i += 32) dst[i] = ok ? __ldg(src + i) : make_uint4(0, 0, 0, 0);
  }
}

// Running (count, mean, M2) of a row; merged pairwise (Chan et al.).
struct Moments {
  float n, mean, m2;
};

__device__ __forceinline__ Moments merge_moments(Moments a, Moments b) {
  const float n = a.n + b.n;
  if (b.n == 0.f) return a;
  if (a.n == 0.f) return b;
  const float delta = b.mean - a.mean, f = b.n / n;
  return {n, a.mean + delta * f, a.m2 + b.m2 + delta * delta * a.n * f};
}

// One warp merges the per-tile (mean, M2) of a row; every lane gets
// (mean, 1/sqrt(var + eps)).
__device__ __forceinline__ float2 row_moments_warp(const float2 *st, int ntiles, int d, float eps) {
  const int lane = threadIdx.x & 31;
  Moments m{0.f, 0.f, 0.f};
  for (int t = lane; t < ntiles; t += 32) {
    const float2 v = st[t];
    m = merge_moments(m, Moments{(float)BN, v.x, v.y});
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    Moments x{__shfl_xor_sync(0xffffffffu, m.n, o), __shfl_xor_sync(0xffffffffu, m.mean, o),
              __shfl_xor_sync(0xffffffffu, m.m2, o)};
    m = merge_moments(m, x);
  }
  return make_float2(m.mean, rsqrtf(m.m2 / (float)d + eps));
}

// ---------------------------------------------------------------------------
// LN_kv + attention pooling with the learnable queries.
// Persistent CTAs; span s goes to CTA s mod grid.  A producer warp copies each
// span's H rows (fp16) and row statistics into a 3-stage shared-memory ring
// with bulk asynchronous copies completing an mbarrier; 8 consumer warps
// compute from shared memory.  With P_jc = (H_jc - mu_j) r_j gamma_c + beta_c,
//   <P_j[head], q_head> = r_j (sum_c H_jc gamma_c q_c - mu_j A_head) + B_head,
//   A_head = sum_c gamma_c q_c,  B_head = sum_c beta_c q_c   (c in head),
// and, because the softmax weights alpha_j sum to one,
//   o_c = sum_j alpha_j P_jc = gamma_c (sum_j w_j H_jc - C_head) + beta_c,
//   w_j = alpha_j r_j,  C_head = sum_j w_j mu_j,
// so each element costs one multiply-add per span row in each pass.  o is
// written in fp16 (11 significant bits) as the A operand of the output
// projection.  16-byte column chunk cc (columns 8 cc .. 8 cc + 7) belongs to
// consumer thread cc mod 256; CH chunks per thread.
// ---------------------------------------------------------------------------
constexpr int kPoolRing = 3;
constexpr int kPoolConsumers = 256;

__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(src), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void consumer_sync() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

__host__ __device__ inline int pool_stage_bytes(int d) {
  return (UMIM_MAX_SPAN_TOKENS * (d * 2 + (d / BN) * 8) + 127) & ~127;
}

template <int CH>
__global__ void __launch_bounds__(kPoolConsumers + 32, CH <= 2 ? 2 : 1)
    pool_kernel(const __half *H, const float2 *stats, const int32_t *offs, int S, int64_t T, int d, int h,
                const __nv_bfloat16 *gamma, const __nv_bfloat16 *beta, const __nv_bfloat16 *query, float eps,
                __half *O, int32_t *status) {
  extern __shared__ __align__(128) uint8_t pool_smem[];
  __shared__ uint64_t full[kPoolRing], empty[kPoolRing];
  __shared__ int s_n[kPoolRing];
  __shared__ float2 s_mom[UMIM_MAX_SPAN_TOKENS];
  __shared__ float s_red[UMIM_MAX_SPAN_TOKENS][128];
  __shared__ float s_w[UMIM_MAX_SPAN_TOKENS][8];
  __shared__ float s_A[8], s_B[8], s_C[8];
  __shared__ int s_abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int ntiles = d / BN;
  const int sbytes = pool_stage_bytes(d);
  const int dh = d / h;
  const int q8 = dh / 8;
  const int seg = min(32, q8 & (-q8));   // lanes per segment: never straddles a head
  const int seg_per_head = q8 / seg;

  if (tid == 0) {
    for (int i = 0; i < kPoolRing; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kPoolConsumers / 32);
    }
    s_abort = 0;
    fence_mbar_init();
  }
  if (tid < 8) {
    s_A[tid] = 0.f;
    s_B[tid] = 0.f;
  }
  __syncthreads();
  griddep_wait();

  if (warp == kPoolConsumers / 32) {
    // ---- producer ----
    if (lane == 0) {
      int k = 0;
      for (int s = blockIdx.x; s < S; s += gridDim.x, ++k) {
        const int st = k % kPoolRing;
        if (!mbar_wait(&empty[st], ((k / kPoolRing) & 1) ^ 1)) {
          set_error(status, UMIM_ERR_TIMEOUT);
          break;
        }
        const int t0 = offs[s], t1 = offs[s + 1];
        int n = t1 - t0;
        if (t0 < 0 || n < 1 || n > UMIM_MAX_SPAN_TOKENS || t1 > T) {
          set_error(status, UMIM_ERR_INVALID_ARG);
          n = 0;
        }
        s_n[st] = n;
        uint8_t *sh = pool_smem + st * sbytes;
        uint8_t *ss = sh + UMIM_MAX_SPAN_TOKENS * d * 2;
        if (n > 0) {
          mbar_arrive_expect_tx(&full[st], n * (d * 2 + ntiles * 8));
          for (int j = 0; j < n; ++j) {
            bulk_g2s(sh + j * d * 2, H + (int64_t)(t0 + j) * d, d * 2, &full[st]);
            bulk_g2s(ss + j * ntiles * 8, stats + (int64_t)(t0 + j) * ntiles, ntiles * 8, &full[st]);
          }
        } else {
          mbar_arrive(&full[st]);
        }
      }
    }
    return;
  }

  // ---- consumers: per-column constants, kept for every span of this CTA ----
  float g[CH][8], b[CH][8], gq[CH][8];
#pragma unroll
  for (int i = 0; i < CH; ++i) {
    const int cc = tid + i * kPoolConsumers;
    if (cc < d / 8) {
      const int c = cc * 8;
      float q[8];
      bf16x8_to_float(*reinterpret_cast<const uint4 *>(gamma + c), g[i]);
      bf16x8_to_float(*reinterpret_cast<const uint4 *>(beta + c), b[i]);
      bf16x8_to_float(*reinterpret_cast<const uint4 *>(query + c), q);   // query [h][dh]: d contiguous values
      float a = 0.f, bb = 0.f;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        gq[i][e] = g[i][e] * q[e];
        a += gq[i][e];
        bb += b[i][e] * q[e];
      }
      for (int o = seg >> 1; o >= 1; o >>= 1) {
        a += __shfl_xor_sync(0xffffffffu, a, o, seg);
        bb += __shfl_xor_sync(0xffffffffu, bb, o, seg);
      }
      if ((lane & (seg - 1)) == 0) {
        atomicAdd(&s_A[c / dh], a);
        atomicAdd(&s_B[c / dh], bb);
      }
    }
  }
  consumer_sync();

  int k = 0;
  for (int s = blockIdx.x; s < S; s += gridDim.x, ++k) {
    const int st = k % kPoolRing;
    if (!mbar_wait(&full[st], (k / kPoolRing) & 1)) {
      set_error(status, UMIM_ERR_TIMEOUT);
      s_abort = 1;
    }
    consumer_sync();
    if (s_abort) break;
    const int n = s_n[st];
    const __half *sh = reinterpret_cast<const __half *>(pool_smem + st * sbytes);
    const float2 *ss = reinterpret_cast<const float2 *>(pool_smem + st * sbytes + UMIM_MAX_SPAN_TOKENS * d * 2);
    if (warp < n) {
      // merge the per-tile (mean, M2) of row `warp`
      Moments m{0.f, 0.f, 0.f};
      for (int t = lane; t < ntiles; t += 32) m = merge_moments(m, Moments{(float)BN, ss[warp * ntiles + t].x,
                                                                           ss[warp * ntiles + t].y});
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) {
        Moments x{__shfl_xor_sync(0xffffffffu, m.n, o), __shfl_xor_sync(0xffffffffu, m.mean, o),
                  __shfl_xor_sync(0xffffffffu, m.m2, o)};
        m = merge_moments(m, x);
      }
      if (lane == 0) s_mom[warp] = make_float2(m.mean, rsqrtf(m.m2 / (float)d + eps));
    }
    // pass 1: sum_c H_jc gamma_c q_c per (row, segment)
#pragma unroll
    for (int i = 0; i < CH; ++i) {
      const int cc = tid + i * kPoolConsumers;
      if (cc < d / 8) {
#pragma unroll
        for (int j = 0; j < UMIM_MAX_SPAN_TOKENS; ++j) {
          if (j < n) {
            const uint4 x = *reinterpret_cast<const uint4 *>(sh + j * d + cc * 8);
            const __half2 *h2 = reinterpret_cast<const __half2 *>(&x);
            float part = 0.f;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float2 f = __half22float2(h2[e]);
              part = fmaf(f.x, gq[i][2 * e], part);
              part = fmaf(f.y, gq[i][2 * e + 1], part);
            }
            for (int o = seg >> 1; o >= 1; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o, seg);
            if ((lane & (seg - 1)) == 0) s_red[j][cc / seg] = part;
          }
        }
      }
    }
    consumer_sync();
    // softmax over the span for each head, then w_j = alpha_j r_j and C_head
    if (tid < h && n > 0) {
      const float inv = rsqrtf((float)dh);
      float sc[UMIM_MAX_SPAN_TOKENS];
      float mx = -INFINITY;
#pragma unroll
      for (int j = 0; j < UMIM_MAX_SPAN_TOKENS; ++j) {
        float v = 0.f;
        if (j < n) {
          for (int i = 0; i < seg_per_head; ++i) v += s_red[j][tid * seg_per_head + i];
          const float2 m = s_mom[j];
          sc[j] = (m.y * (v - m.x * s_A[tid]) + s_B[tid]) * inv;
        } else {
          sc[j] = -INFINITY;
        }
        mx = fmaxf(mx, sc[j]);
      }
      float den = 0.f;
#pragma unroll
      for (int j = 0; j < UMIM_MAX_SPAN_TOKENS; ++j) {
        sc[j] = j < n ? expf(sc[j] - mx) : 0.f;
        den += sc[j];
      }
      float C = 0.f;
#pragma unroll
      for (int j = 0; j < UMIM_MAX_SPAN_TOKENS; ++j) {
        const float2 m = j < n ? s_mom[j] : make_float2(0.f, 0.f);
        const float wj = sc[j] / den * m.y;
        s_w[j][tid] = wj;
        C += wj * m.x;
      }
      s_C[tid] = C;
    }
    consumer_sync();
    // pass 2: o_c = gamma_c (sum_j w_j H_jc - C_head) + beta_c
#pragma unroll
    for (int i = 0; i < CH; ++i) {
      const int cc = tid + i * kPoolConsumers;
      if (cc < d / 8) {
        const int head = cc * 8 / dh;
        float x[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) x[e] = 0.f;
#pragma unroll
        for (int j = 0; j < UMIM_MAX_SPAN_TOKENS; ++j) {
          if (j < n) {
            const float wj = s_w[j][head];
            const uint4 hv = *reinterpret_cast<const uint4 *>(sh + j * d + cc * 8);
            const __half2 *h2 = reinterpret_cast<const __half2 *>(&hv);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float2 f = __half22float2(h2[e]);
              x[2 * e] = fmaf(wj, f.x, x[2 * e]);
              x[2 * e + 1] = fmaf(wj, f.y, x[2 * e + 1]);
            }
          }
        }
        const float C = n > 0 ? s_C[head] : 0.f;
        uint4 packed;
        __half2 *hp = reinterpret_cast<__half2 *>(&packed);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float o0 = n > 0 ? fmaf(g[i][2 * e], x[2 * e] - C, b[i][2 * e]) : 0.f;
          const float o1 = n > 0 ? fmaf(g[i][2 * e + 1], x[2 * e + 1] - C, b[i][2 * e + 1]) : 0.f;
          hp[e] = __floats2half2_rn(o0, o1);
        }
        *reinterpret_cast<uint4 *>(O + (int64_t)s * d + cc * 8) = packed;
      }
    }
    // this warp no longer reads the stage
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[st]);
    consumer_sync();   // s_mom / s_red / s_w / s_C are rewritten for the next span
  }
}

// ---------------------------------------------------------------------------
// LN_o over rows of Z (fp16, the GELU output of the projection; its row
// statistics were taken from the fp32 values), one warp per row, z in fp32
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
    ln_rows_kernel(const __half *Z, float *out, const float2 *stats, int S, int d, const __nv_bfloat16 *gamma,
                   const __nv_bfloat16 *beta, float eps) {
  griddep_wait();
  const int r = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= S) return;
  const float2 m = row_moments_warp(stats + (int64_t)r * (d / BN), d / BN, d, eps);
  const __half *row = Z + (int64_t)r * d;
  float *dst = out + (int64_t)r * d;
#pragma unroll 2
  for (int c = lane * 8; c < d; c += 256) {
    const uint4 u = *reinterpret_cast<const uint4 *>(row + c);
    const __half2 *h2 = reinterpret_cast<const __half2 *>(&u);
    float g[8], b[8];
    bf16x8_to_float(*reinterpret_cast<const uint4 *>(gamma + c), g);
    bf16x8_to_float(*reinterpret_cast<const uint4 *>(beta + c), b);
    float y[8];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 x = __half22float2(h2[e]);
      y[2 * e] = (x.x - m.x) * m.y * g[2 * e] + b[2 * e];
      y[2 * e + 1] = (x.y - m.x) * m.y * g[2 * e + 1] + b[2 * e + 1];
    }
    *reinterpret_cast<float4 *>(dst + c) = make_float4(y[0], y[1], y[2], y[3]);
    *reinterpret_cast<float4 *>(dst + c + 4) = make_float4(y[4], y[5], y[6], y[7]);
  }
}

// W_o from bf16 to fp16 (exact for values in fp16's normal range)
__global__ void bf16_to_f16_kernel(const uint4 *in, uint4 *out, int64_t n_vec) {
  griddep_wait();
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n_vec; i += (int64_t)gridDim.x * blockDim.x) {
    const uint4 u = in[i];
    float f[8];
    bf16x8_to_float(u, f);
    uint4 o;
    __half2 *h = reinterpret_cast<__half2 *>(&o);
#pragma unroll
    for (int e = 0; e < 4; ++e) h[e] = __floats2half2_rn(f[2 * e], f[2 * e + 1]);
    out[i] = o;
  }
}

inline size_t al1k(size_t x) { return (x + 1023) & ~size_t(1023); }

}  // namespace

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *,
                                   CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                   CUtensorMapFloatOOBfill);
EncodeTiledFn get_encode_tiled();

size_t merge_spans_workspace_bytes(int64_t T, int S, int d) {
  const int nt = d / BN;
  size_t b = 0;
  b += al1k((size_t)std::max<int64_t>(std::max<int64_t>(T, S), 1) * d * 2);   // E (bf16), later Z (fp16)
  b += al1k((size_t)std::max<int64_t>(T, 1) * d * 2);          // H (fp16)
  b += al1k((size_t)std::max<int64_t>(T, 1) * nt * 8);         // stats of H
  b += al1k((size_t)std::max(S, 1) * d * 2);                   // o (fp16)
  b += al1k((size_t)d * d * 2);                                 // W_o (fp16)
  b += al1k((size_t)std::max(S, 1) * nt * 8);                  // stats of Z
  return b;
}

static bool encode_kmajor(EncodeTiledFn enc, CUtensorMap *map, const void *base, int64_t rows, int K,
                          int box_rows, bool fp16) {
  const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)K * 2};
  const cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
  const cuuint32_t es[2] = {1, 1};
  return enc(map, fp16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
             const_cast<void *>(base), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// out[M][d] = GELU(A[M][d] B[d][d]^T + bias); A and B both bf16 or both fp16
template <typename OutT>
static umim_status launch_gemm(EncodeTiledFn enc, const void *A, int64_t M, const void *Bw, int d, bool fp16,
                               const void *bias, OutT *out, float2 *stats, int32_t *status, cudaStream_t st,
                               const char *label, int num_sms, const void *cvt_in = nullptr, void *cvt_out = nullptr,
                               int64_t cvt_n = 0) {
  CUtensorMap am, bm;
  if (!encode_kmajor(enc, &am, A, M, d, BM, fp16) || !encode_kmajor(enc, &bm, Bw, d, d, BN, fp16))
    return UMIM_ERR_CUDA;
  GemmArgs<OutT> g;
  g.M = (int)M;
  g.N = d;
  g.K = d;
  g.idesc = idesc_f32acc(BM, BN, fp16);
  g.bias = static_cast<const __nv_bfloat16 *>(bias);
  g.out = out;
  g.stats = stats;
  g.cvt_in = static_cast<const uint4 *>(cvt_in);
  g.cvt_out = static_cast<uint4 *>(cvt_out);
  g.cvt_n = cvt_n;
  g.status = status;
  // set on every call: the attribute belongs to the current device, and calls may
  // come for several devices and from several threads
  if (cudaFuncSetAttribute(gemm_bias_gelu_kernel<OutT>, cudaFuncAttributeMaxDynamicSharedMemorySize, kGemmSmem) !=
      cudaSuccess)
    return UMIM_ERR_CUDA;
  const int64_t tiles = (int64_t)(d / BN) * ((M + BM - 1) / BM);
  const int grid = (int)std::min<int64_t>(tiles, std::max(1, num_sms));
  trace_mark(st, label);
  return launch_pdl(gemm_bias_gelu_kernel<OutT>, dim3(grid), dim3(kGemmThreads), kGemmSmem, st, am, bm, g) ==
                 cudaSuccess
             ? UMIM_OK
             : UMIM_ERR_CUDA;
}

umim_status merge_spans(const void *embeddings, int64_t vocab, const int32_t *token_ids, int64_t T,
                        const int32_t *span_offsets, int S, const umim_merge_weights *w, float *surrogates,
                        void *workspace, int32_t *status, cudaStream_t st, int num_sms) {
  EncodeTiledFn enc = get_encode_tiled();
  if (!enc) return UMIM_ERR_CUDA;
  const int d = w->d_model, nt = d / BN;
  char *p = static_cast<char *>(workspace);
  __nv_bfloat16 *E = reinterpret_cast<__nv_bfloat16 *>(p);
  __half *Z16 = reinterpret_cast<__half *>(p);   // E is dead once GEMM1 has run
  p += al1k((size_t)std::max<int64_t>(std::max<int64_t>(T, S), 1) * d * 2);
  __half *H = reinterpret_cast<__half *>(p);
  p += al1k((size_t)std::max<int64_t>(T, 1) * d * 2);
  float2 *st1 = reinterpret_cast<float2 *>(p);
  p += al1k((size_t)std::max<int64_t>(T, 1) * nt * 8);
  __half *O = reinterpret_cast<__half *>(p);
  p += al1k((size_t)std::max(S, 1) * d * 2);
  __half *Wo16 = reinterpret_cast<__half *>(p);
  p += al1k((size_t)d * d * 2);
  float2 *st2 = reinterpret_cast<float2 *>(p);

  if (S == 0) return UMIM_OK;
  bool wo_in_gemm1 = false;
  if (T > 0) {
    const int blocks = std::max(1, std::min<int>((int)((T + 7) / 8), num_sms * 8));
    trace_mark(st, "merge.gather");
    if (launch_pdl(gather_rows_kernel, dim3(blocks), dim3(256), 0, st, static_cast<const uint4 *>(embeddings), vocab,
                   token_ids, T, d, reinterpret_cast<uint4 *>(E), status) != cudaSuccess)
      return UMIM_ERR_CUDA;
    // W_o -> fp16 rides along in a side warp of GEMM1 when its share is small
    // next to the tiles its CTA computes; else a kernel of its own
    const int64_t tiles1 = (int64_t)(d / BN) * ((T + BM - 1) / BM);
    const int64_t grid1 = std::min<int64_t>(tiles1, std::max(1, num_sms));
    const int64_t n_vec = (int64_t)d * d / 8;
    wo_in_gemm1 = n_vec <= 128 * 32 * grid1 * (tiles1 / grid1);
    umim_status r = launch_gemm(enc, E, T, w->w_kv, d, false, w->b_kv, H, st1, status, st, "merge.gemm1", num_sms,
                                wo_in_gemm1 ? w->w_o : nullptr, wo_in_gemm1 ? Wo16 : nullptr,
                                wo_in_gemm1 ? n_vec : 0);
    if (r != UMIM_OK) return r;
  }
  trace_mark(st, "merge.pool");
  const int psmem = kPoolRing * pool_stage_bytes(d);
  const int chunks = d / 8 / kPoolConsumers;   // 16-byte column chunks per consumer thread (d <= 8192)
  auto pk = chunks <= 1 ? pool_kernel<1> : (chunks == 2 ? pool_kernel<2> : pool_kernel<4>);
  if (cudaFuncSetAttribute(pk, cudaFuncAttributeMaxDynamicSharedMemorySize, psmem) != cudaSuccess)
    return UMIM_ERR_CUDA;
  int pool_per_sm = 1;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&pool_per_sm, pk, kPoolConsumers + 32, psmem) != cudaSuccess ||
      pool_per_sm < 1)
    pool_per_sm = 1;
  const int pool_grid = std::max(1, std::min(S, std::max(1, num_sms) * pool_per_sm));
  if (launch_pdl(pk, dim3(pool_grid), dim3(kPoolConsumers + 32), psmem, st, (const __half *)H, (const float2 *)st1,
                 span_offsets, S, T, d, (int)w->n_heads, static_cast<const __nv_bfloat16 *>(w->ln_kv_gamma),
                 static_cast<const __nv_bfloat16 *>(w->ln_kv_beta), static_cast<const __nv_bfloat16 *>(w->query),
                 w->ln_eps, O, status) != cudaSuccess)
    return UMIM_ERR_CUDA;
  if (!wo_in_gemm1) {
    trace_mark(st, "merge.wo_f16");
    if (launch_pdl(bf16_to_f16_kernel, dim3(std::max(1, num_sms) * 4), dim3(256), 0, st,
                   static_cast<const uint4 *>(w->w_o), reinterpret_cast<uint4 *>(Wo16), (int64_t)d * d / 8) !=
        cudaSuccess)
      return UMIM_ERR_CUDA;
  }
  umim_status r = launch_gemm(enc, O, S, Wo16, d, true, w->b_o, Z16, st2, status, st, "merge.gemm2", num_sms);
  if (r != UMIM_OK) return r;
  trace_mark(st, "merge.ln_o");
  if (launch_pdl(ln_rows_kernel, dim3((S + 7) / 8), dim3(256), 0, st, (const __half *)Z16, surrogates,
                 (const float2 *)st2, S, d,
                 static_cast<const __nv_bfloat16 *>(w->ln_o_gamma), static_cast<const __nv_bfloat16 *>(w->ln_o_beta),
                 w->ln_eps) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(st, nullptr);
  return UMIM_OK;
}

}  // namespace umim
