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
  float cvt_scale;             // applied before the fp16 rounding of the side job
  float acc_scale;             // applied to the accumulator before the bias (undoes an operand scaling)
  int32_t *range_flag;         // set (with UMIM_ERR_UNSUPPORTED) when a value does not fit fp16
  int32_t *status;
};

// fp16's largest finite value is 65504; a value at or above it (or not
// finite) cannot be stored in the fp16 intermediates of the merge module.
constexpr float kF16Limit = 65504.f;

// W_o is staged in fp16 multiplied by this power of two (GEMM2's accumulator is
// multiplied back by its inverse, both exact): entries from 2^-22 up to
// 65504 / 2^8 = 255.875 in magnitude keep a normal fp16 form, so bf16 weights
// of that range are represented exactly.
constexpr float kWoScale = 256.f;

__device__ __forceinline__ void flag_range(int32_t *flag, int32_t *status) {
  set_error(status, UMIM_ERR_UNSUPPORTED);
  if (flag) *reinterpret_cast<volatile int32_t *>(flag) = 1;
}

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
          bool bad = false;
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            f[e] *= g.cvt_scale;
            bad |= !(fabsf(f[e]) < kF16Limit);
          }
          if (bad) flag_range(g.range_flag, g.status);
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
      bool bad = false;
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
            v[8 * i + e] = gelu_erf(fmaf(v[8 * i + e], g.acc_scale, bb[e]));
            sum += v[8 * i + e];
            bad |= !(fabsf(v[8 * i + e]) < kF16Limit);
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
        if (row < g.M && in_bounds(n0 + c * 32 + 31, g.N, g.status, kSiteMergeGemmStore))
          store32(g.out + (int64_t)row * g.N + n0 + c * 32, v);
      }
      if (row < g.M) g.stats[(int64_t)row * tiles_n + n0 / BN] = make_float2(mean, m2);
      if (bad && row < g.M) flag_range(g.range_flag, g.status);   // this row's fp16 output overflowed
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
                                   uint4 *out, int32_t *range_flag, int32_t *status) {
  griddep_wait();
  if (blockIdx.x == 0 && threadIdx.x == 0) *range_flag = 0;   // the first kernel of the call
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
// (mean, 1/sqrt(var + eps)).  Every tile holds BN values, so the row's mean is
// the tiles' average mean and M2 = sum M2_t + BN sum (mean_t - mean)^2.
__device__ __forceinline__ float2 row_moments_warp(const float2 *st, int ntiles, int d, float eps) {
  const int lane = threadIdx.x & 31;
  const float2 v = lane < ntiles ? st[lane] : make_float2(0.f, 0.f);   // ntiles <= 32 (d <= 8192)
  float sm = v.x, s2 = v.y;
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    sm += __shfl_xor_sync(0xffffffffu, sm, o);
    s2 += __shfl_xor_sync(0xffffffffu, s2, o);
  }
  const float mean = sm / (float)ntiles;
  float dv = lane < ntiles ? (v.x - mean) * (v.x - mean) : 0.f;
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) dv += __shfl_xor_sync(0xffffffffu, dv, o);
  return make_float2(mean, rsqrtf((s2 + (float)BN * dv) / (float)d + eps));
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
                __half *O, int32_t *range_flag, int32_t *status) {
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
        bool bad = false;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float o0 = n > 0 ? fmaf(g[i][2 * e], x[2 * e] - C, b[i][2 * e]) : 0.f;
          const float o1 = n > 0 ? fmaf(g[i][2 * e + 1], x[2 * e + 1] - C, b[i][2 * e + 1]) : 0.f;
          bad |= !(fabsf(o0) < kF16Limit) || !(fabsf(o1) < kF16Limit);
          hp[e] = __floats2half2_rn(o0, o1);
        }
        if (bad) flag_range(range_flag, status);
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
// LN_kv + attention pooling, one warp per (span, head) item: the default for
// head widths up to 1024.  Warp w of the grid always takes head w mod h, so
// its lanes keep that head's LayerNorm scale, shift and gamma*q in registers,
// and walks the spans w / h, w / h + (warps / h), ...  Each warp owns two
// shared-memory buffers: lane 0 bulk-copies the next item's rows of H (this
// head's columns) and their per-tile statistics into one buffer while the
// warp computes the current item from the other, so no CTA barrier is ever
// taken.  The LayerNorm algebra is the one of pool_kernel above; a row's
// (mean, M2) comes from its equal-count tiles as mean = avg(mean_t),
// M2 = sum M2_t + 256 sum (mean_t - mean)^2.
// ---------------------------------------------------------------------------
constexpr int kHeadWarps = 12;
constexpr int kHeadBufs = 2;

// one buffer: [4][dh] fp16 rows, then [4][ntiles] float2 statistics; a multiple
// of 128 bytes so that every buffer can take a tensor copy
__host__ __device__ inline int head_buf_bytes(int dh, int ntiles) {
  return (UMIM_MAX_SPAN_TOKENS * (dh * 2 + ntiles * 8) + 127) & ~127;
}

__device__ __forceinline__ void tma_load_3d(void *dst, const CUtensorMap *map, uint64_t *bar, int c0, int c1, int c2,
                                            uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

// H viewed as [T][d / inner][inner] fp16 with inner = 64, 128 or 256 dividing
// the head width; map n - 1 copies n rows of one head (mid = dh / inner boxes
// of inner columns each) in one operation, landing as [n][dh] in shared memory
struct HeadMaps {
  CUtensorMap m[UMIM_MAX_SPAN_TOKENS];
};

// One (span, head) item with N rows, staged in shared memory: hs [N][dh] fp16,
// ts [N][ntiles] per-tile (mean, M2).  Writes the head's slice of o and
// returns nonzero if some fp16 value of it is not finite.
template <int CPL, int N>
__device__ __forceinline__ uint32_t pool_item(const __half *hs, const float2 *ts, const float2 (&gq)[CPL][4],
                                              const uint32_t (&gp)[CPL][4], const uint32_t (&bp)[CPL][4], float A,
                                              float Bq, int lane, int Ch, int dh, int ntiles, float inv_ntiles,
                                              float inv_d, float eps, float inv_sqrt_dh, __half *orow) {
  // scores: per row sum_c H gamma q over the head (packed fp32 pairs, two
  // accumulators per row), then the per-tile moments; the rows' shuffle
  // reductions interleave
  float p[N], sm[N], s2[N], tx[N];
#pragma unroll
  for (int j = 0; j < N; ++j) {
    float2 pa = make_float2(0.f, 0.f), pb = make_float2(0.f, 0.f);
#pragma unroll
    for (int k = 0; k < CPL; ++k) {
      const int ci = k * 32 + lane;
      if (ci < Ch) {
        const uint4 x = *reinterpret_cast<const uint4 *>(hs + j * dh + ci * 8);
        const __half2 *h2 = reinterpret_cast<const __half2 *>(&x);
        pa = __ffma2_rn(__half22float2(h2[0]), gq[k][0], pa);
        pb = __ffma2_rn(__half22float2(h2[1]), gq[k][1], pb);
        pa = __ffma2_rn(__half22float2(h2[2]), gq[k][2], pa);
        pb = __ffma2_rn(__half22float2(h2[3]), gq[k][3], pb);
      }
    }
    const float2 t = lane < ntiles ? ts[j * ntiles + lane] : make_float2(0.f, 0.f);
    p[j] = (pa.x + pb.x) + (pa.y + pb.y);
    tx[j] = t.x;
    sm[j] = t.x;
    s2[j] = t.y;
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
#pragma unroll
    for (int j = 0; j < N; ++j) {
      p[j] += __shfl_xor_sync(0xffffffffu, p[j], o);
      sm[j] += __shfl_xor_sync(0xffffffffu, sm[j], o);
      s2[j] += __shfl_xor_sync(0xffffffffu, s2[j], o);
    }
  }
  float mu[N], dv[N];
#pragma unroll
  for (int j = 0; j < N; ++j) {
    mu[j] = sm[j] * inv_ntiles;
    dv[j] = lane < ntiles ? (tx[j] - mu[j]) * (tx[j] - mu[j]) : 0.f;
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
#pragma unroll
    for (int j = 0; j < N; ++j) dv[j] += __shfl_xor_sync(0xffffffffu, dv[j], o);
  }
  // softmax over the rows; w_j = alpha_j r_j, C = sum_j w_j mu_j
  float rs[N], w[N], mx = -INFINITY;
#pragma unroll
  for (int j = 0; j < N; ++j) {
    rs[j] = rsqrtf((s2[j] + (float)BN * dv[j]) * inv_d + eps);
    w[j] = (rs[j] * (p[j] - mu[j] * A) + Bq) * inv_sqrt_dh;
    mx = fmaxf(mx, w[j]);
  }
  float den = 0.f;
#pragma unroll
  for (int j = 0; j < N; ++j) {
    w[j] = expf(w[j] - mx);
    den += w[j];
  }
  const float inv_den = 1.f / den;
  float C = 0.f;
#pragma unroll
  for (int j = 0; j < N; ++j) {
    w[j] = w[j] * inv_den * rs[j];
    C = fmaf(w[j], mu[j], C);
  }
  // o_c = gamma_c (sum_j w_j H_jc - C) + beta_c; an fp16 result whose exponent
  // bits are all set (inf or NaN) carries into bit 15 of its half when 0x0400
  // is added to the masked exponent
  uint32_t bad = 0;
#pragma unroll
  for (int k = 0; k < CPL; ++k) {
    const int ci = k * 32 + lane;
    if (ci < Ch) {
      float2 x[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) x[e] = make_float2(-C, -C);
#pragma unroll
      for (int j = 0; j < N; ++j) {
        const uint4 hv = *reinterpret_cast<const uint4 *>(hs + j * dh + ci * 8);
        const __half2 *h2 = reinterpret_cast<const __half2 *>(&hv);
        const float2 w2 = make_float2(w[j], w[j]);
#pragma unroll
        for (int e = 0; e < 4; ++e) x[e] = __ffma2_rn(w2, __half22float2(h2[e]), x[e]);
      }
      uint4 packed;
      uint32_t *pw = reinterpret_cast<uint32_t *>(&packed);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 g2 = make_float2(__uint_as_float(gp[k][e] << 16), __uint_as_float(gp[k][e] & 0xFFFF0000u));
        const float2 b2 = make_float2(__uint_as_float(bp[k][e] << 16), __uint_as_float(bp[k][e] & 0xFFFF0000u));
        const __half2 hh = __float22half2_rn(__ffma2_rn(g2, x[e], b2));
        pw[e] = *reinterpret_cast<const uint32_t *>(&hh);
        bad |= (pw[e] & 0x7C007C00u) + 0x04000400u;
      }
      *reinterpret_cast<uint4 *>(orow + ci * 8) = packed;
    }
  }
  return bad & 0x80008000u;
}

template <int CPL>
__global__ void __launch_bounds__(kHeadWarps * 32, 1)
    pool_head_kernel(const __grid_constant__ HeadMaps maps, int mid, const __half *H, const float2 *stats,
                     const int32_t *offs, int S, int64_t T, int d, int h,
                     const __nv_bfloat16 *gamma, const __nv_bfloat16 *beta, const __nv_bfloat16 *query, float eps,
                     __half *O, int32_t *range_flag, int32_t *status) {
  extern __shared__ __align__(128) uint8_t head_smem[];
  __shared__ uint64_t bars[kHeadWarps][kHeadBufs];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int dh = d / h, Ch = dh / 8, ntiles = d / BN;
  const int buf_bytes = head_buf_bytes(dh, ntiles);
  uint8_t *wbuf = head_smem + (size_t)warp * kHeadBufs * buf_bytes;
  const int gw = blockIdx.x * kHeadWarps + warp;
  const int nw = gridDim.x * kHeadWarps;   // a multiple of h (the host sizes the grid so)
  const int head = gw % h;
  const int span_step = nw / h;

  // this lane's columns of the head: chunk ci = k * 32 + lane
  float2 gq[CPL][4];                 // gamma * q, column pairs
  uint32_t gp[CPL][4], bp[CPL][4];   // gamma and beta as bf16 pairs
  float A = 0.f, Bq = 0.f;            // sum over the head of gamma q and of beta q
#pragma unroll
  for (int k = 0; k < CPL; ++k) {
    const int ci = k * 32 + lane;
    float g[8], b[8], q[8];
    uint4 g4 = make_uint4(0, 0, 0, 0), b4 = g4, q4 = g4;
    if (ci < Ch) {
      const int c = head * dh + ci * 8;
      g4 = *reinterpret_cast<const uint4 *>(gamma + c);
      b4 = *reinterpret_cast<const uint4 *>(beta + c);
      q4 = *reinterpret_cast<const uint4 *>(query + c);   // query [h][dh]: d contiguous values
    }
    bf16x8_to_float(g4, g);
    bf16x8_to_float(b4, b);
    bf16x8_to_float(q4, q);
    gp[k][0] = g4.x, gp[k][1] = g4.y, gp[k][2] = g4.z, gp[k][3] = g4.w;
    bp[k][0] = b4.x, bp[k][1] = b4.y, bp[k][2] = b4.z, bp[k][3] = b4.w;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      gq[k][e] = make_float2(g[2 * e] * q[2 * e], g[2 * e + 1] * q[2 * e + 1]);
      A += gq[k][e].x + gq[k][e].y;
      Bq = fmaf(b[2 * e], q[2 * e], Bq);
      Bq = fmaf(b[2 * e + 1], q[2 * e + 1], Bq);
    }
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) {
    A += __shfl_xor_sync(0xffffffffu, A, o);
    Bq += __shfl_xor_sync(0xffffffffu, Bq, o);
  }
  if (lane == 0) {
    for (int i = 0; i < kHeadBufs; ++i) mbar_init(&bars[warp][i], 1);
    fence_mbar_init();
  }
  __syncwarp();
  griddep_wait();   // H and its statistics come from the projection kernel

  const int n_items = (S - gw / h + span_step - 1) / span_step;   // spans gw/h, gw/h + step, ... below S
  const uint64_t pol = policy_evict_first();
  if (lane == 0) prefetch_tensormap(&maps.m[0]);
  // lane 0 loads the span offsets one item ahead of the copies that need them
  int pf_t0 = 0, pf_t1 = 0;
  auto prefetch = [&](int item) {
    if (item < n_items) {
      const int sp = gw / h + item * span_step;
      pf_t0 = offs[sp];
      pf_t1 = offs[sp + 1];
    }
  };
  // lane 0: issue the copies of the item-th span of this warp into buffer `b`
  // (its offsets were prefetched); returns the span's row count (0 for an
  // invalid span)
  auto issue = [&](int b) -> int {
    uint64_t *bar = &bars[warp][b];
    const int t0 = pf_t0, t1 = pf_t1;
    int n = t1 - t0;
    if (t0 < 0 || n < 1 || n > UMIM_MAX_SPAN_TOKENS || t1 > T) {
      if (head == 0) set_error(status, UMIM_ERR_INVALID_ARG);
      n = 0;
    }
    if (n > 0 && !in_bounds((int64_t)t1 * ntiles - 1, T * ntiles, status, kSiteMergePoolStats)) n = 0;
    if (n == 0) {
      mbar_arrive(bar);
      return 0;
    }
    uint8_t *dst = wbuf + b * buf_bytes;
    mbar_arrive_expect_tx(bar, n * (dh * 2 + ntiles * 8));
    // the span's rows of this head in one tensor copy, their statistics (consecutive) in one bulk copy
    tma_load_3d(dst, &maps.m[n - 1], bar, 0, head * mid, t0, pol);
    bulk_g2s(dst + UMIM_MAX_SPAN_TOKENS * dh * 2, stats + (int64_t)t0 * ntiles, n * ntiles * 8, bar);
    return n;
  };

  static_assert(kHeadBufs == 2, "two buffers per warp");
  int n_buf0 = 0, n_buf1 = 0;   // row counts of the items in flight (lane 0's view)
  if (lane == 0) {
    prefetch(0);
    if (n_items > 0) {
      n_buf0 = issue(0);
      prefetch(1);
    }
    if (n_items > 1) {
      n_buf1 = issue(1);
      prefetch(2);
    }
  }
  const float inv_sqrt_dh = rsqrtf((float)dh), inv_ntiles = 1.f / (float)ntiles, inv_d = 1.f / (float)d;
  for (int item = 0; item < n_items; ++item) {
    const int b = item % kHeadBufs;
    const int sp = gw / h + item * span_step;
    const int n = __shfl_sync(0xffffffffu, b ? n_buf1 : n_buf0, 0);
    if (!__all_sync(0xffffffffu, mbar_wait(&bars[warp][b], (item / kHeadBufs) & 1))) {
      set_error(status, UMIM_ERR_TIMEOUT);
      // let the other buffer's copies land (bounded) before leaving
      if (item + 1 < n_items) mbar_wait(&bars[warp][(item + 1) % kHeadBufs], ((item + 1) / kHeadBufs) & 1);
      return;
    }
    const __half *hs = reinterpret_cast<const __half *>(wbuf + b * buf_bytes);
    const float2 *ts = reinterpret_cast<const float2 *>(wbuf + b * buf_bytes + UMIM_MAX_SPAN_TOKENS * dh * 2);
    uint32_t bad = 0;
    __half *orow = O + (int64_t)sp * d + (int64_t)head * dh;
    if (in_bounds(sp, S, status, kSiteMergePoolSpan)) switch (n) {
      case 1: bad = pool_item<CPL, 1>(hs, ts, gq, gp, bp, A, Bq, lane, Ch, dh, ntiles, inv_ntiles, inv_d, eps,
                                      inv_sqrt_dh, orow); break;
      case 2: bad = pool_item<CPL, 2>(hs, ts, gq, gp, bp, A, Bq, lane, Ch, dh, ntiles, inv_ntiles, inv_d, eps,
                                      inv_sqrt_dh, orow); break;
      case 3: bad = pool_item<CPL, 3>(hs, ts, gq, gp, bp, A, Bq, lane, Ch, dh, ntiles, inv_ntiles, inv_d, eps,
                                      inv_sqrt_dh, orow); break;
      case 4: bad = pool_item<CPL, 4>(hs, ts, gq, gp, bp, A, Bq, lane, Ch, dh, ntiles, inv_ntiles, inv_d, eps,
                                      inv_sqrt_dh, orow); break;
      default:   // an invalid span: o = 0
#pragma unroll
        for (int k = 0; k < CPL; ++k)
          if (k * 32 + lane < Ch) *reinterpret_cast<uint4 *>(orow + (k * 32 + lane) * 8) = make_uint4(0, 0, 0, 0);
    }
    if (__any_sync(0xffffffffu, bad != 0) && lane == 0) flag_range(range_flag, status);
    // every lane is done with this buffer: refill it with the item two ahead
    __syncwarp();
    if (lane == 0 && item + kHeadBufs < n_items) {
      const int nn = issue(b);
      prefetch(item + kHeadBufs + 1);
      if (b) n_buf1 = nn;
      else n_buf0 = nn;
    }
  }
}

// ---------------------------------------------------------------------------
// LN_o over rows of Z (fp16, the GELU output of the projection; its row
// statistics were taken from the fp32 values), one warp per row, z in fp32
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
    ln_rows_kernel(const __half *Z, float *out, const float2 *stats, int S, int d, const __nv_bfloat16 *gamma,
                   const __nv_bfloat16 *beta, float eps, const int32_t *range_flag) {
  griddep_wait();
  // an intermediate did not fit fp16 (already reported): write no surrogate
  if (*reinterpret_cast<const volatile int32_t *>(range_flag) != 0) return;
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

// kWoScale * W_o from bf16 to fp16 (exact for |W_o| in [2^-22, 255.875])
__global__ void bf16_to_f16_kernel(const uint4 *in, uint4 *out, int64_t n_vec, int32_t *range_flag,
                                   int32_t *status) {
  griddep_wait();
  bool bad = false;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n_vec; i += (int64_t)gridDim.x * blockDim.x) {
    const uint4 u = in[i];
    float f[8];
    bf16x8_to_float(u, f);
    uint4 o;
    __half2 *h = reinterpret_cast<__half2 *>(&o);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      f[e] *= kWoScale;
      bad |= !(fabsf(f[e]) < kF16Limit);
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) h[e] = __floats2half2_rn(f[2 * e], f[2 * e + 1]);
    out[i] = o;
  }
  if (bad) flag_range(range_flag, status);
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
  b += al1k(sizeof(int32_t));                                   // fp16 range flag
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
                               const void *bias, OutT *out, float2 *stats, int32_t *range_flag, float acc_scale,
                               int32_t *status, cudaStream_t st, const char *label, int num_sms,
                               const void *cvt_in = nullptr, void *cvt_out = nullptr, int64_t cvt_n = 0) {
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
  g.cvt_scale = kWoScale;
  g.acc_scale = acc_scale;
  g.range_flag = range_flag;
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
  p += al1k((size_t)std::max(S, 1) * nt * 8);
  int32_t *range_flag = reinterpret_cast<int32_t *>(p);

  if (S == 0) return UMIM_OK;
  bool wo_in_gemm1 = false;
  if (T > 0) {
    const int blocks = std::max(1, std::min<int>((int)((T + 7) / 8), num_sms * 8));
    trace_mark(st, "merge.gather");
    if (launch_pdl(gather_rows_kernel, dim3(blocks), dim3(256), 0, st, static_cast<const uint4 *>(embeddings), vocab,
                   token_ids, T, d, reinterpret_cast<uint4 *>(E), range_flag, status) != cudaSuccess)
      return UMIM_ERR_CUDA;
    // W_o -> fp16 rides along in a side warp of GEMM1 when its share is small
    // next to the tiles its CTA computes; else a kernel of its own
    const int64_t tiles1 = (int64_t)(d / BN) * ((T + BM - 1) / BM);
    const int64_t grid1 = std::min<int64_t>(tiles1, std::max(1, num_sms));
    const int64_t n_vec = (int64_t)d * d / 8;
    wo_in_gemm1 = n_vec <= 128 * 32 * grid1 * (tiles1 / grid1);
    umim_status r = launch_gemm(enc, E, T, w->w_kv, d, false, w->b_kv, H, st1, range_flag, 1.f, status, st,
                                "merge.gemm1", num_sms, wo_in_gemm1 ? w->w_o : nullptr, wo_in_gemm1 ? Wo16 : nullptr,
                                wo_in_gemm1 ? n_vec : 0);
    if (r != UMIM_OK) return r;
  }
  trace_mark(st, "merge.pool");
  const int Ch = d / w->n_heads / 8;   // 16-byte chunks per head
  if (Ch <= 128) {
    // one warp per (span, head), double-buffered in shared memory
    const int cpl = (Ch + 31) / 32;
    auto pk = cpl == 1 ? pool_head_kernel<1> : cpl == 2 ? pool_head_kernel<2> : cpl == 3 ? pool_head_kernel<3>
                                                                                  : pool_head_kernel<4>;
    const int dh = d / w->n_heads;
    const int inner = 64 * (((dh / 64) % 4 == 0) ? 4 : ((dh / 64) % 2 == 0) ? 2 : 1);
    const int mid = dh / inner;
    HeadMaps maps;
    for (int n = 1; n <= UMIM_MAX_SPAN_TOKENS; ++n) {
      const cuuint64_t dims[3] = {(cuuint64_t)inner, (cuuint64_t)(d / inner), (cuuint64_t)T};
      const cuuint64_t strides[2] = {(cuuint64_t)inner * 2, (cuuint64_t)d * 2};
      const cuuint32_t box[3] = {(cuuint32_t)inner, (cuuint32_t)mid, (cuuint32_t)n};
      const cuuint32_t es[3] = {1, 1, 1};
      if (enc(&maps.m[n - 1], CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, H, dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return UMIM_ERR_CUDA;
    }
    const int psmem = kHeadWarps * kHeadBufs * head_buf_bytes(dh, nt);
    if (cudaFuncSetAttribute(pk, cudaFuncAttributeMaxDynamicSharedMemorySize, psmem) != cudaSuccess)
      return UMIM_ERR_CUDA;
    // warps of the grid: a multiple of h, at most one CTA per SM and no more than the items
    const int h = w->n_heads;
    const int64_t items = (int64_t)S * h;
    int grid = (int)std::min<int64_t>(std::max(1, num_sms), (items + kHeadWarps - 1) / kHeadWarps);
    while (grid > 1 && (grid * kHeadWarps) % h != 0) --grid;
    if ((grid * kHeadWarps) % h != 0) grid = h;   // 12 * h is a multiple of h
    if (launch_pdl(pk, dim3(grid), dim3(kHeadWarps * 32), psmem, st, maps, mid, (const __half *)H,
                   (const float2 *)st1, span_offsets, S, T, d, h, static_cast<const __nv_bfloat16 *>(w->ln_kv_gamma),
                   static_cast<const __nv_bfloat16 *>(w->ln_kv_beta), static_cast<const __nv_bfloat16 *>(w->query),
                   w->ln_eps, O, range_flag, status) != cudaSuccess)
      return UMIM_ERR_CUDA;
  } else {
    // wider heads: the CTA-per-span kernel with a staged ring
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
    if (launch_pdl(pk, dim3(pool_grid), dim3(kPoolConsumers + 32), psmem, st, (const __half *)H,
                   (const float2 *)st1, span_offsets, S, T, d, (int)w->n_heads,
                   static_cast<const __nv_bfloat16 *>(w->ln_kv_gamma),
                   static_cast<const __nv_bfloat16 *>(w->ln_kv_beta), static_cast<const __nv_bfloat16 *>(w->query),
                   w->ln_eps, O, range_flag, status) != cudaSuccess)
      return UMIM_ERR_CUDA;
  }
  if (!wo_in_gemm1) {
    trace_mark(st, "merge.wo_f16");
    if (launch_pdl(bf16_to_f16_kernel, dim3(std::max(1, num_sms) * 4), dim3(256), 0, st,
                   static_cast<const uint4 *>(w->w_o), reinterpret_cast<uint4 *>(Wo16), (int64_t)d * d / 8,
                   range_flag, status) != cudaSuccess)
      return UMIM_ERR_CUDA;
  }
  umim_status r = launch_gemm(enc, O, S, Wo16, d, true, w->b_o, Z16, st2, range_flag, 1.f / kWoScale, status, st,
                              "merge.gemm2", num_sms);
  if (r != UMIM_OK) return r;
  trace_mark(st, "merge.ln_o");
  if (launch_pdl(ln_rows_kernel, dim3((S + 7) / 8), dim3(256), 0, st, (const __half *)Z16, surrogates,
                 (const float2 *)st2, S, d,
                 static_cast<const __nv_bfloat16 *>(w->ln_o_gamma), static_cast<const __nv_bfloat16 *>(w->ln_o_beta),
                 w->ln_eps, (const int32_t *)range_flag) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(st, nullptr);
  return UMIM_OK;
}

}  // namespace umim
