// Merge module M_phi forward (App. C.1; Sec. 3.2 Eq. 1) for a batch of spans:
//   gather     E   = rows of the embedding table for every span token
//   GEMM1      H   = GELU(E W_kv^T + b_kv)        tcgen05, fp32 out + row stats
//   pool       P   = LN_kv(H);  a_i = softmax(P_i q_i / sqrt(d_h));  o_i = a_i^T P_i
//   GEMM2      Z   = GELU(o W_o^T + b_o)          tcgen05, fp32 out + row stats
//   LN_o       z   = LN_o(Z)                      in place in the output
//
// The two d x d projections are the only dense contractions of the module
// and run on the 5th-generation tensor cores: operands staged by TMA in
// 128-byte-swizzled shared memory, accumulator in tensor memory, one thread
// issuing tcgen05.mma, four epilogue warps reading the accumulator with
// tcgen05.ld.  A LayerNorm needs the statistics of a whole d-wide row, which
// spans d/256 output tiles, so each tile's epilogue writes the (mean, M2) of
// its 256 columns per row and the next kernel merges them (Chan et al.).
#include <algorithm>

#include "common.cuh"

namespace umim {
namespace {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int kGemmThreads = 192;   // warp 0: TMA, warp 1: MMA + TMEM owner, warps 2-5: epilogue
constexpr int kStageBytes = (BM + BN) * BK * 2;
constexpr int kGemmSmem = STAGES * kStageBytes + 1024;

struct GemmArgs {
  int M, N, K;                 // A is [M][K]
  int kb_wrap;                 // B is [N][kb_wrap]; A's column k pairs with B's column k % kb_wrap
  const __nv_bfloat16 *bias;   // [N]
  float *out;                  // [M][N]
  float2 *stats;               // [M][N / BN]
  int32_t *status;
};

__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_bias_gelu_kernel(const __grid_constant__ CUtensorMap a_map, const __grid_constant__ CUtensorMap b_map,
                          GemmArgs g) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ uint64_t full_bar[STAGES], empty_bar[STAGES], acc_bar;
  __shared__ uint32_t tmem_base;
  __shared__ float s_bias[BN];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * BN, m0 = blockIdx.y * BM;
  const int num_kb = g.K / BK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], 1);
    }
    mbar_init(&acc_bar, 1);
    fence_mbar_init();
    prefetch_tensormap(&a_map);
    prefetch_tensormap(&b_map);
  }
  if (warp == 1) {
    tmem_alloc(&tmem_base, BN);
    tmem_relinquish();
  }
  for (int i = threadIdx.x; i < BN; i += blockDim.x) s_bias[i] = __bfloat162float(g.bias[n0 + i]);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;

  if (warp == 0) {
    if (lane == 0) {
      const uint64_t pol_a = policy_evict_first();
      const uint64_t pol_b = policy_evict_last();
      for (int kb = 0; kb < num_kb; ++kb) {
        const int s = kb % STAGES;
        const uint32_t ph = (kb / STAGES) & 1;
        if (!mbar_wait(&empty_bar[s], ph ^ 1)) {
          set_error(g.status, UMIM_ERR_TIMEOUT);
          break;
        }
        uint8_t *sa = smem + s * kStageBytes;
        uint8_t *sb = sa + BM * BK * 2;
        mbar_arrive_expect_tx(&full_bar[s], kStageBytes);
        tma_load_2d(sa, &a_map, &full_bar[s], kb * BK, m0, pol_a);
        tma_load_2d(sb, &b_map, &full_bar[s], (kb * BK) % g.kb_wrap, n0, pol_b);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(BM, BN);
      for (int kb = 0; kb < num_kb; ++kb) {
        const int s = kb % STAGES;
        const uint32_t ph = (kb / STAGES) & 1;
        if (!mbar_wait(&full_bar[s], ph)) {
          set_error(g.status, UMIM_ERR_TIMEOUT);
          break;
        }
        tc_fence_after();
        const uint32_t a_base = smem_u32(smem + s * kStageBytes);
        const uint32_t b_base = a_base + BM * BK * 2;
#pragma unroll
        for (int k = 0; k < BK / 16; ++k) {
          const uint64_t ad = sw128_kmajor_desc(a_base + k * 32);
          const uint64_t bd = sw128_kmajor_desc(b_base + k * 32);
          tc_mma_bf16(tmem, ad, bd, idesc, (kb | k) != 0 ? 1u : 0u);
        }
        tc_commit(&empty_bar[s]);
      }
      tc_commit(&acc_bar);
    }
  } else {
    const int q = warp & 3;   // TMEM lane quadrant this warp may read
    const int row = m0 + q * 32 + lane;
    if (!mbar_wait(&acc_bar, 0)) {
      set_error(g.status, UMIM_ERR_TIMEOUT);
    } else {
      tc_fence_after();
      float mean = 0.f, m2 = 0.f, cnt = 0.f;
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        float v[32];
        tmem_ld_32x32b_x32(tmem + (static_cast<uint32_t>(q * 32) << 16) + c * 32, v);
        float sum = 0.f;
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          v[i] = gelu_erf(v[i] + s_bias[c * 32 + i]);
          sum += v[i];
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
        if (row < g.M) {
          float4 *dst = reinterpret_cast<float4 *>(g.out + (int64_t)row * g.N + n0 + c * 32);
#pragma unroll
          for (int i = 0; i < 8; ++i) dst[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
        }
      }
      if (row < g.M) g.stats[(int64_t)row * (g.N / BN) + blockIdx.x] = make_float2(mean, m2);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, BN);
  }
}

// ---------------------------------------------------------------------------
// gather the static embeddings of the span tokens
// ---------------------------------------------------------------------------
__global__ void gather_rows_kernel(const uint4 *table, int64_t vocab, const int32_t *ids, int64_t T, int d,
                                   uint4 *out, int32_t *status) {
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

// merge the per-tile (mean, M2) of one row into mean and 1/sqrt(var + eps)
__device__ __forceinline__ float2 row_moments(const float2 *st, int ntiles, int d, float eps) {
  float mean = 0.f, m2 = 0.f, cnt = 0.f;
  for (int t = 0; t < ntiles; ++t) {
    const float2 v = st[t];
    const float nt = cnt + (float)BN;
    const float delta = v.x - mean;
    mean += delta * ((float)BN / nt);
    m2 += v.y + delta * delta * (cnt * (float)BN / nt);
    cnt = nt;
  }
  const float var = m2 / (float)d;
  return make_float2(mean, rsqrtf(var + eps));
}

// ---------------------------------------------------------------------------
// LN_kv + attention pooling with the learnable queries, one block per span.
// o is written as two bf16 halves, O[s][0:d] = bf16(o) and
// O[s][d:2d] = bf16(o - bf16(o)), so that the output projection, run over
// K = 2d against [W_o | W_o], sees o to about 16 significant bits.
// ---------------------------------------------------------------------------
constexpr int kPoolThreads = 256;

__global__ void __launch_bounds__(kPoolThreads)
    pool_kernel(const float *H, const float2 *stats, const int32_t *offs, int S, int64_t T, int d, int h,
                const __nv_bfloat16 *gamma, const __nv_bfloat16 *beta, const __nv_bfloat16 *query, float eps,
                __nv_bfloat16 *O, int32_t *status) {
  const int s = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int ntiles = d / BN;
  const int cpt = d / kPoolThreads;                // columns per thread, contiguous
  const int c0 = tid * cpt;
  const int dh = d / h;
  const int head = c0 / dh;
  const int tph = kPoolThreads / h;                // threads per head
  __shared__ float2 s_mom[UMIM_MAX_SPAN_TOKENS];
  __shared__ float s_part[UMIM_MAX_SPAN_TOKENS][kPoolThreads / 32];
  __shared__ float s_alpha[UMIM_MAX_SPAN_TOKENS][64];

  const int t0 = offs[s], t1 = offs[s + 1];
  int n = t1 - t0;
  if (t0 < 0 || n < 1 || n > UMIM_MAX_SPAN_TOKENS || t1 > T) {
    if (tid == 0) set_error(status, UMIM_ERR_INVALID_ARG);
    n = 0;
  }
  if (warp < n) {
    const float2 m = row_moments(stats + (int64_t)(t0 + warp) * ntiles, ntiles, d, eps);
    if (lane == 0) s_mom[warp] = m;
  }
  __syncthreads();

  // scores s_j = <P_j[head], q_head> / sqrt(d_h), reduced over the head's threads
  float part[UMIM_MAX_SPAN_TOKENS] = {0.f, 0.f, 0.f, 0.f};
  for (int j = 0; j < n; ++j) {
    const float *hr = H + (int64_t)(t0 + j) * d + c0;
    const float2 mom = s_mom[j];
    float acc = 0.f;
    for (int e = 0; e < cpt; ++e) {
      const int c = c0 + e;
      const float p = (hr[e] - mom.x) * mom.y * __bfloat162float(gamma[c]) + __bfloat162float(beta[c]);
      acc += p * __bfloat162float(query[(int64_t)head * dh + (c - head * dh)]);
    }
    part[j] = acc;
  }
#pragma unroll
  for (int j = 0; j < UMIM_MAX_SPAN_TOKENS; ++j) {
    float v = part[j];
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == 0) s_part[j][warp] = v;
  }
  __syncthreads();
  // softmax over the span for each head (thread `head` of warp 0 handles it)
  if (tid < h && n > 0) {
    const int wph = tph / 32 > 0 ? tph / 32 : 1;    // warps per head
    float sc[UMIM_MAX_SPAN_TOKENS];
    float mx = -INFINITY;
    const float inv = rsqrtf((float)dh);
    for (int j = 0; j < n; ++j) {
      float v = 0.f;
      for (int w = 0; w < wph; ++w) v += s_part[j][tid * wph + w];
      sc[j] = v * inv;
      mx = fmaxf(mx, sc[j]);
    }
    float den = 0.f;
    for (int j = 0; j < n; ++j) {
      sc[j] = expf(sc[j] - mx);
      den += sc[j];
    }
    for (int j = 0; j < n; ++j) s_alpha[j][tid] = sc[j] / den;
  }
  __syncthreads();
  // o = sum_j alpha_j P_j  (bf16, the A operand of the output projection)
  for (int e = 0; e < cpt; e += 2) {
    float o0 = 0.f, o1 = 0.f;
    const int c = c0 + e;
    const float g0 = __bfloat162float(gamma[c]), g1 = __bfloat162float(gamma[c + 1]);
    const float b0 = __bfloat162float(beta[c]), b1 = __bfloat162float(beta[c + 1]);
    for (int j = 0; j < n; ++j) {
      const float2 mom = s_mom[j];
      const float a = s_alpha[j][head];
      const float *hr = H + (int64_t)(t0 + j) * d + c;
      o0 += a * ((hr[0] - mom.x) * mom.y * g0 + b0);
      o1 += a * ((hr[1] - mom.x) * mom.y * g1 + b1);
    }
    const __nv_bfloat162 hi = __floats2bfloat162_rn(o0, o1);
    const __nv_bfloat162 lo = __floats2bfloat162_rn(o0 - __low2float(hi), o1 - __high2float(hi));
    *reinterpret_cast<__nv_bfloat162 *>(O + (int64_t)s * 2 * d + c) = hi;
    *reinterpret_cast<__nv_bfloat162 *>(O + (int64_t)s * 2 * d + d + c) = lo;
  }
}

// ---------------------------------------------------------------------------
// LN_o in place over rows of Z
// ---------------------------------------------------------------------------
__global__ void ln_rows_kernel(float *Z, const float2 *stats, int d, const __nv_bfloat16 *gamma,
                               const __nv_bfloat16 *beta, float eps) {
  const int r = blockIdx.x;
  __shared__ float2 s_m;
  if (threadIdx.x == 0) s_m = row_moments(stats + (int64_t)r * (d / BN), d / BN, d, eps);
  __syncthreads();
  const float2 m = s_m;
  float *row = Z + (int64_t)r * d;
  for (int c = threadIdx.x; c < d; c += blockDim.x)
    row[c] = (row[c] - m.x) * m.y * __bfloat162float(gamma[c]) + __bfloat162float(beta[c]);
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
  b += al1k((size_t)std::max<int64_t>(T, 1) * d * 2);          // E (bf16)
  b += al1k((size_t)std::max<int64_t>(T, 1) * d * 4);          // H (fp32)
  b += al1k((size_t)std::max<int64_t>(T, 1) * nt * 8);         // stats of H
  b += al1k((size_t)std::max(S, 1) * d * 4);                   // o as bf16 hi | lo
  b += al1k((size_t)std::max(S, 1) * nt * 8);                  // stats of Z
  return b;
}

static bool encode_kmajor(EncodeTiledFn enc, CUtensorMap *map, const void *base, int64_t rows, int K,
                          int box_rows) {
  const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)K * 2};
  const cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
  const cuuint32_t es[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// out[M][d] = GELU(A[M][Ka] B[d][d]^T-with-wrap + bias), Ka = d or 2d
static umim_status launch_gemm(EncodeTiledFn enc, const void *A, int64_t M, int Ka, const void *Bw, int d,
                               const void *bias, float *out, float2 *stats, int32_t *status, cudaStream_t st,
                               const char *label) {
  CUtensorMap am, bm;
  if (!encode_kmajor(enc, &am, A, M, Ka, BM) || !encode_kmajor(enc, &bm, Bw, d, d, BN)) return UMIM_ERR_CUDA;
  GemmArgs g;
  g.M = (int)M;
  g.N = d;
  g.K = Ka;
  g.kb_wrap = d;
  g.bias = static_cast<const __nv_bfloat16 *>(bias);
  g.out = out;
  g.stats = stats;
  g.status = status;
  static bool attr_done = false;
  if (!attr_done) {
    if (cudaFuncSetAttribute(gemm_bias_gelu_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kGemmSmem) !=
        cudaSuccess)
      return UMIM_ERR_CUDA;
    attr_done = true;
  }
  dim3 grid(d / BN, (unsigned)((M + BM - 1) / BM));
  trace_mark(st, label);
  gemm_bias_gelu_kernel<<<grid, kGemmThreads, kGemmSmem, st>>>(am, bm, g);
  return cudaGetLastError() == cudaSuccess ? UMIM_OK : UMIM_ERR_CUDA;
}

umim_status merge_spans(const void *embeddings, int64_t vocab, const int32_t *token_ids, int64_t T,
                        const int32_t *span_offsets, int S, const umim_merge_weights *w, float *surrogates,
                        void *workspace, int32_t *status, cudaStream_t st, int num_sms) {
  EncodeTiledFn enc = get_encode_tiled();
  if (!enc) return UMIM_ERR_CUDA;
  const int d = w->d_model, nt = d / BN;
  char *p = static_cast<char *>(workspace);
  __nv_bfloat16 *E = reinterpret_cast<__nv_bfloat16 *>(p);
  p += al1k((size_t)std::max<int64_t>(T, 1) * d * 2);
  float *H = reinterpret_cast<float *>(p);
  p += al1k((size_t)std::max<int64_t>(T, 1) * d * 4);
  float2 *st1 = reinterpret_cast<float2 *>(p);
  p += al1k((size_t)std::max<int64_t>(T, 1) * nt * 8);
  __nv_bfloat16 *O = reinterpret_cast<__nv_bfloat16 *>(p);
  p += al1k((size_t)std::max(S, 1) * d * 4);
  float2 *st2 = reinterpret_cast<float2 *>(p);

  if (S == 0) return UMIM_OK;
  if (T > 0) {
    const int blocks = std::max(1, std::min<int>((int)((T + 7) / 8), num_sms * 8));
    trace_mark(st, "merge.gather");
    gather_rows_kernel<<<blocks, 256, 0, st>>>(static_cast<const uint4 *>(embeddings), vocab, token_ids, T, d,
                                               reinterpret_cast<uint4 *>(E), status);
    umim_status r = launch_gemm(enc, E, T, d, w->w_kv, d, w->b_kv, H, st1, status, st, "merge.gemm1");
    if (r != UMIM_OK) return r;
  }
  trace_mark(st, "merge.pool");
  pool_kernel<<<S, kPoolThreads, 0, st>>>(H, st1, span_offsets, S, T, d, w->n_heads,
                                          static_cast<const __nv_bfloat16 *>(w->ln_kv_gamma),
                                          static_cast<const __nv_bfloat16 *>(w->ln_kv_beta),
                                          static_cast<const __nv_bfloat16 *>(w->query), w->ln_eps, O, status);
  umim_status r = launch_gemm(enc, O, S, 2 * d, w->w_o, d, w->b_o, surrogates, st2, status, st, "merge.gemm2");
  if (r != UMIM_OK) return r;
  trace_mark(st, "merge.ln_o");
  ln_rows_kernel<<<S, 256, 0, st>>>(surrogates, st2, d, static_cast<const __nv_bfloat16 *>(w->ln_o_gamma),
                                    static_cast<const __nv_bfloat16 *>(w->ln_o_beta), w->ln_eps);
  trace_mark(st, nullptr);
  return cudaGetLastError() == cudaSuccess ? UMIM_OK : UMIM_ERR_CUDA;
}

}  // namespace umim
