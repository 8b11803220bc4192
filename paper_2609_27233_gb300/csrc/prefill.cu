// Causal grouped-query prefill attention over packed compressed prompts (App.
// E "Prompt Merging", App. C.5: the compressed embeddings, with contiguous
// positions, go through the frozen backbone's prefill, whose self-attention
// then runs over the shorter sequences).  Sequence b owns rows
// cu_seqlens[b] .. cu_seqlens[b+1]-1 of q [T][Hq][D], k, v [T][Hkv][D].
//
// On the 5th-generation tensor cores: a persistent kernel, two CTAs per SM
// (each allocates half of the tensor memory, so one CTA's products fill the
// tensor cores while the other's softmax runs), each walking work units of
// 128 query rows of one sequence for one query head, heaviest first; the
// next unit's Q and K loads and first S products overlap the current unit's
// last tiles and epilogue.  Warp 0 loads tiles with TMA (a unit's Q; 64-key K
// tiles into a 2-stage ring running a tile ahead of the V^T tiles' 2-stage
// ring), warp 1 issues the S = Q K^T products (tcgen05.mma into one of two
// tensor-memory buffers, reused once the P V product that read it is done),
// warp 6 the O += P V products into a tensor-memory accumulator (a separate
// issuing thread, so that a P V product never waits behind an S product that
// waits for the previous P V), and warps 2-5 run the online
// softmax, one thread per query row: S from tensor memory (tcgen05.ld),
// causal mask, running max, P = exp2(S - max) written back in fp16 over the
// S columns it came from (tcgen05.st; the P V product reads its A operand
// from tensor memory, so P never touches shared memory), row sums.  P V runs
// on fp16 operands (V^T is converted when it is transposed): fp16's 11-bit
// significand keeps P's and V's rounding near 3e-4 relative, where bf16 P
// would cost 1e-3 of the output's error budget; P <= 2^8 by construction and
// |v| < 65504 is checked (UMIM_ERR_UNSUPPORTED otherwise).  The running max
// is only moved when it grows by more than 2^8, so the accumulator in tensor
// memory is rescaled rarely (the result is the same: P and the row sum use
// the same stale max).
//
// V is transposed first (per sequence, padded to a multiple of 64 keys) so
// that both products read K-major operands and every TMA copy starts on a
// 16-byte boundary.  A plan kernel turns cu_seqlens into per-sequence tile
// offsets and padded key offsets (and validates them); tiles run heaviest
// (last in their sequence) first.
#include <cuda_fp16.h>

#include "common.cuh"

namespace umim {

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *,
                                   CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                   CUtensorMapFloatOOBfill);
EncodeTiledFn get_encode_tiled();

namespace {

constexpr int kPfRows = 128;             // query rows per CTA (the MMA's M)
constexpr int kPfKeys = 64;              // keys per K / V tile (the S MMA's N)
constexpr int kPfKStages = 2;            // K ring (K runs kPfKStages - 1 tiles ahead of V^T)
constexpr int kPfVStages = 2;            // V^T ring
constexpr int kPfThreads = 224;          // warp 0 TMA, warp 1 S products + tensor memory, warps 2-5 softmax
                                         // (thread = query row), warp 6 P V products
constexpr int kPfPlanThreads = 1024;
constexpr uint32_t kPfTmemCols = 256;    // S buffers at 0 and 64, O at 128: two CTAs per SM

struct PfArgs {
  __nv_bfloat16 *out;               // [T][Hq][D]
  const int32_t *cu;                // [B + 1]
  int32_t *cu_tiles;                // [B + 1] workspace: query-tile offsets
  int32_t *pcu;                     // [B + 1] workspace: key offsets padded to 64 in V^T
  const __nv_bfloat16 *v;           // [T][Hkv][D]
  __half *vt;                       // [Hkv][D][Tp] workspace, fp16
  int64_t Tp;                       // row length of V^T (a multiple of 64)
  int32_t B, T, Hq, Hkv, G;
  float scale_log2;
  int32_t *status;
};

// One block: validates cu_seqlens, writes the prefix sums of query tiles and
// of sequence lengths rounded up to 64 keys.
__global__ void __launch_bounds__(kPfPlanThreads) prefill_plan_kernel(PfArgs a) {
  griddep_wait();
  __shared__ int s_wsum[2][kPfPlanThreads / 32];
  __shared__ int s_err;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  if (tid == 0) s_err = (a.cu[0] != 0 || a.cu[a.B] > a.T) ? 1 : 0;
  __syncthreads();
  int carry_t = 0, carry_p = 0;
  for (int base = 0; base < a.B; base += kPfPlanThreads) {
    const int b = base + tid;
    int n = 0, pk = 0;
    if (b < a.B) {
      const int len = a.cu[b + 1] - a.cu[b];
      if (len < 0) s_err = 1;
      n = len > 0 ? (len + kPfRows - 1) / kPfRows : 0;
      pk = len > 0 ? (len + kPfKeys - 1) / kPfKeys * kPfKeys : 0;
    }
    int it = n, ip = pk;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, it, o), z = __shfl_up_sync(0xffffffffu, ip, o);
      if (lane >= o) {
        it += y;
        ip += z;
      }
    }
    if (lane == 31) {
      s_wsum[0][wid] = it;
      s_wsum[1][wid] = ip;
    }
    __syncthreads();
    int bt = 0, tt = 0, bp = 0, tp = 0;
    for (int w = 0; w < kPfPlanThreads / 32; ++w) {
      if (w < wid) {
        bt += s_wsum[0][w];
        bp += s_wsum[1][w];
      }
      tt += s_wsum[0][w];
      tp += s_wsum[1][w];
    }
    if (b < a.B) {
      a.cu_tiles[b] = carry_t + bt + it - n;
      a.pcu[b] = carry_p + bp + ip - pk;
    }
    carry_t += tt;
    carry_p += tp;
    __syncthreads();
  }
  if (tid == 0) {
    if (s_err) set_error(a.status, UMIM_ERR_INVALID_ARG);
    a.cu_tiles[a.B] = s_err ? 0 : carry_t;   // invalid offsets: no work at all
    a.pcu[a.B] = s_err ? 0 : carry_p;
  }
}

// last index b in [0, B) with key[b] <= x
__device__ __forceinline__ int pf_find(const int32_t *key, int B, int x) {
  int lo = 0, hi = B;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (key[mid] <= x) lo = mid;
    else hi = mid;
  }
  return lo;
}

// V^T: vt[g][d][pcu[b] + t] = v[cu[b] + t][g][d] for t < len_b, 0 up to the
// next multiple of 64.  One CTA per 64 padded keys and KV head, through a
// shared-memory tile.
template <int D>
__global__ void __launch_bounds__(256) vt_kernel(PfArgs a) {
  griddep_wait();
  __shared__ uint32_t tile[kPfKeys][D / 2 + 1];   // bf16 pairs, padded against bank conflicts
  const int k0 = blockIdx.x * kPfKeys, g = blockIdx.y;
  if (k0 >= a.pcu[a.B]) return;
  const int b = pf_find(a.pcu, a.B, k0);
  const int len = a.cu[b + 1] - a.cu[b];
  const int t0 = k0 - a.pcu[b];
  constexpr int CPR = D / 8;   // 16-byte chunks per key row
  for (int i = threadIdx.x; i < kPfKeys * CPR; i += blockDim.x) {
    const int r = i / CPR, c = i % CPR;
    uint4 u = make_uint4(0, 0, 0, 0);
    if (t0 + r < len)
      u = __ldg(reinterpret_cast<const uint4 *>(a.v + ((int64_t)(a.cu[b] + t0 + r) * a.Hkv + g) * D) + c);
    tile[r][4 * c] = u.x;
    tile[r][4 * c + 1] = u.y;
    tile[r][4 * c + 2] = u.z;
    tile[r][4 * c + 3] = u.w;
  }
  __syncthreads();
  // each thread writes 8 keys of one d row (16 bytes), converted to fp16
  bool too_big = false;
  for (int i = threadIdx.x; i < D * (kPfKeys / 8); i += blockDim.x) {
    const int d = i / (kPfKeys / 8), c = i % (kPfKeys / 8);
    uint32_t w[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t x0 = tile[8 * c + 2 * j][d >> 1], x1 = tile[8 * c + 2 * j + 1][d >> 1];
      const float f0 = __uint_as_float((d & 1) ? (x0 & 0xffff0000u) : (x0 << 16));
      const float f1 = __uint_as_float((d & 1) ? (x1 & 0xffff0000u) : (x1 << 16));
      too_big |= !(fabsf(f0) < 65504.f) || !(fabsf(f1) < 65504.f);
      const __half2 hh = __floats2half2_rn(f0, f1);
      w[j] = *reinterpret_cast<const uint32_t *>(&hh);
    }
    *reinterpret_cast<uint4 *>(a.vt + ((int64_t)g * D + d) * a.Tp + k0 + 8 * c) = make_uint4(w[0], w[1], w[2], w[3]);
  }
  if (too_big) set_error(a.status, UMIM_ERR_UNSUPPORTED);   // |v| outside fp16's range (or not finite)
}

__device__ __forceinline__ void tma_load_3d(void *dst, const CUtensorMap *map, uint64_t *bar, int c0, int c1, int c2,
                                            uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

// 32 lanes x 64 consecutive fp32 columns from tensor memory in one load
// (thread i: row lane base + i), waited for inside the same statement so no
// register is read before it has landed
__device__ __forceinline__ void tmem_ld_32x32b_x64(uint32_t taddr, float (&v)[64]) {
  uint32_t r[64];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x64.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63}, [%64];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]), "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]), "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]), "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]), "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 64; ++i) v[i] = __uint_as_float(r[i]);
}

// 32 lanes x 32 consecutive fp32 columns back into tensor memory (thread i: row lane base + i)
__device__ __forceinline__ void tmem_st_32x32b_x32(uint32_t taddr, const float (&v)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      "f"(v[0]), "f"(v[1]), "f"(v[2]), "f"(v[3]), "f"(v[4]), "f"(v[5]), "f"(v[6]), "f"(v[7]), "f"(v[8]), "f"(v[9]),
      "f"(v[10]), "f"(v[11]), "f"(v[12]), "f"(v[13]), "f"(v[14]), "f"(v[15]), "f"(v[16]), "f"(v[17]), "f"(v[18]),
      "f"(v[19]), "f"(v[20]), "f"(v[21]), "f"(v[22]), "f"(v[23]), "f"(v[24]), "f"(v[25]), "f"(v[26]), "f"(v[27]),
      "f"(v[28]), "f"(v[29]), "f"(v[30]), "f"(v[31])
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// the hardware's approximate base-2 exponential (PTX ex2.approx.ftz: relative
// error about 2^-22, -inf -> 0)
__device__ __forceinline__ float max3f(float x, float y, float z) {   // max of three, one instruction
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(x), "f"(y), "f"(z));
  return r;
}
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 p = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&p);
}

// D[tmem] (+)= A[tmem] * B[smem]^T (kind::f16): A's rows in the 128 lanes,
// two 16-bit values of consecutive K per 32-bit column
__device__ __forceinline__ void tc_mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// shared-memory layout of the attention kernel (bytes, every piece 1024-aligned)
template <int D>
struct PfSmem {
  static constexpr int kQ = kPfRows * D * 2;              // Q of one head: D/64 atoms of [128 rows][128 B]
  static constexpr int kK = kPfKeys * D * 2;              // K tile: D/64 atoms of [64 keys][128 B]
  static constexpr int kV = D * kPfKeys * 2;              // V^T tile: [D rows][128 B]
  static constexpr int kKoff = kQ;
  static constexpr int kVoff = kKoff + kPfKStages * kK;
  static constexpr int kTotal = kVoff + kPfVStages * kV;
};

template <int D>
__global__ void __launch_bounds__(kPfThreads, 2)
    prefill_tc_kernel(const __grid_constant__ CUtensorMap q_map, const __grid_constant__ CUtensorMap k_map,
                      const __grid_constant__ CUtensorMap vt_map, PfArgs a) {
  using L = PfSmem<D>;
  constexpr int DA = D / 64;   // 64-wide atoms along the head dimension
  extern __shared__ __align__(1024) uint8_t pf_raw[];
  __shared__ __align__(8) uint64_t q_full, q_empty, k_full[kPfKStages], k_empty[kPfKStages], v_full[kPfVStages],
      v_empty[kPfVStages], s_full[2], s_empty[2], p_full[2], p_empty, o_done, o_free, mma_done[2];
  __shared__ uint32_t tmem_base;
  __shared__ int s_abort;
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(pf_raw) + 1023) & ~uintptr_t(1023));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    s_abort = 0;
    mbar_init(&q_full, 1);
    mbar_init(&q_empty, 1);    // committed once a unit's S products have read Q
    for (int s = 0; s < kPfKStages; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
    }
    for (int s = 0; s < kPfVStages; ++s) {
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_empty[i], 1);   // committed once the P V product that read P from it is done
      mbar_init(&p_full[i], 4);    // P ready, by tile parity (the four softmax warps)
    }
    mbar_init(&p_empty, 1);       // a P V product has landed
    mbar_init(&o_done, 1);        // a unit's products have landed in O
    mbar_init(&o_free, 4);        // a unit's epilogue has read O (the four softmax warps)
    mbar_init(&mma_done[0], 1);
    mbar_init(&mma_done[1], 1);
    fence_mbar_init();
    prefetch_tensormap(&q_map);
    prefetch_tensormap(&k_map);
    prefetch_tensormap(&vt_map);
  }
  if (warp == 1) {
    tmem_alloc(&tmem_base, kPfTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;
  griddep_wait();

  // Work units: (query tile, query head), the tiles heaviest first (a
  // sequence's last tiles) and the heads of a tile consecutive, so CTAs that
  // run at the same time share K and V tiles in L2.  CTA c takes units c,
  // c + G, c + 2G, ...; every barrier keeps counting across units (tile
  // counters run over the CTA's units).
  const int total = a.cu_tiles[a.B];
  const int n_units = total * a.Hq;
  const int G = (int)gridDim.x;
  struct Unit {
    int s0, len, q0, h, g, n_kv, kbase;
  };
  auto unit_of = [&](int u) {
    Unit w;
    const int t = total - 1 - u / a.Hq;   // a sequence's last (heaviest) tiles first
    const int b = pf_find(a.cu_tiles, a.B, t);
    const int qt = t - a.cu_tiles[b];
    w.s0 = a.cu[b];
    w.len = a.cu[b + 1] - w.s0;
    w.q0 = qt * kPfRows;
    w.h = u % a.Hq;
    w.g = w.h / a.G;
    w.n_kv = (min(w.q0 + kPfRows, w.len) + kPfKeys - 1) / kPfKeys;   // causal key tiles
    w.kbase = a.pcu[b];
    return w;
  };
  // a warp that gave up tells the others, so that no wait is left to time out on its own
  auto aborted = [&]() { return *reinterpret_cast<volatile int *>(&s_abort) != 0; };
  auto give_up = [&]() {
    set_error(a.status, UMIM_ERR_TIMEOUT);
    *reinterpret_cast<volatile int *>(&s_abort) = 1;
  };

  if (warp == 0) {
    if (lane == 0) {
      const uint64_t pol_q = policy_evict_first(), pol_kv = policy_evict_last();
      // K runs kPfKStages - 1 tiles ahead of V^T: a K load never waits behind
      // the P V product that frees a V^T stage
      constexpr int kLead = kPfKStages - 1;
      int nk = 0, nv = 0, nq = 0;   // K and V^T tiles (ring positions) and Q tiles loaded so far
      bool ok = true;
      int k_unit = 0;
      for (int u = (int)blockIdx.x; u < n_units && ok; u += G, ++k_unit) {
        const Unit w = unit_of(u);
        // the unit's last K row and V^T column (a TMA copy past the end of
        // its tensor reads zeros, so these checks only record)
        (void)in_bounds((int64_t)w.s0 + (w.n_kv - 1) * kPfKeys, a.T, a.status, kSitePrefillKvRow);
        (void)in_bounds(w.kbase + (int64_t)(w.n_kv - 1) * kPfKeys, a.Tp, a.status, kSitePrefillKvRow);
        // Q of the previous unit has been read by its last S product
        if (k_unit > 0 && (aborted() || !mbar_wait(&q_empty, (uint32_t)(k_unit - 1) & 1u))) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&q_full, L::kQ);
#pragma unroll
        for (int d = 0; d < DA; ++d)
          tma_load_3d(smem + d * (kPfRows * 128), &q_map, &q_full, d * 64, w.h, w.s0 + w.q0, pol_q);
        ++nq;
        for (int i = 0; i < w.n_kv + kLead && ok; ++i) {
          if (i < w.n_kv) {
            const int s = nk % kPfKStages;
            if (aborted() || !mbar_wait(&k_empty[s], ((nk / kPfKStages) & 1) ^ 1)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&k_full[s], L::kK);
#pragma unroll
            for (int d = 0; d < DA; ++d)
              tma_load_3d(smem + L::kKoff + s * L::kK + d * (kPfKeys * 128), &k_map, &k_full[s], d * 64, w.g,
                          w.s0 + i * kPfKeys, pol_kv);
            ++nk;
          }
          const int j = i - kLead;
          if (j >= 0 && j < w.n_kv) {
            const int s = nv % kPfVStages;
            if (aborted() || !mbar_wait(&v_empty[s], ((nv / kPfVStages) & 1) ^ 1)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&v_full[s], L::kV);
            tma_load_3d(smem + L::kVoff + s * L::kV, &vt_map, &v_full[s], w.kbase + j * kPfKeys, 0, w.g, pol_kv);
            ++nv;
          }
        }
      }
      if (!ok) give_up();
      // copies still in flight when a consumer gave up: wait for them (bounded)
      for (int i = max(0, nk - kPfKStages); i < nk; ++i)
        mbar_wait_for(&k_full[i % kPfKStages], (i / kPfKStages) & 1, kWaitLimitNs);
      for (int i = max(0, nv - kPfVStages); i < nv; ++i)
        mbar_wait_for(&v_full[i % kPfVStages], (i / kPfVStages) & 1, kWaitLimitNs);
      if (nq > 0) mbar_wait_for(&q_full, (uint32_t)(nq - 1) & 1u, kWaitLimitNs);
    }
  } else if (warp == 1) {
    // ---- S = Q K(i)^T into S buffer (tile counter) & 1, once the P V product that read that buffer is done ----
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_f32acc(kPfRows, kPfKeys, false);
      bool ok = true;
      int nt = 0, k_unit = 0;   // tiles and units so far
      for (int u = (int)blockIdx.x; u < n_units && ok; u += G, ++k_unit) {
        const Unit w = unit_of(u);
        if (aborted() || !mbar_wait(&q_full, (uint32_t)k_unit & 1u)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t q_base = smem_u32(smem);
        for (int i = 0; i < w.n_kv; ++i, ++nt) {
          const int s = nt % kPfKStages, sb = nt & 1;
          if (aborted() || !mbar_wait(&k_full[s], (nt / kPfKStages) & 1) ||
              !mbar_wait(&s_empty[sb], ((nt >> 1) & 1) ^ 1)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t k_base = smem_u32(smem + L::kKoff + s * L::kK);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t off = (kk & 3) * 32;
            tc_mma_bf16(tmem + sb * kPfKeys, sw128_kmajor_desc(q_base + (kk >> 2) * (kPfRows * 128) + off),
                        sw128_kmajor_desc(k_base + (kk >> 2) * (kPfKeys * 128) + off), idesc_s, kk != 0 ? 1u : 0u);
          }
          tc_commit(&s_full[sb]);
          tc_commit(&k_empty[s]);
        }
        if (ok) tc_commit(&q_empty);   // the unit's S products have read Q
      }
      if (!ok) give_up();
      // every product this thread issued has finished before tensor memory is released
      tc_commit(&mma_done[0]);
      mbar_wait_for(&mma_done[0], 0, kWaitLimitNs);
    }
  } else if (warp == 6) {
    // ---- O += P V(i) (fp16 operands, P from tensor memory), as soon as P(i) is ready; frees V(i)'s
    // stage and S(i)'s buffer.  A separate issuing thread, so that a P V product never waits behind
    // an S product that waits for the previous P V.  A unit's first product overwrites O once the
    // previous unit's epilogue has read it ----
    if (lane == 0) {
      constexpr uint32_t idesc_o = idesc_f32acc(kPfRows, D, true);   // P and V^T in fp16
      bool ok = true;
      int nt = 0, k_unit = 0;
      for (int u = (int)blockIdx.x; u < n_units && ok; u += G, ++k_unit) {
        const Unit w = unit_of(u);
        if (k_unit > 0 && (aborted() || !mbar_wait(&o_free, (uint32_t)(k_unit - 1) & 1u))) {
          ok = false;
          break;
        }
        for (int i = 0; i < w.n_kv; ++i, ++nt) {
          const int s = nt % kPfVStages, sb = nt & 1;
          if (aborted() || !mbar_wait(&v_full[s], (nt / kPfVStages) & 1) ||
              !mbar_wait(&p_full[sb], (nt >> 1) & 1)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t v_base = smem_u32(smem + L::kVoff + s * L::kV);
          const uint32_t p_tmem = tmem + sb * kPfKeys;   // P(i) sits where S(i) was
#pragma unroll
          for (int kk = 0; kk < kPfKeys / 16; ++kk)
            tc_mma_ts(tmem + 128, p_tmem + kk * 8, sw128_kmajor_desc(v_base + kk * 32), idesc_o,
                      (i | kk) != 0 ? 1u : 0u);
          tc_commit(&p_empty);
          tc_commit(&s_empty[sb]);
          tc_commit(&v_empty[s]);
        }
        if (ok) tc_commit(&o_done);   // the unit's products have landed in O
      }
      if (!ok) give_up();
      tc_commit(&mma_done[1]);
      mbar_wait_for(&mma_done[1], 0, kWaitLimitNs);
    }
  } else if (warp >= 2 && warp < 6) {
    // ---- softmax and epilogue: four warps, thread = query row ----
    const int quad = warp & 3;                 // tensor-memory lanes this warp may access
    const int r = quad * 32 + lane;            // query row within the tile
    const uint32_t t_s = tmem + ((uint32_t)(quad * 32) << 16);   // this row's S buffers
    const uint32_t t_o = t_s + 128;                                // and O
    const float sl2 = a.scale_log2;
    bool ok = true;
    // every lane waits (each needs the acquire), the warp goes on only if all saw the phase:
    // the .sync.aligned tensor-memory instructions below need the whole warp
    auto wwait = [&](uint64_t *m, uint32_t parity) {
      return __all_sync(0xffffffffu, !aborted() && mbar_wait(m, parity)) != 0;
    };
    int nt = 0, k_unit = 0;
    for (int u = (int)blockIdx.x; u < n_units && ok; u += G, ++k_unit) {
      const Unit w = unit_of(u);
      const int qpos = w.q0 + r;                  // position within the sequence
      const int kmax = min(qpos, w.len - 1);      // last key this row sees
      float m_run = -INFINITY, l_run = 0.f;       // running max (log2 units, moved in steps > 8) and row sum
      for (int j = 0; j < w.n_kv; ++j, ++nt) {
        const int sb = nt & 1;
        if (!wwait(&s_full[sb], (nt >> 1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        float s[kPfKeys];
        tmem_ld_32x32b_x64(t_s + sb * kPfKeys, s);
        const int k0 = j * kPfKeys;
        if (k0 + kPfKeys - 1 > kmax) {   // the diagonal tile (or a row past the sequence)
#pragma unroll
          for (int c = 0; c < kPfKeys; ++c) s[c] = (k0 + c <= kmax) ? s[c] : -INFINITY;
        }
        float m4[4] = {s[0], s[1], s[2], s[3]};
#pragma unroll
        for (int c = 4; c < kPfKeys; c += 2) m4[(c >> 1) & 3] = max3f(m4[(c >> 1) & 3], s[c], s[c + 1]);
        const float mx = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3])) * sl2;
        // move the running max only when it grows by more than 2^8
        const bool grow = mx > m_run + 8.f;
        float alpha = 1.f;
        if (grow) {
          alpha = (m_run == -INFINITY) ? 0.f : ex2_approx(m_run - mx);
          m_run = mx;
          l_run *= alpha;
        }
        const float nm = (m_run == -INFINITY) ? 0.f : -m_run;
        // exp2(s * scale - max) and the row sum, two columns per packed instruction
        const float2 sl2x2 = make_float2(sl2, sl2), nm2 = make_float2(nm, nm);
        float2 la = make_float2(0.f, 0.f), lb = la;
#pragma unroll
        for (int c = 0; c < kPfKeys; c += 2) {
          const float2 x = __ffma2_rn(make_float2(s[c], s[c + 1]), sl2x2, nm2);
          s[c] = ex2_approx(x.x);   // masked (-inf): 0
          s[c + 1] = ex2_approx(x.y);
          if (c & 2) lb = __fadd2_rn(lb, make_float2(s[c], s[c + 1]));
          else la = __fadd2_rn(la, make_float2(s[c], s[c + 1]));
        }
        const float2 lab = __fadd2_rn(la, lb);
        l_run += lab.x + lab.y;
        // O is rescaled only once the product of tile j - 1 has landed
        if (j > 0 && __any_sync(0xffffffffu, grow)) {
          if (!wwait(&p_empty, (uint32_t)(nt - 1) & 1u)) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll 1
          for (int c = 0; c < D / 32; ++c) {
            float o[32];
            tmem_ld_32x32b_x32(t_o + c * 32, o);
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] *= alpha;
            tmem_st_32x32b_x32(t_o + c * 32, o);
          }
          tc_fence_before();
        }
        // P(j) in fp16 over S(j)'s columns (this thread has read them), for the P V product
        {
          float pk[32];
#pragma unroll
          for (int c = 0; c < 32; ++c) {
            const __half2 hh = __floats2half2_rn(s[2 * c], s[2 * c + 1]);   // P <= 2^8
            pk[c] = __uint_as_float(*reinterpret_cast<const uint32_t *>(&hh));
          }
          tmem_st_32x32b_x32(t_s + sb * kPfKeys, pk);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&p_full[sb]);
      }
      if (!ok) break;
      // epilogue: O / l once the unit's last product has landed, then O is free for the next unit
      if (!wwait(&o_done, (uint32_t)k_unit & 1u)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
      __nv_bfloat16 *orow = a.out + (((int64_t)w.s0 + qpos) * a.Hq + w.h) * D;
#pragma unroll 1
      for (int c = 0; c < D / 32; ++c) {
        float o[32];
        tmem_ld_32x32b_x32(t_o + c * 32, o);
        if (qpos < w.len && in_bounds((int64_t)w.s0 + qpos, a.T, a.status, kSitePrefillOutRow)) {
          uint4 *dst = reinterpret_cast<uint4 *>(orow + c * 32);
#pragma unroll
          for (int e = 0; e < 4; ++e)
            dst[e] = make_uint4(pack_bf16x2(o[8 * e] * inv, o[8 * e + 1] * inv),
                                pack_bf16x2(o[8 * e + 2] * inv, o[8 * e + 3] * inv),
                                pack_bf16x2(o[8 * e + 4] * inv, o[8 * e + 5] * inv),
                                pack_bf16x2(o[8 * e + 6] * inv, o[8 * e + 7] * inv));
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&o_free);
    }
    if (!ok) give_up();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kPfTmemCols);
  }
}

bool encode_3d(EncodeTiledFn enc, CUtensorMap *map, const void *base, uint64_t d0, uint64_t d1, uint64_t d2,
               uint64_t stride1, uint64_t stride2, uint32_t b0, uint32_t b1, uint32_t b2, bool fp16 = false) {
  const cuuint64_t dims[3] = {d0, d1, d2};
  const cuuint64_t strides[2] = {stride1, stride2};
  const cuuint32_t box[3] = {b0, b1, b2};
  const cuuint32_t es[3] = {1, 1, 1};
  return enc(map, fp16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3,
             const_cast<void *>(base), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// row length of V^T: room for every sequence padded to 64 keys
int64_t vt_row(int B, int T) { return ((int64_t)T + 63LL * B + 63) / 64 * 64; }

}  // namespace

size_t prefill_attention_workspace_bytes(int B, int T, int Hkv, int D) {
  const size_t plan = ((size_t)2 * (B + 1) * sizeof(int32_t) + 1023) & ~size_t(1023);
  return plan + (size_t)Hkv * D * vt_row(B, T) * 2;
}

umim_status prefill_attention(const void *q, const void *k, const void *v, int T, int Hq, int Hkv, int D,
                              const int32_t *cu_seqlens, int B, float scale, void *out, void *ws, int32_t *status,
                              cudaStream_t stream, int num_sms) {
  EncodeTiledFn enc = get_encode_tiled();
  if (!enc) return UMIM_ERR_CUDA;
  PfArgs a{};
  a.out = static_cast<__nv_bfloat16 *>(out);
  a.cu = cu_seqlens;
  a.cu_tiles = static_cast<int32_t *>(ws);
  a.pcu = a.cu_tiles + (B + 1);
  a.v = static_cast<const __nv_bfloat16 *>(v);
  a.vt = reinterpret_cast<__half *>(static_cast<char *>(ws) +
                                           (((size_t)2 * (B + 1) * sizeof(int32_t) + 1023) & ~size_t(1023)));
  a.Tp = vt_row(B, T);
  a.B = B;
  a.T = T;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.G = Hq / Hkv;
  a.scale_log2 = (scale > 0.f ? scale : 1.0f / sqrtf((float)D)) * 1.4426950408889634f;
  a.status = status;
  CUtensorMap qm, km, vm;
  if (!encode_3d(enc, &qm, q, D, Hq, T, (uint64_t)D * 2, (uint64_t)Hq * D * 2, 64, 1, kPfRows) ||
      !encode_3d(enc, &km, k, D, Hkv, T, (uint64_t)D * 2, (uint64_t)Hkv * D * 2, 64, 1, kPfKeys) ||
      !encode_3d(enc, &vm, a.vt, a.Tp, D, Hkv, (uint64_t)a.Tp * 2, (uint64_t)D * a.Tp * 2, kPfKeys, D, 1, true))
    return UMIM_ERR_CUDA;
  trace_mark(stream, "prefill.plan");
  if (launch_pdl(prefill_plan_kernel, dim3(1), dim3(kPfPlanThreads), 0, stream, a) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, "prefill.v_transpose");
  auto vk = D == 128 ? vt_kernel<128> : vt_kernel<64>;
  if (launch_pdl(vk, dim3((unsigned)(a.Tp / kPfKeys), (unsigned)Hkv), dim3(256), 0, stream, a) != cudaSuccess)
    return UMIM_ERR_CUDA;
  auto kern = D == 128 ? prefill_tc_kernel<128> : prefill_tc_kernel<64>;
  const size_t smem = (size_t)(D == 128 ? PfSmem<128>::kTotal : PfSmem<64>::kTotal) + 1024;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return UMIM_ERR_CUDA;
  // persistent: two CTAs per SM walk the (query tile, head) units; no more
  // CTAs than an upper bound of the units (each sequence wastes less than one tile)
  const int64_t units_max = ((int64_t)(T + kPfRows - 1) / kPfRows + B) * Hq;
  const unsigned gx = (unsigned)std::max<int64_t>(1, std::min<int64_t>(2LL * std::max(num_sms, 1), units_max));
  trace_mark(stream, "prefill.attention");
  if (launch_pdl(kern, dim3(gx), dim3(kPfThreads), smem, stream, qm, km, vm, a) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, nullptr);
  return UMIM_OK;
}

}  // namespace umim
