// Causal grouped-query prefill attention over packed compressed prompts (App.
// E "Prompt Merging", App. C.5: the compressed embeddings, with contiguous
// positions, go through the frozen backbone's prefill, whose self-attention
// then runs over the shorter sequences).  Sequence b owns rows
// cu_seqlens[b] .. cu_seqlens[b+1]-1 of q [T][Hq][D], k, v [T][Hkv][D].
//
// Work unit: 64 query rows of one sequence and one query head, one CTA of 4
// warps (16 rows each).  K and V tiles of 64 keys are staged in shared memory
// by cp.async (double-buffered; rows past the sequence are zero-filled) in
// the 128-byte-swizzled layout the decode kernel uses; S = Q K^T and O += P V
// run as mma.sync m16n8k16 (P split into a bf16 high part and a bf16
// remainder, as in decode); the softmax is online in fp32 with the causal
// mask applied on the diagonal tile.  A plan kernel turns cu_seqlens into
// per-sequence query-tile offsets (and validates them); tiles run heaviest
// (last in their sequence) first.
#include "common.cuh"
#include "mma.cuh"

namespace umim {
namespace {

constexpr int kPfWarps = 4;
constexpr int kPfRows = 16 * kPfWarps;   // query rows per CTA
constexpr int kPfKeys = 64;              // keys per K / V tile
constexpr int kPfPlanThreads = 1024;

struct PfArgs {
  const __nv_bfloat16 *q, *k, *v;   // [T][H][D]
  __nv_bfloat16 *out;               // [T][Hq][D]
  const int32_t *cu;                // [B + 1]
  int32_t *cu_tiles;                // [B + 1] workspace: query-tile offsets
  int32_t B, T, Hq, Hkv, G;
  float scale_log2;
  int32_t *status;
};

__global__ void __launch_bounds__(kPfPlanThreads) prefill_plan_kernel(PfArgs a) {
  griddep_wait();
  __shared__ int s_wsum[kPfPlanThreads / 32];
  __shared__ int s_err;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  if (tid == 0) s_err = (a.cu[0] != 0 || a.cu[a.B] > a.T) ? 1 : 0;
  __syncthreads();
  int carry = 0;
  for (int base = 0; base < a.B; base += kPfPlanThreads) {
    const int b = base + tid;
    int n = 0;
    if (b < a.B) {
      const int len = a.cu[b + 1] - a.cu[b];
      if (len < 0) s_err = 1;
      n = len > 0 ? (len + kPfRows - 1) / kPfRows : 0;
    }
    int incl = n;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane == 31) s_wsum[wid] = incl;
    __syncthreads();
    int before = 0, total = 0;
    for (int w = 0; w < kPfPlanThreads / 32; ++w) {
      if (w < wid) before += s_wsum[w];
      total += s_wsum[w];
    }
    if (b < a.B) a.cu_tiles[b] = carry + before + incl - n;
    carry += total;
    __syncthreads();
  }
  if (tid == 0) {
    if (s_err) set_error(a.status, UMIM_ERR_INVALID_ARG);
    a.cu_tiles[a.B] = s_err ? 0 : carry;   // invalid offsets: no work at all
  }
}

// byte offset of 16-byte chunk c16 of key row r in a [64 rows][D] tile stored
// as D / 64 boxes of [64 rows][128 B], 128-byte swizzled
__device__ __forceinline__ uint32_t pf_sw(int r, int c16) {
  return (c16 >> 3) * (kPfKeys * 128) + r * 128 + ((((c16 & 7) ^ (r & 7))) << 4);
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, bool fill) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(fill ? 16 : 0)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

template <int D>
__global__ void __launch_bounds__(kPfWarps * 32) prefill_attn_kernel(PfArgs a) {
  constexpr int KC = D / 16;              // k-chunks of Q K^T
  constexpr int NT = D / 8;               // n-tiles of the output
  constexpr int CPR = D / 8;              // 16-byte chunks per row
  constexpr int kTile = kPfKeys * D * 2;  // bytes of one K (or V) tile
  extern __shared__ __align__(1024) uint8_t pf_smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(pf_smem) + 1023) & ~uintptr_t(1023));

  griddep_wait();
  const int total = a.cu_tiles[a.B];
  if ((int)blockIdx.x >= total) return;
  const int t = total - 1 - (int)blockIdx.x;   // a sequence's last (heaviest) tiles first
  int lo = 0, hi = a.B;                        // sequence: last b with cu_tiles[b] <= t
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (a.cu_tiles[mid] <= t) lo = mid;
    else hi = mid;
  }
  const int b = lo;
  const int qt = t - a.cu_tiles[b];
  const int s0 = a.cu[b], len = a.cu[b + 1] - s0;
  const int q0 = qt * kPfRows;
  const int h = blockIdx.y, g = h / a.G;
  const int n_kv = qt + 1;   // causal: keys up to the tile's last query row

  auto load_kv = [&](int kt, int buf) {
    uint8_t *kd = base + buf * 2 * kTile;
    uint8_t *vd = kd + kTile;
    for (int c = threadIdx.x; c < kPfKeys * CPR; c += kPfWarps * 32) {
      const int r = c / CPR, c16 = c % CPR;
      const int key = kt * kPfKeys + r;
      const bool ok = key < len;
      const int64_t row = (int64_t)s0 + (ok ? key : 0);
      const int64_t off = (row * a.Hkv + g) * D + c16 * 8;
      cp_async16(smem_u32(kd + pf_sw(r, c16)), a.k + off, ok);
      cp_async16(smem_u32(vd + pf_sw(r, c16)), a.v + off, ok);
    }
    cp_async_commit();
  };
  load_kv(0, 0);

  // Q fragments of this warp's 16 rows
  const int qr = lane >> 2, qc = lane & 3;
  const int r0 = q0 + warp * 16 + qr, r1 = r0 + 8;   // rows within the sequence
  uint32_t qa[KC][4];
  {
    const __nv_bfloat16 *q0p = a.q + (((int64_t)s0 + r0) * a.Hq + h) * D;
    const __nv_bfloat16 *q1p = a.q + (((int64_t)s0 + r1) * a.Hq + h) * D;
#pragma unroll
    for (int c = 0; c < KC; ++c) {
      const int k0 = c * 16 + 2 * qc;
      qa[c][0] = r0 < len ? *reinterpret_cast<const uint32_t *>(q0p + k0) : 0u;
      qa[c][1] = r1 < len ? *reinterpret_cast<const uint32_t *>(q1p + k0) : 0u;
      qa[c][2] = r0 < len ? *reinterpret_cast<const uint32_t *>(q0p + k0 + 8) : 0u;
      qa[c][3] = r1 < len ? *reinterpret_cast<const uint32_t *>(q1p + k0 + 8) : 0u;
    }
  }
  float acc[NT][4];
#pragma unroll
  for (int j = 0; j < NT; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;

  for (int kt = 0; kt < n_kv; ++kt) {
    if (kt + 1 < n_kv) {
      load_kv(kt + 1, (kt + 1) & 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const uint32_t ks = smem_u32(base + (kt & 1) * 2 * kTile), vs = ks + kTile;

    // S = Q K^T: 16 rows x 64 keys (8 n-tiles)
    float s[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
    for (int c = 0; c < KC; ++c) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        const int key = np * 16 + (lane & 7) + ((lane >> 4) << 3);
        const int c16 = 2 * c + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(ks + pf_sw(key, c16), b0, b1, b2, b3);
        mma_bf16(s[2 * np], qa[c], b0, b1);
        mma_bf16(s[2 * np + 1], qa[c], b2, b3);
      }
    }
    // scale to log2 units; causal mask (key > row) and keys past the end
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = kt * kPfKeys + nt * 8 + 2 * qc + (e & 1);
        const int row = e < 2 ? r0 : r1;
        const bool keep = key <= row && key < len;
        s[nt][e] = keep ? s[nt][e] * a.scale_log2 : -INFINITY;
        if (e < 2) mx0 = fmaxf(mx0, s[nt][e]);
        else mx1 = fmaxf(mx1, s[nt][e]);
      }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float n0 = fmaxf(m0, mx0), n1 = fmaxf(m1, mx1);
    // rows whose keys are all masked so far keep m = -inf: use 0 as the reference
    const float e0 = n0 == -INFINITY ? 0.f : n0, e1 = n1 == -INFINITY ? 0.f : n1;
    const float c0 = exp2f(m0 - e0), c1 = exp2f(m1 - e1);
    m0 = n0;
    m1 = n1;
    float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      s[nt][0] = exp2f(s[nt][0] - e0);
      s[nt][1] = exp2f(s[nt][1] - e0);
      s[nt][2] = exp2f(s[nt][2] - e1);
      s[nt][3] = exp2f(s[nt][3] - e1);
      rs0 += s[nt][0] + s[nt][1];
      rs1 += s[nt][2] + s[nt][3];
    }
    l0 = l0 * c0 + rs0;
    l1 = l1 * c1 + rs1;
#pragma unroll
    for (int j = 0; j < NT; ++j) {
      acc[j][0] *= c0;
      acc[j][1] *= c0;
      acc[j][2] *= c1;
      acc[j][3] *= c1;
    }
    // O += P V over the tile's 4 groups of 16 keys
#pragma unroll
    for (int kc = 0; kc < 4; ++kc) {
      uint32_t ph[4], pl[4];
      const float v4[4][2] = {{s[2 * kc][0], s[2 * kc][1]}, {s[2 * kc][2], s[2 * kc][3]},
                              {s[2 * kc + 1][0], s[2 * kc + 1][1]}, {s[2 * kc + 1][2], s[2 * kc + 1][3]}};
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const __nv_bfloat162 hh = __floats2bfloat162_rn(v4[r][0], v4[r][1]);
        ph[r] = *reinterpret_cast<const uint32_t *>(&hh);
        pl[r] = pack_bf16(v4[r][0] - __low2float(hh), v4[r][1] - __high2float(hh));
      }
#pragma unroll
      for (int j = 0; j < D / 16; ++j) {
        const int key = kc * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
        const int c16 = 2 * j + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(vs + pf_sw(key, c16), b0, b1, b2, b3);
        mma_bf16(acc[2 * j], ph, b0, b1);
        mma_bf16(acc[2 * j + 1], ph, b2, b3);
        mma_bf16(acc[2 * j], pl, b0, b1);
        mma_bf16(acc[2 * j + 1], pl, b2, b3);
      }
    }
    __syncthreads();   // this buffer is refilled two tiles later
  }

  // normalise and store
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  const float i0 = l0 > 0.f ? 1.f / l0 : 0.f, i1 = l1 > 0.f ? 1.f / l1 : 0.f;
  __nv_bfloat16 *o0 = a.out + (((int64_t)s0 + r0) * a.Hq + h) * D;
  __nv_bfloat16 *o1 = a.out + (((int64_t)s0 + r1) * a.Hq + h) * D;
#pragma unroll
  for (int j = 0; j < NT; ++j) {
    const int col = j * 8 + 2 * qc;
    if (r0 < len) *reinterpret_cast<uint32_t *>(o0 + col) = pack_bf16(acc[j][0] * i0, acc[j][1] * i0);
    if (r1 < len) *reinterpret_cast<uint32_t *>(o1 + col) = pack_bf16(acc[j][2] * i1, acc[j][3] * i1);
  }
}

}  // namespace

size_t prefill_attention_workspace_bytes(int B) { return ((size_t)(B + 1) * sizeof(int32_t) + 255) & ~size_t(255); }

umim_status prefill_attention(const void *q, const void *k, const void *v, int T, int Hq, int Hkv, int D,
                              const int32_t *cu_seqlens, int B, float scale, void *out, void *ws, int32_t *status,
                              cudaStream_t stream) {
  PfArgs a{};
  a.q = static_cast<const __nv_bfloat16 *>(q);
  a.k = static_cast<const __nv_bfloat16 *>(k);
  a.v = static_cast<const __nv_bfloat16 *>(v);
  a.out = static_cast<__nv_bfloat16 *>(out);
  a.cu = cu_seqlens;
  a.cu_tiles = static_cast<int32_t *>(ws);
  a.B = B;
  a.T = T;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.G = Hq / Hkv;
  a.scale_log2 = (scale > 0.f ? scale : 1.0f / sqrtf((float)D)) * 1.4426950408889634f;
  a.status = status;
  trace_mark(stream, "prefill.plan");
  if (launch_pdl(prefill_plan_kernel, dim3(1), dim3(kPfPlanThreads), 0, stream, a) != cudaSuccess)
    return UMIM_ERR_CUDA;
  auto kern = D == 128 ? prefill_attn_kernel<128> : prefill_attn_kernel<64>;
  const size_t smem = (size_t)2 * 2 * kPfKeys * D * 2 + 1024;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return UMIM_ERR_CUDA;
  // an upper bound of the query tiles: each sequence wastes less than one
  const unsigned gx = (unsigned)((T + kPfRows - 1) / kPfRows + B);
  trace_mark(stream, "prefill.attention");
  if (launch_pdl(kern, dim3(gx, (unsigned)Hq), dim3(kPfWarps * 32), smem, stream, a) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, nullptr);
  return UMIM_OK;
}

}  // namespace umim
