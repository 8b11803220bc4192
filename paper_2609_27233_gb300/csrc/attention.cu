// Grouped-query decode attention over the compacted paged bf16 cache
// (App. I.1: decode attends to the accumulated, now shorter, KV cache).
//
// Balanced split-K: the (sequence b, KV head g, page) triples of the whole
// batch are flattened, (b, g)-major, and every warp of a persistent grid
// takes an equal contiguous range of them.  A range piece that lies in one
// (b, g) segment produces one partial (running max m, sum l, unnormalised
// output acc) for the G query heads sharing KV head g; a small combine
// kernel merges the pieces of each segment with log-sum-exp weights.
//
// Per warp: a private ring of NST stages; lane 0 issues TMA tensor loads of
// whole pages (K and V tiles of 16 x D bf16, 128-byte swizzled) into the
// ring and each stage completes an mbarrier.  S = Q K^T (G <= 16 query heads
// as the M=16 side) and O += P V run as mma.sync m16n8k16 on operands read
// with ldmatrix from the swizzled tiles; softmax is online in fp32 with the
// row statistics shared across the 4 threads of an mma row by shuffles.
// Each KV byte is read once from HBM for all G query heads.
#include <algorithm>

#include "common.cuh"
#include "mma.cuh"

namespace umim {
namespace {

// 12 warps x 2 stages (168 registers a thread, 192 KB of rings) moved more bytes
// than 8 x 3, 9 x 3, 10 x 2, 7 x 4, 6 x 4 or 4 x 6; 13 or more warps spill.
constexpr int kAttnWarps = 12;
constexpr int kAttnStages = 2;
constexpr int kPlanThreadsA = 1024;

struct AttnPlan {
  int32_t W;          // pages per warp
  int32_t total;      // flattened pages
  int32_t n_seg;
  int32_t pad[61];
  // followed by seg_off[n_seg+1], seg_pages[n_seg], piece_base[n_seg+1]
};

struct AttnWs {
  AttnPlan *plan;
  int32_t *seg_off;
  int32_t *seg_pages;
  int32_t *piece_base;
  float2 *part_ml;    // [pieces][16]      (m in log2 units, l)
  float *part_acc;    // [pieces][16][D]
};

inline size_t a256(size_t x) { return (x + 255) & ~size_t(255); }

inline size_t attn_ws_bytes(int B, int Hkv, int D, int total_warps) {
  const size_t nseg = (size_t)B * Hkv;
  const size_t pieces = nseg + total_warps;
  size_t b = a256(sizeof(AttnPlan));
  b += 2 * a256(sizeof(int32_t) * (nseg + 1)) + a256(sizeof(int32_t) * nseg);
  b += a256(sizeof(float2) * pieces * 16);
  b += a256(sizeof(float) * pieces * 16 * D);
  return b;
}

inline AttnWs attn_carve(void *ws, int B, int Hkv, int D, int total_warps) {
  const size_t nseg = (size_t)B * Hkv;
  const size_t pieces = nseg + total_warps;
  char *p = static_cast<char *>(ws);
  AttnWs w;
  w.plan = reinterpret_cast<AttnPlan *>(p);
  p += a256(sizeof(AttnPlan));
  w.seg_off = reinterpret_cast<int32_t *>(p);
  p += a256(sizeof(int32_t) * (nseg + 1));
  w.seg_pages = reinterpret_cast<int32_t *>(p);
  p += a256(sizeof(int32_t) * nseg);
  w.piece_base = reinterpret_cast<int32_t *>(p);
  p += a256(sizeof(int32_t) * (nseg + 1));
  w.part_ml = reinterpret_cast<float2 *>(p);
  p += a256(sizeof(float2) * pieces * 16);
  w.part_acc = reinterpret_cast<float *>(p);
  return w;
}

// ---------------------------------------------------------------------------
// plan: segment offsets and pieces (one block)
// ---------------------------------------------------------------------------
__device__ int scan1024(int v, int &total) {
  __shared__ int ws[32];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) ws[w] = x;
  __syncthreads();
  if (w == 0) {
    int s = ws[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    ws[lane] = s;
  }
  __syncthreads();
  const int r = x + (w ? ws[w - 1] : 0);
  total = ws[31];
  __syncthreads();
  return r;
}

__global__ void __launch_bounds__(kPlanThreadsA)
    attn_plan_kernel(const int32_t *seq_lens, int B, int Hkv, int max_pages, int total_warps, AttnWs ws,
                     int32_t *status) {
  griddep_wait();
  const int nseg = B * Hkv;
  // pass 1: segment offsets (segment (b, g) has n_b pages)
  int carry = 0;
  for (int base = 0; base < nseg; base += kPlanThreadsA) {
    const int s = base + threadIdx.x;
    int n = 0;
    if (s < nseg) {
      const int b = s / Hkv;
      int L = seq_lens[b];
      if (L < 0 || (int64_t)L > (int64_t)max_pages * kPageSize) {
        if (s % Hkv == 0) set_error(status, UMIM_ERR_INVALID_ARG);
        L = 0;
      }
      n = ceil_div(L, kPageSize);
      ws.seg_pages[s] = n;
    }
    int tot;
    const int incl = scan1024(n, tot);
    if (s < nseg) ws.seg_off[s] = carry + incl - n;
    carry += tot;
  }
  const int total = carry;
  const int W = max(1, ceil_div(total, total_warps));
  // pass 2: pieces per segment
  int pcarry = 0;
  for (int base = 0; base < nseg; base += kPlanThreadsA) {
    const int s = base + threadIdx.x;
    int np = 0;
    if (s < nseg) {
      const int n = ws.seg_pages[s];
      if (n > 0) {
        const int off = ws.seg_off[s];
        np = (off + n - 1) / W - off / W + 1;
      }
    }
    int tot;
    const int incl = scan1024(np, tot);
    if (s < nseg) ws.piece_base[s] = pcarry + incl - np;
    pcarry += tot;
  }
  if (threadIdx.x == 0) {
    ws.seg_off[nseg] = total;
    ws.piece_base[nseg] = pcarry;
    ws.plan->W = W;
    ws.plan->total = total;
    ws.plan->n_seg = nseg;
  }
}

// ---------------------------------------------------------------------------
// main kernel
// ---------------------------------------------------------------------------
struct AttnArgs {
  const __nv_bfloat16 *q;
  const int32_t *block_table;
  const int32_t *seq_lens;
  int32_t B, Hq, Hkv, G, max_pages, n_pages, layer, n_layers;
  float scale_log2;
  int32_t *status;
};

// swizzled byte offset of 16-byte chunk c16 (0 .. D/8-1) of row r in a tile
// stored as D/64 boxes of [16 rows][128 B] with 128-byte swizzling
__device__ __forceinline__ uint32_t sw_off(int r, int c16) {
  const int box = c16 >> 3, cc = c16 & 7;
  return box * 2048 + r * 128 + ((cc ^ (r & 7)) << 4);
}

template <int D>
__global__ void __launch_bounds__(kAttnWarps * 32, 1)
    attn_decode_kernel(const __grid_constant__ CUtensorMap kv_map, AttnArgs a, AttnWs ws) {
  constexpr int kTile = 16 * D * 2;        // bytes of one K (or V) tile
  constexpr int kStage = 2 * kTile;
  constexpr int NB = D / 64;               // 128-byte boxes per tile row
  constexpr int NT = D / 8;                // n-tiles of the output
  constexpr int KC = D / 16;               // k-chunks of Q K^T
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ uint64_t bars[kAttnWarps][kAttnStages];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gw = blockIdx.x * kAttnWarps + warp;
  uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t *wbuf = base + warp * kAttnStages * kStage;

  if (lane == 0) {
    for (int s = 0; s < kAttnStages; ++s) mbar_init(&bars[warp][s], 1);
    fence_mbar_init();
    if (warp == 0) prefetch_tensormap(&kv_map);
  }
  __syncwarp();
  griddep_wait();

  const int W = ws.plan->W, total = ws.plan->total, nseg = ws.plan->n_seg;
  const int start = gw * W;
  const int end = min(total, start + W);
  if (start >= end) return;

  const int G = a.G;
  const uint64_t pol = policy_evict_first();

  // segment lookup: the last segment whose offset <= pos
  auto seg_of = [&](int pos) {
    int l = 0, h = nseg;
    while (l < h) {
      const int m = (l + h) >> 1;
      if (ws.seg_off[m] <= pos) l = m + 1;
      else h = m;
    }
    return l - 1;
  };

  // ---- loader cursor ----
  int ld_pos = start;
  int ld_seg = seg_of(start);
  auto issue = [&](int pos, int stage) {
    while (pos >= ws.seg_off[ld_seg + 1]) ++ld_seg;
    const int b = ld_seg / a.Hkv, g = ld_seg % a.Hkv;
    const int pi = pos - ws.seg_off[ld_seg];
    const int page = in_bounds(pi, a.max_pages, a.status, kSiteAttnTable)
                         ? a.block_table[(int64_t)b * a.max_pages + pi] : -1;
    int c4 = a.layer * a.n_pages + page;
    if (page < 0 || page >= a.n_pages) {
      // a coordinate past the tensor's last page: the copy reads zeros
      set_error(a.status, UMIM_ERR_INVALID_ARG);
      c4 = a.n_layers * a.n_pages;
    }
    uint64_t *bar = &bars[warp][stage];
    uint8_t *dst = wbuf + stage * kStage;
    mbar_arrive_expect_tx(bar, kStage);
#pragma unroll
    for (int c = 0; c < NB; ++c) {
      tma_load_5d(dst + c * 2048, &kv_map, bar, c * 64, 0, g, 0, c4, pol);
      tma_load_5d(dst + kTile + c * 2048, &kv_map, bar, c * 64, 0, g, 1, c4, pol);
    }
  };
  if (lane == 0) {
    for (int s = 0; s < kAttnStages && ld_pos < end; ++s, ++ld_pos) issue(ld_pos, s);
  }

  // ---- compute state ----
  int cseg = seg_of(start);
  int cb = cseg / a.Hkv, cg = cseg % a.Hkv;
  const int qr = lane >> 2, qc = lane & 3;      // mma fragment row / column group
  uint32_t qa[KC][4];
  auto load_q = [&]() {
    const __nv_bfloat16 *qbase = a.q + ((int64_t)cb * a.Hq + (int64_t)cg * G) * D;
#pragma unroll
    for (int c = 0; c < KC; ++c) {
      const int k0 = c * 16 + 2 * qc;
      const uint32_t *r0 = reinterpret_cast<const uint32_t *>(qbase + (int64_t)qr * D + k0);
      const uint32_t *r1 = reinterpret_cast<const uint32_t *>(qbase + (int64_t)(qr + 8) * D + k0);
      qa[c][0] = qr < G ? r0[0] : 0u;
      qa[c][1] = qr + 8 < G ? r1[0] : 0u;
      qa[c][2] = qr < G ? r0[4] : 0u;
      qa[c][3] = qr + 8 < G ? r1[4] : 0u;
    }
  };
  load_q();
  float acc[NT][4];
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
#pragma unroll
  for (int j = 0; j < NT; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;

  auto flush = [&]() {
    // complete the row sums across the 4 threads of each row
    float s0 = l0, s1 = l1;
    s0 += __shfl_xor_sync(0xffffffffu, s0, 1);
    s0 += __shfl_xor_sync(0xffffffffu, s0, 2);
    s1 += __shfl_xor_sync(0xffffffffu, s1, 1);
    s1 += __shfl_xor_sync(0xffffffffu, s1, 2);
    const int piece = ws.piece_base[cseg] + (gw - ws.seg_off[cseg] / W);
    if (!in_bounds(piece, nseg + (int64_t)gridDim.x * kAttnWarps, a.status, kSiteAttnPiece)) return;
    float2 *ml = ws.part_ml + (int64_t)piece * 16;
    float *pacc = ws.part_acc + (int64_t)piece * 16 * D;
    if (qc == 0) {
      if (qr < G) ml[qr] = make_float2(m0, s0);
      if (qr + 8 < G) ml[qr + 8] = make_float2(m1, s1);
    }
#pragma unroll
    for (int j = 0; j < NT; ++j) {
      const int col = j * 8 + 2 * qc;
      if (qr < G) *reinterpret_cast<float2 *>(pacc + qr * D + col) = make_float2(acc[j][0], acc[j][1]);
      if (qr + 8 < G) *reinterpret_cast<float2 *>(pacc + (qr + 8) * D + col) = make_float2(acc[j][2], acc[j][3]);
    }
  };

  int it = 0;
  for (int pos = start; pos < end; ++pos, ++it) {
    // next segment?
    if (pos >= ws.seg_off[cseg + 1]) {
      flush();
      while (pos >= ws.seg_off[cseg + 1]) ++cseg;
      cb = cseg / a.Hkv;
      cg = cseg % a.Hkv;
      load_q();
      m0 = m1 = -INFINITY;
      l0 = l1 = 0.f;
#pragma unroll
      for (int j = 0; j < NT; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
    }
    const int stage = it % kAttnStages;
    const uint32_t parity = (it / kAttnStages) & 1;
    if (!mbar_wait(&bars[warp][stage], parity)) {
      set_error(a.status, UMIM_ERR_TIMEOUT);
      // let the copies still in flight land (each wait bounded) before leaving
      for (int k = 1; k < kAttnStages && it + k < ld_pos - start; ++k)
        mbar_wait(&bars[warp][(it + k) % kAttnStages], ((it + k) / kAttnStages) & 1);
      return;
    }
    uint8_t *kt = wbuf + stage * kStage;
    uint8_t *vt = kt + kTile;
    const int pi = pos - ws.seg_off[cseg];
    const int L = a.seq_lens[cb];
    const int nvalid = min(16, L - pi * 16);
    if (nvalid < 16) {
      // zero V rows past the end so that 0 * garbage cannot make a NaN
      for (int idx = lane; idx < (16 - nvalid) * NB * 8; idx += 32) {
        const int r = nvalid + idx / (NB * 8);
        const int c16 = idx % (NB * 8);
        *reinterpret_cast<uint4 *>(vt + sw_off(r, c16)) = make_uint4(0, 0, 0, 0);
      }
      // order these generic-proxy writes before the next TMA write of the stage
      fence_proxy_async_smem();
      __syncwarp();
    }
    const uint32_t ks = smem_u32(kt), vs = smem_u32(vt);

    // S = Q K^T   (16 x 16 keys as two n-tiles of 8); even and odd k-chunks
    // accumulate separately to halve the dependent mma chain
    float s[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
    float s2[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
    for (int c = 0; c < KC; ++c) {
      const int key = (lane & 7) + ((lane >> 4) << 3);
      const int c16 = 2 * c + ((lane >> 3) & 1);
      uint32_t b0, b1, b2, b3;
      ldsm_x4(ks + sw_off(key, c16), b0, b1, b2, b3);
      if (c & 1) {
        mma_bf16(s2[0], qa[c], b0, b1);
        mma_bf16(s2[1], qa[c], b2, b3);
      } else {
        mma_bf16(s[0], qa[c], b0, b1);
        mma_bf16(s[1], qa[c], b2, b3);
      }
    }
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) s[nt][e] += s2[nt][e];
    // scale to log2 units and mask keys past the end
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = nt * 8 + 2 * qc + (e & 1);
        s[nt][e] = key < nvalid ? s[nt][e] * a.scale_log2 : -INFINITY;
      }
    float mx0 = fmaxf(fmaxf(s[0][0], s[0][1]), fmaxf(s[1][0], s[1][1]));
    float mx1 = fmaxf(fmaxf(s[0][2], s[0][3]), fmaxf(s[1][2], s[1][3]));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float n0 = fmaxf(m0, mx0), n1 = fmaxf(m1, mx1);
    const float c0 = exp2f(m0 - n0), c1 = exp2f(m1 - n1);
    m0 = n0;
    m1 = n1;
    float p[2][4];
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
      p[nt][0] = exp2f(s[nt][0] - n0);
      p[nt][1] = exp2f(s[nt][1] - n0);
      p[nt][2] = exp2f(s[nt][2] - n1);
      p[nt][3] = exp2f(s[nt][3] - n1);
    }
    l0 = l0 * c0 + p[0][0] + p[0][1] + p[1][0] + p[1][1];
    l1 = l1 * c1 + p[0][2] + p[0][3] + p[1][2] + p[1][3];
#pragma unroll
    for (int j = 0; j < NT; ++j) {
      acc[j][0] *= c0;
      acc[j][1] *= c0;
      acc[j][2] *= c1;
      acc[j][3] *= c1;
    }
    // P as the A operand, split into a bf16 high part and a bf16 remainder
    uint32_t ph[4], pl[4];
    {
      const float v[4][2] = {{p[0][0], p[0][1]}, {p[0][2], p[0][3]}, {p[1][0], p[1][1]}, {p[1][2], p[1][3]}};
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const __nv_bfloat162 h = __floats2bfloat162_rn(v[r][0], v[r][1]);
        ph[r] = *reinterpret_cast<const uint32_t *>(&h);
        pl[r] = pack_bf16(v[r][0] - __low2float(h), v[r][1] - __high2float(h));
      }
    }
    // O += P V
#pragma unroll
    for (int j = 0; j < D / 16; ++j) {
      const int key = (lane & 7) + (((lane >> 3) & 1) << 3);
      const int c16 = 2 * j + (lane >> 4);
      uint32_t b0, b1, b2, b3;
      ldsm_x4_t(vs + sw_off(key, c16), b0, b1, b2, b3);
      mma_bf16(acc[2 * j], ph, b0, b1);
      mma_bf16(acc[2 * j + 1], ph, b2, b3);
      mma_bf16(acc[2 * j], pl, b0, b1);
      mma_bf16(acc[2 * j + 1], pl, b2, b3);
    }
    __syncwarp();
    // refill this stage
    if (lane == 0 && ld_pos < end) {
      issue(ld_pos, stage);
      ++ld_pos;
    }
  }
  flush();
}

// ---------------------------------------------------------------------------
// combine: WPR warps per (b, query head) row, 256 threads per CTA.  The warps
// of a row split its segment's pieces, each merges its share in one pass with
// a running maximum, and (WPR > 1) the warps' (m, l, acc) are merged through
// shared memory.  WPR grows with the pieces per segment (few, long sequences
// split into many pieces).
// ---------------------------------------------------------------------------
constexpr int kCombineThreads = 256;

template <int D, int WPR>
__global__ void __launch_bounds__(kCombineThreads)
    attn_combine_kernel(AttnWs ws, int B, int Hq, int Hkv, int G, __nv_bfloat16 *out) {
  constexpr int E = D / 32;
  constexpr int RPB = kCombineThreads / 32 / WPR;   // rows per CTA
  __shared__ float s_m[kCombineThreads / 32], s_l[kCombineThreads / 32];
  __shared__ float s_acc[WPR > 1 ? kCombineThreads / 32 : 1][D];
  griddep_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row_g = blockIdx.x * RPB + warp / WPR, sub = warp % WPR;
  const bool live = row_g < B * Hq;
  const int b = live ? row_g / Hq : 0, h = live ? row_g % Hq : 0;
  const int seg = b * Hkv + h / G, row = h % G;
  const int p0 = live ? ws.piece_base[seg] : 0, p1 = live ? ws.piece_base[seg + 1] : 0;
  float M = -INFINITY, l = 0.f, o[E];
#pragma unroll
  for (int e = 0; e < E; ++e) o[e] = 0.f;
  for (int pc = p0 + sub; pc < p1; pc += WPR) {
    const float2 ml = ws.part_ml[(int64_t)pc * 16 + row];
    const float *acc = ws.part_acc + ((int64_t)pc * 16 + row) * D + lane * E;
    float av[E];
#pragma unroll
    for (int e = 0; e < E; ++e) av[e] = acc[e];
    const float nm = fmaxf(M, ml.x);
    if (nm == -INFINITY) continue;   // nothing but empty pieces so far
    const float c_old = exp2f(M - nm), c_new = exp2f(ml.x - nm);
    l = l * c_old + ml.y * c_new;
#pragma unroll
    for (int e = 0; e < E; ++e) o[e] = o[e] * c_old + av[e] * c_new;
    M = nm;
  }
  if constexpr (WPR > 1) {
    if (lane == 0) {
      s_m[warp] = M;
      s_l[warp] = l;
    }
#pragma unroll
    for (int e = 0; e < E; ++e) s_acc[warp][lane * E + e] = o[e];
    __syncthreads();
    if (sub != 0) return;
    float Mx = -INFINITY;
#pragma unroll
    for (int w = 0; w < WPR; ++w) Mx = fmaxf(Mx, s_m[warp + w]);
    l = 0.f;
#pragma unroll
    for (int e = 0; e < E; ++e) o[e] = 0.f;
    if (Mx != -INFINITY) {
#pragma unroll
      for (int w = 0; w < WPR; ++w) {
        if (s_m[warp + w] == -INFINITY) continue;
        const float c = exp2f(s_m[warp + w] - Mx);
        l += c * s_l[warp + w];
#pragma unroll
        for (int e = 0; e < E; ++e) o[e] += c * s_acc[warp + w][lane * E + e];
      }
    }
  }
  if (!live) return;
  const float inv = l > 0.f ? 1.f / l : 0.f;
  __nv_bfloat16 *dst = out + ((int64_t)b * Hq + h) * D + lane * E;
#pragma unroll
  for (int e = 0; e < E; ++e) dst[e] = __float2bfloat16_rn(o[e] * inv);
}

}  // namespace

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *,
                                   CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                   CUtensorMapFloatOOBfill);
EncodeTiledFn get_encode_tiled();

int attn_total_warps(int num_sms) { return std::max(1, num_sms) * kAttnWarps; }

size_t decode_attention_workspace_bytes(int B, int Hq, int Hkv, int D, int num_sms) {
  (void)Hq;
  return attn_ws_bytes(B, Hkv, D, attn_total_warps(num_sms));
}

template <int D>
static umim_status run_attention(const void *q, int Hq, const umim_paged_kv *kv, int layer,
                                 const int32_t *block_table, int max_pages, const int32_t *seq_lens, int B,
                                 float scale, void *out, void *workspace, int32_t *status, cudaStream_t stream,
                                 int num_sms) {
  EncodeTiledFn enc = get_encode_tiled();
  if (!enc) return UMIM_ERR_CUDA;
  CUtensorMap map;
  const cuuint64_t dims[5] = {(cuuint64_t)D, 16, (cuuint64_t)kv->n_kv_heads, 2,
                              (cuuint64_t)kv->n_layers * (cuuint64_t)kv->n_pages};
  const cuuint64_t strides[4] = {(cuuint64_t)D * 2, (cuuint64_t)16 * D * 2,
                                 (cuuint64_t)kv->n_kv_heads * 16 * D * 2,
                                 (cuuint64_t)2 * kv->n_kv_heads * 16 * D * 2};
  const cuuint32_t box[5] = {64, 16, 1, 1, 1};
  const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  if (enc(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, kv->base, dims, strides, box, estr,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return UMIM_ERR_CUDA;
  const int total_warps = attn_total_warps(num_sms);
  const int Hkv = kv->n_kv_heads;
  AttnWs ws = attn_carve(workspace, B, Hkv, D, total_warps);
  trace_mark(stream, "attention.plan");
  if (launch_pdl(attn_plan_kernel, dim3(1), dim3(kPlanThreadsA), 0, stream, seq_lens, B, Hkv, max_pages,
                 total_warps, ws, status) != cudaSuccess)
    return UMIM_ERR_CUDA;

  AttnArgs a{};
  a.q = static_cast<const __nv_bfloat16 *>(q);
  a.block_table = block_table;
  a.seq_lens = seq_lens;
  a.B = B;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.G = Hq / Hkv;
  a.max_pages = max_pages;
  a.n_pages = kv->n_pages;
  a.layer = layer;
  a.n_layers = kv->n_layers;
  a.scale_log2 = scale * 1.4426950408889634f;
  a.status = status;
  const size_t smem = (size_t)kAttnWarps * kAttnStages * 2 * 16 * D * 2 + 1024;
  auto kern = attn_decode_kernel<D>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, "attention.decode");
  if (launch_pdl(kern, dim3(total_warps / kAttnWarps), dim3(kAttnWarps * 32), smem, stream, map, a, ws) !=
      cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, "attention.combine");
  // warps per row: about half the pieces a segment has (1 + warps / segments)
  const int per_seg = 1 + total_warps / std::max(1, B * Hkv);
  const int wpr = per_seg >= 16 ? 8 : per_seg >= 8 ? 4 : per_seg >= 4 ? 2 : 1;
  const int rows_per_cta = kCombineThreads / 32 / wpr;
  auto comb = wpr == 8 ? attn_combine_kernel<D, 8>
              : wpr == 4 ? attn_combine_kernel<D, 4>
              : wpr == 2 ? attn_combine_kernel<D, 2> : attn_combine_kernel<D, 1>;
  if (launch_pdl(comb, dim3((unsigned)((B * Hq + rows_per_cta - 1) / rows_per_cta)), dim3(kCombineThreads), 0, stream,
                 ws, B, Hq, Hkv, a.G, static_cast<__nv_bfloat16 *>(out)) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, nullptr);
  return cudaGetLastError() == cudaSuccess ? UMIM_OK : UMIM_ERR_CUDA;
}

umim_status decode_attention(const void *q, int Hq, const umim_paged_kv *kv, int layer, const int32_t *block_table,
                             int max_pages, const int32_t *seq_lens, int B, float scale, void *out,
                             void *workspace, int32_t *status, cudaStream_t stream, int num_sms) {
  if (kv->head_dim == 128)
    return run_attention<128>(q, Hq, kv, layer, block_table, max_pages, seq_lens, B, scale, out, workspace,
                              status, stream, num_sms);
  return run_attention<64>(q, Hq, kv, layer, block_table, max_pages, seq_lens, B, scale, out, workspace, status,
                           stream, num_sms);
}

}  // namespace umim
