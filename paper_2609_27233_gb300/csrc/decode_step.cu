// One layer of a decode step with decoding-time merging, in one launch
// (App. E "Decoding-Time Merging and KV-Cache Update"; Fig. 2 steps (2) and
// (3); App. I.1 on the cost of many small launches per step).
//
// A decode step forwards one token per sequence through the layers in order:
// layer l's new K/V entry exists only once layer l - 1's attention output
// does.  For layer l, per sequence b with L = seq_lens[b] (the length before
// the step) and k = merge_k[b]:
//   k == 0  the forwarded token's entry goes to slot s = L;
//   k >= 1  the forwarded token completes a merge: the surrogate's entry
//           (row merge_row[b]) goes to slot s = L + 1 - k, replacing the k - 1
//           cached entries of the span and the token itself;
// and the query attends over slots [0, s) of the cache plus the entry at s.
// That equals umim_decode_append_merge followed by umim_decode_attention,
// restricted to layer l.  Block tables and lengths keep their pre-step
// values through the step's layer calls; the call with `commit` set (the
// last layer's) records the opened page, releases the page that no longer
// holds an entry and writes the new lengths, once every CTA has finished
// reading them.
//
// Attention is the balanced split-K design of attention.cu in a single
// persistent launch: every CTA derives the same plan from the lengths (a
// prefix sum over the batch in shared memory), every warp streams an equal
// contiguous range of (sequence, KV head, page) units through a private TMA
// ring, and the unit holding slot s takes the entry from the caller's buffer
// (its row is written into the staged tile and into the cache by the same
// warp).  A warp that holds a whole (sequence, KV head) segment writes the
// output itself; a segment split across warps is merged by whichever of its
// warps finishes last (a per-segment arrival counter), so no plan or combine
// kernel is needed.
#include <algorithm>

#include "common.cuh"
#include "mma.cuh"

namespace umim {
namespace {

constexpr int kStepWarps = 12;
constexpr int kStepStages = 2;
constexpr int kStepThreads = kStepWarps * 32;
constexpr int kStepMaxBatch = 4096;

// workspace: a 256-byte header, per-segment arrival counters, then two partial
// slots per warp (a warp's range meets at most two split segments: the one it
// starts in and the one it ends in)
struct StepHeader {
  int32_t done;         // CTAs finished (commit calls only); reset by the last
  int32_t pad[63];
};

inline size_t a256(size_t x) { return (x + 255) & ~size_t(255); }

struct StepWs {
  StepHeader *hdr;
  int32_t *cnt;        // [B * Hkv]
  float2 *part_ml;     // [warps][2][16]   (m in log2 units, l)
  float *part_acc;     // [warps][2][16][D]
};

inline size_t step_ws_bytes(int B, int Hkv, int D, int total_warps) {
  return a256(sizeof(StepHeader)) + a256(sizeof(int32_t) * (size_t)B * Hkv) +
         a256(sizeof(float2) * (size_t)total_warps * 2 * 16) + a256(sizeof(float) * (size_t)total_warps * 2 * 16 * D);
}

inline StepWs step_carve(void *ws, int B, int Hkv, int D, int total_warps) {
  char *p = static_cast<char *>(ws);
  StepWs w;
  w.hdr = reinterpret_cast<StepHeader *>(p);
  p += a256(sizeof(StepHeader));
  w.cnt = reinterpret_cast<int32_t *>(p);
  p += a256(sizeof(int32_t) * (size_t)B * Hkv);
  w.part_ml = reinterpret_cast<float2 *>(p);
  p += a256(sizeof(float2) * (size_t)total_warps * 2 * 16);
  w.part_acc = reinterpret_cast<float *>(p);
  (void)D;
  return w;
}

struct StepArgs {
  const __nv_bfloat16 *q;          // [B][Hq][D]
  uint16_t *pool;                  // the paged cache
  int32_t *block_table;            // [B][max_pages]
  int32_t *seq_lens;               // [B]
  const uint16_t *new_k, *new_v;   // [B] rows of Hkv * D, new_stride elements apart
  int64_t new_stride;
  const int32_t *new_pages;        // [B] or nullptr
  const int32_t *merge_k;          // [B] or nullptr
  const int32_t *merge_row;        // [B]
  int32_t n_rows;
  const uint16_t *sur_k, *sur_v;   // [n_rows][Hkv][D]
  int32_t *released;               // [B] or nullptr
  __nv_bfloat16 *out;              // [B][Hq][D]
  int32_t B, Hq, Hkv, G, max_pages, n_pages, layer, n_layers, commit;
  float scale_log2;
  int32_t *status;
};

// What this step does to sequence b (a pure function of the inputs, so every
// CTA and every warp derives the same answer).
struct SeqStep {
  int keys;      // entries the query attends to: s + 1, or the unchanged length of a rejected sequence
  int slot;      // s, or -1 when nothing is written (rejected sequence)
  int page;      // physical page of slot s
  int row;       // surrogate row (k >= 1) or -1 (the forwarded token's own entry)
  int L, k;
};

__device__ __forceinline__ SeqStep seq_step(const StepArgs &a, int b) {
  SeqStep r;
  const int L = a.seq_lens[b];
  const int k = a.merge_k ? a.merge_k[b] : 0;
  r.L = L;
  r.k = k;
  const int64_t cap = (int64_t)a.max_pages * kPageSize;
  bool ok = L >= 0 && (int64_t)L < cap && k >= 0 && k <= 16 && k <= L + 1;
  const int32_t *bt = a.block_table + (int64_t)b * a.max_pages;
  int page_L = -1;
  if (ok) {
    page_L = L % kPageSize == 0 ? (a.new_pages ? a.new_pages[b] : -1) : bt[L / kPageSize];
    ok = page_L >= 0 && page_L < a.n_pages;
  }
  int slot = L, page = page_L, row = -1;
  if (ok && k > 0) {
    row = a.merge_row ? a.merge_row[b] : -1;
    slot = L + 1 - k;
    page = slot / kPageSize == L / kPageSize ? page_L : bt[slot / kPageSize];
    ok = row >= 0 && row < a.n_rows && page >= 0 && page < a.n_pages;
  }
  if (ok) {
    r.keys = slot + 1;
    r.slot = slot;
    r.page = page;
    r.row = row;
  } else {
    r.keys = (L >= 0 && (int64_t)L <= cap) ? L : 0;
    r.slot = -1;
    r.page = -1;
    r.row = -1;
  }
  return r;
}

// swizzled byte offset of 16-byte chunk c16 of row r in a tile stored as D/64
// boxes of [16 rows][128 B] with 128-byte swizzling
__device__ __forceinline__ uint32_t sw_off(int r, int c16) {
  const int box = c16 >> 3, cc = c16 & 7;
  return box * 2048 + r * 128 + ((cc ^ (r & 7)) << 4);
}

__device__ __forceinline__ uint4 ld_nc_v4(const uint16_t *p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// ---------------------------------------------------------------------------
// the kernel
// ---------------------------------------------------------------------------
template <int D>
__global__ void __launch_bounds__(kStepThreads, 1)
    decode_step_kernel(const __grid_constant__ CUtensorMap kv_map, StepArgs a, StepWs ws) {
  constexpr int kTile = 16 * D * 2;        // bytes of one K (or V) tile
  constexpr int kStage = 2 * kTile;
  constexpr int NB = D / 64;               // 128-byte boxes per tile row
  constexpr int NT = D / 8;                // n-tiles of the output
  constexpr int KC = D / 16;               // k-chunks of Q K^T
  constexpr int CPR = D / 8;               // 16-byte chunks per row
  constexpr int E = D / 32;                // output columns per lane in the merge of split segments
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ uint64_t bars[kStepWarps][kStepStages];
  __shared__ int s_scan[kStepWarps];
  __shared__ int s_last;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gw = blockIdx.x * kStepWarps + warp;
  const int total_warps = gridDim.x * kStepWarps;
  uint8_t *base = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t *wbuf = base + warp * kStepStages * kStage;
  int *pref = reinterpret_cast<int *>(base + kStepWarps * kStepStages * kStage);   // [B + 1] units before b

  if (lane == 0) {
    for (int s = 0; s < kStepStages; ++s) mbar_init(&bars[warp][s], 1);
    fence_mbar_init();
    if (warp == 0) prefetch_tensormap(&kv_map);
  }
  __syncwarp();
  griddep_wait();

  const int B = a.B, Hkv = a.Hkv, G = a.G;
  // ---- plan: ceil(keys / 16) units for every KV head of sequence b, prefix-summed ----
  int carry = 0;
  for (int b0 = 0; b0 < B; b0 += kStepThreads) {
    const int b = b0 + threadIdx.x;
    int n = 0;
    if (b < B) {
      const SeqStep st = seq_step(a, b);
      n = ceil_div(st.keys, kPageSize);
      if (st.slot < 0 && blockIdx.x == 0) set_error(a.status, UMIM_ERR_INVALID_ARG);
      if (n == 0 && blockIdx.x == b % gridDim.x) {
        // a rejected sequence with nothing cached: zero output, like the plain attention
        __nv_bfloat16 *o = a.out + (int64_t)b * a.Hq * D;
        for (int i = 0; i < a.Hq * D; ++i) o[i] = __float2bfloat16_rn(0.f);
      }
    }
    int x = n;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) s_scan[warp] = x;
    __syncthreads();
    if (warp == 0) {
      int v = lane < kStepWarps ? s_scan[lane] : 0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += y;
      }
      if (lane < kStepWarps) s_scan[lane] = v;
    }
    __syncthreads();
    if (b < B) pref[b] = carry + x + (warp ? s_scan[warp - 1] : 0) - n;
    carry += s_scan[kStepWarps - 1];
    __syncthreads();
  }
  if (threadIdx.x == 0) pref[B] = carry;
  __syncthreads();

  const int total = Hkv * carry;
  const int W = max(1, ceil_div(total, total_warps));
  const int64_t start64 = (int64_t)gw * W;
  const int start = start64 < total ? (int)start64 : total;
  const int end = min(total, start + W);

  // (sequence, KV head, page) of a flattened unit index: the last sequence whose
  // first unit is <= pos (sequences without units share their successor's offset)
  auto locate = [&](int pos, int &b, int &g, int &pi) {
    int l = 0, h = B;
    while (h - l > 1) {
      const int m = (l + h) >> 1;
      if (Hkv * pref[m] <= pos) l = m;
      else h = m;
    }
    b = l;
    const int n = pref[b + 1] - pref[b];
    const int r = pos - Hkv * pref[b];
    g = r / n;
    pi = r - g * n;
  };

  if (start < end) {
    const uint64_t pol = policy_evict_first();
    // ---- loader cursor (lane 0 issues the copies) ----
    int lb, lg, lpi;
    locate(start, lb, lg, lpi);
    SeqStep lst = seq_step(a, lb);
    int ld_pos = start;
    auto issue = [&](int stage) {
      uint64_t *bar = &bars[warp][stage];
      uint8_t *dst = wbuf + stage * kStage;
      if (lst.slot >= 0 && lpi == lst.slot / kPageSize && lst.slot % kPageSize == 0) {
        mbar_arrive(bar);   // only the new entry in this unit: nothing to copy
      } else {
        const int page = in_bounds(lpi, a.max_pages, a.status, kSiteStepTable)
                             ? a.block_table[(int64_t)lb * a.max_pages + lpi] : -1;
        int c4 = a.layer * a.n_pages + page;
        if (page < 0 || page >= a.n_pages) {
          set_error(a.status, UMIM_ERR_INVALID_ARG);   // a coordinate past the last page reads zeros
          c4 = a.n_layers * a.n_pages;
        }
        mbar_arrive_expect_tx(bar, kStage);
#pragma unroll
        for (int c = 0; c < NB; ++c) {
          tma_load_5d(dst + c * 2048, &kv_map, bar, c * 64, 0, lg, 0, c4, pol);
          tma_load_5d(dst + kTile + c * 2048, &kv_map, bar, c * 64, 0, lg, 1, c4, pol);
        }
      }
      // advance the cursor
      ++ld_pos;
      if (ld_pos < end) {
        const int n = pref[lb + 1] - pref[lb];
        if (++lpi == n) {
          lpi = 0;
          if (++lg == Hkv) {
            lg = 0;
            do {
              ++lb;
            } while (pref[lb + 1] == pref[lb]);
            lst = seq_step(a, lb);
          }
        }
      }
    };
    if (lane == 0) {
      for (int s = 0; s < kStepStages && ld_pos < end; ++s) issue(s);
    }

    // ---- compute state ----
    int cb, cg, cpi;
    locate(start, cb, cg, cpi);
    SeqStep cst = seq_step(a, cb);
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

    // the current segment (cb, cg) is finished within this warp's range: write
    // its output, or its partial and, if this warp is the segment's last to
    // finish, the merged output
    auto flush = [&]() {
      float s0 = l0, s1 = l1;
      s0 += __shfl_xor_sync(0xffffffffu, s0, 1);
      s0 += __shfl_xor_sync(0xffffffffu, s0, 2);
      s1 += __shfl_xor_sync(0xffffffffu, s1, 1);
      s1 += __shfl_xor_sync(0xffffffffu, s1, 2);
      const int n = pref[cb + 1] - pref[cb];
      const int o = Hkv * pref[cb] + cg * n;
      __nv_bfloat16 *obase = a.out + ((int64_t)cb * a.Hq + (int64_t)cg * G) * D;
      if (o >= start && o + n <= end) {
        const float i0 = s0 > 0.f ? 1.f / s0 : 0.f, i1 = s1 > 0.f ? 1.f / s1 : 0.f;
#pragma unroll
        for (int j = 0; j < NT; ++j) {
          const int col = j * 8 + 2 * qc;
          if (qr < G)
            *reinterpret_cast<__nv_bfloat162 *>(obase + (int64_t)qr * D + col) =
                __floats2bfloat162_rn(acc[j][0] * i0, acc[j][1] * i0);
          if (qr + 8 < G)
            *reinterpret_cast<__nv_bfloat162 *>(obase + (int64_t)(qr + 8) * D + col) =
                __floats2bfloat162_rn(acc[j][2] * i1, acc[j][3] * i1);
        }
        return;
      }
      const int slot = o <= start ? 0 : 1;
      float2 *ml = ws.part_ml + ((int64_t)gw * 2 + slot) * 16;
      float *pacc = ws.part_acc + ((int64_t)gw * 2 + slot) * 16 * D;
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
      __threadfence();   // this lane's partial is visible before the arrival below
      __syncwarp();
      const int seg = cb * Hkv + cg;
      int old = 0;
      if (lane == 0) old = atomicAdd(&ws.cnt[seg], 1);
      old = __shfl_sync(0xffffffffu, old, 0);
      const int w0 = o / W, w1 = (o + n - 1) / W;
      if (old != w1 - w0) return;   // another warp of the segment is still running
      if (!in_bounds(w1, (int64_t)gridDim.x * kStepWarps, a.status, kSiteStepPartial)) return;
      // last to finish: merge the segment's partials (warp w0 used slot 1
      // unless the segment starts its range; every later warp used slot 0),
      // several pieces' loads in flight at a time
      __threadfence();
      constexpr int U = E == 4 ? 4 : 8;
      for (int r = 0; r < G; ++r) {
        float M = -INFINITY, l = 0.f, ov[E];
#pragma unroll
        for (int e = 0; e < E; ++e) ov[e] = 0.f;
        for (int w = w0; w <= w1; w += U) {
          float2 pm[U];
          float av[U][E];
#pragma unroll
          for (int u = 0; u < U; ++u) {
            pm[u] = make_float2(-INFINITY, 0.f);
#pragma unroll
            for (int e = 0; e < E; ++e) av[u][e] = 0.f;
            if (w + u <= w1) {
              const int sl = (w + u == w0 && o != w0 * W) ? 1 : 0;
              const int64_t pc = ((int64_t)(w + u) * 2 + sl) * 16 + r;
              pm[u] = __ldcg(ws.part_ml + pc);
              if constexpr (E == 4) {
                const float4 f = __ldcg(reinterpret_cast<const float4 *>(ws.part_acc + pc * D + lane * E));
                av[u][0] = f.x, av[u][1] = f.y, av[u][2] = f.z, av[u][3] = f.w;
              } else {
                const float2 f = __ldcg(reinterpret_cast<const float2 *>(ws.part_acc + pc * D + lane * E));
                av[u][0] = f.x, av[u][1] = f.y;
              }
            }
          }
          float nm = M;
#pragma unroll
          for (int u = 0; u < U; ++u) nm = fmaxf(nm, pm[u].x);
          if (nm == -INFINITY) continue;
          const float c_old = exp2f(M - nm);
          l *= c_old;
#pragma unroll
          for (int e = 0; e < E; ++e) ov[e] *= c_old;
#pragma unroll
          for (int u = 0; u < U; ++u) {
            const float c = exp2f(pm[u].x - nm);   // 0 for an absent or empty piece
            l = fmaf(pm[u].y, c, l);
#pragma unroll
            for (int e = 0; e < E; ++e) ov[e] = fmaf(av[u][e], c, ov[e]);
          }
          M = nm;
        }
        const float inv = l > 0.f ? 1.f / l : 0.f;
        if constexpr (E == 4) {
          __nv_bfloat162 lo = __floats2bfloat162_rn(ov[0] * inv, ov[1] * inv);
          __nv_bfloat162 hi = __floats2bfloat162_rn(ov[2] * inv, ov[3] * inv);
          uint2 pk;
          pk.x = *reinterpret_cast<uint32_t *>(&lo);
          pk.y = *reinterpret_cast<uint32_t *>(&hi);
          *reinterpret_cast<uint2 *>(obase + (int64_t)r * D + lane * E) = pk;
        } else {
          *reinterpret_cast<__nv_bfloat162 *>(obase + (int64_t)r * D + lane * E) =
              __floats2bfloat162_rn(ov[0] * inv, ov[1] * inv);
        }
      }
      if (lane == 0) ws.cnt[seg] = 0;   // ready for the next call
    };

    int it = 0;
    bool dead = false;
    for (int pos = start; pos < end; ++pos, ++it) {
      const int stage = it % kStepStages;
      const uint32_t parity = (it / kStepStages) & 1;
      // every lane takes the same decision, even if the limit runs out between two lanes' polls
      if (!__all_sync(0xffffffffu, mbar_wait(&bars[warp][stage], parity))) {
        set_error(a.status, UMIM_ERR_TIMEOUT);
        // let the copies still in flight land (each wait bounded) before leaving
        for (int k = 1; k < kStepStages && pos + k < ld_pos; ++k)
          mbar_wait(&bars[warp][(it + k) % kStepStages], ((it + k) / kStepStages) & 1);
        dead = true;
        break;
      }
      uint8_t *kt = wbuf + stage * kStage;
      uint8_t *vt = kt + kTile;
      const int nvalid = min(16, cst.keys - cpi * 16);
      const bool inject = cst.slot >= 0 && cpi == cst.slot / kPageSize;
      if (inject) {
        // the step's entry at slot s: into row s % 16 of the staged tiles and
        // into the cache (lanes 0..CPR-1 carry K, CPR..2*CPR-1 carry V)
        const int r = cst.slot % kPageSize;
        if (lane < 2 * CPR) {
          const int isv = lane >= CPR;
          const int c = isv ? lane - CPR : lane;
          const uint16_t *src =
              cst.row >= 0 ? (isv ? a.sur_v : a.sur_k) + ((int64_t)cst.row * Hkv + cg) * D
                           : (isv ? a.new_v : a.new_k) + (int64_t)cb * a.new_stride + (int64_t)cg * D;
          const uint4 v = ld_nc_v4(src + c * 8);
          *reinterpret_cast<uint4 *>((isv ? vt : kt) + sw_off(r, c)) = v;
          const int64_t off = ((((int64_t)a.layer * a.n_pages + cst.page) * 2 + isv) * Hkv + cg) * (16 * D) +
                              (int64_t)r * D + c * 8;
          if (in_bounds(off, (int64_t)a.n_layers * a.n_pages * 2 * Hkv * 16 * D - 7, a.status,
                        kSiteStepCacheWrite))
            *reinterpret_cast<uint4 *>(a.pool + off) = v;
        }
      }
      if (nvalid < 16) {
        // zero V rows past the end so that 0 * garbage cannot make a NaN
        for (int idx = lane; idx < (16 - nvalid) * NB * 8; idx += 32) {
          const int r = nvalid + idx / (NB * 8);
          const int c16 = idx % (NB * 8);
          *reinterpret_cast<uint4 *>(vt + sw_off(r, c16)) = make_uint4(0, 0, 0, 0);
        }
      }
      if (inject || nvalid < 16) {
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
      if (lane == 0 && ld_pos < end) issue(stage);

      // advance: the end of a segment flushes it
      if (++cpi == pref[cb + 1] - pref[cb]) {
        flush();
        cpi = 0;
        if (pos + 1 < end) {
          if (++cg == Hkv) {
            cg = 0;
            do {
              ++cb;
            } while (pref[cb + 1] == pref[cb]);
            cst = seq_step(a, cb);
          }
          load_q();
          m0 = m1 = -INFINITY;
          l0 = l1 = 0.f;
#pragma unroll
          for (int j = 0; j < NT; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
        }
      } else if (pos + 1 == end) {
        flush();   // the range ends inside this segment
      }
    }
    (void)dead;
  }

  // ---- commit (the step's last layer): once every CTA is done reading ----
  if (a.commit) {
    __syncthreads();
    if (threadIdx.x == 0) {
      __threadfence();
      s_last = atomicAdd(&ws.hdr->done, 1) == (int)gridDim.x - 1;
    }
    __syncthreads();
    if (s_last) {
      __threadfence();
      for (int b = threadIdx.x; b < B; b += kStepThreads) {
        const SeqStep st = seq_step(a, b);
        if (st.slot < 0) {
          if (a.released) a.released[b] = -1;
          continue;   // rejected: left unchanged
        }
        int32_t *bt = a.block_table + (int64_t)b * a.max_pages;
        const int L = st.L, Ln = st.slot + 1;
        if (L % kPageSize == 0) bt[L / kPageSize] = a.new_pages[b];   // the step opened this page
        const int had = ceil_div(L + 1, kPageSize), keep = ceil_div(Ln, kPageSize);
        int rel = -1;
        if (keep < had) {   // k <= 16: at most one page
          rel = bt[keep];
          bt[keep] = -1;
        }
        if (a.released) a.released[b] = rel;
        a.seq_lens[b] = Ln;
      }
      __syncthreads();
      if (threadIdx.x == 0) ws.hdr->done = 0;
    }
  }
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

int decode_step_max_batch() { return kStepMaxBatch; }

size_t decode_step_workspace_bytes(int B, int Hkv, int D, int num_sms) {
  return step_ws_bytes(B, Hkv, D, std::max(1, num_sms) * kStepWarps);
}

template <int D>
static umim_status run_step(const StepArgs &a0, const umim_paged_kv *kv, void *workspace, cudaStream_t stream,
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
  const int grid = std::max(1, num_sms);
  const StepWs ws = step_carve(workspace, a0.B, a0.Hkv, D, grid * kStepWarps);
  const size_t smem = (size_t)kStepWarps * kStepStages * 2 * 16 * D * 2 + 1024 + sizeof(int32_t) * (a0.B + 1);
  auto kern = decode_step_kernel<D>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, a0.commit ? "decode_step.commit" : "decode_step.layer");
  if (launch_pdl(kern, dim3(grid), dim3(kStepThreads), smem, stream, map, a0, ws) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, nullptr);
  return cudaGetLastError() == cudaSuccess ? UMIM_OK : UMIM_ERR_CUDA;
}

umim_status decode_layer_step(const void *q, int Hq, const umim_paged_kv *kv, int layer, int32_t *block_table,
                              int max_pages, int32_t *seq_lens, int B, const void *new_k, const void *new_v,
                              int64_t new_stride, const int32_t *new_pages, const int32_t *merge_k,
                              const int32_t *merge_row, int n_rows, const void *sur_k, const void *sur_v, int commit,
                              int32_t *released, float scale, void *out, void *workspace, int32_t *status,
                              cudaStream_t stream, int num_sms) {
  StepArgs a{};
  a.q = static_cast<const __nv_bfloat16 *>(q);
  a.pool = static_cast<uint16_t *>(kv->base);
  a.block_table = block_table;
  a.seq_lens = seq_lens;
  a.new_k = static_cast<const uint16_t *>(new_k);
  a.new_v = static_cast<const uint16_t *>(new_v);
  a.new_stride = new_stride;
  a.new_pages = new_pages;
  a.merge_k = merge_k;
  a.merge_row = merge_row;
  a.n_rows = n_rows;
  a.sur_k = static_cast<const uint16_t *>(sur_k);
  a.sur_v = static_cast<const uint16_t *>(sur_v);
  a.released = released;
  a.out = static_cast<__nv_bfloat16 *>(out);
  a.B = B;
  a.Hq = Hq;
  a.Hkv = kv->n_kv_heads;
  a.G = Hq / kv->n_kv_heads;
  a.max_pages = max_pages;
  a.n_pages = kv->n_pages;
  a.layer = layer;
  a.n_layers = kv->n_layers;
  a.commit = commit;
  a.scale_log2 = scale * 1.4426950408889634f;
  a.status = status;
  if (kv->head_dim == 128) return run_step<128>(a, kv, workspace, stream, num_sms);
  return run_step<64>(a, kv, workspace, stream, num_sms);
}

}  // namespace umim
