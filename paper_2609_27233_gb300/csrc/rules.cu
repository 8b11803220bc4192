// Merge-rule matching and the surrogate lookup (App. E "Rule Matching",
// "Prompt Merging", "Decoding-Time Merging and KV-Cache Update"; the lookup
// table is the precomputation App. E proposes for context-independent
// surrogates).
//
// Rule table: open addressing with linear probing over a power-of-two number
// (>= 1.5 x rules) of 16-byte slots.  A slot holds the n-gram (four token ids of 24 bits, the
// unused ones set to 0xFFFFFF, packed into three words) and the rule id, so
// one probe is one 16-byte load; an empty slot has rule id 0xFFFFFFFF.  The
// table is built with one thread per rule claiming a slot by compare-and-swap
// on its rule word; a second pass looks every rule up again, which finds a
// repeated n-gram deterministically (the copy in the later slot is not found).
//
// Prompt matching in three kernels:
//   probe    for every position, the longest n in {4, 3, 2} whose n-gram
//            starting there is a rule (all three lookups in flight at once);
//   walk     one CTA per prompt.  The left-to-right scan is sequential, but a
//            jump is at most 4 tokens, so a segment of 8 positions maps the
//            offset (0..3) at which the scan enters it to the offset at which
//            it enters the next one.  Each thread builds that map for its
//            segment; an exclusive scan of map compositions across the CTA
//            gives every segment its actual entry; each thread then re-walks
//            its segment and writes its spans at offsets from a prefix sum.
//            The last CTA turns per-prompt counts into the span CSR offsets;
//   compact  one CTA per prompt copies its spans into the CSR arrays and, if
//            asked, writes the span tokens as the merge module's input.
// Suffix matching (decoding): one thread per sequence tests the raw suffix
// ending at the new token, longest first, and updates the sequence's state;
// merging sequences get consecutive rows in sequence order.
#include <algorithm>

#include "common.cuh"

namespace umim {
namespace {

constexpr uint32_t kEmpty = 0xFFFFFFFFu;
constexpr uint32_t kPadTok = 0xFFFFFFu;   // unused token position of a slot; also the first invalid id

struct Key {
  uint32_t w0, w1, w2;
};

__host__ __device__ __forceinline__ Key pack_key(uint32_t t0, uint32_t t1, uint32_t t2, uint32_t t3) {
  Key k;
  k.w0 = t0 | ((t3 & 0xFFu) << 24);
  k.w1 = t1 | (((t3 >> 8) & 0xFFu) << 24);
  k.w2 = t2 | (((t3 >> 16) & 0xFFu) << 24);
  return k;
}

// the n-gram c[4 - n .. 3] of a 4-token window (n = 2..4), padded
__device__ __forceinline__ Key tail_key(const uint32_t (&c)[4], int n) {
  if (n == 4) return pack_key(c[0], c[1], c[2], c[3]);
  if (n == 3) return pack_key(c[1], c[2], c[3], kPadTok);
  return pack_key(c[2], c[3], kPadTok, kPadTok);
}

// the n-gram c[0 .. n - 1] of a 4-token window, padded
__device__ __forceinline__ Key head_key(const uint32_t (&c)[4], int n) {
  if (n == 4) return pack_key(c[0], c[1], c[2], c[3]);
  if (n == 3) return pack_key(c[0], c[1], c[2], kPadTok);
  return pack_key(c[0], c[1], kPadTok, kPadTok);
}

// 64-bit mix of the key; the finaliser is MurmurHash3's fmix64
__device__ __forceinline__ uint32_t key_hash(Key k) {
  uint64_t x = ((uint64_t)k.w0 << 32) | k.w1;
  x ^= (uint64_t)k.w2 * 0x9E3779B97F4A7C15ull;
  x ^= x >> 33;
  x *= 0xFF51AFD7ED558CCDull;
  x ^= x >> 33;
  x *= 0xC4CEB9FE1A85EC53ull;
  x ^= x >> 33;
  return (uint32_t)x;
}

__device__ __forceinline__ uint4 ld_slot(const uint4 *p) {
  uint4 v;
  asm volatile("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

// Continue probing after slot i held s: rule id of k, or -1.
__device__ __forceinline__ int32_t probe_from(const uint4 *slots, uint32_t mask, Key k, uint32_t i, uint4 s) {
  for (uint32_t n = 0; n <= mask; ++n) {
    if (s.w == kEmpty) return -1;
    if (s.x == k.w0 && s.y == k.w1 && s.z == k.w2) return (int32_t)s.w;
    i = (i + 1) & mask;
    s = ld_slot(slots + i);
  }
  return -1;
}

// Longest of three candidate n-grams (4, 3, 2) that is a rule; the three
// first probes are issued together.  ok[n] says whether the n-gram exists.
template <typename KeyOf>
__device__ __forceinline__ void longest_rule(const uint4 *slots, uint32_t mask, const bool (&ok)[5], KeyOf key_of,
                                             int &best_n, int32_t &best_rule) {
  Key k4 = key_of(4), k3 = key_of(3), k2 = key_of(2);
  const uint32_t i4 = key_hash(k4) & mask, i3 = key_hash(k3) & mask, i2 = key_hash(k2) & mask;
  uint4 s4 = make_uint4(0, 0, 0, kEmpty), s3 = s4, s2 = s4;
  if (ok[4]) s4 = ld_slot(slots + i4);
  if (ok[3]) s3 = ld_slot(slots + i3);
  if (ok[2]) s2 = ld_slot(slots + i2);
  best_n = 0;
  best_rule = -1;
  int32_t r;
  if (ok[4] && (r = probe_from(slots, mask, k4, i4, s4)) >= 0) {
    best_n = 4;
    best_rule = r;
  } else if (ok[3] && (r = probe_from(slots, mask, k3, i3, s3)) >= 0) {
    best_n = 3;
    best_rule = r;
  } else if (ok[2] && (r = probe_from(slots, mask, k2, i2, s2)) >= 0) {
    best_n = 2;
    best_rule = r;
  }
}

// ---------------------------------------------------------------------------
// table build
// ---------------------------------------------------------------------------
// A rule row [4] int32: n >= 2 leading token ids in [0, 0xFFFFFF), then -1s.
__device__ __forceinline__ bool parse_rule(int4 t, Key &k) {
  const int32_t v[4] = {t.x, t.y, t.z, t.w};
  int n = 0;
  while (n < 4 && v[n] >= 0) ++n;
  if (n < 2) return false;
  for (int i = 0; i < 4; ++i) {
    if (i < n && (uint32_t)v[i] >= kPadTok) return false;
    if (i >= n && v[i] != -1) return false;
  }
  k = pack_key((uint32_t)v[0], (uint32_t)v[1], n > 2 ? (uint32_t)v[2] : kPadTok, n > 3 ? (uint32_t)v[3] : kPadTok);
  return true;
}

__global__ void rules_insert_kernel(uint4 *slots, uint32_t mask, const int4 *rules, int64_t n_rules, int32_t *status) {
  griddep_wait();
  for (int64_t r = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; r < n_rules; r += (int64_t)gridDim.x * blockDim.x) {
    Key k;
    if (!parse_rule(rules[r], k)) {
      set_error(status, UMIM_ERR_INVALID_ARG);
      continue;
    }
    uint32_t i = key_hash(k) & mask;
    bool placed = false;
    for (uint32_t n = 0; n <= mask; ++n) {
      uint32_t *w = reinterpret_cast<uint32_t *>(slots + i);
      if (atomicCAS(w + 3, kEmpty, (uint32_t)r) == kEmpty) {
        w[0] = k.w0;
        w[1] = k.w1;
        w[2] = k.w2;
        placed = true;
        break;
      }
      i = (i + 1) & mask;
    }
    if (!placed) set_error(status, UMIM_ERR_WORKSPACE);
  }
}

__global__ void rules_verify_kernel(const uint4 *slots, uint32_t mask, const int4 *rules, int64_t n_rules,
                                    int32_t *status) {
  griddep_wait();
  for (int64_t r = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; r < n_rules; r += (int64_t)gridDim.x * blockDim.x) {
    Key k;
    if (!parse_rule(rules[r], k)) continue;   // reported by the insert pass
    const uint32_t i = key_hash(k) & mask;
    if (probe_from(slots, mask, k, i, ld_slot(slots + i)) != (int32_t)r) set_error(status, UMIM_ERR_INVALID_ARG);
  }
}

// ---------------------------------------------------------------------------
// prompt matching
// ---------------------------------------------------------------------------
constexpr int kWalkThreads = 256;
constexpr int kSeg = 8;                          // positions per thread and pass
constexpr int kPass = kWalkThreads * kSeg;       // positions per pass
constexpr uint32_t kIdentity = 0xE4u;            // entry e -> e, 2 bits per entry

struct MatchHdr {
  int32_t done;   // walk CTAs finished
  int32_t pad[63];
};

struct MatchWs {
  MatchHdr *hdr;
  int8_t *mlen;       // [B][L] longest rule starting at each position (0: none)
  int32_t *mrule;     // [B][L]
  int32_t *sp_start;  // [B][stride] spans of each prompt, in order
  int32_t *sp_len;
  int32_t *sp_rule;
  int32_t *count;     // [B] spans per prompt
  int32_t *ntok;      // [B] span tokens per prompt
  int32_t *tok_base;  // [B + 1] prefix of ntok
};

inline size_t a256(size_t x) { return (x + 255) & ~size_t(255); }

__host__ __device__ inline int64_t span_stride(int L) { return L / 2 > 0 ? L / 2 : 1; }

inline size_t match_ws_bytes(int B, int L) {
  const size_t BL = (size_t)B * L > 0 ? (size_t)B * L : 1;
  const size_t bs = (size_t)(B > 0 ? B : 1) * span_stride(L);
  return a256(sizeof(MatchHdr)) + a256(BL) + a256(4 * BL) + 3 * a256(4 * bs) + 2 * a256(4 * (size_t)(B > 0 ? B : 1)) +
         a256(4 * ((size_t)B + 1));
}

inline MatchWs match_carve(void *ws, int B, int L) {
  const size_t BL = (size_t)B * L > 0 ? (size_t)B * L : 1;
  const size_t bs = (size_t)(B > 0 ? B : 1) * span_stride(L);
  char *p = static_cast<char *>(ws);
  auto take = [&](size_t n) {
    char *r = p;
    p += a256(n);
    return r;
  };
  MatchWs w;
  w.hdr = reinterpret_cast<MatchHdr *>(take(sizeof(MatchHdr)));
  w.mlen = reinterpret_cast<int8_t *>(take(BL));
  w.mrule = reinterpret_cast<int32_t *>(take(4 * BL));
  w.sp_start = reinterpret_cast<int32_t *>(take(4 * bs));
  w.sp_len = reinterpret_cast<int32_t *>(take(4 * bs));
  w.sp_rule = reinterpret_cast<int32_t *>(take(4 * bs));
  w.count = reinterpret_cast<int32_t *>(take(4 * (size_t)(B > 0 ? B : 1)));
  w.ntok = reinterpret_cast<int32_t *>(take(4 * (size_t)(B > 0 ? B : 1)));
  w.tok_base = reinterpret_cast<int32_t *>(take(4 * ((size_t)B + 1)));
  return w;
}

struct MatchArgs {
  const uint4 *slots;
  uint32_t mask;
  const int32_t *tokens;   // [B][L]
  int32_t B, L;
  const int32_t *lens;     // [B] or nullptr
  int32_t *span_offsets, *span_start, *span_len, *span_rule;
  int32_t *merge_tokens, *merge_offsets;   // or nullptr
  int32_t *status;
};

__device__ __forceinline__ int prompt_len(const MatchArgs &a, int b) {
  int Lb = a.lens ? a.lens[b] : a.L;
  if (Lb < 0 || Lb > a.L) {
    Lb = Lb < 0 ? 0 : a.L;
    set_error(a.status, UMIM_ERR_INVALID_ARG);
  }
  return Lb;
}

__global__ void __launch_bounds__(256) rule_probe_kernel(MatchArgs a, MatchWs w) {
  griddep_wait();
  const int64_t total = (int64_t)a.B * a.L;
  for (int64_t g = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; g < total; g += (int64_t)gridDim.x * blockDim.x) {
    const int b = (int)(g / a.L), p = (int)(g % a.L);
    const int Lb = a.lens ? min(max(a.lens[b], 0), a.L) : a.L;
    int n_best = 0;
    int32_t rule = -1;
    if (p < Lb) {
      uint32_t c[4];
      int valid = 0;   // leading tokens of the window that exist and are valid ids
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        c[i] = kPadTok;
        if (p + i < Lb && valid == i) {
          const int32_t t = a.tokens[g + i];
          if (t >= 0 && (uint32_t)t < kPadTok) {
            c[i] = (uint32_t)t;
            ++valid;
          } else if (i == 0) {
            set_error(a.status, UMIM_ERR_INVALID_ARG);
          }
        }
      }
      const bool ok[5] = {false, false, valid >= 2, valid >= 3, valid >= 4};
      longest_rule(a.slots, a.mask, ok, [=](int n) { return head_key(c, n); }, n_best, rule);
    }
    w.mlen[g] = (int8_t)n_best;
    w.mrule[g] = rule;
  }
}

__device__ __forceinline__ uint32_t compose(uint32_t later, uint32_t earlier) {
  uint32_t r = 0;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const uint32_t fe = (earlier >> (2 * e)) & 3u;
    r |= ((later >> (2 * fe)) & 3u) << (2 * e);
  }
  return r;
}

__global__ void __launch_bounds__(kWalkThreads) prompt_walk_kernel(MatchArgs a, MatchWs w) {
  griddep_wait();
  __shared__ int8_t s_m[kPass];
  __shared__ uint32_t s_wmap[kWalkThreads / 32];
  __shared__ int s_wsum[kWalkThreads / 32];
  __shared__ uint32_t s_entry_last;
  __shared__ int s_last;
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int Lb = prompt_len(a, b);
  const int64_t row = (int64_t)b * a.L;
  const int64_t sbase = (int64_t)b * span_stride(a.L);
  uint32_t carry_e = 0;
  int carry_n = 0, carry_t = 0;
  for (int base = 0; base < Lb; base += kPass) {
    for (int i = tid; i < kPass; i += kWalkThreads) s_m[i] = base + i < Lb ? w.mlen[row + base + i] : 0;
    __syncthreads();
    const int8_t *m = s_m + tid * kSeg;
    // the map entry -> exit offset of this segment, and spans / tokens per entry
    uint32_t map = 0, cnt = 0, tok = 0;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      int q = e, c = 0, t = 0;
      while (q < kSeg) {
        const int n = m[q];
        if (n >= 2) {
          ++c;
          t += n;
          q += n;
        } else {
          ++q;
        }
      }
      map |= (uint32_t)(q - kSeg) << (2 * e);
      cnt |= (uint32_t)c << (8 * e);
      tok |= (uint32_t)t << (8 * e);
    }
    // inclusive scan of compositions: P_t = F_t o ... o F_0
    uint32_t P = map;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t other = __shfl_up_sync(0xffffffffu, P, o);
      if (lane >= o) P = compose(P, other);
    }
    if (lane == 31) s_wmap[wid] = P;
    __syncthreads();
    uint32_t wprefix = kIdentity;   // composition of the earlier warps' segments
    for (int v = 0; v < wid; ++v) wprefix = compose(s_wmap[v], wprefix);
    const uint32_t before = __shfl_up_sync(0xffffffffu, P, 1);   // every lane takes part
    const uint32_t excl = lane > 0 ? compose(before, wprefix) : wprefix;
    const uint32_t entry = (excl >> (2 * carry_e)) & 3u;
    if (tid == kWalkThreads - 1) s_entry_last = (compose(P, wprefix) >> (2 * carry_e)) & 3u;
    // spans and tokens before this segment
    const int my_c = (cnt >> (8 * entry)) & 0xFF, my_t = (tok >> (8 * entry)) & 0xFF;
    int x = (my_c << 16) | my_t;
    int incl = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane == 31) s_wsum[wid] = incl;
    __syncthreads();
    int wsum_before = 0, total = 0;
    for (int v = 0; v < kWalkThreads / 32; ++v) {
      if (v < wid) wsum_before += s_wsum[v];
      total += s_wsum[v];
    }
    const int ex = incl - x + wsum_before;
    // re-walk from the actual entry, writing the spans
    int out = carry_n + (ex >> 16);
    for (int q = (int)entry; q < kSeg;) {
      const int n = m[q];
      if (n >= 2) {
        const int p = base + tid * kSeg + q;
        if (in_bounds(out, span_stride(a.L), a.status, kSiteRulesSpanSlot) &&
            in_bounds(p, Lb, a.status, kSiteRulesSpanSlot)) {
          w.sp_start[sbase + out] = p;
          w.sp_len[sbase + out] = n;
          w.sp_rule[sbase + out] = w.mrule[row + p];
        }
        ++out;
        q += n;
      } else {
        ++q;
      }
    }
    carry_n += total >> 16;
    carry_t += total & 0xFFFF;
    __syncthreads();
    carry_e = s_entry_last;
  }
  if (tid == 0) {
    w.count[b] = carry_n;
    w.ntok[b] = carry_t;
  }
  // the last CTA: span and token offsets of every prompt
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    s_last = atomicAdd(&w.hdr->done, 1) == a.B - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  int cs = 0, ct = 0;
  for (int base = 0; base < a.B; base += kWalkThreads) {
    const int i = base + tid;
    const int c = i < a.B ? w.count[i] : 0, t = i < a.B ? w.ntok[i] : 0;
    int ic = c, it = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int yc = __shfl_up_sync(0xffffffffu, ic, o), yt = __shfl_up_sync(0xffffffffu, it, o);
      if (lane >= o) {
        ic += yc;
        it += yt;
      }
    }
    if (lane == 31) {
      s_wsum[wid] = ic;
      s_wmap[wid] = (uint32_t)it;
    }
    __syncthreads();
    int bc = 0, bt = 0, tc = 0, tt = 0;
    for (int v = 0; v < kWalkThreads / 32; ++v) {
      if (v < wid) {
        bc += s_wsum[v];
        bt += (int)s_wmap[v];
      }
      tc += s_wsum[v];
      tt += (int)s_wmap[v];
    }
    if (i < a.B) {
      a.span_offsets[i] = cs + bc + ic - c;
      w.tok_base[i] = ct + bt + it - t;
    }
    cs += tc;
    ct += tt;
    __syncthreads();
  }
  if (tid == 0) {
    a.span_offsets[a.B] = cs;
    w.tok_base[a.B] = ct;
    w.hdr->done = 0;
  }
}

__global__ void __launch_bounds__(256) span_compact_kernel(MatchArgs a, MatchWs w) {
  griddep_wait();
  __shared__ int s_wsum[8];
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int n = w.count[b];
  const int base = a.span_offsets[b];
  const int64_t sbase = (int64_t)b * span_stride(a.L);
  int tcarry = w.tok_base[b];
  for (int c0 = 0; c0 < n; c0 += 256) {
    const int i = c0 + tid;
    int st = 0, ln = 0;
    if (i < n) {
      st = w.sp_start[sbase + i];
      ln = w.sp_len[sbase + i];
      a.span_start[base + i] = st;
      a.span_len[base + i] = ln;
      a.span_rule[base + i] = w.sp_rule[sbase + i];
    }
    if (a.merge_tokens) {
      int incl = ln;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      if (lane == 31) s_wsum[wid] = incl;
      __syncthreads();
      int before = 0, total = 0;
      for (int v = 0; v < 8; ++v) {
        if (v < wid) before += s_wsum[v];
        total += s_wsum[v];
      }
      if (i < n) {
        const int t0 = tcarry + before + incl - ln;
        a.merge_offsets[base + i] = t0;
        if (ln > 0 && in_bounds(st + ln - 1, a.L, a.status, kSiteRulesSpanToken))
          for (int k = 0; k < ln; ++k) a.merge_tokens[t0 + k] = a.tokens[(int64_t)b * a.L + st + k];
      }
      tcarry += total;
      __syncthreads();
    }
  }
  if (a.merge_offsets && b == a.B - 1 && tid == 0) a.merge_offsets[a.span_offsets[a.B]] = w.tok_base[a.B];
}

// ---------------------------------------------------------------------------
// decoding: suffix matching
// ---------------------------------------------------------------------------
constexpr int kSuffixThreads = 1024;

__global__ void __launch_bounds__(kSuffixThreads)
    suffix_match_kernel(const uint4 *slots, uint32_t mask, int4 *state, const int32_t *new_tokens, int B,
                        int32_t *merge_k, int32_t *merge_rule, int32_t *merge_row, int32_t *rows_rule,
                        int32_t *n_merges, int32_t *status) {
  griddep_wait();
  __shared__ int s_wsum[kSuffixThreads / 32];
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  int carry = 0;
  for (int base = 0; base < B; base += kSuffixThreads) {
    const int b = base + tid;
    int k = 0;
    int32_t rule = -1;
    if (b < B) {
      int4 s = state[b];
      const int32_t y = new_tokens[b];
      int n_raw = s.w;
      if (n_raw < 0 || n_raw > 3) {
        set_error(status, UMIM_ERR_INVALID_ARG);
        n_raw = 0;
      }
      if (y < 0 || (uint32_t)y >= kPadTok) {
        // not a token id: no merge, and the raw suffix restarts after it
        set_error(status, UMIM_ERR_INVALID_ARG);
        s = make_int4(-1, -1, -1, 0);
      } else {
        const uint32_t c[4] = {(uint32_t)s.x, (uint32_t)s.y, (uint32_t)s.z, (uint32_t)y};
        const bool ok[5] = {false, false, n_raw >= 1, n_raw >= 2, n_raw >= 3};
        longest_rule(slots, mask, ok, [=](int n) { return tail_key(c, n); }, k, rule);
        if (k > 0) s = make_int4(-1, -1, -1, 0);   // the merged span becomes one marker
        else s = make_int4(s.y, s.z, y, min(n_raw + 1, 3));
      }
      state[b] = s;
      merge_k[b] = k;
      merge_rule[b] = rule;
    }
    // rows of the merging sequences, in sequence order
    const int x = k > 0 ? 1 : 0;
    const unsigned bal = __ballot_sync(0xffffffffu, x);
    if (lane == 0) s_wsum[wid] = __popc(bal);
    __syncthreads();
    int before = 0, total = 0;
    for (int v = 0; v < kSuffixThreads / 32; ++v) {
      if (v < wid) before += s_wsum[v];
      total += s_wsum[v];
    }
    const int row = carry + before + __popc(bal & ((1u << lane) - 1u));
    if (b < B) {
      merge_row[b] = x ? row : -1;
      if (x && rows_rule) rows_rule[row] = rule;
    }
    carry += total;
    __syncthreads();
  }
  if (tid == 0 && n_merges) *n_merges = carry;
}

// ---------------------------------------------------------------------------
// surrogate lookup
// ---------------------------------------------------------------------------
// one CTA per row (grid-stride): 16-byte chunks, four loads in flight per thread
constexpr int kGatherThreads = 256, kGatherUnroll = 4;

__global__ void __launch_bounds__(kGatherThreads) lut_gather_kernel(const float4 *lut, int64_t n_rules, int d4,
                                                                    const int32_t *ids, int n_max,
                                                                    const int32_t *n_dev, float4 *out,
                                                                    int32_t *status) {
  griddep_wait();
  const int n = n_dev ? min(max(*n_dev, 0), n_max) : n_max;
  for (int row = blockIdx.x; row < n; row += gridDim.x) {
    const int32_t id = ids[row];
    const bool ok = id >= 0 && id < n_rules;
    if (!ok && threadIdx.x == 0) set_error(status, UMIM_ERR_INVALID_ARG);
    const float4 *src = lut + (int64_t)(ok ? id : 0) * d4;
    float4 *dst = out + (int64_t)row * d4;
    for (int c0 = threadIdx.x; c0 < d4; c0 += kGatherThreads * kGatherUnroll) {
      float4 v[kGatherUnroll];
#pragma unroll
      for (int u = 0; u < kGatherUnroll; ++u) {
        const int c = c0 + u * kGatherThreads;
        v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (ok && c < d4)
          asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0, %1, %2, %3}, [%4];"
                       : "=f"(v[u].x), "=f"(v[u].y), "=f"(v[u].z), "=f"(v[u].w)
                       : "l"(src + c));
      }
#pragma unroll
      for (int u = 0; u < kGatherUnroll; ++u) {
        const int c = c0 + u * kGatherThreads;
        if (c < d4) dst[c] = v[u];
      }
    }
  }
}

}  // namespace

// slots: a power of two >= 1.5 x rules (load factor <= 2/3), so that the
// 2.2 million rules of a Llama-3 rule set fit 64 MB and stay in L2
size_t rule_table_bytes(int64_t n_rules) {
  uint64_t cap = 16;
  while (cap < ((3 * (uint64_t)n_rules + 1) >> 1)) cap <<= 1;
  return (size_t)cap * 16;
}

umim_status rules_build(void *table, size_t table_bytes, const int32_t *rules, int64_t n_rules, int32_t *status,
                        cudaStream_t stream, int num_sms) {
  const uint64_t cap = table_bytes / 16;
  if (cudaMemsetAsync(table, 0xFF, table_bytes, stream) != cudaSuccess) return UMIM_ERR_CUDA;
  if (n_rules == 0) return UMIM_OK;
  const uint32_t mask = (uint32_t)(cap - 1);
  const int grid = (int)std::min<int64_t>((n_rules + 255) / 256, (int64_t)num_sms * 8);
  trace_mark(stream, "rules.insert");
  if (launch_pdl(rules_insert_kernel, dim3(grid), dim3(256), 0, stream, static_cast<uint4 *>(table), mask,
                 reinterpret_cast<const int4 *>(rules), n_rules, status) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, "rules.verify");
  if (launch_pdl(rules_verify_kernel, dim3(grid), dim3(256), 0, stream, static_cast<const uint4 *>(table), mask,
                 reinterpret_cast<const int4 *>(rules), n_rules, status) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, nullptr);
  return UMIM_OK;
}

size_t match_prompts_workspace_bytes(int B, int L) { return match_ws_bytes(B, L); }

umim_status match_prompts(const void *table, size_t table_bytes, const int32_t *tokens, int B, int L,
                          const int32_t *lens, int32_t *span_offsets, int32_t *span_start, int32_t *span_len,
                          int32_t *span_rule, int32_t *merge_tokens, int32_t *merge_offsets, void *ws,
                          int32_t *status, cudaStream_t stream, int num_sms) {
  MatchWs w = match_carve(ws, B, L);
  MatchArgs a{};
  a.slots = static_cast<const uint4 *>(table);
  a.mask = (uint32_t)(table_bytes / 16 - 1);
  a.tokens = tokens;
  a.B = B;
  a.L = L;
  a.lens = lens;
  a.span_offsets = span_offsets;
  a.span_start = span_start;
  a.span_len = span_len;
  a.span_rule = span_rule;
  a.merge_tokens = merge_tokens;
  a.merge_offsets = merge_offsets;
  a.status = status;
  if (cudaMemsetAsync(w.hdr, 0, sizeof(MatchHdr), stream) != cudaSuccess) return UMIM_ERR_CUDA;
  const int64_t positions = (int64_t)B * L;
  const int grid = (int)std::max<int64_t>(1, std::min<int64_t>((positions + 255) / 256, (int64_t)num_sms * 16));
  trace_mark(stream, "match.probe");
  if (launch_pdl(rule_probe_kernel, dim3(grid), dim3(256), 0, stream, a, w) != cudaSuccess) return UMIM_ERR_CUDA;
  trace_mark(stream, "match.walk");
  if (launch_pdl(prompt_walk_kernel, dim3(B), dim3(kWalkThreads), 0, stream, a, w) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, "match.compact");
  if (launch_pdl(span_compact_kernel, dim3(B), dim3(256), 0, stream, a, w) != cudaSuccess) return UMIM_ERR_CUDA;
  trace_mark(stream, nullptr);
  return UMIM_OK;
}

umim_status match_suffix(const void *table, size_t table_bytes, void *state, const int32_t *new_tokens, int B,
                         int32_t *merge_k, int32_t *merge_rule, int32_t *merge_row, int32_t *rows_rule,
                         int32_t *n_merges, int32_t *status, cudaStream_t stream) {
  trace_mark(stream, "match.suffix");
  if (launch_pdl(suffix_match_kernel, dim3(1), dim3(kSuffixThreads), 0, stream, static_cast<const uint4 *>(table),
                 (uint32_t)(table_bytes / 16 - 1), static_cast<int4 *>(state), new_tokens, B, merge_k, merge_rule,
                 merge_row, rows_rule, n_merges, status) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, nullptr);
  return UMIM_OK;
}

umim_status lookup_surrogates(const float *lut, int64_t n_rules, int d, const int32_t *ids, int n_max,
                              const int32_t *n_dev, float *out, int32_t *status, cudaStream_t stream, int num_sms) {
  const int d4 = d / 4;
  const int grid = std::max(1, std::min(n_max, std::max(1, num_sms) * 8));
  trace_mark(stream, "lut.gather");
  if (launch_pdl(lut_gather_kernel, dim3(grid), dim3(kGatherThreads), 0, stream, reinterpret_cast<const float4 *>(lut), n_rules,
                 d4, ids, n_max, n_dev, reinterpret_cast<float4 *>(out), status) != cudaSuccess)
    return UMIM_ERR_CUDA;
  trace_mark(stream, nullptr);
  return UMIM_OK;
}

}  // namespace umim
