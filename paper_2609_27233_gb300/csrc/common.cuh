// Shared device helpers of libumim: status words, bounded waits, mbarriers,
// TMA (cp.async.bulk.tensor) and tcgen05 wrappers as inline PTX for sm_103a.
#pragma once

#include <atomic>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>

#include "../../include/umim.h"

namespace umim {

// Every spin wait gives up after this many nanoseconds of %globaltimer, records
// UMIM_ERR_TIMEOUT in the call's status word and lets the kernel return.
constexpr uint64_t kWaitLimitNs = 1000000000ull;   // 1 s

constexpr int kPageSize = 16;

// ---------------------------------------------------------------------------
// status word
// ---------------------------------------------------------------------------
__device__ __forceinline__ void set_error(int32_t *status, int32_t code) {
  if (status != nullptr) atomicCAS(status, 0, code);
}

__device__ __forceinline__ int32_t read_status(const int32_t *status) {
  if (status == nullptr) return 0;
  return *reinterpret_cast<const volatile int32_t *>(status);
}

// ---------------------------------------------------------------------------
// debug build
// ---------------------------------------------------------------------------
// Compiled with -DUMIM_DEBUG (libumim_debug.so), the kernels check at their
// access sites that every index they computed from device data lies inside the
// buffer it addresses.  A failed check records UMIM_ERR_BOUNDS | site << 8 in
// the call's status word (the first error wins, as for every code) and the
// access is skipped: a store is dropped, a load yields zeros or reads an
// in-bounds stand-in (where a copy must still complete a barrier).  These are
// checks of the kernels' own invariants (the inputs are validated in both
// builds); in the normal build every check is the constant true and
// compiles to nothing.
#ifdef UMIM_DEBUG
constexpr bool kDebugChecks = true;
#else
constexpr bool kDebugChecks = false;
#endif

// check sites; umim_debug_site_name() gives their names
enum DebugSite : int32_t {
  kSiteSelftest = 1,
  kSiteRollbackMapTable = 2,
  kSiteRollbackDstPage = 3,
  kSiteRollbackSrc = 4,
  kSiteRollbackSurrogate = 5,
  kSiteRollbackReaderRow = 6,
  kSiteAppendDst = 7,
  kSiteAppendSrcRow = 8,
  kSiteAttnTable = 9,
  kSiteAttnPiece = 10,
  kSiteStepTable = 11,
  kSiteStepCacheWrite = 12,
  kSiteStepPartial = 13,
  kSiteMergePoolStats = 14,
  kSiteMergeGemmStore = 15,
  kSiteMergePoolSpan = 16,
  kSiteCompactToken = 17,
  kSitePrefillKvRow = 18,
  kSitePrefillOutRow = 19,
  kSiteDistillTeacherRow = 20,
  kSiteDistillPair = 21,
  kSiteRulesSpanSlot = 22,
  kSiteRulesSpanToken = 23,
  kSiteCount = 24
};

// true when 0 <= i < n; in the debug build a false result is recorded
__device__ __forceinline__ bool in_bounds(int64_t i, int64_t n, int32_t *status, DebugSite site) {
  if constexpr (!kDebugChecks) {
    return true;
  } else {
    const bool ok = (uint64_t)i < (uint64_t)n;
    if (!ok) set_error(status, UMIM_ERR_BOUNDS | ((int32_t)site << 8));
    return ok;
  }
}

__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ---------------------------------------------------------------------------
// global flags with acquire / release semantics (gpu scope)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void st_release(int32_t *p, int32_t v) {
  asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ int32_t ld_acquire(const int32_t *p) {
  int32_t v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// ---------------------------------------------------------------------------
// mbarrier
// ---------------------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Wait for the phase with the given parity to complete; false after limit_ns.
__device__ __forceinline__ bool mbar_wait_for(uint64_t *bar, uint32_t parity, uint64_t limit_ns) {
  const uint32_t a = smem_u32(bar);
  if (mbar_try_wait(a, parity)) return true;
  const uint64_t t0 = globaltimer();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 32; ++i)
      if (mbar_try_wait(a, parity)) return true;
    if (globaltimer() - t0 > limit_ns) return false;
  }
}

__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity) {
  return mbar_wait_for(bar, parity, kWaitLimitNs);
}

// Wait until *cnt >= target (gpu-scope acquire); false when *abort becomes
// nonzero or after limit_ns.
__device__ __forceinline__ bool wait_count_for(const int32_t *cnt, int target, const int32_t *abort,
                                               uint64_t limit_ns) {
  const uint64_t t0 = globaltimer();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 32; ++i)
      if (ld_acquire(cnt) >= target) return true;
    if (ld_acquire(abort) != 0 || globaltimer() - t0 > limit_ns) return false;
  }
}

// ---------------------------------------------------------------------------
// TMA
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

__device__ __forceinline__ void tma_load_2d(void *dst, const CUtensorMap *map, uint64_t *bar, int c0, int c1,
                                            uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

__device__ __forceinline__ void tma_load_5d(void *dst, const CUtensorMap *map, uint64_t *bar, int c0, int c1,
                                            int c2, int c3, int c4, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.5d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4, %5, %6}], [%7], %8;" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(c4), "r"(smem_u32(bar)),
      "l"(policy)
      : "memory");
}

__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap *map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

// ---------------------------------------------------------------------------
// tcgen05 (5th-generation tensor cores, accumulators in tensor memory)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t *dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
}

__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, bf16 inputs, fp32 accumulate.
__device__ __forceinline__ void tc_mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on an mbarrier once every tcgen05 operation this thread issued so far completes.
__device__ __forceinline__ void tc_commit(uint64_t *bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}

// 32 lanes x 32 consecutive fp32 columns: thread i gets row (lane base + i).
__device__ __forceinline__ void tmem_ld_32x32b_x32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Shared-memory matrix descriptor for a K-major bf16 tile written by TMA with
// 128-byte swizzling: rows of 128 bytes, 8-row atoms 1024 bytes apart.
__device__ __forceinline__ uint64_t sw128_kmajor_desc(uint32_t smem_addr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((smem_addr >> 4) & 0x3FFF);          // start address
  d |= static_cast<uint64_t>(1) << 16;                             // leading byte offset (unused here)
  d |= static_cast<uint64_t>(1024 >> 4) << 32;                     // stride byte offset: 8 rows x 128 B
  d |= static_cast<uint64_t>(1) << 46;                             // descriptor version
  d |= static_cast<uint64_t>(2) << 61;                             // 128-byte swizzle
  return d;
}

// Instruction descriptor of kind::f16: both operands bf16 (or both fp16),
// fp32 accumulate, both K-major, M x N tile.
__host__ __device__ constexpr uint32_t idesc_f32acc(int M, int N, bool fp16_operands) {
  return (1u << 4)                                             // D format: fp32
         | (fp16_operands ? 0u : 1u) << 7                      // A format: fp16 = 0, bf16 = 1
         | (fp16_operands ? 0u : 1u) << 10                     // B format (same type as A)
         | (static_cast<uint32_t>(N >> 3) << 17)               // N / 8
         | (static_cast<uint32_t>(M >> 4) << 24);              // M / 16
}

// ---------------------------------------------------------------------------
// misc
// ---------------------------------------------------------------------------
__device__ __forceinline__ float gelu_erf(float x) {
  return 0.5f * x * (1.0f + erff(x * 0.70710678118654752440f));
}

__host__ __device__ __forceinline__ int ceil_div(int a, int b) { return (a + b - 1) / b; }

// Programmatic dependent launch: a kernel launched with launch_pdl may start
// while the previous kernel of the stream is finishing; griddep_wait() blocks
// until that kernel has completed and its writes are visible.  Every kernel
// calls it before its first access to memory another kernel may have written
// (it is a no-op for a kernel launched the ordinary way).
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                              Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// SM count of a device, looked up once per device; atomics, since calls for
// different devices may come from different host threads.
inline int sm_count(int dev) {
  static std::atomic<int> sms_of[64];
  int sms = 0;
  if (dev >= 0 && dev < 64) sms = sms_of[dev].load(std::memory_order_relaxed);
  if (sms == 0) {
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) sms = 0;
    if (sms > 0 && dev >= 0 && dev < 64) sms_of[dev].store(sms, std::memory_order_relaxed);
  }
  return sms;
}

// For the duration of one library call: makes the stream's device current and
// puts the caller's current device back when the call returns.  A stream being
// captured into a CUDA graph refuses cudaStreamGetDevice (and the refusal would
// invalidate the capture), so during a capture the current device is taken as
// the stream's.
class DeviceScope {
 public:
  explicit DeviceScope(cudaStream_t stream) {
    int cur = -1;
    if (cudaGetDevice(&cur) != cudaSuccess) cur = -1;
    dev_ = cur;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    int sdev = -1;
    if (stream != nullptr && cudaStreamIsCapturing(stream, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusNone &&
        cudaStreamGetDevice(stream, &sdev) == cudaSuccess && sdev != cur && cudaSetDevice(sdev) == cudaSuccess) {
      prev_ = cur;
      dev_ = sdev;
    }
    sms_ = dev_ >= 0 ? sm_count(dev_) : 0;
  }
  ~DeviceScope() {
    if (prev_ >= 0) cudaSetDevice(prev_);
  }
  DeviceScope(const DeviceScope &) = delete;
  DeviceScope &operator=(const DeviceScope &) = delete;
  int device() const { return dev_; }
  int sms() const { return sms_; }

 private:
  int dev_ = -1, prev_ = -1, sms_ = 0;
};

// Kernel tracing (trace.cu): records an event labelled with the next kernel,
// or, with a null label, the end of a call.  No-op unless a trace is active.
void trace_mark(cudaStream_t stream, const char *label);

}  // namespace umim
