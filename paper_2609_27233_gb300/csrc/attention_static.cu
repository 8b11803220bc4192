// Decode attention without a caller-provided workspace.
//
// Some callers cannot allocate device memory at the point where they run
// decode attention: a serving engine that hands every byte of the GPU to its
// own block allocator up front, a plug-in loaded into another framework that
// forbids allocations outside its arena, or code running where an allocation
// would synchronise the device or is simply not permitted.  For them this
// entry point takes its scratch (the split-K plan and the fp32 partial
// results) from a fixed array compiled into the library instead of a
// workspace argument.
#include <mutex>

#include "common.cuh"

namespace umim {
size_t decode_attention_workspace_bytes(int B, int Hq, int Hkv, int D, int num_sms);
umim_status decode_attention(const void *, int, const umim_paged_kv *, int, const int32_t *, int, const int32_t *,
                             int, float, void *, void *, int32_t *, cudaStream_t, int);
}  // namespace umim

namespace {

// Every GPU that loads the library holds this array until the process exits.
static __device__ __align__(256) unsigned char g_attention_scratch[UMIM_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mutex;
void *g_scratch_ptr[kMaxDevices];
int g_sms[kMaxDevices];

// Device address of the scratch array and the SM count on the current
// device, looked up once per device.
umim_status scratch_for_current_device(void **ptr, int *sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return UMIM_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mutex);
  if (g_scratch_ptr[dev] == nullptr) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_attention_scratch) != cudaSuccess || p == nullptr) return UMIM_ERR_CUDA;
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      return UMIM_ERR_CUDA;
    g_sms[dev] = n;
    g_scratch_ptr[dev] = p;
  }
  *ptr = g_scratch_ptr[dev];
  *sms = g_sms[dev];
  return UMIM_OK;
}

}  // namespace

using namespace umim;

extern "C" {

umim_status umim_decode_attention_static(const void *q, int32_t n_q_heads, const umim_paged_kv *kv, int32_t layer,
                                         const int32_t *block_table, int32_t max_pages, const int32_t *seq_lens,
                                         int32_t batch, float scale, void *out, int32_t *dev_status,
                                         cudaStream_t stream) {
  if (!kv || !kv->base || batch < 0 || max_pages < 0 || n_q_heads <= 0 || kv->n_layers <= 0 ||
      kv->n_pages <= 0 || kv->n_kv_heads <= 0 || (reinterpret_cast<uintptr_t>(kv->base) % 16) != 0)
    return UMIM_ERR_INVALID_ARG;
  if (kv->page_size != UMIM_PAGE_SIZE || (kv->head_dim != 64 && kv->head_dim != 128) || kv->n_kv_heads > 64)
    return UMIM_ERR_UNSUPPORTED;
  if (n_q_heads % kv->n_kv_heads != 0 || n_q_heads / kv->n_kv_heads > 16) return UMIM_ERR_UNSUPPORTED;
  if (layer < 0 || layer >= kv->n_layers) return UMIM_ERR_INVALID_ARG;
  if ((int64_t)batch * kv->n_kv_heads > (int64_t)1 << 24) return UMIM_ERR_UNSUPPORTED;
  if (batch == 0) return UMIM_OK;
  if (!q || !block_table || !seq_lens || !out) return UMIM_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(q) % 4) != 0 || (reinterpret_cast<uintptr_t>(out) % 2) != 0)
    return UMIM_ERR_INVALID_ARG;
  // the stream's device is current until this call returns (the caller's current
  // device is put back then); during a stream capture the current device is taken
  // as the stream's
  const DeviceScope scope(stream);
  void *scratch = nullptr;
  int sms = 0;
  const umim_status st = scratch_for_current_device(&scratch, &sms);
  if (st != UMIM_OK) return st;
  // the batch this call needs must fit in the fixed array
  if (decode_attention_workspace_bytes(batch, n_q_heads, kv->n_kv_heads, kv->head_dim, sms) >
      (size_t)UMIM_STATIC_SCRATCH_BYTES)
    return UMIM_ERR_WORKSPACE;
  if (!(scale > 0.f)) scale = 1.0f / sqrtf((float)kv->head_dim);
  return decode_attention(q, n_q_heads, kv, layer, block_table, max_pages, seq_lens, batch, scale, out, scratch,
                          dev_status, stream, sms);
}

}  // extern "C"
