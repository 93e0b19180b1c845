// Decode attention for callers that cannot allocate device memory: the
// split-K workspace lives in a fixed device array of this translation unit
// instead of caller memory.  See optr_decode_attention_noalloc in optr.h.
#include <mutex>

#include "optr_internal.cuh"

namespace {

// The scratch array.  In host code its name is only a host-side stand-in
// for the symbol; kernels get its device address from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_decode_scratch[OPTR_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices];  // device address per device, or nullptr

// Device address of the scratch array on the current device (looked up
// once per device, with that device current).
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_ptr[dev]) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_decode_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[dev] = ptr;
  }
  *out = g_scratch_ptr[dev];
  return cudaSuccess;
}

}  // namespace

extern "C" optr_status optr_decode_attention_noalloc(
    const optr_params* p, const void* q, const int32_t* block_table,
    const int32_t* seq_lens, int B, int max_pages, const uint8_t* pool,
    int num_pages, float* out, cudaStream_t stream) {
  if (!p || B <= 0 || max_pages <= 0) return OPTR_ERR_INVALID_ARG;
  const size_t need = optr_decode_workspace_size(p, B, max_pages);
  if (need == 0 || need > OPTR_NOALLOC_SCRATCH_BYTES) return OPTR_ERR_WORKSPACE;
  void* ws = nullptr;
  if (scratch_address(&ws) != cudaSuccess) return OPTR_ERR_CUDA;
  return optr_decode_attention(p, q, block_table, seq_lens, B, max_pages,
                               pool, num_pages, out, ws,
                               OPTR_NOALLOC_SCRATCH_BYTES, stream);
}
