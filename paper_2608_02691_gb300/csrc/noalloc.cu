// Decode attention for callers that cannot allocate device memory: the
// split-K workspace lives in a fixed device array of this translation unit
// instead of caller memory.  See optr_decode_attention_noalloc in optr.h.
#include "optr_internal.cuh"

namespace {

// The scratch array.  In host code its name is only a host-side stand-in
// for the symbol; kernels get its device address from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_decode_scratch[OPTR_NOALLOC_SCRATCH_BYTES];

}  // namespace

namespace optr {

// Called by optr_params_create with the params' device current: the
// array's address belongs to that device's context, so every params object
// carries the address of its own device (and one created after a device
// reset gets the new one).
cudaError_t noalloc_scratch_address(void** out) {
  return cudaGetSymbolAddress(out, g_decode_scratch);
}

}  // namespace optr

extern "C" optr_status optr_decode_attention_noalloc(
    const optr_params* p, const void* q, const int32_t* block_table,
    const int32_t* seq_lens, int B, int max_pages, const uint8_t* pool,
    int num_pages, float* out, cudaStream_t stream) {
  // the checks of optr_decode_attention, in its order, before the size check
  // (params with BF16 windows are refused, as by optr_decode_attention)
  if (p && (p->cfg.sink > 0 || p->cfg.recent > 0)) return OPTR_ERR_INVALID_ARG;
  const optr_status st = optr::decode_args_status(p, q, block_table, seq_lens, B,
                                                  max_pages, pool, num_pages, out);
  if (st != OPTR_OK) return st;
  const size_t need = optr_decode_workspace_size(p, B, max_pages);
  if (need == 0 || need > OPTR_NOALLOC_SCRATCH_BYTES) return OPTR_ERR_WORKSPACE;
  if (!p->noalloc_ws) return OPTR_ERR_CUDA;
  return optr_decode_attention(p, q, block_table, seq_lens, B, max_pages,
                               pool, num_pages, out, p->noalloc_ws,
                               OPTR_NOALLOC_SCRATCH_BYTES, stream);
}
