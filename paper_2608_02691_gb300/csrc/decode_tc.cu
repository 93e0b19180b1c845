// Tensor-core split-K partial kernel (placeholder until implemented).
#include "decode_common.cuh"

namespace optr {

cudaError_t launch_partial_tensor(const optr_params*, const uint8_t*,
                                  const int32_t*, const int32_t*, int, int,
                                  int, const float*, const float*, const int*,
                                  const int*, float*, int, cudaStream_t) {
  return cudaErrorNotSupported;
}

}  // namespace optr
