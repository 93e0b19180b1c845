// The INT2 group quantizer Q2 as the kernels evaluate it (paper Sec. 3.1:
// group-wise affine INT2 with clipping ratio c; the exact float32 formula is
// the one documented in include/optr.h).  Every operation that decides a
// code is an explicit round-to-nearest intrinsic so that no FMA contraction
// changes it.
#pragma once

#include <cuda_fp16.h>

namespace optr {

struct GroupQuant {
  float mn, mx, inv;  // clipped range and 3 / (mx - mn)
  bool degenerate;
  __half scale, min;  // stored metadata
};

__device__ __forceinline__ GroupQuant group_quant_params(float lo, float hi,
                                                         float clip) {
  GroupQuant q;
  q.mn = __fmul_rn(clip, lo);
  q.mx = __fmul_rn(clip, hi);
  const float r = __fsub_rn(q.mx, q.mn);
  q.degenerate = !(r > 1e-30f) || !(r <= 3.402823466e38f);
  q.inv = q.degenerate ? 0.f : __fdiv_rn(3.0f, r);
  q.scale = q.degenerate ? __float2half_rn(0.f) : __float2half_rn(__fdiv_rn(r, 3.0f));
  q.min = __float2half_rn(q.mn);
  return q;
}

__device__ __forceinline__ int quant_code(float z, const GroupQuant& q) {
  const float zc = fminf(fmaxf(z, q.mn), q.mx);
  const float u = __fmul_rn(__fsub_rn(zc, q.mn), q.inv);
  const int c = __float2int_rn(u);
  return q.degenerate ? 0 : min(max(c, 0), 3);
}

}  // namespace optr
