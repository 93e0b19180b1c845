// Register-level helpers of the tensor-core decode kernels (mma.sync
// m16n8k16 with f16 operands and f32 accumulators): INT2 code fields as
// normal fp16 operands, fp16 hi/lo splits of float32 operands, exp2.
#pragma once

#include "decode_common.cuh"

namespace optr {

__device__ __forceinline__ void mma16816(float* d, uint32_t a0, uint32_t a1,
                                         uint32_t a2, uint32_t a3, uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void ldsm_x4_trans(uint32_t& r0, uint32_t& r1,
                                              uint32_t& r2, uint32_t& r3,
                                              const void* smem_row) {
  const unsigned a = static_cast<unsigned>(__cvta_generic_to_shared(smem_row));
  asm volatile(
      "ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
      : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
      : "r"(a));
}

// The two code fields at bit pos of each 16-bit half of src as fp16
// 1024 + code * 2^pos (pos <= 8 keeps the field inside the mantissa).
template <int pos>
__device__ __forceinline__ uint32_t field_f16x2(uint32_t src, uint32_t exp1024) {
  uint32_t x;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;"  // (a & b) | c
      : "=r"(x) : "r"(src), "n"(0x00030003u << pos), "r"(exp1024));
  return x;
}

// The 16 code fields of a word y whose 16-bit halves each hold one byte of
// group 2j (low byte) and one of group 2j+1 (high byte), as MMA A registers
// out[parity][r] = fp16 1024 + code * 2^pos, pos = code_pos(parity, r).
__device__ __forceinline__ void code_fields(uint32_t y, uint32_t e1024,
                                           uint32_t (&out)[2][4]) {
  const uint32_t yl = y << 4, yr = y >> 6;
  out[0][0] = field_f16x2<code_pos(0, 0)>(yl, e1024);
  out[0][1] = field_f16x2<code_pos(0, 1)>(yl, e1024);
  out[0][2] = field_f16x2<code_pos(0, 2)>(y, e1024);
  out[0][3] = field_f16x2<code_pos(0, 3)>(y, e1024);
  out[1][0] = field_f16x2<code_pos(1, 0)>(y, e1024);
  out[1][1] = field_f16x2<code_pos(1, 1)>(yr, e1024);
  out[1][2] = field_f16x2<code_pos(1, 2)>(yr, e1024);
  out[1][3] = field_f16x2<code_pos(1, 3)>(yr, e1024);
}

// A field from code_fields() of group parity par and code index r
// (1024 + code * 2^pos) mapped by one HFMA2 to the exact centered code
// code - 1.5 in {-1.5, -0.5, 0.5, 1.5}: x * 2^-pos - (1024 * 2^-pos + 1.5).
// Both constants are exact fp16 values for pos = 4, 6, 8.
__device__ __forceinline__ uint32_t centered(uint32_t x, int par, int r) {
  const int pos = code_pos(par, r);
  const __half2 sc = __float2half2_rn(1.0f / (float)(1 << pos));
  const __half2 bias = __float2half2_rn(-1024.0f / (float)(1 << pos) - 1.5f);
  const __half2 y = __hfma2(*reinterpret_cast<const __half2*>(&x), sc, bias);
  return *reinterpret_cast<const uint32_t*>(&y);
}

__device__ __forceinline__ float2 h2f(uint32_t u) {
  return __half22float2(*reinterpret_cast<const __half2*>(&u));
}

// fp16 hi / lo split of x, packed (hi in the low half): hi is x with its
// mantissa cut to 11 significant bits (exact in fp16 when |x| is in fp16's
// normal range), lo = x - hi exactly, rounded to fp16.
__device__ __forceinline__ uint32_t split_hilo(float x) {
  const float hi = __uint_as_float(__float_as_uint(x) & 0xffffe000u);
  const float lo = x - hi;
  uint32_t r;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(lo), "f"(hi));
  return r;
}

// 2^x (the MUFU approximation; relative error ~2^-22).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// 2^n as a float, for -126 <= n <= 127 (built from the exponent field).
__device__ __forceinline__ float pow2i(int n) { return __int_as_float((n + 127) << 23); }

// floor(log2 x) of a positive normal float (its exponent field); subnormal
// inputs give -127.
__device__ __forceinline__ int exponent_of(float x) {
  return ((__float_as_int(x) >> 23) & 0xff) - 127;
}

// m16n8k16 with bf16 operands, f32 accumulators (in place)
__device__ __forceinline__ void mma16816_bf16(float* d, uint32_t a0, uint32_t a1,
                                              uint32_t a2, uint32_t a3, uint32_t b0,
                                              uint32_t b1) {
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void ldsm_x4(uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3, const void* smem_row) {
  const unsigned a = static_cast<unsigned>(__cvta_generic_to_shared(smem_row));
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(a));
}

}  // namespace optr
