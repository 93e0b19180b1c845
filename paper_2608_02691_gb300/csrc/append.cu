// Cache write: center, rotate, INT2-quantize, pack and scatter
// (paper Sec. 4.1 "Rotated INT2 Cache Reparameterization"; Appendix,
// "Key-mean estimation and application": (k - mu) R_K = k R_K - mu R_K with
// mu R_K precomputed, subtracted right after the rotation).
#include "optr_internal.cuh"
#include "quant.cuh"
#include "append_common.cuh"
#include "append_small.cuh"

namespace optr {
namespace {

// CUDA-core variant.  Block = 256 threads: warp w < 4 computes key group w,
// warp w >= 4 value group w-4; lane = channel within the group.  Each block
// handles T consecutive new tokens of one KV head; every thread keeps T
// float32 accumulators of z_j = sum_i x_i R[i][j] (j = its channel), reading
// R[i][j] once per i (coalesced) and x from shared memory.
template <int T>
__global__ void __launch_bounds__(256)
append_cuda_core_kernel(const __nv_bfloat16* __restrict__ k,
                        const __nv_bfloat16* __restrict__ v, int n_tok,
                        const int32_t* __restrict__ cu_new,
                        const int32_t* __restrict__ pos0,
                        const int32_t* __restrict__ bt, int B, int max_pages,
                        uint8_t* __restrict__ pool, int num_pages, int h_kv,
                        const float* __restrict__ R_k,
                        const float* __restrict__ R_v,
                        const float* __restrict__ muR, float clip_k,
                        float clip_v, unsigned* err, int group128) {
  __shared__ float xs[2][T][kD];
  __shared__ float2 grange[2][kGroups];  // G = 128: block ranges of a token
  __shared__ long long dst[T];
  __shared__ int dslot[T];
  const int h = blockIdx.y;
  const int t0 = blockIdx.x * T;
  const int tid = threadIdx.x;
  pdl_wait();
  pdl_trigger();

  for (int idx = tid; idx < 2 * T * kD; idx += blockDim.x) {
    int kind = idx / (T * kD);
    int rem = idx - kind * T * kD;
    int t = rem / kD, i = rem % kD;
    int tok = t0 + t;
    float x = 0.f;
    if (tok < n_tok) {
      const __nv_bfloat16* src = kind ? v : k;
      x = __bfloat162float(src[((size_t)tok * h_kv + h) * kD + i]);
    }
    xs[kind][t][i] = x;
  }
  if (tid < T) {
    int tok = t0 + tid;
    int slot = 0;
    long long off = -1;
    if (tok < n_tok)
      off = resolve_slot(tok, h, cu_new, pos0, bt, B, max_pages, num_pages,
                         h_kv, &slot, err, chunk_bytes(group128 != 0));
    dst[tid] = off;
    dslot[tid] = slot;
  }
  __syncthreads();

  const int kind = tid >> 7;   // 0 = key, 1 = value
  const int j = tid & 127;     // rotated channel
  const int g = j >> 5;        // group
  const int lane = j & 31;
  const float* R = (kind ? R_v : R_k) + (size_t)h * kD * kD;
  float acc[T];
#pragma unroll
  for (int t = 0; t < T; ++t) acc[t] = 0.f;
#pragma unroll 8
  for (int i = 0; i < kD; ++i) {
    float r = __ldg(R + i * kD + j);
#pragma unroll
    for (int t = 0; t < T; ++t) acc[t] = fmaf(xs[kind][t][i], r, acc[t]);
  }
  const float sub = kind ? 0.f : __ldg(muR + h * kD + j);
  const float clip = kind ? clip_v : clip_k;
  const int codes_off = kind ? OPTR_V_CODES_OFFSET : OPTR_K_CODES_OFFSET;
  const bool compact = group128 != 0;  // one (scale, min) pair per slot
  const int meta_off = kind ? vmeta_offset(compact) : OPTR_K_META_OFFSET;
#pragma unroll 1
  for (int t = 0; t < T; ++t) {
    const float z = __fsub_rn(acc[t], sub);
    float lo = z, hi = z;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
      hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    if (group128) {  // one range over the four warps (blocks) of this kind
      if (lane == 0) grange[kind][g] = make_float2(lo, hi);
      __syncthreads();
      const float2 r0 = grange[kind][0], r1 = grange[kind][1];
      const float2 r2 = grange[kind][2], r3 = grange[kind][3];
      lo = fminf(fminf(r0.x, r1.x), fminf(r2.x, r3.x));
      hi = fmaxf(fmaxf(r0.y, r1.y), fmaxf(r2.y, r3.y));
      __syncthreads();  // grange is rewritten for the next token
    }
    GroupQuant gq = group_quant_params(lo, hi, clip);
    unsigned bits = (unsigned)quant_code(z, gq) << (2 * (lane & 3));
    bits |= __shfl_xor_sync(0xffffffffu, bits, 1);
    bits |= __shfl_xor_sync(0xffffffffu, bits, 2);
    const long long off = dst[t];
    if (off >= 0) {
      uint8_t* chunk = pool + off;
      const int slot = dslot[t];
      if ((lane & 3) == 0)
        chunk[codes_off + slot * 32 + 4 * (lane >> 2) + g] = (uint8_t)bits;
      if (lane == 0 && (!compact || g == 0))
        *reinterpret_cast<__half2*>(chunk + meta_off + slot * meta_stride(compact) +
                                    (compact ? 0 : 4 * g)) =
            __halves2half2(gq.scale, gq.min);
    }
  }
}

// Decode-step variant for few new tokens: append_small.cuh.
template <int T>
__global__ void __launch_bounds__(512)
append_small_kernel(const __nv_bfloat16* __restrict__ k,
                    const __nv_bfloat16* __restrict__ v, int n_tok,
                    const int32_t* __restrict__ cu_new,
                    const int32_t* __restrict__ pos0,
                    const int32_t* __restrict__ bt, int B, int max_pages,
                    uint8_t* __restrict__ pool, int num_pages, int h_kv,
                    const float* __restrict__ R_k,
                    const float* __restrict__ R_v,
                    const float* __restrict__ muR, float clip_k, float clip_v,
                    unsigned* err, int fold_v, int group128) {
  __shared__ AppendSmallSmemT<T> sm;
  append_small_body<T>(blockIdx.x, blockIdx.y, blockIdx.z, sm, k, v, n_tok,
                    cu_new, pos0, bt, B, max_pages, pool, num_pages, h_kv, R_k,
                    R_v, muR, clip_k, clip_v, err, fold_v && blockIdx.z == 1,
                    group128 != 0);
}

}  // namespace

cudaError_t launch_append_cuda_core(const optr_params* p,
                                    const __nv_bfloat16* k,
                                    const __nv_bfloat16* v, int n_tok,
                                    const int32_t* cu_new, const int32_t* pos0,
                                    const int32_t* bt, int B, int max_pages,
                                    uint8_t* pool, int num_pages,
                                    cudaStream_t s) {
  const int g128 = p->cfg.group == 128 ? 1 : 0;
  // few tokens (decode steps): slice-parallel rotation
  if (n_tok <= 256) {
    const int T = small_tile(n_tok);
    dim3 grid((n_tok + T - 1) / T, p->cfg.h_kv, 2);
    if (T == kSmallTokFew)
      return launch_pdl(append_small_kernel<kSmallTokFew>, grid, dim3(512), 0, s, k, v,
                        n_tok, cu_new, pos0, bt, B, max_pages, pool, num_pages,
                        p->cfg.h_kv, p->R_k, p->R_v, p->muR, p->cfg.clip_k,
                        p->cfg.clip_v, p->err, p->fold_v, g128);
    return launch_pdl(append_small_kernel<kSmallTok>, grid, dim3(512), 0, s, k, v, n_tok,
                      cu_new, pos0, bt, B, max_pages, pool, num_pages,
                      p->cfg.h_kv, p->R_k, p->R_v, p->muR, p->cfg.clip_k,
                      p->cfg.clip_v, p->err, p->fold_v, g128);
  } else {
    constexpr int T = 32;
    dim3 grid((n_tok + T - 1) / T, p->cfg.h_kv);
    return launch_pdl(append_cuda_core_kernel<T>, grid, dim3(256), 0, s, k, v,
                      n_tok, cu_new, pos0, bt, B, max_pages, pool, num_pages,
                      p->cfg.h_kv, p->R_k, p->R_v, p->muR, p->cfg.clip_k,
                      p->cfg.clip_v, p->err, g128);
  }
}

}  // namespace optr
