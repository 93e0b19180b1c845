// Tensor-core cache write on tcgen05 (paper Sec. 4.1; Appendix "Key-mean
// estimation and application": z_K = k R_K - mu R_K, z_V = v R_V, then
// group-wise INT2, Sec. 3.1).
//
// The rotation is a dense GEMM per KV head and kind (K or V),
// Z[tok][128] = X[tok][128] R[128][128], run as 128-token tiles on the
// tensor cores: M = 128 tokens, N = 128 rotated channels, K = 128 input
// channels.  X (bf16) converts to f16 exactly within fp16's range; R is
// prescaled by 2^6 and split into fp16 hi + lo, and both halves accumulate
// into the same float32 accumulator, so the products carry ~22 bits of R
// and the result matches a float32 CUDA-core rotation to rounding.
//
// One CTA per SM works on one (KV head, kind) and loops over its tiles:
//   producer warp   one thread loads the tile's 128 token rows with two TMA
//                   tensor copies (channels 0-63 and 64-127, 128-byte
//                   swizzle) into a shared-memory stage (4 stages in
//                   flight);
//   8 epilogue warps, two groups of 4 taking alternate tiles: thread t owns
//                   token row t; it converts its row to f16 and stores it to
//                   tensor memory as the MMA's A operand, then reads its
//                   row of the accumulator back and quantizes, packs and
//                   scatters its 48-byte record (codes + scale/min);
//   MMA warp        one thread issues the 16 tcgen05.mma of a tile (8
//                   K-steps x {R hi, R lo}) from tensor-memory A and
//                   shared-memory B (R, 64 KB, loaded once) into the
//                   group's tensor-memory accumulator.
// Tensor memory (512 columns): accumulators D[2] (128 columns each) and A
// operands A[2] (64 columns each), one of each per epilogue group.
// The quantizer is quant.cuh's float32 formula.
#include "append_common.cuh"
#include "decode_common.cuh"
#include "quant.cuh"
#include "tc05.cuh"

#include <cudaTypedefs.h>
#include <mutex>

namespace optr {

// Host: B operand of one rotation for tcgen05 (f16, K-major, no swizzle):
// out[term][n][k] = (hi, lo) fp16 parts of 64 R[k][n] at element offset
// ((n / 8) * 2048 + (k / 8) * 128 + (n % 8) * 16 + (k % 8) * 2) / 2 of the
// term's 32 KB, i.e. core matrices of 8 output channels x 8 input channels,
// 128 B apart along k (LBO) and 2048 B apart along n (SBO).
void build_rotation_tc05(const float* R, uint16_t* out) {
  auto h16 = [](float x) -> uint16_t {
    __half_raw r = __half(__float2half_rn(x));
    return r.x;
  };
  auto f16 = [](uint16_t bits) -> float {
    __half_raw r;
    r.x = bits;
    return __half2float(__half(r));
  };
  for (int n = 0; n < kD; ++n)
    for (int k = 0; k < kD; ++k) {
      const float x = R[(size_t)k * kD + n] * 64.0f;
      const uint16_t hi = h16(x), lo = h16(x - f16(hi));
      const size_t off = ((size_t)(n / 8) * 2048 + (k / 8) * 128 + (n % 8) * 16 + (k % 8) * 2) / 2;
      out[off] = hi;
      out[(size_t)kD * kD + off] = lo;
    }
}

namespace {

constexpr int kRows = 128;        // tokens per tile (MMA M)
constexpr int kCuCache = 512;     // sequences whose cu_new / pos0 a CTA caches
constexpr int kStages = 4;        // tiles in flight from global memory
constexpr uint32_t kStageBytes = kRows * kD * 2;  // two 16 KB TMA boxes
constexpr int kEpiWarps = 8;      // two groups of 4
constexpr int kThreads = (kEpiWarps + 2) * 32;
constexpr int kProducerWarp = kEpiWarps, kMmaWarp = kEpiWarps + 1;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColD0 = 0, kColA0 = 256;  // D[g] at 128 g, A[g] at 256 + 64 g
constexpr uint32_t kIdesc = tc05::idesc_f16(128, 128);

struct Smem {
  uint16_t b[2][kD * kD];                 // R' hi, lo (64 KB)
  // token rows, bf16: [channel half][row][128 B], 16-byte chunk c of row r
  // at chunk position c ^ (r % 8) (the TMA 128-byte swizzle)
  uint8_t stage[kStages][kStageBytes];
  alignas(16) float mu[kD];               // mu R_k (keys) or 0 (values)
  int cu[kCuCache + 1];
  int p0[kCuCache];
  uint64_t full[kStages], empty[kStages], aready[2], dready[2];
  uint32_t tmem;
  int abort;
};

__device__ __forceinline__ uint32_t bf16x2_to_f16x2(uint32_t u) {
  const float lo = __uint_as_float(u << 16);
  const float hi = __uint_as_float(u & 0xffff0000u);
  uint32_t r;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// Codes of the 32 values of one group into the 8 code words (byte G of word
// w holds channels 32G + 4w + r at bits 2r).  u + 1.5 * 2^23 rounds u in
// [0, 3] to the nearest integer (ties to even, as __float2int_rn) and leaves
// it in the low mantissa bits of the float: bits = 0x4B400000 + code; the
// constant part is removed from each word once, after all 16 codes are in.
template <bool kClamp>
__device__ __forceinline__ void quantize_group(const float (&z)[32], int G,
                                               const GroupQuant& gq,
                                               uint32_t (&word)[8]) {
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    const int w = j >> 2, r = j & 3;
    // with c = 1, z <= mx always; fmaxf also maps a NaN to mn, as the
    // clamped formula does
    const float zc = kClamp ? fminf(fmaxf(z[j], gq.mn), gq.mx) : fmaxf(z[j], gq.mn);
    const float u = gq.degenerate ? 0.f : __fmul_rn(__fsub_rn(zc, gq.mn), gq.inv);
    const uint32_t bits = __float_as_uint(__fadd_rn(u, 12582912.0f));
    word[w] += bits << (8 * G + 2 * r);
  }
}

// sum over the 16 (G, r) of 0x4B400000 << (8 G + 2 r), mod 2^32
__host__ __device__ constexpr uint32_t magic_sum() {
  uint32_t s = 0;
  for (int G = 0; G < 4; ++G)
    for (int r = 0; r < 4; ++r) s += 0x4B400000u << (8 * G + 2 * r);
  return s;
}

template <bool kClamp>
__global__ void __launch_bounds__(kThreads, 1)
append_tc05_kernel(const __grid_constant__ CUtensorMap tmap_k,
                   const __grid_constant__ CUtensorMap tmap_v, int n_tok,
                   const int32_t* __restrict__ cu_new,
                   const int32_t* __restrict__ pos0,
                   const int32_t* __restrict__ bt, int B, int max_pages,
                   uint8_t* __restrict__ pool, int num_pages, int h_kv,
                   const uint16_t* __restrict__ Rk_t5,
                   const uint16_t* __restrict__ Rv_t5,
                   const float* __restrict__ muR, float clip_k, float clip_v,
                   unsigned* err) {
  extern __shared__ __align__(1024) unsigned char dsm_[];
  Smem& S = *reinterpret_cast<Smem*>(dsm_);
  const int h = blockIdx.y, kind = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int tiles = (n_tok + kRows - 1) / kRows;
  const int my_tiles = tiles > (int)blockIdx.x
                           ? (tiles - 1 - (int)blockIdx.x) / (int)gridDim.x + 1
                           : 0;

  // ---- set-up (library-owned state only before pdl_wait)
  {
    const uint4* src = reinterpret_cast<const uint4*>(kind ? Rv_t5 : Rk_t5) +
                       (size_t)h * (2 * kD * kD * 2 / 16);
    uint4* dst = reinterpret_cast<uint4*>(&S.b[0][0]);
    for (int i = tid; i < 2 * kD * kD * 2 / 16; i += kThreads)
      cp_async16_zfill(dst + i, src + i, true);
    cp_async_commit();
  }
  if (tid < kD) S.mu[tid] = kind ? 0.f : __ldg(muR + h * kD + tid);
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      tc05::bar_init(&S.full[s], 1);
      tc05::bar_init(&S.empty[s], 128);
    }
    for (int g = 0; g < 2; ++g) {
      tc05::bar_init(&S.aready[g], 128);
      tc05::bar_init(&S.dready[g], 1);
    }
    // the 128-byte TMA swizzle wants 1024-byte aligned boxes
    S.abort = (tc05::smem_addr(S.stage[0]) & 1023u) != 0;
    tc05::bar_init_fence();
  }
  if (warp == kProducerWarp) tc05::tmem_alloc(&S.tmem, kTmemCols);
  pdl_wait();  // inputs and the pool may come from earlier kernels
  pdl_trigger();
  const bool cached = B <= kCuCache;
  if (cached) {
    for (int i = tid; i <= B; i += kThreads) S.cu[i] = __ldg(cu_new + i);
    for (int i = tid; i < B; i += kThreads) S.p0[i] = __ldg(pos0 + i);
  }
  cp_async_wait<0>();
  tc05::fence_proxy_async();  // R' (generic-proxy writes) -> tensor core
  tc05::fence_before();
  __syncthreads();
  tc05::fence_after();
  const uint32_t tmem = S.tmem;
  volatile int* abort = &S.abort;

  const CUtensorMap* tmap = kind ? &tmap_v : &tmap_k;
  if (warp == kProducerWarp) {
    // ---------------------------------------------------------- producer
    int last = -1;  // last tile index issued
    for (int i = 0; i < my_tiles; ++i) {
      const int s = i % kStages;
      if (i >= kStages &&
          !__all_sync(0xffffffffu, tc05::bar_wait(&S.empty[s], ((i / kStages) - 1) & 1, abort)))
        break;
      const int tok0 = ((int)blockIdx.x + i * (int)gridDim.x) * kRows;
      if (lane == 0) {
        // rows past n_tok are zero-filled; the transaction counts both boxes
        tc05::bar_arrive_expect_tx(&S.full[s], kStageBytes);
        tc05::tma_load_3d(S.stage[s], tmap, 0, h, tok0, &S.full[s]);
        tc05::tma_load_3d(S.stage[s] + kStageBytes / 2, tmap, 64, h, tok0, &S.full[s]);
      }
      __syncwarp();
      last = i;
    }
    // on abort, let the copies already issued land before the CTA exits
    for (int i = max(0, last - kStages + 1); i <= last; ++i)
      tc05::bar_wait_drain(&S.full[i % kStages], (i / kStages) & 1);
  } else if (warp == kMmaWarp) {
    // --------------------------------------------------------------- MMA
    int last = -1;
    if (lane == 0) {
      const uint32_t b0 = tc05::smem_addr(&S.b[0][0]);
      for (int i = 0; i < my_tiles; ++i) {
        const int g = i & 1;
        if (!tc05::bar_wait(&S.aready[g], (i >> 1) & 1, abort)) break;
        tc05::fence_after();
        const uint32_t d = tmem + kColD0 + 128u * g, a = tmem + kColA0 + 64u * g;
#pragma unroll
        for (int ks = 0; ks < 8; ++ks)
#pragma unroll
          for (int term = 0; term < 2; ++term)
            tc05::mma_ts(d, a + 8u * ks,
                         tc05::smem_desc(b0 + term * kD * kD * 2 + ks * 256, 128, 2048),
                         kIdesc, (ks | term) != 0);
        tc05::mma_commit(&S.dready[g]);
        last = i;
      }
      // the tensor core must be done with tensor memory before it is freed
      if (last >= 0) tc05::bar_wait_drain(&S.dready[last & 1], (last >> 1) & 1);
    }
    __syncwarp();
  } else {
    // ---------------------------------------------------------- epilogue
    const int g = warp >> 2, q = warp & 3, row = 32 * q + lane;
    const float clip = kind ? clip_v : clip_k;
    const int codes_off = kind ? OPTR_V_CODES_OFFSET : OPTR_K_CODES_OFFSET;
    const int meta_off = kind ? OPTR_V_META_OFFSET : OPTR_K_META_OFFSET;
    const uint32_t lane_base = (uint32_t)(32 * q) << 16;
    const uint32_t tA = tmem + lane_base + kColA0 + 64u * g;
    const uint32_t tD = tmem + lane_base + kColD0 + 128u * g;
    for (int i = g; i < my_tiles; i += 2) {
      const int s = i % kStages;
      const int tok = ((int)blockIdx.x + i * (int)gridDim.x) * kRows + row;
      // destination of this row's record (the block-table load overlaps
      // the copy, the conversion and the MMA)
      long long dst = -1;
      int slot = 0;
      if (tok < n_tok)
        dst = cached ? resolve_slot_cached(tok, h, S.cu, S.p0, bt, B, max_pages,
                                           num_pages, h_kv, &slot, err)
                     : resolve_slot(tok, h, cu_new, pos0, bt, B, max_pages,
                                    num_pages, h_kv, &slot, err);
      __syncwarp();  // converged for the warp-wide tensor-memory accesses
      if (!__all_sync(0xffffffffu, tc05::bar_wait(&S.full[s], (i / kStages) & 1, abort))) break;
      // the row as f16 into tensor memory: columns j <-> channels 2j, 2j+1
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const uint8_t* rb = S.stage[s] + half * (kStageBytes / 2) + row * 128;
        uint32_t a[32];
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const uint4 x = *reinterpret_cast<const uint4*>(rb + ((c ^ (row & 7)) << 4));
          a[4 * c + 0] = bf16x2_to_f16x2(x.x);
          a[4 * c + 1] = bf16x2_to_f16x2(x.y);
          a[4 * c + 2] = bf16x2_to_f16x2(x.z);
          a[4 * c + 3] = bf16x2_to_f16x2(x.w);
        }
        tc05::tmem_st32(tA + 32u * half, a);
      }
      tc05::bar_arrive(&S.empty[s]);  // stage s read (values in registers)
      tc05::tmem_wait_st();
      tc05::fence_before();
      tc05::bar_arrive(&S.aready[g]);
      if (!__all_sync(0xffffffffu, tc05::bar_wait(&S.dready[g], (i >> 1) & 1, abort))) break;
      tc05::fence_after();

      uint32_t word[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
      uint32_t meta[4];
      bool range_err = false;
#pragma unroll
      for (int G = 0; G < kGroups; ++G) {
        uint32_t acc[32];
        tc05::tmem_ld32(tD + 32u * G, acc);
        tc05::tmem_wait_ld();
        float z[32];
        const float4* mu4 = reinterpret_cast<const float4*>(S.mu + 32 * G);
#pragma unroll
        for (int j4 = 0; j4 < 8; ++j4) {  // acc / 64 is exact: one rounding, as fmul + fsub
          const float4 m = mu4[j4];
          z[4 * j4 + 0] = fmaf(__uint_as_float(acc[4 * j4 + 0]), 1.0f / 64.0f, -m.x);
          z[4 * j4 + 1] = fmaf(__uint_as_float(acc[4 * j4 + 1]), 1.0f / 64.0f, -m.y);
          z[4 * j4 + 2] = fmaf(__uint_as_float(acc[4 * j4 + 2]), 1.0f / 64.0f, -m.z);
          z[4 * j4 + 3] = fmaf(__uint_as_float(acc[4 * j4 + 3]), 1.0f / 64.0f, -m.w);
        }
        float lo = z[0], hi = z[0];
#pragma unroll
        for (int j = 1; j < 32; ++j) {
          lo = fminf(lo, z[j]);
          hi = fmaxf(hi, z[j]);
        }
        const GroupQuant gq = group_quant_params(lo, hi, clip);
        range_err |= gq.degenerate && !(fabsf(hi - lo) <= 3.402823466e38f);
        quantize_group<kClamp>(z, G, gq, word);
        const __half2 sm = __halves2half2(gq.scale, gq.min);
        meta[G] = *reinterpret_cast<const uint32_t*>(&sm);
      }
      tc05::fence_before();  // accumulator reads done before the next MMA
      if (range_err && tok < n_tok) atomicOr(err, OPTR_DEVERR_FP16_RANGE);
      if (dst >= 0) {
        constexpr uint32_t kMagic = magic_sum();
        uint4 c0, c1;
        c0.x = word[0] - kMagic; c0.y = word[1] - kMagic;
        c0.z = word[2] - kMagic; c0.w = word[3] - kMagic;
        c1.x = word[4] - kMagic; c1.y = word[5] - kMagic;
        c1.z = word[6] - kMagic; c1.w = word[7] - kMagic;
        uint8_t* rec = pool + dst;
        *reinterpret_cast<uint4*>(rec + codes_off + slot * 32) = c0;
        *reinterpret_cast<uint4*>(rec + codes_off + slot * 32 + 16) = c1;
        *reinterpret_cast<uint4*>(rec + meta_off + slot * 16) =
            make_uint4(meta[0], meta[1], meta[2], meta[3]);
      }
    }
  }

  tc05::fence_before();
  __syncthreads();
  if (S.abort && tid == 0) atomicOr(err, OPTR_DEVERR_TIMEOUT);
  if (warp == kProducerWarp) {
    tc05::fence_after();
    tc05::tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace

// cuTensorMapEncodeTiled from the driver, looked up once.
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000,
                                         cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  });
  return fn;
}

// Tensor map of x[n_tok][h_kv][128] bf16: box of 64 channels x 1 head x 128
// tokens, 128-byte swizzle, zero fill past the end.
static bool token_rows_map(CUtensorMap* m, const __nv_bfloat16* x, int n_tok, int h_kv) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[3] = {(cuuint64_t)kD, (cuuint64_t)h_kv, (cuuint64_t)n_tok};
  const cuuint64_t strides[2] = {(cuuint64_t)kD * 2, (cuuint64_t)h_kv * kD * 2};
  const cuuint32_t box[3] = {64, 1, (cuuint32_t)kRows};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<__nv_bfloat16*>(x), dims,
            strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

cudaError_t launch_append_tc05(const optr_params* p, const __nv_bfloat16* k,
                               const __nv_bfloat16* v, int n_tok,
                               const int32_t* cu_new, const int32_t* pos0,
                               const int32_t* bt, int B, int max_pages,
                               uint8_t* pool, int num_pages, cudaStream_t s) {
  const bool clamp = !(p->cfg.clip_k == 1.0f && p->cfg.clip_v == 1.0f);
  const void* fn = clamp ? reinterpret_cast<const void*>(&append_tc05_kernel<true>)
                         : reinterpret_cast<const void*>(&append_tc05_kernel<false>);
  cudaError_t e = ensure_dynamic_smem(fn, sizeof(Smem));
  if (e != cudaSuccess) return e;
  const int h_kv = p->cfg.h_kv;
  CUtensorMap mk, mv;
  if (!token_rows_map(&mk, k, n_tok, h_kv) || !token_rows_map(&mv, v, n_tok, h_kv))
    return cudaErrorInvalidValue;
  const int tiles = (n_tok + kRows - 1) / kRows;
  // one CTA per SM (the shared memory admits no second one, so tensor
  // memory is never contended), spread over the (head, kind) pairs
  int per = max(1, p->num_sms / (2 * h_kv));
  per = min(per, tiles);
  dim3 grid(per, h_kv, 2);
  if (clamp)
    return launch_pdl(append_tc05_kernel<true>, grid, dim3(kThreads), sizeof(Smem), s,
                      mk, mv, n_tok, cu_new, pos0, bt, B, max_pages, pool, num_pages,
                      h_kv, (const uint16_t*)p->Rk_t5, (const uint16_t*)p->Rv_t5,
                      (const float*)p->muR, p->cfg.clip_k, p->cfg.clip_v, p->err);
  return launch_pdl(append_tc05_kernel<false>, grid, dim3(kThreads), sizeof(Smem), s,
                    mk, mv, n_tok, cu_new, pos0, bt, B, max_pages, pool, num_pages,
                    h_kv, (const uint16_t*)p->Rk_t5, (const uint16_t*)p->Rv_t5,
                    (const float*)p->muR, p->cfg.clip_k, p->cfg.clip_v, p->err);
}

}  // namespace optr
