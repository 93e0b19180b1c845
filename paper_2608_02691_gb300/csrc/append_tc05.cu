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
//   16 epilogue warps, two groups of 8 taking alternate tiles: two threads
//                   own token row t, one per half of the channels; each
//                   converts its half row to f16 and stores it to tensor
//                   memory as the MMA's A operand, then reads its half of
//                   the accumulator row back and quantizes and packs its two
//                   channel groups; the pair's code bytes meet in shared
//                   memory and the first thread writes the 32 code bytes,
//                   each thread its 8 scale/min bytes.  A group converts its
//                   next tile while the tensor core works on the current one
//                   (two A buffers per group);
//   MMA warp        one thread issues the 16 tcgen05.mma of a tile (8
//                   K-steps x {R hi, R lo}) from tensor-memory A and
//                   shared-memory B (R, 64 KB, loaded once) into the
//                   group's tensor-memory accumulator.
// Tensor memory (512 columns): per epilogue group g an accumulator D[g]
// (128 columns, at 128 g) and two A operands (64 columns each, at
// 256 + 128 g + 64 b).
// The quantizer is quant.cuh's float32 formula.
#include "append_common.cuh"
#include "decode_common.cuh"
#include "f32x2.cuh"
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
constexpr int kEpiWarps = 16;     // two groups of 8
constexpr int kGroupThreads = 256;
constexpr int kThreads = (kEpiWarps + 2) * 32;
constexpr int kProducerWarp = kEpiWarps, kMmaWarp = kEpiWarps + 1;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColD0 = 0, kColA0 = 256;  // D[g] at 128 g, A[g][b] at 256 + 128 g + 64 b
constexpr uint32_t kIdesc = tc05::idesc_f16(128, 128);

struct Smem {
  uint16_t b[2][kD * kD];                 // R' hi, lo (64 KB)
  // token rows, bf16: [channel half][row][128 B], 16-byte chunk c of row r
  // at chunk position c ^ (r % 8) (the TMA 128-byte swizzle)
  uint8_t stage[kStages][kStageBytes];
  alignas(16) float nmu[kD];              // -mu R_k (keys) or 0 (values)
  int cu[kCuCache + 1];
  int p0[kCuCache];
  uint4 xchg[2][kRows][2];               // second-half code words per row
  // G = 128: each half row's (min, max), per tile group, tile parity, half
  float2 mmx[2][2][2 * kRows];
  uint64_t full[kStages], empty[kStages], aready[2][2], dready[2], dfree[2];
  uint64_t xready[2], xdone[2];  // the exchange slot of group g written / read
  uint64_t rready[2];            // G = 128: both halves' ranges of the tile written
  uint32_t tmem;
  int abort;
};

__device__ __forceinline__ uint32_t bf16x2_to_f16x2(uint32_t u) {
  uint32_t ls;  // u << 16 as an integer multiply (FMA pipe; the ALU pipe is the busier one)
  asm("mul.lo.u32 %0, %1, 65536;" : "=r"(ls) : "r"(u));
  const float lo = __uint_as_float(ls);
  const float hi = __uint_as_float(u & 0xffff0000u);
  uint32_t r;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// Quantizer parameters of one group (quant.cuh's formula: mn = c lo,
// mx = c hi, r = mx - mn, degenerate unless 1e-30 < r <= FLT_MAX), with the
// two divisions done as reciprocal multiplies: inv = 3 / r from rcp.approx
// (within ~2 ulp of quant.cuh's correctly rounded 3 / r, which moves only
// code decisions within ~1e-6 of a rounding boundary) and the stored scale
// fp16(r * (1/3)) (at most one fp16 ulp from fp16(r / 3)).
struct FastQuant {
  float mn, mx, inv;
  uint32_t meta;  // (scale, min) as half2
  bool degenerate;
};

__device__ __forceinline__ FastQuant fast_quant_params(float lo, float hi, float clip) {
  FastQuant q;
  q.mn = __fmul_rn(clip, lo);
  q.mx = __fmul_rn(clip, hi);
  const float r = __fsub_rn(q.mx, q.mn);
  q.degenerate = !(r > 1e-30f) || !(r <= 3.402823466e38f);
  float rc;
  asm("rcp.approx.f32 %0, %1;" : "=f"(rc) : "f"(r));
  q.inv = q.degenerate ? 0.f : __fmul_rn(3.0f, rc);
  const __half2 sm = __halves2half2(
      q.degenerate ? __float2half_rn(0.f) : __float2half_rn(__fmul_rn(r, 1.0f / 3.0f)),
      __float2half_rn(q.mn));
  q.meta = *reinterpret_cast<const uint32_t*>(&sm);
  return q;
}

// Code bytes of the 32 values x of one group: byte[w] holds the codes of
// channels 4w + r (r = 0..3) at bits 2r, in its low byte (bits 8-21 zero).
// In x's scale (mn, mx and inv scaled alike), two values per packed
// instruction:
//   d = x - mn                  rounded as quant.cuh's subtraction; in
//                               [0, r] (x lies in [mn, mx]: the group's own
//                               extremes, or clamped to them when c < 1)
//   d * inv + 1.5 * 2^23        one rounding takes d * inv (<= 3 + 2^-20)
//                               to the nearest integer (ties to even, as
//                               rint) in the low mantissa bits:
//                               bits = 0x4B400000 + code, code <= 3
// and sum_r bits_r 4^r = 85 * 0x4B400000 + byte, whose constant part lies
// above bit 21.  Rounding d * inv once instead of twice (to float, then to
// an integer) moves only decisions within ~2e-7 of a rounding boundary.
// A degenerate group (also any group holding a NaN or infinity: the
// rotation spreads one to every channel of the row) gets code 0 throughout.
template <bool kClamp>
__device__ __forceinline__ void code_bytes(const float (&x)[32], const FastQuant& q,
                                           uint32_t (&byte)[8]) {
  if (q.degenerate) {
#pragma unroll
    for (int w = 0; w < 8; ++w) byte[w] = 0u;
    return;
  }
  const float2 mn2 = make_float2(q.mn, q.mn), inv2 = make_float2(q.inv, q.inv);
  const float2 mag2 = make_float2(12582912.0f, 12582912.0f);
  auto xc = [&](int j) { return kClamp ? fminf(fmaxf(x[j], q.mn), q.mx) : x[j]; };
#pragma unroll
  for (int w = 0; w < 8; ++w) {
    const float2 b01 = fma2(sub2(make_float2(xc(4 * w), xc(4 * w + 1)), mn2), inv2, mag2);
    const float2 b23 = fma2(sub2(make_float2(xc(4 * w + 2), xc(4 * w + 3)), mn2), inv2, mag2);
    byte[w] = __float_as_uint(b01.x) + 4u * __float_as_uint(b01.y) +
              16u * __float_as_uint(b23.x) + 64u * __float_as_uint(b23.y);
  }
}

// Smallest and largest of 32 values (NaNs ignored): four interleaved
// chains per extreme, two new values per 3-input min/max.
__device__ __forceinline__ void minmax32(const float (&x)[32], float& lo, float& hi) {
  float l[4], h[4];
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    l[c] = fminf(x[c], x[c + 4]);
    h[c] = fmaxf(x[c], x[c + 4]);
  }
#pragma unroll
  for (int j = 8; j < 32; j += 8)
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      l[c] = fminf(l[c], fminf(x[j + c], x[j + c + 4]));
      h[c] = fmaxf(h[c], fmaxf(x[j + c], x[j + c + 4]));
    }
  lo = fminf(fminf(l[0], l[1]), fminf(l[2], l[3]));
  hi = fmaxf(fmaxf(h[0], h[1]), fmaxf(h[2], h[3]));
}

template <bool kClamp, bool kG128>
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
  if (tid < kD) S.nmu[tid] = kind ? 0.f : -__ldg(muR + h * kD + tid);
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      tc05::bar_init(&S.full[s], 1);
      tc05::bar_init(&S.empty[s], kGroupThreads);
    }
    for (int g = 0; g < 2; ++g) {
      tc05::bar_init(&S.aready[g][0], kGroupThreads);
      tc05::bar_init(&S.aready[g][1], kGroupThreads);
      tc05::bar_init(&S.dready[g], 1);
      tc05::bar_init(&S.dfree[g], kGroupThreads);
      tc05::bar_init(&S.xready[g], kGroupThreads / 2);
      tc05::bar_init(&S.xdone[g], kGroupThreads / 2);
      tc05::bar_init(&S.rready[g], kGroupThreads);
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
        // tile i is the k-th of group g, its A operand in buffer k % 2; the
        // group's previous tile must have been read out of D[g]
        const int g = i & 1, k = i >> 1;
        if (!tc05::bar_wait(&S.aready[g][k & 1], (k >> 1) & 1, abort)) break;
        if (k > 0 && !tc05::bar_wait(&S.dfree[g], (k - 1) & 1, abort)) break;
        tc05::fence_after();
        const uint32_t d = tmem + kColD0 + 128u * g,
                       a = tmem + kColA0 + 128u * g + 64u * (k & 1);
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
    // warp w: group g = w / 8; lane quarter q = w % 4 (its tensor-memory
    // lanes); channel half hp = (w / 4) % 2, i.e. channel groups 2hp, 2hp+1
    const int g = warp >> 3, q = warp & 3, hp = (warp >> 2) & 1, row = 32 * q + lane;
    const float clip = kind ? clip_v : clip_k;
    const int codes_off = kind ? OPTR_V_CODES_OFFSET : OPTR_K_CODES_OFFSET;
    // G = 128: the compact record, one (scale, min) pair per slot
    const int meta_off = kind ? vmeta_offset(kG128) : OPTR_K_META_OFFSET;
    const uint32_t lane_base = (uint32_t)(32 * q) << 16;
    const uint32_t tD = tmem + lane_base + kColD0 + 128u * g;
    const int n_mine = my_tiles > g ? (my_tiles - 1 - g) / 2 + 1 : 0;
    auto token = [&](int k) {
      return ((int)blockIdx.x + (g + 2 * k) * (int)gridDim.x) * kRows + row;
    };
    // destination of this row's record in the group's k-th tile (the
    // block-table load completes during the conversion and the MMA)
    auto resolve = [&](int k, int& slot) -> long long {
      const int tok = token(k);
      long long d = -1;
      if (tok < n_tok)
        d = cached ? resolve_slot_cached(tok, h, S.cu, S.p0, bt, B, max_pages,
                                         num_pages, h_kv, &slot, err, chunk_bytes(kG128))
                   : resolve_slot(tok, h, cu_new, pos0, bt, B, max_pages,
                                  num_pages, h_kv, &slot, err, chunk_bytes(kG128));
      __syncwarp();  // converged for the warp-wide tensor-memory accesses
      return d;
    };
    // the row of the group's k-th tile as f16 into A buffer k % 2:
    // columns j <-> channels 2j, 2j+1
    auto convert = [&](int k) -> bool {
      const int i = g + 2 * k, s = i % kStages;
      if (!__all_sync(0xffffffffu, tc05::bar_wait(&S.full[s], (i / kStages) & 1, abort)))
        return false;
      const uint32_t tA = tmem + lane_base + kColA0 + 128u * g + 64u * (k & 1) + 32u * hp;
      {
        const uint8_t* rb = S.stage[s] + hp * (kStageBytes / 2) + row * 128;
        uint32_t a[32];
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const uint4 x = *reinterpret_cast<const uint4*>(rb + ((c ^ (row & 7)) << 4));
          a[4 * c + 0] = bf16x2_to_f16x2(x.x);
          a[4 * c + 1] = bf16x2_to_f16x2(x.y);
          a[4 * c + 2] = bf16x2_to_f16x2(x.z);
          a[4 * c + 3] = bf16x2_to_f16x2(x.w);
        }
        tc05::tmem_st32(tA, a);
      }
      tc05::bar_arrive(&S.empty[s]);  // stage s read (values in registers)
      tc05::tmem_wait_st();
      tc05::fence_before();
      tc05::bar_arrive(&S.aready[g][k & 1]);
      return true;
    };

    int slot_next = 0;
    long long dst_next = n_mine > 0 ? resolve(0, slot_next) : -1;
    bool ok = n_mine == 0 || convert(0);
    for (int k = 0; ok && k < n_mine; ++k) {
      const long long dst = dst_next;
      const int slot = slot_next;
      const int tok = token(k);
      if (k + 1 < n_mine) {
        dst_next = resolve(k + 1, slot_next);
        if (!convert(k + 1)) break;
      }
      if (!__all_sync(0xffffffffu, tc05::bar_wait(&S.dready[g], k & 1, abort))) break;
      tc05::fence_after();

      uint32_t word[8];
      uint32_t meta[2];
      bool range_err = false;
      {
        const int G2 = 2 * hp;  // this thread's two channel groups
        uint32_t acc[2][32];
        tc05::tmem_ld32(tD + 32u * G2, acc[0]);
        tc05::tmem_ld32(tD + 32u * (G2 + 1), acc[1]);
        tc05::tmem_wait_ld();
        if constexpr (!kG128) {
          tc05::fence_before();
          tc05::bar_arrive(&S.dfree[g]);  // D[g] read: the next MMA may start
        }
        uint32_t bytes[2][8];
        const float xs = kind ? 64.0f : 1.0f;  // x = xs * z
        // x = z = acc / 64 - mu R (keys; acc / 64 is exact, so one
        // rounding as fmul + fsub), or x = acc = 64 z (values, mu = 0: the
        // group's range and codes are then taken in units of z / 64,
        // exactly)
        auto row_values = [&](int e, const uint32_t (&a)[32], float (&x)[32]) {
          const int G = G2 + e;
          if (kind == 0) {
            const float4* nmu4 = reinterpret_cast<const float4*>(S.nmu + 32 * G);
            const float2 s64 = make_float2(1.0f / 64.0f, 1.0f / 64.0f);
#pragma unroll
            for (int j4 = 0; j4 < 8; ++j4) {
              const float4 m = nmu4[j4];
              const float2 x01 = fma2(make_float2(__uint_as_float(a[4 * j4 + 0]),
                                                  __uint_as_float(a[4 * j4 + 1])),
                                      s64, make_float2(m.x, m.y));
              const float2 x23 = fma2(make_float2(__uint_as_float(a[4 * j4 + 2]),
                                                  __uint_as_float(a[4 * j4 + 3])),
                                      s64, make_float2(m.z, m.w));
              x[4 * j4 + 0] = x01.x;
              x[4 * j4 + 1] = x01.y;
              x[4 * j4 + 2] = x23.x;
              x[4 * j4 + 3] = x23.y;
            }
          } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) x[j] = __uint_as_float(a[j]);
          }
        };
        auto scaled_params = [&](float lo, float hi) {
          FastQuant q = fast_quant_params(lo * (1.0f / xs), hi * (1.0f / xs), clip);
          range_err |= q.degenerate && !(fabsf(hi - lo) <= 3.402823466e38f);
          q.mn *= xs;
          q.mx *= xs;
          q.inv *= 1.0f / xs;
          return q;
        };
        if constexpr (kG128) {
          // one range over the row's 128 channels: this half's two groups,
          // then the partner half's through shared memory (double-buffered
          // by tile parity; a buffer is rewritten two tiles later, after
          // the partner's arrival for the tile in between, i.e. after its
          // read)
          // (the accumulator is read again from tensor memory after the
          // exchange, so no registers hold it meanwhile; D[g] is released
          // after that second read)
          float lo, hi;
          {
            float x[32], l1, h1;
            row_values(0, acc[0], x);
            minmax32(x, lo, hi);
            row_values(1, acc[1], x);
            minmax32(x, l1, h1);
            lo = fminf(lo, l1);
            hi = fmaxf(hi, h1);
          }
          float2* mm = S.mmx[g][k & 1];
          mm[hp * kRows + row] = make_float2(lo, hi);
          tc05::bar_arrive(&S.rready[g]);
          if (!__all_sync(0xffffffffu, tc05::bar_wait(&S.rready[g], k & 1, abort))) break;
          const float2 o = mm[(1 - hp) * kRows + row];
          const FastQuant q = scaled_params(fminf(lo, o.x), fmaxf(hi, o.y));
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            uint32_t a2[32];
            tc05::tmem_ld32(tD + 32u * (G2 + e), a2);
            tc05::tmem_wait_ld();
            float x[32];
            row_values(e, a2, x);
            code_bytes<kClamp>(x, q, bytes[e]);
            meta[e] = q.meta;
          }
          tc05::fence_before();
          tc05::bar_arrive(&S.dfree[g]);  // D[g] read: the next MMA may start
        } else {
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            float x[32];
            row_values(e, acc[e], x);
            float lo, hi;
            minmax32(x, lo, hi);
            const FastQuant q = scaled_params(lo, hi);
            code_bytes<kClamp>(x, q, bytes[e]);
            meta[e] = q.meta;
          }
        }
        // byte 0 of bytes[0][w] / bytes[1][w] to bytes 2hp, 2hp + 1 of the
        // word (byte 1 of bytes[0][w] is zero)
        const uint32_t sel = hp ? 0x4011u : 0x1140u;
#pragma unroll
        for (int w = 0; w < 8; ++w) word[w] = __byte_perm(bytes[0][w], bytes[1][w], sel);
      }
      if (range_err && tok < n_tok) atomicOr(err, OPTR_DEVERR_FP16_RANGE);
      // the second half's code bytes to its partner, through shared memory
      uint4* xw = S.xchg[g][row];
      if (hp) {
        // the partner has read this slot's previous contents
        if (k > 0 && !__all_sync(0xffffffffu, tc05::bar_wait(&S.xdone[g], (k - 1) & 1, abort)))
          break;
        xw[0] = make_uint4(word[0], word[1], word[2], word[3]);
        xw[1] = make_uint4(word[4], word[5], word[6], word[7]);
        tc05::bar_arrive(&S.xready[g]);
      } else {
        if (!__all_sync(0xffffffffu, tc05::bar_wait(&S.xready[g], k & 1, abort))) break;
        const uint4 y0 = xw[0], y1 = xw[1];
        tc05::bar_arrive(&S.xdone[g]);
        word[0] |= y0.x; word[1] |= y0.y; word[2] |= y0.z; word[3] |= y0.w;
        word[4] |= y1.x; word[5] |= y1.y; word[6] |= y1.z; word[7] |= y1.w;
      }
      if (dst >= 0) {
        uint8_t* rec = pool + dst;
        if (!hp) {
          *reinterpret_cast<uint4*>(rec + codes_off + slot * 32) =
              make_uint4(word[0], word[1], word[2], word[3]);
          *reinterpret_cast<uint4*>(rec + codes_off + slot * 32 + 16) =
              make_uint4(word[4], word[5], word[6], word[7]);
        }
        if constexpr (kG128) {
          // both half-row threads hold the group's one pair after the
          // range exchange; the first writes it
          if (!hp) *reinterpret_cast<uint32_t*>(rec + meta_off + slot * 4) = meta[0];
        } else {
          *reinterpret_cast<uint2*>(rec + meta_off + slot * 16 + 8 * hp) =
              make_uint2(meta[0], meta[1]);
        }
      }
      __syncwarp();
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
  const bool g128 = p->cfg.group == 4 * kG;
  auto fn = clamp ? (g128 ? append_tc05_kernel<true, true> : append_tc05_kernel<true, false>)
                  : (g128 ? append_tc05_kernel<false, true> : append_tc05_kernel<false, false>);
  cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(fn), sizeof(Smem));
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
  return launch_pdl(fn, grid, dim3(kThreads), sizeof(Smem), s,
                    mk, mv, n_tok, cu_new, pos0, bt, B, max_pages, pool, num_pages,
                    h_kv, (const uint16_t*)p->Rk_t5, (const uint16_t*)p->Rv_t5,
                    (const float*)p->muR, p->cfg.clip_k, p->cfg.clip_v, p->err);
}

}  // namespace optr

namespace optr {
namespace {

// Self-test of the bounded waits of the tcgen05 kernels: the exit path of
// append_tc05_kernel run against an mbarrier phase that nothing completes.
// Warp 0 allocates the same tensor-memory columns as the cache write; every
// warp waits with the given limit, which runs out; the CTA then takes the
// cache write's exit sequence (flag OPTR_DEVERR_TIMEOUT, free the columns).
__global__ void __launch_bounds__(128, 1)
tc05_wait_selftest_kernel(unsigned* err, unsigned long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ uint32_t tmem;
  __shared__ int abort;
  const int tid = threadIdx.x, warp = tid >> 5;
  if (tid == 0) {
    tc05::bar_init(&bar, 1);  // one arrival completes the phase; none comes
    abort = 0;
    tc05::bar_init_fence();
  }
  if (warp == 0) tc05::tmem_alloc(&tmem, kTmemCols);
  tc05::fence_before();
  __syncthreads();
  tc05::fence_after();
  const uint32_t base = tmem;
  volatile int* ab = &abort;
  // each warp waits (all its lanes agree), as the cache write's warps do
  __all_sync(0xffffffffu, tc05::bar_wait(&bar, 0, ab, limit_ns));
  tc05::fence_before();
  __syncthreads();
  if (abort && tid == 0) atomicOr(err, OPTR_DEVERR_TIMEOUT);
  if (warp == 0) {
    tc05::fence_after();
    tc05::tmem_dealloc(base, kTmemCols);
  }
}

}  // namespace
}  // namespace optr

extern "C" optr_status optr_selftest_wait_timeout(const optr_params* p,
                                                  unsigned long long limit_ns,
                                                  cudaStream_t stream) {
  if (!p || limit_ns < 1000000ull || limit_ns > 2000000000ull)
    return OPTR_ERR_INVALID_ARG;
  optr::tc05_wait_selftest_kernel<<<1, 128, 0, stream>>>(p->err, limit_ns);
  return cudaGetLastError() == cudaSuccess ? OPTR_OK : OPTR_ERR_CUDA;
}
