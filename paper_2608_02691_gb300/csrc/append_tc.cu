// Tensor-core cache write (paper Sec. 4.1; Appendix "Key-mean estimation
// and application": z_K = k R_K - mu R_K, z_V = v R_V, then group-wise INT2).
//
// The rotation is a dense GEMM per KV head, Z[tok][128] = X[tok][128] R[128][128],
// run on mma.sync.m16n8k16 (f16 inputs, f32 accumulate).  X (bf16) converts
// to f16 exactly within fp16's range; R is prescaled by 2^6 and split into
// fp16 hi + lo, so the products carry ~22 bits of R and the float32 result
// matches a float32 CUDA-core rotation to rounding.  One warp computes a
// 16-token tile against all 128 rotated channels (16 n-tiles x 8 k-steps x
// {hi, lo} = 256 MMAs); the B fragments of R (64 KB per head and K/V) are
// staged in shared memory once per CTA.
//
// B columns are permuted so that the C fragment's columns 2c, 2c+1 of the 16
// n-tiles hand lane c exactly the 32 channels of group c: the group min/max
// and the codes are then computed without any shuffle, in the same float32
// formula as the CUDA-core kernel (quant.cuh).
#include "append_common.cuh"
#include "decode_common.cuh"
#include "quant.cuh"

namespace optr {

// Host: B fragments of one rotation R (row-major float32 [128][128]) for
// mma.m16n8k16 row.col: [k-step 8][n-tile 16][lane 32][4 words], the words
// being (hi b0, hi b1, lo b0, lo b1).  Lane (g, c) holds column n = g and
// rows k = 2c, 2c+1 (b0) and 2c+8, 2c+9 (b1) of the 16x8 tile; column n of
// n-tile nt is rotated channel 32*(n/2) + 2*nt + n%2.
void build_rotation_fragments(const float* R, uint32_t* out) {
  auto h16 = [](float x) -> uint32_t {
    __half_raw r = __half(__float2half_rn(x));
    return r.x;
  };
  auto f16 = [](uint32_t bits) -> float {
    __half_raw r;
    r.x = (unsigned short)bits;
    return __half2float(__half(r));
  };
  for (int ks = 0; ks < 8; ++ks)
    for (int nt = 0; nt < 16; ++nt)
      for (int lane = 0; lane < 32; ++lane) {
        const int g = lane >> 2, c = lane & 3;
        const int ch = 32 * (g >> 1) + 2 * nt + (g & 1);
        uint32_t w[4];
        for (int which = 0; which < 2; ++which) {
          const int k0 = 16 * ks + 2 * c + 8 * which;
          uint32_t hi[2], lo[2];
          for (int e = 0; e < 2; ++e) {
            const float x = R[(size_t)(k0 + e) * kD + ch] * 64.0f;
            hi[e] = h16(x);
            lo[e] = h16(x - f16(hi[e]));
          }
          w[which] = hi[0] | (hi[1] << 16);
          w[2 + which] = lo[0] | (lo[1] << 16);
        }
        uint32_t* o = out + (((size_t)ks * 16 + nt) * 32 + lane) * 4;
        for (int i = 0; i < 4; ++i) o[i] = w[i];
      }
}

namespace {

constexpr int kAppendWarps = 4;
constexpr int kTile = 16;  // tokens per warp tile

constexpr int kXPitch = kD + 8;  // padded row (272 B): conflict-free ldmatrix

struct AppendWarpSmem {
  alignas(16) __nv_bfloat16 x[kTile][kXPitch];  // one K or V tile
  alignas(16) uint8_t codes[kTile][32];    // packed codes of the tile
};

__device__ __forceinline__ void ldsm_x4(uint32_t& r0, uint32_t& r1,
                                        uint32_t& r2, uint32_t& r3,
                                        const void* smem_row) {
  const unsigned a = static_cast<unsigned>(__cvta_generic_to_shared(smem_row));
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(a));
}

__device__ __forceinline__ void mma16816(float* d, const uint32_t* a,
                                         uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// bf16 pair -> fp16 pair (exact within fp16's normal range).
__device__ __forceinline__ uint32_t bf16x2_to_f16x2(uint32_t u) {
  const float lo = __uint_as_float(u << 16);
  const float hi = __uint_as_float(u & 0xffff0000u);
  uint32_t r;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

__global__ void __launch_bounds__(kAppendWarps * 32, 2)
append_tensor_kernel(const __nv_bfloat16* __restrict__ k,
                     const __nv_bfloat16* __restrict__ v, int n_tok,
                     const int32_t* __restrict__ cu_new,
                     const int32_t* __restrict__ pos0,
                     const int32_t* __restrict__ bt, int B, int max_pages,
                     uint8_t* __restrict__ pool, int num_pages, int h_kv,
                     const uint32_t* __restrict__ Rk_tc,
                     const uint32_t* __restrict__ Rv_tc,
                     const float* __restrict__ muR, float clip_k, float clip_v,
                     unsigned* err) {
  extern __shared__ uint4 bfrag[];  // [8][16][32] uint4 = 64 KB
  __shared__ AppendWarpSmem wsm[kAppendWarps];
  __shared__ float smu[kD];
  const int h = blockIdx.y, kind = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, c = lane & 3;
  {
    const uint4* src = reinterpret_cast<const uint4*>(kind ? Rv_tc : Rk_tc) +
                       (size_t)h * (kRFragWords / 4);
    for (int i = tid; i < kRFragWords / 4; i += kAppendWarps * 32)
      cp_async16_zfill(&bfrag[i], &src[i], true);
    cp_async_commit();
    smu[tid] = kind ? 0.f : __ldg(muR + h * kD + tid);
    pdl_wait();  // inputs and the pool may come from earlier kernels
    pdl_trigger();
    cp_async_wait<0>();
    __syncthreads();
  }
  AppendWarpSmem& W = wsm[warp];
  const __nv_bfloat16* X = kind ? v : k;
  const float clip = kind ? clip_v : clip_k;
  const int codes_off = kind ? OPTR_V_CODES_OFFSET : OPTR_K_CODES_OFFSET;
  const int meta_off = kind ? OPTR_V_META_OFFSET : OPTR_K_META_OFFSET;
  const int tiles = (n_tok + kTile - 1) / kTile;

  for (int t = blockIdx.x * kAppendWarps + warp; t < tiles;
       t += gridDim.x * kAppendWarps) {
    const int tok0 = t * kTile;
    // stage the tile: 16 rows x 256 B = 256 chunks of 16 B, 8 per lane
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int idx = lane + 32 * j, row = idx >> 4, col = (idx & 15) * 8;
      const int tok = tok0 + row;
      const bool ok = tok < n_tok;
      cp_async16_zfill(&W.x[row][col],
                       X + ((size_t)(ok ? tok : 0) * h_kv + h) * kD + col, ok);
    }
    cp_async_commit();
    // destination of token tok0 + lane (lanes 0..15), during the copy
    long long dst = -1;
    int slot = 0;
    if (lane < kTile && tok0 + lane < n_tok)
      dst = resolve_slot(tok0 + lane, h, cu_new, pos0, bt, B, max_pages,
                         num_pages, h_kv, &slot, err);
    cp_async_wait<0>();
    __syncwarp();

    float acc[16][4];
#pragma unroll
    for (int nt = 0; nt < 16; ++nt)
#pragma unroll
      for (int i = 0; i < 4; ++i) acc[nt][i] = 0.f;
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
      uint32_t a[4];
      ldsm_x4(a[0], a[1], a[2], a[3], &W.x[lane & 15][ks * 16 + (lane >> 4) * 8]);
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = bf16x2_to_f16x2(a[i]);
#pragma unroll
      for (int nt = 0; nt < 16; ++nt) {
        const uint4 bf = bfrag[(ks * 16 + nt) * 32 + lane];
        mma16816(acc[nt], a, bf.x, bf.y);
        mma16816(acc[nt], a, bf.z, bf.w);
      }
    }

    // epilogue: lane (g, c) holds channels 32c + 2nt + e of tokens g (e =
    // 0, 1 -> acc[nt][e]) and g + 8 (acc[nt][2 + e]): all of group c
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int row = g + 8 * half;
      float z[32];
#pragma unroll
      for (int nt = 0; nt < 16; ++nt)
#pragma unroll
        for (int e = 0; e < 2; ++e)
          z[2 * nt + e] = __fsub_rn(__fmul_rn(acc[nt][2 * half + e], 1.0f / 64.0f),
                                    smu[32 * c + 2 * nt + e]);
      float lo = z[0], hi = z[0];
#pragma unroll
      for (int i = 1; i < 32; ++i) {
        lo = fminf(lo, z[i]);
        hi = fmaxf(hi, z[i]);
      }
      const GroupQuant gq = group_quant_params(lo, hi, clip);
      if (gq.degenerate && !(fabsf(hi - lo) <= 3.402823466e38f) && tok0 + row < n_tok)
        atomicOr(err, OPTR_DEVERR_FP16_RANGE);
#pragma unroll
      for (int w = 0; w < 8; ++w) {
        uint32_t byte = 0;
#pragma unroll
        for (int r = 0; r < 4; ++r) byte |= (uint32_t)quant_code(z[4 * w + r], gq) << (2 * r);
        W.codes[row][4 * w + c] = (uint8_t)byte;
      }
      const long long drow = __shfl_sync(0xffffffffu, dst, row);
      const int srow = __shfl_sync(0xffffffffu, slot, row);
      if (drow >= 0)
        *reinterpret_cast<__half2*>(pool + drow + meta_off + srow * 16 + 4 * c) =
            __halves2half2(gq.scale, gq.min);
    }
    __syncwarp();
    {
      const int row = lane >> 1, part = lane & 1;
      const long long drow = __shfl_sync(0xffffffffu, dst, row);
      const int srow = __shfl_sync(0xffffffffu, slot, row);
      if (drow >= 0)
        *reinterpret_cast<uint4*>(pool + drow + codes_off + srow * 32 + 16 * part) =
            *reinterpret_cast<const uint4*>(&W.codes[row][16 * part]);
    }
    __syncwarp();
  }
}

}  // namespace

cudaError_t launch_append_tensor(const optr_params* p, const __nv_bfloat16* k,
                                 const __nv_bfloat16* v, int n_tok,
                                 const int32_t* cu_new, const int32_t* pos0,
                                 const int32_t* bt, int B, int max_pages,
                                 uint8_t* pool, int num_pages, cudaStream_t s) {
  const int smem = kRFragWords * 4;  // 64 KB of B fragments
  cudaError_t e = ensure_dynamic_smem(
      reinterpret_cast<const void*>(&append_tensor_kernel), smem);
  if (e != cudaSuccess) return e;
  const int h_kv = p->cfg.h_kv;
  const int tiles = (n_tok + kTile - 1) / kTile;
  int per_hk = max(1, (2 * p->num_sms) / (2 * h_kv));
  per_hk = min(per_hk, (tiles + kAppendWarps - 1) / kAppendWarps);
  dim3 grid(per_hk, h_kv, 2);
  return launch_pdl(append_tensor_kernel, grid, dim3(kAppendWarps * 32),
                    (size_t)smem, s, k, v, n_tok, cu_new, pos0, bt, B,
                    max_pages, pool, num_pages, h_kv, p->Rk_tc, p->Rv_tc,
                    p->muR, p->cfg.clip_k, p->cfg.clip_v, p->err);
}

}  // namespace optr
