// Single-token cache write body (decode steps), shared by the stand-alone
// kernel in append.cu and the fused decode-step prologue in decode.cu.
#pragma once

#include "optr_internal.cuh"
#include "quant.cuh"
#include "append_common.cuh"

namespace optr {

// Decode-step variant for few new tokens (one per sequence per step): one
// CTA per (tile of T tokens, KV head, K or V), 512 threads = 4 slices x 128
// channels.  Slice s accumulates z_j over i in [32s, 32s+32) for all T
// tokens; the slices are added in shared memory, then warp t quantizes and
// packs token t group by group.  T = 4 for at most 64 new tokens (4x the
// CTAs, a quarter of the FMAs per thread: the decode step's latency), else
// 16.
constexpr int kSmallTok = 16;
constexpr int kSmallTokFew = 4;
constexpr int kSmallCuCache = 512;   // sequences whose cu_new / pos0 a CTA caches

__host__ __device__ constexpr int small_tile(int n_tok) {
  return n_tok <= 64 ? kSmallTokFew : kSmallTok;
}

template <int T>
struct AppendSmallSmemT {
  float xs[T][kD];
  float zp[4][T][kD];
  long long dst[T];
  int dslot[T];
  int s_cu[kSmallCuCache + 1];
  int s_p0[kSmallCuCache];
};
using AppendSmallSmem = AppendSmallSmemT<kSmallTok>;  // the larger one

// CTA (tblk, h, kind) of the cache write: tokens [T*tblk, T*tblk + T),
// KV head h, kind 0 = keys, 1 = values.  512 threads.
template <int T>
__device__ __forceinline__ void append_small_body(
    int tblk, int h, int kind, AppendSmallSmemT<T>& sm,
    const __nv_bfloat16* __restrict__ k, const __nv_bfloat16* __restrict__ v,
    int n_tok, const int32_t* __restrict__ cu_new,
    const int32_t* __restrict__ pos0, const int32_t* __restrict__ bt, int B,
    int max_pages, uint8_t* __restrict__ pool, int num_pages, int h_kv,
    const float* __restrict__ R_k, const float* __restrict__ R_v,
    const float* __restrict__ muR, float clip_k, float clip_v, unsigned* err,
    bool identity = false, bool group128 = false) {
  // identity: z = x, no rotation (values with the rotation folded into the
  // model's projections); group128: Q2 groups of all 128 channels (the
  // pair is stored in each of the four 32-channel metadata entries)
  static_assert(T <= 16, "one quantizing warp per token");
  float (&xs)[T][kD] = sm.xs;
  float (&zp)[4][T][kD] = sm.zp;
  long long (&dst)[T] = sm.dst;
  int (&dslot)[T] = sm.dslot;
  int (&s_cu)[kSmallCuCache + 1] = sm.s_cu;
  int (&s_p0)[kSmallCuCache] = sm.s_p0;
  const int t0 = tblk * T;
  const int tid = threadIdx.x;
  const int sl = tid >> 7, j = tid & 127;
  // rotation column first (independent of everything else): all in flight
  const float* R = (kind ? R_v : R_k) + (size_t)h * kD * kD + (size_t)(32 * sl) * kD + j;
  float rv[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) rv[i] = identity ? 0.f : __ldg(R + i * kD);
  float musub[kGroups];  // mu R_k of this lane's channel in each group (keys)
#pragma unroll
  for (int g = 0; g < kGroups; ++g)
    musub[g] = kind ? 0.f : __ldg(muR + h * kD + 32 * g + (tid & 31));
  pdl_wait();  // inputs and the pool may come from earlier kernels
  pdl_trigger();
  const __nv_bfloat16* src = kind ? v : k;
  for (int idx = tid; idx < T * kD; idx += 512) {
    const int t = idx >> 7, i = idx & 127;
    const int tok = t0 + t;
    xs[t][i] = tok < n_tok ? __bfloat162float(src[((size_t)tok * h_kv + h) * kD + i]) : 0.f;
  }
  const bool cached = B <= kSmallCuCache;
  if (cached) {
    for (int i = tid; i <= B; i += 512) {
      s_cu[i] = __ldg(cu_new + i);
      if (i < B) s_p0[i] = __ldg(pos0 + i);
    }
  }
  __syncthreads();
  // Slot of token t0 + tid (threads < T), in two halves around the
  // rotation: the block-table entry is requested here and checked after the
  // FMAs, so its load latency overlaps them (resolve_slot's checks).
  const int my_tok = t0 + tid;
  const bool resolver = tid < T && my_tok < n_tok;
  long long off = -1;
  int slot = 0, page = -1;
  unsigned bad = 0;
  if (resolver) {
    if (cached) {
      int lo = 0, hi = B;
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (s_cu[mid] <= my_tok) lo = mid; else hi = mid;
      }
      const int c0 = s_cu[lo], c1 = s_cu[lo + 1];
      if (!(c0 <= my_tok && my_tok < c1)) {
        bad = OPTR_DEVERR_CU_NEW;
      } else {
        const long long pos = (long long)s_p0[lo] + (my_tok - c0);
        if (pos < 0 || pos >= (long long)max_pages * kPage) {
          bad = OPTR_DEVERR_POSITION;
        } else {
          slot = (int)(pos % kPage);
          page = __ldg(bt + (size_t)lo * max_pages + pos / kPage);
        }
      }
    } else {
      off = resolve_slot(my_tok, h, cu_new, pos0, bt, B, max_pages, num_pages,
                         h_kv, &slot, err, chunk_bytes(group128));
    }
  }
  if (identity) {
#pragma unroll
    for (int t = 0; t < T; ++t) zp[sl][t][j] = sl == 0 ? xs[t][j] : 0.f;
  } else {
    float acc[T];
#pragma unroll
    for (int t = 0; t < T; ++t) acc[t] = 0.f;
#pragma unroll
    for (int i = 0; i < 32; ++i)
#pragma unroll
      for (int t = 0; t < T; ++t) acc[t] = fmaf(xs[t][32 * sl + i], rv[i], acc[t]);
#pragma unroll
    for (int t = 0; t < T; ++t) zp[sl][t][j] = acc[t];
  }
  if (tid < T) {
    if (resolver && cached) {
      if (bad) {
        atomicOr(err, bad);
      } else if (page < 0 || page >= num_pages) {
        atomicOr(err, OPTR_DEVERR_PAGE_ID);
      } else {
        off = ((long long)page * h_kv + h) * chunk_bytes(group128);
      }
    }
    dst[tid] = off;
    dslot[tid] = slot;
  }
  __syncthreads();

  const int warp = tid >> 5, lane = tid & 31;  // warp = token of the tile
  if (warp >= T) return;
  const long long woff = dst[warp];
  if (t0 + warp >= n_tok || woff < 0) return;
  const int wslot = dslot[warp];
  const float clip = kind ? clip_v : clip_k;
  const int codes_off = kind ? OPTR_V_CODES_OFFSET : OPTR_K_CODES_OFFSET;
  // G = 128: the compact record, one (scale, min) pair per slot
  const int meta_off = kind ? vmeta_offset(group128) : OPTR_K_META_OFFSET;
  uint8_t* chunk = pool + woff;
  float zv[kGroups];
#pragma unroll
  for (int g = 0; g < kGroups; ++g) {
    const int jj = 32 * g + lane;
    const float zsum = ((zp[0][warp][jj] + zp[1][warp][jj]) + zp[2][warp][jj]) + zp[3][warp][jj];
    zv[g] = __fsub_rn(zsum, musub[g]);
  }
  // G = 128: one range over the four blocks of 32 channels
  GroupQuant g128;
  if (group128) {
    float lo = fminf(fminf(zv[0], zv[1]), fminf(zv[2], zv[3]));
    float hi = fmaxf(fmaxf(zv[0], zv[1]), fmaxf(zv[2], zv[3]));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
      hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    g128 = group_quant_params(lo, hi, clip);
  }
  // the four groups' range reductions, parameters and codes interleaved
  // (four independent shuffle chains instead of one after another)
  GroupQuant gq[kGroups];
  if (group128) {
#pragma unroll
    for (int g = 0; g < kGroups; ++g) gq[g] = g128;
  } else {
    float lo[kGroups], hi[kGroups];
#pragma unroll
    for (int g = 0; g < kGroups; ++g) lo[g] = hi[g] = zv[g];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
#pragma unroll
      for (int g = 0; g < kGroups; ++g) {
        lo[g] = fminf(lo[g], __shfl_xor_sync(0xffffffffu, lo[g], o));
        hi[g] = fmaxf(hi[g], __shfl_xor_sync(0xffffffffu, hi[g], o));
      }
#pragma unroll
    for (int g = 0; g < kGroups; ++g) gq[g] = group_quant_params(lo[g], hi[g], clip);
  }
  unsigned bits[kGroups];
#pragma unroll
  for (int g = 0; g < kGroups; ++g) bits[g] = (unsigned)quant_code(zv[g], gq[g]) << (2 * (lane & 3));
#pragma unroll
  for (int g = 0; g < kGroups; ++g) bits[g] |= __shfl_xor_sync(0xffffffffu, bits[g], 1);
#pragma unroll
  for (int g = 0; g < kGroups; ++g) bits[g] |= __shfl_xor_sync(0xffffffffu, bits[g], 2);
#pragma unroll
  for (int g = 0; g < kGroups; ++g) {
    if ((lane & 3) == 0)
      chunk[codes_off + wslot * 32 + 4 * (lane >> 2) + g] = (uint8_t)bits[g];
    if (lane == 0 && (!group128 || g == 0))
      *reinterpret_cast<__half2*>(chunk + meta_off + wslot * meta_stride(group128) +
                                  (group128 ? 0 : 4 * g)) =
          __halves2half2(gq[g].scale, gq[g].min);
  }
}

}  // namespace optr
