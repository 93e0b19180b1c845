// Device helpers shared by the decode kernels: split-K work partition,
// cp.async page staging.
#pragma once

#include "optr_internal.cuh"

namespace optr {

// One (sequence, KV head) run of pages inside a warp's flat range.
struct Segment {
  int b, h, p0, n;   // sequence, KV head, first page, page count
  long long f_end;   // flat index one past the segment
};

// The flat index space orders units as (sequence b, KV head h, page p) with
// index pref[b]*h_kv + h*np(b) + p, np(b) = pref[b+1] - pref[b].  Locate the
// segment that starts at flat index f of a warp whose range ends at f1.
__device__ __forceinline__ Segment locate_segment(long long f, long long f1,
                                                  const int* __restrict__ pref,
                                                  int B, int h_kv) {
  int lo = 0, hi = B;  // largest b with pref[b]*h_kv <= f (non-empty by
                       // construction because f < pref[B]*h_kv)
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if ((long long)__ldcg(pref + mid) * h_kv <= f) lo = mid; else hi = mid;
  }
  Segment s;
  s.b = lo;
  const int np = __ldcg(pref + lo + 1) - __ldcg(pref + lo);
  const long long base = (long long)__ldcg(pref + lo) * h_kv;
  const long long r = f - base;
  s.h = (int)(r / np);
  s.p0 = (int)(r - (long long)s.h * np);
  const long long end = base + (long long)(s.h + 1) * np;
  s.f_end = end < f1 ? end : f1;
  s.n = (int)(s.f_end - f);
  return s;
}

// Key-side code position for the tensor-core decode.  Within a 16-bit half
// holding the code bytes of groups (2j, 2j+1) of one word w (low byte group
// 2j), code r of the even group sits at bit 2r and of the odd group at bit
// 8 + 2r.  The tensor kernel moves every field, with at most one shift of
// the 32-bit word (left by 4 or right by 6), to bit 4, 6 or 8 of its half:
// even group r = 0, 1 from (word << 4), r = 2, 3 in place; odd group r = 0 in
// place, r = 1, 2, 3 from (word >> 6).  This is that final bit position.
__host__ __device__ constexpr int code_pos(int G, int r) {
  return (G & 1) ? (r == 0 ? 8 : 2 + 2 * r) : 4 + 2 * (r & 1);
}

// Warp w owns flat indices [floor(w*F/W), floor((w+1)*F/W)).  The warp that
// owns index f (0 <= f < F) is floor(((f+1)*W - 1) / F).
__device__ __forceinline__ int warp_of(long long f, long long F, int W) {
  long long w = ((f + 1) * W - 1) / F;
  return (int)(w < W - 1 ? w : W - 1);
}

// True when warp w owns no flat index (only possible when F < W).
__device__ __forceinline__ bool warp_empty(int w, long long F, int W) {
  return (long long)w * F / W == (long long)(w + 1) * F / W;
}

// cp.async of 16 bytes that writes zeros (and reads nothing) when !valid.
__device__ __forceinline__ void cp_async16_zfill(void* smem, const void* gmem,
                                                 bool valid) {
  const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
  const int src_size = valid ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(s),
               "l"(gmem), "r"(src_size)
               : "memory");
}

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;\n" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}
__device__ __forceinline__ void cp_async_wait_1() { cp_async_wait<1>(); }

// Stage the record (page, h) of logical page `page_idx` (`chunk` bytes: 1536,
// or 1152 for the compact G = 128 record) into shared memory (up to three
// 16-byte copies per lane) and commit one cp.async group.  An
// out-of-range page id is flagged and not read; the group is still
// committed so that group counting stays uniform.
__device__ __forceinline__ bool issue_page(uint8_t* stage,
                                           const uint8_t* __restrict__ pool,
                                           const int32_t* __restrict__ btb,
                                           int page_idx, int num_pages,
                                           int h_kv, int h, int lane,
                                           unsigned* err, int chunk) {
  const int phys = __ldg(btb + page_idx);
  const bool ok = phys >= 0 && phys < num_pages;
  if (ok) {
    const uint8_t* src = pool + ((size_t)phys * h_kv + h) * chunk;
#pragma unroll
    for (int c = 0; c < 3; ++c)
      if ((lane + 32 * c) * 16 < chunk)
        cp_async16(stage + (lane + 32 * c) * 16, src + (lane + 32 * c) * 16);
  } else if (lane == 0) {
    atomicOr(err, OPTR_DEVERR_PAGE_ID);
  }
  cp_async_commit();
  return ok;
}

// Same as issue_page for a physical page id already in hand.
__device__ __forceinline__ bool issue_phys(uint8_t* stage,
                                           const uint8_t* __restrict__ pool,
                                           int phys, int num_pages, int h_kv,
                                           int h, int lane, unsigned* err,
                                           int chunk) {
  const bool ok = phys >= 0 && phys < num_pages;
  if (ok) {
    const uint8_t* src = pool + ((size_t)phys * h_kv + h) * chunk;
#pragma unroll
    for (int c = 0; c < 3; ++c)
      if ((lane + 32 * c) * 16 < chunk)
        cp_async16(stage + (lane + 32 * c) * 16, src + (lane + 32 * c) * 16);
  } else if (lane == 0) {
    atomicOr(err, OPTR_DEVERR_PAGE_ID);
  }
  cp_async_commit();
  return ok;
}

// exp2(m - M) for a partial whose running max is m, 0 for an empty partial.
__device__ __forceinline__ float merge_weight(float m, float M) {
  return m == -INFINITY ? 0.f : exp2f(m - M);
}

}  // namespace optr
