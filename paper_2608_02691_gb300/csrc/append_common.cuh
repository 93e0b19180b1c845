// Device helpers shared by the cache-write kernels.
#pragma once

#include "optr_internal.cuh"

namespace optr {

// Sequence of new token t: the largest b with cu_new[b] <= t.
__device__ __forceinline__ int find_seq(const int32_t* __restrict__ cu_new,
                                        int B, int t) {
  int lo = 0, hi = B;
  while (hi - lo > 1) {
    int mid = (lo + hi) >> 1;
    if (__ldg(cu_new + mid) <= t) lo = mid; else hi = mid;
  }
  return lo;
}

// Byte offset in the pool of the record (page, h) (records of `chunk`
// bytes) and the slot of new token `tok`, or -1 (after flagging the device error word) when a table entry,
// position or cu_new entry is out of range.
__device__ __forceinline__ long long resolve_slot(int tok, int h, const int32_t* __restrict__ cu_new,
                                  const int32_t* __restrict__ pos0,
                                  const int32_t* __restrict__ bt, int B,
                                  int max_pages, int num_pages, int h_kv,
                                  int* slot, unsigned* err, int chunk) {
  int b = find_seq(cu_new, B, tok);
  int c0 = __ldg(cu_new + b), c1 = __ldg(cu_new + b + 1);
  if (!(c0 <= tok && tok < c1)) {
    atomicOr(err, OPTR_DEVERR_CU_NEW);
    return -1;
  }
  long long pos = (long long)__ldg(pos0 + b) + (tok - c0);
  if (pos < 0 || pos >= (long long)max_pages * kPage) {
    atomicOr(err, OPTR_DEVERR_POSITION);
    return -1;
  }
  int page = __ldg(bt + (size_t)b * max_pages + pos / kPage);
  if (page < 0 || page >= num_pages) {
    atomicOr(err, OPTR_DEVERR_PAGE_ID);
    return -1;
  }
  *slot = (int)(pos % kPage);
  return ((long long)page * h_kv + h) * chunk;
}

// resolve_slot() with cu_new[0..B] and pos0[0..B-1] already in shared
// memory (cu and p0 point there); only the block-table entry is read from
// global memory.
__device__ __forceinline__ long long resolve_slot_cached(
    int tok, int h, const int* cu, const int* p0,
    const int32_t* __restrict__ bt, int B, int max_pages, int num_pages,
    int h_kv, int* slot, unsigned* err, int chunk) {
  int lo = 0, hi = B;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (cu[mid] <= tok) lo = mid; else hi = mid;
  }
  const int b = lo;
  const int c0 = cu[b], c1 = cu[b + 1];
  if (!(c0 <= tok && tok < c1)) {
    atomicOr(err, OPTR_DEVERR_CU_NEW);
    return -1;
  }
  const long long pos = (long long)p0[b] + (tok - c0);
  if (pos < 0 || pos >= (long long)max_pages * kPage) {
    atomicOr(err, OPTR_DEVERR_POSITION);
    return -1;
  }
  const int page = __ldg(bt + (size_t)b * max_pages + pos / kPage);
  if (page < 0 || page >= num_pages) {
    atomicOr(err, OPTR_DEVERR_PAGE_ID);
    return -1;
  }
  *slot = (int)(pos % kPage);
  return ((long long)page * h_kv + h) * chunk;
}

}  // namespace optr
