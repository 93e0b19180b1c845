// Issue rate of tcgen05.mma (kind::f16, M = 128, K = 16, A in tensor
// memory, B in shared memory) against N, on every SM at once.  One thread
// per CTA issues `iters` MMAs, four per loop iteration, into one
// accumulator (or four independent ones) and the CTA waits (bounded) for
// their completion.  Prints cycles per MMA and the aggregate dense rate.
//
// This measures whether a GQA group's decode attention could use tcgen05:
// a group of 4 query heads (x {hi, lo} operand splits) fills N = 8..32
// columns of an M = 128 token tile.  It is a stand-alone program, not part
// of the library:
//   nvcc -gencode arch=compute_103a,code=sm_103a -O2 -std=c++17 \
//        -Ipaper_2608_02691_gb300/csrc -o mma_rate tcgen05_mma_rate.cu
#include <cstdio>
#include <cstdint>

#include "tc05.cuh"

using namespace optr::tc05;

__global__ void __launch_bounds__(128, 1)
rate(int N, int nd, int iters, unsigned long long* cyc, unsigned* status) {
  __shared__ __align__(1024) unsigned char sb[8192];  // B: N <= 128 rows x K = 16
  __shared__ __align__(8) uint64_t bar;
  __shared__ uint32_t tbase;
  __shared__ int abort_flag;
  const int tid = threadIdx.x, warp = tid >> 5;
  for (int i = tid; i < 2048; i += 128) reinterpret_cast<uint32_t*>(sb)[i] = 0x3c003c00u;
  if (tid == 0) {
    bar_init(&bar, 1);
    abort_flag = 0;
    bar_init_fence();
  }
  if (warp == 0) tmem_alloc(&tbase, 512);
  fence_proxy_async();
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem = tbase;
  {
    // A (128 lanes x K = 16 f16 = 8 columns) at column 384: all ones
    uint32_t a[32];
    for (int j = 0; j < 32; ++j) a[j] = 0x3c003c00u;
    tmem_st32(tmem + ((uint32_t)(32 * warp) << 16) + 384, a);
    tmem_wait_st();
  }
  fence_before();
  __syncthreads();
  fence_after();
  if (tid == 0) {
    const uint64_t bd = smem_desc(smem_addr(sb), 128, 256);
    const uint32_t id = idesc_f16(128, N), a = tmem + 384;
    const uint32_t d0 = tmem, d1 = tmem + (nd > 1 ? N : 0), d2 = tmem + (nd > 1 ? 2 * N : 0),
                   d3 = tmem + (nd > 1 ? 3 * N : 0);
    const unsigned long long t0 = clock64();
    for (int i = 0; i < iters; i += 4) {
      const uint32_t acc = i > 0;
      mma_ts(d0, a, bd, id, acc);
      mma_ts(d1, a, bd, id, nd > 1 ? acc : 1u);
      mma_ts(d2, a, bd, id, nd > 1 ? acc : 1u);
      mma_ts(d3, a, bd, id, nd > 1 ? acc : 1u);
    }
    mma_commit(&bar);
    const bool ok = bar_wait(&bar, 0, &abort_flag);
    const unsigned long long t1 = clock64();
    if (!ok) atomicOr(status, 1u);
    if (blockIdx.x == 0) *cyc = t1 - t0;
  }
  fence_before();
  __syncthreads();
  if (warp == 0) {
    fence_after();
    tmem_dealloc(tmem, 512);
  }
}

int main() {
  int nsm = 0;
  cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, 0);
  unsigned long long* dc;
  unsigned* ds;
  cudaMalloc(&dc, 8);
  cudaMalloc(&ds, 4);
  cudaMemset(ds, 0, 4);
  const int iters = 4096;
  printf("tcgen05.mma kind::f16, M = 128, K = 16, A in tensor memory, %d SMs\n", nsm);
  for (int nd : {1, 4})
    for (int N : {16, 32, 64, 128}) {
      if (nd * N > 384) continue;
      rate<<<nsm, 128>>>(N, nd, iters, dc, ds);  // warm-up
      cudaEvent_t a, b;
      cudaEventCreate(&a);
      cudaEventCreate(&b);
      cudaEventRecord(a);
      rate<<<nsm, 128>>>(N, nd, iters, dc, ds);
      cudaEventRecord(b);
      const cudaError_t e = cudaDeviceSynchronize();
      float ms = 0.f;
      cudaEventElapsedTime(&ms, a, b);
      unsigned long long cyc = 0;
      unsigned st = 0;
      cudaMemcpy(&cyc, dc, 8, cudaMemcpyDeviceToHost);
      cudaMemcpy(&st, ds, 4, cudaMemcpyDeviceToHost);
      const double flop = 2.0 * 128 * N * 16 * (double)iters * nsm;
      printf("accumulators %d  N %3d: %s status %u  %6.1f cycles/MMA  %7.0f TFLOP/s\n", nd, N,
             cudaGetErrorString(e), st, (double)cyc / iters, flop / (ms * 1e-3) / 1e12);
      if (e != cudaSuccess) return 1;
    }
  return 0;
}
