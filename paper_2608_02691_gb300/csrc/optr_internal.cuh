// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "optr.h"

namespace optr {

constexpr int kD = OPTR_HEAD_DIM;        // 128
constexpr int kG = OPTR_GROUP;           // 32
constexpr int kGroups = kD / kG;         // 4
constexpr int kPage = OPTR_PAGE_SIZE;    // 16
constexpr int kChunk = OPTR_PAGE_HEAD_BYTES;       // G = 32 record
constexpr int kChunk128 = OPTR_PAGE_HEAD_BYTES_G128;  // compact G = 128 record
// Record layout by group size: bytes per (page, KV head), the value
// metadata's offset and the metadata bytes per slot (four {scale, min}
// pairs for G = 32, one for the compact G = 128 record).
__host__ __device__ constexpr int chunk_bytes(bool compact) {
  return compact ? kChunk128 : kChunk;
}
__host__ __device__ constexpr int vmeta_offset(bool compact) {
  return compact ? OPTR_V_META_OFFSET_G128 : OPTR_V_META_OFFSET;
}
__host__ __device__ constexpr int meta_stride(bool compact) { return compact ? 4 : 16; }
constexpr int kMaxRatio = 8;             // largest supported h_q / h_kv

// Decode split-K: every decode launch uses this many warps per SM for the
// partial kernel; the workspace holds one partial slot per warp plus one per
// (sequence, KV head), see DecodePlan.
constexpr int kDecodeWarpsPerSm = 16;
// with BF16 windows the tensor-core partial kernel keeps 12 of its 16 warps
// per SM on the INT2 pages and gives 4 to the window units
constexpr int kWinIntWarps = 12;
constexpr int kCombineMaxSplit = 16;  // combine CTAs per (sequence, KV head)

}  // namespace optr

struct optr_params {
  optr_config cfg;
  int device;
  int num_sms;
  int ratio;           // h_q / h_kv
  int fold_v;          // R_v folded into the model's W_V / W_O (R_v = I here)
  float* R_k;          // device [h_kv][D][D]
  float* R_v;          // device [h_kv][D][D]
  float* R_vT;         // device [h_kv][D][D], R_vT[h][j][i] = R_v[h][i][j]
  float* muR;          // device [h_kv][D], mu R_k computed in fp64
  float* mu;           // device [h_kv][D], the key mean (window logits)
  uint16_t* Rk_t5;     // device tcgen05 B operands of R_k (append_tc05.cu)
  uint16_t* Rv_t5;     // device tcgen05 B operands of R_v
  unsigned* err;       // device error word
  // device address of the fixed scratch array of
  // optr_decode_attention_noalloc on this params' device (noalloc.cu),
  // looked up once at create with that device current
  void* noalloc_ws;
  // stage timing (optr_profile_enable): ev[0..1] bracket the append kernel,
  // ev[2..5] the decode stages (before qrot, partial, combine, after).
  int prof;
  cudaEvent_t ev[6];
  int ran[2];          // append ran / decode ran since enable
};

namespace optr {
// Argument and range checks shared by every decode entry point (null or
// misaligned pointers, sizes): OPTR_OK or the status the call returns.
optr_status decode_args_status(const optr_params* p, const void* q,
                               const int32_t* block_table,
                               const int32_t* seq_lens, int B, int max_pages,
                               const uint8_t* pool, int num_pages,
                               const float* out);
// Device address of the no-allocation scratch array on the current device.
cudaError_t noalloc_scratch_address(void** out);

// Raise a kernel's dynamic shared memory limit on the current device to at
// least `bytes` (static plus dynamic shared memory may exceed 48 KB only
// after this opt-in).  Cached per (kernel, device) under a lock, so the
// runtime call is made once per new maximum.
cudaError_t ensure_dynamic_smem(const void* kernel, size_t bytes);

// Programmatic dependent launch.  Every kernel of the library is launched
// with launch_pdl(), so the GPU may schedule it while the previous kernel in
// the stream is still draining.  Each kernel calls pdl_wait() before it
// touches any memory that an earlier kernel in the stream may write (or
// read): only the library-owned rotation state in optr_params may be read
// before it.  pdl_wait() returns once the previous grid has completed and
// its writes are visible; since every kernel waits before it completes, the
// order of the whole stream is kept.  pdl_trigger() (right after the wait)
// lets the next kernel's blocks be scheduled.  Data written by the previous
// kernel is read with ld.global.cg (__ldcg), never the non-coherent path.
__device__ __forceinline__ void pdl_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block,
                       size_t smem, cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Record stage event i on stream s when profiling is on.
inline void prof_mark(const optr_params* p, int i, cudaStream_t s) {
  if (p->prof) cudaEventRecord(p->ev[i], s);
}
}  // namespace optr

namespace optr {

// Byte offsets of the decode workspace for a batch shape.
struct DecodePlan {
  int B, h_q, h_kv, max_pages, W;  // W = partial-kernel warps
  int S;                           // combine CTAs per (sequence, KV head)
  int Uw;   // BF16-window units (16 window tokens) per (sequence, KV head)
  int Ww;   // window warps (tensor kernel: 4 per SM; CUDA-core: all W), at most B * h_kv * Uw
  size_t off_qf, off_qs, off_frag, off_koff, off_invs, off_pref, off_cnt,
      off_part, off_cpart, off_wpart, total;
};
DecodePlan decode_plan(const optr_params* p, int B, int max_pages);

// One split-K partial (float32): the unnormalised rotated output o'[4][128]
// of the 4 query heads of a GQA group, then their running maxima m[4]
// (log2 domain) and sums l[4].
// BF16 windows (Sec. 3.1 and 4.1; include/optr.h "BF16 windows"): of a
// sequence holding n tokens, positions s < sink and s >= n - recent are
// window positions; the INT2 positions are [sink, int2_end).  With
// sink = recent = 0 every position is INT2.
__host__ __device__ __forceinline__ int int2_end(int n, int sink, int recent) {
  return n - recent > sink ? n - recent : sink;
}
// INT2 pages of the sequence: logical pages sink/16 .. ceil(int2_end/16)-1
// (sink is a multiple of 16, so the first one is full).
__host__ __device__ __forceinline__ int int2_pages(int n, int sink, int recent) {
  const int e = int2_end(n, sink, recent);
  return e > sink ? (e + kPage - 1) / kPage - sink / kPage : 0;
}
// Window positions of the sequence, listed sink part first: count, and the
// position of list entry i.
__host__ __device__ __forceinline__ int win_count(int n, int sink, int recent) {
  const int ns = n < sink ? n : sink;
  const int r0 = n - recent > sink ? n - recent : sink;
  return ns + (n > r0 ? n - r0 : 0);
}
__host__ __device__ __forceinline__ int win_pos(int i, int n, int sink, int recent) {
  const int ns = n < sink ? n : sink;
  const int r0 = n - recent > sink ? n - recent : sink;
  return i < ns ? i : r0 + (i - ns);
}
// Store row of window position s (recent > 0 whenever s >= sink), in 64
// bits so that positions computed from any int32 pos0 stay exact; the row
// itself lies in [0, sink + recent).
__host__ __device__ __forceinline__ int win_row(long long s, int sink, int recent) {
  return (int)(s < sink ? s : sink + (s - sink) % recent);
}
constexpr int kWinUnit = 16;  // window tokens per decode work unit

// Window store arguments of one call (null when the windows are off).
struct WinArgs {
  __nv_bfloat16* win;     // [n_slots][h_kv][2][sink + recent][D]
  const int32_t* slot;    // [B]
  int n_slots;
};

constexpr int kPartFloats = 4 * kD + 8;
constexpr int kPartM = 4 * kD;
constexpr int kPartL = 4 * kD + 4;

// Launchers (return cudaGetLastError()).
cudaError_t launch_append_cuda_core(const optr_params* p, const __nv_bfloat16* k,
                                    const __nv_bfloat16* v, int n_tok,
                                    const int32_t* cu_new, const int32_t* pos0,
                                    const int32_t* bt, int B, int max_pages,
                                    uint8_t* pool, int num_pages,
                                    cudaStream_t s);
// tcgen05 append operand: [hi, lo][128 x 128] fp16 per head, see append_tc05.cu.
constexpr int kRT5Halves = 2 * kD * kD;
void build_rotation_tc05(const float* R /*[D][D]*/, uint16_t* out);
cudaError_t launch_append_tc05(const optr_params* p, const __nv_bfloat16* k,
                               const __nv_bfloat16* v, int n_tok,
                               const int32_t* cu_new, const int32_t* pos0,
                               const int32_t* bt, int B, int max_pages,
                               uint8_t* pool, int num_pages, cudaStream_t s);
// The decode step's single-token cache write, fused into the decode's first
// launch (optr_decode_step); null for a decode alone.
struct StepAppend {
  const __nv_bfloat16* k;
  const __nv_bfloat16* v;
  int n_tok;
  const int32_t* cu_new;
  const int32_t* pos0;
  uint8_t* pool;
};

cudaError_t launch_decode(const optr_params* p, int variant,
                          const __nv_bfloat16* q, const int32_t* bt,
                          const int32_t* seq_lens, int B, int max_pages,
                          const uint8_t* pool, int num_pages, float* out,
                          void* ws, const DecodePlan& plan, cudaStream_t s,
                          const StepAppend* app, const WinArgs* win);

// Window part of a cache write (positions of the BF16 windows copied into
// the store); a separate launch after the INT2 write.
cudaError_t launch_window_copy(const optr_params* p, const __nv_bfloat16* k,
                               const __nv_bfloat16* v, int n_tok,
                               const int32_t* cu_new, const int32_t* pos0,
                               int B, const WinArgs& win, cudaStream_t s);

}  // namespace optr
