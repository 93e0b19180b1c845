// Host side of the C ABI declared in include/optr.h: argument validation,
// library-owned state (optr_params) and kernel launches.  No entry point
// here allocates or synchronises except optr_params_create/destroy and
// optr_device_error.
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <mutex>
#include <vector>

#include "optr_internal.cuh"

using namespace optr;

namespace {

bool aligned(const void* ptr, size_t a) {
  return (reinterpret_cast<uintptr_t>(ptr) % a) == 0;
}

optr_status cuda_status(cudaError_t e) {
  return e == cudaSuccess ? OPTR_OK : OPTR_ERR_CUDA;
}

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// A per-step activation (k, v, q or out) as the kernels address it: device
// or managed memory as given; page-locked host memory through its device
// mapping (*host set), which the kernels then read or write in place over
// the host link.  Pageable host memory, or a pointer the runtime does not
// know, is refused (false), so no kernel ever dereferences it.
bool io_pointer(const void* ptr, const void** dev, bool* host) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, ptr) != cudaSuccess) {
    (void)cudaGetLastError();  // the failed query leaves no error behind
    return false;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) {
    *dev = ptr;
    if (host) *host = false;
    return true;
  }
  if (a.type == cudaMemoryTypeHost && a.devicePointer != nullptr) {
    *dev = a.devicePointer;
    if (host) *host = true;
    return true;
  }
  return false;
}

}  // namespace

namespace optr {

cudaError_t ensure_dynamic_smem(const void* kernel, size_t bytes) {
  struct Entry {
    const void* kernel;
    int device;
    size_t bytes;
  };
  static std::mutex mu;
  static std::vector<Entry> done;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  Entry* hit = nullptr;
  for (Entry& x : done)
    if (x.kernel == kernel && x.device == dev) hit = &x;
  if (hit && hit->bytes >= bytes) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)bytes);
  if (e != cudaSuccess) return e;
  if (hit)
    hit->bytes = bytes;
  else
    done.push_back(Entry{kernel, dev, bytes});
  return cudaSuccess;
}

// Workspace of one decode call (all offsets 256-byte aligned):
//   qf   float [B][h_q][128]   rotated, pre-scaled queries
//   qs   float [B][h_q][4]     per-group sums of qf
//   frag u32   [B][h_kv][32][16] tensor-core B fragments of qf (hi/lo f16)
//   koff float [B][h_kv][4][4][2] code-offset sums of the fragments
//                               [query head][group][hi/lo] (decode_tc.cu)
//   invs float [B][h_q]         1 / (power-of-two prescale of frag)
//   pref int   [2][B+1]        page prefix sums / non-empty prefix counts
//   cnt  int   [B*h_kv]        combine arrival counters (zeroed by qrot)
//   part float [W + B*h_kv][520] split-K partials (o'[4][128], m[4], l[4])
//   cpart float [B*h_kv*S][520] combine chunk results (only when S > 1)
//   wpart float [Ww + B*h_kv][520] window partials (BF16 windows only)
// S, the combine CTAs per (sequence, KV head), is sized for ~32 partials
// each when every sequence is max_pages long: a segment then overlaps about
// W / (B*h_kv) + 2 warp ranges.
DecodePlan decode_plan(const optr_params* p, int B, int max_pages) {
  DecodePlan d;
  d.B = B;
  d.h_q = p->cfg.h_q;
  d.h_kv = p->cfg.h_kv;
  d.max_pages = max_pages;
  d.W = p->num_sms * kDecodeWarpsPerSm;
  // BF16 windows: Uw units of 16 window tokens per (sequence, KV head);
  // Ww window warps, each owning at least one unit: with the tensor-core
  // partial kernel 4 per SM beside 12 INT2 warps (so W is 12 per SM), with
  // the CUDA-core one every warp takes a share before its pages
  d.Uw = (p->cfg.sink + p->cfg.recent + kWinUnit - 1) / kWinUnit;
  const long long units = (long long)B * d.h_kv * d.Uw;
  d.Ww = 0;
  if (units > 0) {
    if (p->cfg.decode_variant != OPTR_VARIANT_CUDA_CORE) {
      d.W = p->num_sms * kWinIntWarps;
      d.Ww = (int)std::min<long long>((long long)p->num_sms * (kDecodeWarpsPerSm - kWinIntWarps), units);
    } else {
      d.Ww = (int)std::min<long long>(d.W, units);
    }
  }
  size_t o = 0;
  d.off_qf = o;
  o = round_up(o + sizeof(float) * (size_t)B * d.h_q * kD, 256);
  d.off_qs = o;
  o = round_up(o + sizeof(float) * (size_t)B * d.h_q * kGroups, 256);
  d.off_frag = o;
  o = round_up(o + sizeof(uint32_t) * (size_t)B * d.h_kv * 32 * 16, 256);
  d.off_koff = o;
  o = round_up(o + sizeof(float) * (size_t)B * d.h_kv * 32, 256);
  d.off_invs = o;
  o = round_up(o + sizeof(float) * (size_t)B * d.h_q, 256);
  d.off_pref = o;
  o = round_up(o + sizeof(int) * 2 * (size_t)(B + 1), 256);
  d.off_cnt = o;
  o = round_up(o + sizeof(int) * (size_t)B * d.h_kv, 256);
  d.off_part = o;
  o = round_up(o + sizeof(float) * kPartFloats *
                       ((size_t)d.W + (size_t)B * d.h_kv), 256);
  {
    const long long segs = (long long)B * d.h_kv;
    const long long n_est = d.W / segs + 2;
    d.S = (int)std::min<long long>(kCombineMaxSplit,
                                   std::max<long long>(1, (n_est + 31) / 32));
  }
  d.off_cpart = o;
  if (d.S > 1)
    o = round_up(o + sizeof(float) * kPartFloats * (size_t)B * d.h_kv * d.S, 256);
  d.off_wpart = o;
  if (d.Ww > 0)
    o = round_up(o + sizeof(float) * kPartFloats *
                         ((size_t)d.Ww + (size_t)B * d.h_kv), 256);
  d.total = o;
  return d;
}

}  // namespace optr

namespace optr {

optr_status decode_args_status(const optr_params* p, const void* q,
                               const int32_t* block_table,
                               const int32_t* seq_lens, int B, int max_pages,
                               const uint8_t* pool, int num_pages,
                               const float* out) {
  if (!p || B <= 0 || max_pages <= 0 || num_pages <= 0)
    return OPTR_ERR_INVALID_ARG;
  if (!q || !block_table || !seq_lens || !pool || !out)
    return OPTR_ERR_INVALID_ARG;
  if (!aligned(pool, 16) || !aligned(q, 16) || !aligned(out, 16))
    return OPTR_ERR_INVALID_ARG;
  if ((long long)max_pages * kPage > (1LL << 30) || B > (1 << 24))
    return OPTR_ERR_OUT_OF_RANGE;
  // the split-K plan indexes (sequence, KV head, page) units with 32 bits
  if ((long long)B * max_pages * p->cfg.h_kv >= (1LL << 31))
    return OPTR_ERR_OUT_OF_RANGE;
  return OPTR_OK;
}

}  // namespace optr

extern "C" {

const char* optr_strerror(optr_status s) {
  switch (s) {
    case OPTR_OK: return "ok";
    case OPTR_ERR_INVALID_ARG: return "invalid argument";
    case OPTR_ERR_UNSUPPORTED: return "unsupported shape (need D=128, G=32, P=16, h_q = 4*h_kv)";
    case OPTR_ERR_OUT_OF_RANGE: return "size out of the supported range";
    case OPTR_ERR_WORKSPACE: return "workspace missing or too small";
    case OPTR_ERR_CUDA: return "CUDA runtime error";
  }
  return "unknown status";
}

optr_status optr_params_create(const optr_config* cfg, const float* R_k,
                               const float* R_v, const float* mu,
                               optr_params** out) {
  if (out) *out = nullptr;
  if (!cfg || !R_k || !mu || !out) return OPTR_ERR_INVALID_ARG;
  if (cfg->h_kv <= 0 || cfg->h_q <= 0 || cfg->h_q % cfg->h_kv != 0)
    return OPTR_ERR_INVALID_ARG;
  if (cfg->head_dim != kD || (cfg->group != kG && cfg->group != 4 * kG) ||
      cfg->page_size != kPage || cfg->h_q / cfg->h_kv != 4)
    return OPTR_ERR_UNSUPPORTED;
  if (!(cfg->clip_k > 0.f && cfg->clip_k <= 1.f) ||
      !(cfg->clip_v > 0.f && cfg->clip_v <= 1.f))
    return OPTR_ERR_INVALID_ARG;
  if (cfg->h_kv > 1024) return OPTR_ERR_OUT_OF_RANGE;
  if (cfg->sink < 0 || cfg->recent < 0 || cfg->sink % kPage != 0)
    return OPTR_ERR_INVALID_ARG;
  if (cfg->sink > 1024 || cfg->recent > 1024) return OPTR_ERR_OUT_OF_RANGE;

  const int H = cfg->h_kv;
  const size_t mat = (size_t)kD * kD;
  // R_v = NULL: the value rotation is folded into the model's W_V and W_O
  // (Appendix "Equivalent Inference Implementation"); the library then
  // quantizes values as given and returns the output in that basis, i.e.
  // it runs with R_v = I and skips the work where that is cheap.
  const bool fold_v = R_v == nullptr;
  std::vector<float> eye;
  if (fold_v) {
    eye.assign((size_t)H * mat, 0.f);
    for (int h = 0; h < H; ++h)
      for (int i = 0; i < kD; ++i) eye[(size_t)h * mat + (size_t)i * kD + i] = 1.f;
    R_v = eye.data();
  }
  // Host-side preparation: mu R_k in fp64, R_v transposed.
  std::vector<float> muR((size_t)H * kD), RvT((size_t)H * mat);
  for (int h = 0; h < H; ++h) {
    const float* R = R_k + h * mat;
    for (int j = 0; j < kD; ++j) {
      double acc = 0.0;
      for (int i = 0; i < kD; ++i)
        acc += (double)mu[h * kD + i] * (double)R[(size_t)i * kD + j];
      muR[(size_t)h * kD + j] = (float)acc;
    }
    const float* Rv = R_v + h * mat;
    for (int i = 0; i < kD; ++i)
      for (int j = 0; j < kD; ++j)
        RvT[h * mat + (size_t)j * kD + i] = Rv[(size_t)i * kD + j];
  }

  optr_params* p = (optr_params*)calloc(1, sizeof(optr_params));
  if (!p) return OPTR_ERR_OUT_OF_RANGE;
  p->cfg = *cfg;
  p->ratio = cfg->h_q / cfg->h_kv;
  p->fold_v = fold_v ? 1 : 0;
  cudaError_t e = cudaGetDevice(&p->device);
  if (e == cudaSuccess)
    e = cudaDeviceGetAttribute(&p->num_sms, cudaDevAttrMultiProcessorCount,
                               p->device);
  if (e == cudaSuccess) e = cudaMalloc(&p->R_k, sizeof(float) * H * mat);
  if (e == cudaSuccess) e = cudaMalloc(&p->R_v, sizeof(float) * H * mat);
  if (e == cudaSuccess) e = cudaMalloc(&p->R_vT, sizeof(float) * H * mat);
  if (e == cudaSuccess) e = cudaMalloc(&p->muR, sizeof(float) * H * kD);
  if (e == cudaSuccess) e = cudaMalloc(&p->mu, sizeof(float) * H * kD);
  if (e == cudaSuccess) e = cudaMalloc(&p->err, sizeof(unsigned));
  std::vector<uint16_t> t5((size_t)H * kRT5Halves);
  if (e == cudaSuccess) e = cudaMalloc(&p->Rk_t5, sizeof(uint16_t) * t5.size());
  if (e == cudaSuccess) e = cudaMalloc(&p->Rv_t5, sizeof(uint16_t) * t5.size());
  if (e == cudaSuccess) {
    for (int h = 0; h < H; ++h)
      build_rotation_tc05(R_k + h * mat, t5.data() + (size_t)h * kRT5Halves);
    e = cudaMemcpy(p->Rk_t5, t5.data(), sizeof(uint16_t) * t5.size(),
                   cudaMemcpyHostToDevice);
  }
  if (e == cudaSuccess) {
    for (int h = 0; h < H; ++h)
      build_rotation_tc05(R_v + h * mat, t5.data() + (size_t)h * kRT5Halves);
    e = cudaMemcpy(p->Rv_t5, t5.data(), sizeof(uint16_t) * t5.size(),
                   cudaMemcpyHostToDevice);
  }
  if (e == cudaSuccess)
    e = cudaMemcpy(p->R_k, R_k, sizeof(float) * H * mat, cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(p->R_v, R_v, sizeof(float) * H * mat, cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(p->R_vT, RvT.data(), sizeof(float) * H * mat,
                   cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(p->muR, muR.data(), sizeof(float) * H * kD,
                   cudaMemcpyHostToDevice);
  if (e == cudaSuccess)
    e = cudaMemcpy(p->mu, mu, sizeof(float) * H * kD, cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemset(p->err, 0, sizeof(unsigned));
  if (e == cudaSuccess) e = noalloc_scratch_address(&p->noalloc_ws);
  if (e != cudaSuccess) {
    optr_params_destroy(p);
    return OPTR_ERR_CUDA;
  }
  *out = p;
  return OPTR_OK;
}

void optr_params_destroy(optr_params* p) {
  if (!p) return;
  optr_profile_enable(p, 0);
  cudaFree(p->R_k);
  cudaFree(p->R_v);
  cudaFree(p->R_vT);
  cudaFree(p->muR);
  cudaFree(p->mu);
  cudaFree(p->Rk_t5);
  cudaFree(p->Rv_t5);
  cudaFree(p->err);
  free(p);
}

size_t optr_page_bytes(const optr_params* p) {
  return p ? (size_t)p->cfg.h_kv * chunk_bytes(p->cfg.group == 128) : 0;
}

namespace {

bool windows_on(const optr_params* p) {
  return p->cfg.sink > 0 || p->cfg.recent > 0;
}

// The window store of a _win call, validated: null when the windows are
// off; *bad set when they are on and the store is missing or misaligned.
const WinArgs* window_args(const optr_params* p, void* win,
                           const int32_t* win_slot, int n_slots, WinArgs* buf,
                           bool* bad) {
  *bad = false;
  if (!windows_on(p)) return nullptr;
  if (!win || !win_slot || n_slots <= 0 || !aligned(win, 16)) {
    *bad = true;
    return nullptr;
  }
  buf->win = static_cast<__nv_bfloat16*>(win);
  buf->slot = win_slot;
  buf->n_slots = n_slots;
  return buf;
}

}  // namespace

size_t optr_window_bytes(const optr_params* p, int n_slots) {
  if (!p || n_slots <= 0) return 0;
  return (size_t)n_slots * p->cfg.h_kv * 2 * (p->cfg.sink + p->cfg.recent) *
         kD * sizeof(uint16_t);
}

optr_status optr_kv_append_win(const optr_params* p, const void* k,
                               const void* v, int n_tok, const int32_t* cu_new,
                               const int32_t* pos0, const int32_t* block_table,
                               int B, int max_pages, uint8_t* pool,
                               int num_pages, void* win,
                               const int32_t* win_slot, int n_slots,
                               cudaStream_t stream) {
  if (!p || n_tok < 0 || B <= 0 || max_pages <= 0 || num_pages <= 0)
    return OPTR_ERR_INVALID_ARG;
  WinArgs wbuf;
  bool bad = false;
  const WinArgs* wa = window_args(p, win, win_slot, n_slots, &wbuf, &bad);
  if (bad) return OPTR_ERR_INVALID_ARG;
  if (n_tok == 0) return OPTR_OK;
  if (!k || !v || !cu_new || !pos0 || !block_table || !pool)
    return OPTR_ERR_INVALID_ARG;
  if (!aligned(pool, 16) || !aligned(k, 16) || !aligned(v, 16))
    return OPTR_ERR_INVALID_ARG;
  bool k_host = false, v_host = false;
  if (!io_pointer(k, &k, &k_host) || !io_pointer(v, &v, &v_host))
    return OPTR_ERR_INVALID_ARG;
  if ((long long)max_pages * kPage > (1LL << 30)) return OPTR_ERR_OUT_OF_RANGE;
  const int variant = p->cfg.append_variant;
  prof_mark(p, 0, stream);
  cudaError_t e;
  // decode-step sized appends (<= 256 tokens) use the slice-parallel
  // CUDA-core kernel under every variant; larger ones the tensor-core kernel
  // unless the CUDA-core variant is requested or the input is in host
  // memory (the tensor-core kernel loads it by TMA from device memory)
  if (variant == OPTR_VARIANT_CUDA_CORE || n_tok <= 256 || k_host || v_host)
    e = launch_append_cuda_core(p, (const __nv_bfloat16*)k,
                                (const __nv_bfloat16*)v, n_tok, cu_new, pos0,
                                block_table, B, max_pages, pool, num_pages,
                                stream);
  else
    e = launch_append_tc05(p, (const __nv_bfloat16*)k,
                             (const __nv_bfloat16*)v, n_tok, cu_new, pos0,
                             block_table, B, max_pages, pool, num_pages,
                             stream);
  prof_mark(p, 1, stream);
  if (e == cudaSuccess && wa)
    e = launch_window_copy(p, (const __nv_bfloat16*)k, (const __nv_bfloat16*)v,
                           n_tok, cu_new, pos0, B, *wa, stream);
  if (p->prof) const_cast<optr_params*>(p)->ran[0] = 1;
  return cuda_status(e);
}

optr_status optr_kv_append(const optr_params* p, const void* k, const void* v,
                           int n_tok, const int32_t* cu_new,
                           const int32_t* pos0, const int32_t* block_table,
                           int B, int max_pages, uint8_t* pool, int num_pages,
                           cudaStream_t stream) {
  if (p && windows_on(p)) return OPTR_ERR_INVALID_ARG;
  return optr_kv_append_win(p, k, v, n_tok, cu_new, pos0, block_table, B,
                            max_pages, pool, num_pages, nullptr, nullptr, 0,
                            stream);
}

size_t optr_decode_workspace_size(const optr_params* p, int B, int max_pages) {
  if (!p || B <= 0 || max_pages <= 0) return 0;
  return decode_plan(p, B, max_pages).total;
}


optr_status optr_decode_attention_win(const optr_params* p, const void* q,
                                      const int32_t* block_table,
                                      const int32_t* seq_lens, int B,
                                      int max_pages, const uint8_t* pool,
                                      int num_pages, const void* win,
                                      const int32_t* win_slot, int n_slots,
                                      float* out, void* workspace,
                                      size_t ws_bytes, cudaStream_t stream) {
  const optr_status st = decode_args_status(p, q, block_table, seq_lens, B,
                                            max_pages, pool, num_pages, out);
  if (st != OPTR_OK) return st;
  {
    const void* od = nullptr;
    if (!io_pointer(q, &q, nullptr) || !io_pointer(out, &od, nullptr))
      return OPTR_ERR_INVALID_ARG;
    out = static_cast<float*>(const_cast<void*>(od));
  }
  WinArgs wbuf;
  bool bad = false;
  const WinArgs* wa = window_args(p, const_cast<void*>(win), win_slot, n_slots,
                                  &wbuf, &bad);
  if (bad) return OPTR_ERR_INVALID_ARG;
  DecodePlan plan = decode_plan(p, B, max_pages);
  if (!workspace || ws_bytes < plan.total || !aligned(workspace, 256))
    return OPTR_ERR_WORKSPACE;
  int variant = p->cfg.decode_variant;
  cudaError_t e = launch_decode(p, variant, (const __nv_bfloat16*)q,
                                block_table, seq_lens, B, max_pages, pool,
                                num_pages, out, workspace, plan, stream,
                                nullptr, wa);
  if (p->prof) const_cast<optr_params*>(p)->ran[1] = 1;
  return cuda_status(e);
}

optr_status optr_decode_attention(const optr_params* p, const void* q,
                                  const int32_t* block_table,
                                  const int32_t* seq_lens, int B,
                                  int max_pages, const uint8_t* pool,
                                  int num_pages, float* out, void* workspace,
                                  size_t ws_bytes, cudaStream_t stream) {
  if (p && windows_on(p)) return OPTR_ERR_INVALID_ARG;
  return optr_decode_attention_win(p, q, block_table, seq_lens, B, max_pages,
                                   pool, num_pages, nullptr, nullptr, 0, out,
                                   workspace, ws_bytes, stream);
}

optr_status optr_decode_step_win(const optr_params* p, const void* q,
                                 const void* k, const void* v, int n_tok,
                                 const int32_t* cu_new, const int32_t* pos0,
                                 const int32_t* block_table,
                                 const int32_t* seq_lens, int B, int max_pages,
                                 uint8_t* pool, int num_pages, void* win,
                                 const int32_t* win_slot, int n_slots,
                                 float* out, void* workspace, size_t ws_bytes,
                                 cudaStream_t stream) {
  if (!p || n_tok < 0 || B <= 0 || max_pages <= 0 || num_pages <= 0)
    return OPTR_ERR_INVALID_ARG;
  if (!q || !block_table || !seq_lens || !pool || !out)
    return OPTR_ERR_INVALID_ARG;
  if (n_tok > 0 && (!k || !v || !cu_new || !pos0)) return OPTR_ERR_INVALID_ARG;
  if (!aligned(pool, 16) || !aligned(q, 16) || !aligned(out, 16) ||
      (n_tok > 0 && (!aligned(k, 16) || !aligned(v, 16))))
    return OPTR_ERR_INVALID_ARG;
  WinArgs wbuf;
  bool bad = false;
  const WinArgs* wa = window_args(p, win, win_slot, n_slots, &wbuf, &bad);
  if (bad) return OPTR_ERR_INVALID_ARG;
  if ((long long)max_pages * kPage > (1LL << 30) || B > (1 << 24))
    return OPTR_ERR_OUT_OF_RANGE;
  if ((long long)B * max_pages * p->cfg.h_kv >= (1LL << 31))
    return OPTR_ERR_OUT_OF_RANGE;
  DecodePlan plan = decode_plan(p, B, max_pages);
  if (!workspace || ws_bytes < plan.total || !aligned(workspace, 256))
    return OPTR_ERR_WORKSPACE;
  // the fused launch covers decode-step sized writes with the tensor decode;
  // anything else runs as the two calls
  if (n_tok == 0 || n_tok > 256 || p->cfg.decode_variant == OPTR_VARIANT_CUDA_CORE ||
      p->cfg.append_variant == OPTR_VARIANT_CUDA_CORE) {
    optr_status st = optr_kv_append_win(p, k, v, n_tok, cu_new, pos0,
                                        block_table, B, max_pages, pool,
                                        num_pages, win, win_slot, n_slots,
                                        stream);
    if (st != OPTR_OK) return st;
    return optr_decode_attention_win(p, q, block_table, seq_lens, B, max_pages,
                                     pool, num_pages, win, win_slot, n_slots,
                                     out, workspace, ws_bytes, stream);
  }
  {
    const void* od = nullptr;
    if (!io_pointer(q, &q, nullptr) || !io_pointer(k, &k, nullptr) ||
        !io_pointer(v, &v, nullptr) || !io_pointer(out, &od, nullptr))
      return OPTR_ERR_INVALID_ARG;
    out = static_cast<float*>(const_cast<void*>(od));
  }
  StepAppend app{(const __nv_bfloat16*)k, (const __nv_bfloat16*)v, n_tok,
                 cu_new, pos0, pool};
  cudaError_t e = launch_decode(p, p->cfg.decode_variant, (const __nv_bfloat16*)q,
                                block_table, seq_lens, B, max_pages, pool,
                                num_pages, out, workspace, plan, stream, &app,
                                wa);
  if (p->prof) const_cast<optr_params*>(p)->ran[0] = const_cast<optr_params*>(p)->ran[1] = 1;
  return cuda_status(e);
}

optr_status optr_decode_step(const optr_params* p, const void* q,
                             const void* k, const void* v, int n_tok,
                             const int32_t* cu_new, const int32_t* pos0,
                             const int32_t* block_table,
                             const int32_t* seq_lens, int B, int max_pages,
                             uint8_t* pool, int num_pages, float* out,
                             void* workspace, size_t ws_bytes,
                             cudaStream_t stream) {
  if (p && windows_on(p)) return OPTR_ERR_INVALID_ARG;
  return optr_decode_step_win(p, q, k, v, n_tok, cu_new, pos0, block_table,
                              seq_lens, B, max_pages, pool, num_pages, nullptr,
                              nullptr, 0, out, workspace, ws_bytes, stream);
}

optr_status optr_profile_enable(optr_params* p, int on) {
  if (!p) return OPTR_ERR_INVALID_ARG;
  if (on && !p->prof) {
    for (int i = 0; i < 6; ++i)
      if (cudaEventCreate(&p->ev[i]) != cudaSuccess) return OPTR_ERR_CUDA;
    p->ran[0] = p->ran[1] = 0;
    p->prof = 1;
  } else if (!on && p->prof) {
    for (int i = 0; i < 6; ++i) cudaEventDestroy(p->ev[i]);
    p->prof = 0;
  }
  return OPTR_OK;
}

optr_status optr_profile_last(const optr_params* p, float ms[4]) {
  if (!p || !ms) return OPTR_ERR_INVALID_ARG;
  for (int i = 0; i < 4; ++i) ms[i] = 0.f;
  if (!p->prof) return OPTR_ERR_INVALID_ARG;
  cudaError_t e = cudaSuccess;
  if (p->ran[0]) {
    e = cudaEventSynchronize(p->ev[1]);
    if (e == cudaSuccess) e = cudaEventElapsedTime(&ms[0], p->ev[0], p->ev[1]);
  }
  if (e == cudaSuccess && p->ran[1]) {
    e = cudaEventSynchronize(p->ev[5]);
    for (int i = 0; i < 3 && e == cudaSuccess; ++i)
      e = cudaEventElapsedTime(&ms[1 + i], p->ev[2 + i], p->ev[3 + i]);
  }
  return cuda_status(e);
}

optr_status optr_device_error(const optr_params* p, uint32_t* flags) {
  if (!p || !flags) return OPTR_ERR_INVALID_ARG;
  unsigned h = 0;
  cudaError_t e = cudaDeviceSynchronize();
  if (e == cudaSuccess)
    e = cudaMemcpy(&h, p->err, sizeof(unsigned), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemset(p->err, 0, sizeof(unsigned));
  *flags = h;
  return cuda_status(e);
}

}  // extern "C"
