// BF16 sink and recent windows (Sec. 3.1: INT2 long history with a small
// BF16 window; Sec. 4.1: sink and recent tokens stay in BF16, their keys
// centered by the same mu; Sec. 5: 64 sink, 256 recent tokens).
//
//   window_copy_body   cache write: copy the window positions of the new
//                      tokens into the caller's window store.
//   window_phase       decode: the softmax partials of the window positions,
//                      one warp per run of 16-token units, before the warp's
//                      INT2 pages.
#pragma once

#include "decode_common.cuh"

namespace optr {

// ------------------------------------------------------------ cache write

constexpr int kWinCopyTok = 16;  // tokens per copy CTA (512 threads)

struct WinCopySmem {
  long long base[kWinCopyTok];  // store offset (elements) of the token's row
                                // in plane (head 0, keys), or -1
};

// CTA `tile` copies new tokens [16 tile, 16 tile + 16): token t of sequence
// b (rows cu_new[b] .. cu_new[b+1]-1, positions from pos0[b], end = pos0[b]
// + count) is a window position of the written cache when s < sink or, with
// recent > 0, s >= end - recent; its K and V rows of every KV head go to
// row win_row(s) of slot win_slot[b].
__device__ __forceinline__ void window_copy_body(
    int tile, WinCopySmem& sm, const __nv_bfloat16* __restrict__ k,
    const __nv_bfloat16* __restrict__ v, int n_tok,
    const int32_t* __restrict__ cu_new, const int32_t* __restrict__ pos0,
    int B, __nv_bfloat16* __restrict__ win, const int32_t* __restrict__ win_slot,
    int n_slots, int h_kv, int sink, int recent, unsigned* err) {
  const int tid = threadIdx.x;
  const int rows = sink + recent;
  pdl_wait();  // inputs may come from earlier kernels
  pdl_trigger();
  if (tid < kWinCopyTok) {
    const int tok = tile * kWinCopyTok + tid;
    long long base = -1;
    if (tok < n_tok) {
      int lo = 0, hi = B;  // largest b with cu_new[b] <= tok
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (__ldg(cu_new + mid) <= tok) lo = mid; else hi = mid;
      }
      const int c0 = __ldg(cu_new + lo), c1 = __ldg(cu_new + lo + 1);
      if (c0 <= tok && tok < c1) {  // else the INT2 write flags cu_new
        const long long s = (long long)__ldg(pos0 + lo) + (tok - c0);
        const long long end = (long long)__ldg(pos0 + lo) + (c1 - c0);
        if (s >= 0 && (s < sink || (recent > 0 && s >= end - recent))) {
          const int slot = __ldg(win_slot + lo);
          if (slot < 0 || slot >= n_slots) {
            atomicOr(err, OPTR_DEVERR_WIN_SLOT);
          } else {
            const long long row = win_row(s, sink, recent);
            base = (long long)slot * h_kv * 2 * rows * kD + row * kD;
          }
        }
      }
    }
    sm.base[tid] = base;
  }
  __syncthreads();
  // 16-byte pieces: token tt, KV head hh, kind, piece c of the 256-byte row
  const int per_tok = 2 * h_kv * (kD / 8);
  for (int idx = tid; idx < kWinCopyTok * per_tok; idx += blockDim.x) {
    const int tt = idx / per_tok, r = idx - tt * per_tok;
    const long long base = sm.base[tt];
    if (base < 0) continue;
    const int kind = r / (h_kv * (kD / 8));
    const int hh = (r / (kD / 8)) % h_kv, c = r % (kD / 8);
    const int tok = tile * kWinCopyTok + tt;
    const __nv_bfloat16* src = (kind ? v : k) + ((size_t)tok * h_kv + hh) * kD + 8 * c;
    __nv_bfloat16* dst = win + base + (long long)(hh * 2 + kind) * rows * kD + 8 * c;
    *reinterpret_cast<uint4*>(dst) = __ldg(reinterpret_cast<const uint4*>(src));
  }
}

// ------------------------------------------------------------------ decode

// Inputs of the window phase of a partial kernel.
struct WinPhase {
  const __nv_bfloat16* q;      // [B][h_q][D] raw queries
  const __nv_bfloat16* win;    // store
  const int32_t* slot;         // [B]
  const int32_t* seq_lens;     // [B]
  const float* mu;             // [h_kv][D] key mean (library-owned)
  float* wpart;                // [Ww + B*h_kv][kPartFloats]
  unsigned* err;               // device error word
  // the decode step's new tokens (null outside the fused step): their
  // positions are read from these rows, not from the store, because the
  // step's cache write may still be filling the store when this phase runs
  const __nv_bfloat16* k_new;
  const __nv_bfloat16* v_new;
  const int32_t* cu_new;
  const int32_t* pos0;
  int n_slots, B, h_q, h_kv, max_pages, sink, recent, Uw, Ww;
  float qscale;                // log2(e) / sqrt(D)
};

__device__ __forceinline__ void win_mma_bf16(float* d, uint32_t a0, uint32_t a1,
                                             uint32_t a2, uint32_t a3,
                                             uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void win_ldsm_x4(uint32_t (&r)[4], const void* p, bool trans) {
  const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(p));
  if (trans)
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(s));
  else
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(s));
}

__device__ __forceinline__ void win_ldsm_x2t(uint32_t& r0, uint32_t& r1, const void* p) {
  const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(p));
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.trans.shared.b16 {%0,%1}, [%2];\n"
               : "=r"(r0), "=r"(r1) : "r"(s));
}

// 16-byte piece j of staged row r sits at piece (j & 8) | ((j ^ r) & 7) of
// the row: the 8 rows an 8x8 ldmatrix reads then fall on 8 distinct bank
// groups.
__device__ __forceinline__ int win_swz(int j, int r) { return (j & 8) | ((j ^ r) & 7); }

__device__ __forceinline__ float win_sel4(const float (&x)[4], int i) {
  return i == 0 ? x[0] : i == 1 ? x[1] : i == 2 ? x[2] : x[3];
}

constexpr int kWinStageBytes = 2 * kWinUnit * 2 * kD;  // K and V rows: 8 KB
constexpr int kWinPBytes = kWinUnit * 8 * 2;             // P [16 tok][8] bf16

// Window partials of window warp ww (0 <= ww < Ww).  The units (b, h, j) =
// 16 window tokens [16j, 16j + 16) of sequence b, KV head h, indexed
// u = (b * h_kv + h) * Uw + j, are cut into Ww contiguous ranges; a warp
// merges the units of one (b, h) in its range by an online softmax and
// writes one partial (o[4][128], m[4], l[4]; log2 domain, values in the
// unrotated basis) to slot ww + b * h_kv + h.  Units past a sequence's
// window count are empty and skipped, so the slots of (b, h) are those of
// the warps owning its units 0 .. ceil(count / 16) - 1: every window warp
// owns at least one unit, which keeps that run of warps gap-free.
//
// It reads only inputs (queries, lengths, slots, the store, the step's new
// rows) and library-owned state (mu), and writes only its partial slots, so
// a partial kernel runs it before waiting for the previous kernel.  Per
// unit (bf16 tensor cores, mma.sync m16n8k16, fp32 accumulation):
//   stage   the 16 key and value rows by cp.async (zeros past the count)
//           into stage (8 KB, 16-byte aligned; rows swizzled by win_swz);
//   logits  S[16 tok][8] = K[16][128] . Q^T, Q^T columns = the 4 query
//           heads (exact bf16, B fragments straight from global) and 4 zero
//           columns; l = S * qscale - qscale <q, mu> (centered keys);
//   softmax online over the warp's units of (b, h), p split into bf16
//           hi + lo (relative error 2^-16) in pb [16 tok][8 = head x limb];
//   P.V     O^T[128][8] += V^T[128][16] . P[16][8], A = V^T by
//           ldmatrix.trans of the staged value rows.
static __device__ __noinline__ void window_phase(int ww, const WinPhase& a,
                                                 uint8_t* stage, uint8_t* pb) {
  const int lane = threadIdx.x & 31;
  const int g = lane >> 2, c = lane & 3;
  const long long U = (long long)a.B * a.h_kv * a.Uw;
  const long long u0 = ww * U / a.Ww, u1 = (ww + 1) * U / a.Ww;
  const int rows = a.sink + a.recent;
  uint8_t* ks = stage;
  uint8_t* vs = stage + kWinUnit * 2 * kD;
  int cur = -1;  // (b, h) of the running state
  float o[8][4] = {};
  float m[4] = {}, l[4] = {}, qmu[4] = {};
  uint32_t qb[8][2] = {};
  int n = 0, nw = 0, slot = 0;
  bool slot_ok = false;
  int p0n = 0, nn = 0, cn = 0;  // new rows: positions [p0n, p0n + nn) at rows cn..

  auto flush = [&]() {
    float* dst = a.wpart + (size_t)(ww + cur) * kPartFloats + c * kD + g;
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
      dst[16 * mt] = o[mt][0] + o[mt][1];
      dst[16 * mt + 8] = o[mt][2] + o[mt][3];
    }
    if (lane < 4) {
      float* hd = a.wpart + (size_t)(ww + cur) * kPartFloats;
      hd[kPartM + lane] = win_sel4(m, lane);
      hd[kPartL + lane] = win_sel4(l, lane);
    }
  };

  for (long long u = u0; u < u1; ++u) {
    const int bh = (int)(u / a.Uw), j = (int)(u - (long long)bh * a.Uw);
    const int b = bh / a.h_kv, h = bh - b * a.h_kv;
    if (bh != cur) {
      n = __ldg(a.seq_lens + b);
      if (n < 0 || (long long)n > (long long)a.max_pages * kPage) n = 0;  // flagged by qrot
      nw = win_count(n, a.sink, a.recent);
      if (kWinUnit * j >= nw) continue;  // empty unit: no state change
      if (cur >= 0) flush();
      cur = bh;
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        m[r] = -INFINITY;
        l[r] = 0.f;
      }
#pragma unroll
      for (int mt = 0; mt < 8; ++mt)
#pragma unroll
        for (int e = 0; e < 4; ++e) o[mt][e] = 0.f;
      slot = __ldg(a.slot + b);
      slot_ok = slot >= 0 && slot < a.n_slots;
      if (!slot_ok) {  // the run's partial stays empty (m = -inf, l = 0)
        if (lane == 0) atomicOr(a.err, OPTR_DEVERR_WIN_SLOT);
        slot = 0;
      }
      nn = 0;
      if (a.k_new) {
        cn = __ldg(a.cu_new + b);
        nn = __ldg(a.cu_new + b + 1) - cn;
        p0n = __ldg(a.pos0 + b);
      }
      // query B fragments: column g < 4 = head g, k = channels 16kk + 2c
      // (+1) and 16kk + 2c + 8 (+1)
      const __nv_bfloat16* qg = a.q + ((size_t)b * a.h_q + 4 * h) * kD;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        qb[kk][0] = g < 4 ? __ldg(reinterpret_cast<const uint32_t*>(qg + g * kD + 16 * kk + 2 * c)) : 0u;
        qb[kk][1] = g < 4 ? __ldg(reinterpret_cast<const uint32_t*>(qg + g * kD + 16 * kk + 2 * c + 8)) : 0u;
      }
      // qscale * <q_r, mu[h]>: lane takes channels 4 lane .. 4 lane + 3
      const float4 mu4 = __ldg(reinterpret_cast<const float4*>(a.mu + h * kD) + lane);
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const uint2 q4 = __ldg(reinterpret_cast<const uint2*>(qg + r * kD) + lane);
        float x = __uint_as_float(q4.x << 16) * mu4.x;
        x = fmaf(__uint_as_float(q4.x & 0xffff0000u), mu4.y, x);
        x = fmaf(__uint_as_float(q4.y << 16), mu4.z, x);
        x = fmaf(__uint_as_float(q4.y & 0xffff0000u), mu4.w, x);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
        qmu[r] = x * a.qscale;
      }
    } else if (kWinUnit * j >= nw) {
      continue;
    }
    // sources of the unit's 16 rows: lane r < 16 resolves row r
    const int rr = lane & 15;
    const int i = kWinUnit * j + rr;
    const bool rvalid = slot_ok && i < nw;
    const __nv_bfloat16* ksrc = a.win;
    const __nv_bfloat16* vsrc = a.win;
    if (rvalid) {
      const int pos = win_pos(i, n, a.sink, a.recent);
      if (pos >= p0n && pos - p0n < nn) {  // a new token of this step
        const size_t t = (size_t)(cn + pos - p0n) * a.h_kv + h;
        ksrc = a.k_new + t * kD;
        vsrc = a.v_new + t * kD;
      } else {
        const __nv_bfloat16* base = a.win + ((size_t)slot * a.h_kv + h) * 2 * rows * kD;
        const int row = win_row(pos, a.sink, a.recent);
        ksrc = base + (size_t)row * kD;
        vsrc = base + (size_t)(rows + row) * kD;
      }
    }
    __syncwarp();  // the previous unit's reads of stage and pb are done
#pragma unroll
    for (int q = 0; q < kWinUnit / 2; ++q) {
      const int r = 2 * q + (lane >> 4), pc = lane & 15;
      const unsigned long long kp = __shfl_sync(0xffffffffu, reinterpret_cast<unsigned long long>(ksrc), r);
      const unsigned long long vp = __shfl_sync(0xffffffffu, reinterpret_cast<unsigned long long>(vsrc), r);
      const bool ok = __shfl_sync(0xffffffffu, rvalid ? 1 : 0, r) != 0;
      const int dc = win_swz(pc, r);
      cp_async16_zfill(ks + r * 2 * kD + 16 * dc,
                       reinterpret_cast<const __nv_bfloat16*>(kp) + 8 * pc, ok);
      cp_async16_zfill(vs + r * 2 * kD + 16 * dc,
                       reinterpret_cast<const __nv_bfloat16*>(vp) + 8 * pc, ok);
    }
    cp_async_commit();
    cp_async_wait<0>();
    __syncwarp();
    // logits: S[tok][col] for tok g, g + 8 and cols 2c, 2c + 1
    float s[4] = {0.f, 0.f, 0.f, 0.f};
    {
      const int mi = lane >> 3, r = (mi & 1) * 8 + (lane & 7);
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        uint32_t af[4];
        win_ldsm_x4(af, ks + r * 2 * kD + 16 * win_swz(2 * kk + (mi >> 1), r), false);
        win_mma_bf16(s, af[0], af[1], af[2], af[3], qb[kk][0], qb[kk][1]);
      }
    }
    const bool v0 = slot_ok && kWinUnit * j + g < nw;
    const bool v1 = slot_ok && kWinUnit * j + g + 8 < nw;
    const bool hv = c < 2;  // columns 2c, 2c + 1 are heads
    const float qm0 = win_sel4(qmu, (2 * c) & 3), qm1 = win_sel4(qmu, (2 * c + 1) & 3);
    float lg[4];
    lg[0] = hv && v0 ? fmaf(s[0], a.qscale, -qm0) : -INFINITY;
    lg[1] = hv && v0 ? fmaf(s[1], a.qscale, -qm1) : -INFINITY;
    lg[2] = hv && v1 ? fmaf(s[2], a.qscale, -qm0) : -INFINITY;
    lg[3] = hv && v1 ? fmaf(s[3], a.qscale, -qm1) : -INFINITY;
    float mx0 = fmaxf(lg[0], lg[2]), mx1 = fmaxf(lg[1], lg[3]);
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, off));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, off));
    }
    // head h's maximum sits in the lanes with c = h / 2 (lane h / 2 among them)
    float tm[4], alpha[4];
    tm[0] = __shfl_sync(0xffffffffu, mx0, 0);
    tm[1] = __shfl_sync(0xffffffffu, mx1, 0);
    tm[2] = __shfl_sync(0xffffffffu, mx0, 1);
    tm[3] = __shfl_sync(0xffffffffu, mx1, 1);
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const float mn = fmaxf(m[r], tm[r]);  // -inf only with a bad slot
      alpha[r] = m[r] == -INFINITY ? 0.f : exp2f(m[r] - mn);
      m[r] = mn;
    }
    const float mh0 = win_sel4(m, (2 * c) & 3), mh1 = win_sel4(m, (2 * c + 1) & 3);
    float p[4];
    p[0] = lg[0] == -INFINITY ? 0.f : exp2f(lg[0] - mh0);
    p[1] = lg[1] == -INFINITY ? 0.f : exp2f(lg[1] - mh1);
    p[2] = lg[2] == -INFINITY ? 0.f : exp2f(lg[2] - mh0);
    p[3] = lg[3] == -INFINITY ? 0.f : exp2f(lg[3] - mh1);
    float ps0 = p[0] + p[2], ps1 = p[1] + p[3];
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      ps0 += __shfl_xor_sync(0xffffffffu, ps0, off);
      ps1 += __shfl_xor_sync(0xffffffffu, ps1, off);
    }
    {
      float psum[4];
      psum[0] = __shfl_sync(0xffffffffu, ps0, 0);
      psum[1] = __shfl_sync(0xffffffffu, ps1, 0);
      psum[2] = __shfl_sync(0xffffffffu, ps0, 1);
      psum[3] = __shfl_sync(0xffffffffu, ps1, 1);
#pragma unroll
      for (int r = 0; r < 4; ++r) l[r] = fmaf(l[r], alpha[r], psum[r]);
    }
    // P (bf16 hi, lo) into pb[tok][2 head + limb]
    if (hv) {
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const float pa = p[2 * half], pbv = p[2 * half + 1];
        const __nv_bfloat16 ha = __float2bfloat16_rn(pa), hb = __float2bfloat16_rn(pbv);
        const __nv_bfloat16 la = __float2bfloat16_rn(pa - __bfloat162float(ha));
        const __nv_bfloat16 lb = __float2bfloat16_rn(pbv - __bfloat162float(hb));
        uint2 w;
        w.x = (uint32_t)__bfloat16_as_ushort(ha) | ((uint32_t)__bfloat16_as_ushort(la) << 16);
        w.y = (uint32_t)__bfloat16_as_ushort(hb) | ((uint32_t)__bfloat16_as_ushort(lb) << 16);
        *reinterpret_cast<uint2*>(pb + (g + 8 * half) * 16 + 8 * c) = w;
      }
    }
    const float ac = win_sel4(alpha, c);
#pragma unroll
    for (int mt = 0; mt < 8; ++mt)
#pragma unroll
      for (int e = 0; e < 4; ++e) o[mt][e] *= ac;
    __syncwarp();
    uint32_t pb0, pb1;
    win_ldsm_x2t(pb0, pb1, pb + (lane & 15) * 16);
    {
      const int mi = lane >> 3, tok = (mi >> 1) * 8 + (lane & 7);
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        uint32_t af[4];
        win_ldsm_x4(af, vs + tok * 2 * kD + 16 * win_swz(2 * mt + (mi & 1), tok), true);
        win_mma_bf16(o[mt], af[0], af[1], af[2], af[3], pb0, pb1);
      }
    }
  }
  if (cur >= 0) flush();
  __syncwarp();  // the scratch is handed back to the INT2 pages
}

}  // namespace optr
