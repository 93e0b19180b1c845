// Decode attention over the paged INT2 cache.
//
//   qrot     q' = q R_k[h] * log2(e)/sqrt(128) for every query head, per-group
//            sums of q', and the split-K plan (page prefix sums over the
//            batch)  -- paper Appendix, "Rotated-query implementation".
//   partial  persistent warps; the flattened (sequence, KV head, page) space
//            is cut into W equal contiguous ranges, one per warp.  A warp runs
//            an online softmax over each (sequence, KV head) segment of its
//            range and writes one partial (m, l, o') per segment.
//   combine  per (sequence, KV head): log-sum-exp merge of the segment
//            partials, then o = o' R_v^T (Appendix, "Equivalent Inference
//            Implementation": o' = o R_V, recovered with R_V^T).
//
// Logits are kept in the log2 domain: q' carries log2(e)/sqrt(d), so
// softmax weights are exp2(l - m) (Sec. 3 Eq. 1 with the 1/sqrt(d) scale).
#include "decode_common.cuh"
#include "append_small.cuh"
#include "window.cuh"

namespace optr {
namespace {

constexpr float kLog2e = 1.4426950408889634f;

// ---------------------------------------------------------------- qrot

// One CTA per (sequence, KV head), 512 threads = 4 slices x 128 channels:
// slice s sums q[i] R[i][j] over i in [32s, 32s+32) for the 4 query heads of
// the group, the slices are added in shared memory.
constexpr int kQrotThreads = 512;

struct QrotSmem {
  float qsm[4][kD];
  float part[4][4][kD];  // [slice][head][channel]
  float qrs[4][kD];
  float hmax[4][4];
  int warp_tot[2][kQrotThreads / 32];
  long long koff_part[kQrotThreads / 32][kGroups];
};

// CTA (b, h) of the query rotation; 512 threads.
__device__ __forceinline__ void qrot_body(
    int b, int h, QrotSmem& sm, const __nv_bfloat16* __restrict__ q,
    const float* __restrict__ R_k, int B, int h_q, int h_kv, float qscale,
    const int32_t* __restrict__ seq_lens, int max_pages,
    float* __restrict__ qf, float* __restrict__ qs, uint32_t* __restrict__ frag,
    float* __restrict__ koff, float* __restrict__ invs, int* __restrict__ pref,
    int* __restrict__ nzpref, int* __restrict__ cnt_ws, unsigned* err,
    int sink, int recent) {
  float (&qsm)[4][kD] = sm.qsm;
  float (&part)[4][4][kD] = sm.part;
  float (&qrs)[4][kD] = sm.qrs;
  float (&hmax)[4][4] = sm.hmax;
  int (&warp_tot)[2][kQrotThreads / 32] = sm.warp_tot;
  long long (&koff_part)[kQrotThreads / 32][kGroups] = sm.koff_part;
  const int tid = threadIdx.x;
  const int sl = tid >> 7, j = tid & 127;
  const int warp = tid >> 5, lane = tid & 31;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  const float* R = R_k + (size_t)h * kD * kD + (size_t)(32 * sl) * kD + j;
  float rv[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) rv[i] = __ldg(R + i * kD);  // all in flight
  pdl_wait();  // the query, lengths and workspace may belong to earlier kernels
  pdl_trigger();
  // Global stores wait until the end: a __syncthreads() after a store waits
  // for it to complete, which made each phase an L2 round trip.
  {
    const int r = tid >> 7;  // 512 threads load the 4 x 128 query values
    qsm[r][j] = __bfloat162float(q[((size_t)b * h_q + 4 * h + r) * kD + j]);
  }
  __syncthreads();
#pragma unroll
  for (int i4 = 0; i4 < 8; ++i4)
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const float4 qv = *reinterpret_cast<const float4*>(&qsm[r][32 * sl + 4 * i4]);
      acc[r] = fmaf(qv.x, rv[4 * i4 + 0], acc[r]);
      acc[r] = fmaf(qv.y, rv[4 * i4 + 1], acc[r]);
      acc[r] = fmaf(qv.z, rv[4 * i4 + 2], acc[r]);
      acc[r] = fmaf(qv.w, rv[4 * i4 + 3], acc[r]);
    }
#pragma unroll
  for (int r = 0; r < 4; ++r) part[sl][r][j] = acc[r];
  __syncthreads();
  // thread (r, j): the 4 slices of head r, channel j (512 threads)
  const int qr = tid >> 7;
  const size_t qrow = (size_t)b * h_q + 4 * h + qr;
  const float qx = (part[0][qr][j] + part[1][qr][j] + part[2][qr][j] + part[3][qr][j]) * qscale;
  float qsum = qx;
  {
    const int r = qr;
    const float x = qx;
    qrs[r][j] = x;
    float s = x, a = fabsf(x);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      s += __shfl_xor_sync(0xffffffffu, s, o);
      a = fmaxf(a, __shfl_xor_sync(0xffffffffu, a, o));
    }
    qsum = s;
    if (lane == 0) hmax[r][j >> 5] = a;
  }
  __syncthreads();
  // Tensor-core B fragments (see decode_tc.cu): per head a power-of-two
  // prescale 2^e brings max |q'| * 2^e into [2^13, 2^14), so that the fp16
  // hi/lo split stays in the normal range for all but tiny elements.  The
  // key codes enter the MMA as 1024 + code * 2^pos (pos = kCodePos[G&1][r]),
  // so the fragment of channel 32G + 4w + r also carries 2^-pos, and koff
  // holds the offset sum 1024 * sum over the group of the fragment values,
  // per (query head, group, hi/lo column), which the MMA starts from
  // (negated) so that the accumulator sums code * q' exactly as before.
  {
    const int ridx = tid;  // 512 fragment registers, one per thread
    const int L = ridx >> 4, reg = ridx & 15;
    const int G = reg >> 2, kk = (reg >> 1) & 1, which = reg & 1;
    const int g = L >> 2, c = L & 3;
    const int head = g >> 1, part_hl = g & 1;
    const float mx = fmaxf(fmaxf(hmax[head][0], hmax[head][1]),
                           fmaxf(hmax[head][2], hmax[head][3]));
    const int e = max(-100, min(100, mx > 0.f ? 13 - ilogbf(mx) : 0));
    const int r = 2 * kk + which;
    const int ch = 32 * G + 8 * c + r;   // low half; +4 high
    const float sc = ldexpf(1.f, e - code_pos(G, r));
    const float x0 = qrs[head][ch] * sc, x1 = qrs[head][ch + 4] * sc;
    const __half h0 = __float2half_rn(x0), h1 = __float2half_rn(x1);
    __half v0 = h0, v1 = h1;
    if (part_hl) {
      v0 = __float2half_rn(x0 - __half2float(h0));
      v1 = __float2half_rn(x1 - __half2float(h1));
    }
    const uint32_t fragv =
        (uint32_t)__half_as_ushort(v0) | ((uint32_t)__half_as_ushort(v1) << 16);
    // offset sum over the 32 channels of group G for column g: reduce over
    // (kk, which) = lane bits 0-1, c bit 0 = lane bit 4, c bit 1 = warp bit 0.
    // Exact, in fixed point: an fp16 value times 2^24 is an integer below
    // 2^40, so 64 of them sum exactly in int64; one rounding to float, then
    // 1024 * 2^-24 = 2^-14 (exact) gives the correctly rounded koff.
    long long t = __float2ll_rn(__half2float(v0) * 16777216.0f) +
                  __float2ll_rn(__half2float(v1) * 16777216.0f);
    t += __shfl_xor_sync(0xffffffffu, t, 1);
    t += __shfl_xor_sync(0xffffffffu, t, 2);
    t += __shfl_xor_sync(0xffffffffu, t, 16);
    if ((lane & 15) % 4 == 0) koff_part[warp][G] = t;
    __syncthreads();
    if (tid < 32) {  // tid = (g, G): koff[head][G][hl] for column g
      const int gg = tid >> 2, GG = tid & 3;
      const long long tot = koff_part[2 * gg][GG] + koff_part[2 * gg + 1][GG];
      koff[((size_t)b * h_kv + h) * 32 + (gg >> 1) * 8 + GG * 2 + (gg & 1)] =
          __ll2float_rn(tot) * 0x1p-14f;
    }
    if (ridx < 4) {
      const float m2 = fmaxf(fmaxf(hmax[ridx][0], hmax[ridx][1]),
                             fmaxf(hmax[ridx][2], hmax[ridx][3]));
      const int e2 = max(-100, min(100, m2 > 0.f ? 13 - ilogbf(m2) : 0));
      invs[(size_t)b * h_q + 4 * h + ridx] = ldexpf(1.f, -e2);
    }
    frag[((size_t)b * h_kv + h) * 512 + ridx] = fragv;
  }
  qf[qrow * kD + j] = qx;
  if (lane == 0) qs[qrow * kGroups + (j >> 5)] = qsum;
  if (tid == 0) cnt_ws[(size_t)b * h_kv + h] = 0;  // combine arrivals

  if (b != 0 || h != 0) return;
  // Split-K plan: pref[b] = INT2 pages of sequences < b, nzpref[b] =
  // sequences < b with INT2 pages.  Invalid lengths count as empty and are
  // flagged.
  int run_p = 0, run_n = 0;
  constexpr int kW = kQrotThreads / 32;
  for (int base = 0; base < B; base += kQrotThreads) {
    const int bb = base + tid;
    int np = 0;
    if (bb < B) {
      const int len = seq_lens[bb];
      if (len < 0 || (long long)len > (long long)max_pages * kPage)
        atomicOr(err, OPTR_DEVERR_SEQ_LEN);
      else
        np = int2_pages(len, sink, recent);
    }
    int xp = np, xn = np > 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int yp = __shfl_up_sync(0xffffffffu, xp, o);
      const int yn = __shfl_up_sync(0xffffffffu, xn, o);
      if (lane >= o) { xp += yp; xn += yn; }
    }
    if (lane == 31) { warp_tot[0][warp] = xp; warp_tot[1][warp] = xn; }
    __syncthreads();
    int op = run_p, on = run_n;
    for (int w = 0; w < warp; ++w) { op += warp_tot[0][w]; on += warp_tot[1][w]; }
    if (bb < B) { pref[bb + 1] = op + xp; nzpref[bb + 1] = on + xn; }
    if (bb == 0) { pref[0] = 0; nzpref[0] = 0; }
    for (int w = 0; w < kW; ++w) { run_p += warp_tot[0][w]; run_n += warp_tot[1][w]; }
    __syncthreads();
  }
}

__global__ void __launch_bounds__(kQrotThreads)
qrot_kernel(const __nv_bfloat16* __restrict__ q, const float* __restrict__ R_k,
            int B, int h_q, int h_kv, float qscale,
            const int32_t* __restrict__ seq_lens, int max_pages,
            float* __restrict__ qf, float* __restrict__ qs,
            uint32_t* __restrict__ frag, float* __restrict__ koff,
            float* __restrict__ invs, int* __restrict__ pref,
            int* __restrict__ nzpref, int* __restrict__ cnt_ws,
            unsigned* err, int sink, int recent) {
  __shared__ QrotSmem sm;
  qrot_body(blockIdx.x, blockIdx.y, sm, q, R_k, B, h_q, h_kv, qscale, seq_lens,
            max_pages, qf, qs, frag, koff, invs, pref, nzpref, cnt_ws, err,
            sink, recent);
}

// ------------------------------------------------- decode-step prologue
// One launch for the independent first steps of a decode step: the
// single-token cache write of every sequence (CTAs [0, n_app), as
// append_small_kernel), the window copy of the new tokens (the next n_wcp
// CTAs, BF16 windows only) and the query rotation (the following B * h_kv
// CTAs, as qrot_kernel).  All wait for the previous kernel before touching
// inputs; the partial kernel then waits for this grid, i.e. for all.
static_assert(kQrotThreads == 512, "one block size for every body");
static_assert(sizeof(float) * kPage * 4 >= (size_t)kWinPBytes, "window P scratch");

template <int T>
__global__ void __launch_bounds__(512)
step_prologue_kernel(
    int n_app, int app_tiles, const __nv_bfloat16* __restrict__ k,
    const __nv_bfloat16* __restrict__ v, int n_tok,
    const int32_t* __restrict__ cu_new, const int32_t* __restrict__ pos0,
    const int32_t* __restrict__ bt, uint8_t* __restrict__ pool, int num_pages,
    const float* __restrict__ R_v, const float* __restrict__ muR, float clip_k,
    float clip_v, const __nv_bfloat16* __restrict__ q,
    const float* __restrict__ R_k, int B, int h_q, int h_kv, float qscale,
    const int32_t* __restrict__ seq_lens, int max_pages,
    float* __restrict__ qf, float* __restrict__ qs, uint32_t* __restrict__ frag,
    float* __restrict__ koff, float* __restrict__ invs, int* __restrict__ pref,
    int* __restrict__ nzpref, int* __restrict__ cnt_ws, unsigned* err, int fold_v,
    int n_wcp, __nv_bfloat16* __restrict__ win,
    const int32_t* __restrict__ win_slot, int n_slots, int sink, int recent,
    int group128, int lead) {
  extern __shared__ __align__(16) unsigned char dsm_[];
  // Block order: `lead` query-rotation CTAs, the cache-write CTAs, then the
  // remaining query-rotation CTAs.  With lead = SMs - write CTAs, the first
  // wave gives every write CTA (the longest) an SM of its own and the CTAs
  // beyond one per SM are query rotations.
  int bid = blockIdx.x;
  if (bid < lead) {
    bid += n_app + n_wcp;  // a query rotation
  } else if (bid < lead + n_app + n_wcp) {
    bid -= lead;           // a cache write or window copy
  }
  if (bid < n_app) {
    const int tblk = bid % app_tiles, hk = (bid / app_tiles) % h_kv,
              kind = bid / (app_tiles * h_kv);
    append_small_body<T>(tblk, hk, kind, *reinterpret_cast<AppendSmallSmemT<T>*>(dsm_),
                      k, v, n_tok, cu_new, pos0, bt, B, max_pages, pool,
                      num_pages, h_kv, R_k, R_v, muR, clip_k, clip_v, err,
                      fold_v && kind == 1, group128 != 0);
  } else if (bid < n_app + n_wcp) {
    window_copy_body(bid - n_app, *reinterpret_cast<WinCopySmem*>(dsm_), k, v,
                     n_tok, cu_new, pos0, B, win, win_slot, n_slots, h_kv,
                     sink, recent, err);
  } else {
    const int r = bid - n_app - n_wcp;
    qrot_body(r / h_kv, r % h_kv, *reinterpret_cast<QrotSmem*>(dsm_), q, R_k, B,
              h_q, h_kv, qscale, seq_lens, max_pages, qf, qs, frag, koff, invs,
              pref, nzpref, cnt_ws, err, sink, recent);
  }
}

// Window part of a separate cache write (512 threads per 16 new tokens).
__global__ void __launch_bounds__(512)
window_copy_kernel(const __nv_bfloat16* __restrict__ k,
                   const __nv_bfloat16* __restrict__ v, int n_tok,
                   const int32_t* __restrict__ cu_new,
                   const int32_t* __restrict__ pos0, int B,
                   __nv_bfloat16* __restrict__ win,
                   const int32_t* __restrict__ win_slot, int n_slots, int h_kv,
                   int sink, int recent, unsigned* err) {
  __shared__ WinCopySmem sm;
  window_copy_body(blockIdx.x, sm, k, v, n_tok, cu_new, pos0, B, win, win_slot,
                   n_slots, h_kv, sink, recent, err);
}

// ------------------------------------------------- CUDA-core partial kernel

struct WarpSmemCC {
  union {  // the window phase runs before the first page is staged
    alignas(16) uint8_t stage[2][kChunk];
    alignas(16) uint8_t wst[kWinStageBytes];
  };
  float qv[4][kD];
  float qsum[4][kGroups];
  float p[kPage][4];
};

template <bool WIN>  // WIN: with the BF16-window phase
__global__ void __launch_bounds__(128)
partial_cuda_core_kernel(const uint8_t* __restrict__ pool,
                         const int32_t* __restrict__ bt,
                         const int32_t* __restrict__ seq_lens, int B,
                         int max_pages, int num_pages, int h_q, int h_kv,
                         const float* __restrict__ qf,
                         const float* __restrict__ qs,
                         const int* __restrict__ pref,
                         const int* __restrict__ nzpref,
                         float* __restrict__ part, int W, unsigned* err,
                         int sink, int recent, WinPhase wp, int compact) {
  // compact: the G = 128 record (one scale/min pair per slot, 1152 bytes)
  __shared__ WarpSmemCC smem[4];
  const int chunk = chunk_bytes(compact != 0);
  const int mstride = meta_stride(compact != 0);
  const int vmeta = vmeta_offset(compact != 0);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  WarpSmemCC& S = smem[warp];
  const int w = blockIdx.x * 4 + warp;
  // BF16 windows first, before waiting for the previous kernel (the phase
  // reads only inputs and library-owned state); stage and p are free until
  // the first segment
  if constexpr (WIN) {
    if (w < wp.Ww) window_phase(w, wp, S.wst, reinterpret_cast<uint8_t*>(&S.p[0][0]));
  }
  pdl_wait();
  pdl_trigger();
  const int poff = sink / kPage;  // first INT2 page
  const long long F = (long long)__ldcg(pref + B) * h_kv;
  long long f = w * F / W;
  const long long f1 = (w + 1) * F / W;

  while (f < f1) {
    Segment sg = locate_segment(f, f1, pref, B, h_kv);
    const int b = sg.b, h = sg.h;
    const int len = int2_end(__ldg(seq_lens + b), sink, recent);  // INT2 end
    // rotated queries of the GQA group
    for (int i = lane; i < 4 * kD; i += 32)
      S.qv[i / kD][i % kD] = __ldcg(qf + ((size_t)b * h_q + 4 * h) * kD + i);
    if (lane < 16)
      S.qsum[lane / 4][lane % 4] = __ldcg(qs + ((size_t)b * h_q + 4 * h) * kGroups + lane);
    float m[4], l[4], acc[4][4];
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      m[r] = -INFINITY;
      l[r] = 0.f;
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[r][c] = 0.f;
    }
    const int32_t* btb = bt + (size_t)b * max_pages;
    // 2-stage cp.async pipeline over the segment's pages
    bool ok0 = issue_page(S.stage[0], pool, btb, poff + sg.p0, num_pages, h_kv, h, lane, err,
                          chunk);
    bool okn = false;
    for (int i = 0; i < sg.n; ++i) {
      const bool ok = (i == 0) ? ok0 : okn;
      if (i + 1 < sg.n)
        okn = issue_page(S.stage[(i + 1) & 1], pool, btb, poff + sg.p0 + i + 1,
                         num_pages, h_kv, h, lane, err, chunk);
      else
        cp_async_commit();
      cp_async_wait_1();
      __syncwarp();
      const uint8_t* st = S.stage[i & 1];
      const int page = poff + sg.p0 + i;
      int nvalid = ok ? min(kPage, len - page * kPage) : 0;
      __syncwarp();

      // logits: lane -> token t, heads hp and hp+1
      const int t = lane & 15, hp = (lane >> 4) * 2;
      float lg0 = -INFINITY, lg1 = -INFINITY;
      if (t < nvalid) {
        float a0 = 0.f, a1 = 0.f;
        const uint8_t* kc = st + OPTR_K_CODES_OFFSET + t * 32;
        const __half2* km = reinterpret_cast<const __half2*>(st + OPTR_K_META_OFFSET + t * mstride);
#pragma unroll
        for (int G = 0; G < kGroups; ++G) {
          float d0 = 0.f, d1 = 0.f;
#pragma unroll
          for (int wd = 0; wd < 8; ++wd) {
            const unsigned byte = kc[4 * wd + G];
#pragma unroll
            for (int r = 0; r < 4; ++r) {
              const float c = (float)((byte >> (2 * r)) & 3u);
              const int ch = 32 * G + 4 * wd + r;
              d0 = fmaf(S.qv[hp][ch], c, d0);
              d1 = fmaf(S.qv[hp + 1][ch], c, d1);
            }
          }
          const float2 sm = __half22float2(km[compact ? 0 : G]);
          a0 += sm.x * d0 + sm.y * S.qsum[hp][G];
          a1 += sm.x * d1 + sm.y * S.qsum[hp + 1][G];
        }
        lg0 = a0;
        lg1 = a1;
      }
      // online softmax over the 16 tokens of each head
      float t0 = lg0, t1 = lg1;
#pragma unroll
      for (int o = 1; o < 16; o <<= 1) {
        t0 = fmaxf(t0, __shfl_xor_sync(0xffffffffu, t0, o));
        t1 = fmaxf(t1, __shfl_xor_sync(0xffffffffu, t1, o));
      }
      float tmax[4];
      tmax[0] = __shfl_sync(0xffffffffu, t0, 0);
      tmax[1] = __shfl_sync(0xffffffffu, t1, 0);
      tmax[2] = __shfl_sync(0xffffffffu, t0, 16);
      tmax[3] = __shfl_sync(0xffffffffu, t1, 16);
      float alpha[4], mnew[4];
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        mnew[r] = fmaxf(m[r], tmax[r]);
        alpha[r] = (mnew[r] == -INFINITY) ? 1.f : exp2f(m[r] - mnew[r]);
      }
      const float p0 = (lg0 == -INFINITY) ? 0.f : exp2f(lg0 - mnew[hp]);
      const float p1 = (lg1 == -INFINITY) ? 0.f : exp2f(lg1 - mnew[hp + 1]);
      S.p[t][hp] = p0;
      S.p[t][hp + 1] = p1;
      float s0 = p0, s1 = p1;
#pragma unroll
      for (int o = 1; o < 16; o <<= 1) {
        s0 += __shfl_xor_sync(0xffffffffu, s0, o);
        s1 += __shfl_xor_sync(0xffffffffu, s1, o);
      }
      float psum[4];
      psum[0] = __shfl_sync(0xffffffffu, s0, 0);
      psum[1] = __shfl_sync(0xffffffffu, s1, 0);
      psum[2] = __shfl_sync(0xffffffffu, s0, 16);
      psum[3] = __shfl_sync(0xffffffffu, s1, 16);
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        l[r] = l[r] * alpha[r] + psum[r];
        m[r] = mnew[r];
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[r][c] *= alpha[r];
      }
      __syncwarp();
      // PV: lane -> byte `lane` of the value codes (4 channels of group lane%4)
      const int G = lane & 3;
      for (int tt = 0; tt < nvalid; ++tt) {
        const unsigned byte = st[OPTR_V_CODES_OFFSET + tt * 32 + lane];
        const float2 sm = __half22float2(
            reinterpret_cast<const __half2*>(st + vmeta + tt * mstride)[compact ? 0 : G]);
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const float vv = fmaf((float)((byte >> (2 * c)) & 3u), sm.x, sm.y);
#pragma unroll
          for (int r = 0; r < 4; ++r) acc[r][c] = fmaf(S.p[tt][r], vv, acc[r][c]);
        }
      }
      __syncwarp();
    }
    // partial slot of this segment
    float* dst = part + (size_t)(w + nzpref[b] * h_kv + h) * kPartFloats;
    const int wd = lane >> 2, G = lane & 3;
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
      for (int c = 0; c < 4; ++c) dst[r * kD + 32 * G + 4 * wd + c] = acc[r][c];
    if (lane < 4) {
      dst[kPartM + lane] = m[lane];
      dst[kPartL + lane] = l[lane];
    }
    f = sg.f_end;
  }
}

// ------------------------------------------------------------- combine

// Grid (B, h_kv, S), 512 threads.  CTA (b, h, s) merges chunk s of the
// segment partials of (b, h) (log-sum-exp merge, Sec. 3 Eq. 1-2 split over
// the context); with S = 1 it also normalises and rotates back,
// out = o' R_v^T.  With S > 1 each CTA writes its chunk's (m, l, o') to
// the workspace, and the last CTA of (b, h) to arrive (atomic counter,
// zeroed by qrot) merges the S chunk results and rotates.  Before waiting
// for the partial kernel every CTA copies this head's R_v^T (64 KB,
// library-owned) into shared memory, so the rotation never waits on global
// memory.  Partials are read 32 at a time: the headers and the o' float4s
// of a batch are all requested before any is used.
constexpr int kCombineThreads = 512;
constexpr int kCombineBatch = 32;

struct CombineState {
  float M[4], L[4];      // running maxima / sums per query head
  float alpha[4];        // rescale of the accumulators for the batch
  float w[kCombineBatch][4];
  float red[kCombineThreads / 32][4];
};

// Merge cnt (<= kCombineBatch) partials at base + i * kPartFloats into the
// running state st and the thread's float4 accumulator acc (float4 v of
// o'[4][128] over the partials i = ph (mod 4)).  first_w >= 0 marks partial
// slots of warps first_w + i, which may be empty (never written) when
// sparse; their weight is 0 and their values are never accumulated.
__device__ __forceinline__ void combine_batch(const float* base, int cnt,
                                              int first_w, bool sparse,
                                              long long F, int W,
                                              CombineState& st, float4& acc) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int v = tid & 127, ph = tid >> 7, hd = v >> 5;
  // issue every load of the batch first
  float m = -INFINITY, l = 0.f;
  bool hv = false;
  if (tid < 4 * cnt) {
    hv = !(sparse && first_w >= 0 && warp_empty(first_w + (tid >> 2), F, W));
    if (hv) {
      const float* pp = base + (size_t)(tid >> 2) * kPartFloats;
      m = __ldcg(pp + kPartM + (tid & 3));
      l = __ldcg(pp + kPartL + (tid & 3));
    }
  }
  float4 a[kCombineBatch / 4];
#pragma unroll
  for (int j = 0; j < kCombineBatch / 4; ++j) {
    const int i = ph + 4 * j;
    a[j] = i < cnt ? __ldcg(reinterpret_cast<const float4*>(base + (size_t)i * kPartFloats) + v)
                   : make_float4(0.f, 0.f, 0.f, 0.f);
  }
  // batch maximum per head (thread t's head is t & 3 == lane & 3)
  float mx = m;
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  if (lane < 4) st.red[warp][lane] = mx;
  __syncthreads();
  if (tid < 4) {
    float bm = -INFINITY;
    for (int w = 0; w < kCombineThreads / 32; ++w) bm = fmaxf(bm, st.red[w][tid]);
    const float Mn = fmaxf(st.M[tid], bm);
    st.alpha[tid] = merge_weight(st.M[tid], Mn);
    st.M[tid] = Mn;
  }
  __syncthreads();
  const float Mh = st.M[lane & 3];
  float wl = 0.f;
  if (tid < 4 * cnt) {
    const float wgt = hv ? merge_weight(m, Mh) : 0.f;
    st.w[tid >> 2][tid & 3] = wgt;
    wl = l * wgt;
  }
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) wl += __shfl_xor_sync(0xffffffffu, wl, o);
  if (lane < 4) st.red[warp][lane] = wl;
  __syncthreads();
  if (tid < 4) {
    float sl = 0.f;
    for (int w = 0; w < kCombineThreads / 32; ++w) sl += st.red[w][tid];
    st.L[tid] = st.L[tid] * st.alpha[tid] + sl;
  }
  const float al = st.alpha[hd];
  acc.x *= al;
  acc.y *= al;
  acc.z *= al;
  acc.w *= al;
#pragma unroll
  for (int j = 0; j < kCombineBatch / 4; ++j) {
    const int i = ph + 4 * j;
    const float wv = i < cnt ? st.w[i][hd] : 0.f;
    if (wv != 0.f) {
      acc.x = fmaf(a[j].x, wv, acc.x);
      acc.y = fmaf(a[j].y, wv, acc.y);
      acc.z = fmaf(a[j].z, wv, acc.z);
      acc.w = fmaf(a[j].w, wv, acc.w);
    }
  }
  __syncthreads();  // st.w / st.red are reused by the next batch
}

__global__ void __launch_bounds__(kCombineThreads)
combine_kernel(const float* __restrict__ part, const int* __restrict__ pref,
               const int* __restrict__ nzpref, int B, int h_q, int h_kv, int W,
               const float* __restrict__ R_vT, float* __restrict__ cpart,
               int* __restrict__ cnt_ws, float* __restrict__ out, int fold_v,
               const float* __restrict__ wpart,
               const int32_t* __restrict__ seq_lens, int max_pages, int sink,
               int recent, int Uw, int Ww) {
  extern __shared__ float4 dsm[];
  float* rts = reinterpret_cast<float*>(dsm);  // [128][128] R_v^T[h]
  __shared__ float4 msum[4][kD];               // [phase][float4 of o']
  __shared__ float4 msumw[4][kD];              // the same for the windows
  __shared__ float orot[4][kD];
  __shared__ float ow[4][kD];                  // window output (unrotated)
  __shared__ CombineState st;
  __shared__ int last;
  const int b = blockIdx.x, h = blockIdx.y, sp = blockIdx.z, S = gridDim.z;
  const int tid = threadIdx.x;
  if (!fold_v) {
    const float4* src = reinterpret_cast<const float4*>(R_vT + (size_t)h * kD * kD);
#pragma unroll
    for (int u = 0; u < kD * kD / 4 / kCombineThreads; ++u)
      cp_async16(&dsm[tid + u * kCombineThreads], src + tid + u * kCombineThreads);
  }
  cp_async_commit();
  if (tid < 4) {
    st.M[tid] = -INFINITY;
    st.L[tid] = 0.f;
  }
  // The page prefix sums were written by qrot, two kernels back: the
  // partial kernel only lets this grid launch after its own pdl_wait(),
  // i.e. after qrot completed with its writes visible, so they are read
  // (through L2) before waiting for the partials themselves.
  const int np = __ldcg(pref + b + 1) - __ldcg(pref + b);
  const long long F = (long long)__ldcg(pref + B) * h_kv;
  const long long fs = (long long)__ldcg(pref + b) * h_kv + (long long)h * np;
  const int nzb = __ldcg(nzpref + b);
  int w0 = 0, n = 0;
  if (np > 0) {
    w0 = warp_of(fs, F, W);
    n = warp_of(fs + np - 1, F, W) - w0 + 1;
  }
  const bool sparse = F < W;
  const float* pbase = part + ((size_t)nzb * h_kv + h + w0) * kPartFloats;
  const int i0 = sp * n / S, i1 = (sp + 1) * n / S;  // n <= W: no overflow
  // BF16-window partials of (b, h): the window warps that own its units
  // 0 .. nwu - 1 (window.cuh), one slot each, no gaps
  int ww0 = 0, wn = 0;
  if (Ww > 0) {
    int len = __ldg(seq_lens + b);
    if (len < 0 || (long long)len > (long long)max_pages * kPage) len = 0;
    const int nwu = (win_count(len, sink, recent) + kWinUnit - 1) / kWinUnit;
    if (nwu > 0) {
      const long long U = (long long)B * h_kv * Uw;
      const long long u0 = ((long long)b * h_kv + h) * Uw;
      ww0 = warp_of(u0, U, Ww);
      wn = warp_of(u0 + nwu - 1, U, Ww) - ww0 + 1;
    }
  }
  pdl_wait();
  pdl_trigger();
  float* ob = out + ((size_t)b * h_q + 4 * h) * kD;
  if (np == 0 && (wn == 0 || sp != 0)) {  // nothing, or windows only (CTA 0)
    if (sp == 0) ob[tid] = 0.f;
    cp_async_wait<0>();
    return;
  }
  __syncthreads();  // st initialised
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int i = i0; i < i1; i += kCombineBatch)
    combine_batch(pbase + (size_t)i * kPartFloats, min(kCombineBatch, i1 - i),
                  w0 + i, sparse, F, W, st, acc);
  const int v = tid & 127, ph = tid >> 7;
  if (S > 1 && np > 0) {
    msum[ph][v] = acc;
    __syncthreads();
    // publish this chunk: o'[4][128], M[4], L[4] in the partial format
    const size_t seg = (size_t)b * h_kv + h;
    float* cp = cpart + (seg * S + sp) * kPartFloats;
    if (tid < kD) {
      const float4 a = msum[0][tid], b1 = msum[1][tid], c = msum[2][tid], d = msum[3][tid];
      reinterpret_cast<float4*>(cp)[tid] =
          make_float4((a.x + b1.x) + (c.x + d.x), (a.y + b1.y) + (c.y + d.y),
                      (a.z + b1.z) + (c.z + d.z), (a.w + b1.w) + (c.w + d.w));
    } else if (tid < kD + 4) {
      cp[kPartM + tid - kD] = st.M[tid - kD];
      cp[kPartL + tid - kD] = st.L[tid - kD];
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) last = atomicAdd(cnt_ws + seg, 1) == S - 1;
    __syncthreads();
    if (!last) {
      cp_async_wait<0>();
      return;
    }
    __threadfence();
    if (tid < 4) {
      st.M[tid] = -INFINITY;
      st.L[tid] = 0.f;
    }
    if (tid == 0) cnt_ws[seg] = 0;
    __syncthreads();
    acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int i = 0; i < S; i += kCombineBatch)
      combine_batch(cpart + (seg * S + i) * kPartFloats, min(kCombineBatch, S - i),
                    -1, false, F, W, st, acc);
  }
  // The final CTA of (b, h) merges the window partials into a second
  // accumulator under the same running maxima; each batch's rescale of the
  // maxima applies to the INT2 accumulator as well.
  float4 accw = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int i = 0; i < wn; i += kCombineBatch) {
    combine_batch(wpart + (size_t)(ww0 + b * h_kv + h + i) * kPartFloats,
                  min(kCombineBatch, wn - i), -1, false, 0, 1, st, accw);
    const float al = st.alpha[v >> 5];
    acc.x *= al;
    acc.y *= al;
    acc.z *= al;
    acc.w *= al;
  }
  msum[ph][v] = acc;
  msumw[ph][v] = accw;
  __syncthreads();
  if (tid < kD) {
    const float4 a = msum[0][tid], b1 = msum[1][tid], c = msum[2][tid], d = msum[3][tid];
    const int hd = tid >> 5, ch = (tid & 31) * 4;
    const float L = st.L[hd];
    const float il = L > 0.f ? 1.f / L : 0.f;
    orot[hd][ch + 0] = ((a.x + b1.x) + (c.x + d.x)) * il;
    orot[hd][ch + 1] = ((a.y + b1.y) + (c.y + d.y)) * il;
    orot[hd][ch + 2] = ((a.z + b1.z) + (c.z + d.z)) * il;
    orot[hd][ch + 3] = ((a.w + b1.w) + (c.w + d.w)) * il;
    const float4 e = msumw[0][tid], f = msumw[1][tid], g = msumw[2][tid], k = msumw[3][tid];
    ow[hd][ch + 0] = ((e.x + f.x) + (g.x + k.x)) * il;
    ow[hd][ch + 1] = ((e.y + f.y) + (g.y + k.y)) * il;
    ow[hd][ch + 2] = ((e.z + f.z) + (g.z + k.z)) * il;
    ow[hd][ch + 3] = ((e.w + f.w) + (g.w + k.w)) * il;
  }
  cp_async_wait<0>();
  __syncthreads();
  if (fold_v) {  // output in the folded value basis: no R_v^T
    ob[tid] = orot[tid >> 7][tid & 127] + ow[tid >> 7][tid & 127];
    return;
  }
  // out[r][i] = sum_k o'[r][k] R_v[i][k] = sum_k o'[r][k] R_vT[k][i]:
  // thread (i, q) sums k in [32q, 32q + 32) for the 4 heads, reading each
  // R_v^T element once; the 4 quarters are added through shared memory.
  {
    const int i = tid & 127, q = tid >> 7;
    float acc4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
    for (int k = 32 * q; k < 32 * q + 32; ++k) {
      const float rt = rts[k * kD + i];
#pragma unroll
      for (int r = 0; r < 4; ++r) acc4[r] = fmaf(orot[r][k], rt, acc4[r]);
    }
    float* qs4 = reinterpret_cast<float*>(msum);  // reuse: [4 quarters][4][128]
#pragma unroll
    for (int r = 0; r < 4; ++r) qs4[(q * 4 + r) * kD + i] = acc4[r];
    __syncthreads();
    const int r = tid >> 7;
    ob[r * kD + i] = ((qs4[(0 * 4 + r) * kD + i] + qs4[(1 * 4 + r) * kD + i]) +
                      (qs4[(2 * 4 + r) * kD + i] + qs4[(3 * 4 + r) * kD + i])) +
                     ow[r][i];
  }
}

// The one-CTA-per-segment combine (S = 1) without block-wide merging steps:
// grid (B, h_kv), 512 threads, warp (r, qq) = (query head 4h + r, channels
// 32qq .. 32qq + 31).  Every warp merges the segment's partials for its own
// head and channels on its own (the maxima, weights and sums by shuffles),
// with the headers and its o' values of up to kFastBatch partials requested
// at once, then the BF16-window partials of the segment (if any) into a
// second accumulator under the same running maxima; a single barrier then
// hands the normalised o' to the rotation, in which warp (r, qq) produces
// outputs 32qq + lane of head r over all 128 input channels (the window
// part, computed on the unrotated values, is added after it).
constexpr int kFastBatch = 32;

__global__ void __launch_bounds__(kCombineThreads)
combine_fast_kernel(const float* __restrict__ part, const int* __restrict__ pref,
                    const int* __restrict__ nzpref, int B, int h_q, int h_kv, int W,
                    const float* __restrict__ R_vT, float* __restrict__ out,
                    int fold_v, const float* __restrict__ wpart,
                    const int32_t* __restrict__ seq_lens, int max_pages, int sink,
                    int recent, int Uw, int Ww) {
  extern __shared__ float4 dsm[];
  float* rts = reinterpret_cast<float*>(dsm);  // [128][128] R_v^T[h]
  __shared__ __align__(16) float orot[4][kD];
  const int b = blockIdx.x, h = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int r = warp >> 2, ch = 32 * (warp & 3) + lane;
  if (!fold_v) {
    const float4* src = reinterpret_cast<const float4*>(R_vT + (size_t)h * kD * kD);
#pragma unroll
    for (int u = 0; u < kD * kD / 4 / kCombineThreads; ++u)
      cp_async16(&dsm[tid + u * kCombineThreads], src + tid + u * kCombineThreads);
  }
  cp_async_commit();
  // the page prefix sums come from the query rotation, two kernels back
  // (complete before the partial kernel let this grid launch)
  const int np = __ldcg(pref + b + 1) - __ldcg(pref + b);
  const long long F = (long long)__ldcg(pref + B) * h_kv;
  const long long fs = (long long)__ldcg(pref + b) * h_kv + (long long)h * np;
  const int nzb = __ldcg(nzpref + b);
  int w0 = 0, n = 0;
  if (np > 0) {
    w0 = warp_of(fs, F, W);
    n = warp_of(fs + np - 1, F, W) - w0 + 1;
  }
  const bool sparse = F < W;
  const float* pbase = part + ((size_t)nzb * h_kv + h + w0) * kPartFloats;
  // BF16-window partials of (b, h): the window warps that own its units
  // 0 .. nwu - 1 (window.cuh), one slot each, no gaps
  int wn = 0;
  const float* wbase = nullptr;
  if (Ww > 0) {
    int len = __ldg(seq_lens + b);
    if (len < 0 || (long long)len > (long long)max_pages * kPage) len = 0;
    const int nwu = (win_count(len, sink, recent) + kWinUnit - 1) / kWinUnit;
    if (nwu > 0) {
      const long long U = (long long)B * h_kv * Uw;
      const long long u0 = ((long long)b * h_kv + h) * Uw;
      const int ww0 = warp_of(u0, U, Ww);
      wn = warp_of(u0 + nwu - 1, U, Ww) - ww0 + 1;
      wbase = wpart + (size_t)(ww0 + b * h_kv + h) * kPartFloats;
    }
  }
  pdl_wait();
  pdl_trigger();
  float* ob = out + ((size_t)b * h_q + 4 * h) * kD;
  if (np == 0 && wn == 0) {  // no cached token: the output is 0
    ob[tid] = 0.f;
    cp_async_wait<0>();
    return;
  }
  // running maximum M and sum L of head r; accumulators of channel ch:
  // o (INT2 partials) and ow (window partials)
  float M = -INFINITY, L = 0.f, o = 0.f, ow = 0.f;
  // one batch of up to kFastBatch partials at base (empty slots skipped
  // when sparse: only the INT2 slots of warps that own no page); the
  // accumulator acc takes the batch, both are rescaled to the new maximum
  auto merge = [&](const float* base, int cnt, bool sp, int wfirst, float& acc) {
    float m = -INFINITY, l = 0.f;
    if (lane < cnt && !(sp && warp_empty(wfirst + lane, F, W))) {
      const float* pp = base + (size_t)lane * kPartFloats;
      m = __ldcg(pp + kPartM + r);
      l = __ldcg(pp + kPartL + r);
    }
    float ov[kFastBatch];
#pragma unroll
    for (int i = 0; i < kFastBatch; ++i)
      ov[i] = i < cnt ? __ldcg(base + (size_t)i * kPartFloats + r * kD + ch) : 0.f;
    float bm = m;
#pragma unroll
    for (int x = 16; x > 0; x >>= 1) bm = fmaxf(bm, __shfl_xor_sync(0xffffffffu, bm, x));
    const float Mn = fmaxf(M, bm);
    const float alpha = merge_weight(M, Mn);
    const float wgt = merge_weight(m, Mn);  // 0 for an empty partial
    float wl = wgt * l;
#pragma unroll
    for (int x = 16; x > 0; x >>= 1) wl += __shfl_xor_sync(0xffffffffu, wl, x);
    L = L * alpha + wl;
    o *= alpha;
    ow *= alpha;
#pragma unroll
    for (int i = 0; i < kFastBatch; ++i) {
      const float wi = __shfl_sync(0xffffffffu, wgt, i);
      if (wi != 0.f) acc = fmaf(ov[i], wi, acc);
    }
    M = Mn;
  };
  for (int i0 = 0; i0 < n; i0 += kFastBatch)
    merge(pbase + (size_t)i0 * kPartFloats, min(kFastBatch, n - i0), sparse, w0 + i0, o);
  for (int j0 = 0; j0 < wn; j0 += kFastBatch)
    merge(wbase + (size_t)j0 * kPartFloats, min(kFastBatch, wn - j0), false, 0, ow);
  const float il = L > 0.f ? 1.f / L : 0.f;
  orot[r][ch] = o * il;
  const float owin = ow * il;  // window part (values unrotated)
  cp_async_wait<0>();
  __syncthreads();
  if (fold_v) {  // output in the folded value basis: no R_v^T
    ob[r * kD + ch] = orot[r][ch] + owin;
    return;
  }
  // out[r][i] = sum_k o'[r][k] R_v^T[k][i], i = ch
  float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll 8
  for (int k = 0; k < kD; k += 4) {
    const float4 ok = *reinterpret_cast<const float4*>(&orot[r][k]);
    a0 = fmaf(ok.x, rts[(k + 0) * kD + ch], a0);
    a1 = fmaf(ok.y, rts[(k + 1) * kD + ch], a1);
    a2 = fmaf(ok.z, rts[(k + 2) * kD + ch], a2);
    a3 = fmaf(ok.w, rts[(k + 3) * kD + ch], a3);
  }
  ob[r * kD + ch] = ((a0 + a1) + (a2 + a3)) + owin;
}

}  // namespace

cudaError_t launch_partial_tensor(const optr_params* p, const uint8_t* pool,
                                  const int32_t* bt, const int32_t* seq_lens,
                                  int B, int max_pages, int num_pages,
                                  const uint32_t* frag, const float* koff,
                                  const float* invs, const float* qs,
                                  const int* pref, const int* nzpref,
                                  float* part, int W, bool early_pages,
                                  const int32_t* step_cu, const int32_t* step_pos0,
                                  const WinPhase& wp, cudaStream_t s);

cudaError_t launch_window_copy(const optr_params* p, const __nv_bfloat16* k,
                               const __nv_bfloat16* v, int n_tok,
                               const int32_t* cu_new, const int32_t* pos0,
                               int B, const WinArgs& win, cudaStream_t s) {
  const int tiles = (n_tok + kWinCopyTok - 1) / kWinCopyTok;
  return launch_pdl(window_copy_kernel, dim3(tiles), dim3(512), 0, s, k, v,
                    n_tok, cu_new, pos0, B, win.win, win.slot, win.n_slots,
                    p->cfg.h_kv, p->cfg.sink, p->cfg.recent, p->err);
}

cudaError_t launch_decode(const optr_params* p, int variant,
                          const __nv_bfloat16* q, const int32_t* bt,
                          const int32_t* seq_lens, int B, int max_pages,
                          const uint8_t* pool, int num_pages, float* out,
                          void* ws, const DecodePlan& plan, cudaStream_t s,
                          const StepAppend* app, const WinArgs* win) {
  char* w = static_cast<char*>(ws);
  float* qf = reinterpret_cast<float*>(w + plan.off_qf);
  float* qs = reinterpret_cast<float*>(w + plan.off_qs);
  uint32_t* frag = reinterpret_cast<uint32_t*>(w + plan.off_frag);
  float* koff = reinterpret_cast<float*>(w + plan.off_koff);
  float* invs = reinterpret_cast<float*>(w + plan.off_invs);
  int* pref = reinterpret_cast<int*>(w + plan.off_pref);
  int* nzpref = pref + (B + 1);
  float* part = reinterpret_cast<float*>(w + plan.off_part);
  const int h_q = p->cfg.h_q, h_kv = p->cfg.h_kv;
  const int sink = p->cfg.sink, recent = p->cfg.recent;
  const float qscale = kLog2e / sqrtf((float)kD);
  // BF16 windows: the window partials, computed by the partial kernel
  const bool windows = plan.Ww > 0;
  WinPhase wp{};
  wp.Ww = 0;
  if (windows) {
    wp.q = q;
    wp.win = win->win;
    wp.slot = win->slot;
    wp.seq_lens = seq_lens;
    wp.mu = p->mu;
    wp.wpart = reinterpret_cast<float*>(w + plan.off_wpart);
    if (app) {  // the step's new rows, read directly (see WinPhase)
      wp.k_new = app->k;
      wp.v_new = app->v;
      wp.cu_new = app->cu_new;
      wp.pos0 = app->pos0;
    }
    wp.err = p->err;
    wp.n_slots = win->n_slots;
    wp.B = B;
    wp.h_q = h_q;
    wp.h_kv = h_kv;
    wp.max_pages = max_pages;
    wp.sink = sink;
    wp.recent = recent;
    wp.Uw = plan.Uw;
    wp.Ww = plan.Ww;
    wp.qscale = qscale;
  }

  int* cnt_ws = reinterpret_cast<int*>(w + plan.off_cnt);
  cudaError_t e;
  if (app) {
    // the cache write of the step (INT2 records and window copies) and the
    // query rotation in one launch
    prof_mark(p, 0, s);
    const int T = small_tile(app->n_tok);
    const int tiles = (app->n_tok + T - 1) / T;
    const int n_app = tiles * h_kv * 2;
    const int n_wcp = windows ? (app->n_tok + kWinCopyTok - 1) / kWinCopyTok : 0;
    const size_t sm_app = T == kSmallTokFew ? sizeof(AppendSmallSmemT<kSmallTokFew>)
                                            : sizeof(AppendSmallSmemT<kSmallTok>);
    size_t sm_bytes = sm_app > sizeof(QrotSmem) ? sm_app : sizeof(QrotSmem);
    if (sm_bytes < sizeof(WinCopySmem)) sm_bytes = sizeof(WinCopySmem);
    auto fn = T == kSmallTokFew ? step_prologue_kernel<kSmallTokFew>
                                : step_prologue_kernel<kSmallTok>;
    e = ensure_dynamic_smem(reinterpret_cast<const void*>(fn), sm_bytes);
    if (e != cudaSuccess) return e;
    e = launch_pdl(fn, dim3(n_app + n_wcp + B * h_kv), dim3(512),
                   sm_bytes, s, n_app, tiles, app->k, app->v, app->n_tok,
                   app->cu_new, app->pos0, bt, app->pool, num_pages,
                   (const float*)p->R_v, (const float*)p->muR, p->cfg.clip_k,
                   p->cfg.clip_v, q, (const float*)p->R_k, B, h_q, h_kv, qscale,
                   seq_lens, max_pages, qf, qs, frag, koff, invs, pref, nzpref,
                   cnt_ws, p->err, p->fold_v, n_wcp,
                   windows ? win->win : (__nv_bfloat16*)nullptr,
                   windows ? win->slot : (const int32_t*)nullptr,
                   windows ? win->n_slots : 0, sink, recent,
                   p->cfg.group == 128 ? 1 : 0,
                   std::max(0, std::min(B * h_kv, p->num_sms - n_app - n_wcp)));
    if (e != cudaSuccess) return e;
    prof_mark(p, 1, s);  // the append stage covers the fused launch,
    prof_mark(p, 2, s);  // the query-rotation stage is empty
  } else {
    prof_mark(p, 2, s);
    e = launch_pdl(qrot_kernel, dim3(B, h_kv), dim3(kQrotThreads), 0, s, q,
                   p->R_k, B, h_q, h_kv, qscale, seq_lens, max_pages, qf, qs,
                   frag, koff, invs, pref, nzpref, cnt_ws, p->err, sink,
                   recent);
    if (e != cudaSuccess) return e;
  }
  prof_mark(p, 3, s);
  if (variant != OPTR_VARIANT_CUDA_CORE) {
    // after a separate append the pool is complete before qrot starts, so
    // the partial kernel may fetch pages before waiting for qrot; after the
    // fused prologue it must wait first
    e = launch_partial_tensor(p, pool, bt, seq_lens, B, max_pages, num_pages,
                              frag, koff, invs, qs, pref, nzpref, part, plan.W,
                              app == nullptr, app ? app->cu_new : nullptr,
                              app ? app->pos0 : nullptr, wp, s);
  } else {
    e = launch_pdl(windows ? partial_cuda_core_kernel<true> : partial_cuda_core_kernel<false>,
                   dim3(plan.W / 4), dim3(128), 0, s,
                   pool, bt, seq_lens, B, max_pages, num_pages, h_q, h_kv, qf,
                   qs, pref, nzpref, part, plan.W, p->err, sink, recent, wp,
                   p->cfg.group == 128 ? 1 : 0);
  }
  if (e != cudaSuccess) return e;
  prof_mark(p, 4, s);
  // R_v^T (64 KB) plus padding: more than half of an SM's shared memory,
  // so no two combine CTAs share an SM (in a decode step they take SMs as
  // the partial kernel's CTAs leave them)
  const size_t cmb_bytes = 120 * 1024;
  if (plan.S == 1) {
    e = ensure_dynamic_smem(reinterpret_cast<const void*>(&combine_fast_kernel),
                            cmb_bytes);
    if (e != cudaSuccess) return e;
    e = launch_pdl(combine_fast_kernel, dim3(B, h_kv), dim3(kCombineThreads),
                   cmb_bytes, s, (const float*)part, (const int*)pref,
                   (const int*)nzpref, B, h_q, h_kv, plan.W, (const float*)p->R_vT,
                   out, p->fold_v, (const float*)wp.wpart, seq_lens, max_pages,
                   sink, recent, plan.Uw, plan.Ww);
    if (e != cudaSuccess) return e;
    prof_mark(p, 5, s);
    return cudaSuccess;
  }
  e = ensure_dynamic_smem(reinterpret_cast<const void*>(&combine_kernel),
                          cmb_bytes);
  if (e != cudaSuccess) return e;
  e = launch_pdl(combine_kernel, dim3(B, h_kv, plan.S), dim3(kCombineThreads),
                 cmb_bytes, s, (const float*)part, (const int*)pref,
                 (const int*)nzpref, B, h_q, h_kv, plan.W, (const float*)p->R_vT,
                 reinterpret_cast<float*>(w + plan.off_cpart),
                 reinterpret_cast<int*>(w + plan.off_cnt), out, p->fold_v,
                 (const float*)wp.wpart, seq_lens, max_pages, sink, recent,
                 plan.Uw, plan.Ww);
  if (e != cudaSuccess) return e;
  prof_mark(p, 5, s);
  return cudaSuccess;
}

}  // namespace optr
