// Decode attention over the paged INT2 cache in one launch (tensor cores,
// no BF16 windows): query rotation, split-K softmax partials over the
// streamed pages, their log-sum-exp merge and the R_v^T rotation back.
//
// Work order.  The (KV head h, sequence b, INT2 page) units are flattened
// heads-major, f = h * P + pref[b] + page (P = all INT2 pages of the batch,
// pref[b] = pages of the sequences before b), and cut into one contiguous
// range per CTA (one 16-warp CTA per SM), then into one contiguous range
// per warp.  A (h, b) run of pages is a segment; segments are numbered in
// flat order over the sequences that have pages, k = h * NZ + nz[b].
// Heads-major order keeps a CTA on one or two KV heads, so it loads one
// R_k[h] for all its query rotations and one R_v[h] for its outputs; the
// first head of CTA c is floor(c * h_kv / C) whatever the lengths, so its
// rotation rows are requested before the kernel waits for its inputs.
//
//   setup     page prefix sums of the lengths (scanned by every CTA), the
//             CTA's segments, and for each the rotated query of its GQA
//             group q' = q R_k[h] log2(e)/sqrt(d) as tensor-core operands
//             (Appendix "Rotated-query implementation"), in shared memory;
//   pages     each warp streams its range (cp.async, 4 pages in flight) and
//             keeps an online softmax per segment (Sec. 3 Eq. 1-2 on the
//             dequantized rotated keys and values), writing one partial
//             (m, l, o') per segment it touches;
//   finalize  per segment, the CTA merges its warps' partials; a segment
//             inside one CTA is finished there, o = o' R_v[h]^T / l
//             (Appendix "Equivalent Inference Implementation"); a segment
//             spread over several CTAs is finished by the last of them to
//             arrive (an atomic counter in the workspace per CTA where such
//             a segment starts, reset by the last arriver: those counters,
//             at a fixed place whatever the batch, must start at zero and
//             every call leaves them so).
//
// The per-page arithmetic (codes as normal fp16 MMA operands, fp16 hi/lo
// splits of q' and of p * scale, the lazy softmax reference) is the one
// described in mma_frag.cuh and decode_tc.cu.
#include <string.h>

#include <type_traits>

#include "decode_common.cuh"
#include "mma_frag.cuh"

namespace optr {
namespace {

constexpr int kFWarps = 16;
constexpr int kFThreads = kFWarps * 32;
constexpr int kFStages = 4;
constexpr int kSegCap = 16;   // segments whose query data a CTA holds in shared memory
constexpr int kFPref = 1024;  // largest batch whose prefix sums a CTA scans
constexpr float kFLazyTau = 8.f;

// Query data of one segment: the tensor-core B fragments of q' (fp16 hi/lo,
// with the power-of-two prescale and the code-position factors), the key
// MMAs' start values (minus the code-offset sums), the min-term B fragment
// per lane and the inverse prescales.
struct SegQ {
  uint4 qfr[kGroups][32];
  float2 kq[kGroups][4];  // [group][query head] (-offset hi, -offset lo)
  uint32_t bmin[32];
  float invs[4];
};

struct RotSmem {
  // the bf16 query rows of the first batch's segments (cp.async, issued
  // before the first pages so that they do not queue behind them)
  alignas(16) __nv_bfloat16 qall[kSegCap][4][kD];
  float qrs[4][4][kD];  // [segment of the pass][query head][channel]
  float hmax[4][4][4];
  float qsum[4][4][4];
  long long koff_part[4][kFWarps][kGroups];
};

struct FusedCtx {
  int B, h_q, h_kv, P, NZ, k0, nseg, C, cta, fold_v;
  long long F;
  const int* gpref;  // page prefix sums in the workspace (uncached batches)
  const int* gnz;
  float qscale;
};

// One split-K partial in shared memory (the kPartFloats layout).
struct alignas(16) PartSlot {
  float v[kPartFloats];
};
// A warp's value-side B operands (p * scale_v, fp16 hi/lo, two pages); once
// its pages are done, its last partial
union PtOrPart {
  uint32_t pt[2][kGroups][kPage][4];
  PartSlot fin;
};

struct FusedSmem {
  alignas(16) uint8_t stage[kFWarps][kFStages][kChunk];  // cp.async page stages
  PtOrPart ptp[kFWarps];
  int2 info[kFWarps][kFStages];  // per staged page: (local segment, valid tokens)
  SegQ seg[kSegCap];
  // setup scratch; during the pages, one partial per warp of a segment that
  // ended inside its range (when every segment of the CTA fits one batch)
  union {
    RotSmem rot;
    PartSlot mid[kFWarps];
  } u;
  int spref[kFPref + 1];
  int snz[kFPref + 1];
  int wsum[2][kFWarps];
  int fkey[kFWarps];  // local segment of the warp's partial in ptp (or -1)
  int mkey[kFWarps];  // local segment of the warp's partial in u.mid (or -1)
  FusedCtx ctx;       // the launch's geometry, shared by the phases
};
static_assert(sizeof(FusedSmem) <= 227 * 1024, "one CTA per SM");

// d = a * b + c (m16n8k16, f16 operands, f32 accumulators), c given apart
__device__ __forceinline__ void mma16816c(float (&d)[4], uint32_t a0, uint32_t a1,
                                          uint32_t a2, uint32_t a3, uint32_t b0,
                                          uint32_t b1, float c0, float c1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%10,%11,%10,%11};\n"
      : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1), "f"(c0), "f"(c1));
}


// The kernel's dynamic shared memory (one FusedSmem), named here so that
// the out-of-line phases address it as shared memory.
extern __shared__ __align__(16) unsigned char fused_dsm[];
__device__ __forceinline__ FusedSmem& fused_smem() {
  return *reinterpret_cast<FusedSmem*>(fused_dsm);
}

template <bool kCached>
__device__ __forceinline__ int pref_of(const FusedSmem& sm, const FusedCtx& x, int b) {
  return kCached ? sm.spref[b] : __ldcg(x.gpref + b);
}
template <bool kCached>
__device__ __forceinline__ int nz_of(const FusedSmem& sm, const FusedCtx& x, int b) {
  return kCached ? sm.snz[b] : __ldcg(x.gnz + b);
}
// the sequence of segment k (it has pages): largest b with nz[b] <= k mod NZ
template <bool kCached>
__device__ __forceinline__ int seq_of_seg(const FusedSmem& sm, const FusedCtx& x, int k) {
  const int zi = k - (k / x.NZ) * x.NZ;
  int lo = 0, hi = x.B;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (nz_of<kCached>(sm, x, mid) <= zi) lo = mid; else hi = mid;
  }
  return lo;
}

// Query data of the CTA's local segments [kb, kb_end): the first kSegCap
// into the shared table, later ones (CTAs over many short segments) into
// the workspace table gtab, indexed by the global segment number (every CTA
// that touches a segment writes the same values).
// q' = q R_k[h] runs on the tensor cores for up to four segments of one
// head at a time: the m16n8k16 A tile holds their query rows (row 4 s + r:
// segment s, query head r; bf16, exact), B = R_k in three bf16 limbs (24
// significant bits, read from global memory in fragment order: one 16-byte
// load per lane, limb and pair of k-steps), f32 accumulation; warp w
// computes output channels 8w .. 8w + 7.  The query rows come from the
// staged copies (q_staged) or global memory.  All threads of the CTA; ends
// with __syncthreads().
constexpr int kRotSegs = 4;  // segments per rotation pass (16 A rows)
template <bool kCached>
__device__ __forceinline__ void rotate_segs(FusedSmem& sm, const FusedCtx& x,
                                            const __nv_bfloat16* __restrict__ q,
                                            const uint16_t* __restrict__ Rl3, int kb,
                                            int kb_end, bool q_staged, SegQ* gtab) {
  RotSmem& R = sm.u.rot;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g = lane >> 2, c = lane & 3;
  const int jj = tid & 127;
  const int h_q = x.h_q;
  const float qscale = x.qscale;
  for (int s0 = kb; s0 < kb_end;) {
    // the pass: segments s0 .. s0 + ns - 1, all of head h
    const int h = (x.k0 + s0) / x.NZ;
    int ns = 1;
    while (ns < kRotSegs && s0 + ns < kb_end && (x.k0 + s0 + ns) / x.NZ == h) ++ns;
    {
      // A rows g (segment g >> 2) and g + 8 (segment 2 + (g >> 2)), head g & 3
      const __nv_bfloat16* qr[2] = {nullptr, nullptr};
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        const int sg = 2 * hf + (g >> 2);
        if (sg < ns) {
          const int key = s0 + sg;
          if (q_staged && key < kSegCap) {
            qr[hf] = &R.qall[key][g & 3][0];
          } else {
            const int bq = seq_of_seg<kCached>(sm, x, x.k0 + key);
            qr[hf] = q + ((size_t)bq * h_q + 4 * h + (g & 3)) * kD;
          }
        }
      }
      // this warp's B fragments: 12 coalesced 16-byte loads per lane, all
      // issued before the first MMA
      const uint4* Rf = reinterpret_cast<const uint4*>(Rl3 + (size_t)h * kRL3Halves) +
                        (size_t)warp * 4 * 3 * 32 + lane;
      uint4 bq[4][3];
#pragma unroll
      for (int p2 = 0; p2 < 4; ++p2)
#pragma unroll
        for (int limb = 0; limb < 3; ++limb) bq[p2][limb] = __ldg(Rf + (p2 * 3 + limb) * 32);
      uint32_t a[4][2][4];
#pragma unroll
      for (int p2 = 0; p2 < 4; ++p2)
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int k0s = 32 * p2 + 16 * e;
#pragma unroll
          for (int hf = 0; hf < 2; ++hf) {
            a[p2][e][hf] = qr[hf] ? *reinterpret_cast<const uint32_t*>(qr[hf] + k0s + 2 * c) : 0u;
            a[p2][e][2 + hf] = qr[hf] ? *reinterpret_cast<const uint32_t*>(qr[hf] + k0s + 8 + 2 * c) : 0u;
          }
        }
      float d[3][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
      for (int p2 = 0; p2 < 4; ++p2)
#pragma unroll
        for (int limb = 0; limb < 3; ++limb) {
          const uint4 bb = bq[p2][limb];
          // A registers: (row g, k 0-7), (row g + 8, k 0-7), (row g, k 8-15), (row g + 8, k 8-15)
          mma16816_bf16(d[limb], a[p2][0][0], a[p2][0][1], a[p2][0][2], a[p2][0][3], bb.x, bb.y);
          mma16816_bf16(d[limb], a[p2][1][0], a[p2][1][1], a[p2][1][2], a[p2][1][3], bb.z, bb.w);
        }
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        const int sg = 2 * hf + (g >> 2);
        if (sg < ns) {
          R.qrs[sg][g & 3][8 * warp + 2 * c] =
              ((d[0][2 * hf] + d[1][2 * hf]) + d[2][2 * hf]) * qscale;
          R.qrs[sg][g & 3][8 * warp + 2 * c + 1] =
              ((d[0][2 * hf + 1] + d[1][2 * hf + 1]) + d[2][2 * hf + 1]) * qscale;
        }
      }
    }
    __syncthreads();
    for (int sg = 0; sg < ns; ++sg) {
      // thread (r, j): the group sums / maxima of q' of head r
      const int r = tid >> 7;
      const float xv = R.qrs[sg][r][jj];
      float sm_ = xv, am = fabsf(xv);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        sm_ += __shfl_xor_sync(0xffffffffu, sm_, o);
        am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, o));
      }
      if (lane == 0) {
        R.qsum[sg][r][jj >> 5] = sm_;
        R.hmax[sg][r][jj >> 5] = am;
      }
    }
    __syncthreads();
    for (int sg = 0; sg < ns; ++sg) {
      const int key = s0 + sg;
      SegQ& Q = key < kSegCap ? sm.seg[key] : gtab[x.k0 + key];
      // tensor-core B fragment register `reg` of lane L (see the kernel
      // comment of decode_tc.cu): per head a power-of-two prescale 2^e
      // brings max |q'| 2^e into [2^13, 2^14); channel 32G + 4w + r also
      // carries 2^-pos (its code's bit position); koff sums
      // 1024 * fragment over the group exactly (int64 fixed point).
      const int L = tid >> 4, reg = tid & 15;
      const int G = reg >> 2, kk = (reg >> 1) & 1, which = reg & 1;
      const int gl = L >> 2, cl = L & 3;
      const int head = gl >> 1, limb = gl & 1;
      const float mx = fmaxf(fmaxf(R.hmax[sg][head][0], R.hmax[sg][head][1]),
                             fmaxf(R.hmax[sg][head][2], R.hmax[sg][head][3]));
      const int e = max(-100, min(100, mx > 0.f ? 13 - exponent_of(mx) : 0));
      const int r = 2 * kk + which;
      const int ch = 32 * G + 8 * cl + r;
      const float scl = pow2i(e - code_pos(G, r));
      const float x0 = R.qrs[sg][head][ch] * scl, x1 = R.qrs[sg][head][ch + 4] * scl;
      const __half h0 = __float2half_rn(x0), h1 = __float2half_rn(x1);
      __half v0 = h0, v1 = h1;
      if (limb) {
        v0 = __float2half_rn(x0 - __half2float(h0));
        v1 = __float2half_rn(x1 - __half2float(h1));
      }
      const uint32_t fragv =
          (uint32_t)__half_as_ushort(v0) | ((uint32_t)__half_as_ushort(v1) << 16);
      reinterpret_cast<uint32_t*>(&Q.qfr[G][L])[reg & 3] = fragv;
      long long t = __float2ll_rn(__half2float(v0) * 16777216.0f) +
                    __float2ll_rn(__half2float(v1) * 16777216.0f);
      t += __shfl_xor_sync(0xffffffffu, t, 1);
      t += __shfl_xor_sync(0xffffffffu, t, 2);
      t += __shfl_xor_sync(0xffffffffu, t, 16);
      if ((lane & 15) % 4 == 0) R.koff_part[sg][warp][G] = t;
    }
    __syncthreads();
    for (int i = tid; i < ns * 128; i += kFThreads) {
      const int sg = i >> 7, t = i & 127;
      const int key = s0 + sg;
      SegQ& Q = key < kSegCap ? sm.seg[key] : gtab[x.k0 + key];
      if (t < 32) {
        // column gg = (head gg >> 1, limb gg & 1), group GG
        const int gg = t >> 2, GG = t & 3;
        const long long tot = R.koff_part[sg][2 * gg][GG] + R.koff_part[sg][2 * gg + 1][GG];
        reinterpret_cast<float*>(&Q.kq[GG][gg >> 1])[gg & 1] =
            -(__ll2float_rn(tot) * 0x1p-14f);
      } else if (t < 64) {
        // min-term B fragment of lane L = (g, c): limb g & 1 of the group-c
        // sum of q' of head g >> 1, in the high half (rows 2c are 0)
        const int L = t - 32;
        const uint32_t hl = split_hilo(R.qsum[sg][(L >> 2) >> 1][L & 3]);
        Q.bmin[L] = ((L >> 2) & 1) ? (hl & 0xffff0000u) : (hl << 16);
      } else if (t < 68) {
        const int hd = t - 64;
        const float m2 = fmaxf(fmaxf(R.hmax[sg][hd][0], R.hmax[sg][hd][1]),
                               fmaxf(R.hmax[sg][hd][2], R.hmax[sg][hd][3]));
        const int e2 = max(-100, min(100, m2 > 0.f ? 13 - exponent_of(m2) : 0));
        Q.invs[hd] = pow2i(-e2);
      }
    }
    __syncthreads();
    s0 += ns;
  }
}

// Out-of-line entry point of rotate_segs for the segments beyond the shared
// table (CTAs over many short segments), after the first pages are issued.
template <bool kCached>
__device__ __noinline__ void rotate_segs_overflow(const __nv_bfloat16* __restrict__ q,
                                                  const uint16_t* __restrict__ Rl3,
                                                  SegQ* gtab) {
  FusedSmem& sm = fused_smem();
  rotate_segs<kCached>(sm, sm.ctx, q, Rl3, kSegCap, sm.ctx.nseg, false, gtab);
}

// The first kSegCap segments (the shared table) in two phases, so that the
// page loads can be issued in between:
//   rot_mma   q' = q R_k[h] log2(e)/sqrt(d) on the tensor cores, with the
//             three bf16 limbs of R_k[h] staged in the page stages' space
//             (the first head's before the kernel waits; another head's
//             when a pass needs it) and the query rows staged, into qst
//             (the warps' p*scale buffers, unused until the pages): passes
//             of up to four segments of one head, A row 4 s + r = segment s,
//             query head r;
//   rot_frag  per segment, group sums and maxima of q', the prescaled fp16
//             hi/lo B fragments, code-offset sums and min-term fragments.
// Both run on all threads and end with __syncthreads().
template <bool kCached>
__device__ __noinline__ int rot_mma(const uint16_t* __restrict__ Rl3, int h_staged) {
  FusedSmem& sm = fused_smem();
  const FusedCtx& x = sm.ctx;
  uint16_t* Rs = reinterpret_cast<uint16_t*>(&sm.stage[0][0][0]);
  float (*qst)[4][kD] = reinterpret_cast<float (*)[4][kD]>(&sm.ptp[0]);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g = lane >> 2, c = lane & 3;
  const int nA = min(x.nseg, kSegCap);
  for (int s0 = 0; s0 < nA;) {
    const int h = (x.k0 + s0) / x.NZ;
    int ns = 1;
    while (ns < kRotSegs && s0 + ns < nA && (x.k0 + s0 + ns) / x.NZ == h) ++ns;
    if (h != h_staged) {
      __syncthreads();  // every warp is done with the staged limbs
      for (int i = tid; i < kRL3Halves / 8; i += kFThreads)
        cp_async16(Rs + 8 * i, Rl3 + (size_t)h * kRL3Halves + 8 * i);
      cp_async_commit();
      cp_async_wait<0>();
      __syncthreads();
      h_staged = h;
    }
    // A rows g (segment g >> 2) and g + 8 (segment 2 + (g >> 2)), head g & 3
    const __nv_bfloat16* qr[2] = {nullptr, nullptr};
#pragma unroll
    for (int hf = 0; hf < 2; ++hf) {
      const int sg = 2 * hf + (g >> 2);
      if (sg < ns) qr[hf] = &sm.u.rot.qall[s0 + sg][g & 3][0];
    }
    const uint4* Rf = reinterpret_cast<const uint4*>(Rs) + (size_t)warp * 4 * 3 * 32 + lane;
    float d[3][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
    for (int p2 = 0; p2 < 4; ++p2) {
      uint32_t a[2][4];
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int k0s = 32 * p2 + 16 * e;
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
          a[e][hf] = qr[hf] ? *reinterpret_cast<const uint32_t*>(qr[hf] + k0s + 2 * c) : 0u;
          a[e][2 + hf] = qr[hf] ? *reinterpret_cast<const uint32_t*>(qr[hf] + k0s + 8 + 2 * c) : 0u;
        }
      }
#pragma unroll
      for (int limb = 0; limb < 3; ++limb) {
        const uint4 bb = Rf[(p2 * 3 + limb) * 32];
        mma16816_bf16(d[limb], a[0][0], a[0][1], a[0][2], a[0][3], bb.x, bb.y);
        mma16816_bf16(d[limb], a[1][0], a[1][1], a[1][2], a[1][3], bb.z, bb.w);
      }
    }
#pragma unroll
    for (int hf = 0; hf < 2; ++hf) {
      const int sg = 2 * hf + (g >> 2);
      if (sg < ns) {
        qst[s0 + sg][g & 3][8 * warp + 2 * c] =
            ((d[0][2 * hf] + d[1][2 * hf]) + d[2][2 * hf]) * x.qscale;
        qst[s0 + sg][g & 3][8 * warp + 2 * c + 1] =
            ((d[0][2 * hf + 1] + d[1][2 * hf + 1]) + d[2][2 * hf + 1]) * x.qscale;
      }
    }
    s0 += ns;
  }
  __syncthreads();
  return h_staged;
}

template <bool kCached>
__device__ __noinline__ void rot_frag() {
  FusedSmem& sm = fused_smem();
  const FusedCtx& x = sm.ctx;
  RotSmem& R = sm.u.rot;
  const float (*qst)[4][kD] = reinterpret_cast<const float (*)[4][kD]>(&sm.ptp[0]);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int jj = tid & 127;
  const int nA = min(x.nseg, kSegCap);
  for (int s0 = 0; s0 < nA; s0 += 4) {
    const int ns = min(4, nA - s0);
    for (int sg = 0; sg < ns; ++sg) {
      const int r = tid >> 7;
      const float xv = qst[s0 + sg][r][jj];
      float sm_ = xv, am = fabsf(xv);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        sm_ += __shfl_xor_sync(0xffffffffu, sm_, o);
        am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, o));
      }
      if (lane == 0) {
        R.qsum[sg][r][jj >> 5] = sm_;
        R.hmax[sg][r][jj >> 5] = am;
      }
    }
    __syncthreads();
    for (int sg = 0; sg < ns; ++sg) {
      SegQ& Q = sm.seg[s0 + sg];
      const int L = tid >> 4, reg = tid & 15;
      const int G = reg >> 2, kk = (reg >> 1) & 1, which = reg & 1;
      const int gl = L >> 2, cl = L & 3;
      const int head = gl >> 1, limb = gl & 1;
      const float mx = fmaxf(fmaxf(R.hmax[sg][head][0], R.hmax[sg][head][1]),
                             fmaxf(R.hmax[sg][head][2], R.hmax[sg][head][3]));
      const int e = max(-100, min(100, mx > 0.f ? 13 - exponent_of(mx) : 0));
      const int r = 2 * kk + which;
      const int ch = 32 * G + 8 * cl + r;
      const float scl = pow2i(e - code_pos(G, r));
      const float x0 = qst[s0 + sg][head][ch] * scl, x1 = qst[s0 + sg][head][ch + 4] * scl;
      const __half h0 = __float2half_rn(x0), h1 = __float2half_rn(x1);
      __half v0 = h0, v1 = h1;
      if (limb) {
        v0 = __float2half_rn(x0 - __half2float(h0));
        v1 = __float2half_rn(x1 - __half2float(h1));
      }
      const uint32_t fragv =
          (uint32_t)__half_as_ushort(v0) | ((uint32_t)__half_as_ushort(v1) << 16);
      reinterpret_cast<uint32_t*>(&Q.qfr[G][L])[reg & 3] = fragv;
      long long t = __float2ll_rn(__half2float(v0) * 16777216.0f) +
                    __float2ll_rn(__half2float(v1) * 16777216.0f);
      t += __shfl_xor_sync(0xffffffffu, t, 1);
      t += __shfl_xor_sync(0xffffffffu, t, 2);
      t += __shfl_xor_sync(0xffffffffu, t, 16);
      if ((lane & 15) % 4 == 0) R.koff_part[sg][warp][G] = t;
    }
    __syncthreads();
    for (int i = tid; i < ns * 128; i += kFThreads) {
      const int sg = i >> 7, t = i & 127;
      SegQ& Q = sm.seg[s0 + sg];
      if (t < 32) {
        const int gg = t >> 2, GG = t & 3;
        const long long tot = R.koff_part[sg][2 * gg][GG] + R.koff_part[sg][2 * gg + 1][GG];
        reinterpret_cast<float*>(&Q.kq[GG][gg >> 1])[gg & 1] =
            -(__ll2float_rn(tot) * 0x1p-14f);
      } else if (t < 64) {
        const int L = t - 32;
        const uint32_t hl = split_hilo(R.qsum[sg][(L >> 2) >> 1][L & 3]);
        Q.bmin[L] = ((L >> 2) & 1) ? (hl & 0xffff0000u) : (hl << 16);
      } else if (t < 68) {
        const int hd = t - 64;
        const float m2 = fmaxf(fmaxf(R.hmax[sg][hd][0], R.hmax[sg][hd][1]),
                               fmaxf(R.hmax[sg][hd][2], R.hmax[sg][hd][3]));
        const int e2 = max(-100, min(100, m2 > 0.f ? 13 - exponent_of(m2) : 0));
        Q.invs[hd] = pow2i(-e2);
      }
    }
    __syncthreads();
  }
}

// Finalization scratch, in the query-data table's space (free once every
// warp is done with its pages).
constexpr int kWave = 4;  // segments finalized together, 128 threads each
constexpr int kMaxCtas = 256;  // largest grid (SM count) the tables allow
struct FinScratch {
  int wbnd[kFWarps + 1];          // flat starts of this CTA's warp ranges
  int cbnd[kMaxCtas + 1];         // flat starts of every CTA's range
  float orot[kWave][4][kD];       // o' / l of the wave's segments
  float qs4[4][4][kD];            // quarter sums of the R_v^T product
  float red_m[kWave][kFWarps][4];
  float red_l[kWave][kFWarps][4];
  int flag[kWave];                // 1: this CTA finishes the segment
};
static_assert(sizeof(FinScratch) <= sizeof(SegQ) * kSegCap, "finalize scratch");
// R_v^T of up to two heads, staged in the page stages' space
static_assert(kD * kD * sizeof(float) <= sizeof(FusedSmem::stage), "R_v^T staging");

__device__ __forceinline__ void group_sync(int grp) {
  asm volatile("bar.sync %0, 128;" ::"r"(grp + 1) : "memory");
}

// Log-sum-exp merge of n (<= kFWarps) partials slot(i) into the running
// (M, L, acc) of one 128-thread group: thread v holds float4 v of o'
// (query head v >> 5) and, for v % 32 == 0, that head's M and L.  red_m /
// red_l are the group's scratch.  Ends with a group barrier.
// exp2(m - M) for a partial with running maximum m (0 for an empty one);
// the MUFU approximation (relative error ~2^-22), as the pages' weights.
__device__ __forceinline__ float merge_w(float m, float M) {
  return m == -INFINITY ? 0.f : ex2(m - M);
}

// Log-sum-exp merge of up to kFWarps candidate partials slot(i), i <
// kFWarps (slot(i) null: no partial), into the running (M, L, acc) of one
// 128-thread group: thread v holds float4 v of o' (query head v >> 5) and
// that head's M and L.  kOther: the partials are other CTAs' (global
// memory, read through L2); else this CTA's own (shared or global memory,
// generic loads).  Fixed, unrolled candidate loops keep every value in
// registers.  Ends with a group barrier.
template <bool kOther, typename Slot>
__device__ __forceinline__ void group_merge(int grp, int v, Slot slot,
                                            float (&red_m)[kFWarps][4],
                                            float (&red_l)[kFWarps][4], float& M,
                                            float& L, float4& acc) {
  const int hd = v >> 5;
  float4 o[kFWarps];
#pragma unroll
  for (int i = 0; i < kFWarps; ++i) {
    const float* p = slot(i);
    o[i] = !p ? make_float4(0.f, 0.f, 0.f, 0.f)
           : kOther ? __ldcg(reinterpret_cast<const float4*>(p) + v)
                    : *(reinterpret_cast<const float4*>(p) + v);
  }
  if (v < 4 * kFWarps) {
    const int i = v >> 2, r = v & 3;
    const float* p = slot(i);
    float m = -INFINITY, l = 0.f;
    if (p) {
      m = kOther ? __ldcg(p + kPartM + r) : p[kPartM + r];
      l = kOther ? __ldcg(p + kPartL + r) : p[kPartL + r];
    }
    red_m[i][r] = m;
    red_l[i][r] = l;
  }
  group_sync(grp);
  float Mn = M;
#pragma unroll
  for (int i = 0; i < kFWarps; ++i) Mn = fmaxf(Mn, red_m[i][hd]);
  const float al = merge_w(M, Mn);
  acc.x *= al;
  acc.y *= al;
  acc.z *= al;
  acc.w *= al;
  L *= al;
#pragma unroll
  for (int i = 0; i < kFWarps; ++i) {
    const float wv = merge_w(red_m[i][hd], Mn);  // 0 for an empty candidate
    acc.x = fmaf(o[i].x, wv, acc.x);
    acc.y = fmaf(o[i].y, wv, acc.y);
    acc.z = fmaf(o[i].z, wv, acc.z);
    acc.w = fmaf(o[i].w, wv, acc.w);
    L = fmaf(red_l[i][hd], wv, L);
  }
  M = Mn;
  group_sync(grp);  // red_m / red_l may be rewritten
}

// Per segment of the CTA, four at a time (one 128-thread group each): merge
// this CTA's warp partials; a segment inside the CTA is finished here, one
// spread over several CTAs is published and finished by the last of them
// to arrive; then, with all threads, o = o' / l and out = o R_v^T, with
// R_v^T of the wave's heads staged in shared memory while the merges run.
// Rows of sequences without pages are zeroed.  The page stages are free.
template <bool kCached>
__device__ __noinline__ void finalize_segs(const float* __restrict__ part,
                                           float* __restrict__ cpart,
                                           int* __restrict__ cnt,
                                           float* __restrict__ out,
                                           const float* __restrict__ R_vT) {
  FusedSmem& sm = fused_smem();
  const FusedCtx& x = sm.ctx;
  const int tid = threadIdx.x;
  const int B = x.B, h_q = x.h_q, NZ = x.NZ, k0 = x.k0, nseg = x.nseg;
  const int C = x.C, cta = x.cta, fold_v = x.fold_v;
  const long long F = x.F;
  const int W = C * kFWarps;
  FinScratch& fz = *reinterpret_cast<FinScratch*>(&sm.seg[0]);
  float (*rvt)[kD] = reinterpret_cast<float (*)[kD]>(&sm.stage[0][0][0]);
  const int grp = tid >> 7, v = tid & 127, hd = v >> 5;
  // range boundaries (one 64-bit division each, once), so that the tests
  // below are comparisons: warp i of this CTA owns [wbnd[i], wbnd[i+1]),
  // CTA c owns [cbnd[c], cbnd[c+1])
  if (tid <= kFWarps) fz.wbnd[tid] = (int)((long long)(cta * kFWarps + tid) * F / W);
  for (int c = tid; c <= C; c += kFThreads) fz.cbnd[c] = (int)((long long)c * F / C);
  __syncthreads();
  for (int s0 = 0; s0 < nseg; s0 += kWave) {
    const int nw = min(kWave, nseg - s0);
    // R_v^T of the wave's first head into shared memory (the page stages'
    // space; a second head of the wave is read from global memory)
    const int h_a = (k0 + s0) / NZ;
    if (!fold_v)
      for (int i = tid; i < kD * kD / 4; i += kFThreads)
        cp_async16(&rvt[0][0] + 4 * i, R_vT + (size_t)h_a * kD * kD + 4 * i);
    cp_async_commit();
    if (grp < nw) {
      const int key = s0 + grp;
      const int k = k0 + key;
      const int h = k / NZ;
      const int b = seq_of_seg<kCached>(sm, x, k);
      const int fs0 = h * x.P + pref_of<kCached>(sm, x, b);
      const int fs1 = fs0 + (pref_of<kCached>(sm, x, b + 1) - pref_of<kCached>(sm, x, b));
      // each of this CTA's warps with pages of the segment: its partial is
      // in its own shared slot (its last segment), in its mid slot, or in
      // the workspace
      float M = -INFINITY, L = 0.f;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      group_merge<false>(grp, v, [&](int wl) -> const float* {
        if (fz.wbnd[wl] >= fs1 || fz.wbnd[wl + 1] <= fs0 || fz.wbnd[wl] == fz.wbnd[wl + 1])
          return nullptr;
        return sm.fkey[wl] == key ? sm.ptp[wl].fin.v
               : sm.mkey[wl] == key ? sm.u.mid[wl].v
                                    : part + (size_t)(cta * kFWarps + wl + k) * kPartFloats;
      }, fz.red_m[grp], fz.red_l[grp], M, L, acc);
      // CTAs whose ranges hold pages of the segment
      int ca = 0, cb = C;  // last c with cbnd[c] <= fs0 / <= fs1 - 1
      {
        int lo = 0, hi = C;
        while (hi - lo > 1) {
          const int mid = (lo + hi) >> 1;
          if (fz.cbnd[mid] <= fs0) lo = mid; else hi = mid;
        }
        ca = lo;
        lo = ca;
        hi = C;
        while (hi - lo > 1) {
          const int mid = (lo + hi) >> 1;
          if (fz.cbnd[mid] <= fs1 - 1) lo = mid; else hi = mid;
        }
        cb = lo;
      }
      bool mine = true;
      if (ca != cb) {
        // publish this CTA's merge; the last CTA to arrive finishes
        float* cp = cpart + (size_t)(cta + k) * kPartFloats;
        reinterpret_cast<float4*>(cp)[v] = acc;
        if ((v & 31) == 0) {
          cp[kPartM + hd] = M;
          cp[kPartL + hd] = L;
        }
        __threadfence();
        group_sync(grp);
        if (v == 0) {
          // the counter of the CTA where the segment starts: a CTA's range
          // ends inside at most one segment, so at most one spread segment
          // starts in each CTA
          int n_arr = 0;
          for (int c = ca; c <= cb; ++c) n_arr += fz.cbnd[c] < fz.cbnd[c + 1] ? 1 : 0;
          const int old = atomicAdd(cnt + ca, 1);
          fz.flag[grp] = old == n_arr - 1;
          if (old == n_arr - 1) cnt[ca] = 0;  // reset for the next call
        }
        group_sync(grp);
        mine = fz.flag[grp] != 0;
        if (mine) {
          __threadfence();
          M = -INFINITY;
          L = 0.f;
          acc = make_float4(0.f, 0.f, 0.f, 0.f);
          for (int c0 = ca; c0 <= cb; c0 += kFWarps) {
            group_merge<true>(grp, v, [&](int i) -> const float* {
              const int c = c0 + i;
              if (c > cb || fz.cbnd[c] == fz.cbnd[c + 1]) return nullptr;
              return cpart + (size_t)(c + k) * kPartFloats;
            }, fz.red_m[grp], fz.red_l[grp], M, L, acc);
          }
        }
      }
      if (v == 0) fz.flag[grp] = mine ? 1 : 0;
      if (mine) {
        const float il = L > 0.f ? 1.f / L : 0.f;
        const int ch = (v & 31) * 4;
        fz.orot[grp][hd][ch + 0] = acc.x * il;
        fz.orot[grp][hd][ch + 1] = acc.y * il;
        fz.orot[grp][hd][ch + 2] = acc.z * il;
        fz.orot[grp][hd][ch + 3] = acc.w * il;
      }
    }
    cp_async_wait<0>();
    __syncthreads();
    // o R_v^T for the segments this CTA finishes, all threads: thread
    // (i, quarter) sums k in [32 quarter, 32 quarter + 32) for the 4 heads
    for (int j = 0; j < nw; ++j) {
      if (!fz.flag[j]) continue;
      const int k = k0 + s0 + j;
      const int h = k / NZ;
      const int b = seq_of_seg<kCached>(sm, x, k);
      float* ob = out + ((size_t)b * h_q + 4 * h) * kD;
      if (fold_v) {
        ob[tid] = fz.orot[j][tid >> 7][tid & 127];
        continue;
      }
      const int i = tid & 127, qq = tid >> 7;
      const float* rs = h == h_a ? &rvt[0][0] : nullptr;
      float a4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
      for (int kk = 32 * qq; kk < 32 * qq + 32; ++kk) {
        const float rt = rs ? rs[kk * kD + i] : __ldg(R_vT + (size_t)h * kD * kD + kk * kD + i);
#pragma unroll
        for (int r = 0; r < 4; ++r) a4[r] = fmaf(fz.orot[j][r][kk], rt, a4[r]);
      }
#pragma unroll
      for (int r = 0; r < 4; ++r) fz.qs4[qq][r][i] = a4[r];
      __syncthreads();
      const int r = tid >> 7;
      ob[r * kD + i] = (fz.qs4[0][r][i] + fz.qs4[1][r][i]) + (fz.qs4[2][r][i] + fz.qs4[3][r][i]);
      __syncthreads();
    }
    __syncthreads();  // the staged R_v^T and the scratch are reused
  }
  // rows of sequences without pages are zero
  for (int b = cta; b < B; b += C) {
    if (pref_of<kCached>(sm, x, b + 1) == pref_of<kCached>(sm, x, b)) {
      float* ob = out + (size_t)b * h_q * kD;
      for (int i = tid; i < h_q * kD; i += kFThreads) ob[i] = 0.f;
    }
  }
}

// kCached: the batch is small enough (B <= kFPref) for every CTA to scan
// the page prefix sums into shared memory; otherwise a plan launch wrote
// them to the workspace.
template <bool kCached>
__global__ void __launch_bounds__(kFThreads, 1)
decode_fused_kernel(const uint8_t* __restrict__ pool,
                    const int32_t* __restrict__ bt,
                    const int32_t* __restrict__ seq_lens, int B, int max_pages,
                    int num_pages, int h_q, int h_kv,
                    const __nv_bfloat16* __restrict__ q,
                    const uint16_t* __restrict__ Rl3,
                    const float* __restrict__ R_vT, int fold_v, float qscale,
                    const int* __restrict__ gpref, const int* __restrict__ gnz,
                    float* __restrict__ part, float* __restrict__ cpart,
                    int* __restrict__ cnt, float* __restrict__ out,
                    SegQ* __restrict__ gtab, unsigned* err, int inputs_ready) {
  FusedSmem& sm = fused_smem();
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, c = lane & 3;
  const int C = gridDim.x, cta = blockIdx.x;
  const int W = C * kFWarps;
  const int w = cta * kFWarps + warp;

  // ---------------------------------------------------------------- setup
  // R_k of this CTA's first head (floor(cta * h_kv / C) whatever the
  // lengths), as bf16 limbs in fragment order, into the page stages' space,
  // requested before any input is read: it is library-owned.
  int h_staged = (int)((long long)cta * h_kv / C);
  {
    uint16_t* Rs = reinterpret_cast<uint16_t*>(&sm.stage[0][0][0]);
    for (int i = tid; i < kRL3Halves / 8; i += kFThreads)
      cp_async16(Rs + 8 * i, Rl3 + (size_t)h_staged * kRL3Halves + 8 * i);
    cp_async_commit();
  }
  // The caller's inputs may come from earlier kernels in the stream.  After
  // the step's cache-write launch (inputs_ready) the query, lengths and
  // tables were complete before that launch began; only the pool is
  // written by it, so pages are read after the wait.
  if (!inputs_ready) {
    pdl_wait();
    pdl_trigger();
  }

  // page prefix sums: pref[b] = INT2 pages of sequences < b, nz[b] =
  // sequences < b with pages; invalid lengths count as empty (flagged once)
  constexpr bool cached = kCached;
  if (cached) {
    int np0 = 0, np1 = 0;
    const int b0 = 2 * tid, b1 = 2 * tid + 1;
    bool bad = false;
    if (b0 < B) {
      const int len = __ldg(seq_lens + b0);
      if (len < 0 || (long long)len > (long long)max_pages * kPage) bad = true;
      else np0 = (len + kPage - 1) / kPage;
    }
    if (b1 < B) {
      const int len = __ldg(seq_lens + b1);
      if (len < 0 || (long long)len > (long long)max_pages * kPage) bad = true;
      else np1 = (len + kPage - 1) / kPage;
    }
    if (bad && cta == 0) atomicOr(err, OPTR_DEVERR_SEQ_LEN);
    int xp = np0 + np1, xn = (np0 > 0) + (np1 > 0);
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int yp = __shfl_up_sync(0xffffffffu, xp, o);
      const int yn = __shfl_up_sync(0xffffffffu, xn, o);
      if (lane >= o) { xp += yp; xn += yn; }
    }
    if (lane == 31) { sm.wsum[0][warp] = xp; sm.wsum[1][warp] = xn; }
    __syncthreads();
    int op = 0, on = 0;
    for (int i = 0; i < warp; ++i) { op += sm.wsum[0][i]; on += sm.wsum[1][i]; }
    // inclusive prefix at b1 is op + xp; at b0 it is that minus np1
    if (b0 < B) {
      sm.spref[b0 + 1] = op + xp - np1;
      sm.snz[b0 + 1] = on + xn - (np1 > 0);
    }
    if (b1 < B) {
      sm.spref[b1 + 1] = op + xp;
      sm.snz[b1 + 1] = on + xn;
    }
    if (tid == 0) { sm.spref[0] = 0; sm.snz[0] = 0; }
  } else {
    // the plan launch before this one wrote them (it waited for the inputs)
    if (inputs_ready) {
      pdl_wait();
      pdl_trigger();
    }
  }
  __syncthreads();
  auto pref_at = [&](int b) { return cached ? sm.spref[b] : __ldcg(gpref + b); };
  auto nz_at = [&](int b) { return cached ? sm.snz[b] : __ldcg(gnz + b); };
  const int P = pref_at(B);
  const int NZ = nz_at(B);
  const long long F = (long long)h_kv * P;
  // the sequence of flat offset r in [0, P) (it has pages)
  auto seq_of = [&](int r) {
    int lo = 0, hi = B;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (pref_at(mid) <= r) lo = mid; else hi = mid;
    }
    return lo;
  };
  // global segment index of flat index f
  auto seg_of = [&](long long f) {
    const int h = (int)(f / P);
    const int b = seq_of((int)(f - (long long)h * P));
    return h * NZ + nz_at(b);
  };

  const long long C0 = (long long)cta * F / C, C1 = (long long)(cta + 1) * F / C;
  const int k0 = C0 < C1 ? seg_of(C0) : 0;
  const int nseg = C0 < C1 ? seg_of(C1 - 1) - k0 + 1 : 0;
  FusedCtx& x = sm.ctx;
  if (tid == 0) {
    x.B = B;
    x.h_q = h_q;
    x.h_kv = h_kv;
    x.P = P;
    x.NZ = NZ;
    x.k0 = k0;
    x.nseg = nseg;
    x.C = C;
    x.cta = cta;
    x.fold_v = fold_v;
    x.F = F;
    x.gpref = gpref;
    x.gnz = gnz;
    x.qscale = qscale;
  }
  __syncthreads();

  // ---------------------------------------------------------- page issue
  // flat indices fit in 32 bits (B * max_pages * h_kv < 2^31, host-checked)
  const int f0 = (int)((long long)w * F / W), f1 = (int)((long long)(w + 1) * F / W);
  uint8_t (&stage)[kFStages][kChunk] = sm.stage[warp];
  uint32_t (&pt)[2][kGroups][kPage][4] = sm.ptp[warp].pt;
  int2 (&info)[kFStages] = sm.info[warp];
  if (lane == 0) {
    sm.fkey[warp] = -1;
    sm.mkey[warp] = -1;
  }
  // lane l of a chunk resolves flat page base + l: physical unit
  // (page * h_kv + h, or -1 when the table entry is out of range: its
  // tokens count as masked), local segment and valid tokens
  int ch_base = f0;
  int ch_unit = -1, ch_key = 0, ch_nv = 0;
  auto load_chunk = [&](int base) {
    ch_base = base;
    ch_unit = -1;
    ch_key = 0;
    ch_nv = 0;
    const int f = base + lane;
    if (f < f1) {
      const int h = f / P;
      const int r = f - h * P;
      const int b = seq_of(r);
      const int page = r - pref_at(b);
      const int phys = __ldg(bt + (size_t)b * max_pages + page);
      ch_key = h * NZ + nz_at(b) - k0;
      if (phys >= 0 && phys < num_pages) {
        ch_unit = phys * h_kv + h;
        ch_nv = min(kPage, __ldg(seq_lens + b) - page * kPage);
      } else {
        atomicOr(err, OPTR_DEVERR_PAGE_ID);
      }
    }
  };
  int f_issue = f0;
  // issue the next page into its stage (or nothing past the range) and
  // commit one cp.async group either way, so that the group count stays
  // uniform: every consumed page has kFStages - 1 groups after it
  auto issue = [&]() {
    if (f_issue < f1) {
      if (f_issue - ch_base == 32) load_chunk(f_issue);
      const int j = f_issue - ch_base;
      const int unit = __shfl_sync(0xffffffffu, ch_unit, j);
      const int key = __shfl_sync(0xffffffffu, ch_key, j);
      const int nv = __shfl_sync(0xffffffffu, ch_nv, j);
      const bool ok = unit >= 0;
      const int s = (f_issue - f0) & (kFStages - 1);
      const uint8_t* src = pool + (size_t)(ok ? unit : 0) * kChunk + lane * 16;
      uint8_t* dst = stage[s] + lane * 16;
      cp_async16_zfill(dst, src, ok);
      cp_async16_zfill(dst + 512, src + 512, ok);
      cp_async16_zfill(dst + 1024, src + 1024, ok);
      info[s] = make_int2(key, nv);
      ++f_issue;
    }
    cp_async_commit();
  };

  // ------------------------------------------------------- page state
  uint32_t e1024;
  asm volatile("mov.b32 %0, 0x64006400;" : "=r"(e1024));
  uint32_t bmin = 0;
  float inv_s = 0.f;
  float acc_o[kGroups][2][4];
  float mv[kGroups];
  float m_ref = -INFINITY, l_lane = 0.f, m_lazy = -INFINITY;
  int k_s = -30;
  float s_cap = 0x1p-30f;
  int cur_key = -1;
  const SegQ* sq = &sm.seg[0];  // query data of the current segment

  // The warp's partial of segment cur_key: its last one into its own
  // shared slot (ptp, free once its pages are done), the first one that
  // ends inside its range into u.mid (when the CTA's segments fit one
  // batch: later batches reuse that space for their query rotation), any
  // other to the workspace.
  int n_mid = 0;
  auto flush = [&](bool last) {
    float l = l_lane;
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
#pragma unroll
    for (int G = 0; G < kGroups; ++G)
#pragma unroll
      for (int o = 4; o < 32; o <<= 1) mv[G] += __shfl_xor_sync(0xffffffffu, mv[G], o);
    float* slot;
    if (last) {
      slot = sm.ptp[warp].fin.v;
      if (lane == 0) sm.fkey[warp] = cur_key;
    } else if (n_mid == 0) {
      slot = sm.u.mid[warp].v;
      if (lane == 0) sm.mkey[warp] = cur_key;
      n_mid = 1;
    } else {
      slot = part + (size_t)(w + k0 + cur_key) * kPartFloats;
    }
    float* dst = slot + c * kD;
#pragma unroll
    for (int G = 0; G < kGroups; ++G) {
      float4 o4;
      o4.x = (acc_o[G][0][0] + acc_o[G][0][1]) + mv[G];
      o4.y = (acc_o[G][0][2] + acc_o[G][0][3]) + mv[G];
      o4.z = (acc_o[G][1][0] + acc_o[G][1][1]) + mv[G];
      o4.w = (acc_o[G][1][2] + acc_o[G][1][3]) + mv[G];
      *reinterpret_cast<float4*>(dst + 32 * G + 4 * g) = o4;
    }
    if (g == 0) {
      slot[kPartM + c] = m_ref;
      slot[kPartL + c] = l;
    }
  };

  auto begin_segment = [&](int key) {
    cur_key = key;
    sq = key < kSegCap ? &sm.seg[key] : gtab + k0 + key;
    bmin = sq->bmin[lane];
    inv_s = sq->invs[c];
#pragma unroll
    for (int G = 0; G < kGroups; ++G) {
      mv[G] = 0.f;
#pragma unroll
      for (int hf = 0; hf < 2; ++hf)
#pragma unroll
        for (int k = 0; k < 4; ++k) acc_o[G][hf][k] = 0.f;
    }
    m_ref = -INFINITY;
    m_lazy = -INFINITY;
    k_s = -30;
    s_cap = 0x1p-30f;
    l_lane = 0.f;
  };

  auto logits = [&](const uint8_t* st, float& sc0, float& sc1) {
    const uint2 k0w = *reinterpret_cast<const uint2*>(st + OPTR_K_CODES_OFFSET + g * 32 + 8 * c);
    const uint2 k1w = *reinterpret_cast<const uint2*>(st + OPTR_K_CODES_OFFSET + (g + 8) * 32 + 8 * c);
    const uint32_t y01_0 = __byte_perm(k0w.x, k0w.y, 0x5410);
    const uint32_t y23_0 = __byte_perm(k0w.x, k0w.y, 0x7632);
    const uint32_t y01_1 = __byte_perm(k1w.x, k1w.y, 0x5410);
    const uint32_t y23_1 = __byte_perm(k1w.x, k1w.y, 0x7632);
    float s_acc[kGroups][4];
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      uint32_t fa[2][4], fb[2][4];
      code_fields(j ? y23_0 : y01_0, e1024, fa);
      code_fields(j ? y23_1 : y01_1, e1024, fb);
#pragma unroll
      for (int par = 0; par < 2; ++par) {
        const int G = 2 * j + par;
        const uint4 qv = sq->qfr[G][lane];
        const float2 kv = sq->kq[G][c];
        mma16816c(s_acc[G], fa[par][0], fb[par][0], fa[par][1], fb[par][1], qv.x, qv.y,
                  kv.x, kv.y);
        mma16816(s_acc[G], fa[par][2], fb[par][2], fa[par][3], fb[par][3], qv.z, qv.w);
      }
    }
    const uint4 km0 = *reinterpret_cast<const uint4*>(st + OPTR_K_META_OFFSET + g * 16);
    const uint4 km1 = *reinterpret_cast<const uint4*>(st + OPTR_K_META_OFFSET + (g + 8) * 16);
    const uint32_t kmv0[4] = {km0.x, km0.y, km0.z, km0.w};
    const uint32_t kmv1[4] = {km1.x, km1.y, km1.z, km1.w};
    float u[4] = {0.f, 0.f, 0.f, 0.f};
    {
      const uint32_t w0 = *reinterpret_cast<const uint32_t*>(st + OPTR_K_META_OFFSET + g * 16 + 4 * c);
      const uint32_t w1 = *reinterpret_cast<const uint32_t*>(st + OPTR_K_META_OFFSET + (g + 8) * 16 + 4 * c);
      mma16816(u, w0, w1, 0u, 0u, bmin, 0u);
    }
    float t0 = 0.f, t1 = 0.f;
#pragma unroll
    for (int G = 0; G < kGroups; ++G) {
      const float a = __low2float(*reinterpret_cast<const __half2*>(&kmv0[G]));
      const float bb = __low2float(*reinterpret_cast<const __half2*>(&kmv1[G]));
      t0 = fmaf(a, s_acc[G][0] + s_acc[G][1], t0);
      t1 = fmaf(bb, s_acc[G][2] + s_acc[G][3], t1);
    }
    sc0 = fmaf(inv_s, t0, u[0] + u[1]);
    sc1 = fmaf(inv_s, t1, u[2] + u[3]);
  };

  auto vmeta = [&](const uint8_t* st, uint32_t (&vm)[2 * kGroups]) {
    const uint4 m0 = *reinterpret_cast<const uint4*>(st + OPTR_V_META_OFFSET + g * 16);
    const uint4 m1 = *reinterpret_cast<const uint4*>(st + OPTR_V_META_OFFSET + (g + 8) * 16);
    vm[0] = m0.x; vm[1] = m0.y; vm[2] = m0.z; vm[3] = m0.w;
    vm[4] = m1.x; vm[5] = m1.y; vm[6] = m1.z; vm[7] = m1.w;
    __half2 mx = *reinterpret_cast<const __half2*>(&vm[0]);
#pragma unroll
    for (int i = 1; i < 2 * kGroups; ++i) mx = __hmax2(mx, *reinterpret_cast<const __half2*>(&vm[i]));
    return __low2float(mx);
  };

  auto reference = [&](float lmax, float smax) {
    if (__any_sync(0xffffffffu, lmax > m_lazy || smax > s_cap)) {
      float tmax = lmax, smx = smax;
#pragma unroll
      for (int o = 4; o < 32; o <<= 1) {
        tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, o));
        smx = fmaxf(smx, __shfl_xor_sync(0xffffffffu, smx, o));
      }
      if (tmax > m_lazy) m_lazy = tmax + kFLazyTau;
      if (smx > s_cap) {
        k_s = exponent_of(smx) + 1;  // smx: an fp16 scale, normal in float
        s_cap = pow2i(k_s);
      }
      const float m_new = m_lazy + (float)(k_s - 15);
      if (m_new != m_ref) {
        const float alpha = (m_ref == -INFINITY) ? 0.f : ex2(m_ref - m_new);
        l_lane *= alpha;
#pragma unroll
        for (int G = 0; G < kGroups; ++G) {
          mv[G] *= alpha;
#pragma unroll
          for (int hf = 0; hf < 2; ++hf)
#pragma unroll
            for (int k = 0; k < 4; ++k) acc_o[G][hf][k] *= alpha;
        }
        m_ref = m_new;
      }
    }
  };

  auto vprod = [&](float p0, float p1, const uint32_t (&vm)[2 * kGroups],
                   uint32_t (&pt)[kGroups][kPage][4]) {
#pragma unroll
    for (int G = 0; G < kGroups; ++G) {
      const float2 va = h2f(vm[G]), vb = h2f(vm[kGroups + G]);
      const float ps0 = p0 * va.x, ps1 = p1 * vb.x;
      mv[G] = fmaf(1.5f, ps0, fmaf(p0, va.y, fmaf(1.5f, ps1, fmaf(p1, vb.y, mv[G]))));
      pt[G][g][c] = split_hilo(ps0);
      pt[G][g + 8][c] = split_hilo(ps1);
    }
  };

  auto vcodes = [&](const uint8_t* st, uint32_t (&pt)[kGroups][kPage][4]) {
    uint32_t bv[kGroups][2];
    {
      const int r = lane & 15, gsel = lane >> 4;
      ldsm_x4_trans(bv[0][0], bv[0][1], bv[1][0], bv[1][1], &pt[gsel][r][0]);
      ldsm_x4_trans(bv[2][0], bv[2][1], bv[3][0], bv[3][1], &pt[2 + gsel][r][0]);
    }
    const uint8_t* vc = st + OPTR_V_CODES_OFFSET + 4 * g;
    const uint32_t x0 = *reinterpret_cast<const uint32_t*>(vc + (2 * c) * 32);
    const uint32_t x1 = *reinterpret_cast<const uint32_t*>(vc + (2 * c + 1) * 32);
    const uint32_t x2 = *reinterpret_cast<const uint32_t*>(vc + (2 * c + 8) * 32);
    const uint32_t x3 = *reinterpret_cast<const uint32_t*>(vc + (2 * c + 9) * 32);
    const uint32_t a01 = __byte_perm(x0, x1, 0x5410), a23 = __byte_perm(x0, x1, 0x7632);
    const uint32_t b01 = __byte_perm(x2, x3, 0x5410), b23 = __byte_perm(x2, x3, 0x7632);
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      uint32_t fa[2][4], fb[2][4];
      code_fields(j ? a23 : a01, e1024, fa);
      code_fields(j ? b23 : b01, e1024, fb);
#pragma unroll
      for (int par = 0; par < 2; ++par) {
        const int G = 2 * j + par;
        mma16816(acc_o[G][0], centered(fa[par][0], par, 0), centered(fa[par][1], par, 1),
                 centered(fb[par][0], par, 0), centered(fb[par][1], par, 1),
                 bv[G][0], bv[G][1]);
        mma16816(acc_o[G][1], centered(fa[par][2], par, 2), centered(fa[par][3], par, 3),
                 centered(fb[par][2], par, 2), centered(fb[par][3], par, 3),
                 bv[G][0], bv[G][1]);
      }
    }
  };

  auto page = [&](const uint8_t* st, int nvalid, auto full_tag) {
    constexpr bool FULL = decltype(full_tag)::value;
    const bool v0 = FULL || g < nvalid, v1 = FULL || g + 8 < nvalid;
    float sc0, sc1;
    logits(st, sc0, sc1);
    uint32_t vm[2 * kGroups];
    if (!FULL) {
      sc0 = v0 ? sc0 : -INFINITY;
      sc1 = v1 ? sc1 : -INFINITY;
    }
    float smax = vmeta(st, vm);
    if (!FULL) {
#pragma unroll
      for (int G = 0; G < kGroups; ++G) {
        vm[G] = v0 ? vm[G] : 0u;
        vm[kGroups + G] = v1 ? vm[kGroups + G] : 0u;
      }
      __half2 mx = *reinterpret_cast<const __half2*>(&vm[0]);
#pragma unroll
      for (int i = 1; i < 2 * kGroups; ++i) mx = __hmax2(mx, *reinterpret_cast<const __half2*>(&vm[i]));
      smax = __low2float(mx);
    }
    reference(fmaxf(sc0, sc1), smax);
    float p0 = ex2(sc0 - m_ref), p1 = ex2(sc1 - m_ref);
    if (!FULL) {
      p0 = v0 ? p0 : 0.f;
      p1 = v1 ? p1 : 0.f;
    }
    l_lane += p0 + p1;
    vprod(p0, p1, vm, pt[0]);
    __syncwarp();
    vcodes(st, pt[0]);
  };

  auto page_pair = [&](const uint8_t* sa, const uint8_t* sb) {
    float a0, a1, b0, b1;
    logits(sa, a0, a1);
    logits(sb, b0, b1);
    uint32_t vma[2 * kGroups], vmb[2 * kGroups];
    const float smax = fmaxf(vmeta(sa, vma), vmeta(sb, vmb));
    reference(fmaxf(fmaxf(a0, a1), fmaxf(b0, b1)), smax);
    const float pa0 = ex2(a0 - m_ref), pa1 = ex2(a1 - m_ref);
    const float pb0 = ex2(b0 - m_ref), pb1 = ex2(b1 - m_ref);
    l_lane += (pa0 + pa1) + (pb0 + pb1);
    vprod(pa0, pa1, vma, pt[0]);
    vprod(pb0, pb1, vmb, pt[1]);
    __syncwarp();
    vcodes(sa, pt[0]);
    vcodes(sb, pt[1]);
  };

  // ------------------------------------------------------------ run
  // query rows of the first batch's segments: 1 KB each (the 4 query heads
  // of the group are consecutive rows), 16 bytes per copy
  const int kb_end0 = min(nseg, kSegCap);  // segments whose query rows are staged
  for (int i = tid; i < kb_end0 * 64; i += kFThreads) {
    const int key = i >> 6;
    const int k = k0 + key;
    const int h = k / NZ;
    const int b = seq_of_seg<kCached>(sm, x, k);
    cp_async16(reinterpret_cast<uint8_t*>(&sm.u.rot.qall[key][0][0]) + (i & 63) * 16,
               reinterpret_cast<const uint8_t*>(q + ((size_t)b * h_q + 4 * h) * kD) +
                   (i & 63) * 16);
  }
  cp_async_commit();
  if (f0 < f1) load_chunk(f0);
  cp_async_wait<0>();  // R_k's limbs and the query rows
  __syncthreads();
  h_staged = rot_mma<kCached>(Rl3, h_staged);
  if (inputs_ready && cached) {
    // step: the pool is written by the step's cache-write launch
    pdl_wait();
    pdl_trigger();
  }
#pragma unroll 1
  for (int s = 0; s < kFStages; ++s) issue();
  // the fragments of q' while the first pages are in flight
  rot_frag<kCached>();
  if (nseg > kSegCap) rotate_segs_overflow<kCached>(q, Rl3, gtab);

  int f_cons = f0;
#pragma unroll 1
  while (f_cons < f1) {
    cp_async_wait<kFStages - 2>();  // pages f_cons and f_cons + 1 landed
    __syncwarp();
    const int sa = (f_cons - f0) & (kFStages - 1);
    const int2 ia = info[sa];
    if (ia.x != cur_key) {
      if (cur_key >= 0) flush(false);
      begin_segment(ia.x);
    }
    const int sb = (f_cons + 1 - f0) & (kFStages - 1);
    const int2 ib = info[sb];
    if (f_cons + 1 < f1 && ib.x == cur_key && ia.y == kPage && ib.y == kPage) {
      page_pair(stage[sa], stage[sb]);
      __syncwarp();
      f_cons += 2;
      issue();
      issue();
    } else {
      if (ia.y == kPage)
        page(stage[sa], ia.y, std::true_type{});
      else
        page(stage[sa], ia.y, std::false_type{});
      __syncwarp();
      f_cons += 1;
      issue();
    }
  }
  cp_async_wait<0>();
  __syncwarp();
  if (cur_key >= 0) flush(true);

  // ------------------------------------------------------------ finalize
  __threadfence();
  __syncthreads();  // every warp's partials written; page stages free
  finalize_segs<kCached>(part, cpart, cnt, out, R_vT);
}

// Page prefix sums of a batch too large for a CTA to scan itself (one CTA).
__global__ void __launch_bounds__(512)
decode_plan_kernel(const int32_t* __restrict__ seq_lens, int B, int max_pages,
                   int* __restrict__ pref, int* __restrict__ nz, unsigned* err) {
  __shared__ int wt[2][16];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  pdl_wait();
  pdl_trigger();
  int run_p = 0, run_n = 0;
  for (int base = 0; base < B; base += 512) {
    const int b = base + tid;
    int np = 0;
    if (b < B) {
      const int len = seq_lens[b];
      if (len < 0 || (long long)len > (long long)max_pages * kPage)
        atomicOr(err, OPTR_DEVERR_SEQ_LEN);
      else
        np = (len + kPage - 1) / kPage;
    }
    int xp = np, xn = np > 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int yp = __shfl_up_sync(0xffffffffu, xp, o);
      const int yn = __shfl_up_sync(0xffffffffu, xn, o);
      if (lane >= o) { xp += yp; xn += yn; }
    }
    if (lane == 31) { wt[0][warp] = xp; wt[1][warp] = xn; }
    __syncthreads();
    int op = run_p, on = run_n;
    for (int i = 0; i < warp; ++i) { op += wt[0][i]; on += wt[1][i]; }
    if (b < B) { pref[b + 1] = op + xp; nz[b + 1] = on + xn; }
    if (b == 0) { pref[0] = 0; nz[0] = 0; }
    for (int i = 0; i < 16; ++i) { run_p += wt[0][i]; run_n += wt[1][i]; }
    __syncthreads();
  }
}

}  // namespace

size_t fused_decode_smem() { return sizeof(FusedSmem); }
size_t fused_qtab_entry_bytes() { return sizeof(SegQ); }

cudaError_t launch_decode_fused(const optr_params* p, const __nv_bfloat16* q,
                                const int32_t* bt, const int32_t* seq_lens,
                                int B, int max_pages, const uint8_t* pool,
                                int num_pages, float* out, int* pref, int* nz,
                                float* part, float* cpart, int* cnt, void* qtab,
                                bool inputs_ready, cudaStream_t s) {
  cudaError_t e;
  if (B > kFPref) {
    e = launch_pdl(decode_plan_kernel, dim3(1), dim3(512), 0, s, seq_lens, B,
                   max_pages, pref, nz, p->err);
    if (e != cudaSuccess) return e;
    // the fused kernel now follows the plan launch, which waited for the
    // inputs: they may be read before its own wait
    inputs_ready = true;
  }
  if (p->num_sms > kMaxCtas) return cudaErrorInvalidConfiguration;
  const size_t smem = sizeof(FusedSmem);
  auto fn = B <= kFPref ? decode_fused_kernel<true> : decode_fused_kernel<false>;
  e = ensure_dynamic_smem(reinterpret_cast<const void*>(fn), smem);
  if (e != cudaSuccess) return e;
  const float qscale = 1.4426950408889634f / sqrtf((float)kD);
  return launch_pdl(fn, dim3(p->num_sms), dim3(kFThreads), smem, s,
                    pool, bt, seq_lens, B, max_pages, num_pages, p->cfg.h_q,
                    p->cfg.h_kv, q, (const uint16_t*)p->Rk_l3, (const float*)p->R_vT,
                    p->fold_v, qscale, (const int*)pref, (const int*)nz, part,
                    cpart, cnt, out, reinterpret_cast<SegQ*>(qtab), p->err,
                    inputs_ready ? 1 : 0);
}

}  // namespace optr

namespace optr {

void build_rotation_l3(const float* R, uint16_t* out) {
  // bf16 round-to-nearest-even of a float (finite inputs)
  auto bf = [](float x) -> uint16_t {
    uint32_t u;
    memcpy(&u, &x, 4);
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
  };
  auto fl = [](uint16_t b) -> float {
    const uint32_t u = (uint32_t)b << 16;
    float x;
    memcpy(&x, &u, 4);
    return x;
  };
  // B fragments of m16n8k16 (B[k][n] = R[k][n]: input channel k, output
  // channel n), in the order the rotation loads them: warp w (outputs
  // 8w .. 8w + 7), k-step pair p2, limb, lane (g, c), then its four
  // registers mi (k chunk 4 p2 + mi), each the pair k = 8 kc + 2c, + 1 of
  // output n = 8w + g (low half first)
  for (int w = 0; w < kD / 8; ++w)
    for (int p2 = 0; p2 < 4; ++p2)
      for (int lane = 0; lane < 32; ++lane)
        for (int mi = 0; mi < 4; ++mi)
          for (int e = 0; e < 2; ++e) {
            const int n = 8 * w + (lane >> 2);
            const int kk = 8 * (4 * p2 + mi) + 2 * (lane & 3) + e;
            const float x = R[(size_t)kk * kD + n];
            const uint16_t hi = bf(x);
            const float r1 = x - fl(hi);
            const uint16_t mid = bf(r1);
            const uint16_t lo = bf(r1 - fl(mid));
            const uint16_t lim[3] = {hi, mid, lo};
            for (int limb = 0; limb < 3; ++limb)
              out[((((size_t)w * 4 + p2) * 3 + limb) * 32 + lane) * 8 + mi * 2 + e] = lim[limb];
          }
}

}  // namespace optr
