// Tensor-core split-K partial kernel of the decode attention.
//
// Work partition, partial format and combine are those of decode.cu: the
// flattened (sequence, KV head, page) space is cut into W equal contiguous
// ranges, one per warp; a warp writes one partial (m, l, o') per
// (sequence, KV head) segment of its range.
//
// Per 16-token page a warp runs two tiny GEMMs on mma.sync.m16n8k16
// (f16 inputs, f32 accumulate), N = 8 = 4 GQA query heads x {hi, lo}:
//
//   logits   S[tok][n] = sum_ch code[tok][ch] * q'[n][ch], one accumulator
//            per 32-channel group, then l = sum_g scale_g * S_g
//            + sum_g min_g * sum(q' over group g)      (Sec. 3 Eq. 1 on the
//            dequantized rotated key, Appendix "Rotated-query implementation")
//   values   O[ch][n] += (code[ch][tok] - 1.5) * (p[tok] * scale_g[tok])_{hi,lo},
//            plus sum_tok p * (min_g + 1.5 scale_g)[tok] per group
//                                                          (Sec. 3 Eq. 2)
//
// The 2-bit codes enter the MMA as normal fp16 values.  One LOP3 masks a
// code field and ORs in the exponent of 1024, giving 1024 + code * 2^pos;
// every field is first moved to bit pos = 4, 6 or 8 of its 16-bit half by at
// most one shift of the 32-bit word (code_pos), so that the offset 1024 is at
// most 64x the code's weight.  Raw masked fields would be fp16 subnormals,
// and the MMA keeps only ~17 bits below its largest product for subnormal A
// operands, against ~21 for normal ones.
//   keys    the LOP3 result goes to the MMA as is: the query fragment of that
//           channel carries 2^-pos, and the MMA starts from minus the group's
//           offset sum 1024 * sum(fragment), leaving sum code * q'.
//   values  one HFMA2 maps it to the exact centered code - 1.5, and the min
//           term carries min + 1.5 * scale.  Centering keeps the tensor-core
//           accumulator o' a random walk over the pages instead of a sum that
//           grows with the context and cancels against the min term, so its
//           rounding error grows far more slowly with the pages per warp.
// q' and p*scale are split into fp16 hi + lo parts, which fill the 8 MMA
// columns and keep ~22 bits of the float32 operands.
#include <type_traits>

#include "decode_common.cuh"
#include "window.cuh"

namespace optr {
namespace {

constexpr int kStages = 4;            // cp.async pages in flight per warp
constexpr int kWarps = 16;            // warps per CTA: one CTA per SM
constexpr float kLazyTau = 8.f;       // log2-domain slack before rescaling

struct WarpSmemTC {
  alignas(16) uint8_t stage[kStages][kChunk];
  alignas(16) uint32_t pt[2][kGroups][kPage][4];  // p*scale_v (hi, lo) per head, 2 pages
  int2 info[kStages];  // per staged page: (segment key b*h_kv+h, valid tokens)
  // per segment, per lane (kept here, not in registers, so that the page
  // loop has registers to spare): query B fragments, and the key MMAs'
  // start values (-offset hi, -offset lo) twice, in accumulator order
  uint4 qfr[kGroups][32];
  float4 kq[kGroups][32];
};

// the window phase stages 16 key and 16 value rows (8 KB) in the page
// stages and pt, and its P tile in qfr, before any of them is used
static_assert(offsetof(WarpSmemTC, pt) + sizeof(WarpSmemTC::pt) -
                      offsetof(WarpSmemTC, stage) >= (size_t)kWinStageBytes,
              "window row scratch");
static_assert(sizeof(WarpSmemTC::qfr) >= (size_t)kWinPBytes, "window P scratch");

constexpr int kPrefCache = 256;  // sequences whose page prefix sums a CTA caches

__device__ __forceinline__ void mma16816(float* d, uint32_t a0, uint32_t a1,
                                         uint32_t a2, uint32_t a3, uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void ldsm_x4_trans(uint32_t& r0, uint32_t& r1,
                                              uint32_t& r2, uint32_t& r3,
                                              const void* smem_row) {
  const unsigned a = static_cast<unsigned>(__cvta_generic_to_shared(smem_row));
  asm volatile(
      "ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
      : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
      : "r"(a));
}

// The two code fields at bit pos of each 16-bit half of src as fp16
// 1024 + code * 2^pos (pos <= 8 keeps the field inside the mantissa).
template <int pos>
__device__ __forceinline__ uint32_t field_f16x2(uint32_t src, uint32_t exp1024) {
  uint32_t x;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;"  // (a & b) | c
      : "=r"(x) : "r"(src), "n"(0x00030003u << pos), "r"(exp1024));
  return x;
}

// The 16 code fields of a word y whose 16-bit halves each hold one byte of
// group 2j (low byte) and one of group 2j+1 (high byte), as MMA A registers
// out[parity][r] = fp16 1024 + code * 2^pos, pos = code_pos(parity, r).
__device__ __forceinline__ void code_fields(uint32_t y, uint32_t e1024,
                                           uint32_t (&out)[2][4]) {
  const uint32_t yl = y << 4, yr = y >> 6;
  out[0][0] = field_f16x2<code_pos(0, 0)>(yl, e1024);
  out[0][1] = field_f16x2<code_pos(0, 1)>(yl, e1024);
  out[0][2] = field_f16x2<code_pos(0, 2)>(y, e1024);
  out[0][3] = field_f16x2<code_pos(0, 3)>(y, e1024);
  out[1][0] = field_f16x2<code_pos(1, 0)>(y, e1024);
  out[1][1] = field_f16x2<code_pos(1, 1)>(yr, e1024);
  out[1][2] = field_f16x2<code_pos(1, 2)>(yr, e1024);
  out[1][3] = field_f16x2<code_pos(1, 3)>(yr, e1024);
}

// A field from code_fields() of group parity par and code index r
// (1024 + code * 2^pos) mapped by one HFMA2 to the exact centered code
// code - 1.5 in {-1.5, -0.5, 0.5, 1.5}: x * 2^-pos - (1024 * 2^-pos + 1.5).
// Both constants are exact fp16 values for pos = 4, 6, 8.
__device__ __forceinline__ uint32_t centered(uint32_t x, int par, int r) {
  const int pos = code_pos(par, r);
  const __half2 sc = __float2half2_rn(1.0f / (float)(1 << pos));
  const __half2 bias = __float2half2_rn(-1024.0f / (float)(1 << pos) - 1.5f);
  const __half2 y = __hfma2(*reinterpret_cast<const __half2*>(&x), sc, bias);
  return *reinterpret_cast<const uint32_t*>(&y);
}

__device__ __forceinline__ float2 h2f(uint32_t u) {
  return __half22float2(*reinterpret_cast<const __half2*>(&u));
}

// fp16 hi / lo split of x, packed (hi in the low half): hi is x with its
// mantissa cut to 11 significant bits (exact in fp16 when |x| is in fp16's
// normal range), lo = x - hi exactly, rounded to fp16.
__device__ __forceinline__ uint32_t split_hilo(float x) {
  const float hi = __uint_as_float(__float_as_uint(x) & 0xffffe000u);
  const float lo = x - hi;
  uint32_t r;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(lo), "f"(hi));
  return r;
}

// 2^x (the MUFU approximation; relative error ~2^-22).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// The issuing side of a warp describes its flat page range
// (sequence-major, then KV head, then page) 32 pages at a time: lane l of a
// chunk resolves flat page base + l to its physical page, segment key
// (b * h_kv + h) and valid token count, so that issuing a page is a shuffle
// and an address computation with no dependent global load.
struct PageChunk {
  int base;        // first flat page of the chunk
  int unit;        // this lane's page: physical page * h_kv + h, or -1
  int key, nvalid; // segment key b * h_kv + h and valid tokens
};

__device__ __forceinline__ void load_chunk(PageChunk& ch, int base, int f1,
                                           const int* __restrict__ pref,
                                           const int* spref, bool cached,
                                           const int32_t* __restrict__ seq_lens,
                                           const int32_t* __restrict__ bt,
                                           int B, int h_kv, int max_pages,
                                           int num_pages, unsigned* err,
                                           int lane, int sink, int recent,
                                           int& lpage) {
  ch.base = base;
  lpage = 0;
  ch.unit = -1;
  ch.key = -1;
  ch.nvalid = 0;
  const int f = base + lane;
  if (f < f1) {
    int lo = 0, hi = B;  // largest b with pref[b] * h_kv <= f
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      const int pm = cached ? spref[mid] : __ldcg(pref + mid);
      if (pm * h_kv <= f) lo = mid; else hi = mid;
    }
    const int p0 = cached ? spref[lo] : __ldcg(pref + lo);
    const int np = (cached ? spref[lo + 1] : __ldcg(pref + lo + 1)) - p0;
    const int r = f - p0 * h_kv;
    const int h = r / np;
    const int page = sink / kPage + (r - h * np);  // logical page (INT2 range)
    lpage = page;
    const int phys = __ldg(bt + (size_t)lo * max_pages + page);
    ch.key = lo * h_kv + h;
    if (phys >= 0 && phys < num_pages) {
      ch.unit = phys * h_kv + h;
      ch.nvalid = min(kPage, int2_end(__ldg(seq_lens + lo), sink, recent) - page * kPage);
    } else {
      atomicOr(err, OPTR_DEVERR_PAGE_ID);  // skipped: its tokens count as masked
    }
  }
}

// spref[b] = pages of sequences < b (b <= B <= kPrefCache; invalid lengths
// count as empty), by one block-wide scan; ends with __syncthreads().  In a
// decode step (step_cu set) also sstep[0][b] = the step's new tokens of
// sequence b and sstep[1][b] = their first position, loaded together with
// the lengths.
__device__ __noinline__ void page_prefix(const int32_t* __restrict__ seq_lens,
                                         int B, int max_pages, int* spref,
                                         int* wsum, int sink, int recent,
                                         const int32_t* __restrict__ step_cu,
                                         const int32_t* __restrict__ step_pos0,
                                         int (*sstep)[kPrefCache]) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int np = 0;
  if ((int)threadIdx.x < B) {
    if (step_cu != nullptr) {
      sstep[0][threadIdx.x] = __ldg(step_cu + threadIdx.x + 1) - __ldg(step_cu + threadIdx.x);
      sstep[1][threadIdx.x] = __ldg(step_pos0 + threadIdx.x);
    }
    const int len = __ldg(seq_lens + threadIdx.x);
    if (len >= 0 && (long long)len <= (long long)max_pages * kPage)
      np = int2_pages(len, sink, recent);
  }
  int x = np;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) wsum[warp] = x;
  __syncthreads();
  int off = 0;
  for (int i = 0; i < warp; ++i) off += wsum[i];
  if ((int)threadIdx.x < B) spref[threadIdx.x + 1] = off + x;
  if (threadIdx.x == 0) spref[0] = 0;
  __syncthreads();
}

// WIN: the BF16-window phase is compiled in (a separate instance, so that
// the INT2-only kernel keeps its own register allocation).  CMP: the compact
// G = 128 record (1152 bytes per page and KV head, one (scale, min) pair per
// slot at 4-byte stride), read as the G = 32 record's four entries with the
// pair repeated, so the page arithmetic is the same.
template <bool WIN, bool CMP>
__global__ void __launch_bounds__(kWarps * 32, 1)
partial_tensor_kernel(const uint8_t* __restrict__ pool,
                      const int32_t* __restrict__ bt,
                      const int32_t* __restrict__ seq_lens, int B,
                      int max_pages, int num_pages, int h_q, int h_kv,
                      const uint32_t* __restrict__ frag,
                      const float* __restrict__ koff,
                      const float* __restrict__ invs,
                      const float* __restrict__ qs,
                      const int* __restrict__ pref,
                      const int* __restrict__ nzpref,
                      float* __restrict__ part, int W, int early_pages,
                      const int32_t* __restrict__ step_cu,
                      const int32_t* __restrict__ step_pos0,
                      unsigned* err, int sink, int recent, WinPhase wp) {
  // One 16-warp CTA per SM: the warp schedulers favour the CTAs that
  // arrived first on an SM, and with four 4-warp CTAs per SM the last CTA
  // finished ~20% after the first; within one CTA the warps keep pace.
  extern __shared__ __align__(16) unsigned char dsm_[];
  WarpSmemTC* smem = reinterpret_cast<WarpSmemTC*>(dsm_);  // [kWarps]
  __shared__ int spref[kPrefCache + 1];
  __shared__ int sstep[2][kPrefCache];  // decode step: new tokens, first position
  __shared__ int wsum[kWarps];
  uint32_t e1024;
  asm volatile("mov.b32 %0, 0x64006400;" : "=r"(e1024));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, c = lane & 3;
  WarpSmemTC& S = smem[warp];
  // With BF16 windows, warps kWinIntWarps.. of every CTA are window warps
  // (their loads overlap the INT2 pages of the others); the INT2 work is
  // split over the first kWinIntWarps warps of each CTA.
  constexpr int kInt = WIN ? kWinIntWarps : kWarps;
  const int w = blockIdx.x * kInt + warp;  // INT2 warp index (warp < kInt)

  // Page prefix sums.  For up to kPrefCache sequences the CTA scans the
  // lengths itself (the values qrot writes to pref for the combine): the
  // lengths and the block table are inputs, complete before the previous
  // kernel (qrot, or the fused step prologue) began, since that kernel
  // passes its pdl_wait() before it lets this grid launch.  So the page
  // tables are set up before this grid's own pdl_wait(), overlapping the
  // previous kernel.  The first page copies also go before the wait when the
  // pool was complete before the previous kernel began (early_pages: a
  // separate append); after the fused step prologue, which writes the pool,
  // they follow the wait.
  const bool cached = B <= kPrefCache;
  static_assert(kPrefCache < kWarps * 32, "one thread per sequence");
  int F;
  if (cached) {
    page_prefix(seq_lens, B, max_pages, spref, wsum, sink, recent, step_cu, step_pos0,
                sstep);
    F = spref[B] * h_kv;
  } else {
    pdl_wait();
    F = __ldcg(pref + B) * h_kv;
  }
  if constexpr (WIN) {
    if (warp >= kInt) {
      // window warp ww, numbered across the CTAs first so that a partial set
      // is spread over the SMs.  The phase reads only inputs and
      // library-owned state, so it runs before this grid waits for the
      // previous kernel, in the warp's own page stages.
      const int ww = (warp - kInt) * gridDim.x + blockIdx.x;
      if (ww < wp.Ww)
        window_phase(ww, wp, &S.stage[0][0], reinterpret_cast<uint8_t*>(&S.qfr[0][0]));
      pdl_wait();
      pdl_trigger();
      return;
    }
  }
  const int f0 = (int)((long long)w * F / W), f1 = (int)((long long)(w + 1) * F / W);
  if (f0 >= f1) {
    pdl_wait();
    pdl_trigger();
    return;
  }
  PageChunk chk;
  int f_issue = f0;
  int lpage;
  load_chunk(chk, f0, f1, pref, spref, cached, seq_lens, bt, B, h_kv,
             max_pages, num_pages, err, lane, sink, recent, lpage);

  // issue one page into stage s (no commit); every lane records what the
  // stage holds
  auto issue = [&](int s) {
    if (f_issue < f1) {
      if (f_issue - chk.base == 32)
        load_chunk(chk, f_issue, f1, pref, spref, cached, seq_lens, bt, B, h_kv,
                   max_pages, num_pages, err, lane, sink, recent, lpage);
      const int j = f_issue - chk.base;
      const int unit = __shfl_sync(0xffffffffu, chk.unit, j);
      const int key = __shfl_sync(0xffffffffu, chk.key, j);
      const int nv = __shfl_sync(0xffffffffu, chk.nvalid, j);
      // an invalid page (flagged, all tokens masked) is filled with zeros
      const bool ok = unit >= 0;
      const uint8_t* src = pool + (size_t)(ok ? unit : 0) * chunk_bytes(CMP) + lane * 16;
      uint8_t* dst = S.stage[s] + lane * 16;
      cp_async16_zfill(dst, src, ok);
      cp_async16_zfill(dst + 512, src + 512, ok);
      if (!CMP || lane < 8)  // the compact record's last 128 bytes
        cp_async16_zfill(dst + 1024, src + 1024, ok);
      S.info[s] = make_int2(key, nv);  // same value from every lane
      ++f_issue;
    }
  };
  // the next two pages into stages 2q, 2q+1, one cp.async group
  auto issue_pair = [&](int q) {
    issue(2 * q);
    issue(2 * q + 1);
    cp_async_commit();
  };
  // In a decode step the previous kernel writes the step's new tokens, at
  // positions [pos0[b], pos0[b] + n_b) of each sequence b (n_b from cu_new,
  // an input complete before that kernel began).  A page of the first pair
  // none of whose 16 positions is among them holds only records written
  // before the step, so the pair is fetched before the wait when both pages
  // are such (a step's written pages are not read by another sequence).
  bool pre = early_pages != 0;
  if (!pre && step_cu != nullptr) {
    bool safe = true;
    if (lane < 2 && f0 + lane < f1 && chk.key >= 0) {
      const int b = chk.key / h_kv;
      const long long n = cached ? sstep[0][b]
                                 : (long long)__ldg(step_cu + b + 1) - __ldg(step_cu + b);
      const long long s0 = cached ? sstep[1][b] : __ldg(step_pos0 + b);
      const long long t0 = (long long)lpage * kPage;
      safe = n <= 0 || s0 >= t0 + kPage || s0 + n <= t0;
    }
    pre = __all_sync(0xffffffffu, safe);
  }
  if (pre) issue_pair(0);
  pdl_wait();  // (returns at once when already passed above)
  pdl_trigger();
  if (!pre) issue_pair(0);

  // per-segment state
  uint32_t bmin = 0;           // key min-term B fragment (sum q' per group)
  float inv_s = 0.f;           // 1 / prescale of head c
  float acc_o[kGroups][2][4];  // values: [group][half][c-frag]
  float mv[kGroups];           // sum_tok p * min_v per group (this lane)
  float m_ref = -INFINITY, l_lane = 0.f;
  float m_lazy = -INFINITY;    // kLazyTau above the running maximum logit
  int k_s = -30;               // 2^k_s bounds the value scales seen
  float s_cap = 0x1p-30f;      // 2^k_s
  int cur_key = -1;

  auto flush = [&]() {
    // reduce l and the min-terms over the 8 lanes of head c, then write
    float l = l_lane;
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
#pragma unroll
    for (int G = 0; G < (CMP ? 1 : kGroups); ++G)
#pragma unroll
      for (int o = 4; o < 32; o <<= 1)
        mv[G] += __shfl_xor_sync(0xffffffffu, mv[G], o);
    const int cb = cur_key / h_kv, ch = cur_key - cb * h_kv;
    float* slot = part + (size_t)(w + __ldcg(nzpref + cb) * h_kv + ch) * kPartFloats;
    float* dst = slot + c * kD;
#pragma unroll
    for (int G = 0; G < kGroups; ++G) {
      // rows g (r = 2*half) and g+8 (r = 2*half+1) of tile (G, half) are
      // channels 32G + 4g + r
      const float mvG = mv[CMP ? 0 : G];  // CMP: one (scale, min) per token
      float4 o4;
      o4.x = (acc_o[G][0][0] + acc_o[G][0][1]) + mvG;
      o4.y = (acc_o[G][0][2] + acc_o[G][0][3]) + mvG;
      o4.z = (acc_o[G][1][0] + acc_o[G][1][1]) + mvG;
      o4.w = (acc_o[G][1][2] + acc_o[G][1][3]) + mvG;
      *reinterpret_cast<float4*>(dst + 32 * G + 4 * g) = o4;
    }
    if (g == 0) {
      slot[kPartM + c] = m_ref;
      slot[kPartL + c] = l;
    }
  };

  auto begin_segment = [&](int key) {
    cur_key = key;
    const int cb = key / h_kv, ch = key - cb * h_kv;
    const uint4* fq = reinterpret_cast<const uint4*>(
        frag + (((size_t)cb * h_kv + ch) * 32 + lane) * 16);
#pragma unroll
    for (int G = 0; G < kGroups; ++G) {
      const uint4 v = __ldcg(fq + G);
      S.qfr[G][lane] = v;
    }
    {
      const float4* ko = reinterpret_cast<const float4*>(
          koff + ((size_t)cb * h_kv + ch) * 32 + c * 8);
      const float4 k01 = __ldcg(ko), k23 = __ldcg(ko + 1);
      if constexpr (CMP) {
        // one scale per token: the four groups share one accumulator,
        // started from the sum of their offsets
        const float hi = -((k01.x + k01.z) + (k23.x + k23.z));
        const float lo = -((k01.y + k01.w) + (k23.y + k23.w));
        S.kq[0][lane] = make_float4(hi, lo, hi, lo);
      } else {
        S.kq[0][lane] = make_float4(-k01.x, -k01.y, -k01.x, -k01.y);
        S.kq[1][lane] = make_float4(-k01.z, -k01.w, -k01.z, -k01.w);
        S.kq[2][lane] = make_float4(-k23.x, -k23.y, -k23.x, -k23.y);
        S.kq[3][lane] = make_float4(-k23.z, -k23.w, -k23.z, -k23.w);
      }
    }
    const size_t row = (size_t)cb * h_q + 4 * ch + c;
    {
      // column g of the min-term MMA: head g/2, fp16 limb g%2 of the
      // group-c sum of q'; rows k = 2c (scale entries) are 0
      const float qg = __ldcg(qs + ((size_t)cb * h_q + 4 * ch + (g >> 1)) * kGroups + c);
      const uint32_t hl = split_hilo(qg);
      bmin = (g & 1) ? (hl & 0xffff0000u) : (hl << 16);
    }
    inv_s = __ldcg(invs + row);
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

  // ------------------------------------------------ parts of one page
  // logits of tokens g and g+8 (head c) of the page staged at st
  // the four (scale, min) entries of slot t in a metadata region (the
  // compact record's one pair repeated)
  auto meta4 = [&](const uint8_t* region, int t) -> uint4 {
    if constexpr (CMP) {
      const uint32_t x = *reinterpret_cast<const uint32_t*>(region + t * 4);
      return make_uint4(x, x, x, x);
    } else {
      return *reinterpret_cast<const uint4*>(region + t * 16);
    }
  };

  auto logits = [&](const uint8_t* st, float& sc0, float& sc1) {
    const uint2 k0 = *reinterpret_cast<const uint2*>(st + OPTR_K_CODES_OFFSET + g * 32 + 8 * c);
    const uint2 k1 = *reinterpret_cast<const uint2*>(st + OPTR_K_CODES_OFFSET + (g + 8) * 32 + 8 * c);
    // bytes [G0 w2c, G1 w2c, G0 w2c+1, G1 w2c+1] and the same for G2/G3
    const uint32_t y01_0 = __byte_perm(k0.x, k0.y, 0x5410);
    const uint32_t y23_0 = __byte_perm(k0.x, k0.y, 0x7632);
    const uint32_t y01_1 = __byte_perm(k1.x, k1.y, 0x5410);
    const uint32_t y23_1 = __byte_perm(k1.x, k1.y, 0x7632);
    float s_acc[kGroups][4];
    if constexpr (CMP) {
      const float4 kv = S.kq[0][lane];
      s_acc[0][0] = kv.x; s_acc[0][1] = kv.y; s_acc[0][2] = kv.z; s_acc[0][3] = kv.w;
    }
#pragma unroll
    for (int j = 0; j < 2; ++j) {  // groups 2j, 2j+1
      uint32_t f0[2][4], f1[2][4];  // token rows g, g+8
      code_fields(j ? y23_0 : y01_0, e1024, f0);
      code_fields(j ? y23_1 : y01_1, e1024, f1);
#pragma unroll
      for (int par = 0; par < 2; ++par) {
        const int G = 2 * j + par;
        const int A = CMP ? 0 : G;  // accumulator of the group's scale
        const uint4 qv = S.qfr[G][lane];
        if constexpr (!CMP) {
          const float4 kv = S.kq[G][lane];
          s_acc[G][0] = kv.x; s_acc[G][1] = kv.y; s_acc[G][2] = kv.z; s_acc[G][3] = kv.w;
        }
        mma16816(s_acc[A], f0[par][0], f1[par][0], f0[par][1], f1[par][1], qv.x, qv.y);
        mma16816(s_acc[A], f0[par][2], f1[par][2], f0[par][3], f1[par][3], qv.z, qv.w);
      }
    }
    float t0 = 0.f, t1 = 0.f;
    if constexpr (!CMP) {
      const uint4 km0 = meta4(st + OPTR_K_META_OFFSET, g);
      const uint4 km1 = meta4(st + OPTR_K_META_OFFSET, g + 8);
      const uint32_t kmv0[4] = {km0.x, km0.y, km0.z, km0.w};
      const uint32_t kmv1[4] = {km1.x, km1.y, km1.z, km1.w};
#pragma unroll
      for (int G = 0; G < kGroups; ++G) {
        const float a = __low2float(*reinterpret_cast<const __half2*>(&kmv0[G]));   // scale, token g
        const float bb = __low2float(*reinterpret_cast<const __half2*>(&kmv1[G]));  // token g+8
        t0 = fmaf(a, s_acc[G][0] + s_acc[G][1], t0);
        t1 = fmaf(bb, s_acc[G][2] + s_acc[G][3], t1);
      }
    }
    // sum_g min_g * sum(q' over g) on the tensor core: A row t = the 8
    // (scale, min) halves of token t, B = (0, Q_g) per (scale, min) pair
    float u[4] = {0.f, 0.f, 0.f, 0.f};
    const uint32_t w0 = *reinterpret_cast<const uint32_t*>(
        st + OPTR_K_META_OFFSET + g * meta_stride(CMP) + (CMP ? 0 : 4 * c));
    const uint32_t w1 = *reinterpret_cast<const uint32_t*>(
        st + OPTR_K_META_OFFSET + (g + 8) * meta_stride(CMP) + (CMP ? 0 : 4 * c));
    mma16816(u, w0, w1, 0u, 0u, bmin, 0u);
    if constexpr (CMP) {
      // the one (scale, min) pair of tokens g and g+8 is w0 and w1
      t0 = __low2float(*reinterpret_cast<const __half2*>(&w0)) * (s_acc[0][0] + s_acc[0][1]);
      t1 = __low2float(*reinterpret_cast<const __half2*>(&w1)) * (s_acc[0][2] + s_acc[0][3]);
    }
    sc0 = fmaf(inv_s, t0, u[0] + u[1]);
    sc1 = fmaf(inv_s, t1, u[2] + u[3]);
  };

  // value (scale, min) halves of tokens g (vm[0..3]) and g+8 (vm[4..7])
  // per group, kept packed; returns their largest scale
  // (CMP: the one pair of tokens g and g+8 in vm[0] and vm[kGroups])
  auto vmeta = [&](const uint8_t* st, uint32_t (&vm)[2 * kGroups]) {
    if constexpr (CMP) {
      const uint8_t* region = st + vmeta_offset(true);
      vm[0] = *reinterpret_cast<const uint32_t*>(region + g * 4);
      vm[kGroups] = *reinterpret_cast<const uint32_t*>(region + (g + 8) * 4);
      const __half2 mx = __hmax2(*reinterpret_cast<const __half2*>(&vm[0]),
                                 *reinterpret_cast<const __half2*>(&vm[kGroups]));
      return __low2float(mx);
    } else {
      const uint4 m0 = meta4(st + vmeta_offset(CMP), g);
      const uint4 m1 = meta4(st + vmeta_offset(CMP), g + 8);
      vm[0] = m0.x; vm[1] = m0.y; vm[2] = m0.z; vm[3] = m0.w;
      vm[4] = m1.x; vm[5] = m1.y; vm[6] = m1.z; vm[7] = m1.w;
      __half2 mx = *reinterpret_cast<const __half2*>(&vm[0]);
#pragma unroll
      for (int i = 1; i < 2 * kGroups; ++i) mx = __hmax2(mx, *reinterpret_cast<const __half2*>(&vm[i]));
      return __low2float(mx);  // scales are >= 0 (fp16 max ignores a NaN min half)
    }
  };

  // Lazy reference: p = 2^(l - m_ref) with m_ref = m_lazy + k_s - 15,
  // where m_lazy lies kLazyTau (log2 units) above the head's running
  // maximum logit and 2^k_s bounds every value scale seen.  Then
  // p * scale <= 2^15 always fits fp16, and the largest products sit near
  // 2^15, so their fp16 lo parts stay normal whatever the magnitude of the
  // values.  m_lazy and k_s move only when a logit exceeds m_lazy or a
  // scale exceeds 2^k_s; each lane tests its own tokens, and only then are
  // the head maxima reduced over the 8 lanes of the head and the
  // accumulators rescaled.
  auto reference = [&](float lmax, float smax) {
    if (__any_sync(0xffffffffu, lmax > m_lazy || smax > s_cap)) {
      float tmax = lmax, smx = smax;
#pragma unroll
      for (int o = 4; o < 32; o <<= 1) {
        tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, o));
        smx = fmaxf(smx, __shfl_xor_sync(0xffffffffu, smx, o));
      }
      // uniform over the lanes of head c
      if (tmax > m_lazy) m_lazy = tmax + kLazyTau;
      if (smx > s_cap) {
        k_s = ilogbf(smx) + 1;  // smx < 2^k_s
        s_cap = ldexpf(1.f, k_s);
      }
      const float m_new = m_lazy + (float)(k_s - 15);
      if (m_new != m_ref) {
        const float alpha = (m_ref == -INFINITY) ? 0.f : ex2(m_ref - m_new);
        l_lane *= alpha;
#pragma unroll
        for (int G = 0; G < kGroups; ++G) {
          if (!CMP || G == 0) mv[G] *= alpha;
#pragma unroll
          for (int hf = 0; hf < 2; ++hf)
#pragma unroll
            for (int k = 0; k < 4; ++k) acc_o[G][hf][k] *= alpha;
        }
        m_ref = m_new;
      }
    }
  };

  // value-side B operands p * scale (hi, lo) into pt, min terms into mv
  auto vprod = [&](float p0, float p1, const uint32_t (&vm)[2 * kGroups],
                   uint32_t (&pt)[kGroups][kPage][4]) {
#pragma unroll
    for (int G = 0; G < (CMP ? 1 : kGroups); ++G) {  // CMP: one pair per token
      const float2 va = h2f(vm[G]), vb = h2f(vm[kGroups + G]);  // tokens g, g+8
      // the MMA sees centered codes (code - 1.5): the min term carries
      // min + 1.5 * scale
      const float ps0 = p0 * va.x, ps1 = p1 * vb.x;
      mv[G] = fmaf(1.5f, ps0, fmaf(p0, va.y, fmaf(1.5f, ps1, fmaf(p1, vb.y, mv[G]))));
      pt[G][g][c] = split_hilo(ps0);
      pt[G][g + 8][c] = split_hilo(ps1);
    }
  };

  // P.V of the page at st with the B operands in pt (after a __syncwarp)
  auto vcodes = [&](const uint8_t* st, uint32_t (&pt)[kGroups][kPage][4]) {
    uint32_t bv[kGroups][2];
    {
      // lanes 0-7 address rows 0-7 of group G, 8-15 rows 8-15, 16-31 the
      // same for group G+1 (CMP: every group's operand is group 0's)
      const int r = lane & 15, gsel = CMP ? 0 : lane >> 4;
      ldsm_x4_trans(bv[0][0], bv[0][1], bv[1][0], bv[1][1], &pt[gsel][r][0]);
      if constexpr (CMP) {
        bv[2][0] = bv[0][0]; bv[2][1] = bv[0][1];
        bv[3][0] = bv[0][0]; bv[3][1] = bv[0][1];
      } else {
        ldsm_x4_trans(bv[2][0], bv[2][1], bv[3][0], bv[3][1], &pt[2 + gsel][r][0]);
      }
    }
    const uint8_t* vc = st + OPTR_V_CODES_OFFSET + 4 * g;
    const uint32_t x0 = *reinterpret_cast<const uint32_t*>(vc + (2 * c) * 32);
    const uint32_t x1 = *reinterpret_cast<const uint32_t*>(vc + (2 * c + 1) * 32);
    const uint32_t x2 = *reinterpret_cast<const uint32_t*>(vc + (2 * c + 8) * 32);
    const uint32_t x3 = *reinterpret_cast<const uint32_t*>(vc + (2 * c + 9) * 32);
    const uint32_t a01 = __byte_perm(x0, x1, 0x5410), a23 = __byte_perm(x0, x1, 0x7632);
    const uint32_t b01 = __byte_perm(x2, x3, 0x5410), b23 = __byte_perm(x2, x3, 0x7632);
#pragma unroll
    for (int j = 0; j < 2; ++j) {  // groups 2j, 2j+1
      uint32_t fa[2][4], fb[2][4];  // tokens (2c, 2c+1), (2c+8, 2c+9)
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

  // One page on its own (segment starts, partial pages).  FULL = all 16
  // tokens valid (no masking code).
  auto page = [&](const uint8_t* st, int nvalid, auto full_tag) {
    constexpr bool FULL = decltype(full_tag)::value;
    const bool v0 = FULL || g < nvalid, v1 = FULL || g + 8 < nvalid;
    float sc0, sc1;
    logits(st, sc0, sc1);
    uint32_t vm[2 * kGroups];
    if (!FULL) {
      // masked tokens have p = 0 and their (possibly garbage) metadata is
      // zeroed before it is read, so it is never multiplied in
      sc0 = v0 ? sc0 : -INFINITY;
      sc1 = v1 ? sc1 : -INFINITY;
    }
    float smax = vmeta(st, vm);
    if (!FULL) {
      constexpr int nG = CMP ? 1 : kGroups;
#pragma unroll
      for (int G = 0; G < nG; ++G) {
        vm[G] = v0 ? vm[G] : 0u;
        vm[kGroups + G] = v1 ? vm[kGroups + G] : 0u;
      }
      __half2 mx = *reinterpret_cast<const __half2*>(&vm[0]);
#pragma unroll
      for (int G = 0; G < nG; ++G) {
        mx = __hmax2(mx, *reinterpret_cast<const __half2*>(&vm[G]));
        mx = __hmax2(mx, *reinterpret_cast<const __half2*>(&vm[kGroups + G]));
      }
      smax = __low2float(mx);
    }
    reference(fmaxf(sc0, sc1), smax);
    float p0 = ex2(sc0 - m_ref), p1 = ex2(sc1 - m_ref);  // ex2(-inf) = 0
    if (!FULL) {  // a fully masked page before any finite max: -inf - -inf
      p0 = v0 ? p0 : 0.f;
      p1 = v1 ? p1 : 0.f;
    }
    l_lane += p0 + p1;
    vprod(p0, p1, vm, S.pt[0]);
    __syncwarp();
    vcodes(st, S.pt[0]);
  };

  // Two full pages of the current segment: the same steps with the two
  // pages' independent work interleaved and one softmax update.
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
    vprod(pa0, pa1, vma, S.pt[0]);
    vprod(pb0, pb1, vmb, S.pt[1]);
    __syncwarp();
    vcodes(sa, S.pt[0]);
    vcodes(sb, S.pt[1]);
  };

  // one staged page through the segment bookkeeping
  auto single = [&](int s) {
    const int2 inf = S.info[s];
    if (inf.x != cur_key) {
      if (cur_key >= 0) flush();
      begin_segment(inf.x);
    }
    if (inf.y == kPage)
      page(S.stage[s], inf.y, std::true_type{});
    else
      page(S.stage[s], inf.y, std::false_type{});
    __syncwarp();
  };

  // Pages go through the stages in pairs: pair q (stages 2q, 2q+1) is
  // processed while the other pair is in flight.
  // the first segment's query data, loaded while the first pages land
  begin_segment(__shfl_sync(0xffffffffu, chk.key, 0));
  static_assert(kStages == 4, "two pairs of stages");
  const int total = f1 - f0;
#pragma unroll 1
  for (int done = 0; done < total; done += 2) {
    const int q = (done >> 1) & 1;
    issue_pair(1 - q);
    cp_async_wait<1>();
    __syncwarp();
    const int2 ia = S.info[2 * q], ib = S.info[2 * q + 1];
    if (done + 1 < total && ia.x == cur_key && ib.x == cur_key && ia.y == kPage &&
        ib.y == kPage) {
      page_pair(S.stage[2 * q], S.stage[2 * q + 1]);
      __syncwarp();
    } else {
      single(2 * q);
      if (done + 1 < total) single(2 * q + 1);
    }
  }
  flush();
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
                                  const WinPhase& wp, cudaStream_t s) {
  const size_t dsmem = sizeof(WarpSmemTC) * kWarps;
  const bool win = wp.Ww > 0;
  const bool cmp = p->cfg.group == 128;
  auto fn = win ? (cmp ? partial_tensor_kernel<true, true> : partial_tensor_kernel<true, false>)
                : (cmp ? partial_tensor_kernel<false, true> : partial_tensor_kernel<false, false>);
  cudaError_t e = ensure_dynamic_smem(reinterpret_cast<const void*>(fn), dsmem);
  if (e != cudaSuccess) return e;
  return launch_pdl(fn, dim3(W / (win ? kWinIntWarps : kWarps)), dim3(kWarps * 32),
                    dsmem, s, pool, bt, seq_lens, B, max_pages, num_pages,
                    p->cfg.h_q, p->cfg.h_kv, frag, koff, invs, qs, pref, nzpref,
                    part, W, early_pages ? 1 : 0, step_cu, step_pos0, p->err, p->cfg.sink,
                    p->cfg.recent, wp);
}

}  // namespace optr
