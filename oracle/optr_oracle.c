/*
 * optr_oracle.c -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, obviously correct CPU statement of the OptR rotated-INT2
 * paged KV-cache path (arXiv 2608.02691), used to check the CUDA library.
 * Only the tests, the package's smoke check and the benchmark's CPU-baseline
 * leg may load it; the library never calls it and shares no code with it.
 *
 * Precision: every rotation, logit, softmax and output is computed in
 * float64 from the exact widening of the bf16 / fp16 / fp32 inputs.  The one
 * place where floating point decides an integer -- the INT2 code of a rotated
 * value -- is evaluated in IEEE float32 on the float32 rounding of the fp64
 * rotated value, because that is the precision the kernels decide it in and
 * the paper fixes none (its quantizer is "group-wise affine INT2", Sec. 3.1).
 *
 * Conventions: row vectors, z' = z R (Sec. 3.1 Eq. 4); contiguous GQA
 * grouping; logits scaled by 1/sqrt(d) (Sec. 3 Eq. 1).  The pool layout and
 * the quantizer reading are the ones documented in include/optr.h; they are
 * restated here from that specification, not shared as code.
 *
 * Build: gcc -O2 -std=gnu11 -ffp-contract=off -fopenmp -fPIC -shared.
 * fp-contract is off so that x86-64 and aarch64 builds round identically.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define OR_D 128
#define OR_G 32
#define OR_P 16
#define OR_KC 0
#define OR_VC 512
#define OR_KM 1024

/* ---------------------------------------------------------------- scalars */

static double bf16_to_f64(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

static uint16_t f32_to_f16_bits(float x) {
  _Float16 h = (_Float16)x; /* IEEE round-to-nearest-even */
  uint16_t b;
  memcpy(&b, &h, sizeof b);
  return b;
}

static double f16_bits_to_f64(uint16_t b) {
  _Float16 h;
  memcpy(&h, &b, sizeof h);
  return (double)h;
}

/* ------------------------------------------------------------- quantizer */

/*
 * Q2 on one group of n rotated values (Sec. 3.1: "Q2(.; c, G), the INT2
 * quantize-dequantize map with clipping ratio c and group size G"; four
 * levels, affine (scale and min) per group).  Reading fixed by the library
 * specification: range [c*min, c*max], codes round_half_even((z-mn)*3/r)
 * clamped to 0..3, fp16 scale r/3 and fp16 min.  Evaluated in float32.
 * Outputs one code per element (unpacked), the fp16 bit patterns of scale
 * and min, and the pre-rounding values u (0 for a degenerate group).
 * Returns 1 for a degenerate group, else 0.
 */
int oracle_quantize_group(const float* z, int n, float clip, uint8_t* codes,
                          uint16_t* scale_bits, uint16_t* min_bits, float* u) {
  float lo = z[0], hi = z[0];
  for (int i = 1; i < n; ++i) {
    if (z[i] < lo) lo = z[i];
    if (z[i] > hi) hi = z[i];
  }
  float mn = clip * lo;
  float mx = clip * hi;
  float r = mx - mn;
  if (!(r > 1e-30f) || !isfinite(r)) {
    for (int i = 0; i < n; ++i) {
      codes[i] = 0;
      if (u) u[i] = 0.0f;
    }
    *scale_bits = 0;
    *min_bits = f32_to_f16_bits(mn);
    return 1;
  }
  float inv = 3.0f / r;
  for (int i = 0; i < n; ++i) {
    float zc = z[i];
    if (zc < mn) zc = mn;
    if (zc > mx) zc = mx;
    float ui = (zc - mn) * inv;
    float c = rintf(ui); /* default rounding mode: nearest, ties to even */
    if (c < 0.0f) c = 0.0f;
    if (c > 3.0f) c = 3.0f;
    codes[i] = (uint8_t)c;
    if (u) u[i] = ui;
  }
  *scale_bits = f32_to_f16_bits(r / 3.0f);
  *min_bits = f32_to_f16_bits(mn);
  return 0;
}

/* Dequantized value of one code: code * scale + min (fp16 metadata). */
static double dequant(int code, uint16_t scale_bits, uint16_t min_bits) {
  return (double)code * f16_bits_to_f64(scale_bits) + f16_bits_to_f64(min_bits);
}

/* ------------------------------------------------------------ pool layout */

/* Byte of a slot's 32 code bytes that holds channel ch, and its bit shift:
 * ch = 32*g + 4*w + r lives in byte 4*w + g at bits [2r, 2r+1]. */
int oracle_code_byte(int ch) { return 4 * ((ch % OR_G) / 4) + ch / OR_G; }
int oracle_code_shift(int ch) { return 2 * (ch % 4); }

/* Pool record layout per (page, KV head) as a function of the group size:
 *   G = 32:  1536 bytes: K codes [16][32] at 0, V codes at 512, K meta
 *            [16 slots][4 blocks][fp16 scale, fp16 min] at 1024, V meta at
 *            1280 (16 bytes per slot);
 *   G = 128: 1152 bytes (the paper's compact record, Sec. 5: one scale and
 *            min per 128 channels, 2 + 0.25 bits per element): codes as
 *            above, K meta [16 slots][fp16 scale, fp16 min] at 1024, V meta
 *            at 1088 (4 bytes per slot). */
static int chunk_bytes(int group) { return group == 128 ? 1152 : 1536; }
static int vmeta_off(int group) { return group == 128 ? 1088 : 1280; }
static int meta_stride(int group) { return group == 128 ? 4 : 16; }

static uint8_t* chunk_of(uint8_t* pool, int page, int h_kv, int h, int group) {
  return pool + ((size_t)page * h_kv + h) * chunk_bytes(group);
}

static void store_slot(uint8_t* chunk, int codes_off, int meta_off, int slot,
                       const uint8_t* codes /*[128]*/,
                       const uint16_t* scale /*[4]*/,
                       const uint16_t* mn /*[4]*/, int group) {
  uint8_t* cb = chunk + codes_off + slot * 32;
  memset(cb, 0, 32);
  for (int ch = 0; ch < OR_D; ++ch)
    cb[oracle_code_byte(ch)] |= (uint8_t)(codes[ch] << oracle_code_shift(ch));
  uint8_t* mb = chunk + meta_off + slot * meta_stride(group);
  /* G = 128: the four 32-channel blocks share one pair, stored once */
  for (int g = 0; g < (group == 128 ? 1 : OR_D / OR_G); ++g) {
    mb[4 * g + 0] = (uint8_t)(scale[g] & 0xff);
    mb[4 * g + 1] = (uint8_t)(scale[g] >> 8);
    mb[4 * g + 2] = (uint8_t)(mn[g] & 0xff);
    mb[4 * g + 3] = (uint8_t)(mn[g] >> 8);
  }
}

/* Dequantized rotated vector of one slot (kind 0 = key, 1 = value). */
static void load_slot(const uint8_t* chunk, int kind, int slot,
                      double* out /*[128]*/, int group) {
  const uint8_t* cb = chunk + (kind ? OR_VC : OR_KC) + slot * 32;
  const uint8_t* mb = chunk + (kind ? vmeta_off(group) : OR_KM) + slot * meta_stride(group);
  for (int ch = 0; ch < OR_D; ++ch) {
    int code = (cb[oracle_code_byte(ch)] >> oracle_code_shift(ch)) & 3;
    int g = group == 128 ? 0 : ch / OR_G;
    uint16_t s = (uint16_t)(mb[4 * g] | (mb[4 * g + 1] << 8));
    uint16_t m = (uint16_t)(mb[4 * g + 2] | (mb[4 * g + 3] << 8));
    out[ch] = dequant(code, s, m);
  }
}

/* Exported for tests: dequantized K and V of one slot of the pool. */
int oracle_read_slot(const uint8_t* pool, int h_kv, int page, int h, int slot,
                     double* khat, double* vhat, int group) {
  if (group != 32 && group != 128) return -1;
  const uint8_t* c = pool + ((size_t)page * h_kv + h) * chunk_bytes(group);
  load_slot(c, 0, slot, khat, group);
  load_slot(c, 1, slot, vhat, group);
  return 0;
}

/* ------------------------------------------------------------- rotations */

/* y = x R for one row vector x (Sec. 3.1 Eq. 4: the cache vector z becomes
 * zR); R row-major float32 [128][128]. */
static void rotate(const double* x, const float* R, double* y) {
  for (int j = 0; j < OR_D; ++j) {
    double acc = 0.0;
    for (int i = 0; i < OR_D; ++i) acc += x[i] * (double)R[i * OR_D + j];
    y[j] = acc;
  }
}

/* y = x R^T, the inverse of rotate() for orthogonal R. */
static void rotate_back(const double* x, const float* R, double* y) {
  for (int i = 0; i < OR_D; ++i) {
    double acc = 0.0;
    for (int j = 0; j < OR_D; ++j) acc += x[j] * (double)R[i * OR_D + j];
    y[i] = acc;
  }
}

/* Q2 applied group by group to a rotated 128-vector, groups of G = 32 or
 * 128 consecutive channels (Sec. 3.1, group size G; the paper's default is
 * 128, Sec. 5); codes and (optionally) the pre-rounding values are
 * returned, and scale/min per 32-channel block of the stored layout: with
 * G = 128 the one group's pair is repeated in its four blocks. */
static void quantize_vector(const double* z, float clip, int G, uint8_t* codes,
                            uint16_t* scale, uint16_t* mn, float* u) {
  for (int g0 = 0; g0 < OR_D; g0 += G) {
    float zf[OR_D];
    uint16_t s, m;
    for (int i = 0; i < G; ++i) zf[i] = (float)z[g0 + i];
    oracle_quantize_group(zf, G, clip, codes + g0, &s, &m, u ? u + g0 : NULL);
    for (int blk = g0 / OR_G; blk < (g0 + G) / OR_G; ++blk) {
      scale[blk] = s;
      mn[blk] = m;
    }
  }
}

/* -------------------------------------------------------- threads option */

static int g_threads = 1;
void oracle_set_threads(int n) { g_threads = n > 0 ? n : 1; }
int oracle_get_threads(void) { return g_threads; }

/* ----------------------------------------------------------- cache write */

/*
 * Cache write (Sec. 4.1, "Rotated INT2 Cache Reparameterization"; Appendix,
 * "Key-mean estimation and application"): for every new token t of
 * sequence b and KV head h,
 *     z_K = (k - mu_h) R_K,h      z_V = v R_V,h          (fp64)
 * then Q2 per group of 32 rotated channels (float32 decision), packed into
 * the page block_table[b][pos / 16], slot pos % 16, pos = pos0[b] + i.
 * Arrays: k, v bf16 bits [n_tok][h_kv][128]; R_k, R_v float32
 * [h_kv][128][128]; mu float32 [h_kv][128].  u_out (optional, float32
 * [n_tok][h_kv][2][128]) receives the pre-rounding values of the key
 * (index 0) and value (index 1) codes.  group: Q2 group size, 32 or 128.
 * Returns 0, or -1 when a table entry or position is out of range (nothing
 * is written for that token) or the group size is not supported.
 */
int oracle_kv_append(const uint16_t* k, const uint16_t* v, int n_tok,
                     const int32_t* cu_new, const int32_t* pos0,
                     const int32_t* block_table, int B, int max_pages,
                     uint8_t* pool, int num_pages, int h_kv, const float* R_k,
                     const float* R_v, const float* mu, float clip_k,
                     float clip_v, float* u_out, int group) {
  int bad = 0;
  if (group != 32 && group != 128) return -1;
  if (cu_new[0] != 0 || cu_new[B] != n_tok) return -1;
#pragma omp parallel for schedule(dynamic, 16) num_threads(g_threads) reduction(|: bad)
  for (int t = 0; t < n_tok; ++t) {
    int b = 0;
    while (b < B && !(cu_new[b] <= t && t < cu_new[b + 1])) ++b;
    if (b == B) { bad = 1; continue; }
    int pos = pos0[b] + (t - cu_new[b]);
    if (pos < 0 || pos >= max_pages * OR_P) { bad = 1; continue; }
    int page = block_table[(size_t)b * max_pages + pos / OR_P];
    if (page < 0 || page >= num_pages) { bad = 1; continue; }
    int slot = pos % OR_P;
    for (int h = 0; h < h_kv; ++h) {
      double x[OR_D], zk[OR_D], zv[OR_D];
      const uint16_t* kr = k + ((size_t)t * h_kv + h) * OR_D;
      const uint16_t* vr = v + ((size_t)t * h_kv + h) * OR_D;
      for (int i = 0; i < OR_D; ++i)
        x[i] = bf16_to_f64(kr[i]) - (double)mu[h * OR_D + i];
      rotate(x, R_k + (size_t)h * OR_D * OR_D, zk);
      for (int i = 0; i < OR_D; ++i) x[i] = bf16_to_f64(vr[i]);
      rotate(x, R_v + (size_t)h * OR_D * OR_D, zv);

      uint8_t ck[OR_D], cv[OR_D];
      uint16_t sk[4], mk[4], sv[4], mv[4];
      float* uk = u_out ? u_out + (((size_t)t * h_kv + h) * 2 + 0) * OR_D : NULL;
      float* uv = u_out ? u_out + (((size_t)t * h_kv + h) * 2 + 1) * OR_D : NULL;
      quantize_vector(zk, clip_k, group, ck, sk, mk, uk);
      quantize_vector(zv, clip_v, group, cv, sv, mv, uv);
      uint8_t* c = chunk_of(pool, page, h_kv, h, group);
      store_slot(c, OR_KC, OR_KM, slot, ck, sk, mk, group);
      store_slot(c, OR_VC, vmeta_off(group), slot, cv, sv, mv, group);
    }
  }
  return bad ? -1 : 0;
}

/* ------------------------------------------------------------ attention */

/* One query head against n dequantized rotated keys / values
 * (Sec. 3 Eq. 1-2 in the rotated basis): logits <qr, khat_s> / sqrt(d),
 * two-pass softmax, o' = sum_s p_s vhat_s.  Writes o' and (optionally) p. */
static void attend(const double* qr, const double* khat, const double* vhat,
                   int n, double* o_rot, double* p_out) {
  double* l = (double*)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
  double mx = -INFINITY;
  const double scale = 1.0 / sqrt((double)OR_D);
  for (int s = 0; s < n; ++s) {
    double acc = 0.0;
    for (int i = 0; i < OR_D; ++i) acc += qr[i] * khat[(size_t)s * OR_D + i];
    l[s] = acc * scale;
    if (l[s] > mx) mx = l[s];
  }
  double z = 0.0;
  for (int s = 0; s < n; ++s) {
    l[s] = exp(l[s] - mx);
    z += l[s];
  }
  for (int i = 0; i < OR_D; ++i) o_rot[i] = 0.0;
  for (int s = 0; s < n; ++s) {
    double p = l[s] / z;
    if (p_out) p_out[s] = p;
    for (int i = 0; i < OR_D; ++i) o_rot[i] += p * vhat[(size_t)s * OR_D + i];
  }
  free(l);
}

/* ------------------------------------------------------- BF16 windows */

/*
 * BF16 windows (Sec. 3.1, opening paragraph: the long history is stored in
 * INT2 while a small BF16 window is kept; Sec. 4.1: sink and recent tokens
 * stay in BF16 and their keys receive the same centering by mu; Sec. 5,
 * "Implementation Details": 64 sink and 256 recent tokens).  Of a sequence
 * that holds n tokens, position s is a window position when s < sink (the
 * attention sink) or s >= n - recent (the most recent tokens).  Its
 * effective key is k_s - mu and its effective value v_s, from the exact bf16
 * inputs, with no rotation or quantization; every other position attends
 * with its rotated INT2 record.
 *
 * Window store (the library's layout, restated from include/optr.h):
 * bf16 bits [n_slots][h_kv][2][sink + recent][128], index 0 keys, 1 values;
 * position s lives in row s when s < sink, else in row
 * sink + (s - sink) % recent.
 */
static int in_window(int s, int n, int sink, int recent) {
  return s < sink || s >= n - recent;
}

static int window_row(int s, int sink, int recent) {
  return s < sink ? s : sink + (s - sink) % recent;
}

static const uint16_t* window_vec(const uint16_t* win, int slot, int h_kv,
                                  int h, int kind, int row, int sink,
                                  int recent) {
  size_t rows = (size_t)(sink + recent);
  return win + ((((size_t)slot * h_kv + h) * 2 + kind) * rows + row) * OR_D;
}

/*
 * Window part of a cache write.  Sequence b's new tokens (rows cu_new[b] ..
 * cu_new[b+1]-1 of k / v) take positions pos0[b] .. end-1; a position s is
 * copied into the store when s < sink, or when recent > 0 and
 * s >= end - recent (those still in the recent window once this write is
 * cached; the ring row of an older position is overwritten in position
 * order).  k, v: bf16 bits [n_tok][h_kv][128].  Returns 0, or -1 when a
 * window slot is out of range (nothing is written for that sequence).
 */
int oracle_window_write(const uint16_t* k, const uint16_t* v, int n_tok,
                        const int32_t* cu_new, const int32_t* pos0, int B,
                        const int32_t* win_slot, int n_slots, int h_kv,
                        int sink, int recent, uint16_t* win) {
  int bad = 0;
  if (cu_new[0] != 0 || cu_new[B] != n_tok) return -1;
  for (int b = 0; b < B; ++b) {
    int m = cu_new[b + 1] - cu_new[b];
    if (m <= 0) continue;
    int slot = win_slot[b];
    if (slot < 0 || slot >= n_slots) { bad = 1; continue; }
    int end = pos0[b] + m;
    for (int i = 0; i < m; ++i) {
      int s = pos0[b] + i;
      if (!(s < sink || (recent > 0 && s >= end - recent))) continue;
      int row = window_row(s, sink, recent);
      int t = cu_new[b] + i;
      for (int h = 0; h < h_kv; ++h) {
        memcpy((void*)window_vec(win, slot, h_kv, h, 0, row, sink, recent),
               k + ((size_t)t * h_kv + h) * OR_D, OR_D * sizeof(uint16_t));
        memcpy((void*)window_vec(win, slot, h_kv, h, 1, row, sink, recent),
               v + ((size_t)t * h_kv + h) * OR_D, OR_D * sizeof(uint16_t));
      }
    }
  }
  return bad ? -1 : 0;
}

/*
 * Decode attention over the paged INT2 cache (Sec. 3 Eq. 1-2; Appendix,
 * "Rotated-query implementation": the cache stores k_R = Q2((k-mu)R_K) and
 * the query is rotated instead, q' = q R_K; Appendix, "Equivalent Inference
 * Implementation": o' = o R_V and o = o' R_V^T), with BF16 windows (above).
 * For each selected (b, j): h = j / (h_q / h_kv), tokens s < n = seq_lens[b],
 *     INT2 s:    l_s = <q_j R_K,h, khat_R,s> / sqrt(128), value vhat_R,s
 *     window s:  l_s = <q_j, k_s - mu_h> / sqrt(128),     value v_s
 *     p = softmax(l),
 *     out_j = (sum_INT2 p_s vhat_R,s) R_V,h^T + sum_window p_s v_s.
 * Without windows (sink = recent = 0) this is the INT2 path alone, and the
 * query-independent -q.mu term of the INT2 logits needs no explicit
 * treatment (softmax invariance); with windows the window logits carry it
 * explicitly so that both kinds of logits are those of centered keys.
 * q: bf16 bits [B][h_q][128].  out: float64 [B][h_q][128]; only selected
 * rows are written (sel_b/sel_j of length n_sel; n_sel = 0 selects all).
 * p_out (optional, float64, used with exactly one selected row) receives
 * the softmax weights.  mu float32 [h_kv][128]; win / win_slot may be NULL
 * when sink = recent = 0.  Returns 0, or -1 on an out-of-range table entry
 * or window slot.
 */
int oracle_decode_attention_win(const uint16_t* q, const int32_t* block_table,
                                const int32_t* seq_lens, int B, int max_pages,
                                const uint8_t* pool, int num_pages, int h_q,
                                int h_kv, const float* R_k, const float* R_v,
                                const float* mu, const uint16_t* win,
                                const int32_t* win_slot, int n_slots, int sink,
                                int recent, double* out, const int32_t* sel_b,
                                const int32_t* sel_j, int n_sel, double* p_out,
                                int group) {
  if (group != 32 && group != 128) return -1;
  int n_rows = n_sel > 0 ? n_sel : B * h_q;
  int ratio = h_q / h_kv;
  int bad = 0;
  const double scale = 1.0 / sqrt((double)OR_D);
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads) reduction(|: bad)
  for (int r = 0; r < n_rows; ++r) {
    int b = n_sel > 0 ? sel_b[r] : r / h_q;
    int j = n_sel > 0 ? sel_j[r] : r % h_q;
    int h = j / ratio;
    int n = seq_lens[b];
    double* o = out + ((size_t)b * h_q + j) * OR_D;
    if (n <= 0) {
      for (int i = 0; i < OR_D; ++i) o[i] = 0.0;
      continue;
    }
    if (n > max_pages * OR_P) { bad = 1; continue; }
    int slot = (sink > 0 || recent > 0) ? win_slot[b] : 0;
    if ((sink > 0 || recent > 0) && (slot < 0 || slot >= n_slots)) {
      bad = 1;
      continue;
    }
    double qx[OR_D], qr[OR_D];
    const uint16_t* qrow = q + ((size_t)b * h_q + j) * OR_D;
    for (int i = 0; i < OR_D; ++i) qx[i] = bf16_to_f64(qrow[i]);
    rotate(qx, R_k + (size_t)h * OR_D * OR_D, qr);
    /* per token: logit, value, and whether the value is in the rotated basis */
    double* l = (double*)malloc(sizeof(double) * (size_t)n);
    double* val = (double*)malloc(sizeof(double) * (size_t)n * OR_D);
    char* rot = (char*)malloc((size_t)n);
    int ok = 1;
    for (int s = 0; s < n && ok; ++s) {
      double* vs = val + (size_t)s * OR_D;
      double acc = 0.0;
      if (in_window(s, n, sink, recent)) {
        int row = window_row(s, sink, recent);
        const uint16_t* kw = window_vec(win, slot, h_kv, h, 0, row, sink, recent);
        const uint16_t* vw = window_vec(win, slot, h_kv, h, 1, row, sink, recent);
        for (int i = 0; i < OR_D; ++i)
          acc += qx[i] * (bf16_to_f64(kw[i]) - (double)mu[h * OR_D + i]);
        for (int i = 0; i < OR_D; ++i) vs[i] = bf16_to_f64(vw[i]);
        rot[s] = 0;
      } else {
        int page = block_table[(size_t)b * max_pages + s / OR_P];
        if (page < 0 || page >= num_pages) { ok = 0; break; }
        const uint8_t* c = pool + ((size_t)page * h_kv + h) * chunk_bytes(group);
        double kh[OR_D];
        load_slot(c, 0, s % OR_P, kh, group);
        load_slot(c, 1, s % OR_P, vs, group);
        for (int i = 0; i < OR_D; ++i) acc += qr[i] * kh[i];
        rot[s] = 1;
      }
      l[s] = acc * scale;
    }
    if (ok) {
      /* two-pass softmax, then the two value sums */
      double mx = -INFINITY, z = 0.0;
      for (int s = 0; s < n; ++s)
        if (l[s] > mx) mx = l[s];
      for (int s = 0; s < n; ++s) {
        l[s] = exp(l[s] - mx);
        z += l[s];
      }
      double orot[OR_D], owin[OR_D], oback[OR_D];
      for (int i = 0; i < OR_D; ++i) orot[i] = owin[i] = 0.0;
      for (int s = 0; s < n; ++s) {
        double p = l[s] / z;
        if (p_out && n_sel == 1) p_out[s] = p;
        double* acc = rot[s] ? orot : owin;
        for (int i = 0; i < OR_D; ++i) acc[i] += p * val[(size_t)s * OR_D + i];
      }
      rotate_back(orot, R_v + (size_t)h * OR_D * OR_D, oback);
      for (int i = 0; i < OR_D; ++i) o[i] = oback[i] + owin[i];
    } else {
      bad = 1;
    }
    free(l);
    free(val);
    free(rot);
  }
  return bad ? -1 : 0;
}

/* The INT2 path alone (no windows): oracle_decode_attention_win with
 * sink = recent = 0. */
int oracle_decode_attention(const uint16_t* q, const int32_t* block_table,
                            const int32_t* seq_lens, int B, int max_pages,
                            const uint8_t* pool, int num_pages, int h_q,
                            int h_kv, const float* R_k, const float* R_v,
                            double* out, const int32_t* sel_b,
                            const int32_t* sel_j, int n_sel, double* p_out,
                            int group) {
  return oracle_decode_attention_win(q, block_table, seq_lens, B, max_pages,
                                     pool, num_pages, h_q, h_kv, R_k, R_v,
                                     NULL, NULL, NULL, 0, 0, 0, out, sel_b,
                                     sel_j, n_sel, p_out, group);
}

/*
 * Dense single-head statement in the main paper's inverse-rotation form
 * (Sec. 3.1 Eq. 4 and Sec. 4.1): kbar_s = D_{R_K,c_K}(k_s - mu) =
 * Q2((k_s - mu) R_K) R_K^T, vbar_s = D_{R_V,c_V}(v_s) = Q2(v_s R_V) R_V^T,
 * then Eq. 1-2 with the plain query: a_s = <q, kbar_s>/sqrt(d),
 * p = softmax(a), out = sum_s p_s vbar_s.  With quantize = 0 the map Q2 is
 * the identity, so D_{R,c}(z) = z (Sec. 3.1).  Window positions (s < sink or
 * s >= n - recent; Sec. 3.1 and Sec. 4.1, BF16 sink and recent tokens with
 * the same key centering) keep kbar_s = k_s - mu and vbar_s = v_s.
 * q float64 [128]; K, V float64 [n][128]; R_k, R_v float32 [128][128];
 * mu float64 [128].
 */
int oracle_attention_dense_win(const double* q, const double* K,
                               const double* V, int n, const float* R_k,
                               const float* R_v, const double* mu,
                               int quantize, float clip_k, float clip_v,
                               int sink, int recent, double* out,
                               double* p_out, int group) {
  if (n <= 0) {
    for (int i = 0; i < OR_D; ++i) out[i] = 0.0;
    return 0;
  }
  double* kbar = (double*)malloc(sizeof(double) * (size_t)n * OR_D);
  double* vbar = (double*)malloc(sizeof(double) * (size_t)n * OR_D);
  for (int s = 0; s < n; ++s) {
    double x[OR_D], z[OR_D], zq[OR_D];
    for (int i = 0; i < OR_D; ++i) x[i] = K[(size_t)s * OR_D + i] - mu[i];
    if (in_window(s, n, sink, recent)) {
      for (int i = 0; i < OR_D; ++i) {
        kbar[(size_t)s * OR_D + i] = x[i];
        vbar[(size_t)s * OR_D + i] = V[(size_t)s * OR_D + i];
      }
      continue;
    }
    rotate(x, R_k, z);
    if (quantize) {
      uint8_t c[OR_D];
      uint16_t sc[4], mn[4];
      quantize_vector(z, clip_k, group, c, sc, mn, NULL);
      for (int i = 0; i < OR_D; ++i) zq[i] = dequant(c[i], sc[i / OR_G], mn[i / OR_G]);
    } else {
      for (int i = 0; i < OR_D; ++i) zq[i] = z[i];
    }
    rotate_back(zq, R_k, kbar + (size_t)s * OR_D);

    for (int i = 0; i < OR_D; ++i) x[i] = V[(size_t)s * OR_D + i];
    rotate(x, R_v, z);
    if (quantize) {
      uint8_t c[OR_D];
      uint16_t sc[4], mn[4];
      quantize_vector(z, clip_v, group, c, sc, mn, NULL);
      for (int i = 0; i < OR_D; ++i) zq[i] = dequant(c[i], sc[i / OR_G], mn[i / OR_G]);
    } else {
      for (int i = 0; i < OR_D; ++i) zq[i] = z[i];
    }
    rotate_back(zq, R_v, vbar + (size_t)s * OR_D);
  }
  attend(q, kbar, vbar, n, out, p_out);
  free(kbar);
  free(vbar);
  return 0;
}

/* The dense statement without windows. */
int oracle_attention_dense(const double* q, const double* K, const double* V,
                           int n, const float* R_k, const float* R_v,
                           const double* mu, int quantize, float clip_k,
                           float clip_v, double* out, double* p_out) {
  return oracle_attention_dense_win(q, K, V, n, R_k, R_v, mu, quantize, clip_k,
                                    clip_v, 0, 0, out, p_out, OR_G);
}

/* Exported for tests: z = x R (fp64) and the group quantization of z, for
 * one 128-vector, groups of `group` (32 or 128) channels. */
int oracle_rotate_quantize_g(const double* x, const float* R, float clip,
                             double* z, uint8_t* codes, uint16_t* scale,
                             uint16_t* mn, float* u, int group) {
  if (group != 32 && group != 128) return -1;
  rotate(x, R, z);
  quantize_vector(z, clip, group, codes, scale, mn, u);
  return 0;
}

int oracle_rotate_quantize(const double* x, const float* R, float clip,
                           double* z, uint8_t* codes, uint16_t* scale,
                           uint16_t* mn, float* u) {
  return oracle_rotate_quantize_g(x, R, clip, z, codes, scale, mn, u, OR_G);
}
