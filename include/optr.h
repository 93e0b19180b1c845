/*
 * optr.h -- C ABI of the rotated INT2 paged KV-cache hot path of OptR
 * ("Output-Aware Rotation for INT2 KV-Cache Quantization", arXiv 2608.02691).
 *
 * Two operations are exported:
 *
 *   optr_kv_append         cache write: center keys by mu, rotate K by R_k and
 *                          V by R_v, group-wise asymmetric INT2 quantize, pack
 *                          four codes per byte, scatter into paged blocks.
 *   optr_decode_attention  decode read: rotate each GQA query by its KV head's
 *                          R_k, stream the paged INT2 cache, dequantize in
 *                          registers, split-K online softmax, combine, apply
 *                          R_v^T to the attention output.
 *
 * Conventions (fixed for every entry point)
 * ------------------------------------------
 *  - Vectors are ROW vectors and a rotation acts on the right: z' = z R, i.e.
 *    z'[j] = sum_i z[i] * R[i][j]  (paper, Introduction and Sec. 3.1, Eq. 4).
 *    Every matrix argument is row-major float32, R[i][j] at offset i*D + j.
 *  - GQA grouping is contiguous: query head j reads KV head j / (h_q / h_kv)
 *    (Sec. 3, "Preliminaries": the set G_h of query heads sharing KV head h).
 *  - Attention logits use the scale 1/sqrt(D) (Sec. 3, Eq. 1).
 *  - Supported shape: head_dim D = 128, group G = 32 or 128, page_size
 *    P = 16.  Anything else returns OPTR_ERR_UNSUPPORTED.
 *
 * Quantizer Q2 (Sec. 3.1 "group-wise affine INT2 with clipping ratio c and
 * group size G"; Table "Default experimental settings").  The paper does not
 * write the formula out; this library fixes the following reading.  For one
 * token, one KV head and one group of G consecutive ROTATED channels
 * z_0..z_{G-1} (G = cfg.group: 32, or the paper's 128), evaluated in IEEE
 * float32 arithmetic:
 *      mn = c * min_i z_i,  mx = c * max_i z_i          (c = clip ratio)
 *      r  = mx - mn
 *      degenerate group (r is not > 1e-30 or r is not finite):
 *          all codes 0, scale = 0, min = fp16_rn(mn)
 *      otherwise:
 *          inv    = 3.0f / r
 *          u_i    = (clamp(z_i, mn, mx) - mn) * inv
 *          code_i = clamp(round_half_even(u_i), 0, 3)
 *          scale  = fp16_rn(r / 3.0f),  min = fp16_rn(mn)
 *      dequantized value: zhat_i = code_i * scale + min
 * Codes are decided from the unrounded range, never from the fp16 scale.
 * Inputs must be finite; NaN or Inf inputs give unspecified codes.
 *
 * Cache write (Sec. 4.1, "Rotated INT2 Cache Reparameterization"; Appendix,
 * "Key-mean estimation and application"):
 *      keys:   z_K = k R_k[h] - (mu[h] R_k[h])   ( = (k - mu[h]) R_k[h] )
 *      values: z_V = v R_v[h]
 * then Q2 with clip_k / clip_v.  mu[h] R_k[h] is precomputed once per head by
 * optr_params_create.  The dequantized rotated key is what the decode
 * attends with (Appendix, "Rotated-query implementation").
 *
 * Decode (Sec. 3 Eq. 1-2; Appendix, "Rotated-query implementation" and
 * "Equivalent Inference Implementation"), for sequence b, query head j,
 * KV head h = j / (h_q / h_kv), cached tokens s = 0 .. seq_lens[b]-1:
 *      q'_j  = q_j R_k[h]
 *      l_s   = <q'_j, khat_R,s> / sqrt(D)
 *      p     = softmax_s(l)
 *      o'_j  = sum_s p_s vhat_R,s
 *      out_j = o'_j R_v[h]^T                                   (float32)
 * The constant -q.mu term of the centered logits is omitted: softmax is
 * invariant to it (Appendix, "Equivalent Inference Implementation").
 * A sequence with seq_lens[b] == 0 gets an all-zero output.
 *
 * Paged pool layout (this library's choice; the paper inherits its layout
 * from its serving stack).  The pool is a byte array
 *      pool[num_pages][h_kv][OPTR_PAGE_HEAD_BYTES = 1536],
 * 16-byte aligned, and token position pos of sequence b lives in physical
 * page block_table[b * max_pages + pos / 16], slot pos % 16.  One
 * (page, KV head) chunk is:
 *      offset    0: K codes  [16 slots][32 bytes]
 *      offset  512: V codes  [16 slots][32 bytes]
 *      offset 1024: K meta   [16 slots][4 groups] {fp16 scale, fp16 min}
 *      offset 1280: V meta   [16 slots][4 groups] {fp16 scale, fp16 min}
 * The metadata has one {scale, min} entry per 32-channel block.  With
 * G = 128 the record is the paper's compact one (Sec. 5: one fp16 scale and
 * min per 128 channels, 2.25 bits per element), OPTR_PAGE_HEAD_BYTES_G128 =
 * 1152 bytes per (page, KV head):
 *      offset    0: K codes  [16 slots][32 bytes]
 *      offset  512: V codes  [16 slots][32 bytes]
 *      offset 1024: K meta   [16 slots] {fp16 scale, fp16 min}
 *      offset 1088: V meta   [16 slots] {fp16 scale, fp16 min}
 * and the pool is pool[num_pages][h_kv][1152] (optr_page_bytes).
 * Within a slot's 32 code bytes the groups are interleaved word-major:
 * channel ch = 32*g + 4*w + r  (group g in 0..3, w in 0..7, r in 0..3) is
 * stored in byte 4*w + g, bits [2r, 2r+1].  Byte 4*w + g therefore holds the
 * four codes of channels 32g+4w .. 32g+4w+3, lowest channel in the lowest
 * bits.  (Interleaving lets one decode lane fetch whole 32/64-bit words that
 * carry every group it needs.)  Every slot owns whole bytes, so appends to
 * different slots of one page never touch the same byte.
 *
 * Ownership and synchronisation
 * -----------------------------
 * The caller owns every tensor: q, k, v, tables, pool, out and workspace.
 * The library owns only optr_params (device copies of R_k, R_v, mu R_k, the
 * tensor-core splits of R, and a device error word).  optr_kv_append and
 * optr_decode_attention allocate nothing and never synchronise; they enqueue
 * kernels on the given stream and return.  Pointers named "device" must be
 * device memory of the current CUDA device; "host" pointers are read
 * synchronously before the call returns.
 *
 * Activations in host memory
 * --------------------------
 * The per-step activations -- k and v of a cache write, q and out of a
 * decode, all four of a decode step ("device or pinned host" below) -- may
 * instead be page-locked host memory (cudaHostAlloc, or host memory
 * registered with cudaHostRegister) that the runtime maps into the
 * device's address space.  The kernels then read and write them in place
 * over the host link (NVLink-C2C on a Grace host), so a step's host-device
 * transfers happen inside its own kernels, with no staging copies.
 * Pageable host memory, or a pointer the CUDA runtime does not know, is
 * refused with OPTR_ERR_INVALID_ARG before any launch.  A cache write of
 * more than 256 tokens from host memory runs on the CUDA-core kernel (the
 * tensor-core kernel loads its input by TMA from device memory).
 *
 * Errors
 * ------
 * Argument errors are detected on the host before any launch and return a
 * negative status; nothing is enqueued then.  Table contents (page ids,
 * positions, sequence lengths) live in device memory and are checked by the
 * kernels: an out-of-range entry is skipped (never dereferenced) and a bit is
 * set in the params' device error word, read with optr_device_error().  No
 * kernel traps, asserts or waits without bound.  A failed launch returns
 * OPTR_ERR_CUDA.
 */
#ifndef OPTR_H_
#define OPTR_H_

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

#define OPTR_HEAD_DIM 128
#define OPTR_GROUP 32
#define OPTR_PAGE_SIZE 16
#define OPTR_PAGE_HEAD_BYTES 1536
#define OPTR_K_CODES_OFFSET 0
#define OPTR_V_CODES_OFFSET 512
#define OPTR_K_META_OFFSET 1024
#define OPTR_V_META_OFFSET 1280
/* the compact record of G = 128 (one scale and min per 128 channels) */
#define OPTR_PAGE_HEAD_BYTES_G128 1152
#define OPTR_V_META_OFFSET_G128 1088

typedef enum {
  OPTR_OK = 0,
  OPTR_ERR_INVALID_ARG = -1, /* null pointer, non-positive size, bad ratio */
  OPTR_ERR_UNSUPPORTED = -2, /* D, G or P other than 128 / 32 / 16        */
  OPTR_ERR_OUT_OF_RANGE = -3,/* a size exceeds what the library handles    */
  OPTR_ERR_WORKSPACE = -4,   /* workspace null or smaller than required    */
  OPTR_ERR_CUDA = -5         /* a CUDA runtime call or launch failed        */
} optr_status;

/* Bits of the device error word (optr_device_error). */
#define OPTR_DEVERR_PAGE_ID 1u   /* block_table entry < 0 or >= num_pages  */
#define OPTR_DEVERR_POSITION 2u  /* append position >= max_pages * 16 or <0 */
#define OPTR_DEVERR_SEQ_LEN 4u   /* seq_lens[b] < 0 or > max_pages * 16     */
#define OPTR_DEVERR_CU_NEW 8u    /* cu_new not non-decreasing within n_tok  */
#define OPTR_DEVERR_FP16_RANGE 16u /* tensor-core append: |k| or |v| >= 65504 */
#define OPTR_DEVERR_TIMEOUT 32u  /* internal: a kernel's bounded wait gave up */
#define OPTR_DEVERR_WIN_SLOT 64u /* window slot of a sequence < 0 or >= n_slots */
#define OPTR_DEVERR_CALIB_RANGE 128u /* calibration: generator norm past exp's scaling range */

/* Kernel variants (for measurement; 0 picks the library default). */
#define OPTR_VARIANT_DEFAULT 0
#define OPTR_VARIANT_CUDA_CORE 1  /* float32 FMA on CUDA cores             */
#define OPTR_VARIANT_TENSOR 2     /* tensor-core path                      */

typedef struct optr_params optr_params; /* opaque, library-owned */

typedef struct {
  int h_q;            /* query heads; a positive multiple of h_kv          */
  int h_kv;           /* KV heads                                          */
  int head_dim;       /* must be 128                                       */
  int group;          /* Q2 group size: 32, or 128 (the paper's default)  */
  int page_size;      /* must be 16                                        */
  float clip_k;       /* key clip ratio c_K in (0, 1]; 1 = min-max          */
  float clip_v;       /* value clip ratio c_V in (0, 1]; 1 = min-max        */
  int append_variant; /* OPTR_VARIANT_*                                    */
  int decode_variant; /* OPTR_VARIANT_*                                    */
  int sink;           /* BF16 sink window: positions 0 .. sink-1; a multiple
                         of 16 in [0, 1024]; 0 = none (see BF16 windows)    */
  int recent;         /* BF16 recent window: the last `recent` positions;
                         [0, 1024]; 0 = none                               */
} optr_config;

/*
 * Create the per-layer rotation state (paper Algorithm "OptR offline
 * calibration": its output {R_K, R_V, mu} per KV head is this call's input).
 *   cfg   host; shapes and clip ratios (copied).
 *   R_k   host float32 [h_kv][D][D]: key rotation per KV head (orthogonal;
 *         orthogonality is the caller's contract and is not checked).
 *   R_v   host float32 [h_kv][D][D]: value rotation per KV head, or NULL
 *         when the value rotation is folded into the model's projections
 *         (Appendix "Equivalent Inference Implementation": W_V and W_O
 *         pre-multiplied by R_v): values are then quantized as given and
 *         the decode output is returned in that basis (as R_v = I; the
 *         decode skips its R_v^T step, the decode-step cache write its
 *         value rotation).
 *   mu    host float32 [h_kv][D]: per-channel key mean (Appendix, key-mean
 *         estimation).  Pass all zeros for no centering.
 *   out   host; receives the new handle, or NULL on error.
 * Allocates device memory on the current device (about h_kv * 200 KB) and
 * copies synchronously.  Returns OPTR_OK or a negative status.
 */
optr_status optr_params_create(const optr_config* cfg, const float* R_k,
                               const float* R_v, const float* mu,
                               optr_params** out);

/* Free a handle (NULL is ignored).  The caller ensures no enqueued work
 * still uses it. */
void optr_params_destroy(optr_params* p);

/* Bytes of one page across all KV heads: h_kv * 1536 (G = 32) or
 * h_kv * 1152 (the compact G = 128 record). */
size_t optr_page_bytes(const optr_params* p);

/*
 * Cache write (Sec. 4.1; Appendix, key-mean estimation and application).
 *   k, v        device or pinned host bf16 [n_tok][h_kv][D]: new keys
 *               (post-RoPE) and values.
 *   n_tok       host; total new tokens (0 is a no-op).
 *   cu_new      device int32 [B+1]: tokens of sequence b are rows
 *               cu_new[b] .. cu_new[b+1]-1 of k / v; cu_new[0] = 0,
 *               non-decreasing, cu_new[B] = n_tok.
 *   pos0        device int32 [B]: cache position of sequence b's first new
 *               token; token i of the sequence goes to position pos0[b] + i.
 *   block_table device int32 [B][max_pages]: logical page -> physical page.
 *   pool        device bytes [num_pages][h_kv][1536], written in place.
 * Each written slot's codes and metadata are replaced entirely.  Two appends
 * that target the same slot concurrently race.  The tensor-core variant
 * (the default for more than 256 new tokens, with either group size)
 * converts k and v to fp16: values of magnitude 65504 or more set
 * OPTR_DEVERR_FP16_RANGE and leave their token's record unspecified (use
 * the CUDA-core variant for such inputs).  Out-of-range table entries
 * or positions skip that token and set a device error bit.
 */
optr_status optr_kv_append(const optr_params* p, const void* k, const void* v,
                           int n_tok, const int32_t* cu_new,
                           const int32_t* pos0, const int32_t* block_table,
                           int B, int max_pages, uint8_t* pool, int num_pages,
                           cudaStream_t stream);

/* Workspace bytes optr_decode_attention (and _win, optr_decode_step and
 * _win) needs for this batch shape on the current device: split-K
 * partials, the rotated queries and, when p has BF16 windows, the window
 * partials. */
size_t optr_decode_workspace_size(const optr_params* p, int B, int max_pages);

/*
 * Decode attention over the paged INT2 cache (Sec. 3 Eq. 1-2; Appendix,
 * rotated-query implementation and equivalent inference implementation).
 *   q           device or pinned host bf16 [B][h_q][D]: post-RoPE queries,
 *               one per sequence.
 *   block_table device int32 [B][max_pages].
 *   seq_lens    device int32 [B]: cached tokens per sequence, 0 .. max_pages*16.
 *   pool        device bytes [num_pages][h_kv][1536] (read only).
 *   out         device or pinned host float32 [B][h_q][D]: attention output
 *               o = o' R_v^T.
 *   workspace   device, at least optr_decode_workspace_size(p, B, max_pages)
 *               bytes, 256-byte aligned; contents need no initialisation and
 *               are scratch between calls (concurrent calls need distinct
 *               workspaces).
 */
optr_status optr_decode_attention(const optr_params* p, const void* q,
                                  const int32_t* block_table,
                                  const int32_t* seq_lens, int B,
                                  int max_pages, const uint8_t* pool,
                                  int num_pages, float* out, void* workspace,
                                  size_t ws_bytes, cudaStream_t stream);

/*
 * One decode step: optr_kv_append(p, k, v, n_tok, cu_new, pos0, ...) of the
 * step's new tokens followed by optr_decode_attention(p, q, ...) over the
 * updated cache, with the same arguments, layouts, results and errors
 * (seq_lens counts the new tokens).  The paper's serving loop writes each
 * new token's rotated INT2 record and then attends over the cache (Sec. 4.1;
 * Appendix, key-mean estimation and rotated-query implementation); the two
 * first launches of that pair are independent (the cache write does not
 * touch the query), so for decode-step sized writes (n_tok <= 256) with the
 * default variants they run as one launch.  Other cases run exactly as the
 * two calls.  The decode may read pages that the step does not write
 * before the write has finished, so a physical page that receives one of
 * the step's tokens must not also be mapped by another sequence's block
 * table (pages holding a sequence's newest tokens are never shared in a
 * paged cache).  No allocation, no synchronisation.
 */
optr_status optr_decode_step(const optr_params* p, const void* q,
                             const void* k, const void* v, int n_tok,
                             const int32_t* cu_new, const int32_t* pos0,
                             const int32_t* block_table,
                             const int32_t* seq_lens, int B, int max_pages,
                             uint8_t* pool, int num_pages, float* out,
                             void* workspace, size_t ws_bytes,
                             cudaStream_t stream);

/*
 * Read and clear the device error word of p (OPTR_DEVERR_* bits).
 * Synchronises the device.  *flags receives 0 when no kernel reported a
 * table error since the last call.
 */
optr_status optr_device_error(const optr_params* p, uint32_t* flags);

/*
 * Stage timing for measurement (off by default).  optr_profile_enable(p, 1)
 * creates library-owned CUDA events; afterwards every optr_kv_append,
 * optr_decode_attention and optr_decode_step call made with p records an
 * event on its stream before and after each kernel it launches (for the
 * step's fused first launch the append stage covers it and the query
 * rotation stage is empty).  optr_profile_last waits for the
 * most recent calls' events and returns their durations in milliseconds:
 *   ms[0] append kernel, ms[1] query rotation + plan, ms[2] split-K partial,
 *   ms[3] combine (a stage that did not run reports 0).
 * Calls that overlap on the GPU share the events, so time one call at a
 * time.  optr_profile_enable(p, 0) destroys the events.
 */
optr_status optr_profile_enable(optr_params* p, int on);
optr_status optr_profile_last(const optr_params* p, float ms[4]);

/*
 * Decode attention without a caller-supplied workspace.  The paper has no
 * counterpart: this entry point exists for callers that cannot allocate
 * device memory at decode time -- for example an inference-engine plugin
 * whose host interface hands it tensors but no allocator, or a latency-
 * critical decode loop that must never call cudaMalloc (which synchronises
 * the device and can fail under memory pressure).
 *
 * Same arguments, result and errors as optr_decode_attention, minus the
 * workspace: the same argument and range checks run first, in the same
 * order; params with BF16 windows (cfg.sink or cfg.recent > 0) are refused
 * with OPTR_ERR_INVALID_ARG, as optr_decode_attention refuses them (there
 * is no windowed variant of this call).  The scratch memory is a fixed
 * array of OPTR_NOALLOC_SCRATCH_BYTES (16 MiB) in the library's device
 * image; every GPU that loads the library holds it until the process
 * exits.  A batch whose workspace would exceed it
 * (optr_decode_workspace_size(p, B, max_pages) > OPTR_NOALLOC_SCRATCH_BYTES;
 * about B > 230 at 8 KV heads on a 152-SM GPU) is rejected with
 * OPTR_ERR_WORKSPACE before any launch.
 *
 * optr_params_create looks up the array's device address on its device
 * (with that device current) and keeps it in the params, so this call does
 * no set-up of its own; params created after a cudaDeviceReset carry the
 * new address.  Nothing in the scratch needs to start at zero.  All calls
 * on a device share the one array, so calls that overlap on the GPU
 * (different streams, or different threads without ordering) race and
 * corrupt each other's results; serialise them.  This call allocates
 * nothing and never calls cudaMalloc or cudaFree.
 */
#define OPTR_NOALLOC_SCRATCH_BYTES (16u << 20)
optr_status optr_decode_attention_noalloc(const optr_params* p, const void* q,
                                          const int32_t* block_table,
                                          const int32_t* seq_lens, int B,
                                          int max_pages, const uint8_t* pool,
                                          int num_pages, float* out,
                                          cudaStream_t stream);

/*
 * BF16 windows (Sec. 3.1, opening paragraph: the long history is INT2 while
 * a small BF16 window is kept; Sec. 4.1: sink and recent tokens stay in
 * BF16 and their keys receive the same centering by mu; Sec. 5,
 * "Implementation Details": 64 sink and 256 recent tokens).  With
 * cfg.sink or cfg.recent > 0, a position s of a sequence holding n tokens
 * is a window position when s < sink or s >= n - recent.  The decode then
 * attends to it with its exact bf16 key and value:
 *      l_s = <q_j, k_s - mu[h]> / sqrt(D),   value v_s (not rotated),
 * and to every other position with its rotated INT2 record as above:
 *      out_j = (sum_INT2 p_s vhat_R,s) R_v[h]^T + sum_window p_s v_s.
 * Every token is still written to the INT2 pool (a token leaving the recent
 * window needs no re-quantization); window positions are not read from it.
 *
 * Window store (caller-owned, optr_window_bytes(p, n_slots) bytes, 16-byte
 * aligned): bf16 [n_slots][h_kv][2][sink + recent][D], plane 0 keys (as
 * given, not centered), plane 1 values (as given: with R_v = NULL that is
 * the folded basis).  Sequence b owns slot win_slot[b] (device int32 [B]);
 * position s lives in row s when s < sink, else in row
 * sink + (s - sink) % recent (a ring).  The cache write copies, for each
 * sequence, the positions s < sink and the positions s >= end - recent,
 * end = pos0[b] + its new-token count (those in the recent window once
 * the write is cached); ring rows of older positions are overwritten, so
 * a sequence's positions must be written in order.  A slot outside
 * [0, n_slots) skips the sequence's window work and sets
 * OPTR_DEVERR_WIN_SLOT.
 *
 * The entry points without _win require sink = recent = 0 and return
 * OPTR_ERR_INVALID_ARG otherwise; the _win entry points take the same
 * arguments plus the store (win, win_slot, n_slots), and with
 * sink = recent = 0 behave exactly as the plain ones (the store arguments
 * may then be NULL / 0).
 */
size_t optr_window_bytes(const optr_params* p, int n_slots);

optr_status optr_kv_append_win(const optr_params* p, const void* k,
                               const void* v, int n_tok, const int32_t* cu_new,
                               const int32_t* pos0, const int32_t* block_table,
                               int B, int max_pages, uint8_t* pool,
                               int num_pages, void* win,
                               const int32_t* win_slot, int n_slots,
                               cudaStream_t stream);

optr_status optr_decode_attention_win(const optr_params* p, const void* q,
                                      const int32_t* block_table,
                                      const int32_t* seq_lens, int B,
                                      int max_pages, const uint8_t* pool,
                                      int num_pages, const void* win,
                                      const int32_t* win_slot, int n_slots,
                                      float* out, void* workspace,
                                      size_t ws_bytes, cudaStream_t stream);

optr_status optr_decode_step_win(const optr_params* p, const void* q,
                                 const void* k, const void* v, int n_tok,
                                 const int32_t* cu_new, const int32_t* pos0,
                                 const int32_t* block_table,
                                 const int32_t* seq_lens, int B, int max_pages,
                                 uint8_t* pool, int num_pages, void* win,
                                 const int32_t* win_slot, int n_slots,
                                 float* out, void* workspace, size_t ws_bytes,
                                 cudaStream_t stream);

/* Static description of a status code. */
const char* optr_strerror(optr_status s);

/*
 * Offline rotation calibration of one KV head (Sec. 4.2 "Orthogonal
 * Rotation Refinement", Sec. 4.3 output-aware key objective, Sec. 4.4 value
 * objective, Sec. 4.5 INT2-aware calibration with the straight-through
 * estimator; Appendix, "OptR Algorithm"; Sec. 5: 80 Adam steps, lr 0.02,
 * held-out selection every 20 steps).  It produces the R_k[h], R_v[h] and
 * mu[h] that optr_params_create takes.  With d = 128, scale = 1/sqrt(d):
 *   mu      = mean over the calibration trace's keys
 *   R_K     = R0_K exp(A_K - A_K^T),  R_V = R0_V exp(A_V - A_V^T)
 *   keys    kt_s = Q2((k_s - mu) R_K, clip_k) R_K^T   (window pairs: k_s - mu)
 *   values  vt_s = Q2(v_s R_V, clip_v) R_V^T          (window pairs: v_s)
 *   p_t     = softmax_{s <= t}(scale q_t . k_s),  p^K_t the same on kt
 *   L_K     = mean_{t,j} [KL(p_t || p^K_t)
 *                         + lam |((p^K_t - p_t) V) W_O[j]^T|^2 / d_model]
 *   L_V     = mean_{t,j} |(phat_t (Vt - V)) W_O[j]^T|^2 / d_model,
 *             phat the key attention under the selected R_K
 * with Q2 the cache's quantizer (group cfg.group, fp16 scale and min taken
 * from the float32 rounding of the float64 values) and its gradient the
 * indicator of the clipped range [c min, c max] of the value's group.  A
 * position s is a BF16-window position for query position t when
 * s < sink or s > t - recent.  Adam (b1 0.9, b2 0.999, eps 1e-8) runs
 * `steps` steps on A_K from 0, scoring R_K on the held-out trace at step
 * 0, every select_every steps and after the last step and keeping the best;
 * then the same for A_V under the selected R_K.  Float64 throughout, on the
 * GPU; the gradient is written out (Frechet derivative of the matrix
 * exponential from a Taylor series with scaling and squaring).
 *
 * All arrays are device float64 (int32 positions), row-major:
 *   q [nt][g][128] (the g query heads of the KV head at query positions
 *   t_pos[nt], each in 0 .. T-1), K, V [T][128], W_O [g][d_model][128]
 *   (W_O[j] maps query head j's output to the model); the held-out trace
 *   likewise with T_held / nt_held (T_held = 0: scored on the calibration
 *   trace, pointers may be NULL); R0_K, R0_V [128][128] or NULL for the
 *   normalised Hadamard matrix.  Outputs R_K, R_V [128][128], mu [128],
 *   hist_k, hist_v [steps] (the training loss before each step).
 * The workspace (optr_calib_workspace_size bytes, 256-byte aligned) is
 * scratch.  The call enqueues its kernels on `stream` and synchronises it
 * before returning; OPTR_ERR_OUT_OF_RANGE reports a generator whose norm
 * left the exponential's scaling range (|A - A^T| above 2^15).
 */
typedef struct {
  int g;              /* query heads of the KV head (1 .. 64)                */
  int d_model;        /* rows of each W_O[j]                                 */
  int T, nt;          /* calibration trace: tokens, query positions          */
  int T_held, nt_held;/* held-out trace; T_held = 0: none                    */
  int steps;          /* Adam steps per rotation (paper: 80)                 */
  int select_every;   /* held-out selection period (paper: 20)               */
  int group;          /* Q2 group size: 32 or 128                            */
  int sink, recent;   /* BF16 windows (0, 0: none)                           */
  double lr, lam;     /* Adam learning rate (0.02), key-loss lambda          */
  double clip_k, clip_v; /* Q2 clipping ratios in (0, 1]                     */
} optr_calib_config;

/* Workspace bytes of optr_calibrate_head / optr_calib_loss_grad for this
 * configuration, or 0 when the configuration is invalid. */
size_t optr_calib_workspace_size(const optr_calib_config* c);

optr_status optr_calibrate_head(
    const optr_calib_config* c, const double* q, const double* K,
    const double* V, const int32_t* t_pos, const double* W_O,
    const double* q_held, const double* K_held, const double* V_held,
    const int32_t* t_pos_held, const double* R0_K, const double* R0_V,
    double* R_K, double* R_V, double* mu, double* hist_k, double* hist_v,
    void* workspace, size_t ws_bytes, cudaStream_t stream);

/* One evaluation of the objective on the calibration trace (held-out
 * fields unused): which = 0, L_K at R_K = R0 exp(A - A^T); which = 1, L_V at
 * R_V = R0 exp(A - A^T) under the key rotation R_K.  mu is given.  Writes
 * the loss (device double) and, when dA is not NULL, its gradient with
 * respect to A (device [128][128]).  Synchronises the stream. */
optr_status optr_calib_loss_grad(const optr_calib_config* c, int which,
                                 const double* q, const double* K,
                                 const double* V, const int32_t* t_pos,
                                 const double* W_O, const double* mu,
                                 const double* R_K, const double* R0,
                                 const double* A, double* loss, double* dA,
                                 void* workspace, size_t ws_bytes,
                                 cudaStream_t stream);

/*
 * Self-test of the bounded waits (library machinery; the paper has no
 * counterpart).  Every mbarrier wait in the tcgen05 kernels gives up after
 * a time limit, flags OPTR_DEVERR_TIMEOUT, drains its own copies and frees
 * its tensor memory, so that no wait can hang the GPU.  This call launches
 * one CTA that allocates the cache write's tensor-memory columns, waits
 * with the limit limit_ns (1 ms .. 2 s, else OPTR_ERR_INVALID_ARG) on an
 * mbarrier phase that nothing completes, and leaves through the cache
 * write's exit path: OPTR_DEVERR_TIMEOUT is then set in p's device error
 * word (optr_device_error) and the columns are free again.  Asynchronous on
 * `stream`; no allocation.
 */
optr_status optr_selftest_wait_timeout(const optr_params* p,
                                       unsigned long long limit_ns,
                                       cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* OPTR_H_ */
