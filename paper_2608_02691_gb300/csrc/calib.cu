// Offline rotation calibration on the GPU (Sec. 4.2-4.5; Appendix, "OptR
// Algorithm"): per KV head, Adam on the skew generators A_K and A_V of
//   R_K = R_K^0 exp(A_K - A_K^T),  R_V = R_V^0 exp(A_V - A_V^T)
// against the output-aware objectives
//   L_K = mean_{t,j} KL(p_t || p_t^K) + lambda ||e_K(t,j)||^2 / d_model,
//   L_V = mean_{t,j} ||e_V(t,j)||^2 / d_model,
// with the cache's INT2 quantizer Q2 inside the effective keys and values and
// its straight-through gradient, and held-out selection of the rotations.
//
// Everything runs in float64 on the CUDA cores in this file's kernels: the
// calibration is a one-time offline pass, this GPU's tensor cores have no
// float64 path, and float64 keeps the 80-step trajectory reproducible.
// The gradient is written out (no autograd):
//   keys    Z = (K - mu) R, Zh = Q2(Z), Kt = Zh R^T, l = scale q Kt^T
//           dl = c [(pk - p) + pk (gv - sum_s pk gv)],  gv = U V^T,
//           U = (2 lambda / d_model) e W_O,  c = 1 / (nt g)
//           dKt = dl^T q,  dR = dKt^T Zh + (K - mu)^T (1{inside} (dKt R))
//   values  Vt = Q2(V R) R^T, e = phat_nw (Vt - V) W_O^T
//           dVt = phat_nw^T U,  U = 2 c / d_model e W_O
//           dR = dVt^T Zh + V^T (1{inside} (dVt R))
//   both    dE = R0^T dR, dS = L_exp(S^T, dE), dA = dS - dS^T
// where L_exp(X, H) is the Frechet derivative of the matrix exponential
// (the adjoint of L_exp(S, .) is L_exp(S^T, .)).  exp and L_exp come from
// one Taylor series of the block matrix [[X, H], [0, X]] with scaling and
// squaring: the upper-right block of its exponential is L_exp(X, H).
#include <math.h>
#include <string.h>

#include <algorithm>
#include <vector>

#include "optr_internal.cuh"

namespace optr {
namespace {

constexpr int kCD = 128;  // head dimension d

// ------------------------------------------------------------------ GEMM
// C[b] = alpha op(A[b]) op(B[b]) + beta C[b] + diag I, float64, row-major
// with leading dimensions; op = transpose when tA / tB.  Square output tiles
// of 64, 32 or 16 (gemm_f64_kernel below), 16-deep k slices in shared
// memory, 256 threads per CTA.
// gate: when non-null and gate_idx >= *gate, the launch instead copies
// `pass` into C (or does nothing when pass is null); this lets a fixed
// number of launches apply a device-decided number of squarings.
struct Gemm {
  int M, N, K;
  const double* A;
  long long lda, sA;
  int tA;
  const double* B;
  long long ldb, sB;
  int tB;
  double* C;
  long long ldc, sC;
  double alpha, beta, diag;
  const int* gate;
  int gate_idx;
  const double* pass;
};

constexpr int kTK = 16;

// TILE x TILE outputs per CTA of 256 threads ((TILE / 16)^2 outputs each).
// The host picks the largest tile, then a split of K into kc chunks, so that
// a call covers about two CTAs per SM (float64 runs at a few FMAs per clock
// per SM on this GPU).  With kc > 1 chunk z of a product writes its raw sum
// to P[z][b]; the last of the tile's kc CTAs to finish (a per-tile arrival
// counter, left at 0 again) adds the chunks in a fixed order, z = 0 .. kc-1,
// so the result does not depend on which CTA that is.
template <int TILE>
__global__ void __launch_bounds__(256) gemm_f64_kernel(Gemm g, int kc, double* P,
                                                       int* tcnt) {
  constexpr int R = TILE / 16;  // outputs per thread per dimension
  __shared__ double As[kTK][TILE + 1];
  __shared__ double Bs[kTK][TILE + 1];
  __shared__ int s_last;
  const int b = blockIdx.z / kc, z = blockIdx.z % kc;
  const int m0 = blockIdx.y * TILE, n0 = blockIdx.x * TILE;
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  double* C = g.C + (long long)b * g.sC;
  if (g.gate != nullptr && g.gate_idx >= *g.gate) {
    if (g.pass != nullptr && z == 0) {
      for (int i = tid; i < TILE * TILE; i += 256) {
        const int r = m0 + i / TILE, c = n0 + i % TILE;
        if (r < g.M && c < g.N) C[r * g.ldc + c] = g.pass[r * g.ldc + c];
      }
    }
    return;
  }
  const double* A = g.A + (long long)b * g.sA;
  const double* B = g.B + (long long)b * g.sB;
  // this CTA's K range: chunk z of kc, in whole kTK slices
  const int nsl = (g.K + kTK - 1) / kTK;
  const int kb = (int)((long long)z * nsl / kc) * kTK;
  const int ke = min(g.K, (int)((long long)(z + 1) * nsl / kc) * kTK);
  double acc[R][R];
#pragma unroll
  for (int i = 0; i < R; ++i)
#pragma unroll
    for (int j = 0; j < R; ++j) acc[i][j] = 0.0;
  for (int k0 = kb; k0 < ke; k0 += kTK) {
    for (int i = tid; i < TILE * kTK; i += 256) {
      int mm, kk;
      if (g.tA) { kk = i / TILE; mm = i % TILE; } else { mm = i / kTK; kk = i % kTK; }
      const int gm = m0 + mm, gk = k0 + kk;
      double x = 0.0;
      if (gm < g.M && gk < ke) x = g.tA ? A[gk * g.lda + gm] : A[gm * g.lda + gk];
      As[kk][mm] = x;
    }
    for (int i = tid; i < kTK * TILE; i += 256) {
      int kk, nn;
      if (g.tB) { nn = i / kTK; kk = i % kTK; } else { kk = i / TILE; nn = i % TILE; }
      const int gk = k0 + kk, gn = n0 + nn;
      double x = 0.0;
      if (gk < ke && gn < g.N) x = g.tB ? B[gn * g.ldb + gk] : B[gk * g.ldb + gn];
      Bs[kk][nn] = x;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < kTK; ++kk) {
      double a[R], bb[R];
#pragma unroll
      for (int i = 0; i < R; ++i) a[i] = As[kk][ty * R + i];
#pragma unroll
      for (int j = 0; j < R; ++j) bb[j] = Bs[kk][tx * R + j];
#pragma unroll
      for (int i = 0; i < R; ++i)
#pragma unroll
        for (int j = 0; j < R; ++j) acc[i][j] = fma(a[i], bb[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < R; ++i) {
    const int r = m0 + ty * R + i;
    if (r >= g.M) continue;
#pragma unroll
    for (int j = 0; j < R; ++j) {
      const int c = n0 + tx * R + j;
      if (c >= g.N) continue;
      if (kc > 1) {
        P[(((long long)z * gridDim.z / kc + b) * g.M + r) * g.N + c] = acc[i][j];
        continue;
      }
      double x = g.alpha * acc[i][j];
      if (g.beta != 0.0) x += g.beta * C[r * g.ldc + c];
      if (r == c) x += g.diag;
      C[r * g.ldc + c] = x;
    }
  }
  if (kc == 1) return;
  // split K: the tile's last CTA to arrive adds the kc chunk sums in order
  __threadfence();
  __syncthreads();
  const int tile_id = (b * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x;
  if (tid == 0) s_last = atomicAdd(tcnt + tile_id, 1) == kc - 1;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const int batch = gridDim.z / kc;
  for (int i = tid; i < TILE * TILE; i += 256) {
    const int r = m0 + i / TILE, c = n0 + i % TILE;
    if (r >= g.M || c >= g.N) continue;
    double sum = 0.0;
    for (int zz = 0; zz < kc; ++zz)
      sum += __ldcg(P + (((long long)zz * batch + b) * g.M + r) * g.N + c);
    double x = g.alpha * sum;
    if (g.beta != 0.0) x += g.beta * C[r * g.ldc + c];
    if (r == c) x += g.diag;
    C[r * g.ldc + c] = x;
  }
  if (tid == 0) tcnt[tile_id] = 0;
}

// ------------------------------------------------------- small kernels

__global__ void col_mean_kernel(const double* __restrict__ K, int T,
                                double* __restrict__ mu) {
  const int c = threadIdx.x;  // 128 threads
  double s = 0.0;
  for (int t = 0; t < T; ++t) s += K[(long long)t * kCD + c];
  mu[c] = s / (double)T;
}

// Kc = K - mu (rows of d)
__global__ void center_kernel(const double* __restrict__ K,
                              const double* __restrict__ mu, long long n,
                              double* __restrict__ Kc) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x)
    Kc[i] = K[i] - mu[i % kCD];
}

// S = X - X^T (d x d)
__global__ void skew_kernel(const double* __restrict__ X, double* __restrict__ S) {
  const int i = blockIdx.x, j = threadIdx.x;
  S[i * kCD + j] = X[i * kCD + j] - X[j * kCD + i];
}

// normalised Sylvester-Hadamard matrix: (-1)^popcount(i & j) / sqrt(d)
__global__ void hadamard_kernel(double* __restrict__ H) {
  const int i = blockIdx.x, j = threadIdx.x;
  H[i * kCD + j] = (__popc(i & j) & 1 ? -1.0 : 1.0) / sqrt((double)kCD);
}

__global__ void fill_kernel(double* __restrict__ x, long long n, double v) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x)
    x[i] = v;
}

__global__ void copy_kernel(const double* __restrict__ x, long long n,
                            double* __restrict__ y) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x)
    y[i] = x[i];
}

// C = A - B
__global__ void sub_kernel(const double* __restrict__ A, const double* __restrict__ B,
                           long long n, double* __restrict__ C) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x)
    C[i] = A[i] - B[i];
}

// X *= M elementwise (M is 0 or 1)
__global__ void mask_mul_kernel(double* __restrict__ X, const double* __restrict__ M,
                                long long n) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x)
    X[i] = X[i] * M[i];
}

// log(max(p, 1e-300))
__global__ void logclamp_kernel(const double* __restrict__ P, long long n,
                                double* __restrict__ L) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n;
       i += (long long)gridDim.x * blockDim.x)
    L[i] = log(fmax(P[i], 1e-300));
}

__device__ __forceinline__ bool is_window(int s, int t, int sink, int recent) {
  return s < sink || s > t - recent;
}

// Q2 (Sec. 3.1: group-wise asymmetric INT2 with clipping ratio c, fp16 scale
// and min; the cache quantizer's rule) with the straight-through indicator
// (Sec. 4.5): per row and group of G channels of Z, mn = c min, mx = c max,
// r = mx - mn, u = (clamp(z, mn, mx) - mn) * 3 / r, code = clamp(rint(u), 0,
// 3), zh = code * fp16(r / 3) + fp16(mn) (fp16 values of the float32
// rounding), inside = mn <= z <= mx.  Degenerate groups (r <= 1e-30): code
// 0, scale 0.  One warp per (row, group).
__global__ void q2_kernel(const double* __restrict__ Z, int rows, int G,
                          double clip, double* __restrict__ Zh,
                          double* __restrict__ inside) {
  const int lane = threadIdx.x & 31;
  const long long wid = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5;
  const int groups = kCD / G;
  if (wid >= (long long)rows * groups) return;
  const long long row = wid / groups;
  const int g0 = (int)(wid % groups) * G;
  const int per = G / 32;  // 1 or 4 channels per lane
  double z[4];
  double lo = INFINITY, hi = -INFINITY;
  for (int e = 0; e < per; ++e) {
    z[e] = Z[row * kCD + g0 + e * 32 + lane];
    lo = fmin(lo, z[e]);
    hi = fmax(hi, z[e]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = fmin(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    hi = fmax(hi, __shfl_xor_sync(0xffffffffu, hi, o));
  }
  const double mn = clip * lo, mx = clip * hi;
  const double r = mx - mn;
  const bool deg = !(r > 1e-30);
  const double inv = deg ? 0.0 : 3.0 / r;
  const double scale = deg ? 0.0 : (double)__half2float(__float2half_rn(__double2float_rn(r / 3.0)));
  const double mn16 = (double)__half2float(__float2half_rn(__double2float_rn(mn)));
  for (int e = 0; e < per; ++e) {
    const double u = (fmin(fmax(z[e], mn), mx) - mn) * inv;
    const double code = fmin(fmax(rint(u), 0.0), 3.0);
    const long long i = row * kCD + g0 + e * 32 + lane;
    Zh[i] = __dadd_rn(__dmul_rn(code, scale), mn16);
    inside[i] = (z[e] >= mn && z[e] <= mx) ? 1.0 : 0.0;
  }
}

// Row (j, t) of [g][nt][T]: logits scale * x (x = the row of X, or of Xc
// at the BF16-window pairs when windows), masked to s <= t_pos[t]; the
// softmax goes to P.  When Pref is given, rowv[row] = KL(Pref || P) =
// sum_s pref (logpref - log max(p, 1e-300)), with log p = l - m - log(sum)
// (p = 0 entries: log 1e-300; below 1e-300 the clamp).  One block of 256
// threads per row; exp(l - m) is stored in the sum pass and normalised in
// the last.
__device__ __forceinline__ double block_reduce(double v, bool is_max, double* sh) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const double u = __shfl_xor_sync(0xffffffffu, v, o);
    v = is_max ? fmax(v, u) : v + u;
  }
  __syncthreads();  // sh free from an earlier reduction
  if (lane == 0) sh[w] = v;
  __syncthreads();
  double r = sh[0];
  for (int i = 1; i < 8; ++i) r = is_max ? fmax(r, sh[i]) : r + sh[i];
  return r;
}

__global__ void __launch_bounds__(256) softmax_rows_kernel(
    const double* __restrict__ X, const double* __restrict__ Xc, int rows, int nt,
    int T, const int32_t* __restrict__ t_pos, double scale, int sink, int recent,
    double* __restrict__ P, const double* __restrict__ Pref,
    const double* __restrict__ logPref, double* __restrict__ rowv) {
  __shared__ double sh[8];
  const long long row = blockIdx.x;
  const int t = t_pos[row % nt];
  const bool win = Xc != nullptr;
  const double* x = X + row * (long long)T;
  const double* xc = win ? Xc + row * (long long)T : nullptr;
  auto logit = [&](int s) {
    const double v = (win && is_window(s, t, sink, recent)) ? xc[s] : x[s];
    return v * scale;
  };
  double m = -INFINITY;
  for (int s = threadIdx.x; s < T; s += 256)
    if (s <= t) m = fmax(m, logit(s));
  m = block_reduce(m, true, sh);
  double* p = P + row * (long long)T;
  double sum = 0.0;
  for (int s = threadIdx.x; s < T; s += 256) {
    const double e = s <= t ? exp(logit(s) - m) : 0.0;
    p[s] = e;
    sum += e;
  }
  sum = block_reduce(sum, false, sh);
  const double lsum = Pref != nullptr ? log(sum) : 0.0;
  double kl = 0.0;
  for (int s = threadIdx.x; s < T; s += 256) {
    const double v = p[s] / sum;
    p[s] = v;
    if (Pref != nullptr) {
      const double lp = v > 1e-300 ? (logit(s) - m) - lsum : log(1e-300);
      kl += Pref[row * (long long)T + s] * (logPref[row * (long long)T + s] - lp);
    }
  }
  if (Pref != nullptr) {
    kl = block_reduce(kl, false, sh);
    if (threadIdx.x == 0) rowv[row] = kl;
  }
}

// Gradient of the key loss with respect to the raw logits x of row (j, t)
// (l = scale x): G[s] = coef * ((pk - p) + pk (gv - sum_s pk gv)) at the
// causal non-window pairs, 0 elsewhere.  In place over GV.  One warp per row.
__global__ void key_row_grad_kernel(const double* __restrict__ PK,
                                    const double* __restrict__ Pref,
                                    double* __restrict__ GV, int rows, int nt,
                                    int T, const int32_t* __restrict__ t_pos,
                                    double coef, int sink, int recent, int win) {
  const int lane = threadIdx.x & 31;
  const long long row = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5;
  if (row >= rows) return;
  const int t = t_pos[row % nt];
  const double* pk = PK + row * (long long)T;
  const double* p = Pref + row * (long long)T;
  double* gv = GV + row * (long long)T;
  double gbar = 0.0;
  for (int s = lane; s < T; s += 32) gbar += pk[s] * gv[s];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) gbar += __shfl_xor_sync(0xffffffffu, gbar, o);
  for (int s = lane; s < T; s += 32) {
    double gsum = 0.0;
    if (s <= t && !(win && is_window(s, t, sink, recent)))
      gsum = coef * ((pk[s] - p[s]) + pk[s] * (gv[s] - gbar));
    gv[s] = gsum;
  }
}

// Zero the BF16-window pairs of rows (j, t) of [g][nt][T].
__global__ void zero_window_kernel(double* __restrict__ P, int rows, int nt, int T,
                                   const int32_t* __restrict__ t_pos, int sink,
                                   int recent) {
  const int lane = threadIdx.x & 31;
  const long long row = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5;
  if (row >= rows) return;
  const int t = t_pos[row % nt];
  for (int s = lane; s < T; s += 32)
    if (is_window(s, t, sink, recent)) P[row * (long long)T + s] = 0.0;
}

// rowv[row] = (add ? rowv[row] : 0) + lam * (sum_c E[row][c]^2) / dm
__global__ void row_sqsum_kernel(const double* __restrict__ E, int rows, int dm,
                                 double lam, int add, double* __restrict__ rowv) {
  const int lane = threadIdx.x & 31;
  const long long row = (blockIdx.x * (long long)blockDim.x + threadIdx.x) >> 5;
  if (row >= rows) return;
  double s = 0.0;
  for (int c = lane; c < dm; c += 32) {
    const double e = E[row * (long long)dm + c];
    s += e * e;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (lane == 0) {
    const double v = lam * s / (double)dm;
    rowv[row] = add ? rowv[row] + v : v;
  }
}

// out = (sum_i rowv[i]) / n, one block of 1024 threads, fixed order
__global__ void __launch_bounds__(1024) loss_reduce_kernel(const double* __restrict__ rowv,
                                                           int rows, double n,
                                                           double* __restrict__ out) {
  __shared__ double red[1024];
  double s = 0.0;
  for (int i = threadIdx.x; i < rows; i += 1024) s += rowv[i];
  red[threadIdx.x] = s;
  __syncthreads();
  for (int w = 512; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) *out = red[0] / n;
}

// Adam (Kingma & Ba), in the order m = b1 m + (1 - b1) g,
// v = b2 v + ((1 - b2) g) g, x -= (lr mh) / (sqrt(vh) + eps), mh = m / bc1,
// vh = v / bc2; separate roundings (no contraction).
__global__ void adam_kernel(double* __restrict__ x, const double* __restrict__ g,
                            double* __restrict__ m, double* __restrict__ v,
                            int n, double lr, double b1, double omb1, double b2,
                            double omb2, double bc1, double bc2, double eps) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const double gi = g[i];
  const double mi = __dadd_rn(__dmul_rn(b1, m[i]), __dmul_rn(omb1, gi));
  const double vi = __dadd_rn(__dmul_rn(b2, v[i]), __dmul_rn(__dmul_rn(omb2, gi), gi));
  m[i] = mi;
  v[i] = vi;
  const double mh = __ddiv_rn(mi, bc1), vh = __ddiv_rn(vi, bc2);
  x[i] = __dsub_rn(x[i], __ddiv_rn(__dmul_rn(lr, mh), __dadd_rn(__dsqrt_rn(vh), eps)));
}

// Held-out selection: keep R when its score is the first or a lower one.
__global__ void select_kernel(const double* __restrict__ score,
                              double* __restrict__ best, int first,
                              const double* __restrict__ R,
                              double* __restrict__ bestR) {
  __shared__ int take;
  if (threadIdx.x == 0) {
    take = first || *score < *best;
    if (take) *best = *score;
  }
  __syncthreads();
  if (take)
    for (int i = threadIdx.x; i < kCD * kCD; i += blockDim.x) bestR[i] = R[i];
}

// Scaling for exp: s = smallest integer with max(|S|_1, |S|_inf) 2^-s <= 1/2
// (at most kMaxSquare), X = sign * S * 2^-s and, when H is given,
// Hs = H * 2^-s (the block matrix [[X, H], [0, X]] is scaled as a whole).
constexpr int kMaxSquare = 16;  // norms up to 2^15
__global__ void expm_prep_kernel(const double* __restrict__ S, double sign,
                                 const double* __restrict__ H,
                                 double* __restrict__ Xs, double* __restrict__ Hs,
                                 int* __restrict__ s_out, unsigned* err) {
  __shared__ double red[kCD];
  __shared__ int s_sh;
  const int i = threadIdx.x;  // 128 threads
  double rs = 0.0, cs = 0.0;
  for (int j = 0; j < kCD; ++j) {
    rs += fabs(S[i * kCD + j]);
    cs += fabs(S[j * kCD + i]);
  }
  red[i] = fmax(rs, cs);
  __syncthreads();
  for (int w = kCD / 2; w > 0; w >>= 1) {
    if (i < w) red[i] = fmax(red[i], red[i + w]);
    __syncthreads();
  }
  if (i == 0) {
    int s = 0;
    double nrm = red[0];
    while (nrm > 0.5 && s < kMaxSquare) {
      nrm *= 0.5;
      ++s;
    }
    if (nrm > 0.5 || !(red[0] == red[0])) atomicOr(err, OPTR_DEVERR_CALIB_RANGE);
    s_sh = s;
    *s_out = s;
  }
  __syncthreads();
  const double f = sign * ldexp(1.0, -s_sh);
  for (int j = 0; j < kCD; ++j) {
    Xs[i * kCD + j] = f * S[i * kCD + j];
    if (H != nullptr) Hs[i * kCD + j] = ldexp(H[i * kCD + j], -s_sh);
  }
}

}  // namespace

// ------------------------------------------------------------ host side

namespace {

constexpr int kTaylor = 18;        // Taylor degree of exp on ||X|| <= 1/2
constexpr int kSquareLaunches = kMaxSquare;  // one gated launch per possible squaring

__global__ void eye_kernel(double* __restrict__ X) {
  const int i = blockIdx.x, j = threadIdx.x;
  X[i * kCD + j] = i == j ? 1.0 : 0.0;
}

// blocks of 256 threads for one warp per row (no grid-stride loop)
inline int nwarp_blocks(long long rows) { return (int)((rows * 32 + 255) / 256); }

inline int nblk(long long n, int t = 256) {
  long long b = (n + t - 1) / t;
  return (int)(b < 4096 ? (b > 0 ? b : 1) : 4096);
}

constexpr long long kGemmScratch = 1 << 21;  // split-K doubles (16 MiB)
constexpr int kGemmTiles = 512;  // K is split only while a call has < 300 tiles

struct GemmCall {
  cudaStream_t s;
  double* scratch;        // split-K partial sums
  long long scratch_len;  // doubles
  int* tcnt;              // split-K arrival counters, one per output tile (0)
  void operator()(int M, int N, int K, const double* A, long long lda, bool tA,
                  const double* B, long long ldb, bool tB, double* C, long long ldc,
                  double alpha = 1.0, double beta = 0.0, int batch = 1,
                  long long sA = 0, long long sB = 0, long long sC = 0,
                  double diag = 0.0, const int* gate = nullptr, int gate_idx = 0,
                  const double* pass = nullptr) const {
    Gemm g{M, N, K, A, lda, sA, tA ? 1 : 0, B, ldb, sB, tB ? 1 : 0, C, ldc, sC,
           alpha, beta, diag, gate, gate_idx, pass};
    auto ctas = [&](int t) {
      return (long long)((N + t - 1) / t) * ((M + t - 1) / t) * batch;
    };
    const int tile = ctas(64) >= 300 ? 64 : (ctas(32) >= 300 ? 32 : 16);
    // split K when the output alone gives too few CTAs (chunks of >= 64)
    int kc = 1;
    while (kc < 64 && ctas(tile) * kc < 300 && K / (2 * kc) >= 64 &&
           (long long)(2 * kc) * batch * M * N <= scratch_len)
      kc *= 2;
    const dim3 grid((N + tile - 1) / tile, (M + tile - 1) / tile, batch * kc);
    if (tile == 64) gemm_f64_kernel<64><<<grid, 256, 0, s>>>(g, kc, scratch, tcnt);
    else if (tile == 32) gemm_f64_kernel<32><<<grid, 256, 0, s>>>(g, kc, scratch, tcnt);
    else gemm_f64_kernel<16><<<grid, 256, 0, s>>>(g, kc, scratch, tcnt);
  }
};

// One trace: the inputs and what stays fixed over the Adam steps.
struct Trace {
  const double *q, *K, *V;
  const int32_t* tpos;
  int T, nt;
  double *Kc;       // [T][d]     K - mu
  double *Pref;     // [g][nt][T] softmax of the BF16 logits
  double *logPref;  // [g][nt][T] log max(Pref, 1e-300)
  double *Lc;       // [g][nt][T] raw window logits q (K - mu)^T (windows only)
  double *Phat;     // [g][nt][T] key-phase attention, window pairs zeroed
};

struct Calib {
  optr_calib_config c;
  int windows;
  double scale;  // 1 / sqrt(d)
  Trace tr[2];   // calibration, held-out
  // working buffers (sized for the larger trace)
  double *Z, *Zh, *inside, *Kt, *dKt, *dZh;  // [T][d]
  double *L, *PK, *GV;                       // [g][nt][T]
  double *rowv;                              // [g][nt]
  double *DV, *U;                            // [g][nt][d]
  double *E;                                 // [g][nt][d_model]
  // d x d
  double *R0[2], *A, *m, *v, *dA, *S, *Xs, *Hs, *T1[2], *T2[2], *R, *dR, *dE, *best;
  double* scal;  // [0] training loss scratch, [1] score, [2] best score
  int* s_dev;
  unsigned* err;
  const double* W;  // [g][d_model][d]
  double* gsc;      // split-K scratch of the GEMMs
  int* gcnt;        // split-K arrival counters (kGemmTiles, zero between calls)
  cudaStream_t st;
  GemmCall gemm() const { return GemmCall{st, gsc, kGemmScratch, gcnt}; }
};

struct Layout {
  size_t off = 0;
  char* base = nullptr;
  template <typename T>
  T* take(size_t n) {
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += (n * sizeof(T) + 255) & ~(size_t)255;
    return p;
  }
};

// Carves the workspace (base == nullptr: only sizes it).
size_t carve(Calib& C, char* base) {
  const optr_calib_config& c = C.c;
  Layout L;
  L.base = base;
  const int Th = c.T_held > 0 ? c.T_held : c.T, nh = c.T_held > 0 ? c.nt_held : c.nt;
  const long long Tm = c.T > Th ? c.T : Th, nm = c.nt > nh ? c.nt : nh;
  const long long g = c.g, D = kCD, D2 = kCD * kCD;
  C.err = L.take<unsigned>(1);
  C.s_dev = L.take<int>(1);
  C.scal = L.take<double>(8);
  for (int k = 0; k < 2; ++k) {
    const long long T = k ? Th : c.T, nt = k ? nh : c.nt;
    Trace& t = C.tr[k];
    t.Kc = L.take<double>(T * D);
    t.Pref = L.take<double>(g * nt * T);
    t.logPref = L.take<double>(g * nt * T);
    t.Lc = C.windows ? L.take<double>(g * nt * T) : nullptr;
    t.Phat = L.take<double>(g * nt * T);
  }
  C.Z = L.take<double>(Tm * D);
  C.Zh = L.take<double>(Tm * D);
  C.inside = L.take<double>(Tm * D);
  C.Kt = L.take<double>(Tm * D);
  C.dKt = L.take<double>(Tm * D);
  C.dZh = L.take<double>(Tm * D);
  C.L = L.take<double>(g * nm * Tm);
  C.PK = L.take<double>(g * nm * Tm);
  C.GV = L.take<double>(g * nm * Tm);
  C.rowv = L.take<double>(g * nm);
  C.DV = L.take<double>(g * nm * D);
  C.U = L.take<double>(g * nm * D);
  C.E = L.take<double>(g * nm * c.d_model);
  C.gsc = L.take<double>(kGemmScratch);
  C.gcnt = L.take<int>(kGemmTiles);
  double** dd[] = {&C.R0[0], &C.R0[1], &C.A, &C.m, &C.v, &C.dA, &C.S, &C.Xs,
                   &C.Hs, &C.T1[0], &C.T1[1], &C.T2[0], &C.T2[1], &C.R, &C.dR,
                   &C.dE, &C.best};
  for (double** p : dd) *p = L.take<double>(D2);
  return L.off;
}

// E = exp(sign * S) into T1[*], and with H, L = L_exp(sign * S, H) into
// T2[*]; returns the buffer index holding the results.  Taylor series of
// the block matrix [[X, H], [0, X]] in Horner form (T1 <- I + X T1 / k,
// T2 <- (X T2 + H T1) / k), X = sign S 2^-s, H scaled alike, then s
// squarings ([[E, L], [0, E]]^2 = [[E E, E L + L E], [0, E E]]), s decided
// on the device.
int expm(Calib& C, const double* S, double sign, const double* H) {
  GemmCall gm = C.gemm();
  expm_prep_kernel<<<1, kCD, 0, C.st>>>(S, sign, H, C.Xs, C.Hs, C.s_dev, C.err);
  int cur = 0;
  eye_kernel<<<kCD, kCD, 0, C.st>>>(C.T1[0]);
  if (H) fill_kernel<<<nblk(kCD * kCD), 256, 0, C.st>>>(C.T2[0], kCD * kCD, 0.0);
  for (int k = kTaylor; k >= 1; --k) {
    const int nx = cur ^ 1;
    const double a = 1.0 / (double)k;
    gm(kCD, kCD, kCD, C.Xs, kCD, false, C.T1[cur], kCD, false, C.T1[nx], kCD, a, 0.0,
       1, 0, 0, 0, 1.0);
    if (H) {
      gm(kCD, kCD, kCD, C.Xs, kCD, false, C.T2[cur], kCD, false, C.T2[nx], kCD, a, 0.0);
      gm(kCD, kCD, kCD, C.Hs, kCD, false, C.T1[cur], kCD, false, C.T2[nx], kCD, a, 1.0);
    }
    cur = nx;
  }
  for (int i = 0; i < kSquareLaunches; ++i) {
    const int nx = cur ^ 1;
    gm(kCD, kCD, kCD, C.T1[cur], kCD, false, C.T1[cur], kCD, false, C.T1[nx], kCD,
       1.0, 0.0, 1, 0, 0, 0, 0.0, C.s_dev, i, C.T1[cur]);
    if (H) {
      gm(kCD, kCD, kCD, C.T1[cur], kCD, false, C.T2[cur], kCD, false, C.T2[nx], kCD,
         1.0, 0.0, 1, 0, 0, 0, 0.0, C.s_dev, i, C.T2[cur]);
      gm(kCD, kCD, kCD, C.T2[cur], kCD, false, C.T1[cur], kCD, false, C.T2[nx], kCD,
         1.0, 1.0, 1, 0, 0, 0, 0.0, C.s_dev, i, nullptr);
    }
    cur = nx;
  }
  return cur;
}

// R = R0 exp(A - A^T) into C.R (S = A - A^T kept in C.S)
void rotation(Calib& C, const double* R0) {
  skew_kernel<<<kCD, kCD, 0, C.st>>>(C.A, C.S);
  const int e = expm(C, C.S, 1.0, nullptr);
  C.gemm()(kCD, kCD, kCD, R0, kCD, false, C.T1[e], kCD, false, C.R, kCD);
}

// dA = dS - dS^T with dS = L_exp(S^T, R0^T dR) (S^T = -S)
void generator_grad(Calib& C, const double* R0) {
  C.gemm()(kCD, kCD, kCD, R0, kCD, true, C.dR, kCD, false, C.dE, kCD);
  const int e = expm(C, C.S, -1.0, C.dE);
  skew_kernel<<<kCD, kCD, 0, C.st>>>(C.T2[e], C.dA);
}

}  // namespace

namespace {

// Inputs that stay fixed over the steps: K - mu, the BF16 reference
// attention p (and log p), the raw window logits.
void trace_setup(Calib& C, Trace& t, const double* mu) {
  GemmCall gm = C.gemm();
  const int g = C.c.g, D = kCD;
  const long long nT = (long long)t.T * D, r = (long long)g * t.nt;
  center_kernel<<<nblk(nT), 256, 0, C.st>>>(t.K, mu, nT, t.Kc);
  // raw BF16 logits q_j K^T into L, softmax into Pref
  gm(t.nt, t.T, D, t.q, (long long)g * D, false, t.K, D, true, C.L, t.T, 1.0, 0.0,
     g, D, 0, (long long)t.nt * t.T);
  softmax_rows_kernel<<<(unsigned)r, 256, 0, C.st>>>(
      C.L, nullptr, (int)r, t.nt, t.T, t.tpos, C.scale, 0, 0, t.Pref, nullptr,
      nullptr, nullptr);
  logclamp_kernel<<<nblk(r * t.T), 256, 0, C.st>>>(t.Pref, r * t.T, t.logPref);
  if (C.windows)
    gm(t.nt, t.T, D, t.q, (long long)g * D, false, t.Kc, D, true, t.Lc, t.T, 1.0,
       0.0, g, D, 0, (long long)t.nt * t.T);
}

// Effective rotated-and-back rows Q2(X R) R^T into C.Kt (Zh, inside kept).
void q2_roundtrip(Calib& C, const double* X, int T, double clip) {
  GemmCall gm = C.gemm();
  gm(T, kCD, kCD, X, kCD, false, C.R, kCD, false, C.Z, kCD);
  const long long warps = (long long)T * (kCD / C.c.group);
  q2_kernel<<<nwarp_blocks(warps), 256, 0, C.st>>>(C.Z, T, C.c.group, clip, C.Zh, C.inside);
  gm(T, kCD, kCD, C.Zh, kCD, false, C.R, kCD, true, C.Kt, kCD);
}

// L_K of trace t under C.R into *out; leaves PK, E for the backward.
void key_forward(Calib& C, Trace& t, double* out) {
  GemmCall gm = C.gemm();
  const int g = C.c.g, D = kCD, dm = C.c.d_model;
  const long long r = (long long)g * t.nt, nTT = (long long)t.nt * t.T;
  q2_roundtrip(C, t.Kc, t.T, C.c.clip_k);
  gm(t.nt, t.T, D, t.q, (long long)g * D, false, C.Kt, D, true, C.L, t.T, 1.0, 0.0,
     g, D, 0, nTT);
  softmax_rows_kernel<<<(unsigned)r, 256, 0, C.st>>>(
      C.L, C.windows ? t.Lc : nullptr, (int)r, t.nt, t.T, t.tpos, C.scale,
      C.c.sink, C.c.recent, C.PK, t.Pref, t.logPref, C.rowv);
  // e_j = ((pk - p) V) W_j^T
  sub_kernel<<<nblk(r * t.T), 256, 0, C.st>>>(C.PK, t.Pref, r * t.T, C.GV);
  gm(t.nt, D, t.T, C.GV, t.T, false, t.V, D, false, C.DV, D, 1.0, 0.0, g, nTT, 0,
     (long long)t.nt * D);
  gm(t.nt, dm, D, C.DV, D, false, C.W, D, true, C.E, dm, 1.0, 0.0, g,
     (long long)t.nt * D, (long long)dm * D, (long long)t.nt * dm);
  row_sqsum_kernel<<<nwarp_blocks(r), 256, 0, C.st>>>(C.E, (int)r, dm, C.c.lam, 1, C.rowv);
  loss_reduce_kernel<<<1, 1024, 0, C.st>>>(C.rowv, (int)r, (double)r, out);
}

}  // namespace

namespace {

// dR of L_K (after key_forward on the same trace and rotation).
void key_backward(Calib& C, Trace& t) {
  GemmCall gm = C.gemm();
  const int g = C.c.g, D = kCD, dm = C.c.d_model;
  const long long r = (long long)g * t.nt, nTT = (long long)t.nt * t.T;
  // U_j = (2 lambda / d_model) e_j W_j;  GV_j = U_j V^T
  gm(t.nt, D, dm, C.E, dm, false, C.W, D, false, C.U, D, 2.0 * C.c.lam / dm, 0.0, g,
     (long long)t.nt * dm, (long long)dm * D, (long long)t.nt * D);
  gm(t.nt, t.T, D, C.U, D, false, t.V, D, true, C.GV, t.T, 1.0, 0.0, g,
     (long long)t.nt * D, 0, nTT);
  key_row_grad_kernel<<<nwarp_blocks(r), 256, 0, C.st>>>(
      C.PK, t.Pref, C.GV, (int)r, t.nt, t.T, t.tpos, C.scale / (double)r, C.c.sink,
      C.c.recent, C.windows);
  // dKt = sum_j dl_j^T q_j
  for (int j = 0; j < g; ++j)
    gm(t.T, D, t.nt, C.GV + j * nTT, t.T, true, t.q + j * D, (long long)g * D, false,
       C.dKt, D, 1.0, j ? 1.0 : 0.0);
  // dR = dKt^T Zh + Kc^T (inside * (dKt R))
  gm(t.T, D, D, C.dKt, D, false, C.R, D, false, C.dZh, D);
  gm(D, D, t.T, C.dKt, D, true, C.Zh, D, false, C.dR, D);
  mask_mul_kernel<<<nblk((long long)t.T * D), 256, 0, C.st>>>(C.dZh, C.inside,
                                                             (long long)t.T * D);
  gm(D, D, t.T, t.Kc, D, true, C.dZh, D, false, C.dR, D, 1.0, 1.0);
}

// Phat of trace t: the key-phase attention under C.R (the selected R_K),
// window pairs zeroed (their values are exact, so they add no error).
void value_setup(Calib& C, Trace& t) {
  key_forward(C, t, C.scal + 3);
  const long long r = (long long)C.c.g * t.nt;
  copy_kernel<<<nblk(r * t.T), 256, 0, C.st>>>(C.PK, r * t.T, t.Phat);
  if (C.windows)
    zero_window_kernel<<<nwarp_blocks(r), 256, 0, C.st>>>(t.Phat, (int)r, t.nt, t.T,
                                                        t.tpos, C.c.sink, C.c.recent);
}

// L_V of trace t under C.R (the value rotation) into *out.
void value_forward(Calib& C, Trace& t, double* out) {
  GemmCall gm = C.gemm();
  const int g = C.c.g, D = kCD, dm = C.c.d_model;
  const long long r = (long long)g * t.nt, nTT = (long long)t.nt * t.T;
  q2_roundtrip(C, t.V, t.T, C.c.clip_v);
  sub_kernel<<<nblk((long long)t.T * D), 256, 0, C.st>>>(C.Kt, t.V, (long long)t.T * D,
                                                        C.Kt);
  gm(t.nt, D, t.T, t.Phat, t.T, false, C.Kt, D, false, C.DV, D, 1.0, 0.0, g, nTT, 0,
     (long long)t.nt * D);
  gm(t.nt, dm, D, C.DV, D, false, C.W, D, true, C.E, dm, 1.0, 0.0, g,
     (long long)t.nt * D, (long long)dm * D, (long long)t.nt * dm);
  row_sqsum_kernel<<<nwarp_blocks(r), 256, 0, C.st>>>(C.E, (int)r, dm, 1.0, 0, C.rowv);
  loss_reduce_kernel<<<1, 1024, 0, C.st>>>(C.rowv, (int)r, (double)r, out);
}

// dR of L_V (after value_forward on the same trace and rotation).
void value_backward(Calib& C, Trace& t) {
  GemmCall gm = C.gemm();
  const int g = C.c.g, D = kCD, dm = C.c.d_model;
  const long long r = (long long)g * t.nt, nTT = (long long)t.nt * t.T;
  gm(t.nt, D, dm, C.E, dm, false, C.W, D, false, C.U, D, 2.0 / ((double)dm * r), 0.0,
     g, (long long)t.nt * dm, (long long)dm * D, (long long)t.nt * D);
  for (int j = 0; j < g; ++j)
    gm(t.T, D, t.nt, t.Phat + j * nTT, t.T, true, C.U + (long long)j * t.nt * D, D,
       false, C.dKt, D, 1.0, j ? 1.0 : 0.0);
  gm(t.T, D, D, C.dKt, D, false, C.R, D, false, C.dZh, D);
  gm(D, D, t.T, C.dKt, D, true, C.Zh, D, false, C.dR, D);
  mask_mul_kernel<<<nblk((long long)t.T * D), 256, 0, C.st>>>(C.dZh, C.inside,
                                                             (long long)t.T * D);
  gm(D, D, t.T, t.V, D, true, C.dZh, D, false, C.dR, D, 1.0, 1.0);
}

// One Adam run of the appendix algorithm on generator A (from 0) for the
// key (kind 0) or value (kind 1) objective; the best-scoring rotation on
// the held-out trace (scored at step 0, every select_every steps and after
// the last step) ends in C.best; hist[i] = the training loss at step i.
void adam_run(Calib& C, int kind, const double* R0, double* hist) {
  const optr_calib_config& c = C.c;
  const int n = kCD * kCD;
  fill_kernel<<<nblk(n), 256, 0, C.st>>>(C.A, n, 0.0);
  fill_kernel<<<nblk(n), 256, 0, C.st>>>(C.m, n, 0.0);
  fill_kernel<<<nblk(n), 256, 0, C.st>>>(C.v, n, 0.0);
  const double b1 = 0.9, b2 = 0.999, eps = 1e-8;
  for (int i = 0; i <= c.steps; ++i) {
    rotation(C, R0);
    if (i % c.select_every == 0 || i == c.steps) {
      if (kind == 0) key_forward(C, C.tr[1], C.scal + 1);
      else value_forward(C, C.tr[1], C.scal + 1);
      select_kernel<<<1, 256, 0, C.st>>>(C.scal + 1, C.scal + 2, i == 0, C.R, C.best);
    }
    if (i == c.steps) break;
    if (kind == 0) {
      key_forward(C, C.tr[0], hist + i);
      key_backward(C, C.tr[0]);
    } else {
      value_forward(C, C.tr[0], hist + i);
      value_backward(C, C.tr[0]);
    }
    generator_grad(C, R0);
    const int t = i + 1;
    adam_kernel<<<nblk(n), 256, 0, C.st>>>(C.A, C.dA, C.m, C.v, n, c.lr, b1, 1.0 - b1,
                                           b2, 1.0 - b2, 1.0 - pow(b1, (double)t),
                                           1.0 - pow(b2, (double)t), eps);
  }
}

}  // namespace

namespace {

bool calib_config_ok(const optr_calib_config* c) {
  if (!c) return false;
  const bool held = c->T_held > 0;
  // tokens and query rows: GEMM grids stay within 65535 row tiles
  const double lim = 4000000.0;
  return c->g >= 1 && c->g <= 64 && c->d_model >= 1 && c->d_model <= (1 << 20) &&
         c->T >= 1 && c->T <= lim && c->nt >= 1 &&
         (double)c->g * c->nt <= lim && c->T_held >= 0 &&
         (!held || (c->nt_held >= 1 && c->T_held <= lim &&
                    (double)c->g * c->nt_held <= lim)) &&
         c->steps >= 0 && c->steps <= 100000 && c->select_every >= 1 &&
         (c->group == 32 || c->group == 128) && c->sink >= 0 && c->recent >= 0 &&
         c->clip_k > 0.0 && c->clip_k <= 1.0 && c->clip_v > 0.0 && c->clip_v <= 1.0 &&
         c->lr > 0.0 && c->lr < 1e6 && c->lam >= 0.0 && c->lam < 1e12;
}

void calib_init(Calib& C, const optr_calib_config* c, void* ws, const double* W_O,
                cudaStream_t s) {
  C = Calib{};
  C.c = *c;
  C.windows = c->sink > 0 || c->recent > 0;
  C.scale = 1.0 / sqrt((double)kCD);
  carve(C, static_cast<char*>(ws));
  C.W = W_O;
  C.st = s;
}

optr_status calib_finish(Calib& C) {
  if (cudaGetLastError() != cudaSuccess) return OPTR_ERR_CUDA;
  unsigned e = 0;
  if (cudaMemcpyAsync(&e, C.err, sizeof(unsigned), cudaMemcpyDeviceToHost, C.st) !=
          cudaSuccess ||
      cudaStreamSynchronize(C.st) != cudaSuccess)
    return OPTR_ERR_CUDA;
  return e ? OPTR_ERR_OUT_OF_RANGE : OPTR_OK;
}

}  // namespace
}  // namespace optr

using namespace optr;

extern "C" size_t optr_calib_workspace_size(const optr_calib_config* c) {
  if (!calib_config_ok(c)) return 0;
  Calib C{};
  C.c = *c;
  C.windows = c->sink > 0 || c->recent > 0;
  return carve(C, nullptr);
}

extern "C" optr_status optr_calibrate_head(
    const optr_calib_config* c, const double* q, const double* K, const double* V,
    const int32_t* t_pos, const double* W_O, const double* q_held,
    const double* K_held, const double* V_held, const int32_t* t_pos_held,
    const double* R0_K, const double* R0_V, double* R_K, double* R_V, double* mu,
    double* hist_k, double* hist_v, void* workspace, size_t ws_bytes,
    cudaStream_t stream) {
  if (!calib_config_ok(c)) return OPTR_ERR_INVALID_ARG;
  if (!q || !K || !V || !t_pos || !W_O || !R_K || !R_V || !mu) return OPTR_ERR_INVALID_ARG;
  if (c->steps > 0 && (!hist_k || !hist_v)) return OPTR_ERR_INVALID_ARG;
  const bool held = c->T_held > 0;
  if (held && (!q_held || !K_held || !V_held || !t_pos_held)) return OPTR_ERR_INVALID_ARG;
  const size_t need = optr_calib_workspace_size(c);
  if (!workspace || ws_bytes < need || (reinterpret_cast<uintptr_t>(workspace) & 255))
    return OPTR_ERR_WORKSPACE;
  Calib C;
  calib_init(C, c, workspace, W_O, stream);
  const int n = kCD * kCD;
  if (cudaMemsetAsync(C.err, 0, sizeof(unsigned), stream) != cudaSuccess ||
      cudaMemsetAsync(C.gcnt, 0, sizeof(int) * kGemmTiles, stream) != cudaSuccess)
    return OPTR_ERR_CUDA;
  col_mean_kernel<<<1, kCD, 0, stream>>>(K, c->T, mu);
  const double* r0[2] = {R0_K, R0_V};
  for (int k = 0; k < 2; ++k) {
    if (r0[k]) copy_kernel<<<nblk(n), 256, 0, stream>>>(r0[k], n, C.R0[k]);
    else hadamard_kernel<<<kCD, kCD, 0, stream>>>(C.R0[k]);
  }
  C.tr[0].q = q; C.tr[0].K = K; C.tr[0].V = V; C.tr[0].tpos = t_pos;
  C.tr[0].T = c->T; C.tr[0].nt = c->nt;
  trace_setup(C, C.tr[0], mu);
  if (held) {
    C.tr[1].q = q_held; C.tr[1].K = K_held; C.tr[1].V = V_held;
    C.tr[1].tpos = t_pos_held; C.tr[1].T = c->T_held; C.tr[1].nt = c->nt_held;
    trace_setup(C, C.tr[1], mu);
  } else {
    C.tr[1] = C.tr[0];
  }
  adam_run(C, 0, C.R0[0], hist_k);
  copy_kernel<<<nblk(n), 256, 0, stream>>>(C.best, n, R_K);
  copy_kernel<<<nblk(n), 256, 0, stream>>>(C.best, n, C.R);
  value_setup(C, C.tr[0]);
  if (held) value_setup(C, C.tr[1]);
  adam_run(C, 1, C.R0[1], hist_v);
  copy_kernel<<<nblk(n), 256, 0, stream>>>(C.best, n, R_V);
  return calib_finish(C);
}

extern "C" optr_status optr_calib_loss_grad(
    const optr_calib_config* c, int which, const double* q, const double* K,
    const double* V, const int32_t* t_pos, const double* W_O, const double* mu,
    const double* R_K, const double* R0, const double* A, double* loss, double* dA,
    void* workspace, size_t ws_bytes, cudaStream_t stream) {
  if (!calib_config_ok(c) || (which != 0 && which != 1)) return OPTR_ERR_INVALID_ARG;
  if (!q || !K || !V || !t_pos || !W_O || !mu || !R0 || !A || !loss)
    return OPTR_ERR_INVALID_ARG;
  if (which == 1 && !R_K) return OPTR_ERR_INVALID_ARG;
  const size_t need = optr_calib_workspace_size(c);
  if (!workspace || ws_bytes < need || (reinterpret_cast<uintptr_t>(workspace) & 255))
    return OPTR_ERR_WORKSPACE;
  Calib C;
  calib_init(C, c, workspace, W_O, stream);
  const int n = kCD * kCD;
  if (cudaMemsetAsync(C.err, 0, sizeof(unsigned), stream) != cudaSuccess ||
      cudaMemsetAsync(C.gcnt, 0, sizeof(int) * kGemmTiles, stream) != cudaSuccess)
    return OPTR_ERR_CUDA;
  C.tr[0].q = q; C.tr[0].K = K; C.tr[0].V = V; C.tr[0].tpos = t_pos;
  C.tr[0].T = c->T; C.tr[0].nt = c->nt;
  trace_setup(C, C.tr[0], mu);
  if (which == 1) {
    copy_kernel<<<nblk(n), 256, 0, stream>>>(R_K, n, C.R);
    value_setup(C, C.tr[0]);
  }
  copy_kernel<<<nblk(n), 256, 0, stream>>>(A, n, C.A);
  rotation(C, R0);
  if (which == 0) key_forward(C, C.tr[0], loss);
  else value_forward(C, C.tr[0], loss);
  if (dA) {
    if (which == 0) key_backward(C, C.tr[0]);
    else value_backward(C, C.tr[0]);
    generator_grad(C, R0);
    copy_kernel<<<nblk(n), 256, 0, stream>>>(C.dA, n, dA);
  }
  return calib_finish(C);
}
