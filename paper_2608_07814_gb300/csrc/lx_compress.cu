// Compression of one member projection (Sec. 3.2 Stage 3 (ii)): the residual
// R = W_mem - W_dom ([rows][cols], Eq. svd), its rank-r randomized SVD (range
// finder with power iterations, Halko-Martinsson-Tropp, with the Gaussian test
// matrix given by the caller) and the symmetric split of Eq. factors,
// U = U_r S_r^(1/2) [rows][r], V = V_r S_r^(1/2) [cols][r].
//
// Kernels:
//   k_cgemm     fp32 GEMM (CUDA-core FMA, 64 x 64 tiles, 32-deep K chunks in
//               shared memory); its A operand is R (rows of W_mem - W_dom,
//               formed on load), R^T (columns of the same), or an fp32 matrix.
//   k_gram      G = X^T X in float64 (fp32 inputs, float64 products and sums).
//   k_chol32    one CTA: Cholesky G + s I = L L^T (fp32 in shared memory; a
//               small relative shift in the first of the two passes keeps
//               rank-deficient bases factorable) and T = L^-T, so that X T has
//               orthonormal columns (CholeskyQR, run twice per
//               orthonormalisation).
//   k_trmm      M = L1 L2, the triangular factor of R^T Q = Z2 M^T.
//   k_onesided  one CTA: one-sided Jacobi SVD of M (fp32 rotations, shared
//               memory), M W = U S.
//   k_ritz      sigma_j = |M w_j| / |w_j| in float64 (Rayleigh quotients).
//   k_finish    the r largest sigma and the fp32 matrices that turn the bases
//               into the split factors.
//   k_sign      each factor column's largest-magnitude entry of U made
//               positive (U and V negated together).
// Only the Gram sums and the Rayleigh quotients use float64: a single SM's
// float64 rate is a small fraction of its fp32 rate on this GPU.
#include <algorithm>
#include <cmath>
#include <type_traits>

#include "lx_internal.cuh"

namespace lx {
namespace {

constexpr int CG_TILE = 64;
constexpr int CG_KC = 32;
constexpr int CG_LD = CG_TILE + 4;
constexpr int CG_THREADS = 256;

enum { A_RES = 0, A_RES_T = 1, A_F32 = 2 };

__device__ __forceinline__ void cload8(const __nv_bfloat16* p, float (&v)[8]) {
  const uint4 q = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&q);
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float2 f = __bfloat1622float2(h[e]);
    v[2 * e] = f.x;
    v[2 * e + 1] = f.y;
  }
}
__device__ __forceinline__ void cload8(const float* p, float (&v)[8]) {
  const float4 a = *reinterpret_cast<const float4*>(p);
  const float4 b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

// C [M][N] = A [M][K] * B [K][N] (fp32, row-major).  A element (m, k):
//   A_RES:   Wm[m * ldw + k] - Wd[m * ldw + k]   (R itself; M = rows, K = cols = ldw)
//   A_RES_T: Wm[k * ldw + m] - Wd[k * ldw + m]   (R^T; M = cols = ldw, K = rows)
//   A_F32:   X[m * K + k]
// A_RES / A_RES_T need ldw % 8 == 0 and 16-byte aligned weights (8-element
// vector loads); A_F32 and B take scalar loads (any K, N).
template <typename TW, int MODE>
__global__ void __launch_bounds__(CG_THREADS)
k_cgemm(const TW* __restrict__ Wm, const TW* __restrict__ Wd, const float* __restrict__ X,
        int ldw, const float* __restrict__ B, float* __restrict__ C, int M, int N, int K) {
  __shared__ __align__(16) float As[CG_KC][CG_LD];
  __shared__ __align__(16) float Bs[CG_KC][CG_LD];
  const int tid = threadIdx.x;
  const int m0 = blockIdx.y * CG_TILE, n0 = blockIdx.x * CG_TILE;
  const int ty = tid >> 4, tx = tid & 15;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += CG_KC) {
    const int kc = min(CG_KC, K - k0);
    if (MODE == A_RES) {
      const int row = tid >> 2, kq = (tid & 3) * 8;
      const bool ok = m0 + row < M && kq < kc;  // kc is a multiple of 8 here
      float a[8], d[8];
      if (ok) {
        cload8(Wm + (size_t)(m0 + row) * ldw + k0 + kq, a);
        cload8(Wd + (size_t)(m0 + row) * ldw + k0 + kq, d);
      }
#pragma unroll
      for (int e = 0; e < 8; ++e) As[kq + e][row] = ok ? a[e] - d[e] : 0.f;
    } else if (MODE == A_RES_T) {
      const int kr = tid >> 3, mq = (tid & 7) * 8;
      const bool ok = kr < kc && m0 + mq < M;
      float a[8], d[8];
      if (ok) {
        cload8(Wm + (size_t)(k0 + kr) * ldw + m0 + mq, a);
        cload8(Wd + (size_t)(k0 + kr) * ldw + m0 + mq, d);
      }
#pragma unroll
      for (int e = 0; e < 8; ++e) As[kr][mq + e] = ok ? a[e] - d[e] : 0.f;
    } else {
      const int row = tid >> 2, kq = (tid & 3) * 8;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const bool ok = m0 + row < M && kq + e < kc;
        As[kq + e][row] = ok ? X[(size_t)(m0 + row) * K + k0 + kq + e] : 0.f;
      }
    }
    {
      const int kr = tid >> 3, nq = (tid & 7) * 8;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const bool ok = kr < kc && n0 + nq + e < N;
        Bs[kr][nq + e] = ok ? B[(size_t)(k0 + kr) * N + n0 + nq + e] : 0.f;
      }
    }
    __syncthreads();
#pragma unroll 8
    for (int k = 0; k < CG_KC; ++k) {
      const float4 a = *reinterpret_cast<const float4*>(&As[k][ty * 4]);
      const float4 b = *reinterpret_cast<const float4*>(&Bs[k][tx * 4]);
      const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
      for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(av[r], bv[c], acc[r][c]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int m = m0 + ty * 4 + r;
    if (m >= M) continue;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int n = n0 + tx * 4 + c;
      if (n < N) C[(size_t)m * N + n] = acc[r][c];
    }
  }
}

// G [L][L] = X^T X for X [n][L] fp32 row-major; float64 products and sums in
// ascending row order.  16 x 16 outputs per CTA; only the tiles on or below
// the diagonal are computed (the Cholesky reads the lower triangle alone).
constexpr int GR_T = 16;
constexpr int GR_KC = 32;
__global__ void __launch_bounds__(GR_T * GR_T)
k_gram(const float* __restrict__ X, int n, int L, double* __restrict__ G) {
  __shared__ double Xi[GR_KC][GR_T], Xj[GR_KC][GR_T];
  if (blockIdx.x > blockIdx.y) return;  // strictly above the diagonal
  const int ti = threadIdx.x / GR_T, tj = threadIdx.x % GR_T;
  const int i0 = blockIdx.y * GR_T, j0 = blockIdx.x * GR_T;
  double acc = 0.0;
  for (int m0 = 0; m0 < n; m0 += GR_KC) {
    for (int q = threadIdx.x; q < GR_KC * GR_T; q += GR_T * GR_T) {
      const int mr = q / GR_T, c = q % GR_T;
      const bool okm = m0 + mr < n;
      Xi[mr][c] = (okm && i0 + c < L) ? (double)X[(size_t)(m0 + mr) * L + i0 + c] : 0.0;
      Xj[mr][c] = (okm && j0 + c < L) ? (double)X[(size_t)(m0 + mr) * L + j0 + c] : 0.0;
    }
    __syncthreads();
#pragma unroll 8
    for (int mr = 0; mr < GR_KC; ++mr) acc = fma(Xi[mr][ti], Xj[mr][tj], acc);
    __syncthreads();
  }
  if (i0 + ti < L && j0 + tj < L) G[(size_t)(i0 + ti) * L + j0 + tj] = acc;
}

// One CTA (L <= 256).  Cholesky of G + s I in fp32 (G float64, rounded once;
// s = shift_rel * max diag(G)) in a packed lower triangle in shared memory
// (L (L + 1) / 2 floats), pivots floored at 1e-30; then X = L^-1 by forward
// substitution (thread c owns column c; X packed like L, in shared memory
// when x_in_smem, else in the global scratch Xg, so that a warp reads one
// contiguous piece of a row per step) and T = X^T, so that Y T = Y L^-T has
// orthonormal columns when Y^T Y = G (CholeskyQR).  The factor itself is
// written to Lout [L][L] (zero above the diagonal).  A zero Gram gives
// Lout = T = 0.
constexpr int CH_THREADS = 1024;
__global__ void __launch_bounds__(CH_THREADS)
k_chol32(const double* __restrict__ G, int L, float shift_rel, float* __restrict__ Lout,
         float* __restrict__ Xg, int x_in_smem, float* __restrict__ T) {
  extern __shared__ float Ls[];
  float* Xp = x_in_smem ? Ls + L * (L + 1) / 2 : Xg;  // packed lower X
  __shared__ double s_md;
  __shared__ float s_diag[256];  // the factor's diagonal (Ls keeps the raw pivots)
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = CH_THREADS / 32;
  if (tid == 0) {
    double md = 0.0;
    for (int i = 0; i < L; ++i) md = fmax(md, G[(size_t)i * L + i]);
    s_md = md;
  }
  __syncthreads();
  const double md = s_md;
  if (!(md > 0.0)) {
    for (int q = tid; q < L * L; q += CH_THREADS) {
      Lout[q] = 0.f;
      T[q] = 0.f;
    }
    return;
  }
  const float shift = (float)(shift_rel * md);
  for (int i = warp; i < L; i += nw)
    for (int j = lane; j <= i; j += 32)
      Ls[i * (i + 1) / 2 + j] = (float)G[(size_t)i * L + j] + (i == j ? shift : 0.f);
  __syncthreads();
  for (int j = 0; j < L; ++j) {
    // every thread takes the pivot from the raw entry, which nothing writes
    // after the previous step's barrier; the factor's diagonal goes to s_diag
    const float ljj = sqrtf(fmaxf(Ls[j * (j + 1) / 2 + j], 1e-30f));
    if (tid == 0) s_diag[j] = ljj;
    for (int i = j + 1 + tid; i < L; i += CH_THREADS) Ls[i * (i + 1) / 2 + j] /= ljj;
    __syncthreads();
    for (int i = j + 1 + warp; i < L; i += nw) {
      const float lij = Ls[i * (i + 1) / 2 + j];
      for (int c = j + 1 + lane; c <= i; c += 32) Ls[i * (i + 1) / 2 + c] -= lij * Ls[c * (c + 1) / 2 + j];
    }
    __syncthreads();
  }
  for (int j = tid; j < L; j += CH_THREADS) Ls[j * (j + 1) / 2 + j] = s_diag[j];
  __syncthreads();
  for (int q = tid; q < L * L; q += CH_THREADS) {
    const int i = q / L, c = q % L;
    Lout[q] = c <= i ? Ls[i * (i + 1) / 2 + c] : 0.f;
  }
  if (tid < L) {
    const int c = tid;
    for (int i = c; i < L; ++i) {
      const float* Li = Ls + i * (i + 1) / 2;
      float acc = 0.f;
      for (int k = c; k < i; ++k) acc = fmaf(Li[k], Xp[k * (k + 1) / 2 + c], acc);
      Xp[i * (i + 1) / 2 + c] = i == c ? 1.f / Li[i] : -acc / Li[i];
    }
  }
  __syncthreads();
  for (int q = tid; q < L * L; q += CH_THREADS) {
    const int k = q / L, n = q % L;  // T[k][n] = X[n][k], zero below the diagonal
    T[q] = k <= n ? Xp[n * (n + 1) / 2 + k] : 0.f;
  }
}

// Mt (column-major, Mt[j][i] = M[i][j]) of M = L1 L2 for lower-triangular
// L1, L2 [L][L] (fp32, float64 sums).  CTA i, thread j.
__global__ void k_trmm(const float* __restrict__ L1, const float* __restrict__ L2, int L,
                       float* __restrict__ Mt) {
  const int i = blockIdx.x, j = threadIdx.x;
  if (j >= L) return;
  double acc = 0.0;
  for (int k = j; k <= i; ++k) acc = fma((double)L1[(size_t)i * L + k], (double)L2[(size_t)k * L + j], acc);
  Mt[(size_t)j * L + i] = (float)acc;
}

// One-sided Jacobi SVD of M (Hestenes), one CTA: the columns of M are
// orthogonalised by plane rotations applied from the right, M W = U S, W
// orthogonal.  Lp = L rounded up to even (a zero padding column never rotates);
// each round pairs the columns by the circle method, a warp takes a pair:
// alpha = |m_p|^2, beta = |m_q|^2, gamma = m_p . m_q (fp32), and unless
// |gamma| <= 1e-6 sqrt(alpha beta) (a little above the rounding of an fp32 dot
// product, so that sweeps terminate) rotates columns p, q of M and of W by the
// angle that makes them orthogonal (zeta = (beta - alpha) / (2 gamma),
// t = sign(zeta) / (|zeta| + sqrt(1 + zeta^2)), c = 1 / sqrt(1 + t^2), s = c t).  Sweeps end when one makes no rotation, or after OS_MAX_SWEEPS.
// M and W are column-major, in shared memory when they fit, else in Mg / Wg.
// Output: Wt [L][L], Wt[j][k] = W[k][j].
constexpr int OS_THREADS = 1024;
constexpr int OS_MAX_SWEEPS = 30;
__global__ void __launch_bounds__(OS_THREADS)
k_onesided(const float* __restrict__ Mt, int L, float* __restrict__ Mg, float* __restrict__ Wg,
           int in_smem, float* __restrict__ Wt) {
  extern __shared__ float osm[];
  __shared__ int s_rot;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = OS_THREADS / 32;
  const int Lp = L + (L & 1), half = Lp / 2;
  float* M = in_smem ? osm : Mg;                       // [Lp][L]
  float* W = in_smem ? osm + (size_t)Lp * L : Wg;      // [Lp][Lp]
  for (int q = tid; q < Lp * L; q += OS_THREADS) M[q] = q < L * L ? Mt[q] : 0.f;
  for (int q = tid; q < Lp * Lp; q += OS_THREADS) W[q] = (q / Lp == q % Lp) ? 1.f : 0.f;
  __syncthreads();
  for (int sweep = 0; sweep < OS_MAX_SWEEPS; ++sweep) {
    if (tid == 0) s_rot = 0;
    __syncthreads();
    for (int round = 0; round < Lp - 1; ++round) {
      for (int P = warp; P < half; P += nw) {
        int p, q;
        if (P == 0) {
          p = round;
          q = Lp - 1;
        } else {
          p = round + P;
          if (p >= Lp - 1) p -= Lp - 1;
          q = round - P;
          if (q < 0) q += Lp - 1;
        }
        float* mp = M + (size_t)p * L;
        float* mq = M + (size_t)q * L;
        float a = 0.f, b = 0.f, g = 0.f;
        for (int i = lane; i < L; i += 32) {
          const float x = mp[i], y = mq[i];
          a = fmaf(x, x, a);
          b = fmaf(y, y, b);
          g = fmaf(x, y, g);
        }
        for (int o = 16; o; o >>= 1) {
          a += __shfl_xor_sync(0xffffffffu, a, o);
          b += __shfl_xor_sync(0xffffffffu, b, o);
          g += __shfl_xor_sync(0xffffffffu, g, o);
        }
        if (g == 0.f || fabsf(g) <= 1e-6f * sqrtf(a * b)) continue;  // warp-uniform
        // (an overflowing zeta gives t = 0: no rotation, never a NaN)
        const float z = (b - a) / (2.f * g);
        const float t = (z >= 0.f ? 1.f : -1.f) / (fabsf(z) + sqrtf(1.f + z * z));
        const float c = 1.f / sqrtf(1.f + t * t), s = t * c;
        float* wp = W + (size_t)p * Lp;
        float* wq = W + (size_t)q * Lp;
        for (int i = lane; i < Lp; i += 32) {  // Lp >= L: one loop for M and W
          if (i < L) {
            const float x = mp[i], y = mq[i];
            mp[i] = c * x - s * y;
            mq[i] = s * x + c * y;
          }
          const float x = wp[i], y = wq[i];
          wp[i] = c * x - s * y;
          wq[i] = s * x + c * y;
        }
        if (lane == 0) s_rot = 1;
      }
      __syncthreads();
    }
    if (s_rot == 0) break;  // read after the round's barrier; every thread sees the same value
    __syncthreads();        // before thread 0 clears s_rot for the next sweep
  }
  for (int q = tid; q < L * L; q += OS_THREADS) {
    const int j = q / L, k = q % L;
    Wt[q] = W[(size_t)j * Lp + k];
  }
}

// CTA j: v = M w_j in float64, sigma_j = |v| / |w_j| (the Rayleigh quotient of
// the converged rotation, second-order accurate in the rotation's error);
// MWn[j] = v / |w_j|, Wn[j] = w_j / |w_j| (fp32, column j stored contiguously).
__global__ void __launch_bounds__(256)
k_ritz(const float* __restrict__ Mt, const float* __restrict__ Wt, int L, float* __restrict__ MWn,
       float* __restrict__ Wn, double* __restrict__ sig64) {
  __shared__ float w[256];
  __shared__ double red[2][8];
  const int j = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int k = tid; k < L; k += 256) w[k] = Wt[(size_t)j * L + k];
  __syncthreads();
  double v = 0.0, ww = 0.0;
  if (tid < L) {
    for (int k = 0; k < L; ++k) v = fma((double)Mt[(size_t)k * L + tid], (double)w[k], v);
    ww = (double)w[tid] * (double)w[tid];
  }
  double v2 = v * v, w2 = ww;
  for (int o = 16; o; o >>= 1) {
    v2 += __shfl_xor_sync(0xffffffffu, v2, o);
    w2 += __shfl_xor_sync(0xffffffffu, w2, o);
  }
  if (lane == 0) {
    red[0][warp] = v2;
    red[1][warp] = w2;
  }
  __syncthreads();
  double tv = 0.0, tw = 0.0;
  for (int q = 0; q < 8; ++q) {
    tv += red[0][q];
    tw += red[1][q];
  }
  const double nw_ = sqrt(tw);
  if (tid < L) {
    MWn[(size_t)j * L + tid] = nw_ > 0.0 ? (float)(v / nw_) : 0.f;
    Wn[(size_t)j * L + tid] = nw_ > 0.0 ? (float)((double)w[tid] / nw_) : 0.f;
  }
  if (tid == 0) sig64[j] = nw_ > 0.0 ? sqrt(tv) / nw_ : 0.0;
}

// One CTA: the r largest sigma (ties: lower index first) and the fp32
// matrices Wu [L][r] = MWn[i_c] / sqrt(sigma_c), Wv [L][r] = Wn[i_c] sqrt(sigma_c)
// (zero for sigma_c <= 1e-6 sigma_0), so that Q Wu = U_r S_r^(1/2) and
// Z2 Wv = V_r S_r^(1/2) (Eq. factors); sig [r] fp32.
__global__ void __launch_bounds__(256)
k_finish(const double* __restrict__ sig64, const float* __restrict__ MWn,
         const float* __restrict__ Wn, int L, int r, float* __restrict__ Wu,
         float* __restrict__ Wv, float* __restrict__ sig) {
  __shared__ int order[256];
  const int tid = threadIdx.x;
  for (int i = tid; i < L; i += 256) {
    const double si = sig64[i];
    int rk = 0;
    for (int j = 0; j < L; ++j) {
      const double sj = sig64[j];
      rk += (sj > si || (sj == si && j < i)) ? 1 : 0;
    }
    order[rk] = i;
  }
  __syncthreads();
  const double s0 = sig64[order[0]];
  for (int q = tid; q < L * r; q += 256) {
    const int k = q / r, c = q % r;
    const int i = order[c];
    const double sg = sig64[i];
    const bool keep = sg > 1e-6 * s0 && sg > 0.0;
    const float rs = (float)sqrt(sg);
    Wu[q] = keep ? MWn[(size_t)i * L + k] / rs : 0.f;
    Wv[q] = keep ? Wn[(size_t)i * L + k] * rs : 0.f;
    if (k == 0) sig[c] = (float)sg;
  }
}

// Column c of U [rows][r]: the entry of largest magnitude (lowest row on
// ties) is made positive by negating U[:, c] and V[:, c] together.
__global__ void k_sign(float* __restrict__ U, float* __restrict__ V, int rows, int cols, int r) {
  __shared__ float bv[32];
  __shared__ int bi[32];
  __shared__ float s_sign;
  const int c = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  float best = -1.f;
  int bidx = 0x7fffffff;
  for (int m = tid; m < rows; m += blockDim.x) {
    const float a = fabsf(U[(size_t)m * r + c]);
    if (a > best || (a == best && m < bidx)) {
      best = a;
      bidx = m;
    }
  }
  for (int o = 16; o; o >>= 1) {
    const float ob = __shfl_xor_sync(0xffffffffu, best, o);
    const int oi = __shfl_xor_sync(0xffffffffu, bidx, o);
    if (ob > best || (ob == best && oi < bidx)) {
      best = ob;
      bidx = oi;
    }
  }
  if (lane == 0) {
    bv[warp] = best;
    bi[warp] = bidx;
  }
  __syncthreads();
  if (tid == 0) {
    float b = -1.f;
    int i = 0x7fffffff;
    for (int w = 0; w < (int)(blockDim.x / 32); ++w)
      if (bv[w] > b || (bv[w] == b && bi[w] < i)) {
        b = bv[w];
        i = bi[w];
      }
    s_sign = (i < rows && U[(size_t)i * r + c] < 0.f) ? -1.f : 1.f;
  }
  __syncthreads();
  if (s_sign < 0.f) {
    for (int m = tid; m < rows; m += blockDim.x) U[(size_t)m * r + c] = -U[(size_t)m * r + c];
    for (int m = tid; m < cols; m += blockDim.x) V[(size_t)m * r + c] = -V[(size_t)m * r + c];
  }
}

bool g_ch_cap[64] = {};
bool g_os_cap[64] = {};

}  // namespace
}  // namespace lx

namespace lx {
namespace {
constexpr int CP_MAX_L = 256;
constexpr size_t CP_SMEM_CAP = 200 * 1024;

size_t al256(size_t v) { return (v + 255) / 256 * 256; }

struct CompressWs {
  float *y0, *y1, *z0, *z1, *T, *Wu, *Wv, *L1, *L2, *Xg, *Mt, *Wt, *MWn, *Wn, *Mg, *Wg;
  double *G, *sig64;
  char* tc;  // the tensor-core residual products' scratch (bf16 weights)
  size_t bytes;
};

// Carves the workspace (each piece 256-byte aligned from `base`; base == NULL
// only sizes it).
CompressWs carve(char* base, long rows, long cols, long l, long r) {
  const long Lp = l + (l & 1);
  CompressWs w{};
  size_t off = 0;
  auto take = [&](size_t bytes) {
    char* p = base ? base + off : nullptr;
    off += al256(bytes);
    return p;
  };
  w.y0 = (float*)take(4 * rows * l);
  w.y1 = (float*)take(4 * rows * l);
  w.z0 = (float*)take(4 * cols * l);
  w.z1 = (float*)take(4 * cols * l);
  w.T = (float*)take(4 * l * l);
  w.Wu = (float*)take(4 * l * r);
  w.Wv = (float*)take(4 * l * r);
  w.L1 = (float*)take(4 * l * l);
  w.L2 = (float*)take(4 * l * l);
  w.Xg = (float*)take(4 * l * l);
  w.Mt = (float*)take(4 * l * l);
  w.Wt = (float*)take(4 * l * l);
  w.MWn = (float*)take(4 * l * l);
  w.Wn = (float*)take(4 * l * l);
  w.Mg = (float*)take(4 * Lp * l);
  w.Wg = (float*)take(4 * Lp * Lp);
  w.G = (double*)take(8 * l * l);
  w.sig64 = (double*)take(8 * l);
  w.tc = take(res_tc_workspace(rows, cols, l));
  w.bytes = off;
  return w;
}

lx_status check_compress(int32_t rows, int32_t cols, int32_t l, int32_t r) {
  if (rows < 8 || cols < 8 || rows % 8 || cols % 8 || rows > 65536 || cols > 65536)
    return fail(LX_ERR_SHAPE, "rows and cols must be multiples of 8 in 8..65536");
  if (r < 1 || l < r || l > CP_MAX_L || l > std::min(rows, cols))
    return fail(LX_ERR_SHAPE, "need 1 <= r <= l <= min(rows, cols, 256)");
  return LX_OK;
}

template <typename TW>
lx_status run_compress(int rows, int cols, const TW* Wd, const TW* Wm, const float* omega, int l,
                       int r, int q, float* U, float* V, float* sigma, const CompressWs& w,
                       int dev, cudaStream_t s) {
  int num_sms = 0;
  LX_CUDA(cudaDeviceGetAttribute(&num_sms, cudaDevAttrMultiProcessorCount, dev));
  // bf16 weights: the residual products R X and R^T X on the tensor cores
  constexpr bool bf16_w = std::is_same<TW, __nv_bfloat16>::value;
  const bool res_tc = bf16_w && res_tc_fits(rows, cols, l);
  lx_status tc_status = LX_OK;
  auto gemm = [&](int mode, const float* X, const float* B, float* C, int M, int N, int K) {
    const dim3 grid((N + CG_TILE - 1) / CG_TILE, (M + CG_TILE - 1) / CG_TILE);
    if constexpr (bf16_w) {
      if (res_tc && (mode == A_RES || mode == A_RES_T)) {
        const lx_status st = res_gemm_tc(mode == A_RES_T, reinterpret_cast<const __nv_bfloat16*>(Wm),
                                         reinterpret_cast<const __nv_bfloat16*>(Wd), rows, cols, B, N,
                                         C, w.tc, num_sms, dev, s);
        if (st != LX_OK) tc_status = st;
        return;
      }
    }
    if (mode == A_RES)
      k_cgemm<TW, A_RES><<<grid, CG_THREADS, 0, s>>>(Wm, Wd, nullptr, cols, B, C, M, N, K);
    else if (mode == A_RES_T)
      k_cgemm<TW, A_RES_T><<<grid, CG_THREADS, 0, s>>>(Wm, Wd, nullptr, cols, B, C, M, N, K);
    else
      k_cgemm<TW, A_F32><<<grid, CG_THREADS, 0, s>>>(nullptr, nullptr, X, cols, B, C, M, N, K);
  };
  auto gram = [&](const float* X, int n) {
    const dim3 grid((l + GR_T - 1) / GR_T, (l + GR_T - 1) / GR_T);
    k_gram<<<grid, GR_T * GR_T, 0, s>>>(X, n, l, w.G);
  };
  const size_t tri = sizeof(float) * (size_t)l * (l + 1) / 2;
  const bool x_smem = 2 * tri <= CP_SMEM_CAP;  // L and X both in shared memory
  const size_t ch_smem = x_smem ? 2 * tri : tri;
  LX_CUDA(smem_cap_once((const void*)k_chol32, (int)CP_SMEM_CAP, dev, g_ch_cap));
  // CholeskyQR twice (the first pass shifted by 1e-6 of the largest Gram
  // diagonal, so rank-deficient bases stay factorable); X [n][l] ends
  // orthonormal, tmp is scratch; the two factors stay in L1, L2.
  auto orth2 = [&](float* X, float* tmp, int n) {
    gram(X, n);
    k_chol32<<<1, CH_THREADS, ch_smem, s>>>(w.G, l, 1e-6f, w.L1, w.Xg, x_smem ? 1 : 0, w.T);
    gemm(A_F32, X, w.T, tmp, n, l, l);
    gram(tmp, n);
    k_chol32<<<1, CH_THREADS, ch_smem, s>>>(w.G, l, 0.f, w.L2, w.Xg, x_smem ? 1 : 0, w.T);
    gemm(A_F32, tmp, w.T, X, n, l, l);
  };
  gemm(A_RES, nullptr, omega, w.y0, rows, l, cols);  // Y = R Omega
  orth2(w.y0, w.y1, rows);                            // Q
  for (int it = 0; it < q; ++it) {
    gemm(A_RES_T, nullptr, w.y0, w.z0, cols, l, rows);  // R^T Q
    orth2(w.z0, w.z1, cols);
    gemm(A_RES, nullptr, w.z0, w.y0, rows, l, cols);    // R Z
    orth2(w.y0, w.y1, rows);
  }
  // Z = R^T Q = Bs^T = Z2 (L1 L2)^T with Z2 orthonormal, so Bs = M Z2^T for
  // M = L1 L2, and the SVD of Bs follows from the small SVD of M.
  gemm(A_RES_T, nullptr, w.y0, w.z0, cols, l, rows);
  orth2(w.z0, w.z1, cols);
  k_trmm<<<l, 256, 0, s>>>(w.L1, w.L2, l, w.Mt);
  const int Lp = l + (l & 1);
  const size_t os_bytes = sizeof(float) * ((size_t)Lp * l + (size_t)Lp * Lp);
  const bool os_smem = os_bytes <= CP_SMEM_CAP;
  if (os_smem) LX_CUDA(smem_cap_once((const void*)k_onesided, (int)CP_SMEM_CAP, dev, g_os_cap));
  k_onesided<<<1, OS_THREADS, os_smem ? os_bytes : 0, s>>>(w.Mt, l, w.Mg, w.Wg, os_smem ? 1 : 0,
                                                          w.Wt);
  k_ritz<<<l, 256, 0, s>>>(w.Mt, w.Wt, l, w.MWn, w.Wn, w.sig64);
  k_finish<<<1, 256, 0, s>>>(w.sig64, w.MWn, w.Wn, l, r, w.Wu, w.Wv, sigma);
  gemm(A_F32, w.y0, w.Wu, U, rows, r, l);   // U_r S^(1/2)
  gemm(A_F32, w.z0, w.Wv, V, cols, r, l);   // V_r S^(1/2)
  k_sign<<<r, 256, 0, s>>>(U, V, rows, cols, r);
  LX_CUDA(cudaGetLastError());
  return tc_status;
}
}  // namespace
}  // namespace lx

extern "C" lx_status lx_compress_workspace(int32_t rows, int32_t cols, int32_t l, int32_t r,
                                           uint64_t* bytes) {
  using namespace lx;
  if (!bytes) return fail(LX_ERR_ARG, "bytes is NULL");
  LX_TRY(check_compress(rows, cols, l, r));
  *bytes = carve(nullptr, rows, cols, l, r).bytes;
  return LX_OK;
}

extern "C" lx_status lx_compress_factor(int32_t dtype, int32_t rows, int32_t cols,
                                        const void* w_dom, const void* w_mem, const float* omega,
                                        int32_t l, int32_t r, int32_t power_iters, float* U,
                                        float* V, float* sigma, void* workspace,
                                        uint64_t workspace_bytes, void* stream) {
  using namespace lx;
  if (dtype != LX_F32 && dtype != LX_BF16) return fail(LX_ERR_ARG, "unknown dtype");
  LX_TRY(check_compress(rows, cols, l, r));
  if (power_iters < 0 || power_iters > 16) return fail(LX_ERR_ARG, "power_iters outside 0..16");
  if (!w_dom || !w_mem || !omega || !U || !V || !sigma || !workspace)
    return fail(LX_ERR_ARG, "NULL pointer");
  if (((uintptr_t)w_dom & 15u) || ((uintptr_t)w_mem & 15u))
    return fail(LX_ERR_ARG, "w_dom and w_mem must be 16-byte aligned");
  if ((uintptr_t)workspace & 255u) return fail(LX_ERR_ARG, "workspace must be 256-byte aligned");
  const CompressWs w = carve((char*)workspace, rows, cols, l, r);
  if (workspace_bytes < w.bytes) return fail(LX_ERR_ARG, "workspace too small");
  int dev = 0;
  LX_CUDA(cudaGetDevice(&dev));
  cudaStream_t s = (cudaStream_t)stream;
  if (dtype == LX_BF16)
    return run_compress(rows, cols, (const __nv_bfloat16*)w_dom, (const __nv_bfloat16*)w_mem,
                        omega, l, r, power_iters, U, V, sigma, w, dev, s);
  return run_compress(rows, cols, (const float*)w_dom, (const float*)w_mem, omega, l, r,
                      power_iters, U, V, sigma, w, dev, s);
}
