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
//   k_chol_inv  one CTA: Cholesky G + s I = L L^T (float64, a small relative
//               shift keeps rank-deficient bases factorable) and T = L^-T
//               (fp32) so that X T has orthonormal columns (CholeskyQR; run
//               twice per orthonormalisation).
//   k_jacobi    one CTA: cyclic parallel Jacobi eigensolver (float64) of the
//               l x l Gram of the projected residual, the r largest
//               eigenpairs and the fp32 matrices that turn the basis into the
//               split factors.
//   k_sign      each factor column's largest-magnitude entry of U made
//               positive (U and V negated together).
#include <algorithm>
#include <cmath>

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
// ascending row order.  16 x 16 outputs per CTA.
constexpr int GR_T = 16;
constexpr int GR_KC = 32;
__global__ void __launch_bounds__(GR_T * GR_T)
k_gram(const float* __restrict__ X, int n, int L, double* __restrict__ G) {
  __shared__ double Xi[GR_KC][GR_T], Xj[GR_KC][GR_T];
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

// One CTA (blockDim >= L, L <= 256).  Lw [L][L] float64 workspace.
// Cholesky of G + s I with s = 1e-11 * trace(G) (s = 1 when G = 0), then
// X = L^-1 column by column (thread c solves L x = e_c) and T = X^T (fp32,
// upper triangular), so that Y T = Y L^-T has orthonormal columns when
// Y^T Y = G.
constexpr int CH_THREADS = 256;
__global__ void __launch_bounds__(CH_THREADS)
k_chol_inv(const double* __restrict__ G, int L, double* __restrict__ Lw,
           double* __restrict__ Xw, float* __restrict__ T) {
  __shared__ double s_shift;
  const int tid = threadIdx.x;
  if (tid == 0) {
    double tr = 0.0;
    for (int i = 0; i < L; ++i) tr += G[(size_t)i * L + i];
    s_shift = tr > 0.0 ? 1e-11 * tr : 1.0;
  }
  __syncthreads();
  // lower triangle of G + s I (the upper triangle of Lw is never read)
  for (int q = tid; q < L * L; q += CH_THREADS) {
    const int i = q / L, j = q % L;
    Lw[q] = j <= i ? G[q] + (i == j ? s_shift : 0.0) : 0.0;
  }
  __syncthreads();
  for (int j = 0; j < L; ++j) {
    if (tid == 0) {
      const double d = Lw[(size_t)j * L + j];
      Lw[(size_t)j * L + j] = sqrt(d > 1e-300 ? d : 1e-300);
    }
    __syncthreads();
    const double ljj = Lw[(size_t)j * L + j];
    for (int i = j + 1 + tid; i < L; i += CH_THREADS) Lw[(size_t)i * L + j] /= ljj;
    __syncthreads();
    // trailing update of the lower triangle: A[i][c] -= L[i][j] L[c][j], j < c <= i
    const int w = L - j - 1;
    for (int q = tid; q < w * w; q += CH_THREADS) {
      const int i = j + 1 + q / w, c = j + 1 + q % w;
      if (c <= i) Lw[(size_t)i * L + c] -= Lw[(size_t)i * L + j] * Lw[(size_t)c * L + j];
    }
    __syncthreads();
  }
  // X = L^-1, row by row: thread c owns column c (x_i = -sum_{c<=k<i} L[i][k]
  // x_k / L[i][i]); uniform loops, so a warp reads one broadcast L[i][k] and a
  // contiguous piece of row k of X per step.  Each thread reads back only its
  // own column, so the rows need no barrier between them.
  if (tid < L) {
    const int c = tid;
    for (int i = 0; i < L; ++i) {
      double acc = 0.0;
      for (int k = 0; k < i; ++k)
        if (k >= c) acc = fma(Lw[(size_t)i * L + k], Xw[(size_t)k * L + c], acc);
      const double lii = Lw[(size_t)i * L + i];
      Xw[(size_t)i * L + c] = i < c ? 0.0 : (i == c ? 1.0 / lii : -acc / lii);
    }
  }
  __syncthreads();
  for (int q = tid; q < L * L; q += CH_THREADS) {
    const int k = q / L, n = q % L;  // T[k][n] = X[n][k]
    T[q] = (float)Xw[(size_t)n * L + k];
  }
}

// Symmetric eigensolver for the l x l Gram S = Z^T Z (Z = R^T Q, so S = Bs Bs^T
// for Bs = Q^T R), then the factor matrices of the r largest eigenpairs.
// Cyclic Jacobi, parallel form: Lp = l rounded up to even; in each of the
// Lp - 1 rounds of a sweep the indices are split into Lp / 2 disjoint pairs
// (circle method: index Lp - 1 fixed, the others rotated), every pair's
// rotation J = [[c, s], [-s, c]] zeroes its off-diagonal entry, and
// A <- J^T A J, V <- V J are applied as independent 2 x 2 blocks (each entry
// has one writer per round).  A padding index (odd l) stays decoupled: its row
// and column are zero, so its rotations are the identity.  Sweeps stop when
// the off-diagonal mass is below 1e-28 of the total (squared norms) or after
// JB_MAX_SWEEPS.  A lives in shared memory when it fits, else in `Ag`.
// Outputs, for c < r with i_c the c-th largest eigenvalue lambda (ties: lower
// index first) and sigma_c = sqrt(max(lambda, 0)):
//   sig[c] = sigma_c;  Wu[k][c] = V[k][i_c] sqrt(sigma_c);
//   Wv[k][c] = V[k][i_c] / sqrt(sigma_c), or 0 when sigma_c <= 1e-6 sigma_0.
// Q Wu = U_r S_r^(1/2) and Z Wv = V_r S_r^(1/2) (Eq. factors).
constexpr int JB_THREADS = 512;
constexpr int JB_MAX_L = 256;
constexpr int JB_MAX_SWEEPS = 30;

__global__ void __launch_bounds__(JB_THREADS)
k_jacobi(const double* __restrict__ S, int L, int r, double* __restrict__ Ag,
         double* __restrict__ V, int a_in_smem, float* __restrict__ Wu,
         float* __restrict__ Wv, float* __restrict__ sig) {
  extern __shared__ double Asm[];
  __shared__ double pc[JB_MAX_L / 2], ps[JB_MAX_L / 2];
  __shared__ int pp[JB_MAX_L / 2], pq[JB_MAX_L / 2];
  __shared__ int order[JB_MAX_L];
  __shared__ double red[2][JB_THREADS / 32];
  __shared__ int s_done;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int Lp = L + (L & 1), half = Lp / 2;
  double* A = a_in_smem ? Asm : Ag;
  for (int q = tid; q < Lp * Lp; q += JB_THREADS) {
    const int i = q / Lp, j = q % Lp;
    A[q] = (i < L && j < L) ? S[(size_t)i * L + j] : 0.0;
    V[q] = i == j ? 1.0 : 0.0;
  }
  __syncthreads();
  for (int sweep = 0; sweep < JB_MAX_SWEEPS; ++sweep) {
    // convergence: off-diagonal and total squared mass
    double off = 0.0, tot = 0.0;
    for (int q = tid; q < Lp * Lp; q += JB_THREADS) {
      const double a = A[q];
      tot += a * a;
      if (q / Lp != q % Lp) off += a * a;
    }
    for (int o = 16; o; o >>= 1) {
      off += __shfl_xor_sync(0xffffffffu, off, o);
      tot += __shfl_xor_sync(0xffffffffu, tot, o);
    }
    if (lane == 0) {
      red[0][warp] = off;
      red[1][warp] = tot;
    }
    __syncthreads();
    if (tid == 0) {
      double o2 = 0.0, t2 = 0.0;
      for (int w = 0; w < JB_THREADS / 32; ++w) {
        o2 += red[0][w];
        t2 += red[1][w];
      }
      s_done = (t2 == 0.0 || o2 <= 1e-28 * t2) ? 1 : 0;
    }
    __syncthreads();
    if (s_done) break;
    for (int round = 0; round < Lp - 1; ++round) {
      if (tid < half) {
        int p, q;
        if (tid == 0) {
          p = round;
          q = Lp - 1;
        } else {
          p = (round + tid) % (Lp - 1);
          q = (round - tid + (Lp - 1)) % (Lp - 1);
        }
        const double app = A[(size_t)p * Lp + p], aqq = A[(size_t)q * Lp + q];
        const double apq = A[(size_t)p * Lp + q];
        double c = 1.0, s = 0.0;
        if (apq != 0.0 && fabs(apq) > 1e-300) {
          const double tau = (aqq - app) / (2.0 * apq);
          const double t = (tau >= 0.0 ? 1.0 : -1.0) / (fabs(tau) + sqrt(1.0 + tau * tau));
          c = 1.0 / sqrt(1.0 + t * t);
          s = t * c;
        }
        pc[tid] = c;
        ps[tid] = s;
        pp[tid] = p;
        pq[tid] = q;
      }
      __syncthreads();
      // A <- J^T A J by 2 x 2 blocks (pair P rows, pair P2 columns)
      for (int w = tid; w < half * half; w += JB_THREADS) {
        const int P = w / half, P2 = w % half;
        const int p = pp[P], q = pq[P], p2 = pp[P2], q2 = pq[P2];
        const double c = pc[P], s = ps[P], c2 = pc[P2], s2 = ps[P2];
        const double b00 = A[(size_t)p * Lp + p2], b01 = A[(size_t)p * Lp + q2];
        const double b10 = A[(size_t)q * Lp + p2], b11 = A[(size_t)q * Lp + q2];
        // rows: J^T B
        const double r00 = c * b00 - s * b10, r01 = c * b01 - s * b11;
        const double r10 = s * b00 + c * b10, r11 = s * b01 + c * b11;
        // columns: (J^T B) J2
        double n00 = c2 * r00 - s2 * r01, n01 = s2 * r00 + c2 * r01;
        double n10 = c2 * r10 - s2 * r11, n11 = s2 * r10 + c2 * r11;
        if (P == P2) n01 = n10 = 0.0;  // the entry this rotation annihilates
        A[(size_t)p * Lp + p2] = n00;
        A[(size_t)p * Lp + q2] = n01;
        A[(size_t)q * Lp + p2] = n10;
        A[(size_t)q * Lp + q2] = n11;
      }
      // V <- V J
      for (int w = tid; w < Lp * half; w += JB_THREADS) {
        const int i = w / half, P = w % half;
        const int p = pp[P], q = pq[P];
        const double c = pc[P], s = ps[P];
        const double vp = V[(size_t)i * Lp + p], vq = V[(size_t)i * Lp + q];
        V[(size_t)i * Lp + p] = c * vp - s * vq;
        V[(size_t)i * Lp + q] = s * vp + c * vq;
      }
      __syncthreads();
    }
  }
  // rank of every real index by (eigenvalue descending, index ascending)
  for (int i = tid; i < L; i += JB_THREADS) {
    const double li = A[(size_t)i * Lp + i];
    int rk = 0;
    for (int j = 0; j < L; ++j) {
      const double lj = A[(size_t)j * Lp + j];
      rk += (lj > li || (lj == li && j < i)) ? 1 : 0;
    }
    order[rk] = i;
  }
  __syncthreads();
  const double sig0 = sqrt(fmax(A[(size_t)order[0] * Lp + order[0]], 0.0));
  for (int q = tid; q < L * r; q += JB_THREADS) {
    const int k = q / r, c = q % r;
    const int i = order[c];
    const double sg = sqrt(fmax(A[(size_t)i * Lp + i], 0.0));
    const double rs = sqrt(sg);
    const double v = V[(size_t)k * Lp + i];
    Wu[q] = (float)(v * rs);
    Wv[q] = (sg > 1e-6 * sig0 && sg > 0.0) ? (float)(v / rs) : 0.f;
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

bool g_jb_cap[64] = {};

}  // namespace
}  // namespace lx

namespace lx {
namespace {
constexpr int CP_MAX_L = 256;

size_t al256(size_t v) { return (v + 255) / 256 * 256; }

struct CompressWs {
  float *y0, *y1, *z0, *z1, *T, *Wu, *Wv;
  double *G, *Lw, *Xw, *A, *V;
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
  w.G = (double*)take(8 * l * l);
  w.Lw = (double*)take(8 * l * l);
  w.Xw = (double*)take(8 * l * l);
  w.A = (double*)take(8 * Lp * Lp);
  w.V = (double*)take(8 * Lp * Lp);
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
  auto gemm = [&](int mode, const float* X, const float* B, float* C, int M, int N, int K) {
    const dim3 grid((N + CG_TILE - 1) / CG_TILE, (M + CG_TILE - 1) / CG_TILE);
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
  // CholeskyQR twice: X [n][l] -> orthonormal columns, result in X (tmp scratch)
  auto orth2 = [&](float* X, float* tmp, int n) {
    gram(X, n);
    k_chol_inv<<<1, CH_THREADS, 0, s>>>(w.G, l, w.Lw, w.Xw, w.T);
    gemm(A_F32, X, w.T, tmp, n, l, l);
    gram(tmp, n);
    k_chol_inv<<<1, CH_THREADS, 0, s>>>(w.G, l, w.Lw, w.Xw, w.T);
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
  gemm(A_RES_T, nullptr, w.y0, w.z0, cols, l, rows);    // Z = R^T Q = Bs^T
  gram(w.z0, cols);                                     // Bs Bs^T
  const int Lp = l + (l & 1);
  const size_t a_bytes = (size_t)Lp * Lp * 8;
  const bool in_smem = a_bytes <= 200 * 1024;
  if (in_smem)
    LX_CUDA(smem_cap_once((const void*)k_jacobi, 200 * 1024, dev, g_jb_cap));
  k_jacobi<<<1, JB_THREADS, in_smem ? a_bytes : 0, s>>>(w.G, l, r, w.A, w.V, in_smem ? 1 : 0,
                                                        w.Wu, w.Wv, sigma);
  gemm(A_F32, w.y0, w.Wu, U, rows, r, l);   // U_r S^(1/2)
  gemm(A_F32, w.z0, w.Wv, V, cols, r, l);   // V_r S^(1/2)
  k_sign<<<r, 256, 0, s>>>(U, V, rows, cols, r);
  LX_CUDA(cudaGetLastError());
  return LX_OK;
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
