// Compression of one member projection (Sec. 3.2 Stage 3 (ii)): the residual
// R = W_mem - W_dom ([rows][cols], Eq. svd), its rank-r randomized SVD (range
// finder with power iterations, Halko-Martinsson-Tropp, with the Gaussian test
// matrix given by the caller) and the symmetric split of Eq. factors,
// U = U_r S_r^(1/2) [rows][r], V = V_r S_r^(1/2) [cols][r].
//
// Kernels (the products with R of bf16 weights run on the tensor cores, in
// lx_compress_tc.cu):
//   k_cgemm     fp32 GEMM (CUDA-core FMA, 64 x 64 tiles, 32-deep K chunks in
//               shared memory); its A operand is R (rows of W_mem - W_dom,
//               formed on load; fp32 weights), R^T (columns of the same), or an
//               fp32 matrix (the bases times the small factors).
//   k_gram      G = X^T X to float64 accuracy (exact fp32 products, error-free
//               two-sum accumulation on the fp32 pipes), stored in float64.
//   k_chol32    one CTA: Cholesky G + s I = L L^T (fp32 in shared memory,
//               blocked by 16 columns; a small relative shift in the first
//               pass keeps rank-deficient bases factorable) and T = L^-T,
//               blocked the same way, so that X T has orthonormal columns
//               (CholeskyQR).
//   k_trmm      M = L1 L2, the triangular factor of R^T Q = Z2 M^T.
//   k_onesided_v, k_onesided
//               one CTA: one-sided Jacobi SVD of M (fp32 rotations in shared
//               memory, one 8-lane group per column pair so that every pair
//               of a round runs at once), M W = U S; the _v form keeps the
//               pair's columns in registers (l <= 144).
//   k_ritz      sigma_j = |M w_j| / |w_j| in float64 (Rayleigh quotients).
//   k_finish    the r largest sigma and the fp32 matrices that turn the bases
//               into the split factors.
//   k_sign      each factor column's largest-magnitude entry of U made
//               positive (U and V negated together).
// Only the Rayleigh quotients use float64 arithmetic, and the Gram sums reach
// float64 accuracy by compensated fp32 arithmetic: this GPU's float64 rate is
// a small fraction of its fp32 rate.
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

// G [L][L] = X^T X for X [n][L] fp32 row-major, to float64 accuracy on the
// fp32 pipes (this GPU's float64 rate is a small fraction of its fp32 rate).
// Each product is formed exactly as the pair p + e (p = x y rounded,
// e = fma(x, y, -p)); the sum is carried as an unevaluated pair hi + lo, hi
// taking the products through Knuth's error-free two-sum and lo collecting the
// two-sum and product errors (the compensated dot product "Dot2" of Ogita,
// Rump and Oishi, 2005), so G = hi + lo is as accurate as a dot product in
// twice the fp32 precision: within 2^-24 |G| + (n 2^-24)^2 sum |x y| of the
// exact sum, far below the fp32 rounding the Cholesky applies to it.  Four
// such pairs per thread take the rows of a chunk in turn (independent chains)
// and are added pairwise at the end; each 64-row chunk is staged in shared
// memory while the next one is already loading into registers.  16 x 16
// outputs per CTA; only the tiles on or below the diagonal are computed (the
// Cholesky reads the lower triangle alone).
constexpr int GR_T = 16;
constexpr int GR_KC = 64;
constexpr int GR_CH = 4;
static_assert(GR_KC * GR_T % (GR_T * GR_T) == 0, "whole staged values per thread");

struct DF {
  float hi, lo;
};
// hi + lo += p + e, by the two-sum of hi and p (every step rounded on its own:
// the intrinsics are never contracted into fused operations)
__device__ __forceinline__ void df_add(DF& d, float p, float e) {
  const float s = __fadd_rn(d.hi, p);
  const float v = __fsub_rn(s, d.hi);
  const float err = __fadd_rn(__fsub_rn(d.hi, __fsub_rn(s, v)), __fsub_rn(p, v));
  d.hi = s;
  d.lo = __fadd_rn(d.lo, __fadd_rn(err, e));
}

__global__ void __launch_bounds__(GR_T * GR_T)
k_gram(const float* __restrict__ X, int n, int L, double* __restrict__ G) {
  constexpr int PER = GR_KC * GR_T / (GR_T * GR_T);  // staged values per thread and side
  __shared__ float Xi[GR_KC][GR_T], Xj[GR_KC][GR_T];
  if (blockIdx.x > blockIdx.y) return;  // strictly above the diagonal
  const int ti = threadIdx.x / GR_T, tj = threadIdx.x % GR_T;
  const int i0 = blockIdx.y * GR_T, j0 = blockIdx.x * GR_T;
  DF acc[GR_CH];
#pragma unroll
  for (int c = 0; c < GR_CH; ++c) acc[c] = DF{0.f, 0.f};
  // the next chunk's rows are loaded into registers while this one is summed
  float ri[PER], rj[PER];
  auto fetch = [&](int m0) {
#pragma unroll
    for (int e = 0; e < PER; ++e) {
      const int q = threadIdx.x + e * GR_T * GR_T;
      const int mr = q / GR_T, c = q % GR_T;
      const bool okm = m0 + mr < n;
      ri[e] = (okm && i0 + c < L) ? X[(size_t)(m0 + mr) * L + i0 + c] : 0.f;
      rj[e] = (okm && j0 + c < L) ? X[(size_t)(m0 + mr) * L + j0 + c] : 0.f;
    }
  };
  fetch(0);
  for (int m0 = 0; m0 < n; m0 += GR_KC) {
#pragma unroll
    for (int e = 0; e < PER; ++e) {
      const int q = threadIdx.x + e * GR_T * GR_T;
      Xi[q / GR_T][q % GR_T] = ri[e];
      Xj[q / GR_T][q % GR_T] = rj[e];
    }
    __syncthreads();
    if (m0 + GR_KC < n) fetch(m0 + GR_KC);
#pragma unroll
    for (int mr = 0; mr < GR_KC; mr += GR_CH) {
#pragma unroll
      for (int c = 0; c < GR_CH; ++c) {
        const float x = Xi[mr + c][ti], y = Xj[mr + c][tj];
        const float p = __fmul_rn(x, y);
        df_add(acc[c], p, __fmaf_rn(x, y, -p));
      }
    }
    __syncthreads();
  }
  // (chain 0 + chain 1) + (chain 2 + chain 3), each pair added as hi + lo
  DF s01 = acc[0], s23 = acc[2];
  df_add(s01, acc[1].hi, acc[1].lo);
  df_add(s23, acc[3].hi, acc[3].lo);
  df_add(s01, s23.hi, s23.lo);
  if (i0 + ti < L && j0 + tj < L)
    G[(size_t)(i0 + ti) * L + j0 + tj] = (double)s01.hi + (double)s01.lo;
}

// One CTA (L <= 256).  Cholesky of G + s I in fp32 (G float64, rounded once;
// s = shift_rel * max diag(G)) in a packed lower triangle in shared memory
// (L (L + 1) / 2 floats, row i from i (i + 1) / 2), pivots floored at 1e-30,
// blocked by 16 columns (right-looking): warp 0 factors the diagonal block in
// place (lane i updates row i; warp barriers only), one thread per row below
// solves its 16 panel entries against it (forward substitution), and the
// trailing triangle takes the panel's rank-16 update in 4 x 4 register tiles
// from a transposed copy of the panel.  Then X = L^-1, blocked the same way:
// the diagonal blocks' inverses
// (one warp each, lane m column m), and for block row i and every block
// column k < i, X_ik = -X_ii (sum_{k <= m < i} L_im X_mk) in two tiled
// products.  X is packed like L, in shared memory when x_in_smem, else in the
// global scratch Xg.  T = X^T, so that Y T = Y L^-T has orthonormal columns
// when Y^T Y = G (CholeskyQR).  The factor is written to Lout [L][L] (zero
// above the diagonal).  A zero Gram gives Lout = T = 0.
constexpr int CH_THREADS = 512;  // 16 warps: nb <= 16 diagonal blocks, 128 registers a thread
constexpr int CH_B = 16;  // block width
__device__ __forceinline__ int tri_off(int i) { return i * (i + 1) / 2; }

// row-major 4 x 4 tile index blk of a lower block triangle -> (bi, bc), bc <= bi
__device__ __forceinline__ void tri_tile(int blk, int& bi, int& bc) {
  int b = (int)((sqrtf(8.f * (float)blk + 1.f) - 1.f) * 0.5f);
  while (b * (b + 1) / 2 > blk) --b;
  while ((b + 1) * (b + 2) / 2 <= blk) ++b;
  bi = b;
  bc = blk - b * (b + 1) / 2;
}

__global__ void __launch_bounds__(CH_THREADS, 1)
k_chol32(const double* __restrict__ G, int L, float shift_rel, float* __restrict__ Lout,
         float* __restrict__ Xg, int x_in_smem, float* __restrict__ T) {
  extern __shared__ __align__(16) float Ls[];
  const int ldp = (L + 3) & ~3;                      // panel copy: [CH_B][ldp], also S below
  float* Pt = Ls + ((tri_off(L) + 3) & ~3);
  float* Xp = x_in_smem ? Pt + CH_B * ldp : Xg;      // packed lower X
  __shared__ double s_md;
  __shared__ float s_rdiag[256];  // reciprocals of the factor's diagonal
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = CH_THREADS / 32;
  const int nb = (L + CH_B - 1) / CH_B;
  // the lower triangle of G rounded to fp32, every load of a batch in flight
  // (packed element e -> row i, column e - i (i + 1) / 2), while warp 0 also
  // takes the largest diagonal entry
  const int ntri = tri_off(L);
  for (int e0 = tid; e0 < ntri; e0 += 4 * CH_THREADS) {
    double g[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int e = e0 + u * CH_THREADS;
      int i = (int)((sqrtf(8.f * (float)e + 1.f) - 1.f) * 0.5f);
      while (tri_off(i) > e) --i;
      while (tri_off(i + 1) <= e) ++i;
      g[u] = e < ntri ? G[(size_t)i * L + (e - tri_off(i))] : 0.0;
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (e0 + u * CH_THREADS < ntri) Ls[e0 + u * CH_THREADS] = (float)g[u];
  }
  if (warp == 0) {
    double md = 0.0;
    for (int i = lane; i < L; i += 32) md = fmax(md, G[(size_t)i * L + i]);
#pragma unroll
    for (int o = 16; o; o >>= 1) md = fmax(md, __shfl_xor_sync(0xffffffffu, md, o));
    if (lane == 0) s_md = md;
  }
  __syncthreads();
  const double md = s_md;
  if (!(md > 0.0)) {
    for (int i = warp; i < L; i += nw)
      for (int c = lane; c < L; c += 32) {
        Lout[(size_t)i * L + c] = 0.f;
        T[(size_t)i * L + c] = 0.f;
      }
    return;
  }
  const float shift = (float)(shift_rel * md);
  for (int i = tid; i < L; i += CH_THREADS) Ls[tri_off(i) + i] += shift;  // (float) g_ii + shift
  __syncthreads();
  // ---- factorization
  for (int kb = 0; kb < nb; ++kb) {
    const int j0 = kb * CH_B, bw = min(CH_B, L - j0), j1 = j0 + bw, nt = L - j1;
    if (warp == 0) {
      // lane i: row j0 + i of the diagonal block, in place in the packed triangle
      float* Ar = Ls + tri_off(j0 + min(lane, bw - 1)) + j0;
      for (int j = 0; j < bw; ++j) {
        const float d = sqrtf(fmaxf(Ls[tri_off(j0 + j) + j0 + j], 1e-30f));
        const float rd = 1.f / d;
        __syncwarp();
        if (lane == j) Ar[j] = d;
        else if (lane > j && lane < bw) Ar[j] *= rd;  // l_ij
        __syncwarp();
        if (lane > j && lane < bw) {
          const float lij = Ar[j];
          for (int c = j + 1; c <= lane; ++c) Ar[c] = fmaf(-lij, Ls[tri_off(j0 + c) + j0 + j], Ar[c]);
        }
        if (lane == 0) s_rdiag[j0 + j] = rd;
        __syncwarp();
      }
    }
    __syncthreads();
    if (nt > 0) {
      // panel: row i solves x L_kk^T = a_i[j0 : j1]
      for (int i = j1 + tid; i < L; i += CH_THREADS) {
        float x[CH_B];
        float* Ai = Ls + tri_off(i) + j0;
#pragma unroll
        for (int c = 0; c < CH_B; ++c) x[c] = c < bw ? Ai[c] : 0.f;
#pragma unroll
        for (int c = 0; c < CH_B; ++c) {
          if (c < bw) {
            x[c] *= s_rdiag[j0 + c];
#pragma unroll
            for (int c2 = c + 1; c2 < CH_B; ++c2)
              if (c2 < bw) x[c2] = fmaf(-x[c], Ls[tri_off(j0 + c2) + j0 + c], x[c2]);
          }
        }
#pragma unroll
        for (int c = 0; c < CH_B; ++c)
          if (c < bw) {
            Ai[c] = x[c];
            Pt[c * ldp + (i - j1)] = x[c];
          }
      }
      __syncthreads();
      // trailing triangle: A_ic -= sum_m P_im P_cm, 4 x 4 tiles
      const int n4 = (nt + 3) / 4;
      for (int blk = tid; blk < n4 * (n4 + 1) / 2; blk += CH_THREADS) {
        int bi, bc;
        tri_tile(blk, bi, bc);
        float acc[4][4] = {};
        for (int m = 0; m < bw; ++m) {
          const float4 a = *reinterpret_cast<const float4*>(Pt + m * ldp + 4 * bi);
          const float4 b = *reinterpret_cast<const float4*>(Pt + m * ldp + 4 * bc);
          const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
          for (int u = 0; u < 4; ++u)
#pragma unroll
            for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(av[u], bv[v], acc[u][v]);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int i = j1 + 4 * bi + u;
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            const int c = j1 + 4 * bc + v;
            if (i < L && c <= i) Ls[tri_off(i) + c] -= acc[u][v];
          }
        }
      }
      __syncthreads();
    }
  }
  // ---- X = L^-1: the diagonal blocks, one warp each (lane m: column m)
  if (warp < nb) {
    const int j0 = warp * CH_B, bw = min(CH_B, L - j0);
    float x[CH_B];
#pragma unroll
    for (int i = 0; i < CH_B; ++i) x[i] = i == lane ? 1.f : 0.f;
#pragma unroll
    for (int p = 0; p < CH_B; ++p) {
      if (p < bw) {
        x[p] *= s_rdiag[j0 + p];
#pragma unroll
        for (int i = p + 1; i < CH_B; ++i)
          if (i < bw) x[i] = fmaf(-Ls[tri_off(j0 + i) + j0 + p], x[p], x[i]);
      }
    }
    if (lane < bw) {
#pragma unroll
      for (int i = 0; i < CH_B; ++i)
        if (i >= lane && i < bw) Xp[tri_off(j0 + i) + j0 + lane] = x[i];
    }
  }
  __syncthreads();
  // block row ib: S_k = sum_{k <= m < ib} L_{ib,m} X_{m,k} (into the panel
  // buffer), then X_{ib,k} = -X_{ib,ib} S_k, for every k < ib
  float* S = Pt;  // [k][CH_B rows][CH_B columns]
  for (int ib = 1; ib < nb; ++ib) {
    const int i0 = ib * CH_B, bwi = min(CH_B, L - i0), r4 = (bwi + 3) / 4;
    const int ntile = ib * r4 * (CH_B / 4);
    for (int tt = tid; tt < ntile; tt += CH_THREADS) {
      const int kb = tt / (r4 * (CH_B / 4)), rem = tt - kb * r4 * (CH_B / 4);
      const int rt = rem / (CH_B / 4), ct = rem - rt * (CH_B / 4);
      const int col0 = kb * CH_B + 4 * ct;
      float acc[4][4] = {};
      for (int q = kb * CH_B; q < i0; ++q) {
        float a[4], b[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int i = i0 + 4 * rt + u;
          a[u] = i < L ? Ls[tri_off(i) + q] : 0.f;
          b[u] = q >= col0 + u ? Xp[tri_off(q) + col0 + u] : 0.f;
        }
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
          for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(a[u], b[v], acc[u][v]);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) S[(kb * CH_B + 4 * rt + u) * CH_B + 4 * ct + v] = acc[u][v];
    }
    __syncthreads();
    for (int tt = tid; tt < ntile; tt += CH_THREADS) {
      const int kb = tt / (r4 * (CH_B / 4)), rem = tt - kb * r4 * (CH_B / 4);
      const int rt = rem / (CH_B / 4), ct = rem - rt * (CH_B / 4);
      float acc[4][4] = {};
      for (int p = 0; p < min(bwi, 4 * rt + 4); ++p) {
        float a[4], b[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int r = 4 * rt + u;
          a[u] = (r < bwi && p <= r) ? Xp[tri_off(i0 + r) + i0 + p] : 0.f;
          b[u] = S[(kb * CH_B + p) * CH_B + 4 * ct + u];
        }
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
          for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(a[u], b[v], acc[u][v]);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int r = 4 * rt + u;
        if (r < bwi)
#pragma unroll
          for (int v = 0; v < 4; ++v) Xp[tri_off(i0 + r) + kb * CH_B + 4 * ct + v] = -acc[u][v];
      }
    }
    __syncthreads();
  }
  for (int i = warp; i < L; i += nw) {
    const float* Ai = Ls + tri_off(i);
    for (int c = lane; c < L; c += 32) {
      Lout[(size_t)i * L + c] = c <= i ? Ai[c] : 0.f;
      T[(size_t)i * L + c] = c >= i ? Xp[tri_off(c) + i] : 0.f;  // T[k][n] = X[n][k]
    }
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
// each round pairs the columns by the circle method and a group of OS_GROUP = 8
// lanes takes one pair, so the 128 groups of the CTA cover every pair of a
// round (Lp / 2 <= 128) at once and a round costs one pair's latency and one
// barrier.  For a pair: alpha = |m_p|^2, beta = |m_q|^2, gamma = m_p . m_q
// (fp32, each lane a strided share, then a butterfly inside the group, which
// leaves every lane of the group the same sums), and unless
// |gamma| <= 1e-6 sqrt(alpha beta) (a little above the rounding of an fp32
// dot product, so that sweeps terminate) columns p, q of M and of W are
// rotated by the angle that makes them orthogonal (zeta = (beta - alpha) /
// (2 gamma), t = sign(zeta) / (|zeta| + sqrt(1 + zeta^2)), c = 1 / sqrt(1 + t^2),
// s = c t).  Sweeps end when one makes no rotation, or after OS_MAX_SWEEPS.
// M [Lp][ldm] and W [Lp][ldw] are column-major with column strides of 8 mod 32
// floats (the four groups of a warp take consecutive columns, which then fall
// on distinct banks), in shared memory when they fit, else in Mg / Wg.
// Output: Wt [L][L], Wt[j][k] = W[k][j].
constexpr int OS_THREADS = 1024;
constexpr int OS_GROUP = 8;
constexpr int OS_MAX_SWEEPS = 30;
static_assert(OS_THREADS / OS_GROUP >= 128, "one group per pair of a round (l <= 256)");

__global__ void __launch_bounds__(OS_THREADS)
k_onesided(const float* __restrict__ Mt, int L, float* __restrict__ Mg, float* __restrict__ Wg,
           int in_smem, int ldm, int ldw, float* __restrict__ Wt) {
  extern __shared__ float osm[];
  __shared__ int s_rot;
  const int tid = threadIdx.x, grp = tid / OS_GROUP, u = tid % OS_GROUP;
  const int Lp = L + (L & 1), half = Lp / 2;
  float* M = in_smem ? osm : Mg;                       // [Lp][ldm]
  float* W = in_smem ? osm + (size_t)Lp * ldm : Wg;    // [Lp][ldw]
  for (int e = tid; e < Lp * ldm; e += OS_THREADS) {
    const int c = e / ldm, i = e - c * ldm;
    M[e] = (c < L && i < L) ? Mt[(size_t)c * L + i] : 0.f;
  }
  for (int e = tid; e < Lp * ldw; e += OS_THREADS) {
    const int c = e / ldw, i = e - c * ldw;
    W[e] = i == c ? 1.f : 0.f;
  }
  const bool active = grp < half;
  for (int sweep = 0; sweep < OS_MAX_SWEEPS; ++sweep) {
    if (tid == 0) s_rot = 0;
    __syncthreads();
    bool rotated = false;
    for (int round = 0; round < Lp - 1; ++round) {
      int p = 0, q = 1;
      if (grp == 0) {
        p = round;
        q = Lp - 1;
      } else if (active) {
        p = round + grp;
        if (p >= Lp - 1) p -= Lp - 1;
        q = round - grp;
        if (q < 0) q += Lp - 1;
      }
      float* mp = M + (size_t)p * ldm;
      float* mq = M + (size_t)q * ldm;
      float a = 0.f, b = 0.f, g = 0.f;
      if (active) {
#pragma unroll 4
        for (int i = u; i < L; i += OS_GROUP) {
          const float x = mp[i], y = mq[i];
          a = fmaf(x, x, a);
          b = fmaf(y, y, b);
          g = fmaf(x, y, g);
        }
      }
      // (xor offsets below OS_GROUP stay inside the aligned group)
#pragma unroll
      for (int o = OS_GROUP / 2; o; o >>= 1) {
        a += __shfl_xor_sync(0xffffffffu, a, o);
        b += __shfl_xor_sync(0xffffffffu, b, o);
        g += __shfl_xor_sync(0xffffffffu, g, o);
      }
      if (active && g != 0.f && fabsf(g) > 1e-6f * sqrtf(a * b)) {  // group-uniform
        // (an overflowing zeta gives t = 0: no rotation, never a NaN)
        const float z = (b - a) / (2.f * g);
        const float t = (z >= 0.f ? 1.f : -1.f) / (fabsf(z) + sqrtf(1.f + z * z));
        const float c = 1.f / sqrtf(1.f + t * t), sn = t * c;
#pragma unroll 4
        for (int i = u; i < L; i += OS_GROUP) {
          const float x = mp[i], y = mq[i];
          mp[i] = c * x - sn * y;
          mq[i] = sn * x + c * y;
        }
        float* wp = W + (size_t)p * ldw;
        float* wq = W + (size_t)q * ldw;
#pragma unroll 4
        for (int i = u; i < Lp; i += OS_GROUP) {
          const float x = wp[i], y = wq[i];
          wp[i] = c * x - sn * y;
          wq[i] = sn * x + c * y;
        }
        rotated = true;
      }
      __syncthreads();
    }
    if (rotated) s_rot = 1;
    __syncthreads();
    if (s_rot == 0) break;  // every thread reads the same value after the barrier
    __syncthreads();        // before thread 0 clears s_rot for the next sweep
  }
  for (int e = tid; e < L * L; e += OS_THREADS) {
    const int j = e / L, k = e - j * L;
    Wt[e] = W[(size_t)j * ldw + k];
  }
}

// The same Jacobi for L <= 16 NV with M and W in shared memory: each lane of
// a group holds NV float2 pieces of each of its two columns (elements
// 16 v + 2 u, + 1), loaded once for the dot products and kept in registers
// for the rotation; W's columns stream through as float2 too.  Column strides
// ldm, ldw >= 16 NV are multiples of 8 but not of 32, so the four groups of a
// warp (consecutive columns) spread each 256-byte access over two wavefronts.
// The padding rows beyond L (beyond Lp for W) are zero and stay zero.
template <int NV>
__global__ void __launch_bounds__(OS_THREADS)
k_onesided_v(const float* __restrict__ Mt, int L, int ldm, int ldw, float* __restrict__ Wt) {
  extern __shared__ __align__(16) float osm[];
  __shared__ int s_rot;
  const int tid = threadIdx.x, grp = tid / OS_GROUP, u = tid % OS_GROUP;
  const int Lp = L + (L & 1), half = Lp / 2;
  float* M = osm;                       // [Lp][ldm]
  float* W = osm + (size_t)Lp * ldm;    // [Lp][ldw]
  for (int e = tid; e < Lp * ldm; e += OS_THREADS) {
    const int c = e / ldm, i = e - c * ldm;
    M[e] = (c < L && i < L) ? Mt[(size_t)c * L + i] : 0.f;
  }
  for (int e = tid; e < Lp * ldw; e += OS_THREADS) {
    const int c = e / ldw, i = e - c * ldw;
    W[e] = i == c ? 1.f : 0.f;
  }
  const bool active = grp < half;
  for (int sweep = 0; sweep < OS_MAX_SWEEPS; ++sweep) {
    if (tid == 0) s_rot = 0;
    __syncthreads();
    bool rotated = false;
    for (int round = 0; round < Lp - 1; ++round) {
      int p = 0, q = 1;
      if (grp == 0) {
        p = round;
        q = Lp - 1;
      } else if (active) {
        p = round + grp;
        if (p >= Lp - 1) p -= Lp - 1;
        q = round - grp;
        if (q < 0) q += Lp - 1;
      }
      float2* mp = reinterpret_cast<float2*>(M + (size_t)p * ldm) + u;
      float2* mq = reinterpret_cast<float2*>(M + (size_t)q * ldm) + u;
      float2 xp[NV], xq[NV];
      float a = 0.f, b = 0.f, g = 0.f;
      if (active) {
#pragma unroll
        for (int v = 0; v < NV; ++v) {
          xp[v] = mp[8 * v];
          xq[v] = mq[8 * v];
        }
#pragma unroll
        for (int v = 0; v < NV; ++v) {
          a = fmaf(xp[v].x, xp[v].x, a);
          a = fmaf(xp[v].y, xp[v].y, a);
          b = fmaf(xq[v].x, xq[v].x, b);
          b = fmaf(xq[v].y, xq[v].y, b);
          g = fmaf(xp[v].x, xq[v].x, g);
          g = fmaf(xp[v].y, xq[v].y, g);
        }
      }
#pragma unroll
      for (int o = OS_GROUP / 2; o; o >>= 1) {
        a += __shfl_xor_sync(0xffffffffu, a, o);
        b += __shfl_xor_sync(0xffffffffu, b, o);
        g += __shfl_xor_sync(0xffffffffu, g, o);
      }
      if (active && g != 0.f && fabsf(g) > 1e-6f * sqrtf(a * b)) {  // group-uniform
        const float z = (b - a) / (2.f * g);
        const float t = (z >= 0.f ? 1.f : -1.f) / (fabsf(z) + sqrtf(1.f + z * z));
        const float c = 1.f / sqrtf(1.f + t * t), sn = t * c;
#pragma unroll
        for (int v = 0; v < NV; ++v) {
          mp[8 * v] = make_float2(c * xp[v].x - sn * xq[v].x, c * xp[v].y - sn * xq[v].y);
          mq[8 * v] = make_float2(sn * xp[v].x + c * xq[v].x, sn * xp[v].y + c * xq[v].y);
        }
        float2* wp = reinterpret_cast<float2*>(W + (size_t)p * ldw) + u;
        float2* wq = reinterpret_cast<float2*>(W + (size_t)q * ldw) + u;
#pragma unroll
        for (int v = 0; v < NV; ++v) {
          const float2 x = wp[8 * v], y = wq[8 * v];
          wp[8 * v] = make_float2(c * x.x - sn * y.x, c * x.y - sn * y.y);
          wq[8 * v] = make_float2(sn * x.x + c * y.x, sn * x.y + c * y.y);
        }
        rotated = true;
      }
      __syncthreads();
    }
    if (rotated) s_rot = 1;
    __syncthreads();
    if (s_rot == 0) break;
    __syncthreads();
  }
  for (int e = tid; e < L * L; e += OS_THREADS) {
    const int j = e / L, k = e - j * L;
    Wt[e] = W[(size_t)j * ldw + k];
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
bool g_osv_cap[16][64] = {};

}  // namespace
}  // namespace lx

namespace lx {
namespace {
constexpr int CP_MAX_L = 256;
constexpr size_t CP_SMEM_CAP = 200 * 1024;

size_t al256(size_t v) { return (v + 255) / 256 * 256; }

// Column stride (floats) of the Jacobi's M and W for columns of n entries: a
// multiple of 8 that is 8 mod 32 (n + 39 at most).
long os_ld(long n) {
  long ld = (n + 7) / 8 * 8;
  ld += ((8 - ld % 32) + 32) % 32;
  return ld;
}
// Column stride of the register form: a multiple of 8 that is not one of 32.
long os_ld_v(long n) {
  long ld = (n + 7) / 8 * 8;
  return ld % 32 == 0 ? ld + 8 : ld;
}

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
  w.Mg = (float*)take(4 * Lp * os_ld(l));
  w.Wg = (float*)take(4 * Lp * os_ld(Lp));
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
  // packed L (rounded to 16 bytes), the panel copy, and packed X
  // when it fits too
  const size_t tri = sizeof(float) * (size_t)l * (l + 1) / 2;
  const size_t ch_base = (tri + 15) / 16 * 16 + sizeof(float) * CH_B * (size_t)((l + 3) & ~3);
  const bool x_smem = ch_base + tri <= CP_SMEM_CAP;
  const size_t ch_smem = x_smem ? ch_base + tri : ch_base;
  LX_CUDA(smem_cap_once((const void*)k_chol32, (int)CP_SMEM_CAP, dev, g_ch_cap));
  // CholeskyQR (the first pass shifted by 1e-6 of the largest Gram diagonal,
  // so rank-deficient bases stay factorable).  orth2 runs it twice, X [n][l]
  // ends orthonormal and its two factors stay in L1, L2; orth1 runs the
  // shifted pass once, for the intermediate bases of the power iterations,
  // whose span is all the next product uses (the final Q and Z take orth2).
  // Both leave the result in *X and swap *X with the scratch *tmp.
  auto orth1 = [&](float** X, float** tmp, int n) {
    gram(*X, n);
    k_chol32<<<1, CH_THREADS, ch_smem, s>>>(w.G, l, 1e-6f, w.L1, w.Xg, x_smem ? 1 : 0, w.T);
    gemm(A_F32, *X, w.T, *tmp, n, l, l);
    std::swap(*X, *tmp);
  };
  auto orth2 = [&](float** X, float** tmp, int n) {
    gram(*X, n);
    k_chol32<<<1, CH_THREADS, ch_smem, s>>>(w.G, l, 1e-6f, w.L1, w.Xg, x_smem ? 1 : 0, w.T);
    gemm(A_F32, *X, w.T, *tmp, n, l, l);
    gram(*tmp, n);
    k_chol32<<<1, CH_THREADS, ch_smem, s>>>(w.G, l, 0.f, w.L2, w.Xg, x_smem ? 1 : 0, w.T);
    gemm(A_F32, *tmp, w.T, *X, n, l, l);
  };
  float *yc = w.y0, *yt = w.y1, *zc = w.z0, *zt = w.z1;
  gemm(A_RES, nullptr, omega, yc, rows, l, cols);  // Y = R Omega
  if (q == 0) orth2(&yc, &yt, rows);              // Q
  else orth1(&yc, &yt, rows);
  for (int it = 0; it < q; ++it) {
    gemm(A_RES_T, nullptr, yc, zc, cols, l, rows);  // R^T Q
    orth1(&zc, &zt, cols);
    gemm(A_RES, nullptr, zc, yc, rows, l, cols);    // R Z
    if (it + 1 == q) orth2(&yc, &yt, rows);
    else orth1(&yc, &yt, rows);
  }
  // Z = R^T Q = Bs^T = Z2 (L1 L2)^T with Z2 orthonormal, so Bs = M Z2^T for
  // M = L1 L2, and the SVD of Bs follows from the small SVD of M.
  gemm(A_RES_T, nullptr, yc, zc, cols, l, rows);
  orth2(&zc, &zt, cols);
  k_trmm<<<l, 256, 0, s>>>(w.L1, w.L2, l, w.Mt);
  const int Lp = l + (l & 1);
  // register form when the columns fit NV float2 pieces per lane (NV <= 9,
  // l <= 144) and M, W fit shared memory; else the strided form
  const int nv = Lp <= 32 ? 2 : Lp <= 48 ? 3 : Lp <= 80 ? 5 : Lp <= 144 ? 9 : 0;
  const long ldv = nv ? os_ld_v(16 * nv) : 0;
  const size_t osv_bytes = sizeof(float) * (size_t)Lp * 2 * ldv;
  if (nv && osv_bytes <= CP_SMEM_CAP) {
    auto launch_v = [&](auto kern) -> lx_status {
      LX_CUDA(smem_cap_once((const void*)kern, (int)CP_SMEM_CAP, dev, g_osv_cap[nv]));
      kern<<<1, OS_THREADS, osv_bytes, s>>>(w.Mt, l, (int)ldv, (int)ldv, w.Wt);
      return LX_OK;
    };
    if (nv == 2) LX_TRY(launch_v(k_onesided_v<2>));
    else if (nv == 3) LX_TRY(launch_v(k_onesided_v<3>));
    else if (nv == 5) LX_TRY(launch_v(k_onesided_v<5>));
    else LX_TRY(launch_v(k_onesided_v<9>));
  } else {
    const long ldm = os_ld(l), ldw = os_ld(Lp);
    const size_t os_bytes = sizeof(float) * (size_t)Lp * (ldm + ldw);
    const bool os_smem = os_bytes <= CP_SMEM_CAP;
    if (os_smem) LX_CUDA(smem_cap_once((const void*)k_onesided, (int)CP_SMEM_CAP, dev, g_os_cap));
    k_onesided<<<1, OS_THREADS, os_smem ? os_bytes : 0, s>>>(w.Mt, l, w.Mg, w.Wg, os_smem ? 1 : 0,
                                                            (int)ldm, (int)ldw, w.Wt);
  }
  k_ritz<<<l, 256, 0, s>>>(w.Mt, w.Wt, l, w.MWn, w.Wn, w.sig64);
  k_finish<<<1, 256, 0, s>>>(w.sig64, w.MWn, w.Wn, l, r, w.Wu, w.Wv, sigma);
  gemm(A_F32, yc, w.Wu, U, rows, r, l);   // U_r S^(1/2)
  gemm(A_F32, zc, w.Wv, V, cols, r, l);   // V_r S^(1/2)
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
