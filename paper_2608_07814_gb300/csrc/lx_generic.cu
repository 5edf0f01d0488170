// Generic expert path (CUDA cores, fp32 accumulation, every dtype and shape).
//
// For every node n and every token t in its bucket the shared product is
// evaluated once (Sec. 5.1):
//   anchor:     h[(t,n)] = x_t [Wg;Wu]^T                       (2I values)
//   correction: P[(t,n)] = x_t [Vg|Vu],  h[(t,n)] = [Pg Ug^T | Pu Uu^T]
// then per (t, n) the SwiGLU outputs of the selected experts whose path holds n
// are aggregated with their gates (linearity of the down projection):
//   z[(t,n)] = sum_{s : n in path(e_s)} g_s * silu(sum_l h_g[(t,path_l)]) * (sum_l h_u[...])
// and the down projection is again evaluated once per (t, n):
//   anchor:     ypart[(t,n)] = z Wd^T;   correction: ypart[(t,n)] = (z Vd) Ud^T
// y_t is the sum of ypart over t's rows in ascending node order.
#include <algorithm>
#include <type_traits>

#include "lx_internal.cuh"

namespace lx {

namespace {

constexpr int GG_THREADS = 256;

// OPK only names the instantiation (one kernel symbol per op in profiles)
template <typename TA, typename TW, int OPK>
__global__ void __launch_bounds__(GG_THREADS)
k_grouped_gemm(GemmArgs g) {
  pdl_wait();
  __shared__ float As[G_BK][G_BM + 1];
  __shared__ float Ws[G_BK][G_BN + 1];
  const int total = g.tile_off[g.n_items];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;  // 16 x 16 threads
  for (int tile = blockIdx.x; tile < total; tile += gridDim.x) {
    // item = last index with tile_off[item] <= tile
    int lo = 0, hi = g.n_items;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (g.tile_off[mid] <= tile) lo = mid; else hi = mid;
    }
    const int n = g.items[lo];
    const int local = tile - g.tile_off[lo];
    const int r = g.rank[n];
    const int Ng = g.shape.n_const + g.shape.n_rank * r;
    const int K = g.shape.k_const + g.shape.k_rank * r;
    const int ncol = (Ng + G_BN - 1) / G_BN;
    const int per_rt = ncol * g.shape.groups;
    const int rt = local / per_rt, rem = local % per_rt;
    const int grp = rem / ncol, ct = rem % ncol;
    const int row0 = g.node_off[n] + rt * G_BM;
    const int rows = min(G_BM, g.node_off[n + 1] - row0);
    const int col0 = ct * G_BN;
    const TW* W = reinterpret_cast<const TW*>(g.W[n]) + (size_t)grp * Ng * K;
    const TA* A = reinterpret_cast<const TA*>(g.A);
    const long acol = (long)grp * K;

    float acc[2][4];
#pragma unroll
    for (int i = 0; i < 2; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

    for (int k0 = 0; k0 < K; k0 += G_BK) {
      for (int idx = threadIdx.x; idx < G_BM * G_BK; idx += GG_THREADS) {
        const int i = idx / G_BK, kk = idx % G_BK;
        float v = 0.f;
        if (i < rows && k0 + kk < K) {
          const int grow = row0 + i;
          const long src = g.gather ? g.gather[grow] : grow;
          v = to_f32(A[src * g.lda + acol + k0 + kk]);
        }
        As[kk][i] = v;
      }
      for (int idx = threadIdx.x; idx < G_BN * G_BK; idx += GG_THREADS) {
        const int j = idx / G_BK, kk = idx % G_BK;
        float v = 0.f;
        if (col0 + j < Ng && k0 + kk < K) {
          const int c = col0 + j, kx = k0 + kk;
          const size_t wi = g.tiled ? ((((size_t)(c >> 6) * (K >> 6) + (kx >> 6)) * 64 + (c & 63)) * 64 + (kx & 63))
                                    : (size_t)c * K + kx;
          v = to_f32(W[wi]);
        }
        Ws[kk][j] = v;
      }
      __syncthreads();
#pragma unroll 8
      for (int kk = 0; kk < G_BK; ++kk) {
        const float a0 = As[kk][ty * 2], a1 = As[kk][ty * 2 + 1];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float w = Ws[kk][tx * 4 + j];
          acc[0][j] = fmaf(a0, w, acc[0][j]);
          acc[1][j] = fmaf(a1, w, acc[1][j]);
        }
      }
      __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int ri = ty * 2 + i;
      if (ri >= rows) continue;
      float* o = g.out + (size_t)(row0 + ri) * g.ldo + (size_t)grp * Ng + col0;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (col0 + tx * 4 + j < Ng) o[tx * 4 + j] = acc[i][j];
    }
  }
}

__device__ __forceinline__ float silu_f(float v) { return v / (1.f + expf(-v)); }
// the bf16 paths' SiLU: CUDA's fast exponential and division intrinsics (their
// error is far below the bf16 rounding of the operands)
__device__ __forceinline__ float silu_fast(float v) { return __fdividef(v, 1.f + __expf(-v)); }

// One CTA per token.  Its k selected experts' gated SwiGLU outputs,
//   a_s = g_s * silu(sum_l h_gate[row(s,l)]) * sum_l h_up[row(s,l)],
// are added, slot by slot in ascending order, into the z row of every node on
// the slot's path: z[(t,n)] = sum_{s : n in path(e_s)} a_s.  Each thread owns
// four columns; its per-row partial sums live in its own shared-memory slice.
constexpr int SW_T = 256;


template <typename TZ>
__device__ __forceinline__ void store4(TZ* p, float4 v);
template <>
__device__ __forceinline__ void store4<float>(float* p, float4 v) {
  *reinterpret_cast<float4*>(p) = v;
}
template <>
__device__ __forceinline__ void store4<__nv_bfloat16>(__nv_bfloat16* p, float4 v) {
  __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y), b = __floats2bfloat162_rn(v.z, v.w);
  uint2 u;
  u.x = *reinterpret_cast<uint32_t*>(&a);
  u.y = *reinterpret_cast<uint32_t*>(&b);
  *reinterpret_cast<uint2*>(p) = u;
}

template <typename TZ>
__global__ void __launch_bounds__(SW_T)
k_swiglu_aggregate(const int* __restrict__ topk_id, const float* __restrict__ topk_w,
                   const int* __restrict__ node_row, int T, int k, int D,
                   const float* __restrict__ h, int I, TZ* __restrict__ z) {
  pdl_wait();
  extern __shared__ float4 zacc[];  // [distinct rows][SW_T]
  __shared__ int rows[LX_MAX_K * LX_MAX_DEPTH], lrow[LX_MAX_K * LX_MAX_DEPTH];
  __shared__ int drow[LX_MAX_K * LX_MAX_DEPTH];
  __shared__ float gw[LX_MAX_K];
  __shared__ int nd_s;
  const int kD = k * D;
  for (int t = blockIdx.x; t < T; t += gridDim.x) {
    for (int j = threadIdx.x; j < kD; j += blockDim.x) rows[j] = node_row[(size_t)t * kD + j];
    for (int j = threadIdx.x; j < k; j += blockDim.x) gw[j] = topk_w[(size_t)t * k + j];
    __syncthreads();
    // distinct rows, numbered in order of first appearance (entry j owns the
    // number of first appearances before it)
    if (threadIdx.x < 32) {
      const int lane = threadIdx.x;
      int base = 0;
      for (int j0 = 0; j0 < kD; j0 += 32) {
        const int j = j0 + lane;
        const int r = j < kD ? rows[j] : -1;
        bool first = r >= 0;
        for (int q = 0; q < j && first; ++q) first = rows[q] != r;
        const uint32_t fm = __ballot_sync(0xffffffffu, first);
        if (first) {
          const int d = base + __popc(fm & ((1u << lane) - 1u));
          drow[d] = r;
        }
        base += __popc(fm);
      }
      if (lane == 0) nd_s = base;
    }
    __syncthreads();
    for (int j = threadIdx.x; j < kD; j += blockDim.x) {
      const int r = rows[j];
      int d = -1;
      if (r >= 0)
        for (int q = 0; q < nd_s; ++q)
          if (drow[q] == r) d = q;
      lrow[j] = d;
    }
    __syncthreads();
    const int nd = nd_s;
    for (int c0 = 0; c0 < I; c0 += 4 * SW_T) {
      const int i = c0 + 4 * threadIdx.x;
      if (i < I) {
        for (int d = 0; d < nd; ++d) zacc[d * SW_T + threadIdx.x] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
        for (int sl = 0; sl < k; ++sl) {
          float4 pg = make_float4(0.f, 0.f, 0.f, 0.f), pu = pg;
          for (int l = 0; l < D; ++l) {
            const int r = rows[sl * D + l];
            if (r < 0) continue;
            const float4 a = *reinterpret_cast<const float4*>(h + (size_t)r * 2 * I + i);
            const float4 b = *reinterpret_cast<const float4*>(h + (size_t)r * 2 * I + I + i);
            pg.x += a.x; pg.y += a.y; pg.z += a.z; pg.w += a.w;
            pu.x += b.x; pu.y += b.y; pu.z += b.z; pu.w += b.w;
          }
          const float g = gw[sl];
          const float4 act = make_float4(g * silu_f(pg.x) * pu.x, g * silu_f(pg.y) * pu.y,
                                         g * silu_f(pg.z) * pu.z, g * silu_f(pg.w) * pu.w);
          for (int l = 0; l < D; ++l) {
            const int d = lrow[sl * D + l];
            if (d < 0) continue;
            float4& acc = zacc[d * SW_T + threadIdx.x];
            acc.x += act.x; acc.y += act.y; acc.z += act.z; acc.w += act.w;
          }
        }
        for (int d = 0; d < nd; ++d) store4<TZ>(z + (size_t)drow[d] * I + i, zacc[d * SW_T + threadIdx.x]);
      }
    }
    __syncthreads();
  }
}

// y[t] = sum of ypart over t's distinct rows in ascending row (= node) order;
// each thread owns four columns and issues four rows' loads at a time.
template <typename TY>
__global__ void __launch_bounds__(256)
k_combine(const int* __restrict__ node_row, int k, int D, const float* __restrict__ ypart, int H,
          TY* __restrict__ y, int T) {
  pdl_wait();
  __shared__ int raw_s[LX_MAX_K * LX_MAX_DEPTH];
  __shared__ int rows_s[LX_MAX_K * LX_MAX_DEPTH];
  __shared__ int nrows_s;
  for (int t = blockIdx.x; t < T; t += gridDim.x) {
    for (int j = threadIdx.x; j < k * D; j += blockDim.x) raw_s[j] = node_row[(long)t * k * D + j];
    __syncthreads();
    // distinct rows in ascending order: each first occurrence takes the rank
    // of its value among the distinct values
    for (int j = threadIdx.x; j < k * D; j += blockDim.x) {
      const int r = raw_s[j];
      bool first = r >= 0;
      for (int q = 0; q < j && first; ++q) first = raw_s[q] != r;
      if (first) {
        int rank = 0;
        for (int q = 0; q < k * D; ++q) {
          const int v = raw_s[q];
          bool fq = v >= 0 && v < r;
          for (int u = 0; u < q && fq; ++u) fq = raw_s[u] != v;
          rank += fq;
        }
        rows_s[rank] = r;
      }
    }
    if (threadIdx.x < 32) {
      int cntd = 0;
      for (int j0 = 0; j0 < k * D; j0 += 32) {
        const int j = j0 + threadIdx.x;
        const int r = j < k * D ? raw_s[j] : -1;
        bool first = r >= 0;
        for (int q = 0; q < j && first; ++q) first = raw_s[q] != r;
        cntd += __popc(__ballot_sync(0xffffffffu, first));
      }
      if (threadIdx.x == 0) nrows_s = cntd;
    }
    __syncthreads();
    const int m = nrows_s;
    for (int c = 4 * threadIdx.x; c < H; c += 4 * blockDim.x) {
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      int q = 0;
      for (; q + 4 <= m; q += 4) {
        float4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u)
          v[u] = *reinterpret_cast<const float4*>(ypart + (size_t)rows_s[q + u] * H + c);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          acc.x += v[u].x; acc.y += v[u].y; acc.z += v[u].z; acc.w += v[u].w;
        }
      }
      for (; q < m; ++q) {
        const float4 v = *reinterpret_cast<const float4*>(ypart + (size_t)rows_s[q] * H + c);
        acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
      }
      store4<TY>(y + (size_t)t * H + c, acc);
    }
    __syncthreads();
  }
}

// ---------------------------------------------------------------------------
// Warp-per-token SwiGLU aggregation and combine (k <= 8, k * D <= 32).
//
// A warp reads the token's k * D path rows (node_row), finds its distinct rows
// with match/ballot/shuffle (no block barrier), and keeps them, in ascending
// order, in a per-warp shared-memory block with, for each distinct row, the
// bit mask of the top-k slots whose path passes through it.
// ---------------------------------------------------------------------------
constexpr int WT_WARPS = 8;
constexpr int WT_SLOTS = 8;

struct WarpRows {
  int rows[32];       // entry j = slot j / D, level j % D (-1: none)
  int lrow[32];       // entry j: index of its row among the distinct rows (-1: none)
  int drow[32];       // distinct rows, ascending
  unsigned dmask[32]; // slots whose path holds distinct row d
  float g[WT_SLOTS];
  int nd;
  unsigned anchor_rows;  // bit d: distinct row d belongs to an anchor
};

// v: entry `lane` of the token's node rows (-1 for lanes >= kD)
__device__ __forceinline__ void warp_token_rows(int v, int kD, int D, WarpRows& wr) {
  const int lane = threadIdx.x & 31;
  const int key = v >= 0 ? v : INT_MAX;
  const unsigned same = __match_any_sync(0xffffffffu, key);
  const bool first = key != INT_MAX && lane == __ffs(same) - 1;
  const unsigned fm = __ballot_sync(0xffffffffu, first);
  // rank of this entry's row among the distinct rows (the loop is warp-uniform)
  int rank = 0;
  for (unsigned b = fm; b; b &= b - 1) {
    const int q = __ffs(b) - 1;
    rank += __shfl_sync(0xffffffffu, key, q) < key;
  }
  if (lane < kD) {
    wr.rows[lane] = v;
    wr.lrow[lane] = key != INT_MAX ? rank : -1;
  }
  if (first) wr.drow[rank] = key;
  // entry j holds its path's anchor if it is the path's last valid level
  // (paths are stored from the expert's own node up to the anchor)
  const int v_next = __shfl_down_sync(0xffffffffu, v, 1);
  const bool anchor_entry = v >= 0 && (lane % D == D - 1 || lane + 1 >= kD || v_next < 0);
  const unsigned am = __ballot_sync(0xffffffffu, anchor_entry);
  unsigned mask = 0, anc = 0;
  for (int j = 0; j < kD; ++j) {
    const int rj = __shfl_sync(0xffffffffu, key != INT_MAX ? rank : -1, j);
    if (rj == lane) mask |= 1u << (j / D);
    if (rj >= 0 && ((am >> j) & 1u)) anc |= 1u << rj;
  }
  wr.dmask[lane] = mask;
  if (lane == 0) {
    wr.nd = __popc(fm);
    wr.anchor_rows = anc;
  }
  __syncwarp();
}

// CPL consecutive columns of one row (CPL = 1: one float per lane, for small
// batches, where every row load of a token can then be in flight at once;
// CPL = 4: one 16-byte load)
template <int CPL>
struct Cols {
  float v[CPL];
};
template <int CPL>
__device__ __forceinline__ Cols<CPL> ld_cols(const float* p) {
  Cols<CPL> r;
  if constexpr (CPL == 8) {
    const float4 f = __ldg(reinterpret_cast<const float4*>(p));
    const float4 g = __ldg(reinterpret_cast<const float4*>(p + 4));
    r.v[0] = f.x; r.v[1] = f.y; r.v[2] = f.z; r.v[3] = f.w;
    r.v[4] = g.x; r.v[5] = g.y; r.v[6] = g.z; r.v[7] = g.w;
  } else if constexpr (CPL == 4) {
    const float4 f = __ldg(reinterpret_cast<const float4*>(p));
    r.v[0] = f.x; r.v[1] = f.y; r.v[2] = f.z; r.v[3] = f.w;
  } else if constexpr (CPL == 2) {
    const float2 f = __ldg(reinterpret_cast<const float2*>(p));
    r.v[0] = f.x; r.v[1] = f.y;
  } else {
#pragma unroll
    for (int i = 0; i < CPL; ++i) r.v[i] = __ldg(p + i);
  }
  return r;
}
template <int CPL>
__device__ __forceinline__ Cols<CPL> ld_cols(const __nv_bfloat16* p) {
  Cols<CPL> r;
  if constexpr (CPL == 8) {
    const uint4 u = __ldg(reinterpret_cast<const uint4*>(p));
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      r.v[2 * i] = __uint_as_float(w[i] << 16);
      r.v[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
  } else if constexpr (CPL == 4) {
    const uint2 u = __ldg(reinterpret_cast<const uint2*>(p));
    r.v[0] = __uint_as_float(u.x << 16); r.v[1] = __uint_as_float(u.x & 0xFFFF0000u);
    r.v[2] = __uint_as_float(u.y << 16); r.v[3] = __uint_as_float(u.y & 0xFFFF0000u);
  } else if constexpr (CPL == 2) {
    const uint32_t u = __ldg(reinterpret_cast<const unsigned int*>(p));
    r.v[0] = __uint_as_float(u << 16); r.v[1] = __uint_as_float(u & 0xFFFF0000u);
  } else {
#pragma unroll
    for (int i = 0; i < CPL; ++i) r.v[i] = __bfloat162float(p[i]);
  }
  return r;
}
// CPL raw bf16 values (CPL = 4: one 8-byte load) and their widening
template <int CPL>
struct RawB {
  uint32_t w[(CPL + 1) / 2];
};
template <int CPL>
__device__ __forceinline__ RawB<CPL> ld_raw(const __nv_bfloat16* p) {
  RawB<CPL> r;
  if constexpr (CPL == 4) {
    const uint2 u = __ldg(reinterpret_cast<const uint2*>(p));
    r.w[0] = u.x;
    r.w[1] = u.y;
  } else if constexpr (CPL == 2) {
    r.w[0] = __ldg(reinterpret_cast<const unsigned int*>(p));
  } else {
    r.w[0] = (uint32_t)__ldg(reinterpret_cast<const unsigned short*>(p));
  }
  return r;
}
template <int CPL>
__device__ __forceinline__ void add_raw(Cols<CPL>& a, const RawB<CPL>& r, bool valid) {
  if constexpr (CPL == 4) {
    if (valid) {
      a.v[0] += __uint_as_float(r.w[0] << 16); a.v[1] += __uint_as_float(r.w[0] & 0xFFFF0000u);
      a.v[2] += __uint_as_float(r.w[1] << 16); a.v[3] += __uint_as_float(r.w[1] & 0xFFFF0000u);
    }
  } else if constexpr (CPL == 2) {
    if (valid) {
      a.v[0] += __uint_as_float(r.w[0] << 16); a.v[1] += __uint_as_float(r.w[0] & 0xFFFF0000u);
    }
  } else {
    if (valid) a.v[0] += __uint_as_float(r.w[0] << 16);
  }
}
template <typename T, int CPL>
__device__ __forceinline__ void st_cols(T* p, const Cols<CPL>& c) {
  if constexpr (CPL == 8 && std::is_same<T, __nv_bfloat16>::value) {
    uint4 u;
    uint32_t* w = reinterpret_cast<uint32_t*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const __nv_bfloat162 b = __floats2bfloat162_rn(c.v[2 * i], c.v[2 * i + 1]);
      w[i] = *reinterpret_cast<const uint32_t*>(&b);
    }
    *reinterpret_cast<uint4*>(p) = u;
  } else if constexpr (CPL == 8) {
    store4<T>(p, make_float4(c.v[0], c.v[1], c.v[2], c.v[3]));
    store4<T>(p + 4, make_float4(c.v[4], c.v[5], c.v[6], c.v[7]));
  } else if constexpr (CPL == 4) {
    store4<T>(p, make_float4(c.v[0], c.v[1], c.v[2], c.v[3]));
  } else if constexpr (CPL == 2 && std::is_same<T, __nv_bfloat16>::value) {
    *reinterpret_cast<__nv_bfloat162*>(p) = __floats2bfloat162_rn(c.v[0], c.v[1]);
  } else if constexpr (std::is_same<T, float>::value) {
#pragma unroll
    for (int i = 0; i < CPL; ++i) p[i] = c.v[i];
  } else {
#pragma unroll
    for (int i = 0; i < CPL; ++i) p[i] = __float2bfloat16_rn(c.v[i]);
  }
}
template <int CPL>
__device__ __forceinline__ void add_cols(Cols<CPL>& a, const Cols<CPL>& b) {
#pragma unroll
  for (int i = 0; i < CPL; ++i) a.v[i] += b.v[i];
}

template <typename TH, typename TZ, int D, bool SPLIT, int CPL>
__global__ void __launch_bounds__(WT_WARPS * 32, (sizeof(TH) == 2 && CPL >= 4 && D <= 2) ? 3 : 2)
k_swiglu_warp(const float* __restrict__ topk_w, const int* __restrict__ node_row, int T, int k,
              const TH* __restrict__ h, int I, TZ* __restrict__ z, int cols_per_item,
              const SplitParts hs) {
  extern __shared__ float zsm[];  // bf16 path: [warp][k slots][32 lanes * CPL] activations
  __shared__ WarpRows wrs[WT_WARPS];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  WarpRows& wr = wrs[warp];
  const int kD = k * D;
  const int per_tok = (I + cols_per_item - 1) / cols_per_item;
  const long items = (long)T * per_tok;
  long it = (long)blockIdx.x * WT_WARPS + warp;
  // The routing tables (node rows, gates) come from the routing and bucketing
  // kernels, at least two launches before this one: the first item's entries
  // are loaded before the wait for the preceding kernel.
  int v_pre = -1;
  float g_pre = 0.f;
  if (it < items) {
    const int t = (int)(it / per_tok);
    if (lane < kD) v_pre = node_row[(size_t)t * kD + lane];
    if (lane < k) g_pre = topk_w[(size_t)t * k + lane];
  }
  pdl_wait();
  for (bool first = true; it < items; it += (long)gridDim.x * WT_WARPS, first = false) {
    const int t = (int)(it / per_tok);
    const int c_begin = (int)(it % per_tok) * cols_per_item;
    const int c_end = min(I, c_begin + cols_per_item);
    warp_token_rows(first ? v_pre : (lane < kD ? node_row[(size_t)t * kD + lane] : -1), kD, D, wr);
    if (lane < k) wr.g[lane] = first ? g_pre : topk_w[(size_t)t * k + lane];
    __syncwarp();
    const int nd = wr.nd;
    for (int c = c_begin + CPL * lane; c < c_end; c += 32 * CPL) {
      Cols<CPL> act[WT_SLOTS];
      if constexpr (sizeof(TH) == 2) {
        // bf16 rows, in batches of SG slots: every path-row load of a batch
        // first (rows past a path's end are not read), so that they are in
        // flight at once; each slot's act then goes to this lane's slice of
        // the warp's shared block
        float* as = zsm + (size_t)warp * k * 32 * CPL;
        constexpr int NS = SPLIT ? LX_STREAM_MAX_SPLIT : 1;
        constexpr int SG = (CPL >= 4 && D >= 2) ? 4 : WT_SLOTS;  // bounds the live registers
#pragma unroll
        for (int s0 = 0; s0 < WT_SLOTS; s0 += SG) {
          if (s0 >= k) break;
          RawB<CPL> rg[SG][D], ru[SG][D];
          bool val[SG][D], anc[SG][D];
          Cols<CPL> sg[SG][NS], su[SG][NS];  // the anchor row's split-K partials
#pragma unroll
          for (int j = 0; j < SG; ++j) {
            const int sl = s0 + j;
            int ra = 0;
#pragma unroll
            for (int l = 0; l < D; ++l) {
              const int r = sl < k ? wr.rows[sl * D + l] : -1;
              const int rn = (sl < k && l + 1 < D) ? wr.rows[sl * D + l + 1] : -1;
              val[j][l] = r >= 0;
              anc[j][l] = SPLIT && r >= 0 && rn < 0;  // the path's anchor row
              if (anc[j][l]) ra = r;
              if (r >= 0 && !anc[j][l]) {
                const __nv_bfloat16* hp =
                    reinterpret_cast<const __nv_bfloat16*>(h) + (size_t)r * 2 * I + c;
                rg[j][l] = ld_raw<CPL>(hp);
                ru[j][l] = ld_raw<CPL>(hp + I);
              }
            }
            if constexpr (SPLIT) {
#pragma unroll
              for (int sp = 0; sp < NS; ++sp) {
                const float* hp2 = hs.part + (long)(sp < hs.splits ? sp : 0) * hs.stride +
                                   (size_t)ra * 2 * I + c;
                sg[j][sp] = ld_cols<CPL>(hp2);
                su[j][sp] = ld_cols<CPL>(hp2 + I);
              }
            }
          }
#pragma unroll
          for (int j = 0; j < SG; ++j) {
            const int sl = s0 + j;
            Cols<CPL> pg, pu;
#pragma unroll
            for (int i = 0; i < CPL; ++i) pg.v[i] = pu.v[i] = 0.f;
#pragma unroll
            for (int l = 0; l < D; ++l) {  // path order: the expert's node up to its anchor
              if (anc[j][l]) {
                // anchor row: its split-K partials (not h), in split order
#pragma unroll
                for (int sp = 0; sp < NS; ++sp) {
                  if (sp < hs.splits) {
                    add_cols(pg, sg[j][sp]);
                    add_cols(pu, su[j][sp]);
                  }
                }
              } else {
                add_raw(pg, rg[j][l], val[j][l]);
                add_raw(pu, ru[j][l], val[j][l]);
              }
            }
            if (sl < k) {
              const float g = wr.g[sl];
#pragma unroll
              for (int i = 0; i < CPL; ++i)
                as[(sl * 32 + lane) * CPL + i] = g * silu_fast(pg.v[i]) * pu.v[i];
            }
          }
        }
        // z: every distinct row's z is the sum of the acts of the slots whose
        // path holds it (the row's slot mask), slots ascending
        for (int d = 0; d < nd; ++d) {
          Cols<CPL> zc;
#pragma unroll
          for (int i = 0; i < CPL; ++i) zc.v[i] = 0.f;
          for (unsigned m = wr.dmask[d]; m; m &= m - 1) {
            const int sl = __ffs(m) - 1;
#pragma unroll
            for (int i = 0; i < CPL; ++i) zc.v[i] += as[(sl * 32 + lane) * CPL + i];
          }
          st_cols<TZ, CPL>(z + (size_t)wr.drow[d] * I + c, zc);
        }
        continue;
      } else {
#pragma unroll
      for (int sl = 0; sl < WT_SLOTS; ++sl) {
#pragma unroll
        for (int i = 0; i < CPL; ++i) act[sl].v[i] = 0.f;
        if (sl < k) {
          Cols<CPL> pg, pu;
#pragma unroll
          for (int i = 0; i < CPL; ++i) pg.v[i] = pu.v[i] = 0.f;
#pragma unroll
          for (int l = 0; l < D; ++l) {  // path order: the expert's node up to its anchor
            const int r = wr.rows[sl * D + l];
            if (r >= 0) {
              if (SPLIT && (l + 1 == D || wr.rows[sl * D + l + 1] < 0)) {
                // anchor row: its split-K partials, in split order
#pragma unroll
                for (int sp = 0; sp < LX_STREAM_MAX_SPLIT; ++sp) {
                  if (sp < hs.splits) {
                    const float* hp = hs.part + sp * hs.stride + (size_t)r * 2 * I;
                    add_cols(pg, ld_cols<CPL>(hp + c));
                    add_cols(pu, ld_cols<CPL>(hp + I + c));
                  }
                }
              } else {
                add_cols(pg, ld_cols<CPL>(h + (size_t)r * 2 * I + c));
                add_cols(pu, ld_cols<CPL>(h + (size_t)r * 2 * I + I + c));
              }
            }
          }
          const float g = wr.g[sl];
#pragma unroll
          for (int i = 0; i < CPL; ++i) act[sl].v[i] = g * silu_f(pg.v[i]) * pu.v[i];
        }
      }
      }
      for (int d = 0; d < nd; ++d) {
        const unsigned m = wr.dmask[d];
        Cols<CPL> acc;
#pragma unroll
        for (int i = 0; i < CPL; ++i) acc.v[i] = 0.f;
#pragma unroll
        for (int sl = 0; sl < WT_SLOTS; ++sl)  // slots ascending
          if ((m >> sl) & 1u) add_cols(acc, act[sl]);
        st_cols<TZ, CPL>(z + (size_t)wr.drow[d] * I + c, acc);
      }
    }
    __syncwarp();
  }
}

// y[t] = sum of ypart over t's distinct rows in ascending row order (an
// anchor row split into K ranges contributes its partials in split order)
template <typename TP, typename TY, int CPL, bool SPLIT, bool ANCHORS = false>
__global__ void __launch_bounds__(WT_WARPS * 32, 2)
k_combine_warp(const int* __restrict__ node_row, int k, int D, const TP* __restrict__ ypart,
               int H, TY* __restrict__ y, int T, int cols_per_item, const SplitParts ys) {
  __shared__ WarpRows wrs[WT_WARPS];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  WarpRows& wr = wrs[warp];
  const int kD = k * D;
  const int per_tok = (H + cols_per_item - 1) / cols_per_item;
  const long items = (long)T * per_tok;
  long it = (long)blockIdx.x * WT_WARPS + warp;
  // node rows come from the bucketing, several launches before this one: the
  // first item's entries are loaded before the wait for the preceding kernel
  int v_pre = -1;
  if (it < items && lane < kD) v_pre = node_row[(size_t)(it / per_tok) * kD + lane];
  pdl_wait();
  for (bool first = true; it < items; it += (long)gridDim.x * WT_WARPS, first = false) {
    const int t = (int)(it / per_tok);
    const int c_begin = (int)(it % per_tok) * cols_per_item;
    const int c_end = min(H, c_begin + cols_per_item);
    int v_cur;
    if constexpr (ANCHORS) {
      // the next item's node rows are requested now, ahead of their use
      v_cur = v_pre;
      const long itn = it + (long)gridDim.x * WT_WARPS;
      v_pre = (itn < items && lane < kD) ? node_row[(size_t)(itn / per_tok) * kD + lane] : -1;
    } else {
      v_cur = first ? v_pre : (lane < kD ? node_row[(size_t)t * kD + lane] : -1);
    }
    warp_token_rows(v_cur, kD, D, wr);
    const int nd = wr.nd;
    if constexpr (ANCHORS && !SPLIT && CPL == 8 && sizeof(TP) == 2) {
      {
        // only the anchor rows (their down tiles already hold the members'
        // corrections), ascending; four column passes' 16-byte loads of a
        // batch of four rows in flight at once, each column summed in row order
        for (int c0 = c_begin + CPL * lane; c0 < c_end; c0 += 4 * 32 * CPL) {
          Cols<CPL> acc[4];
#pragma unroll
          for (int u = 0; u < 4; ++u)
#pragma unroll
            for (int i = 0; i < CPL; ++i) acc[u].v[i] = 0.f;
          for (unsigned am = wr.anchor_rows; am;) {
            int rq[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              rq[q] = -1;
              if (am) {
                rq[q] = wr.drow[__ffs(am) - 1];
                am &= am - 1u;
              }
            }
            uint4 v[4][4];
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
              for (int q = 0; q < 4; ++q)
                if (rq[q] >= 0 && c0 + u * 32 * CPL < c_end)
                  v[u][q] = __ldg(reinterpret_cast<const uint4*>(ypart + (size_t)rq[q] * H + c0 +
                                                                 u * 32 * CPL));
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
              for (int q = 0; q < 4; ++q)
                if (rq[q] >= 0 && c0 + u * 32 * CPL < c_end) {
                  const uint32_t w4[4] = {v[u][q].x, v[u][q].y, v[u][q].z, v[u][q].w};
#pragma unroll
                  for (int i = 0; i < 4; ++i) {
                    acc[u].v[2 * i] += __uint_as_float(w4[i] << 16);
                    acc[u].v[2 * i + 1] += __uint_as_float(w4[i] & 0xFFFF0000u);
                  }
                }
          }
#pragma unroll
          for (int u = 0; u < 4; ++u)
            if (c0 + u * 32 * CPL < c_end) st_cols<TY, CPL>(y + (size_t)t * H + c0 + u * 32 * CPL, acc[u]);
        }
        __syncwarp();
        continue;
      }
    }
    for (int c = c_begin + CPL * lane; c < c_end; c += 32 * CPL) {
      Cols<CPL> acc;
#pragma unroll
      for (int i = 0; i < CPL; ++i) acc.v[i] = 0.f;
      if constexpr (SPLIT) {
        // four distinct rows per batch, every load of the batch first: an
        // anchor row contributes its split partials (fp32, split order), any
        // other row its ypart row
        constexpr int NS = LX_STREAM_MAX_SPLIT;
        for (int q0 = 0; q0 < nd; q0 += 4) {
          Cols<CPL> v[4][NS];
          bool isa[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int d = q0 + u < nd ? q0 + u : q0;
            const size_t ro = (size_t)wr.drow[d] * H + c;
            isa[u] = q0 + u < nd && ((wr.anchor_rows >> d) & 1u);
            if (isa[u]) {
#pragma unroll
              for (int sp = 0; sp < NS; ++sp)
                v[u][sp] = ld_cols<CPL>(ys.part + (long)(sp < ys.splits ? sp : 0) * ys.stride + ro);
            } else {
              v[u][0] = ld_cols<CPL>(ypart + ro);
            }
          }
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            if (q0 + u >= nd) break;
            if (isa[u]) {
#pragma unroll
              for (int sp = 0; sp < NS; ++sp)
                if (sp < ys.splits) add_cols(acc, v[u][sp]);
            } else {
              add_cols(acc, v[u][0]);
            }
          }
        }
      } else {
        int q = 0;
        for (; q + 8 <= nd; q += 8) {
          Cols<CPL> v[8];
#pragma unroll
          for (int u = 0; u < 8; ++u) v[u] = ld_cols<CPL>(ypart + (size_t)wr.drow[q + u] * H + c);
#pragma unroll
          for (int u = 0; u < 8; ++u) add_cols(acc, v[u]);
        }
        for (; q < nd; ++q) add_cols(acc, ld_cols<CPL>(ypart + (size_t)wr.drow[q] * H + c));
      }
      st_cols<TY, CPL>(y + (size_t)t * H + c, acc);
    }
    __syncwarp();
  }
}

}  // namespace

bool warp_kernels_fit(const lx_layer* L, int k) {
  return k <= WT_SLOTS && k * L->max_depth <= 32 && L->I % 4 == 0 && L->H % 8 == 0;
}

// Columns per warp work item: whole rows when the batch alone fills the GPU
// (the distinct-row search then runs once per token), else blocks of `unit`
// columns so that a small batch still spreads over the SMs.
static int warp_item_cols(const lx_layer* L, int T, int width, int unit) {
  const long want = (long)L->num_sms * 4 * WT_WARPS;
  const int blocks = (width + unit - 1) / unit;
  int per = blocks;
  while (per > 1 && (long)T * ((blocks + per - 1) / per) < want) per = (per + 1) / 2;
  return per * unit;
}

static int warp_grid(const lx_layer* L, int T, int width, int cols) {
  const long items = (long)T * ((width + cols - 1) / cols);
  return (int)std::min<long>((items + WT_WARPS - 1) / WT_WARPS, (long)L->num_sms * 4);
}

// One float per lane for batches too small to fill the GPU with 128-column items.
static bool narrow_cols(const lx_layer* L, int T, int width) {
  return (long)T * ((width + 127) / 128) < (long)L->num_sms * 4 * WT_WARPS;
}

template <typename TH, typename TZ, int D, int CPL>
static void launch_swiglu_c(lx_layer* L, int T, int k, const TH* h, TZ* z, cudaStream_t s,
                            const SplitParts& hs) {
  Workspace& w = L->ws;
  const int cols = warp_item_cols(L, T, L->I, 32 * CPL);
  const int grid = warp_grid(L, T, L->I, cols);
  const size_t zs = sizeof(TH) == 2 ? (size_t)WT_WARPS * k * 32 * CPL * 4 : 0;
  if (zs > 0) {  // the accumulators plus the static rows may pass the 48 KB default
    static bool done_s[64] = {}, done_n[64] = {};
    if constexpr (CPL == 1) {
      if (hs.splits > 1)
        (void)smem_cap_once((const void*)k_swiglu_warp<TH, TZ, D, true, CPL>, 128 * 1024,
                            L->device, done_s);
    }
    (void)smem_cap_once((const void*)k_swiglu_warp<TH, TZ, D, false, CPL>, 128 * 1024, L->device,
                        done_n);
  }
  if constexpr (CPL == 1) {
    if (hs.splits > 1) {
      launch_k(L, k_swiglu_warp<TH, TZ, D, true, CPL>, grid, WT_WARPS * 32, zs, s, w.topk_w,
               w.node_row, T, k, h, L->I, z, cols, hs);
      return;
    }
  }
  launch_k(L, k_swiglu_warp<TH, TZ, D, false, CPL>, grid, WT_WARPS * 32, zs, s, w.topk_w,
           w.node_row, T, k, h, L->I, z, cols, hs);
}

template <typename TH, typename TZ, int D>
static void launch_swiglu_d(lx_layer* L, int T, int k, const TH* h, TZ* z, cudaStream_t s,
                            const SplitParts& hs) {
  // split partials (small batches only) take the one-column-per-lane form
  // (measured on GB300: four columns per lane beat two for large batches)
  if (narrow_cols(L, T, L->I) || hs.splits > 1)
    launch_swiglu_c<TH, TZ, D, 1>(L, T, k, h, z, s, hs);
  else
    launch_swiglu_c<TH, TZ, D, 4>(L, T, k, h, z, s, hs);
}

template <typename TH, typename TZ>
static void launch_swiglu_warp(lx_layer* L, int T, int k, const TH* h, TZ* z, cudaStream_t s,
                               const SplitParts& hs) {
  switch (L->max_depth) {
    case 1: launch_swiglu_d<TH, TZ, 1>(L, T, k, h, z, s, hs); break;
    case 2: launch_swiglu_d<TH, TZ, 2>(L, T, k, h, z, s, hs); break;
    case 3: launch_swiglu_d<TH, TZ, 3>(L, T, k, h, z, s, hs); break;
    default: launch_swiglu_d<TH, TZ, 4>(L, T, k, h, z, s, hs); break;
  }
}

// (the combine reads few rows per token: 16-byte columns measured faster at
// every batch size)
template <typename TP, typename TY>
static void launch_combine_warp(lx_layer* L, int T, int k, const TP* ypart, TY* y, cudaStream_t s,
                                const SplitParts& ys, bool anchors_only = false) {
  Workspace& w = L->ws;
  if (ys.splits > 1) {
    const int cols = warp_item_cols(L, T, L->H, 128);
    const int grid = warp_grid(L, T, L->H, cols);
    launch_k(L, k_combine_warp<TP, TY, 4, true>, grid, WT_WARPS * 32, 0, s, w.node_row, k,
             L->max_depth, ypart, L->H, y, T, cols, ys);
    return;
  }
  // eight columns per lane (16-byte bf16 loads): half the per-element address
  // and loop instructions of four (measured faster at decode and prefill)
  const int cols = warp_item_cols(L, T, L->H, 256);
  const int grid = warp_grid(L, T, L->H, cols);
  if (anchors_only && sizeof(TP) == 2) {
    launch_k(L, k_combine_warp<TP, TY, 8, false, true>, grid, WT_WARPS * 32, 0, s, w.node_row, k,
             L->max_depth, ypart, L->H, y, T, cols, ys);
    return;
  }
  launch_k(L, k_combine_warp<TP, TY, 8, false>, grid, WT_WARPS * 32, 0, s, w.node_row, k,
           L->max_depth, ypart, L->H, y, T, cols, ys);
}

lx_status launch_swiglu(lx_layer* L, int T, int k, bool bf16, cudaStream_t s, SplitParts hs) {
  Workspace& w = L->ws;
  ProfScope ps(L, s, bf16 ? "swiglu" : "generic_swiglu");
  if (warp_kernels_fit(L, k)) {
    if (bf16)
      launch_swiglu_warp(L, T, k, w.hb, w.zb, s, hs);
    else
      launch_swiglu_warp(L, T, k, w.h, w.z, s, hs);
    LX_CUDA(cudaGetLastError());
    return LX_OK;
  }
  // large k or deep paths: the block-per-token form (generic path only)
  if (bf16 || hs.splits > 1) return fail(LX_ERR_STATE, "bf16 SwiGLU needs k <= 8, k * depth <= 32");
  const int grid = std::min(T, L->num_sms * 8);
  const size_t smem = sizeof(float4) * SW_T * k * L->max_depth;
  static bool done_f[64] = {};
  LX_CUDA(smem_cap_once((const void*)k_swiglu_aggregate<float>, 200 * 1024, L->device, done_f));
  launch_k(L, k_swiglu_aggregate<float>, grid, SW_T, smem, s, w.topk_id, w.topk_w, w.node_row, T,
           k, L->max_depth, w.h, L->I, w.z);
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

lx_status launch_combine(lx_layer* L, int T, int k, void* y, bool bf16, cudaStream_t s,
                         SplitParts ys, bool anchors_only) {
  Workspace& w = L->ws;
  ProfScope ps(L, s, "combine");
  if (anchors_only && !(bf16 && ys.splits <= 1 && warp_kernels_fit(L, k)))
    return fail(LX_ERR_STATE, "anchor-row combine needs the bf16 warp form");
  if (warp_kernels_fit(L, k)) {
    if (bf16)
      launch_combine_warp(L, T, k, L->ws.yb, static_cast<__nv_bfloat16*>(y), s, ys, anchors_only);
    else if (L->dtype == LX_BF16)
      launch_combine_warp(L, T, k, L->ws.ypart, static_cast<__nv_bfloat16*>(y), s, ys);
    else
      launch_combine_warp(L, T, k, L->ws.ypart, static_cast<float*>(y), s, ys);
    LX_CUDA(cudaGetLastError());
    return LX_OK;
  }
  if (bf16 || ys.splits > 1) return fail(LX_ERR_STATE, "bf16 combine needs k <= 8, k * depth <= 32");
  const int grid = std::min(T, L->num_sms * 8);
  if (L->dtype == LX_BF16)
    launch_k(L, k_combine<__nv_bfloat16>, grid, 256, 0, s, w.node_row, k, L->max_depth, w.ypart, L->H,
                                                  (__nv_bfloat16*)y, T);
  else
    launch_k(L, k_combine<float>, grid, 256, 0, s, w.node_row, k, L->max_depth, w.ypart, L->H, (float*)y, T);
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

namespace {

template <typename TA, typename TW, int op>
lx_status run_gemm(lx_layer* L, const void* A, long lda, const int* gather,
                   const void* const* W, float* out, long ldo, cudaStream_t s, const char* name) {
  const OpShape sh = op_shape(L, op);
  GemmArgs g;
  g.items = sh.on_anchors ? L->d_anchors : L->d_corrs;
  g.n_items = sh.on_anchors ? L->n_anchor : L->n_corr;
  if (g.n_items == 0) return LX_OK;
  g.tile_off = L->ws.tile_off + op * (op_max_items(L) + 1);
  g.node_off = L->ws.key_off;
  g.gather = gather;
  g.A = A;
  g.lda = lda;
  g.W = W;
  g.rank = L->d_rank;
  g.shape = sh;
  g.out = out;
  g.ldo = ldo;
  g.tiled = L->tiled ? 1 : 0;
  ProfScope ps(L, s, name);
  launch_k(L, k_grouped_gemm<TA, TW, op>, L->num_sms * 4, GG_THREADS, 0, s, g);
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

template <typename TX>
lx_status generic_impl(lx_layer* L, const void* x, int T, int k, void* y, cudaStream_t s) {
  Workspace& w = L->ws;
  const long H = L->H, I = L->I, rmax = std::max(1, L->max_rank);
  const int D = L->max_depth;
  // x-side products
  LX_TRY((run_gemm<TX, TX, OP_UP_ANCHOR>(L, x, H, w.node_tok, (const void* const*)L->d_w_up,
                           w.h, 2 * I, s, "generic_up_anchor")));
  LX_TRY((run_gemm<TX, TX, OP_UP_V>(L, x, H, w.node_tok, (const void* const*)L->d_w_up, w.P,
                           2 * rmax, s, "generic_up_V")));
  LX_TRY((run_gemm<float, TX, OP_UP_U>(L, w.P, 2 * rmax, nullptr,
                              (const void* const*)L->d_w_upU, w.h, 2 * I, s, "generic_up_U")));
  LX_TRY(launch_swiglu(L, T, k, false, s));
  // z-side products
  LX_TRY((run_gemm<float, TX, OP_DN_ANCHOR>(L, w.z, I, nullptr, (const void* const*)L->d_w_dn,
                              w.ypart, H, s, "generic_dn_anchor")));
  LX_TRY((run_gemm<float, TX, OP_DN_V>(L, w.z, I, nullptr, (const void* const*)L->d_w_dn, w.Q,
                              rmax, s, "generic_dn_V")));
  LX_TRY((run_gemm<float, TX, OP_DN_U>(L, w.Q, rmax, nullptr, (const void* const*)L->d_w_dnU,
                              w.ypart, H, s, "generic_dn_U")));
  LX_TRY(launch_combine(L, T, k, y, false, s));
  return LX_OK;
}

}  // namespace

lx_status launch_generic_experts(lx_layer* L, const void* x, int T, int k, void* y,
                                 cudaStream_t s) {
  if (L->dtype == LX_BF16) return generic_impl<__nv_bfloat16>(L, x, T, k, y, s);
  return generic_impl<float>(L, x, T, k, y, s);
}

}  // namespace lx
