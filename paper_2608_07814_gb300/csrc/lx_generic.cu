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

#include "lx_internal.cuh"

namespace lx {

namespace {

constexpr int GG_THREADS = 256;

// OPK only names the instantiation (one kernel symbol per op in profiles)
template <typename TA, typename TW, int OPK>
__global__ void __launch_bounds__(GG_THREADS)
k_grouped_gemm(GemmArgs g) {
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
        if (col0 + j < Ng && k0 + kk < K) v = to_f32(W[(size_t)(col0 + j) * K + k0 + kk]);
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

// z[row] for every (token, node) row
template <typename TZ>
__global__ void k_swiglu_aggregate(const int* __restrict__ key_off, int N,
                                   const int* __restrict__ node_tok,
                                   const int* __restrict__ row_node,
                                   const int* __restrict__ topk_id,
                                   const float* __restrict__ topk_w,
                                   const int* __restrict__ node_row, int k, int D, int E,
                                   const int* __restrict__ paths, const int* __restrict__ path_len,
                                   const float* __restrict__ h, int I, TZ* __restrict__ z) {
  const int R = key_off[N];
  for (int row = blockIdx.x; row < R; row += gridDim.x) {
    const int t = node_tok[row];
    const int n = row_node[row];
    for (int i = threadIdx.x; i < I; i += blockDim.x) {
      float acc = 0.f;
      for (int s = 0; s < k; ++s) {
        const long a = (long)t * k + s;
        const int e = topk_id[a];
        if (e < 0 || e >= E) continue;
        const int len = path_len[e];
        bool on_path = false;
        for (int l = 0; l < len; ++l) on_path |= paths[e * LX_MAX_DEPTH + l] == n;
        if (!on_path) continue;
        float pg = 0.f, pu = 0.f;
        for (int l = 0; l < len; ++l) {
          const int rr = node_row[a * D + l];
          if (rr < 0) continue;
          pg += h[(size_t)rr * 2 * I + i];
          pu += h[(size_t)rr * 2 * I + I + i];
        }
        acc = fmaf(topk_w[a], silu_f(pg) * pu, acc);
      }
      z[(size_t)row * I + i] = from_f32<TZ>(acc);
    }
  }
}

// y[t] = sum of ypart over t's distinct rows, ascending
template <typename TY>
__global__ void k_combine(const int* __restrict__ node_row, int k, int D,
                          const float* __restrict__ ypart, int H, TY* __restrict__ y, int T) {
  __shared__ int rows_s[LX_MAX_K * LX_MAX_DEPTH];
  __shared__ int nrows_s;
  for (int t = blockIdx.x; t < T; t += gridDim.x) {
    if (threadIdx.x == 0) {
      int m = 0;
      for (int j = 0; j < k * D; ++j) {
        const int r = node_row[(long)t * k * D + j];
        if (r < 0) continue;
        bool dup = false;
        for (int q = 0; q < m; ++q) dup |= rows_s[q] == r;
        if (dup) continue;
        int p = m++;  // insertion sort, ascending
        while (p > 0 && rows_s[p - 1] > r) { rows_s[p] = rows_s[p - 1]; --p; }
        rows_s[p] = r;
      }
      nrows_s = m;
    }
    __syncthreads();
    const int m = nrows_s;
    for (int c = threadIdx.x; c < H; c += blockDim.x) {
      float acc = 0.f;
      for (int q = 0; q < m; ++q) acc += ypart[(size_t)rows_s[q] * H + c];
      y[(size_t)t * H + c] = from_f32<TY>(acc);
    }
    __syncthreads();
  }
}

}  // namespace

lx_status launch_swiglu(lx_layer* L, int k, void* z, bool z_bf16, cudaStream_t s) {
  Workspace& w = L->ws;
  ProfScope ps(L, s, z_bf16 ? "swiglu" : "generic_swiglu");
  const dim3 grid(L->num_sms * 8);
  if (z_bf16)
    k_swiglu_aggregate<__nv_bfloat16><<<grid, 256, 0, s>>>(
        w.key_off, L->N, w.node_tok, w.row_node, w.topk_id, w.topk_w, w.node_row, k,
        L->max_depth, L->E, L->d_paths, L->d_path_len, w.h, L->I, (__nv_bfloat16*)z);
  else
    k_swiglu_aggregate<float><<<grid, 256, 0, s>>>(
        w.key_off, L->N, w.node_tok, w.row_node, w.topk_id, w.topk_w, w.node_row, k,
        L->max_depth, L->E, L->d_paths, L->d_path_len, w.h, L->I, (float*)z);
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

lx_status launch_combine(lx_layer* L, int T, int k, void* y, cudaStream_t s) {
  Workspace& w = L->ws;
  ProfScope ps(L, s, "combine");
  const int grid = std::min(T, L->num_sms * 8);
  if (L->dtype == LX_BF16)
    k_combine<__nv_bfloat16><<<grid, 256, 0, s>>>(w.node_row, k, L->max_depth, w.ypart, L->H,
                                                  (__nv_bfloat16*)y, T);
  else
    k_combine<float><<<grid, 256, 0, s>>>(w.node_row, k, L->max_depth, w.ypart, L->H, (float*)y, T);
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
  ProfScope ps(L, s, name);
  k_grouped_gemm<TA, TW, op><<<L->num_sms * 4, GG_THREADS, 0, s>>>(g);
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
  LX_TRY(launch_swiglu(L, k, w.z, false, s));
  // z-side products
  LX_TRY((run_gemm<float, TX, OP_DN_ANCHOR>(L, w.z, I, nullptr, (const void* const*)L->d_w_dn,
                              w.ypart, H, s, "generic_dn_anchor")));
  LX_TRY((run_gemm<float, TX, OP_DN_V>(L, w.z, I, nullptr, (const void* const*)L->d_w_dn, w.Q,
                              rmax, s, "generic_dn_V")));
  LX_TRY((run_gemm<float, TX, OP_DN_U>(L, w.Q, rmax, nullptr, (const void* const*)L->d_w_dnU,
                              w.ypart, H, s, "generic_dn_U")));
  LX_TRY(launch_combine(L, T, k, y, s));
  return LX_OK;
}

}  // namespace

lx_status launch_generic_experts(lx_layer* L, const void* x, int T, int k, void* y,
                                 cudaStream_t s) {
  if (L->dtype == LX_BF16) return generic_impl<__nv_bfloat16>(L, x, T, k, y, s);
  return generic_impl<float>(L, x, T, k, y, s);
}

}  // namespace lx
