// Bucketing: per node the ascending list of tokens whose selected experts' root
// paths contain the node (the (token, node) pairs whose products the amortised
// forward computes once, Sec. 5.1), per assignment and path level the row of
// that pair, and per expert its assignments in token order.
//
// Keys are the N nodes followed by the E experts.  A byte matrix marks[key][t]
// records which (key, token) pairs occur; one CTA per key turns its row into
// exclusive ranks with a block scan (so the order inside a bucket is the token
// order, with no atomics); a single CTA scans the per-key counts into offsets
// and builds the tile plans of the grouped GEMMs; a last pass scatters.
// Everything is deterministic.
#include <mutex>

#include "lx_internal.cuh"

namespace lx {

namespace {

constexpr int SCAN_THREADS = 512;

__global__ void k_mark(const int* __restrict__ topk_id, int T, int k, int N, int E, long Tp,
                       const int* __restrict__ paths, const int* __restrict__ path_len,
                       uint8_t* __restrict__ marks) {
  pdl_wait();
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= T) return;
  for (int s = 0; s < k; ++s) {
    const int e = topk_id[(size_t)t * k + s];
    if (e < 0 || e >= E) continue;  // invalid ids are ignored
    marks[(size_t)(N + e) * Tp + t] = 1;
    const int len = path_len[e];
    for (int l = 0; l < len; ++l) marks[(size_t)paths[e * LX_MAX_DEPTH + l] * Tp + t] = 1;
  }
}

// block-wide exclusive scan of one int per thread; returns the block total
__device__ int block_excl_scan(int v, int* total) {
  __shared__ int warp_sums[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int incl = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int o = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += o;
  }
  if (lane == 31) warp_sums[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int ws = lane < nw ? warp_sums[lane] : 0;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int o = __shfl_up_sync(0xffffffffu, ws, off);
      if (lane >= off) ws += o;
    }
    if (lane < nw) warp_sums[lane] = ws;  // inclusive
  }
  __syncthreads();
  const int warp_base = warp > 0 ? warp_sums[warp - 1] : 0;
  *total = warp_sums[nw - 1];
  __syncthreads();
  return warp_base + incl - v;
}

__global__ void __launch_bounds__(SCAN_THREADS)
k_key_scan(const uint8_t* __restrict__ marks, int T, long Tp, int* __restrict__ rank_in,
           int* __restrict__ key_cnt) {
  pdl_wait();
  const int key = blockIdx.x;
  const uint8_t* m = marks + (size_t)key * Tp;
  int* r = rank_in + (size_t)key * Tp;
  int running = 0;
  for (int base = 0; base < T; base += blockDim.x * 4) {
    const int i0 = base + threadIdx.x * 4;
    int v[4], c = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      v[j] = (i0 + j < T) ? m[i0 + j] : 0;
      c += v[j];
    }
    int total;
    int run = running + block_excl_scan(c, &total);
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (v[j]) r[i0 + j] = run++;
    running += total;
  }
  if (threadIdx.x == 0) key_cnt[key] = running;
}

struct PlanArgs {
  const int* items[N_PLANS];
  int n_items[N_PLANS];
  OpShape shape[N_PLANS];
  int bm[N_PLANS], bn[N_PLANS];  // token rows and output columns per tile
  int n_plans;
  int first;                      // plan p fills tile-plan slot first + p
};

// tiles of one node in one plan
__device__ __forceinline__ int plan_tiles(const PlanArgs& pa, int p, int r, int rows) {
  const OpShape sh = pa.shape[p];
  const int Ng = sh.n_const + sh.n_rank * r;
  const int ncol = (Ng + pa.bn[p] - 1) / pa.bn[p];
  return ((rows + pa.bm[p] - 1) / pa.bm[p]) * sh.groups * ncol;
}



// Work items of the streaming launches: one (node, token block) pair per
// `blk` rows of every active node's bucket, anchors then corrections, in
// node-table order, packed as node * STREAM_DEP_TB + block; and zeroed tile
// counters.  blk = 0 (batches the streaming kernels do not take) publishes
// empty lists.  One CTA; warps 0 and 1 each compact one list.
__device__ void publish_active(const int* cnt, const int* anchors, int n_anchor,
                               const int* corrs, int n_corr, int blk, int* act, int* act_n,
                               int* sctr, int n_sctr) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (warp < 2) {
    const int* list = warp == 0 ? anchors : corrs;
    const int n = warp == 0 ? n_anchor : n_corr;
    int* out = act + (warp == 0 ? 0 : n_anchor * STREAM_DEP_TB);
    int base = 0;
    for (int i0 = 0; i0 < n && blk > 0; i0 += 32) {
      const int i = i0 + lane;
      const int node = i < n ? list[i] : -1;
      // blocks of this node's bucket (the host passes blk only for batches of
      // at most STREAM_DEP_TB blocks)
      const int nb = node >= 0 ? (cnt[node] + blk - 1) / blk : 0;
      int incl = nb;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int x = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += x;
      }
      for (int b = 0; b < nb; ++b) out[base + incl - nb + b] = node * STREAM_DEP_TB + b;
      base += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) act_n[warp] = base;
  }
  for (int i = threadIdx.x; i < n_sctr; i += blockDim.x) sctr[i] = 0;
}

// one CTA: node/expert offsets and the tile prefix of every plan
__global__ void k_offsets_plan(const int* __restrict__ key_cnt, int N, int E,
                               int* __restrict__ key_off, const int* __restrict__ rank,
                               int* __restrict__ tile_off, int max_items, PlanArgs pa,
                               const int* __restrict__ anchors, int n_anchor,
                               const int* __restrict__ corrs, int n_corr, int blk,
                               int* __restrict__ act, int* __restrict__ act_n,
                               int* __restrict__ sctr, int n_sctr) {
  pdl_wait();
  if (act)
    publish_active(key_cnt, anchors, n_anchor, corrs, n_corr, blk, act, act_n, sctr, n_sctr);
  // node offsets then expert offsets
  for (int part = 0; part < 2; ++part) {
    const int n0 = part == 0 ? 0 : N, cnt = part == 0 ? N : E;
    int* out = key_off + (part == 0 ? 0 : N + 1);
    int carry = 0;
    for (int base = 0; base < cnt; base += blockDim.x) {
      const int i = base + threadIdx.x;
      const int v = i < cnt ? key_cnt[n0 + i] : 0;
      int total;
      const int ex = block_excl_scan(v, &total);
      if (i < cnt) out[i] = carry + ex;
      carry += total;
    }
    if (threadIdx.x == 0) out[cnt] = carry;
    __syncthreads();
  }
  for (int p = 0; p < pa.n_plans; ++p) {
    int* to = tile_off + (pa.first + p) * (max_items + 1);
    int carry = 0;
    for (int base = 0; base < pa.n_items[p]; base += blockDim.x) {
      const int i = base + threadIdx.x;
      int v = 0;
      if (i < pa.n_items[p]) {
        const int n = pa.items[p][i];
        v = plan_tiles(pa, p, rank[n], key_cnt[n]);
      }
      int total;
      const int ex = block_excl_scan(v, &total);
      if (i < pa.n_items[p]) to[i] = carry + ex;
      carry += total;
    }
    if (threadIdx.x == 0) to[pa.n_items[p]] = carry;
    __syncthreads();
  }
}

__global__ void k_scatter(const uint8_t* __restrict__ marks, const int* __restrict__ rank_in,
                          const int* __restrict__ key_off, const int* __restrict__ topk_id, int T,
                          int k, int N, long Tp, int* __restrict__ node_tok,
                          int* __restrict__ row_node, int* __restrict__ perm) {
  pdl_wait();
  const int key = blockIdx.y;
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= T) return;
  const size_t idx = (size_t)key * Tp + t;
  if (!marks[idx]) return;
  const int rk = rank_in[idx];
  if (key < N) {
    const int row = key_off[key] + rk;
    node_tok[row] = t;
    row_node[row] = key;
  } else {
    const int e = key - N;
    const int pos = key_off[N + 1 + e] + rk;
    for (int s = 0; s < k; ++s)
      if (topk_id[(size_t)t * k + s] == e) {
        perm[pos] = t * k + s;
        break;
      }
  }
}

__global__ void k_node_row(const int* __restrict__ topk_id, int T, int k, int E, int D, long Tp,
                           const int* __restrict__ paths, const int* __restrict__ path_len,
                           const int* __restrict__ key_off, const int* __restrict__ rank_in,
                           int* __restrict__ node_row) {
  pdl_wait();
  const long a = (long)blockIdx.x * blockDim.x + threadIdx.x;
  if (a >= (long)T * k) return;
  const int t = (int)(a / k);
  const int e = topk_id[a];
  const int len = (e >= 0 && e < E) ? path_len[e] : 0;
  for (int l = 0; l < D; ++l) {
    int row = -1;
    if (l < len) {
      const int n = paths[e * LX_MAX_DEPTH + l];
      row = key_off[n] + rank_in[(size_t)n * Tp + t];
    }
    node_row[a * D + l] = row;
  }
}

// The fused path's per-cluster-row tables (flat layers on the tensor-core
// path; al_g == nullptr: none): see k_assign_rows.
struct CtMeta {
  const float* topk_w;
  float* al_g;
  int* al_row;
  int* rho2al;
  const int* child_col;
  int nch, gstride, rstride, pslot;
};

// The rows of every assignment, one warp per token (lane s = top-k slot s):
// its position in its expert's bucket (perm), the rows of the nodes on its
// path (node_row; the (token, node) pairs shared by several slots write the
// same node_tok / row_node values), and, for flat layers on the fused
// tensor-core path, the per-cluster-row tables: for each anchor row a of the
// token, al_g[a] = {dominant's gate, gates of child slots 0, 1, ...} (0 where
// not selected; slots whose experts share a node add up, in slot order) and
// al_row[a] = the child rows (-1 where not selected), written by the first
// slot of that anchor row; rho2al maps every child row to its anchor row.
__global__ void __launch_bounds__(256)
k_assign_rows(const int* __restrict__ topk_id, int T, int k, int N, int E, int D, long Tp,
              const int* __restrict__ paths, const int* __restrict__ path_len,
              const int* __restrict__ key_off, const int* __restrict__ rank_in,
              int* __restrict__ node_tok, int* __restrict__ row_node, int* __restrict__ perm,
              int* __restrict__ node_row, const CtMeta cm) {
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int t = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  if (t >= T) return;
  const size_t a = (size_t)t * k + lane;
  int e = -1, len = 0;
  if (lane < k) {
    e = topk_id[a];
    if (e >= 0 && e < E) {
      len = path_len[e];
      perm[key_off[N + 1 + e] + rank_in[(size_t)(N + e) * Tp + t]] = (int)a;
    } else {
      e = -1;
    }
  }
  int r0 = -1, r1 = -1, n0 = -1;
#pragma unroll
  for (int l = 0; l < LX_MAX_DEPTH; ++l) {
    if (l >= D) break;
    int row = -1;
    if (l < len) {
      const int n = paths[e * LX_MAX_DEPTH + l];
      row = key_off[n] + rank_in[(size_t)n * Tp + t];
      node_tok[row] = t;
      row_node[row] = n;
      if (l == 0) n0 = n;
    }
    if (lane < k) node_row[a * D + l] = row;
    if (l == 0) r0 = row;
    if (l == 1) r1 = row;
  }
  if (!cm.al_g) return;
  // flat layers: a path is [anchor] (the dominant) or [member, anchor]
  const bool member = len >= 2;
  const int an = lane < k && e >= 0 ? (member ? r1 : r0) : -1;
  const int j = member ? cm.child_col[n0] / cm.pslot : -1;
  const float g = an >= 0 ? cm.topk_w[a] : 0.f;
  if (member) cm.rho2al[r0] = an;
  const unsigned same = __match_any_sync(0xffffffffu, an);
  const bool leader = an >= 0 && lane == __ffs(same) - 1;
  float rg[1 + CT_MAX_CH];
  int rr[CT_MAX_CH];
#pragma unroll
  for (int i = 0; i <= CT_MAX_CH; ++i) rg[i] = 0.f;
#pragma unroll
  for (int i = 0; i < CT_MAX_CH; ++i) rr[i] = -1;
  for (int sl = 0; sl < k; ++sl) {
    const int as = __shfl_sync(0xffffffffu, an, sl), js = __shfl_sync(0xffffffffu, j, sl);
    const int rs = __shfl_sync(0xffffffffu, r0, sl);
    const float gs = __shfl_sync(0xffffffffu, g, sl);
    if (as == an && as >= 0) {
#pragma unroll
      for (int i = 0; i <= CT_MAX_CH; ++i)
        if (i == js + 1) rg[i] += gs;
#pragma unroll
      for (int i = 0; i < CT_MAX_CH; ++i)
        if (i == js) rr[i] = rs;
    }
  }
  if (leader) {
#pragma unroll
    for (int i = 0; i <= CT_MAX_CH; ++i)
      if (i <= cm.nch) cm.al_g[(size_t)an * cm.gstride + i] = rg[i];
#pragma unroll
    for (int i = 0; i < CT_MAX_CH; ++i)
      if (i < cm.nch) cm.al_row[(size_t)an * cm.rstride + i] = rr[i];
  }
}

// ---------------------------------------------------------------------------
// Small batches (decode): top-k and the whole bucketing in one CTA, with the
// marks and ranks in shared memory (ranks fit a byte since T <= 256).  Same
// outputs, same order, as the multi-kernel path above.
// ---------------------------------------------------------------------------
constexpr int SB_THREADS = 1024;
constexpr int SB_MAX_T = 256;
constexpr size_t SB_SMEM_LIMIT = 160 * 1024;

__host__ __device__ inline size_t sb_smem(int T, int k, int keys, int E, int N, int max_items) {
  const size_t Tp = ((size_t)T + 15) / 16 * 16;
  return (size_t)T * k * 4 + 2 * (size_t)keys * Tp + (size_t)keys * 4 + ((size_t)keys + 2) * 4 +
         (size_t)E * (LX_MAX_DEPTH + 1) * 4 + 2 * (size_t)N * 4 + 64;
}

__global__ void __launch_bounds__(SB_THREADS)
k_bucket_small(const float* __restrict__ logits, const int* __restrict__ ids_in, int T, int k,
               int E, int N, int D, const int* __restrict__ paths,
               const int* __restrict__ path_len, const int* __restrict__ rank,
               int* __restrict__ topk_id, float* __restrict__ topk_w, int* __restrict__ key_off_g,
               int* __restrict__ node_tok, int* __restrict__ row_node, int* __restrict__ node_row,
               int* __restrict__ perm, int* __restrict__ tile_off, int max_items, PlanArgs pa,
               const int* __restrict__ anchors, int n_anchor, const int* __restrict__ corrs,
               int n_corr, int blk, int* __restrict__ act, int* __restrict__ act_n,
               int* __restrict__ sctr, int n_sctr) {
  extern __shared__ __align__(16) unsigned char sm[];
  const int keys = N + E;
  const int Tp = (T + 15) & ~15;
  int* ids = reinterpret_cast<int*>(sm);
  uint8_t* marks = reinterpret_cast<uint8_t*>(ids + T * k);
  uint8_t* rk = marks + (size_t)keys * Tp;
  int* cnt = reinterpret_cast<int*>(rk + (((size_t)keys * Tp + 3) & ~(size_t)3));
  int* off = cnt + keys;
  int* spaths = off + keys + 2;                 // [E][LX_MAX_DEPTH]
  int* splen = spaths + E * LX_MAX_DEPTH;       // [E]
  int* srank = splen + E;                       // [N]
  int* slist = srank + N;                       // [N]: the anchors, then the corrections
  const int tid = threadIdx.x, nth = blockDim.x;
  const int warp = tid >> 5, lane = tid & 31, nw = nth >> 5;
  // Before the wait for the preceding kernel: zeroed marks and the layer's
  // tables (constants of the layer) staged in shared memory.
  {
    uint32_t* m32 = reinterpret_cast<uint32_t*>(marks);  // keys*Tp is a multiple of 16
    for (int i = tid; i < keys * Tp / 4; i += nth) m32[i] = 0;
  }
  {
    const int n_paths = E * LX_MAX_DEPTH, n_tab = n_paths + E + N;
    for (int i = tid; i < n_tab + N; i += nth) {
      if (i < n_paths) spaths[i] = paths[i];
      else if (i < n_paths + E) splen[i - n_paths] = path_len[i - n_paths];
      else if (i < n_tab) srank[i - n_paths - E] = rank[i - n_paths - E];
      else if (i < n_tab + n_anchor) slist[i - n_tab] = anchors[i - n_tab];
      else slist[i - n_tab] = corrs[i - n_tab - n_anchor];
    }
  }
  pdl_wait();
  if (!logits)  // the given ids (written by the preceding kernel)
    for (int i = tid; i < T * k; i += nth) ids[i] = ids_in[i];
  // 1. routing (or the given ids)
  if (logits) {
    for (int t = warp; t < T; t += nw) {
      int id;
      float w;
      warp_topk(logits + (size_t)t * E, E, k, id, w);
      if (lane < k) {
        ids[t * k + lane] = id;
        topk_id[(size_t)t * k + lane] = id;
        topk_w[(size_t)t * k + lane] = w;
      }
    }
  }
  __syncthreads();
  // 2. marks
  for (int a = tid; a < T * k; a += nth) {
    const int t = a / k, e = ids[a];
    if (e < 0 || e >= E) continue;
    marks[(N + e) * Tp + t] = 1;
    const int len = splen[e];
    for (int l = 0; l < len; ++l) marks[spaths[e * LX_MAX_DEPTH + l] * Tp + t] = 1;
  }
  __syncthreads();
  // 3. per-key ranks in token order (warp ballots; four keys per warp at a
  // time, so that their ballot chains overlap)
  for (int kb0 = warp; kb0 < keys; kb0 += 4 * nw) {
    int running[4] = {0, 0, 0, 0};
    for (int t0 = 0; t0 < T; t0 += 32) {
      const int t = t0 + lane;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int key = kb0 + j * nw;
        const bool m = key < keys && t < T && marks[key * Tp + t];
        const uint32_t b = __ballot_sync(0xffffffffu, m);
        if (m) rk[key * Tp + t] = (uint8_t)(running[j] + __popc(b & ((1u << lane) - 1u)));
        running[j] += __popc(b);
      }
    }
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (lane == 0 && kb0 + j * nw < keys) cnt[kb0 + j * nw] = running[j];
  }
  __syncthreads();
  // 4. node offsets (warp 0) and expert offsets (warp 1): warp scans with a carry
  if (warp < 2) {
    const int n0 = warp == 0 ? 0 : N, n = warp == 0 ? N : E;
    const int o0 = warp == 0 ? 0 : N + 1;
    int carry = 0;
    for (int base = 0; base < n; base += 32) {
      const int i = base + lane;
      const int v = i < n ? cnt[n0 + i] : 0;
      int incl = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int x = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += x;
      }
      if (i < n) off[o0 + i] = carry + incl - v;
      carry += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) off[o0 + n] = carry;
  }
  __syncthreads();
  for (int i = tid; i < keys + 2; i += nth) key_off_g[i] = off[i];
  publish_active(cnt, slist, n_anchor, slist + n_anchor, n_corr, blk, act, act_n, sctr, n_sctr);
  // 5. tile plans: one warp per plan
  for (int p = warp; p < pa.n_plans; p += nw) {
    int* to = tile_off + (pa.first + p) * (max_items + 1);
    int carry = 0;
    for (int base = 0; base < pa.n_items[p]; base += 32) {
      const int i = base + lane;
      int v = 0;
      if (i < pa.n_items[p]) {
        const int n = pa.items[p][i];
        v = plan_tiles(pa, p, srank[n], cnt[n]);
      }
      int incl = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int x = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += x;
      }
      if (i < pa.n_items[p]) to[i] = carry + incl - v;
      carry += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) to[pa.n_items[p]] = carry;
  }
  // 6. scatter from the assignments: bucket rows, node rows, permutation
  for (int a = tid; a < T * k; a += nth) {
    const int t = a / k, e = ids[a];
    const bool valid = e >= 0 && e < E;
    const int len = valid ? splen[e] : 0;
    if (valid) perm[off[N + 1 + e] + rk[(N + e) * Tp + t]] = a;
    for (int l = 0; l < D; ++l) {
      int row = -1;
      if (l < len) {
        const int n = spaths[e * LX_MAX_DEPTH + l];
        row = off[n] + rk[n * Tp + t];
        node_tok[row] = t;   // (t, n) pairs shared by several slots write the same values
        row_node[row] = n;
      }
      node_row[(size_t)a * D + l] = row;
    }
  }
}

}  // namespace

// plans 0..N_OPS-1: generic tiles; N_OPS..2*N_OPS-1: streaming tiles
// Plans for slots [first, first + n_plans): 0 = the generic GEMMs' six ops,
// PLAN_TC = the tensor-core GEMMs' six ops.
static PlanArgs make_plans(const lx_layer* L, int n_plans, int first = 0) {
  PlanArgs pa;
  pa.n_plans = n_plans;
  pa.first = first;
  for (int p = 0; p < n_plans; ++p) {
    const int slot = first + p;
    const int op = slot % N_OPS;
    pa.shape[p] = op_shape(L, op);
    pa.items[p] = pa.shape[p].on_anchors ? L->d_anchors : L->d_corrs;
    pa.n_items[p] = pa.shape[p].on_anchors ? L->n_anchor : L->n_corr;
    pa.bm[p] = slot < PLAN_TC ? G_BM : tc_tile_rows(L, op);
    pa.bn[p] = slot < PLAN_TC ? G_BN : tc_tile_cols();
    if (L->ct && slot == PLAN_TC + OP_UP_U) {
      // the fused correction + SwiGLU kernel takes this slot: tiles of 128
      // cluster rows x CT_CW d_ff columns over the anchors
      pa.shape[p] = OpShape{L->I, 0, 0, 0, 1, 1};
      pa.items[p] = L->d_anchors;
      pa.n_items[p] = L->n_anchor;
      pa.bm[p] = 128;
      pa.bn[p] = CT_CW;
    }
  }
  return pa;
}

// Token rows per streaming work item, or 0 for batches the streaming kernels
// do not take (more blocks than the dependency counters cover).
static int stream_item_rows(int T) {
  const int blk = stream_tile_tokens();
  return T <= STREAM_DEP_TB * blk ? blk : 0;
}

bool bucket_small_fits(const lx_layer* L, int T, int k) {
  return T <= SB_MAX_T &&
         sb_smem(T, k, L->N + L->E, L->E, L->N, op_max_items(L)) <= SB_SMEM_LIMIT;
}

lx_status launch_bucket_small(lx_layer* L, const float* logits, const int* ids_in, int T, int k,
                              int* topk_id, float* topk_w, cudaStream_t s, bool plans) {
  Workspace& w = L->ws;
  const size_t smem = sb_smem(T, k, L->N + L->E, L->E, L->N, op_max_items(L));
  const PlanArgs pa = make_plans(L, plans ? N_OPS : 0);
  static bool done[64] = {};
  LX_CUDA(smem_cap_once((const void*)k_bucket_small, (int)SB_SMEM_LIMIT, L->device, done));
  ProfScope ps(L, s, logits ? "topk_bucket_small" : "bucket_small");
  launch_k(L, k_bucket_small, 1, SB_THREADS, smem, s, logits, ids_in, T, k, L->E, L->N, L->max_depth,
                                             L->d_paths, L->d_path_len, L->d_rank, topk_id, topk_w,
                                             w.key_off, w.node_tok, w.row_node, w.node_row, w.perm,
                                             w.tile_off, op_max_items(L), pa, L->d_anchors,
                                             L->n_anchor, L->d_corrs, L->n_corr,
                                             stream_item_rows(T), w.act, w.act_n, w.sctr,
                                             sctr_ints(L));
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

lx_status launch_bucket(lx_layer* L, const int* topk_id, int T, int k, cudaStream_t s,
                        int plan_first) {
  Workspace& w = L->ws;
  const long Tp = (w.cap_T + 15) / 16 * 16;
  const int keys = L->N + L->E;
  {
    ProfScope ps(L, s, "bucket_clear");
    LX_CUDA(cudaMemsetAsync(w.marks, 0, (size_t)keys * Tp, s));
  }
  {
    ProfScope ps(L, s, "bucket_mark");
    launch_k(L, k_mark, (T + 255) / 256, 256, 0, s, topk_id, T, k, L->N, L->E, Tp, L->d_paths,
             L->d_path_len, w.marks);
    LX_CUDA(cudaGetLastError());
  }
  {
    ProfScope ps(L, s, "bucket_scan");
    launch_k(L, k_key_scan, keys, SCAN_THREADS, 0, s, w.marks, T, Tp, w.rank_in, w.key_cnt);
    LX_CUDA(cudaGetLastError());
  }
  {
    const PlanArgs pa = plan_first < 0 ? make_plans(L, 0) : make_plans(L, N_OPS, plan_first);
    ProfScope ps(L, s, "bucket_offsets");
    launch_k(L, k_offsets_plan, 1, 1024, 0, s, w.key_cnt, L->N, L->E, w.key_off, L->d_rank, w.tile_off,
                                      op_max_items(L), pa, L->d_anchors, L->n_anchor, L->d_corrs,
                                      L->n_corr, stream_item_rows(T), w.act, w.act_n, w.sctr,
                                      sctr_ints(L));
    LX_CUDA(cudaGetLastError());
  }
  {
    // the fused tensor-core path of flat layers also takes its per-cluster-row
    // tables from this pass
    CtMeta cm{};
    if (L->ct && plan_first == PLAN_TC) {
      cm.topk_w = w.topk_w;
      cm.al_g = w.al_g;
      cm.al_row = w.al_row;
      cm.rho2al = w.rho2al;
      cm.child_col = L->d_child_col;
      cm.nch = L->ct_nch;
      cm.gstride = ct_gstride(L);
      cm.rstride = ct_rstride(L);
      cm.pslot = 2 * std::max(1, L->max_rank);
    }
    ProfScope ps(L, s, "bucket_rows");
    launch_k(L, k_assign_rows, (unsigned)((T + 7) / 8), 256, 0, s, topk_id, T, k, L->N, L->E,
             L->max_depth, Tp, L->d_paths, L->d_path_len, w.key_off, w.rank_in, w.node_tok,
             w.row_node, w.perm, w.node_row, cm);
    LX_CUDA(cudaGetLastError());
  }
  return LX_OK;
}

}  // namespace lx

// ---------------------------------------------------------------------------
// lx_bucket_noalloc: the same kernels, with every temporary buffer carved out
// of one static device array instead of the layer's (cudaMalloc'd) workspace.
// ---------------------------------------------------------------------------
namespace lx {
namespace {

// The scratch itself.  In host code this name is only a handle for
// cudaGetSymbolAddress, never a device address.
static __device__ __align__(256) unsigned char g_bucket_scratch[LX_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of g_bucket_scratch on `device` (which must be current).
lx_status scratch_address(int device, void** out) {
  if (device < 0 || device >= kMaxDevices) return fail(LX_ERR_UNSUPPORTED, "device id above 63");
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_addr[device]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_bucket_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(g_bucket_scratch)");
    g_scratch_addr[device] = p;
  }
  *out = g_scratch_addr[device];
  return LX_OK;
}

size_t round256(size_t v) { return (v + 255) / 256 * 256; }

}  // namespace

}  // namespace lx

extern "C" lx_status lx_bucket_noalloc(lx_layer* L, const int32_t* topk_id, int32_t T, int32_t k,
                                       int32_t* node_off, int32_t* node_tok, int32_t* node_row,
                                       int32_t* expert_off, int32_t* perm, void* stream) {
  using namespace lx;
  if (!L) return fail(LX_ERR_ARG, "layer is NULL");
  if (T < 0) return fail(LX_ERR_ARG, "T < 0");
  if (k < 1 || k > LX_MAX_K || k > L->E) return fail(LX_ERR_ARG, "k must be in 1..min(E, LX_MAX_K)");
  cudaStream_t s = (cudaStream_t)stream;
  if (T == 0) {
    // no assignments: every bucket is empty, so both offset arrays are zero
    if (node_off) LX_CUDA(cudaMemsetAsync(node_off, 0, sizeof(int) * (L->N + 1), s));
    if (expert_off) LX_CUDA(cudaMemsetAsync(expert_off, 0, sizeof(int) * (L->E + 1), s));
    return LX_OK;
  }
  if (!topk_id || !node_off || !node_tok || !node_row || !expert_off || !perm)
    return fail(LX_ERR_ARG, "NULL topk_id or output pointer");
  int dev = -1;
  LX_CUDA(cudaGetDevice(&dev));
  if (dev != L->device) return fail(LX_ERR_ARG, "the layer's device must be current");

  // carve the scratch: marks, ranks, counts, offsets, row->node (no tile plans:
  // nothing reads them here)
  const long Tp = ((long)T + 15) / 16 * 16;
  const long keys = (long)L->N + L->E;
  const long D = L->max_depth;
  const size_t b_marks = round256((size_t)keys * Tp);
  const size_t b_rank = round256(sizeof(int) * (size_t)keys * Tp);
  const size_t b_cnt = round256(sizeof(int) * (size_t)keys);
  const size_t b_off = round256(sizeof(int) * (size_t)(keys + 2));
  const size_t b_rown = round256(sizeof(int) * (size_t)T * k * D);
  const size_t need = b_marks + b_rank + b_cnt + b_off + b_rown;
  if (need > (size_t)LX_NOALLOC_SCRATCH_BYTES)
    return fail(LX_ERR_SHAPE, "lx_bucket_noalloc: T=" + std::to_string(T) + " needs " +
                                  std::to_string(need) + " scratch bytes, the fixed array has " +
                                  std::to_string((size_t)LX_NOALLOC_SCRATCH_BYTES));
  void* base = nullptr;
  LX_TRY(scratch_address(dev, &base));
  char* p = static_cast<char*>(base);
  uint8_t* marks = reinterpret_cast<uint8_t*>(p);
  int* rank_in = reinterpret_cast<int*>(p += b_marks);
  int* key_cnt = reinterpret_cast<int*>(p += b_rank);
  int* key_off = reinterpret_cast<int*>(p += b_cnt);
  int* row_node = reinterpret_cast<int*>(p += b_off);

  LX_CUDA(cudaMemsetAsync(marks, 0, (size_t)keys * Tp, s));  // previous call's marks
  k_mark<<<(T + 255) / 256, 256, 0, s>>>(topk_id, T, k, L->N, L->E, Tp, L->d_paths,
                                         L->d_path_len, marks);
  LX_CUDA(cudaGetLastError());
  k_key_scan<<<(unsigned)keys, SCAN_THREADS, 0, s>>>(marks, T, Tp, rank_in, key_cnt);
  LX_CUDA(cudaGetLastError());
  const PlanArgs pa = make_plans(L, 0);
  k_offsets_plan<<<1, 1024, 0, s>>>(key_cnt, L->N, L->E, key_off, L->d_rank, nullptr,
                                    op_max_items(L), pa, nullptr, 0, nullptr, 0, 0, nullptr,
                                    nullptr, nullptr, 0);
  LX_CUDA(cudaGetLastError());
  k_scatter<<<dim3((T + 255) / 256, (unsigned)keys), 256, 0, s>>>(
      marks, rank_in, key_off, topk_id, T, k, L->N, Tp, node_tok, row_node, perm);
  LX_CUDA(cudaGetLastError());
  const long A = (long)T * k;
  k_node_row<<<(unsigned)((A + 255) / 256), 256, 0, s>>>(topk_id, T, k, L->E, L->max_depth, Tp,
                                                         L->d_paths, L->d_path_len, key_off,
                                                         rank_in, node_row);
  LX_CUDA(cudaGetLastError());
  LX_CUDA(cudaMemcpyAsync(node_off, key_off, sizeof(int) * (L->N + 1), cudaMemcpyDeviceToDevice, s));
  LX_CUDA(cudaMemcpyAsync(expert_off, key_off + L->N + 1, sizeof(int) * (L->E + 1),
                          cudaMemcpyDeviceToDevice, s));
  return LX_OK;
}
