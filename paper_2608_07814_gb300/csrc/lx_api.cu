// C ABI of liblx: validation, layer installation (Sec. 3.2 Stage 3 iii),
// workspace management, profiling and the forward's orchestration.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <string>
#include <vector>

#include "lx_internal.cuh"

namespace lx {

static thread_local std::string g_last_error;

lx_status fail(lx_status s, const std::string& msg) {
  g_last_error = msg;
  return s;
}

lx_status cuda_fail(cudaError_t e, const char* what) {
  g_last_error = std::string(what) + ": " + cudaGetErrorString(e);
  return e == cudaErrorMemoryAllocation ? LX_ERR_OOM : LX_ERR_CUDA;
}

static size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// ---------------------------------------------------------------------------
// profiling
// ---------------------------------------------------------------------------
static cudaEvent_t take_event(lx_layer* L) {
  if (!L->event_pool.empty()) {
    cudaEvent_t e = L->event_pool.back();
    L->event_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

// Under stream capture the events become external record nodes of the graph,
// so every replay stamps them.
static void record(cudaEvent_t e, cudaStream_t s) {
  cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
  cudaStreamIsCapturing(s, &st);
  if (st == cudaStreamCaptureStatusActive) cudaEventRecordWithFlags(e, s, cudaEventRecordExternal);
  else cudaEventRecord(e, s);
}

ProfScope::ProfScope(lx_layer* L_, cudaStream_t s_, const char* n) : L(L_), s(s_), name(n) {
  if (L->profiling) {
    b = take_event(L);
    if (b) record(b, s);
  }
}

ProfScope::~ProfScope() {
  if (L->profiling && b) {
    cudaEvent_t e = take_event(L);
    if (e) {
      record(e, s);
      L->prof.push_back(ProfRec{name, b, e});
    } else {
      L->event_pool.push_back(b);
    }
  }
}

// ---------------------------------------------------------------------------
// op shapes of the generic grouped GEMMs
// ---------------------------------------------------------------------------
OpShape op_shape(const lx_layer* L, int op) {
  switch (op) {
    case OP_UP_ANCHOR: return OpShape{2 * L->I, 0, L->H, 0, 1, 1};
    case OP_UP_V:      return OpShape{0, 2, L->H, 0, 1, 0};
    case OP_UP_U:      return OpShape{L->I, 0, 0, 1, 2, 0};
    case OP_DN_ANCHOR: return OpShape{L->H, 0, L->I, 0, 1, 1};
    case OP_DN_V:      return OpShape{0, 1, L->I, 0, 1, 0};
    default:           return OpShape{L->H, 0, 0, 1, 1, 0};  // OP_DN_U
  }
}

int op_max_items(const lx_layer* L) { return std::max(L->n_anchor, L->n_corr); }

static PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  cudaError_t ce = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                    cudaEnableDefault, &q);
  if (ce != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) return nullptr;
  return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
}

bool encode_bf16_2d(CUtensorMap* m, const void* base, long inner, long outer, int box_inner,
                    int box_outer) {
  auto encode = get_encode();
  if (!encode) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)inner, (cuuint64_t)outer};
  const cuuint64_t strides[1] = {(cuuint64_t)inner * 2};
  const cuuint32_t box[2] = {(cuuint32_t)box_inner, (cuuint32_t)box_outer};
  const cuuint32_t estr[2] = {1, 1};
  return encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

// TMA store map of a bf16 output buffer [rows][ld]: 32 x 32 boxes staged with
// the 64-byte swizzle (the 256-row tensor-core epilogue)
static bool encode_store_map(CUtensorMap* m, void* base, long rows, long ld) {
  auto encode = get_encode();
  if (!encode || (ld * 2) % 16 != 0) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)ld, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
  const cuuint32_t box[2] = {32, 32};
  const cuuint32_t estr[2] = {1, 1};
  return encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
                CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

// TMA map of a bf16 activation buffer [rows][ld] read as box_rows x 64-column
// boxes with the 128-byte swizzle (an A operand whose rows are already in
// node-row order)
static bool encode_rows_map(CUtensorMap* m, void* base, long rows, long ld, int box_rows) {
  auto encode = get_encode();
  if (!encode) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)ld, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
  const cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

// ---------------------------------------------------------------------------
// workspace
// ---------------------------------------------------------------------------
// Batches up to this size take the weight-streaming kernels.
constexpr int kStreamMaxT = 256;

static lx_status ensure_workspace(lx_layer* L, int T, int k, cudaStream_t s) {
  Workspace& w = L->ws;
  if (T <= w.cap_T && k <= w.cap_k) return LX_OK;
  const int cT = std::max(T, w.cap_T), ck = std::max(k, w.cap_k);
  const long Tp = align_up((size_t)cT, 16);
  const long D = L->max_depth;
  const long keys = (long)L->N + L->E;
  const long Rmax = std::max<long>(1, (long)cT * std::min<long>(L->N, (long)ck * D));
  const long rmax = std::max(1, L->max_rank);
  // split-K partial rows of the streaming path (batches up to kStreamMaxT)
  const long Rsplit =
      L->stream_ok ? std::max<long>(1, (long)std::min(cT, kStreamMaxT) *
                                           std::min<long>(L->N, (long)ck * D))
                   : 0;
  struct Item { void** p; size_t bytes; };
  std::vector<Item> items = {
      {(void**)&w.logits, sizeof(float) * cT * L->E},
      {(void**)&w.topk_id, sizeof(int) * cT * ck},
      {(void**)&w.tile_cnt, sizeof(int) * std::max(1, router_tile_counters(cT))},
      {(void**)&w.topk_w, sizeof(float) * cT * ck},
      {(void**)&w.marks, (size_t)keys * Tp},
      {(void**)&w.rank_in, sizeof(int) * keys * Tp},
      {(void**)&w.key_cnt, sizeof(int) * keys},
      {(void**)&w.key_off, sizeof(int) * (keys + 2)},
      {(void**)&w.node_tok, sizeof(int) * cT * ck * D},
      {(void**)&w.row_node, sizeof(int) * cT * ck * D},
      {(void**)&w.node_row, sizeof(int) * cT * ck * D},
      {(void**)&w.perm, sizeof(int) * cT * ck},
      {(void**)&w.tile_off, sizeof(int) * N_PLANS * (op_max_items(L) + 1)},
      {(void**)&w.h, sizeof(float) * Rmax * 2 * L->I},
      {(void**)&w.P, sizeof(float) * Rmax * 2 * rmax},
      {(void**)&w.z, sizeof(float) * Rmax * L->I},
      {(void**)&w.Q, sizeof(float) * Rmax * rmax},
      {(void**)&w.ypart, sizeof(float) * Rmax * L->H},
      {(void**)&w.Pb, (size_t)2 * Rmax * 2 * rmax},
      {(void**)&w.zb, (size_t)2 * Rmax * L->I},
      {(void**)&w.Qb, (size_t)2 * Rmax * rmax},
      {(void**)&w.act, sizeof(int) * STREAM_DEP_TB * std::max(1, L->n_anchor + L->n_corr)},
      {(void**)&w.act_n, sizeof(int) * 2},
      {(void**)&w.sctr, sizeof(int) * sctr_ints(L)},
      {(void**)&w.xmaps, sizeof(CUtensorMap) * 3},
      {(void**)&w.smaps, sizeof(CUtensorMap) * 3},
      {(void**)&w.gmap, sizeof(CUtensorMap)},
      {(void**)&w.xg, L->stream_ok ? (size_t)2 * Rmax * L->H : 0},
      {(void**)&w.hsplit, sizeof(float) * LX_STREAM_MAX_SPLIT * Rsplit * 2 * L->I},
      {(void**)&w.ysplit, sizeof(float) * LX_STREAM_MAX_SPLIT * Rsplit * L->H},
      {(void**)&w.err, 256},
      // fused correction + SwiGLU tables (flat layers on the tensor-core path)
      {(void**)&w.al_g, L->ct ? sizeof(float) * Rmax * ct_gstride(L) : 0},
      {(void**)&w.al_row, L->ct ? sizeof(int) * Rmax * ct_rstride(L) : 0},
      {(void**)&w.rho2al, L->ct ? sizeof(int) * Rmax : 0},
      {(void**)&w.Pal, L->ct ? (size_t)2 * Rmax * L->ct_nch * 2 * rmax : 0},
      {(void**)&w.Qal, L->ct ? (size_t)2 * Rmax * L->ct_nch * rmax : 0},
      {(void**)&w.pamap, L->ct ? 3 * sizeof(CUtensorMap) : 0},
      {(void**)&w.omaps, 2 * sizeof(CUtensorMap)},
      {(void**)&w.rs_part, L->router_screen
                               ? sizeof(float) * RS_MAX_SPLITS * (size_t)cT * router_epad(L) : 0},
  };
  size_t total = 0;
  for (auto& it : items) total += align_up(it.bytes, 256);
  if (w.base) {
    LX_CUDA(cudaStreamSynchronize(s));
    LX_CUDA(cudaFree(w.base));
    w.base = nullptr;
  }
  void* base = nullptr;
  cudaError_t e = cudaMalloc(&base, total);
  if (e != cudaSuccess) {
    w.cap_T = w.cap_k = 0;
    return cuda_fail(e, "cudaMalloc(workspace)");
  }
  size_t off = 0;
  for (auto& it : items) {
    *it.p = (char*)base + off;
    off += align_up(it.bytes, 256);
  }
  w.base = base;
  w.bytes = total;
  e = cudaMemsetAsync(w.err, 0, sizeof(int), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(w.tile_cnt, 0, sizeof(int) * std::max(1, router_tile_counters(cT)), s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "clear workspace error word");
  w.cap_T = cT;
  w.cap_k = ck;
  w.rows_cap = Rmax;
  w.hb = reinterpret_cast<__nv_bfloat16*>(w.h);
  w.yb = reinterpret_cast<__nv_bfloat16*>(w.ypart);
  w.split_rows = Rsplit;
  if (Rsplit == 0) w.hsplit = w.ysplit = nullptr;
  if (L->stream_ok) {
    CUtensorMap maps[7];
    std::memset(maps, 0, sizeof(maps));
    const int tb = tc_tile_tokens(), sb = stream_tile_tokens();
    const bool okm = encode_rows_map(&maps[0], w.Pb, Rmax, 2 * rmax, tb) &&
                     encode_rows_map(&maps[1], w.zb, Rmax, L->I, tb) &&
                     encode_rows_map(&maps[2], w.Qb, Rmax, rmax, tb) &&
                     encode_rows_map(&maps[3], w.Pb, Rmax, 2 * rmax, sb) &&
                     encode_rows_map(&maps[4], w.zb, Rmax, L->I, sb) &&
                     encode_rows_map(&maps[5], w.Qb, Rmax, rmax, sb) &&
                     encode_rows_map(&maps[6], w.xg, Rmax, L->H, tb);
    if (!okm) return fail(LX_ERR_CUDA, "cuTensorMapEncodeTiled(activation maps) failed");
    e = cudaMemcpyAsync(w.xmaps, maps, 3 * sizeof(CUtensorMap), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(w.smaps, maps + 3, 3 * sizeof(CUtensorMap), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(w.gmap, maps + 6, sizeof(CUtensorMap), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "copy activation maps");
  }
  if (L->ct) {
    CUtensorMap pm[3];
    std::memset(pm, 0, sizeof(pm));
    if (!encode_rows_map(&pm[0], w.Pal, Rmax, (long)L->ct_nch * 2 * rmax, tc_tile_tokens()) ||
        !encode_rows_map(&pm[1], w.hb, Rmax, 2L * L->I, tc_tile_tokens()) ||
        !encode_rows_map(&pm[2], w.Qal, Rmax, (long)L->ct_nch * rmax, tc_tile_tokens()))
      return fail(LX_ERR_CUDA, "cuTensorMapEncodeTiled(Pal, h, Qal) failed");
    e = cudaMemcpyAsync(w.pamap, pm, 3 * sizeof(CUtensorMap), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "copy Pal map");
  }
  {
    // TMA store maps of the anchor products' outputs (hb [R][2I], yb [R][H]);
    // left null (row-by-row stores) where the row pitch is not 16-byte aligned
    CUtensorMap om[2];
    std::memset(om, 0, sizeof(om));
    if (encode_store_map(&om[0], w.hb, Rmax, 2L * L->I) && encode_store_map(&om[1], w.yb, Rmax, L->H)) {
      e = cudaMemcpyAsync(w.omaps, om, 2 * sizeof(CUtensorMap), cudaMemcpyHostToDevice, s);
      if (e == cudaSuccess) e = cudaStreamSynchronize(s);
      if (e != cudaSuccess) return cuda_fail(e, "copy store maps");
    } else {
      w.omaps = nullptr;
    }
  }
  L->last_T = L->last_k = 0;
  return LX_OK;
}

static lx_status check_call(lx_layer* L, int T, int k) {
  if (!L) return fail(LX_ERR_ARG, "layer is NULL");
  if (T < 0) return fail(LX_ERR_ARG, "T < 0");
  if (k < 1 || k > LX_MAX_K || k > L->E)
    return fail(LX_ERR_ARG, "k must be in 1..min(E, LX_MAX_K)");
  if ((long)T * k * L->max_depth > (1L << 30)) return fail(LX_ERR_SHAPE, "T*k too large");
  return LX_OK;
}

// plan_first: which tile plans the forward's GEMMs read (0 = generic, PLAN_TC =
// tensor-core, -1 = none: the streaming kernels and lx_get_buckets read none)
static lx_status bucket_ids(lx_layer* L, const int* ids, int T, int k, cudaStream_t s,
                            int plan_first) {
  if (bucket_small_fits(L, T, k))
    return launch_bucket_small(L, nullptr, ids, T, k, nullptr, nullptr, s, plan_first == 0);
  return launch_bucket(L, ids, T, k, s, plan_first);
}

static lx_status route_and_bucket(lx_layer* L, const void* x, int T, int k, int* ids, float* w,
                                  float* logits_user, cudaStream_t s, int plan_first) {
  float* logits = logits_user ? logits_user : L->ws.logits;
  LX_TRY(launch_router(L, x, T, k, logits, ids, w, s, logits_user != nullptr));
  return bucket_ids(L, ids, T, k, s, plan_first);
}


// Largest batch the weight-streaming (decode) kernels take; beyond it every
// weight would be re-streamed per 64-token block.

static bool use_stream(const lx_layer* L, int T, int k) {
  return L->path_mode == LX_PATH_AUTO && L->stream_ok && warp_kernels_fit(L, k) &&
         T <= kStreamMaxT;
}

// Larger batches: the tensor-core kernels (same layer requirements).
static bool use_tc(const lx_layer* L, int T, int k) {
  return L->path_mode == LX_PATH_AUTO && L->stream_ok && warp_kernels_fit(L, k) &&
         T > kStreamMaxT;
}

// TMA descriptors of every weight matrix the streaming kernels read: each
// matrix is a 4-D tensor {64 K, 64 rows, K/64 tiles, rows/64 tiles} over the
// tiled layout, read one 64x64 box (8 KiB, contiguous) at a time.
static lx_status encode_tensor_maps(lx_layer* L, cudaStream_t s) {
  L->stream_ok = false;
  if (!L->tiled) return LX_OK;
  auto encode = get_encode();
  if (!encode) return LX_OK;
  std::vector<CUtensorMap> maps((size_t)N_OPS * L->N);
  std::memset(maps.data(), 0, maps.size() * sizeof(CUtensorMap));
  for (int op = 0; op < N_OPS; ++op) {
    const OpShape sh = op_shape(L, op);
    for (int n = 0; n < L->N; ++n) {
      const bool anchor = L->parent[n] < 0;
      if ((sh.on_anchors != 0) != anchor) continue;
      const int r = L->rank[n];
      const cuuint64_t K = sh.k_const + sh.k_rank * r;
      const cuuint64_t rows = (cuuint64_t)sh.groups * (sh.n_const + sh.n_rank * r);
      const void* base = op == OP_UP_ANCHOR || op == OP_UP_V ? L->h_w_up[n]
                         : op == OP_UP_U                     ? L->h_w_upU[n]
                         : op == OP_DN_U                     ? L->h_w_dnU[n]
                                                             : L->h_w_dn[n];
      const cuuint64_t dims[4] = {64, 64, K / 64, rows / 64};
      const cuuint64_t strides[3] = {128, 8192, (K / 64) * 8192};
      const cuuint32_t box[4] = {64, 64, 1, 1};
      const cuuint32_t estr[4] = {1, 1, 1, 1};
      CUresult cr = encode(&maps[(size_t)op * L->N + n], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4,
                           const_cast<void*>(base), dims, strides, box, estr,
                           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
      if (cr != CUDA_SUCCESS) return LX_OK;  // streaming path stays off
    }
  }
  void* d = nullptr;
  LX_CUDA(cudaMalloc(&d, maps.size() * sizeof(CUtensorMap)));
  L->d_tmaps = static_cast<CUtensorMap*>(d);
  LX_CUDA(cudaMemcpyAsync(d, maps.data(), maps.size() * sizeof(CUtensorMap),
                          cudaMemcpyHostToDevice, s));
  LX_CUDA(cudaStreamSynchronize(s));
  L->stream_ok = true;
  return LX_OK;
}

}  // namespace lx

using namespace lx;

// ---------------------------------------------------------------------------
// load
// ---------------------------------------------------------------------------
static lx_status validate_desc(const lx_layer_desc* d, const void* const* node_w,
                               const void* router_w) {
  if (!d || !node_w || !router_w) return fail(LX_ERR_ARG, "NULL descriptor/weights/router");
  if (!d->node_parent || !d->node_rank || !d->expert_node)
    return fail(LX_ERR_ARG, "NULL node table");
  if (d->dtype != LX_F32 && d->dtype != LX_BF16) return fail(LX_ERR_ARG, "unknown dtype");
  const long H = d->d_model, I = d->d_ff, E = d->n_experts, N = d->n_nodes;
  if (H < 8 || I < 8 || H % 8 || I % 8)
    return fail(LX_ERR_SHAPE, "d_model and d_ff must be positive multiples of 8");
  if (H > 65536 || I > 65536) return fail(LX_ERR_SHAPE, "d_model/d_ff above 65536");
  if (E < 1 || E > LX_MAX_EXPERTS) return fail(LX_ERR_SHAPE, "n_experts outside 1..1024");
  if (N < 1 || N > 4096) return fail(LX_ERR_SHAPE, "n_nodes outside 1..4096");
  for (long n = 0; n < N; ++n) {
    const int p = d->node_parent[n], r = d->node_rank[n];
    if (p < -1 || p >= N || p == n) return fail(LX_ERR_SHAPE, "bad node_parent");
    if (p == -1 && r != 0) return fail(LX_ERR_SHAPE, "anchor node with rank != 0");
    if (p >= 0 && (r < 1 || r > std::min(H, I)))
      return fail(LX_ERR_SHAPE, "correction rank outside 1..min(d_model, d_ff)");
    const int nw = p == -1 ? 3 : 6;
    for (int j = 0; j < nw; ++j)
      if (!node_w[6 * n + j]) return fail(LX_ERR_ARG, "NULL node weight pointer");
    // root path must reach an anchor within LX_MAX_DEPTH nodes (no cycles)
    long m = n;
    int depth = 1;
    while (d->node_parent[m] >= 0) {
      m = d->node_parent[m];
      if (++depth > LX_MAX_DEPTH) return fail(LX_ERR_SHAPE, "node path deeper than LX_MAX_DEPTH or cyclic");
    }
  }
  for (long e = 0; e < E; ++e)
    if (d->expert_node[e] < 0 || d->expert_node[e] >= N)
      return fail(LX_ERR_SHAPE, "expert_node out of range");
  if (d->node_sign)
    for (long n = 0; n < N; ++n) {
      const int sg = d->node_sign[n];
      if (sg != 1 && sg != -1) return fail(LX_ERR_SHAPE, "node_sign must be +1 or -1");
      if (d->node_parent[n] < 0 && sg != 1) return fail(LX_ERR_SHAPE, "anchor with node_sign -1");
    }
  return LX_OK;
}

// Flips the sign bit of every element (bf16 or fp32): exact negation.
static void negate_bytes(void* buf, size_t n_elems, int esz) {
  if (esz == 2) {
    uint16_t* p = (uint16_t*)buf;
    for (size_t i = 0; i < n_elems; ++i) p[i] ^= 0x8000u;
  } else {
    uint32_t* p = (uint32_t*)buf;
    for (size_t i = 0; i < n_elems; ++i) p[i] ^= 0x80000000u;
  }
}

// dst[c][r] = src[r][c] for a [rows][cols] matrix of esz-byte elements
static void transpose_bytes(const void* src, void* dst, long rows, long cols, int esz) {
  const char* s = (const char*)src;
  char* o = (char*)dst;
  for (long r = 0; r < rows; ++r)
    for (long c = 0; c < cols; ++c) std::memcpy(o + (c * rows + r) * esz, s + (r * cols + c) * esz, esz);
}

extern "C" lx_status lx_load_compressed_layer(const lx_layer_desc* d, const void* const* node_w,
                                              const void* router_w, const float* router_bias,
                                              void* stream, lx_layer** out) {
  if (!out) return fail(LX_ERR_ARG, "out is NULL");
  *out = nullptr;
  LX_TRY(validate_desc(d, node_w, router_w));
  cudaStream_t s = (cudaStream_t)stream;
  lx_layer* L = new lx_layer();
  {
    // LX_PDL=0 turns programmatic dependent launch off (for A/B timing)
    const char* pdl = std::getenv("LX_PDL");
    L->pdl = !(pdl && pdl[0] == '0');
  }
  L->H = d->d_model;
  L->I = d->d_ff;
  L->E = d->n_experts;
  L->N = d->n_nodes;
  L->dtype = d->dtype;
  L->esz = d->dtype == LX_BF16 ? 2 : 4;
  L->parent.assign(d->node_parent, d->node_parent + L->N);
  L->rank.assign(d->node_rank, d->node_rank + L->N);
  L->expert_node.assign(d->expert_node, d->expert_node + L->E);
  for (int n = 0; n < L->N; ++n) {
    if (L->parent[n] < 0) L->anchors.push_back(n);
    else L->corrs.push_back(n);
    L->max_rank = std::max(L->max_rank, L->rank[n]);
  }
  L->n_anchor = (int)L->anchors.size();
  L->n_corr = (int)L->corrs.size();
  std::vector<int> paths((size_t)L->E * LX_MAX_DEPTH, -1), plen(L->E, 0);
  for (int e = 0; e < L->E; ++e) {
    int n = L->expert_node[e], l = 0;
    while (n >= 0) {
      paths[(size_t)e * LX_MAX_DEPTH + l++] = n;
      n = L->parent[n];
    }
    plen[e] = l;
    L->max_depth = std::max(L->max_depth, l);
  }
  auto cleanup = [&](lx_status st) {
    lx_free_layer(L);
    return st;
  };
  cudaError_t ce = cudaGetDevice(&L->device);
  if (ce != cudaSuccess) return cleanup(cuda_fail(ce, "cudaGetDevice"));
  cudaDeviceGetAttribute(&L->num_sms, cudaDevAttrMultiProcessorCount, L->device);

  // ---- weight arena layout.  Layers the streaming kernels serve (bf16, every
  // dimension and rank a multiple of 64) store each weight matrix [rows][K] as
  // 64x64 tiles [rows/64][K/64][64][64]: one TMA box is then one contiguous
  // 8 KiB run, and a 64-row block's whole K extent is sequential in memory.
  L->tiled = L->dtype == LX_BF16 && L->H % 64 == 0 && L->I % 64 == 0;
  for (int n = 0; n < L->N; ++n)
    if (L->parent[n] >= 0 && L->rank[n] % 64) L->tiled = false;
  const long H = L->H, I = L->I, esz = L->esz;
  struct Piece { int node; int slot; size_t off; size_t bytes; };
  std::vector<Piece> pieces;
  size_t off = 0;
  auto add = [&](int node, int slot, size_t bytes) {
    pieces.push_back(Piece{node, slot, off, bytes});
    off += align_up(bytes, 256);
  };
  for (int n = 0; n < L->N; ++n) {
    if (L->parent[n] < 0) {
      add(n, 0, 2 * I * H * esz);  // [Wg;Wu]
      add(n, 2, H * I * esz);      // Wd
    } else {
      const long r = L->rank[n];
      add(n, 0, 2 * r * H * esz);  // [Vg^T;Vu^T]
      add(n, 1, 2 * I * r * esz);  // [Ug;Uu]
      add(n, 2, r * I * esz);      // Vd^T
      add(n, 3, H * r * esz);      // Ud
    }
  }
  const size_t router_off = off;
  off += align_up((size_t)L->E * H * esz, 256);
  const size_t bias_off = off;
  if (router_bias) off += align_up((size_t)L->E * 4, 256);
  L->arena_bytes = off;
  ce = cudaMalloc(&L->arena, off);
  if (ce != cudaSuccess) return cleanup(cuda_fail(ce, "cudaMalloc(weights)"));

  L->h_w_up.assign(L->N, nullptr);
  L->h_w_upU.assign(L->N, nullptr);
  L->h_w_dn.assign(L->N, nullptr);
  L->h_w_dnU.assign(L->N, nullptr);
  std::vector<char> stage, tiled;
  for (const Piece& p : pieces) {
    char* dst = (char*)L->arena + p.off;
    const int n = p.node;
    const void* const* w = node_w + 6 * (size_t)n;
    // edge sign -1 (Fig. 2): the correction enters as (-U) V^T
    const bool negative = d->node_sign && d->node_sign[n] < 0;
    stage.resize(p.bytes);
    if (L->parent[n] < 0) {
      if (p.slot == 0) {
        std::memcpy(stage.data(), w[0], I * H * esz);
        std::memcpy(stage.data() + I * H * esz, w[1], I * H * esz);
        L->h_w_up[n] = dst;
      } else {
        std::memcpy(stage.data(), w[2], H * I * esz);
        L->h_w_dn[n] = dst;
      }
    } else {
      const long r = L->rank[n];
      if (p.slot == 0) {  // Vg [H][r] -> [r][H]; Vu likewise
        transpose_bytes(w[1], stage.data(), H, r, esz);
        transpose_bytes(w[3], stage.data() + r * H * esz, H, r, esz);
        L->h_w_up[n] = dst;
      } else if (p.slot == 1) {
        std::memcpy(stage.data(), w[0], I * r * esz);
        std::memcpy(stage.data() + I * r * esz, w[2], I * r * esz);
        if (negative) negate_bytes(stage.data(), (size_t)2 * I * r, (int)esz);
        L->h_w_upU[n] = dst;
      } else if (p.slot == 2) {  // Vd [I][r] -> [r][I]
        transpose_bytes(w[5], stage.data(), I, r, esz);
        L->h_w_dn[n] = dst;
      } else {
        std::memcpy(stage.data(), w[4], H * r * esz);
        if (negative) negate_bytes(stage.data(), (size_t)H * r, (int)esz);
        L->h_w_dnU[n] = dst;
      }
    }
    const char* src = stage.data();
    if (L->tiled) {
      const long r = L->parent[n] < 0 ? 0 : L->rank[n];
      long rows, K;
      if (L->parent[n] < 0) { rows = p.slot == 0 ? 2 * I : H; K = p.slot == 0 ? H : I; }
      else if (p.slot == 0) { rows = 2 * r; K = H; }
      else if (p.slot == 1) { rows = 2 * I; K = r; }
      else if (p.slot == 2) { rows = r; K = I; }
      else { rows = H; K = r; }
      tiled.resize(p.bytes);
      const long nkt = K / 64;
      for (long row = 0; row < rows; ++row)
        for (long kt = 0; kt < nkt; ++kt)
          std::memcpy(tiled.data() + ((((row / 64) * nkt + kt) * 64 + row % 64) * 64) * esz,
                      stage.data() + (row * K + kt * 64) * esz, 64 * esz);
      src = tiled.data();
    }
    ce = cudaMemcpyAsync(dst, src, p.bytes, cudaMemcpyHostToDevice, s);
    if (ce == cudaSuccess) ce = cudaStreamSynchronize(s);
    if (ce != cudaSuccess) return cleanup(cuda_fail(ce, "copy weights"));
  }
  L->router_w = (char*)L->arena + router_off;
  ce = cudaMemcpyAsync(L->router_w, router_w, (size_t)L->E * H * esz, cudaMemcpyHostToDevice, s);
  if (ce == cudaSuccess && router_bias) {
    L->router_bias = (float*)((char*)L->arena + bias_off);
    ce = cudaMemcpyAsync(L->router_bias, router_bias, (size_t)L->E * 4, cudaMemcpyHostToDevice, s);
  }
  if (ce != cudaSuccess) return cleanup(cuda_fail(ce, "copy router"));

  // ---- small device tables
  const size_t nptr = (size_t)L->N;
  size_t toff = 0;
  auto tadd = [&](size_t bytes) {
    size_t o = toff;
    toff += align_up(bytes, 256);
    return o;
  };
  const size_t o_rank = tadd(4 * L->N), o_paths = tadd(4 * paths.size()), o_plen = tadd(4 * L->E);
  const size_t o_anc = tadd(4 * std::max(1, L->n_anchor)), o_cor = tadd(4 * std::max(1, L->n_corr));
  const size_t o_p0 = tadd(sizeof(void*) * nptr), o_p1 = tadd(sizeof(void*) * nptr);
  const size_t o_p2 = tadd(sizeof(void*) * nptr), o_p3 = tadd(sizeof(void*) * nptr);
  // children of every anchor (fused correction + SwiGLU of flat layers): a
  // layer qualifies when every correction node is a direct child of an anchor
  // and no anchor has more than CT_MAX_CH children
  std::vector<int> child((size_t)L->N * CT_MAX_CH, -1), child_col(L->N, 0), child_qcol(L->N, 0);
  std::vector<int> nchild(L->N, 0);
  bool flat = L->max_depth <= 2 && L->n_corr > 0;
  for (int n = 0; n < L->N && flat; ++n) {
    const int p = L->parent[n];
    if (p < 0) continue;
    if (L->parent[p] >= 0 || nchild[p] >= CT_MAX_CH) {
      flat = false;
      break;
    }
    child[(size_t)p * CT_MAX_CH + nchild[p]] = n;
    child_col[n] = nchild[p] * 2 * std::max(1, L->max_rank);
    child_qcol[n] = nchild[p] * std::max(1, L->max_rank);
    ++nchild[p];
  }
  L->ct_nch = 0;
  for (int n = 0; n < L->N; ++n) L->ct_nch = std::max(L->ct_nch, nchild[n]);
  {
    // LX_FUSED_SWIGLU=0 keeps the unfused tensor-core path (for A/B timing)
    const char* env = std::getenv("LX_FUSED_SWIGLU");
    L->ct = flat && L->tiled && !(env && env[0] == '0');
  }
  const size_t o_child = tadd(4 * child.size()), o_ccol = tadd(4 * (size_t)L->N);
  const size_t o_cqcol = tadd(4 * (size_t)L->N);
  std::vector<char> tb(toff, 0);
  std::memcpy(tb.data() + o_child, child.data(), 4 * child.size());
  std::memcpy(tb.data() + o_ccol, child_col.data(), 4 * (size_t)L->N);
  std::memcpy(tb.data() + o_cqcol, child_qcol.data(), 4 * (size_t)L->N);
  std::memcpy(tb.data() + o_rank, L->rank.data(), 4 * L->N);
  std::memcpy(tb.data() + o_paths, paths.data(), 4 * paths.size());
  std::memcpy(tb.data() + o_plen, plen.data(), 4 * L->E);
  if (L->n_anchor) std::memcpy(tb.data() + o_anc, L->anchors.data(), 4 * L->n_anchor);
  if (L->n_corr) std::memcpy(tb.data() + o_cor, L->corrs.data(), 4 * L->n_corr);
  std::memcpy(tb.data() + o_p0, L->h_w_up.data(), sizeof(void*) * nptr);
  std::memcpy(tb.data() + o_p1, L->h_w_upU.data(), sizeof(void*) * nptr);
  std::memcpy(tb.data() + o_p2, L->h_w_dn.data(), sizeof(void*) * nptr);
  std::memcpy(tb.data() + o_p3, L->h_w_dnU.data(), sizeof(void*) * nptr);
  ce = cudaMalloc(&L->tables, toff);
  if (ce != cudaSuccess) return cleanup(cuda_fail(ce, "cudaMalloc(tables)"));
  char* tbase = (char*)L->tables;
  L->d_rank = (int*)(tbase + o_rank);
  L->d_paths = (int*)(tbase + o_paths);
  L->d_path_len = (int*)(tbase + o_plen);
  L->d_anchors = (int*)(tbase + o_anc);
  L->d_corrs = (int*)(tbase + o_cor);
  L->d_w_up = (const void**)(tbase + o_p0);
  L->d_w_upU = (const void**)(tbase + o_p1);
  L->d_w_dn = (const void**)(tbase + o_p2);
  L->d_w_dnU = (const void**)(tbase + o_p3);
  L->d_child = (int*)(tbase + o_child);
  L->d_child_col = (int*)(tbase + o_ccol);
  L->d_child_qcol = (int*)(tbase + o_cqcol);
  ce = cudaMemcpyAsync(L->tables, tb.data(), toff, cudaMemcpyHostToDevice, s);
  if (ce == cudaSuccess) ce = cudaStreamSynchronize(s);
  if (ce != cudaSuccess) return cleanup(cuda_fail(ce, "copy tables"));
  const lx_status st = encode_tensor_maps(L, s);
  if (st != LX_OK) return cleanup(st);
  L->ct = L->ct && L->stream_ok;
  {
    // screened routing: bf16 router rows of a multiple of 64, at most 256
    // experts (one N tile); the bound of its candidate test needs the largest
    // row norm of the router matrix
    const char* env = std::getenv("LX_ROUTER_SCREEN");
    L->router_screen = L->dtype == LX_BF16 && L->H % 64 == 0 && L->E <= 256 &&
                       !(env && env[0] == '0');
    if (L->router_screen) {
      const uint16_t* rw = static_cast<const uint16_t*>(router_w);
      double wmax = 0.0;
      for (int e = 0; e < L->E; ++e) {
        double ss = 0.0;
        for (long h = 0; h < H; ++h) {
          const uint32_t bits = (uint32_t)rw[(size_t)e * H + h] << 16;
          float f;
          std::memcpy(&f, &bits, 4);
          ss += (double)f * f;
        }
        wmax = std::max(wmax, std::sqrt(ss));
      }
      L->router_wmax = (float)(wmax * (1.0 + 1e-6));
      std::memset(&L->router_map, 0, sizeof(L->router_map));
      if (!std::isfinite(L->router_wmax) ||
          !encode_bf16_2d(&L->router_map, L->router_w, H, L->E, 64, router_epad(L)))
        L->router_screen = false;
    }
  }
  *out = L;
  return LX_OK;
}

extern "C" lx_status lx_free_layer(lx_layer* L) {
  if (!L) return fail(LX_ERR_ARG, "layer is NULL");
  cudaDeviceSynchronize();
  for (auto& r : L->prof) {
    cudaEventDestroy(r.a);
    cudaEventDestroy(r.b);
  }
  for (auto e : L->event_pool) cudaEventDestroy(e);
  if (L->ws.base) cudaFree(L->ws.base);
  if (L->arena) cudaFree(L->arena);
  if (L->tables) cudaFree(L->tables);
  if (L->d_tmaps) cudaFree(L->d_tmaps);
  delete L;
  return LX_OK;
}

extern "C" lx_status lx_reserve(lx_layer* L, int32_t max_tokens, int32_t k) {
  LX_TRY(check_call(L, max_tokens, k));
  LX_TRY(ensure_workspace(L, std::max(1, max_tokens), k, nullptr));
  LX_CUDA(cudaDeviceSynchronize());
  return LX_OK;
}

extern "C" lx_status lx_route(lx_layer* L, const void* x, int32_t T, int32_t k, int32_t* topk_id,
                              float* topk_w, float* logits, void* stream) {
  LX_TRY(check_call(L, T, k));
  if (T == 0) return LX_OK;
  if (!x || !topk_id || !topk_w) return fail(LX_ERR_ARG, "NULL x/topk_id/topk_w");
  cudaStream_t s = (cudaStream_t)stream;
  LX_TRY(ensure_workspace(L, T, k, s));
  LX_TRY(route_and_bucket(L, x, T, k, topk_id, topk_w, logits, s, -1));
  L->last_T = T;
  L->last_k = k;
  return LX_OK;
}

extern "C" lx_status lx_bucket(lx_layer* L, const int32_t* topk_id, int32_t T, int32_t k,
                               void* stream) {
  LX_TRY(check_call(L, T, k));
  if (T == 0) return LX_OK;
  if (!topk_id) return fail(LX_ERR_ARG, "NULL topk_id");
  cudaStream_t s = (cudaStream_t)stream;
  LX_TRY(ensure_workspace(L, T, k, s));
  LX_TRY(bucket_ids(L, topk_id, T, k, s, -1));
  L->last_T = T;
  L->last_k = k;
  return LX_OK;
}

extern "C" lx_status lx_moe_forward(lx_layer* L, const void* x, int32_t T, int32_t k, void* y,
                                    void* stream) {
  LX_TRY(check_call(L, T, k));
  if (T == 0) return LX_OK;
  if (!x || !y) return fail(LX_ERR_ARG, "NULL x/y");
  if (reinterpret_cast<uintptr_t>(x) % 16 || reinterpret_cast<uintptr_t>(y) % 16)
    return fail(LX_ERR_ARG, "x and y must be 16-byte aligned");
  {
    const uintptr_t xb = reinterpret_cast<uintptr_t>(x), yb = reinterpret_cast<uintptr_t>(y);
    const uintptr_t bytes = (uintptr_t)T * L->H * L->esz;
    if (xb < yb + bytes && yb < xb + bytes) return fail(LX_ERR_ARG, "y may not overlap x");
  }
  cudaStream_t s = (cudaStream_t)stream;
  LX_TRY(ensure_workspace(L, T, k, s));
  Workspace& w = L->ws;
  // the generic and tensor-core GEMMs read tile plans; the streaming kernels do not
  const int plan_first = use_stream(L, T, k) ? -1 : use_tc(L, T, k) ? PLAN_TC : 0;
  LX_TRY(route_and_bucket(L, x, T, k, w.topk_id, w.topk_w, nullptr, s, plan_first));
  L->last_T = T;
  L->last_k = k;
  if (use_stream(L, T, k)) {
    LX_TRY(launch_fast_experts(L, x, T, k, y, s));
  } else if (use_tc(L, T, k)) {
    LX_TRY(launch_tc_experts(L, x, T, k, y, s));
  } else {
    LX_TRY(launch_generic_experts(L, x, T, k, y, s));
  }
  return LX_OK;
}

extern "C" lx_status lx_get_buckets(lx_layer* L, int32_t* node_off, int32_t* node_tok,
                                    int32_t* node_row, int32_t* expert_off, int32_t* perm,
                                    void* stream) {
  if (!L) return fail(LX_ERR_ARG, "layer is NULL");
  if (L->last_T == 0) return fail(LX_ERR_STATE, "nothing bucketed yet");
  cudaStream_t s = (cudaStream_t)stream;
  const Workspace& w = L->ws;
  const long T = L->last_T, k = L->last_k, D = L->max_depth;
  if (node_off)
    LX_CUDA(cudaMemcpyAsync(node_off, w.key_off, 4 * (L->N + 1), cudaMemcpyDeviceToDevice, s));
  if (expert_off)
    LX_CUDA(cudaMemcpyAsync(expert_off, w.key_off + L->N + 1, 4 * (L->E + 1),
                            cudaMemcpyDeviceToDevice, s));
  if (node_tok)
    LX_CUDA(cudaMemcpyAsync(node_tok, w.node_tok, 4 * T * k * D, cudaMemcpyDeviceToDevice, s));
  if (node_row)
    LX_CUDA(cudaMemcpyAsync(node_row, w.node_row, 4 * T * k * D, cudaMemcpyDeviceToDevice, s));
  if (perm) LX_CUDA(cudaMemcpyAsync(perm, w.perm, 4 * T * k, cudaMemcpyDeviceToDevice, s));
  return LX_OK;
}

extern "C" lx_status lx_layer_info(lx_layer* L, lx_layer_info_t* info) {
  if (!L || !info) return fail(LX_ERR_ARG, "NULL argument");
  info->d_model = L->H;
  info->d_ff = L->I;
  info->n_experts = L->E;
  info->n_nodes = L->N;
  info->dtype = L->dtype;
  info->n_anchors = L->n_anchor;
  info->n_corrections = L->n_corr;
  info->max_depth = L->max_depth;
  info->max_rank = L->max_rank;
  info->weight_bytes = (int64_t)L->arena_bytes;
  info->last_T = L->last_T;
  info->last_k = L->last_k;
  info->last_rows = 0;
  info->device_error = 0;
  info->stream_path = L->stream_ok ? 1 : 0;
  if (L->ws.base) {
    LX_CUDA(cudaDeviceSynchronize());
    int err = 0;
    LX_CUDA(cudaMemcpy(&err, L->ws.err, 4, cudaMemcpyDeviceToHost));
    info->device_error = err;
    if (L->last_T > 0) {
      int rows = 0;
      LX_CUDA(cudaMemcpy(&rows, L->ws.key_off + L->N, 4, cudaMemcpyDeviceToHost));
      info->last_rows = rows;
    }
  }
  return LX_OK;
}

extern "C" lx_status lx_set_path(lx_layer* L, int32_t path) {
  if (!L) return fail(LX_ERR_ARG, "layer is NULL");
  if (path != LX_PATH_AUTO && path != LX_PATH_GENERIC) return fail(LX_ERR_ARG, "unknown path");
  L->path_mode = path;
  return LX_OK;
}

extern "C" lx_status lx_set_wait_limit(lx_layer* L, uint64_t cycles) {
  if (!L) return fail(LX_ERR_ARG, "layer is NULL");
  L->wait_cycles = cycles;
  return LX_OK;
}

extern "C" lx_status lx_inject_unmet_wait(lx_layer* L, int32_t site) {
  if (!L) return fail(LX_ERR_ARG, "layer is NULL");
  if (site != LX_WAIT_NONE && site != LX_WAIT_STREAM_DEP && site != LX_WAIT_TC_MMA)
    return fail(LX_ERR_ARG, "unknown wait site");
  L->unmet_wait = site;
  return LX_OK;
}

extern "C" lx_status lx_clear_device_error(lx_layer* L) {
  if (!L) return fail(LX_ERR_ARG, "layer is NULL");
  if (L->ws.base) {
    LX_CUDA(cudaDeviceSynchronize());
    LX_CUDA(cudaMemset(L->ws.err, 0, sizeof(int)));
    LX_CUDA(cudaDeviceSynchronize());
  }
  return LX_OK;
}

extern "C" lx_status lx_set_profiling(lx_layer* L, int32_t enable) {
  if (!L) return fail(LX_ERR_ARG, "layer is NULL");
  L->profiling = enable != 0;
  return LX_OK;
}

extern "C" lx_status lx_read_profile(lx_layer* L, lx_kernel_time* out, int32_t cap, int32_t* n) {
  if (!L || !n || (cap > 0 && !out)) return fail(LX_ERR_ARG, "NULL argument");
  *n = 0;
  if (!L->prof.empty()) LX_CUDA(cudaEventSynchronize(L->prof.back().b));
  int w = 0;
  for (auto& r : L->prof) {
    float ms = 0.f;
    cudaEventElapsedTime(&ms, r.a, r.b);
    if (w < cap) out[w++] = lx_kernel_time{r.name, ms};
    L->event_pool.push_back(r.a);
    L->event_pool.push_back(r.b);
  }
  L->prof.clear();
  *n = w;
  return LX_OK;
}

extern "C" const char* lx_last_error(void) { return g_last_error.c_str(); }
