// Internal declarations shared by the CUDA translation units of liblx.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include <string>
#include <vector>

#include "../../include/lx.h"

namespace lx {

// ---------------------------------------------------------------------------
// error handling
// ---------------------------------------------------------------------------
lx_status fail(lx_status s, const std::string& msg);
lx_status cuda_fail(cudaError_t e, const char* what);

#define LX_CUDA(call)                                              \
  do {                                                             \
    cudaError_t e_ = (call);                                       \
    if (e_ != cudaSuccess) return ::lx::cuda_fail(e_, #call);      \
  } while (0)

#define LX_TRY(call)                                               \
  do {                                                             \
    lx_status s_ = (call);                                         \
    if (s_ != LX_OK) return s_;                                    \
  } while (0)

// ---------------------------------------------------------------------------
// element helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ float to_f32(float v) { return v; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 v) { return __bfloat162float(v); }
template <typename T> __device__ __forceinline__ T from_f32(float v);
template <> __device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) {
  return __float2bfloat16_rn(v);
}

// ---------------------------------------------------------------------------
// top-k of one token's logits by one warp: k rounds of a warp arg-max with
// the order (logit descending, expert id ascending); softmax over the k
// selected logits.  Lane j ends with slot j's id and gate (j < k).  A NaN
// logit is never preferred; if only NaNs remain the lowest free id is taken,
// so ids always stay in [0, E).
// ---------------------------------------------------------------------------
// Order-preserving integer key of a non-NaN logit (+0 and -0 map alike, as
// they compare equal); 0 marks "no candidate" and lies below every logit.
__device__ __forceinline__ uint32_t topk_key(float v) {
  const uint32_t u = __float_as_uint(v == 0.f ? 0.f : v);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float topk_key_value(uint32_t key) {
  return __uint_as_float((key & 0x80000000u) ? (key & 0x7fffffffu) : ~key);
}

// Each round: every lane's best free candidate (largest key, then lowest id),
// the warp maximum of the keys and the lowest id holding it by two warp
// reductions (redux.sync).
template <int EPL>  // candidates per lane: E <= 32 * EPL
__device__ __forceinline__ void warp_topk_t(const float* lt, int E, int k, int& sel_id,
                                            float& sel_w) {
  const int lane = threadIdx.x & 31;
  uint32_t key[EPL];  // this lane's candidates e = lane + 32 i (0: absent or NaN)
#pragma unroll
  for (int i = 0; i < EPL; ++i) {
    const int e = lane + 32 * i;
    const float v = e < E ? lt[e] : 0.f;
    key[i] = (e < E && v == v) ? topk_key(v) : 0u;
  }
  uint32_t taken = 0;  // bit i <-> expert lane + 32 i
  float m = 0.f, denom = 0.f, selv = 0.f;
  int seli = 0;
  for (int j = 0; j < k; ++j) {
    uint32_t bk = 0;
    int be = 0x7fffffff;
#pragma unroll
    for (int i = 0; i < EPL; ++i) {
      const uint32_t ki = ((taken >> i) & 1u) ? 0u : key[i];
      if (ki > bk) {  // ascending i: the first of equal keys (lowest id) stays
        bk = ki;
        be = lane + 32 * i;
      }
    }
    const uint32_t mk = __reduce_max_sync(0xffffffffu, bk);
    int bi;
    float bv;
    if (mk != 0u) {
      bi = __reduce_min_sync(0xffffffffu, bk == mk ? be : 0x7fffffff);
      bv = topk_key_value(mk);
    } else {  // only NaNs left: lowest free id
      int fi = 0x7fffffff;
#pragma unroll
      for (int i = EPL - 1; i >= 0; --i) {
        const int e = lane + 32 * i;
        if (e < E && !((taken >> i) & 1u)) fi = e;
      }
      bi = __reduce_min_sync(0xffffffffu, fi);
      bv = lt[bi];
    }
    if ((bi & 31) == lane) taken |= 1u << (bi >> 5);
    if (j == 0) m = bv;
    const float ex = expf(bv - m);
    denom += ex;
    if (lane == j) { selv = ex; seli = bi; }
  }
  sel_id = seli;
  sel_w = selv / denom;
}

__device__ __forceinline__ void warp_topk(const float* lt, int E, int k, int& sel_id,
                                          float& sel_w) {
  if (E <= 32) warp_topk_t<1>(lt, E, k, sel_id, sel_w);
  else if (E <= 64) warp_topk_t<2>(lt, E, k, sel_id, sel_w);
  else if (E <= 128) warp_topk_t<4>(lt, E, k, sel_id, sel_w);
  else if (E <= 256) warp_topk_t<8>(lt, E, k, sel_id, sel_w);
  else warp_topk_t<32>(lt, E, k, sel_id, sel_w);
}

// ---------------------------------------------------------------------------
// grouped GEMM over node buckets (the generic CUDA-core path)
// ---------------------------------------------------------------------------
// Op kinds, indexing the per-op tile plans.
enum OpKind {
  OP_UP_ANCHOR = 0,  // h[row, 0:2I]   = x[tok] . [Wg;Wu]^T          (anchors)
  OP_UP_V = 1,       // P[row, 0:2r]   = x[tok] . [Vg|Vu]            (corrections)
  OP_UP_U = 2,       // h[row, gI:(g+1)I] = P[row, g r:(g+1) r] . U_g^T, g in {gate, up}
  OP_DN_ANCHOR = 3,  // ypart[row, 0:H] = z[row] . Wd^T              (anchors)
  OP_DN_V = 4,       // Q[row, 0:r]    = z[row] . Vd
  OP_DN_U = 5,       // ypart[row, 0:H] = Q[row] . Ud^T
  N_OPS = 6
};

// Tile plans (prefix of the tiles per node, built by the bucketing): plan p <
// N_OPS is op p for the generic kernel (32-token x 64-column tiles); plan
// PLAN_TC + p is op p for the tensor-core kernel (128 tokens x 256 columns).
// The streaming kernels decode their tiles from the streaming work items instead.
constexpr int N_PLANS = 2 * N_OPS;
constexpr int PLAN_TC = N_OPS;
constexpr int N_TILE_COUNTERS = 16;  // dynamic tile counters, zeroed by the bucketing

// Per-op shape rule: for node n with rank r, each group has
//   N_g = n_const + n_rank * r output columns and K = k_const + k_rank * r.
struct OpShape {
  int n_const, n_rank, k_const, k_rank, groups;
  int on_anchors;  // 1: items are anchors; 0: corrections
};

// Generic tile sizes
constexpr int G_BM = 32, G_BN = 64, G_BK = 32;

struct GemmArgs {
  const int* items;        // node ids [n_items]
  int n_items;
  const int* tile_off;     // [n_items+1] tile prefix (device, from the plan)
  const int* node_off;     // [n_nodes+1]
  const int* gather;       // row -> A row index (e.g. node_tok), or null = identity
  const void* A;           // activations (f32 or layer dtype)
  long lda;                // elements
  const void* const* W;    // per node id: weight [groups*N_g][K] row-major
  const int* rank;         // per node
  OpShape shape;
  float* out;
  long ldo;
  int tiled;               // W stored as [rows/64][K/64][64][64] tiles
};

// Streaming (decode) grouped GEMM: one op of a launch
struct StreamOp {
  const CUtensorMap* tmaps;  // [n_nodes] weight tensor maps of this op
  const int* items;          // work items node * STREAM_DEP_TB + token block (written by the bucketing)
  const int* n_active;       // device count of items
  int n_items;               // upper bound of the count (host)
  const int* tile_off;       // [n_items+1] stream plan
  const int* node_off;
  const int* gather;         // row -> X row (token ids), or null = identity
  const __nv_bfloat16* X;    // activations, bf16
  const CUtensorMap* xmap;   // TMA map of X (rows in node-row order) when gather is null
  long ldx;
  void* out;                 // fp32 or bf16
  long ldo;
  int out_f32;
  OpShape shape;
  const int* rank;
  int ncol_max;              // column tiles of the widest node of this op
  int ncb;                   // 64-row column blocks per tile
  // split-K: K-range s of a tile (kbs 64-wide K blocks) writes fp32 partial s
  // to split_out + s * split_stride (`out` is not written)
  int nsplit;
  int kbs;
  float* split_out;
  long split_stride;
  // in-launch dependency of a factor product on the rows another op of the
  // same launch writes: each consumer warp of a tile of `sig`'s op adds 1 to
  // sig[node * STREAM_DEP_TB + token block] once its half of the rows is
  // stored; a tile of `dep`'s op waits (bounded) until dep[...] reaches
  // 2 * ceil(dep_nrank * rank / 64), both halves of every column tile of its
  // node's producer op
  int* sig;
  const int* dep;
  int dep_nrank;
};

// Dynamic tile counters of the launches: 0 = the x-side streaming launch, 2 =
// the z-side one, N_STREAM_GROUPS + op = the tensor-core launch of op.
constexpr int N_STREAM_GROUPS = 4;

constexpr int STREAM_DEP_TB = 8;  // token blocks per node covered by the dependency counters

struct StreamLaunch {
  StreamOp op[3];
  int n_ops;
  // 1: the launch's weights and tile lists do not depend on the preceding
  // kernel (only its token rows do): the producer issues the first tile's
  // weight boxes before griddepcontrol.wait
  int early_weights;
  int* ctr;                  // tile counter of this launch (zeroed by the bucketing)
  int* err;                  // device error word (LX_ERR_TIMEOUT on a bounded wait)
  unsigned long long wait_cycles;  // bound of every wait (SM clock cycles)
  int unmet_wait;            // lx_wait_site whose wait is made to run out (test hook), 0 = none
};

// Tensor-core (prefill) grouped GEMM: one op per launch
struct TcLaunch {
  OpShape shape;
  const int* items;          // node ids of the op's plan
  int n_items;
  const int* tile_off;       // [n_items+1] tensor-core plan
  const int* node_off;
  const int* rank;
  const CUtensorMap* wmaps;  // [n_nodes] weight tensor maps of the op
  const CUtensorMap* xmap;   // TMA map of the A buffer (rows in node-row order)
  int xcol;                  // column offset of A inside xmap
  void* out;
  long ldo;
  int out_f32;
  long rows_cap;             // rows of the output buffer (bounds check)
  int* ctr;                  // dynamic tile counter (zeroed by the bucketing)
  int* err;
  unsigned long long wait_cycles;  // bound of every wait (SM clock cycles)
  int unmet_wait;            // lx_wait_site whose wait is made to run out (test hook), 0 = none
  int bm;                    // tile rows: 128 or 256 (tc_tile_rows of the op)
  int epi;                   // epilogue warps: 4 or 8
  // optional output remap (bf16 outputs): row r of the tile plan is stored at
  // row row_map[r], columns shifted by node_col[node] (null: identity)
  const int* row_map;
  const int* node_col;
  // optional K concatenation (anchor down tiles of flat layers): after its own
  // K, an anchor tile runs over each child c of kc_child[node] (CT_MAX_CH per
  // node, -1 padded) for rank(c) more: A from kc_xmap at columns j * kc_slot
  // (the child's slot j), B from kc_wmaps[c]
  const int* kc_child;
  const CUtensorMap* kc_wmaps;
  const CUtensorMap* kc_xmap;
  int kc_slot;
  // optional gathered A rows (in place of xmap): row r of the plan reads row
  // gather[r] of xsrc [.][ldx] (bf16), copied into shared memory by a warp
  const int* gather;
  const __nv_bfloat16* xsrc;
  long ldx;
  // optional TMA map of out (bf16, 32 x 32 boxes, 64-byte swizzle): 256-row
  // tiles store whole 32-row blocks with TMA (row_map null)
  const CUtensorMap* omap;
};

// Fused correction + SwiGLU of flat layers (every correction node a direct
// child of an anchor): children per anchor at most CT_MAX_CH.
constexpr int CT_MAX_CH = 7;

// ---------------------------------------------------------------------------
// device workspace of one forward
// ---------------------------------------------------------------------------
struct Workspace {
  int cap_T = 0, cap_k = 0;
  long rows_cap = 0;            // Rmax
  void* base = nullptr;
  size_t bytes = 0;
  // routing
  float* logits = nullptr;   // [T][E]
  int* topk_id = nullptr;    // [T][k]
  int* tile_cnt = nullptr;   // [router_tile_counters(T)] router slices done per token tile (self-resetting)
  float* topk_w = nullptr;   // [T][k]
  // bucketing
  uint8_t* marks = nullptr;  // [(N+E)][Tp]
  int* rank_in = nullptr;    // [(N+E)][Tp]
  int* key_cnt = nullptr;    // [N+E]
  int* key_off = nullptr;    // [N+1 + E+1]: node_off then expert_off
  int* node_tok = nullptr;   // [T*k*D]
  int* row_node = nullptr;   // [T*k*D]
  int* node_row = nullptr;   // [T*k*D]
  int* perm = nullptr;       // [T*k]
  int* tile_off = nullptr;   // [N_PLANS][max_items+1]
  // generic path intermediates (fp32)
  float* h = nullptr;        // [Rmax][2I]
  float* P = nullptr;        // [Rmax][2 rmax]
  float* z = nullptr;        // [Rmax][I]
  float* Q = nullptr;        // [Rmax][rmax]
  float* ypart = nullptr;    // [Rmax][H]
  // streaming and tensor-core path intermediates, bf16: pre-activations hb
  // [Rmax][2I] and down partials yb [Rmax][H] (aliasing h and ypart, which only
  // the generic path uses), and the operands of the next product
  __nv_bfloat16* hb = nullptr;
  __nv_bfloat16* yb = nullptr;
  __nv_bfloat16* Pb = nullptr;  // [Rmax][2 rmax]
  __nv_bfloat16* zb = nullptr;  // [Rmax][I]
  __nv_bfloat16* Qb = nullptr;  // [Rmax][rmax]
  int* act = nullptr;           // [STREAM_DEP_TB * (n_anchor + n_corr)] streaming work items:
                                // (anchor, token block) pairs, then (correction, token block)
  int* act_n = nullptr;         // [2] their counts
  int* sctr = nullptr;          // [sctr_ints] streaming / tensor-core tile counters, then the
                                // streaming launches' dependency counters [2][N][STREAM_DEP_TB]
  CUtensorMap* xmaps = nullptr; // [3] TMA maps of Pb, zb, Qb (tensor-core A operands)
  CUtensorMap* smaps = nullptr; // [3] the same buffers in streaming-tile boxes
  __nv_bfloat16* xg = nullptr;  // [Rmax][H] token rows in node-row order (tensor-core path)
  CUtensorMap* gmap = nullptr;  // TMA map of xg (tensor-core A operand boxes)
  // split-K partials of the anchor products on the streaming path (fp32):
  // [LX_STREAM_MAX_SPLIT][split_rows][2I] and [..][split_rows][H]
  float* hsplit = nullptr;
  float* ysplit = nullptr;
  long split_rows = 0;
  int* err = nullptr;           // device error word
  // fused correction + SwiGLU (flat layers): per anchor row a, the gates
  // al_g[a][0] (the dominant's, 0 if not selected) and al_g[a][1 + j] (child
  // slot j's), the child rows al_row[a][j] (-1: not selected), the anchor row
  // of every child row (rho2al), and the children's x V products aligned to
  // the anchor rows: Pal[a][j * 2 rmax + (0..2r)]
  float* al_g = nullptr;
  int* al_row = nullptr;
  int* rho2al = nullptr;
  __nv_bfloat16* Pal = nullptr;
  __nv_bfloat16* Qal = nullptr;  // [R][nch * rmax] the children's z Vd rows, aligned likewise
  CUtensorMap* pamap = nullptr;  // [3] TMA maps of Pal, hb and Qal (128-row boxes)
  CUtensorMap* omaps = nullptr;  // [2] TMA store maps of hb and yb (null: not encodable)
  // screened routing: the tensor-core logit partials [splits][T][Epad]
  float* rs_part = nullptr;
};

struct ProfRec {
  const char* name;
  cudaEvent_t a, b;
};

}  // namespace lx

struct lx_layer {
  int H = 0, I = 0, E = 0, N = 0, dtype = 0, esz = 0;
  int n_anchor = 0, n_corr = 0, max_depth = 0, max_rank = 0;
  int path_mode = LX_PATH_AUTO;
  int device = 0, num_sms = 0;
  std::vector<int> parent, rank, expert_node;
  std::vector<int> anchors, corrs;  // node ids
  // device copies of the tables
  int* d_rank = nullptr;
  int* d_paths = nullptr;           // [E][LX_MAX_DEPTH] node ids, -1 padded
  int* d_path_len = nullptr;        // [E]
  int* d_anchors = nullptr;
  int* d_corrs = nullptr;
  const void** d_w_up = nullptr;    // per node: anchor [Wg;Wu] [2I][H] | corr [Vg^T;Vu^T] [2r][H]
  const void** d_w_upU = nullptr;   // per node: corr [Ug;Uu] [2I][r] (null for anchors)
  const void** d_w_dn = nullptr;    // per node: anchor Wd [H][I] | corr Vd^T [r][I]
  const void** d_w_dnU = nullptr;   // per node: corr Ud [H][r] (null for anchors)
  CUtensorMap* d_tmaps = nullptr;   // [N_OPS][N] TMA descriptors (bf16 layers)
  bool stream_ok = false;           // the streaming kernels support this layer
  bool tiled = false;               // weights stored as 64x64 tiles (see lx_api.cu)
  std::vector<const void*> h_w_up, h_w_upU, h_w_dn, h_w_dnU;  // same, host copies
  void* router_w = nullptr;         // [E][H]
  float* router_bias = nullptr;     // [E] or null
  void* arena = nullptr;            // weights
  size_t arena_bytes = 0;
  void* tables = nullptr;           // small device tables
  lx::Workspace ws;
  int last_T = 0, last_k = 0;       // last bucketing
  bool profiling = false;
  bool pdl = true;                  // programmatic dependent launch between kernels
  unsigned long long wait_cycles = 0;  // bound of the kernels' device-side waits (0: default)
  int unmet_wait = 0;               // lx_wait_site made to run out (test hook), 0 = none
  // screened routing (large bf16 batches): approximate logits on the tensor
  // cores, exact canonical-order logits for the candidates only
  bool router_screen = false;
  float router_wmax = 0.f;          // max over experts of ||W_r[e]||_2
  CUtensorMap router_map;           // W_r [E][H], 64 x Epad boxes
  // fused correction + SwiGLU on the tensor-core path (flat layers)
  bool ct = false;
  int ct_nch = 0;                   // most children of an anchor (table stride)
  int* d_child = nullptr;           // [N][CT_MAX_CH] an anchor's children in node order, -1 padded
  int* d_child_col = nullptr;       // [N] column of a child's slot in Pal (j * 2 rmax), 0 for anchors
  int* d_child_qcol = nullptr;      // [N] column of a child's slot in Qal (j * rmax)
  std::vector<lx::ProfRec> prof;
  std::vector<cudaEvent_t> event_pool;
};

namespace lx {

// Default bound of every device-side wait: about 2 s at the GB300's clock.
constexpr unsigned long long kDefaultWaitCycles = 4000000000ull;
inline unsigned long long wait_limit(const lx_layer* L) {
  return L->wait_cycles ? L->wait_cycles : kDefaultWaitCycles;
}

// ints of the counter block zeroed by every bucketing
inline int sctr_ints(const lx_layer* L) { return N_TILE_COUNTERS + 2 * L->N * STREAM_DEP_TB; }

// Raises a kernel's dynamic shared-memory cap once per device (the flag array
// belongs to the calling launcher).
inline cudaError_t smem_cap_once(const void* func, int bytes, int device, bool (&done)[64]) {
  if (device >= 0 && device < 64 && done[device]) return cudaSuccess;
  const cudaError_t e =
      cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess && device >= 0 && device < 64) done[device] = true;
  return e;
}

// Kernel launch with programmatic dependent launch: the next kernel of the
// stream may be scheduled while this one drains, and every kernel of the
// library starts with griddepcontrol.wait (pdl_wait), which returns once its
// predecessor has completed and its writes are visible.  Off while profiling,
// so that the per-kernel events time one kernel each.  Launch errors surface
// through cudaGetLastError at the call site.
template <typename... KArgs, typename... Args>
inline void launch_k(const lx_layer* L, void (*kern)(KArgs...), dim3 grid, dim3 block,
                     size_t smem, cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = (L->pdl && !L->profiling) ? 1 : 0;
  (void)cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// Device side of the dependent launch: wait for the predecessor grid, then let
// the successor be scheduled on SMs this grid leaves free.
__device__ __forceinline__ void pdl_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Launch-time timing helper: records events around a launch when profiling.
struct ProfScope {
  lx_layer* L;
  cudaStream_t s;
  cudaEvent_t b = nullptr;
  const char* name;
  ProfScope(lx_layer* L_, cudaStream_t s_, const char* n);
  ~ProfScope();
};

// kernels / launchers (defined in the .cu files)
// need_logits = false: the caller reads only the ids and gates, so large bf16
// batches may take the screened path (logits of the candidates only)
lx_status launch_router(lx_layer* L, const void* x, int T, int k, float* logits, int* topk_id,
                        float* topk_w, cudaStream_t s, bool need_logits = true);
constexpr int RS_MAX_SPLITS = 8;
inline int router_epad(const lx_layer* L) { return (L->E + 15) / 16 * 16; }
bool router_is_tiled(const lx_layer* L, int T);
int router_tile_counters(int T);  // token tiles of the small-batch router
// plan_first: tile plans for the generic GEMMs (0), the tensor-core GEMMs
// (PLAN_TC), or none (-1)
lx_status launch_bucket(lx_layer* L, const int* topk_id, int T, int k, cudaStream_t s,
                        int plan_first);
lx_status launch_generic_experts(lx_layer* L, const void* x, int T, int k, void* y,
                                 cudaStream_t s);
// Anchor split-K partials the SwiGLU / combine kernels read for the anchor rows
// (the last node of each expert's path) in place of h / ypart: partial s of
// row r at part + s * stride + r * width, summed in split order.
struct SplitParts {
  const float* part = nullptr;
  int splits = 1;
  long stride = 0;
};
constexpr int LX_STREAM_MAX_SPLIT = 4;
bool warp_kernels_fit(const lx_layer* L, int k);
// bf16 = true: the streaming / tensor-core form (h = hb, z = zb, ypart = yb,
// all bf16); false: the generic form (fp32 h, z, ypart)
lx_status launch_swiglu(lx_layer* L, int T, int k, bool bf16, cudaStream_t s,
                        SplitParts hs = SplitParts());
// anchors_only: sum only the anchor rows of each token (their down tiles
// already hold the members' corrections)
lx_status launch_combine(lx_layer* L, int T, int k, void* y, bool bf16, cudaStream_t s,
                         SplitParts ys = SplitParts(), bool anchors_only = false);
lx_status launch_fast_experts(lx_layer* L, const void* x, int T, int k, void* y, cudaStream_t s);
lx_status launch_tc_experts(lx_layer* L, const void* x, int T, int k, void* y, cudaStream_t s);
int tc_tile_tokens();  // rows of the TMA boxes of the tensor-core A operands
int tc_tile_cols();
int tc_tile_rows(const lx_layer* L, int op);  // token rows of a tensor-core tile of op (its tile plan)
lx_status launch_tc(lx_layer* L, const TcLaunch& P, cudaStream_t s, const char* name);
// 2-D TMA map of a row-major bf16 matrix [outer][inner] read as box_inner x
// box_outer boxes with the 128-byte swizzle
bool encode_bf16_2d(CUtensorMap* m, const void* base, long inner, long outer, int box_inner,
                    int box_outer);
// the residual products of the member compression on the tensor cores
// (bf16 weights): C [M][N] = R X (transposed = false: M = rows, K = cols) or
// R^T X (M = cols, K = rows), R = Wm - Wd [rows][cols], X fp32 [K][N]
constexpr int RES_TC_MAX_SPLITS = 32;
size_t res_tc_workspace(long rows, long cols, long l);
bool res_tc_fits(long rows, long cols, long l);
lx_status res_gemm_tc(bool transposed, const __nv_bfloat16* Wm, const __nv_bfloat16* Wd,
                      long rows, long cols, const float* X, long N, float* C, char* ws,
                      int num_sms, int dev, cudaStream_t s);
// split-K tensor-core product part[s][M][Npad] = A . B^T over K range s (see
// lx_compress_tc.cu); the number of ranges used is returned in splits_out
lx_status tc_splitk_gemm_chunks(const CUtensorMap& a, const CUtensorMap& b, int M, int Npad,
                                int nz, int K, float* part, int max_splits, int* splits_out,
                                int num_sms, int dev, cudaStream_t s);
lx_status tc_splitk_gemm(lx_layer* L, const CUtensorMap& a, const CUtensorMap& b, int M, int Npad,
                         int K, float* part, int max_splits, int* splits_out, cudaStream_t s,
                         const char* name);
// fused correction + SwiGLU (flat layers): the kernel over (anchor, 128-row
// block, 64 d_ff columns); its per-cluster-row gate / child-row tables are
// written by the bucketing (k_assign_rows)
lx_status launch_ct_swiglu(lx_layer* L, cudaStream_t s);
constexpr int CT_CW = 64;  // d_ff columns of a fused tile
// row strides (4-byte words, 16-byte rows) of the per-anchor-row tables
inline int ct_gstride(const lx_layer* L) { return (1 + L->ct_nch + 3) / 4 * 4; }
inline int ct_rstride(const lx_layer* L) { return (L->ct_nch + 3) / 4 * 4; }
lx_status launch_stream(lx_layer* L, const StreamLaunch& P, cudaStream_t s, const char* name);
// plans = false: skip the generic GEMMs' tile plans (not read by the
// streaming kernels or by lx_get_buckets)
lx_status launch_bucket_small(lx_layer* L, const float* logits, const int* ids_in, int T, int k,
                              int* topk_id, float* topk_w, cudaStream_t s, bool plans = true);
bool bucket_small_fits(const lx_layer* L, int T, int k);
int stream_tile_rows();
int stream_tile_tokens();
int stream_box();

OpShape op_shape(const lx_layer* L, int op);
int op_max_items(const lx_layer* L);

}  // namespace lx
