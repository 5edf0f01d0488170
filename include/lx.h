/*
 * lx.h -- C ABI of the GB300 (sm_103a) LorExperts / BTExperts compressed-MoE
 * forward (arXiv 2608.07814).
 *
 * The layer (Sec. 3.1 "Representation", Sec. 5 "BTExperts") is a node table:
 *   - an ANCHOR node (parent -1, rank 0) stores full SwiGLU matrices
 *       gate [I][H], up [I][H], down [H][I]      (nn.Linear [out][in] row-major,
 *     the paper's W_e in R^{I x H} applied as x W^T, Sec. 2 and Sec. 5.1);
 *   - a CORRECTION node (parent >= 0, rank r > 0) stores, per projection, the
 *     factors of W_m ~ W_dom + B_m A_m (Sec. 3.1) as U = B_m [out][r] and
 *     V = A_m^T [in][r]:  Ug [I][r], Vg [H][r], Uu [I][r], Vu [H][r],
 *     Ud [H][r], Vd [I][r]   (row-major);
 *   - expert e is the sum of the contributions on the root path of
 *     expert_node[e]:  W_e = W_anchor + sum_{corrections n on the path} s_n U_n V_n^T,
 *     s_n = +1 unless the descriptor labels the edge into n with -1 (Fig. 2).
 * Flat LorExperts: one anchor per cluster (the dominant maps to it, so it
 * carries no correction) and one rank-r child per member; a protection-set
 * singleton is an anchor without children.  BTExperts: anchors are tree roots
 * (which need not be experts), corrections at any depth <= LX_MAX_DEPTH - 1,
 * e.g. Fig. 2's binary tree with signed edges and experts at the leaves.  A
 * single shared base (Sec. 5.2's single-shared-component layout) is one anchor
 * that is no expert, with every expert a correction below it.
 *
 * The forward (Sec. 5.1: each shared product evaluated once per token) routes every
 * token top-k over all E experts with the unchanged router (Sec. 1, Fig. 1),
 * evaluates each anchor's product once per (token, anchor) and each correction
 * once per (token, node), applies SwiGLU per selected expert and combines
 * y_t = sum_s g_{t,s} W_{e_s}^down act_{t,s}, using linearity so that the
 * down-projection of shared nodes is also evaluated once per (token, node).
 *
 * Conventions for every call:
 *   - All device pointers are caller-owned CUDA device memory of the current
 *     device; host pointers are only read during the call.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *     Work is enqueued on it; no call synchronises the host except
 *     lx_load_compressed_layer, lx_reserve (and a forward that has to grow its
 *     workspace), lx_layer_info's row count and lx_read_profile.
 *   - Errors are returned as lx_status; lx_last_error() gives a message for the
 *     calling thread.  Arguments are validated on the host before any launch;
 *     an invalid call launches nothing.  T == 0 is a valid no-op.
 *   - A layer may be used from one host thread at a time.
 */
#ifndef LX_H_
#define LX_H_

#include <stdint.h>

#if defined(__GNUC__)
#define LX_API __attribute__((visibility("default")))
#else
#define LX_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

#define LX_MAX_DEPTH 4   /* nodes on a root path, anchor included */
#define LX_MAX_K 32      /* router top-k */
#define LX_MAX_EXPERTS 1024

typedef enum {
  LX_OK = 0,
  LX_ERR_ARG = 1,          /* null pointer, k out of range, bad option */
  LX_ERR_SHAPE = 2,        /* inconsistent or unsupported sizes / node table */
  LX_ERR_CUDA = 3,         /* a CUDA runtime call failed */
  LX_ERR_OOM = 4,          /* device allocation failed */
  LX_ERR_TIMEOUT = 5,      /* a bounded device-side wait gave up */
  LX_ERR_STATE = 6,        /* call out of order (e.g. buckets before a forward) */
  LX_ERR_UNSUPPORTED = 7   /* valid request the library does not implement */
} lx_status;

typedef enum { LX_F32 = 0, LX_BF16 = 1 } lx_dtype;

typedef struct lx_layer lx_layer; /* opaque, library-owned */

typedef struct {
  int32_t d_model;            /* H */
  int32_t d_ff;               /* I */
  int32_t n_experts;          /* E, 1..LX_MAX_EXPERTS */
  int32_t n_nodes;            /* >= 1 */
  int32_t dtype;              /* lx_dtype of weights, x and y */
  const int32_t* node_parent; /* host [n_nodes]: -1 for an anchor, else parent id */
  const int32_t* node_rank;   /* host [n_nodes]: 0 for an anchor, 1..min(I,H) else */
  const int32_t* expert_node; /* host [n_experts]: node defining expert e */
  const int8_t* node_sign;    /* host [n_nodes] or NULL: sign s_n in {+1, -1} of the edge
                                 into node n (Fig. 2 labels the edges of the BTExperts tree
                                 -1/+1); a correction then contributes s_n U_n V_n^T.
                                 Anchors must carry +1.  NULL = every edge +1. */
} lx_layer_desc;

/*
 * Load ("install", Sec. 3.2 Stage 3 iii) a compressed layer.
 *   node_w:      host array of 6*n_nodes host pointers.  For an anchor n:
 *                node_w[6n+0..2] = gate, up, down; node_w[6n+3..5] unused.
 *                For a correction n: node_w[6n+0..5] = Ug, Vg, Uu, Vu, Ud, Vd.
 *                Element type = desc->dtype (bf16 as uint16 bit patterns).
 *   router_w:    host [E][H] (desc->dtype).
 *   router_bias: host [E] fp32 added to the logits, or NULL.
 * Copies (and repacks) everything to device memory owned by the layer; a
 * correction whose edge sign is -1 is stored with negated U factors (exact), so
 * every kernel sees an unsigned tree.  Synchronises `stream`.  Errors:
 * LX_ERR_ARG (null pointers), LX_ERR_SHAPE (sizes, cycles, depth >
 * LX_MAX_DEPTH, anchor with rank != 0, correction rank outside 1..min(I,H),
 * H or I not a multiple of 8, a sign other than +1/-1 or an anchor sign of -1),
 * LX_ERR_OOM, LX_ERR_CUDA.
 */
LX_API lx_status lx_load_compressed_layer(const lx_layer_desc* desc, const void* const* node_w,
                                   const void* router_w, const float* router_bias,
                                   void* stream, lx_layer** out);

/* Releases all device memory of the layer (synchronises the device first). */
LX_API lx_status lx_free_layer(lx_layer* layer);

/*
 * Pre-sizes the layer's device workspace for up to max_tokens tokens with
 * top-k (synchronous).  A forward with more tokens grows the workspace itself
 * (and then synchronises its stream once).
 */
LX_API lx_status lx_reserve(lx_layer* layer, int32_t max_tokens, int32_t k);

/*
 * Router (Sec. 1, Fig. 1): logits l = x W_r^T (+ bias) in the canonical fp32
 * order (H in chunks of 8; lane j = chunk mod 32 accumulates its chunks with
 * fused multiply-adds in ascending h; the 32 partials are added pairwise at
 * offsets 16, 8, 4, 2, 1; then the bias), top-k by (logit desc, id asc),
 * gates = softmax over the k selected logits (fp32).
 *   x:       device [T][H] (layer dtype)
 *   topk_id: device [T][k] int32 out;  topk_w: device [T][k] fp32 out
 *   logits:  device [T][E] fp32 out, or NULL
 * With logits == NULL, large bf16 batches (at least 8 tokens per SM; H a
 * multiple of 64, E <= 256) may take the screened form: approximate logits on
 * the tensor cores, and the canonical logits only of the experts whose
 * approximate logit is within twice a proven error bound of the k-th largest
 * (a set that contains the exact top-k); topk_id and topk_w are then identical
 * to the full router's, bit for bit.  lx_moe_forward routes this way.
 * Also leaves the routing in the layer for lx_bucket / lx_get_buckets.
 * Errors: LX_ERR_ARG (k < 1, k > min(E, LX_MAX_K), T < 0, null pointers).
 */
LX_API lx_status lx_route(lx_layer* layer, const void* x, int32_t T, int32_t k, int32_t* topk_id,
                   float* topk_w, float* logits, void* stream);

/*
 * Bucketing of given assignments (device [T][k] int32 expert ids, each row
 * holding k distinct ids in [0, E)): per node the ascending list of tokens
 * whose selected experts' root paths contain the node, per (assignment, path
 * level) the row of that (token, node) pair, and per expert its assignments in
 * ascending token order.  Results stay in the layer (lx_get_buckets).
 */
LX_API lx_status lx_bucket(lx_layer* layer, const int32_t* topk_id, int32_t T, int32_t k,
                    void* stream);

/*
 * The compressed-MoE forward (Sec. 5.1: a dominant's or ancestor's product is
 * evaluated one time per token and reused by every selected expert below it;
 * Sec. 3.1: a member's projection is W_dom + B_m A_m, never re-materialised): route, bucket, shared anchor GEMMs with the low-rank
 * corrections and SwiGLU, down-projection and weighted combine.
 *   x: device [T][H], y: device [T][H] (layer dtype), both 16-byte aligned;
 *   y may not overlap x.
 * Kernels: bf16 layers whose H, I and ranks are multiples of 64 (with k <= 8,
 * k * max_depth <= 32) take the weight-streaming kernels for T <= 256 and the
 * tcgen05 tensor-core kernels above; every other layer, and LX_PATH_GENERIC,
 * the CUDA-core kernels.  All products accumulate in fp32; on the streaming
 * and tensor-core paths the intermediates that cross device memory (the
 * gate/up pre-activations, x V, the SwiGLU aggregate, z Vd and the down
 * partials) are stored as bf16, on the CUDA-core path as fp32.
 * Errors: LX_ERR_ARG (k, T, alignment, aliasing, null pointers), LX_ERR_OOM /
 * LX_ERR_CUDA while growing the workspace; a kernel's bounded wait that gave up
 * is reported by lx_layer_info (device_error).
 */
LX_API lx_status lx_moe_forward(lx_layer* layer, const void* x, int32_t T, int32_t k, void* y,
                         void* stream);

/*
 * Copies the last bucketing (from lx_bucket, lx_route or lx_moe_forward) into
 * caller device buffers (stream-ordered).  The buckets are the (token, node)
 * pairs whose products the forward evaluates once and shares (Sec. 5.1): node
 * n's bucket holds every token that selected an expert whose root path
 * contains n.  With D = info.max_depth:
 *   node_off   [n_nodes+1]  exclusive prefix of the node bucket sizes
 *   node_tok   [T*k*D]      capacity; first node_off[n_nodes] entries written:
 *                           node n's tokens ascending, nodes in id order
 *   node_row   [T*k*D]      row of (t, path(e)[l]) for assignment a = t*k+s at
 *                           index a*D + l, -1 beyond the path's end
 *   expert_off [E+1]        exclusive prefix of the per-expert firing counts N_e
 *   perm       [T*k]        assignments a = t*k+s ordered by (expert, token)
 * Any pointer may be NULL (that output is skipped).  LX_ERR_STATE if nothing
 * has been bucketed yet.
 */
LX_API lx_status lx_get_buckets(lx_layer* layer, int32_t* node_off, int32_t* node_tok,
                         int32_t* node_row, int32_t* expert_off, int32_t* perm, void* stream);

typedef struct {
  int32_t d_model, d_ff, n_experts, n_nodes, dtype;
  int32_t n_anchors, n_corrections, max_depth, max_rank;
  int64_t weight_bytes;       /* device bytes of the repacked weights + router */
  int32_t last_T, last_k;     /* sizes of the last bucketing (0 if none) */
  int32_t last_rows;          /* node_off[n_nodes] of the last bucketing (synchronises) */
  int32_t device_error;       /* lx_status recorded by a kernel (e.g. LX_ERR_TIMEOUT when a
                                 bounded device-side wait gave up), 0 if none (synchronises) */
  int32_t stream_path;        /* 1 if the weight-streaming (T <= 256) and tcgen05 (T > 256)
                                 kernels serve the layer under LX_PATH_AUTO */
} lx_layer_info_t;

LX_API lx_status lx_layer_info(lx_layer* layer, lx_layer_info_t* info);

/* Execution paths.  LX_PATH_AUTO picks the fastest kernels that support the
 * layer and batch; LX_PATH_GENERIC forces the plain CUDA-core kernels (every
 * dtype and shape). */
typedef enum { LX_PATH_AUTO = 0, LX_PATH_GENERIC = 1 } lx_path;
LX_API lx_status lx_set_path(lx_layer* layer, int32_t path);

/*
 * Kernel timing.  While enabled, every kernel the layer launches is bracketed by
 * CUDA events on its stream (and kernels are launched without programmatic
 * dependent launch, so each event pair times one kernel; the events add the
 * launch latency to each).  lx_read_profile synchronises on the last event,
 * writes up to `cap` records of the launches since the previous read (oldest
 * first) and clears the list; *n receives the number written.
 */
typedef struct {
  const char* name;  /* static string */
  float ms;          /* device time between the bracketing events */
} lx_kernel_time;
LX_API lx_status lx_set_profiling(lx_layer* layer, int32_t enable);
LX_API lx_status lx_read_profile(lx_layer* layer, lx_kernel_time* out, int32_t cap, int32_t* n);

/*
 * Bounded device-side waits.  The kernels wait in two places: the weight
 * streaming kernels (T <= 256) wait inside a launch for the rows another tile
 * of the same launch writes (a factor product U after its x V), and every
 * kernel with a TMA/tensor-core pipeline waits on shared-memory barriers.
 * Each wait gives up after a bound, records LX_ERR_TIMEOUT in the layer's
 * device error word (lx_layer_info's device_error), makes the CTA's other
 * roles stop, lets the CTA's copies and tensor-core operations in flight
 * finish and frees its tensor memory; the launch then ends normally, so the
 * CUDA context stays usable, and that forward's output is undefined.
 *
 * lx_set_wait_limit: the bound in SM clock cycles of every later wait of the
 * layer's kernels (0 restores the default, 4e9 cycles, about 2 s at the GB300's
 * clock).  Copies that are already in flight are always waited for with the
 * default bound.  Errors: LX_ERR_ARG (NULL layer).
 *
 * lx_inject_unmet_wait (test hook): from the next forward on, the wait at
 * `site` waits for a condition that nothing fulfils -- LX_WAIT_STREAM_DEP: one
 * arrival more than the streaming producer tiles make; LX_WAIT_TC_MMA: a
 * barrier that only the abort path arrives on, before the tensor-core MMA
 * issuer's first tile -- so that it runs out after the bound.  LX_WAIT_NONE
 * turns the hook off.  Errors: LX_ERR_ARG (NULL layer, unknown site).
 *
 * lx_clear_device_error: zeroes the device error word (stream-ordered on the
 * legacy default stream; synchronises the device).  Errors: LX_ERR_ARG.
 */
typedef enum { LX_WAIT_NONE = 0, LX_WAIT_STREAM_DEP = 1, LX_WAIT_TC_MMA = 2 } lx_wait_site;
LX_API lx_status lx_set_wait_limit(lx_layer* layer, uint64_t cycles);
LX_API lx_status lx_inject_unmet_wait(lx_layer* layer, int32_t site);
LX_API lx_status lx_clear_device_error(lx_layer* layer);

/*
 * Size of the fixed device array that lx_bucket_noalloc uses as scratch.  The
 * array is a static device variable of the library, so every GPU on which the
 * library's code is loaded holds these bytes until the process exits.
 */
#define LX_NOALLOC_SCRATCH_BYTES (16u << 20)

/*
 * lx_bucket_noalloc -- the bucketing of lx_bucket, for callers that must not
 * allocate device memory during the call.  The paper has no counterpart; this
 * is an integration entry point.
 *
 * Who needs it: serving runtimes that hand all device memory to their own
 * pooling allocator or run under a fixed memory budget, and latency-critical
 * loops in which cudaMalloc/cudaFree are not allowed because they can
 * synchronise the device and fragment memory.  lx_bucket itself may grow the
 * layer's workspace with cudaMalloc; this variant never allocates: its
 * temporary buffers (per-(node|expert, token) marks and ranks, counts and
 * offsets) live in one static device array of LX_NOALLOC_SCRATCH_BYTES bytes.
 *
 * Arguments: as lx_bucket, plus caller-owned device outputs in the layout of
 * lx_get_buckets (all required, D = max path length of the layer):
 *   node_off [n_nodes+1], node_tok [T*k*D] (capacity), node_row [T*k*D],
 *   expert_off [E+1], perm [T*k].
 * Must be called with the layer's device current.  The first call on a device
 * looks up the array's device address (cudaGetSymbolAddress) and caches it;
 * make that first call before any stream capture.  With keys = n_nodes + E
 * and Tp = round_up(T, 16), the call needs
 *   r(keys*Tp) + r(4*keys*Tp) + r(4*keys) + r(4*(keys+2)) + r(4*T*k*D)
 * bytes of the array, r(v) = v rounded up to 256, and returns LX_ERR_SHAPE,
 * launching nothing, when that exceeds LX_NOALLOC_SCRATCH_BYTES (the
 * Qwen3-30B-A3B-shaped layer, keys = 256, k = 8, D = 2: T <= 12480).
 * T == 0 writes zeros to node_off and expert_off (if not NULL) and nothing else.
 * All calls in the process share the one array per device and the array keeps
 * the previous call's contents (the call clears what must start at zero):
 * calls whose GPU work can overlap (different streams, or different layers on
 * concurrent streams) race on it and must be serialised by the caller.
 * Results do not update the layer's own bucketing (lx_get_buckets).
 */
LX_API lx_status lx_bucket_noalloc(lx_layer* layer, const int32_t* topk_id, int32_t T, int32_t k,
                                   int32_t* node_off, int32_t* node_tok, int32_t* node_row,
                                   int32_t* expert_off, int32_t* perm, void* stream);

/*
 * Router profiling statistics (Sec. 3.2 Stage 1 accumulates per-layer firing
 * counts N_e by reading the router; Sec. 2.2 weights the expert co-activation
 * graph by normalised pointwise mutual information, NPMI, and Stage 2's
 * Coact-NPMI variant clusters on 1 - NPMI).  Standalone: no layer needed.
 *
 * lx_coact_accumulate ADDS one batch of top-k assignments to the counters:
 *   topk_id: device [T][k] int32.  A token's selected set is the set of its ids
 *            in [0, E); ids outside are skipped and a repeated id counts once.
 *   fire:    device [E] uint64 or NULL:  fire[e] += tokens whose set holds e (N_e)
 *   coact:   device [E][E] uint64 row-major or NULL:  coact[i][j] += tokens
 *            whose set holds both i and j; coact[i][i] += N_i.
 * The caller zeroes the counters before the first batch; counts are exact
 * (integer) and independent of launch order.  Stream-ordered; no allocation.
 * Errors: LX_ERR_ARG (T < 0, k outside 1..LX_MAX_K, E outside
 * 1..LX_MAX_EXPERTS, fire and coact both NULL, topk_id NULL with T > 0).
 * T == 0 is a no-op.
 */
LX_API lx_status lx_coact_accumulate(const int32_t* topk_id, int32_t T, int32_t k, int32_t E,
                                     uint64_t* fire, uint64_t* coact, void* stream);

/*
 * lx_coact_npmi: NPMI matrix of accumulated counts over n_tokens tokens, in
 * float64:  with p_i = coact[i][i] / n and p_ij = coact[i][j] / n,
 *   npmi[i][j] = ln(p_ij / (p_i p_j)) / (-ln p_ij)   for 0 < p_ij < 1,
 *              = -1 for p_ij = 0 (never together), +1 for p_ij = 1.
 *   coact: device [E][E] uint64 (from lx_coact_accumulate); npmi: device [E][E]
 *   double out.  Errors: LX_ERR_ARG (E out of range, n_tokens < 0, NULL).
 */
LX_API lx_status lx_coact_npmi(const uint64_t* coact, int32_t E, int64_t n_tokens, double* npmi,
                               void* stream);

/*
 * Neuron alignment of a member expert to its dominant (Sec. 3.2 Stage 3 (i)).
 * Standalone: the experts are given as plain matrices, not as a layer.
 * Neuron i of an expert is a_i = (gate[i][:], up[i][:], down[:][i]), length 3H.
 *
 * lx_align_cost: C[i][j] = ||a_i||^2 + ||b_j||^2 - 2 a_i . b_j (Eq. cost) for
 * dominant neurons a_i and member neurons b_j, fp32 accumulation.
 *   dtype: LX_F32 or LX_BF16 (bf16 as uint16 bit patterns); d_model H, d_ff I
 *          multiples of 8.
 *   dom_gate, dom_up, mem_gate, mem_up: device [I][H]; dom_down, mem_down:
 *          device [H][I] (row-major, the x W^T storage of lx_load_compressed_layer);
 *   cost:  device [I][I] fp32 out.  Every pointer 16-byte aligned.
 * Stream-ordered; no allocation.  Errors: LX_ERR_ARG (dtype, NULL, alignment),
 * LX_ERR_SHAPE (sizes).
 */
LX_API lx_status lx_align_cost(int32_t dtype, int32_t d_model, int32_t d_ff,
                               const void* dom_gate, const void* dom_up, const void* dom_down,
                               const void* mem_gate, const void* mem_up, const void* mem_down,
                               float* cost, void* stream);

/*
 * lx_lap_solve (host): the permutation P minimising sum_i cost[i][P(i)]
 * (Eq. assign), solved exactly (shortest augmenting paths with dual
 * potentials, the scheme of Jonker and Volgenant; float64 arithmetic, O(n^3)).
 *   cost:   HOST [n][n] fp32 (e.g. copied back from lx_align_cost), finite;
 *   assign: HOST [n] int32 out, assign[i] = P(i);
 *   total:  HOST double out (sum_i cost[i][P(i)] in float64), or NULL.
 * Among several optimal permutations any one may be returned.  Errors:
 * LX_ERR_ARG (n outside 1..65536, NULL, a NaN or infinite cost).
 */
LX_API lx_status lx_lap_solve(const float* cost, int32_t n, int32_t* assign, double* total);

/*
 * lx_lap_solve_batch (host): lx_lap_solve for `count` independent problems
 * (e.g. every member of a layer), spread over `threads` host threads
 * (<= 0: the hardware concurrency).
 *   costs:  HOST [count][n][n] fp32;  assign: HOST [count][n] int32 out;
 *   totals: HOST [count] double out, or NULL.
 * Every cost is checked before any problem is solved.  Errors: LX_ERR_ARG
 * (n outside 1..65536, count < 0, NULL, a NaN or infinite cost).
 */
LX_API lx_status lx_lap_solve_batch(const float* costs, int32_t n, int32_t count, int32_t* assign,
                                    double* totals, int32_t threads);

/*
 * lx_permute_neurons: the aligned member, neuron i <- neuron perm[i]:
 *   gate_out[i][:] = gate[perm[i]][:], up_out likewise,
 *   down_out[:][i] = down[:][perm[i]]   (bit-exact copies).
 *   perm: device [I] int32, a permutation of 0..I-1 (an entry outside that
 *         range yields a zero neuron);  weights as lx_align_cost, outputs
 *         device buffers of the same shapes that overlap no input.
 * Stream-ordered; no allocation.  Errors: LX_ERR_ARG (dtype, NULL, alignment,
 * overlap), LX_ERR_SHAPE (sizes).
 */
LX_API lx_status lx_permute_neurons(int32_t dtype, int32_t d_model, int32_t d_ff,
                                    const int32_t* perm, const void* gate, const void* up,
                                    const void* down, void* gate_out, void* up_out, void* down_out,
                                    void* stream);

/*
 * Compression of one member projection (Sec. 3.2 Stage 3 (ii)): the residual
 * R = W_mem - W_dom (Eq. svd; W_mem already aligned) and its rank-r randomized
 * SVD with the symmetric split of Eq. factors:
 *   U = U_r S_r^(1/2) [rows][r] (the paper's B_m),  V = V_r S_r^(1/2) [cols][r]
 *   (A_m^T), so that U V^T ~ R, plus the singular values s [r].
 * Solver: Y = R Omega, Q = orth(Y); power_iters times Q = orth(R orth(R^T Q));
 * then the SVD of Bs = Q^T R: Z = R^T Q is orthonormalised too, Z = Z2 M^T with
 * M the l x l triangular factor, and the small SVD of M (one-sided Jacobi)
 * gives Bs's.  orth is CholeskyQR run twice (float64 Gram sums, fp32 Cholesky;
 * the first pass is shifted by 1e-6 of the largest Gram diagonal); the
 * products with R are fp32 (CUDA cores); singular values are float64 Rayleigh
 * quotients.  The sign of each factor column is fixed so that the
 * largest-magnitude entry of U's column is positive.  Singular values at or
 * below 1e-6 of the largest give zero U and V columns.  The call is latency
 * bound (one-CTA stages): independent projections run concurrently when given
 * their own streams and workspaces.
 *   dtype:      LX_F32 or LX_BF16 of w_dom / w_mem
 *   rows, cols: the projection's [out][in] shape, multiples of 8 (gate / up:
 *               [I][H], down: [H][I]); w_dom, w_mem device, 16-byte aligned
 *   omega:      device [cols][l] fp32, the Gaussian test matrix (the caller
 *               draws it: the random numbers are an input)
 *   l, r:       1 <= r <= l <= min(rows, cols, 256) (l = r + oversampling)
 *   power_iters 0..16
 *   U, V, s:    device fp32 outputs [rows][r], [cols][r], [r]
 *   workspace:  device, 256-byte aligned, >= lx_compress_workspace bytes
 *               (caller-owned; nothing is allocated)
 * Stream-ordered.  Errors: LX_ERR_ARG (dtype, NULL, alignment, power_iters,
 * workspace too small), LX_ERR_SHAPE (sizes).
 */
LX_API lx_status lx_compress_workspace(int32_t rows, int32_t cols, int32_t l, int32_t r,
                                       uint64_t* bytes);
LX_API lx_status lx_compress_factor(int32_t dtype, int32_t rows, int32_t cols, const void* w_dom,
                                    const void* w_mem, const float* omega, int32_t l, int32_t r,
                                    int32_t power_iters, float* U, float* V, float* s,
                                    void* workspace, uint64_t workspace_bytes, void* stream);

/* Message of the last failed call on this thread ("" if none). */
LX_API const char* lx_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* LX_H_ */
