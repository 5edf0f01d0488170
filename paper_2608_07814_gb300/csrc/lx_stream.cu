// Weight-streaming grouped GEMM for small token counts (decode).
//
// out[rows of node n][cols] = X[rows][K] . W_n[cols][K]^T for every active node,
// where X holds at most 32 rows per tile.  Decode is bound by reading each
// touched weight byte once from HBM (Sec. 5.2: the projections run at about one
// FLOP per byte), so the kernel is organised around the weight stream:
//
//   * one tile = 64 weight rows (output columns) x 32 tokens of one node,
//     over the full K or, for the anchors, one of up to four K ranges (split-K:
//     every range writes an fp32 partial that the next kernel adds in order),
//     so that the tiles left at the end of a launch are short;
//   * a producer warp streams the tile's weights with TMA loads
//     (cp.async.bulk.tensor, 64x64 bf16 boxes, 128-byte swizzle) into a
//     3-stage shared-memory ring guarded by mbarriers;
//   * two consumer warps (32 weight rows each) multiply with mma.sync
//     m16n8k16 (weights as the 16-row operand, tokens as the 8-column
//     operand).  Inside each 64-wide K box the contraction index is
//     permuted so that every lane reads 8 consecutive K values of a weight
//     row and of a token row (16-byte shared loads, conflict-free under the
//     128-byte swizzle); the same permutation on both operands leaves the sum
//     unchanged;
//   * persistent CTAs claim tiles from a device-built list of (node, token
//     block) work items, each near the end of the previous tile; every mbarrier wait is
//     bounded, and a wait that gives up records LX_ERR_TIMEOUT in a device
//     word and drains the CTA's copies in flight before returning.
#include <cuda.h>

#include <algorithm>
#include <initializer_list>


#include "lx_internal.cuh"

namespace lx {

namespace {

constexpr int SW_ROWS = 64;         // weight rows per tile
// Tokens per tile.  Decode buckets are small (at 64 tokens top-8 over 32
// clusters the median anchor bucket holds a handful of tokens), so a 32-token
// slot keeps the stage at 12 KiB and five CTAs of three stages fit an SM (more
// CTAs streaming measured faster than fewer CTAs with deeper rings).  Larger
// buckets take several token blocks.
constexpr int SW_TOK = 32;
constexpr int SW_BOX = 64;          // K per stage = one TMA box of 64 K x 64 rows
constexpr int SW_BOX_BYTES = SW_BOX * SW_ROWS * 2;
// Token rows of a stage: SW_TOK rows x 128 bytes in the 128-byte swizzle (the
// layout a TMA box of contiguous rows lands in; gathered rows are written in
// the same layout by cp.async).
constexpr int SW_XBYTES = SW_TOK * SW_BOX * 2;
constexpr int SW_STAGE_BYTES = SW_BOX_BYTES + SW_XBYTES;
constexpr int SW_STAGES = 3;
// bf16 output staging per consumer warp: SW_TOK token rows of its 32 output
// columns, rows padded to 80 bytes (conflict-free writes and 16-byte reads)
constexpr int SW_OST = 40;
constexpr int SW_OST_BYTES = 2 * SW_TOK * SW_OST * 2;
constexpr int SW_CTAS_PER_SM = 5;
constexpr int SW_CONSUMERS = 2;
constexpr int SW_MT = SW_ROWS / (16 * SW_CONSUMERS);  // 16-row MMA tiles per consumer warp
constexpr int SW_THREADS = 32 * (1 + SW_CONSUMERS);
constexpr unsigned long long SW_TIMEOUT_CYCLES = 4000000000ull;  // ~2 s
// stages of the current tile still to be issued when the next tile is decoded
// (measured at a decode batch of 64: 1 before 3 before 6)
constexpr int kClaimLead = 1;
static_assert(SW_STAGE_BYTES % 1024 == 0, "stages must keep the 128B-swizzle alignment");
static_assert(SW_TOK % 8 == 0 && SW_TOK <= 64, "token slot: whole 8-token MMA columns");

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

// Consumer release of a stage.  The stage's shared-memory reads are complete
// (their values fed the MMAs before this point in program order), so no
// release ordering is needed -- which keeps the arrive from waiting on the
// consumer's earlier global stores.
__device__ __forceinline__ void mbar_arrive_relaxed(uint32_t bar) {
  asm volatile("mbarrier.arrive.relaxed.cta.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

// try_wait with a suspend-time hint: a waiting thread is parked by the
// hardware (up to ~0.5 us per call) instead of spinning on issue slots that
// the working warps of the SM need.
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(500)
      : "memory");
  return ok != 0;
}

// Bounded wait: false if the phase did not complete within `limit` SM clock
// cycles or the CTA aborted.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          unsigned long long limit) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = clock64();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (clock64() - t0 > limit) return false;
  }
}

// Bounded wait for an in-launch dependency counter (acquire); false on
// timeout or when the CTA aborts.
__device__ __forceinline__ bool dep_wait(const int* p, int need, volatile int* abort_flag,
                                         unsigned long long limit) {
  const unsigned long long t0 = clock64();
  while (true) {
    int v;
    asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    if (v >= need) return true;
    if (*abort_flag) return false;
    if (clock64() - t0 > limit) return false;
    __nanosleep(128);
  }
}

// L2 policy of the weight boxes: every weight byte is read once per launch, so
// its lines are evicted first and the activations, factor projections and
// split-K partials the launch writes stay in L2 for the kernels that read them.
__device__ __forceinline__ uint64_t evict_first_policy() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// one 64x64 tile (box) of a tiled weight matrix: K tile kt of row tile rt
__device__ __forceinline__ void tma_load_tile(uint32_t dst, const CUtensorMap* map, int kt, int rt,
                                              uint32_t bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%2, %3, %4, %5}], [%6], %7;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(0), "r"(0), "r"(kt), "r"(rt), "r"(bar),
      "l"(policy)
      : "memory");
}

// SW_TOK contiguous rows x 64 columns of a bf16 activation buffer (2-D map)
__device__ __forceinline__ void tma_load_rows(uint32_t dst, const CUtensorMap* map, int col,
                                              int row, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(col), "r"(row), "r"(bar)
      : "memory");
}
// 16-byte asynchronous copy global -> shared on the load/store path (cp.async);
// the TMA unit is kept for the weight boxes, whose requests it serialises.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst),
               "l"(reinterpret_cast<uint64_t>(src))
               : "memory");
}

// arrive on `bar` once this thread's earlier cp.async copies have landed
__device__ __forceinline__ void cp_async_arrive(uint32_t bar) {
  asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint4 lds_v4(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr));
  return v;
}

struct TileInfo {
  int op, node, grp, row0, tok0, M, Ng, K, ncb;
  int tb;               // token block of the node's bucket
  int kb0, nkb, split;  // K blocks [kb0, kb0 + nkb) of split `split`
  bool active;
};

__device__ __forceinline__ int op_tiles(const StreamOp& op) {
  return *op.n_active * op.shape.groups * op.ncol_max * op.nsplit;
}

// Tile index -> (op, node, token block, group, column tile, K split).
// tiles0 / tiles1: first tile of op 1 / op 2 (the ops' tiles are consecutive)
__device__ __forceinline__ void decode_tile(const StreamLaunch& P, int tile, int tiles0,
                                            int tiles1, TileInfo& ti) {
  int o = 0, local = tile;
  if (P.n_ops > 2 && tile >= tiles1) {
    o = 2;
    local = tile - tiles1;
  } else if (P.n_ops > 1 && tile >= tiles0) {
    o = 1;
    local = tile - tiles0;
  }
  const StreamOp& op = P.op[o];
  // (work item = node and token block, group, column tile, split), split fastest
  const int per_item = op.shape.groups * op.ncol_max * op.nsplit;
  const int item = local / per_item;
  int rem = local - item * per_item;
  const int grp = rem / (op.ncol_max * op.nsplit);
  rem -= grp * op.ncol_max * op.nsplit;
  const int ct = rem / op.nsplit, split = rem - ct * op.nsplit;
  const int packed = op.items[item];
  const int n = packed / STREAM_DEP_TB, tb = packed - n * STREAM_DEP_TB;
  const int r = op.rank[n];
  const int b0 = op.node_off[n], b1 = op.node_off[n + 1];
  ti.op = o;
  ti.tb = tb;
  ti.node = n;
  ti.grp = grp;
  ti.row0 = ct * SW_ROWS * op.ncb;
  ti.Ng = op.shape.n_const + op.shape.n_rank * r;
  ti.K = op.shape.k_const + op.shape.k_rank * r;
  ti.tok0 = b0 + tb * SW_TOK;
  ti.M = min(SW_TOK, b1 - ti.tok0);
  ti.ncb = min(op.ncb, (ti.Ng - ti.row0 + SW_ROWS - 1) / SW_ROWS);
  const int nkb_all = (ti.K + SW_BOX - 1) / SW_BOX;
  ti.split = split;
  ti.kb0 = split * op.kbs;
  ti.nkb = min(op.kbs, nkb_all - ti.kb0);
  ti.active = ti.M > 0 && ti.row0 < ti.Ng && ti.nkb > 0;
}

template <int NT>
__device__ __forceinline__ bool consume_tile(const StreamLaunch& P, const TileInfo& ti,
                                             uint32_t smem_base, uint32_t full0, uint32_t empty0,
                                             uint32_t& it, volatile int* abort_flag,
                                             __nv_bfloat16* ost) {
  const StreamOp& op = P.op[ti.op];
  const int lane = threadIdx.x & 31, cw = (threadIdx.x >> 5) - 1;
  const int g = lane >> 2, q = lane & 3;
  const int nkb = ti.nkb;
  const int wrow = cw * 16 * SW_MT + g;  // first of this lane's weight rows in a 64-row block
  // split-K tiles write their fp32 partial, the others `out`
  float* const part = op.nsplit > 1 ? op.split_out + ti.split * op.split_stride : nullptr;
  for (int cb = 0; cb < ti.ncb; ++cb) {
    float acc[SW_MT][NT][4];
#pragma unroll
    for (int i = 0; i < SW_MT; ++i)
#pragma unroll
      for (int j = 0; j < NT; ++j)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[i][j][c] = 0.f;
    for (int kb = 0; kb < nkb; ++kb, ++it) {
      const uint32_t s = it % SW_STAGES;
      if (!mbar_wait(full0 + 8 * s, (it / SW_STAGES) & 1, abort_flag, P.wait_cycles)) return false;
      const uint32_t wbox = smem_base + s * SW_STAGE_BYTES;
      const uint32_t xbox = wbox + SW_BOX_BYTES;
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        // Lane q of half c reads the 16-byte K unit u = 2q + c of its rows (the
        // same unit of the weight and of the token row, so the MMA sum is a
        // permutation of K), stored at u ^ (r & 7) by the 128-byte swizzle with
        // r & 7 == g.  Rows g and g + 1 then read units of opposite parity:
        // the 8 lanes of a shared-memory phase touch 8 distinct bank groups.
        const uint32_t unit = (((q << 1) | c) ^ g) * 16;
        // token rows 8j+g beyond M hold stale data; they only reach masked columns
        uint4 xv[NT];
#pragma unroll
        for (int j = 0; j < NT; ++j)
          xv[j] = lds_v4(xbox + (8 * j + g) * 128 + unit);
#pragma unroll
        for (int i = 0; i < SW_MT; ++i) {
          const uint4 w0 = lds_v4(wbox + (wrow + 16 * i) * 128 + unit);
          const uint4 w1 = lds_v4(wbox + (wrow + 16 * i + 8) * 128 + unit);
#pragma unroll
          for (int j = 0; j < NT; ++j) {
            mma_bf16(acc[i][j], w0.x, w1.x, w0.y, w1.y, xv[j].x, xv[j].y);
            mma_bf16(acc[i][j], w0.z, w1.z, w0.w, w1.w, xv[j].z, xv[j].w);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive_relaxed(empty0 + 8 * s);
    }
    // epilogue: D[weight row][token] -> out[token row][grp*Ng + weight row]
    if (!part && !op.out_f32) {
      // bf16: stage the warp's 32 columns x 8 NT tokens, then 16-byte row pieces
      __nv_bfloat16* st = ost + cw * (SW_TOK * SW_OST);
#pragma unroll
      for (int i = 0; i < SW_MT; ++i)
#pragma unroll
        for (int j = 0; j < NT; ++j)
#pragma unroll
          for (int c = 0; c < 4; ++c)
            st[(8 * j + 2 * q + (c & 1)) * SW_OST + 16 * i + g + (c >= 2 ? 8 : 0)] =
                __float2bfloat16_rn(acc[i][j][c]);
      __syncwarp();
      const int ch = lane & 3;
      const int wr0 = ti.row0 + cb * SW_ROWS + cw * 16 * SW_MT + 8 * ch;
#pragma unroll
      for (int pss = 0; pss < NT; ++pss) {
        const int m = 8 * pss + (lane >> 2);
        if (m < ti.M && wr0 < ti.Ng) {
          const uint4 v = *reinterpret_cast<const uint4*>(st + m * SW_OST + 8 * ch);
          *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(op.out) +
                                    (size_t)(ti.tok0 + m) * op.ldo + (size_t)ti.grp * ti.Ng +
                                    wr0) = v;
        }
      }
      if (op.sig) {
        // this warp's half of the column tile is stored: count it
        __threadfence();
        __syncwarp();
        if (lane == 0) atomicAdd(op.sig + ti.node * STREAM_DEP_TB + ti.tb, 1);
      }
      __syncwarp();
      continue;
    }
#pragma unroll
    for (int i = 0; i < SW_MT; ++i) {
#pragma unroll
      for (int j = 0; j < NT; ++j) {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int wr = ti.row0 + cb * SW_ROWS + wrow + 16 * i + (c >= 2 ? 8 : 0);
          const int m = 8 * j + 2 * q + (c & 1);
          if (wr < ti.Ng && m < ti.M) {
            const size_t o = (size_t)(ti.tok0 + m) * op.ldo + (size_t)ti.grp * ti.Ng + wr;
            if (part) part[o] = acc[i][j][c];
            else if (op.out_f32) static_cast<float*>(op.out)[o] = acc[i][j][c];
            else static_cast<__nv_bfloat16*>(op.out)[o] = __float2bfloat16_rn(acc[i][j][c]);
          }
        }
      }
    }
  }
  return true;
}

__global__ void __launch_bounds__(SW_THREADS, SW_CTAS_PER_SM)
k_stream_gemm(const __grid_constant__ StreamLaunch P) {
  if (!P.early_weights) pdl_wait();
  else asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  __nv_bfloat16* ost = reinterpret_cast<__nv_bfloat16*>(smem + SW_STAGES * SW_STAGE_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + SW_STAGES * SW_STAGE_BYTES + SW_OST_BYTES);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 2 * SW_STAGES);
  const __nv_bfloat16** xsrc = reinterpret_cast<const __nv_bfloat16**>(bars + 2 * SW_STAGES + 2);
  TileInfo* slot = reinterpret_cast<TileInfo*>(xsrc + 2 * SW_TOK);  // [SW_STAGES]
  const uint32_t smem_base = smem_u32(smem);
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * SW_STAGES;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < SW_STAGES; ++s) {
      // the producer lane's arrival plus one cp.async arrival per producer lane
      mbar_init(full0 + 8 * s, 1 + 32);
      mbar_init(empty0 + 8 * s, SW_CONSUMERS);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  uint32_t it = 0;
  if (warp == 0) {
    // ---- producer warp.  Tiles are claimed from the launch's counter while
    // the previous tile's last stages stream; the decoded tile rides in the
    // shared slot of its first stage.  Lane 0 waits and issues the weight box,
    // all lanes copy token rows.
    const uint64_t wpol = evict_first_policy();
    const int tiles0 = op_tiles(P.op[0]);
    const int tiles1 = tiles0 + (P.n_ops > 1 ? op_tiles(P.op[1]) : 0);
    const int total = tiles1 + (P.n_ops > 2 ? op_tiles(P.op[2]) : 0);
    // token-row sources of a tile, double-buffered so the next tile's are
    // prepared while the current one streams
    auto prepare = [&](const TileInfo& t, int buf) {
      const StreamOp& op = P.op[t.op];
      if (!op.gather) return;  // contiguous rows come by TMA
      const long acol = (long)t.grp * t.K;
#pragma unroll
      for (int h = 0; h < (SW_TOK + 31) / 32; ++h) {
        const int m = lane + 32 * h;
        if (t.active && m < t.M) {
          const int row = t.tok0 + m;
          const long r = op.gather ? op.gather[row] : row;
          xsrc[buf * SW_TOK + m] = op.X + r * op.ldx + acol;
        }
      }
    };
    // CTA b starts on tile b; later tiles come from the counter, offset by the
    // grid (a first claim by every CTA at once would be a contended round
    // trip).  A factor-product tile among the first ones waits only for tiles
    // of lower index, i.e. of CTAs dispatched no later than its own.
    int cur = blockIdx.x;
    TileInfo ti;
    if (cur < total) {
      decode_tile(P, cur, tiles0, tiles1, ti);
      prepare(ti, 0);
    }
    __syncwarp();
    // Dependent launch whose weights do not depend on the preceding kernel: the
    // first tile's first weight boxes go out before the wait for it (stage
    // it < npre already holds its box and expected bytes); token rows after.
    uint32_t npre = 0;
    if (P.early_weights) {
      if (cur < total && ti.active && ti.ncb >= 1) {
        const StreamOp& op = P.op[ti.op];
        npre = (uint32_t)min(ti.nkb, SW_STAGES);
        if (lane == 0) {
          const int rt0 = (ti.grp * ti.Ng + ti.row0) / SW_ROWS;
          for (uint32_t kb = 0; kb < npre; ++kb) {  // fresh stages: nothing to wait for
            const uint32_t wbox = smem_base + kb * SW_STAGE_BYTES;
            if (kb == 0) slot[0] = ti;
            mbar_expect_tx(full0 + 8 * kb, SW_BOX_BYTES + (op.gather ? 0 : SW_XBYTES));
            tma_load_tile(wbox, op.tmaps + ti.node, ti.kb0 + kb, rt0, full0 + 8 * kb, wpol);
          }
        }
      }
      __syncwarp();
      asm volatile("griddepcontrol.wait;" ::: "memory");
    }
    int buf = 0;
    bool ok = true;
    while (cur < total && ok) {
      int nxt = 0;
      TileInfo tn;
      bool claimed = false, prepared = false;
      if (ti.active) {
        const StreamOp& op = P.op[ti.op];
        const CUtensorMap* map = op.tmaps + ti.node;
        const int rt0 = (ti.grp * ti.Ng + ti.row0) / SW_ROWS;
        const __nv_bfloat16* const* xs = xsrc + buf * SW_TOK;
        const int nkb = ti.nkb, kb0 = ti.kb0;
        // The next tile is claimed kClaimLead stages before this tile's last
        // one and decoded a stage later: a tile claimed earlier would wait
        // behind a long one (whole-K factor tiles stream 32 stages) instead of
        // going to a CTA that is about to be free.
        const int nst = ti.ncb * nkb;
        const int jd = max(nst - 1 - kClaimLead, min(1, nst - 1)), jc = max(jd - 1, 0);
        if (op.dep) {
          // the token rows of this tile are written by another op of this
          // launch: wait for every column tile of them (both consumer warps'
          // halves), then order the async-proxy row loads after the acquire
          int good = 1;
          if (lane == 0) {
            // (an injected unmet wait asks for one arrival more than the
            // producer tiles ever make, so that the bounded wait runs out)
            const int need = SW_CONSUMERS * ((op.dep_nrank * ti.K + SW_ROWS - 1) / SW_ROWS) +
                             (P.unmet_wait == LX_WAIT_STREAM_DEP ? 1 : 0);
            good = dep_wait(op.dep + ti.node * STREAM_DEP_TB + ti.tb, need, abort_flag,
                            P.wait_cycles) ? 1 : 0;
            asm volatile("fence.proxy.async.global;" ::: "memory");
          }
          good = __shfl_sync(0xffffffffu, good, 0);
          if (!good) ok = false;
        }
        for (int cb = 0; cb < ti.ncb && ok; ++cb) {
          for (int kb = 0; kb < nkb; ++kb, ++it) {
            const int j = cb * nkb + kb;
            if (j == jc) {
              if (lane == 0) nxt = (int)gridDim.x + atomicAdd(P.ctr, 1);  // in flight until j == jd
              claimed = true;
            }
            const uint32_t s = it % SW_STAGES;
            int good = 1;
            const bool pre = it < npre;  // weight box issued before the dependency wait
            if (lane == 0 && !pre) {
              good = mbar_wait(empty0 + 8 * s, ((it / SW_STAGES) & 1) ^ 1, abort_flag,
                               P.wait_cycles) ? 1 : 0;
              if (good) {
                if (cb == 0 && kb == 0) slot[s] = ti;
                mbar_expect_tx(full0 + 8 * s, SW_BOX_BYTES + (op.gather ? 0 : SW_XBYTES));
              }
            }
            good = __shfl_sync(0xffffffffu, good, 0);
            if (!good) {
              ok = false;
              break;
            }
            const uint32_t wbox = smem_base + s * SW_STAGE_BYTES;
            if (lane == 0) {
              if (!pre) tma_load_tile(wbox, map, kb0 + kb, rt0 + cb, full0 + 8 * s, wpol);
              // contiguous token rows: one box of SW_TOK rows (rows past the
              // bucket belong to the next node and are never stored)
              if (!op.gather)
                tma_load_rows(wbox + SW_BOX_BYTES, op.xmap,
                              (int)(ti.grp * ti.K) + (kb0 + kb) * SW_BOX, ti.tok0, full0 + 8 * s);
            }
            if (op.gather) {
              // gathered token rows: M rows x 128 bytes as 16-byte pieces over
              // the 32 lanes, piece u of row m to 16-byte unit u ^ (m & 7)
              for (int piece = lane; piece < ti.M * 8; piece += 32) {
                const int m = piece >> 3, u = piece & 7;
                cp_async16(wbox + SW_BOX_BYTES + m * 128 + ((u ^ (m & 7)) << 4),
                           xs[m] + (kb0 + kb) * SW_BOX + u * 8);
              }
            }
            cp_async_arrive(full0 + 8 * s);
            if (j == jd) {
              // the next tile: decode and prepare its rows while these stages stream
              nxt = __shfl_sync(0xffffffffu, nxt, 0);
              if (nxt < total) {
                decode_tile(P, nxt, tiles0, tiles1, tn);
                prepare(tn, buf ^ 1);
                if (lane == 0 && tn.active)
                  asm volatile("prefetch.tensormap [%0];" ::"l"(
                      reinterpret_cast<uint64_t>(P.op[tn.op].tmaps + tn.node)) : "memory");
              }
              prepared = true;
            }
          }
        }
      }
      if (!claimed && lane == 0) nxt = (int)gridDim.x + atomicAdd(P.ctr, 1);
      if (!prepared) {
        nxt = __shfl_sync(0xffffffffu, nxt, 0);
        if (nxt < total) {
          decode_tile(P, nxt, tiles0, tiles1, tn);
          prepare(tn, buf ^ 1);
        }
      }
      __syncwarp();
      cur = nxt;
      ti = tn;
      buf ^= 1;
    }
    if (ok) {
      // sentinel stage: tells the consumers that no tile follows
      const uint32_t s = it % SW_STAGES;
      int good = 1;
      if (lane == 0) {
        good = mbar_wait(empty0 + 8 * s, ((it / SW_STAGES) & 1) ^ 1, abort_flag, P.wait_cycles)
                   ? 1 : 0;
        if (good) {
          slot[s].op = -1;
          mbar_arrive(full0 + 8 * s);
        }
      }
      good = __shfl_sync(0xffffffffu, good, 0);
      if (good) {
        cp_async_arrive(full0 + 8 * s);
        ++it;
      } else {
        ok = false;
      }
    }
    if (!ok && lane == 0) {
      atomicExch(P.err, LX_ERR_TIMEOUT);
      *abort_flag = 1;
      // drain: every issued stage's copies must land before the CTA exits (the
      // copies were issued, so these waits end; they keep the full bound)
      const uint32_t first = it > SW_STAGES ? it - SW_STAGES : 0;
      volatile int never = 0;
      for (uint32_t j = first; j < it; ++j)
        mbar_wait(full0 + 8 * (j % SW_STAGES), (j / SW_STAGES) & 1, &never, SW_TIMEOUT_CYCLES);
    }
    return;
  }
  // ---- consumers: the first stage of every tile carries its description
  while (true) {
    const uint32_t s = it % SW_STAGES;
    if (!mbar_wait(full0 + 8 * s, (it / SW_STAGES) & 1, abort_flag, P.wait_cycles)) {
      if (lane == 0) {
        atomicExch(P.err, LX_ERR_TIMEOUT);
        *abort_flag = 1;
      }
      return;
    }
    const TileInfo ti = slot[s];
    if (ti.op < 0) return;  // sentinel
    const int nt = (ti.M + 7) / 8;
    bool ok;
    if (nt <= 1) ok = consume_tile<1>(P, ti, smem_base, full0, empty0, it, abort_flag, ost);
    else if (nt <= 2) ok = consume_tile<2>(P, ti, smem_base, full0, empty0, it, abort_flag, ost);
    else if (SW_TOK <= 32 || nt <= 4)
      ok = consume_tile<SW_TOK <= 32 ? SW_TOK / 8 : 4>(P, ti, smem_base, full0, empty0, it, abort_flag, ost);
    else ok = consume_tile<SW_TOK / 8>(P, ti, smem_base, full0, empty0, it, abort_flag, ost);
    if (!ok) {
      if (lane == 0) {
        atomicExch(P.err, LX_ERR_TIMEOUT);
        *abort_flag = 1;
      }
      return;
    }
  }
}

}  // namespace

int stream_smem_bytes() {
  return SW_STAGES * SW_STAGE_BYTES + SW_OST_BYTES + 2 * SW_STAGES * 8 + 16 + 2 * SW_TOK * 8 +
         SW_STAGES * (int)sizeof(TileInfo) + 1024;
}

lx_status launch_stream(lx_layer* L, const StreamLaunch& P, cudaStream_t s, const char* name) {
  const int smem = stream_smem_bytes();
  static bool done[64] = {};
  LX_CUDA(smem_cap_once((const void*)k_stream_gemm, smem, L->device, done));
  ProfScope ps(L, s, name);
  launch_k(L, k_stream_gemm, L->num_sms * SW_CTAS_PER_SM, SW_THREADS, smem, s, P);
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

constexpr int kStreamUBlocks = 1;

static StreamOp make_op(lx_layer* L, int op, const __nv_bfloat16* X, long ldx,
                        const int* gather, const CUtensorMap* xmap, void* out, long ldo,
                        bool out_f32) {
  StreamOp o;
  o.shape = op_shape(L, op);
  o.tmaps = L->d_tmaps + (size_t)op * L->N;
  o.items = L->ws.act + (o.shape.on_anchors ? 0 : (size_t)L->n_anchor * STREAM_DEP_TB);
  o.n_active = L->ws.act_n + (o.shape.on_anchors ? 0 : 1);
  o.n_items = o.shape.on_anchors ? L->n_anchor : L->n_corr;
  o.tile_off = nullptr;
  o.node_off = L->ws.key_off;
  o.gather = gather;
  o.X = X;
  o.xmap = xmap;
  o.ldx = ldx;
  o.out = out;
  o.ldo = ldo;
  o.out_f32 = out_f32 ? 1 : 0;
  o.rank = L->d_rank;
  int ng_max = 0;
  for (int n : (o.shape.on_anchors ? L->anchors : L->corrs))
    ng_max = std::max(ng_max, o.shape.n_const + o.shape.n_rank * L->rank[n]);
  // short-K factor products (U) take several column blocks per tile, so that
  // a tile streams more than two stages
  o.ncb = (op == OP_UP_U || op == OP_DN_U) ? kStreamUBlocks : 1;
  o.ncol_max = ((ng_max + SW_ROWS - 1) / SW_ROWS + o.ncb - 1) / o.ncb;
  o.nsplit = 1;
  o.kbs = 1 << 20;
  o.split_out = nullptr;
  o.split_stride = 0;
  o.sig = nullptr;
  o.dep = nullptr;
  o.dep_nrank = 0;
  return o;
}

// Split the anchor op's K into at most LX_STREAM_MAX_SPLIT ranges of about
// `blocks` 64-wide blocks, so that the last tiles of a launch are short.
// Partials go to `part`.  Measured on GB300 at a decode batch of 64: the
// gate/up side (K = H) gains with 8-block (64 KB) ranges; the down side
// (K = I) is faster unsplit up to 16 blocks, where the partials' extra traffic
// outweighs the shorter tail.
constexpr int kStreamSplitBlocksUp = 8;
constexpr int kStreamSplitBlocksDown = 16;
static void split_op(lx_layer* L, StreamOp& o, float* part, long stride, int blocks) {
  if (!part) return;
  const int K = o.shape.k_const;  // anchors: K does not depend on a rank
  const int nkb = (K + SW_BOX - 1) / SW_BOX;
  int ns = std::min(LX_STREAM_MAX_SPLIT, (nkb + blocks - 1) / blocks);
  if (ns <= 1) return;
  o.kbs = (nkb + ns - 1) / ns;
  o.nsplit = (nkb + o.kbs - 1) / o.kbs;
  o.split_out = part;
  o.split_stride = stride;
  (void)L;
}

// Whether the anchors' split-K pays at this batch: measured on GB300 (decode
// forwards of the Qwen3-30B-A3B-shaped and the high-expert-count layers, T from
// 1 to 256), it shortens the launches only while the batch's tokens times the
// anchors' gate/up column tiles lie between about 1.5 and 3 times the
// streaming grid -- the whole-K anchor tiles then make a last partial wave --
// and costs time elsewhere (fewer, longer tiles already balance, or every tile
// fits the first wave), through the partials' extra traffic.
static bool split_pays(const lx_layer* L, int T) {
  const long grid = (long)L->num_sms * SW_CTAS_PER_SM;
  const long work = (long)T * ((2L * L->I + SW_ROWS - 1) / SW_ROWS);
  return 2 * work >= 3 * grid && 10 * work <= 31 * grid;
}

// One streaming launch (launch group g) over up to three ops' tile grids, in
// claim order.
static lx_status run_stream(lx_layer* L, int g, std::initializer_list<const StreamOp*> ops,
                            cudaStream_t s, const char* name) {
  StreamLaunch P;
  P.n_ops = 0;
  for (const StreamOp* o : ops) {
    if (!o || o->n_items == 0) continue;
    P.op[P.n_ops++] = *o;
  }
  if (P.n_ops == 0) return LX_OK;
  P.ctr = L->ws.sctr + g;
  P.err = L->ws.err;
  P.wait_cycles = wait_limit(L);
  P.unmet_wait = L->unmet_wait;
  // the z-side launch follows the SwiGLU kernel, whose output only its token
  // rows read
  P.early_weights = g == 2 ? 1 : 0;
  return launch_stream(L, P, s, name);
}

// The decode forward: every touched weight byte is streamed once.  Two
// streaming launches: {x V of every correction, the shared anchor gate/up,
// then P U of every correction (each waits for its P rows)} and the same on
// the z side; the factor products fill the tail of the anchor products.
lx_status launch_fast_experts(lx_layer* L, const void* x, int T, int k, void* y, cudaStream_t s) {
  Workspace& w = L->ws;
  const long H = L->H, I = L->I, rmax = L->max_rank;
  const __nv_bfloat16* xb = static_cast<const __nv_bfloat16*>(x);
  const bool split = w.hsplit && w.ysplit && warp_kernels_fit(L, k) &&
                     (long)T * std::min<long>(L->N, (long)k * L->max_depth) <= w.split_rows &&
                     split_pays(L, T);
  int* dep_up = w.sctr + N_TILE_COUNTERS;
  int* dep_dn = dep_up + (size_t)L->N * STREAM_DEP_TB;
  // x-side: x V of every correction (whole-K tiles, claimed first), the shared
  // anchor gate/up in split-K slices, then the corrections' U products
  StreamOp up_v = make_op(L, OP_UP_V, xb, H, w.node_tok, nullptr, w.Pb, 2 * rmax, false);
  up_v.sig = dep_up;
  StreamOp up_a = make_op(L, OP_UP_ANCHOR, xb, H, w.node_tok, nullptr, w.hb, 2 * I, false);
  if (split) split_op(L, up_a, w.hsplit, w.split_rows * 2 * I, kStreamSplitBlocksUp);
  StreamOp up_u = make_op(L, OP_UP_U, w.Pb, 2 * rmax, nullptr, w.smaps + 0, w.hb, 2 * I, false);
  up_u.dep = dep_up;
  up_u.dep_nrank = 2;  // P = [x Vg | x Vu]: 2r columns
  LX_TRY(run_stream(L, 0, {&up_v, &up_a, &up_u}, s, "stream_up"));
  SplitParts hs, ys;
  if (up_a.nsplit > 1) {
    hs.part = up_a.split_out;
    hs.splits = up_a.nsplit;
    hs.stride = up_a.split_stride;
  }
  LX_TRY(launch_swiglu(L, T, k, true, s, hs));
  // z-side: z Vd of every correction first, the shared anchor down
  // projection, then the corrections' Ud products
  StreamOp dn_v = make_op(L, OP_DN_V, w.zb, I, nullptr, w.smaps + 1, w.Qb, rmax, false);
  dn_v.sig = dep_dn;
  StreamOp dn_a = make_op(L, OP_DN_ANCHOR, w.zb, I, nullptr, w.smaps + 1, w.yb, H, false);
  if (split) split_op(L, dn_a, w.ysplit, w.split_rows * H, kStreamSplitBlocksDown);
  StreamOp dn_u = make_op(L, OP_DN_U, w.Qb, rmax, nullptr, w.smaps + 2, w.yb, H, false);
  dn_u.dep = dep_dn;
  dn_u.dep_nrank = 1;  // Q = z Vd: r columns
  LX_TRY(run_stream(L, 2, {&dn_v, &dn_a, &dn_u}, s, "stream_dn"));
  if (dn_a.nsplit > 1) {
    ys.part = dn_a.split_out;
    ys.splits = dn_a.nsplit;
    ys.stride = dn_a.split_stride;
  }
  LX_TRY(launch_combine(L, T, k, y, true, s, ys));
  return LX_OK;
}

int stream_tile_rows() { return SW_ROWS; }
int stream_tile_tokens() { return SW_TOK; }
int stream_box() { return SW_BOX; }

}  // namespace lx
