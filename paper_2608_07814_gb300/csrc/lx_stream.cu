// Weight-streaming grouped GEMM for small token counts (decode).
//
// out[rows of node n][cols] = X[rows][K] . W_n[cols][K]^T for every active node,
// where X holds at most 64 rows per tile.  Decode is bound by reading each
// touched weight byte once from HBM (Sec. 5.2: the projections run at about one
// FLOP per byte), so the kernel is organised around the weight stream:
//
//   * one tile = 64 weight rows (output columns) x 64 tokens of one node,
//     over the full K;
//   * a producer warp streams the tile's weights with 2-D TMA loads
//     (cp.async.bulk.tensor, 64x64 bf16 boxes, 128-byte swizzle) into a
//     4-stage shared-memory ring guarded by mbarriers;
//   * two consumer warps (32 weight rows each) multiply with mma.sync
//     m16n8k16 (weights as the 16-row operand, tokens as the 8-column
//     operand).  Inside each 32-wide K chunk the contraction index is
//     permuted so that every lane reads 8 consecutive K values of a weight
//     row (one 16-byte shared load) and of a token row (one 16-byte global
//     load); the same permutation on both operands leaves the sum unchanged;
//   * persistent CTAs walk a device-built tile list; every mbarrier wait is
//     bounded, and a wait that gives up records LX_ERR_TIMEOUT in a device
//     word and drains the CTA's copies in flight before returning.
#include <cuda.h>


#include "lx_internal.cuh"

namespace lx {

namespace {

constexpr int SW_ROWS = 64;         // weight rows per tile
constexpr int SW_TOK = 64;          // tokens per tile
constexpr int SW_BOX = 64;          // K per stage = one TMA box of 64 K x 64 rows
constexpr int SW_BOX_BYTES = SW_BOX * SW_ROWS * 2;
constexpr int SW_XROW = SW_BOX * 2 + 16;           // padded token row in shared memory
constexpr int SW_STAGE_BYTES = SW_BOX_BYTES + SW_TOK * SW_XROW;  // 17 KiB, 1024-aligned
constexpr int SW_STAGES = 6;
constexpr int SW_CONSUMERS = 2;
constexpr int SW_THREADS = 32 * (1 + SW_CONSUMERS);
constexpr unsigned long long SW_TIMEOUT_CYCLES = 4000000000ull;  // ~2 s
static_assert(SW_STAGE_BYTES % 1024 == 0, "stages must keep the 128B-swizzle alignment");

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: false if the phase did not complete in time or the CTA aborted.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag) {
  if (mbar_try_wait(bar, parity)) return true;
  const unsigned long long t0 = clock64();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort_flag) return false;
    if (clock64() - t0 > SW_TIMEOUT_CYCLES) return false;
  }
}

// one 64x64 tile (box) of a tiled weight matrix: K tile kt of row tile rt
__device__ __forceinline__ void tma_load_tile(uint32_t dst, const CUtensorMap* map, int kt, int rt,
                                              uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(0), "r"(0), "r"(kt), "r"(rt), "r"(bar)
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
};

__device__ __forceinline__ void fetch_tile(const StreamLaunch& P, int tile, int total, int4& a,
                                           int4& b) {
  if (tile < total) {
    a = P.tiles[2 * tile];
    b = P.tiles[2 * tile + 1];
  }
}

__device__ __forceinline__ void unpack_tile(const StreamLaunch& P, const int4& a, const int4& b,
                                            TileInfo& ti) {
  ti.op = (P.n_ops > 1 && a.x == P.op_id[1]) ? 1 : 0;
  ti.node = a.y;
  ti.row0 = a.z;
  ti.tok0 = a.w;
  ti.M = b.x;
  ti.K = b.y;
  ti.Ng = b.z;
  ti.grp = b.w & 15;
  ti.ncb = b.w >> 4;
}

template <int NT>
__device__ __forceinline__ bool consume_tile(const StreamLaunch& P, const TileInfo& ti,
                                             uint32_t smem_base, uint32_t full0, uint32_t empty0,
                                             uint32_t& it, volatile int* abort_flag) {
  const StreamOp& op = P.op[ti.op];
  const int lane = threadIdx.x & 31, cw = (threadIdx.x >> 5) - 1;
  const int g = lane >> 2, q = lane & 3;
  const int nkb = (ti.K + SW_BOX - 1) / SW_BOX;
  const int wrow = cw * 32 + g;  // first of this lane's weight rows inside a 64-row block
  for (int cb = 0; cb < ti.ncb; ++cb) {
    float acc[2][NT][4];
#pragma unroll
    for (int i = 0; i < 2; ++i)
#pragma unroll
      for (int j = 0; j < NT; ++j)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[i][j][c] = 0.f;
    for (int kb = 0; kb < nkb; ++kb, ++it) {
      const uint32_t s = it % SW_STAGES;
      if (!mbar_wait(full0 + 8 * s, (it / SW_STAGES) & 1, abort_flag)) return false;
      const uint32_t wbox = smem_base + s * SW_STAGE_BYTES;
      const uint32_t xbox = wbox + SW_BOX_BYTES;
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        // token rows 8j+g beyond M hold stale data; they only reach masked columns
        uint4 xv[NT];
#pragma unroll
        for (int j = 0; j < NT; ++j)
          xv[j] = lds_v4(xbox + (8 * j + g) * SW_XROW + c * 64 + 16 * q);
        const uint32_t unit = ((c * 4 + q) ^ g) * 16;  // 128-byte swizzle (row & 7 == g)
#pragma unroll
        for (int i = 0; i < 2; ++i) {
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
      if (lane == 0) mbar_arrive(empty0 + 8 * s);
    }
    // epilogue: D[weight row][token] -> out[token row][grp*Ng + weight row]
#pragma unroll
    for (int i = 0; i < 2; ++i) {
#pragma unroll
      for (int j = 0; j < NT; ++j) {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const int wr = ti.row0 + cb * SW_ROWS + wrow + 16 * i + (c >= 2 ? 8 : 0);
          const int m = 8 * j + 2 * q + (c & 1);
          if (wr < ti.Ng && m < ti.M) {
            const size_t o = (size_t)(ti.tok0 + m) * op.ldo + (size_t)ti.grp * ti.Ng + wr;
            if (op.out_f32) static_cast<float*>(op.out)[o] = acc[i][j][c];
            else static_cast<__nv_bfloat16*>(op.out)[o] = __float2bfloat16_rn(acc[i][j][c]);
          }
        }
      }
    }
  }
  return true;
}

__global__ void __launch_bounds__(SW_THREADS)
k_stream_gemm(const __grid_constant__ StreamLaunch P) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + SW_STAGES * SW_STAGE_BYTES);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 2 * SW_STAGES);
  const __nv_bfloat16** xsrc = reinterpret_cast<const __nv_bfloat16**>(bars + 2 * SW_STAGES + 2);
  const uint32_t smem_base = smem_u32(smem);
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * SW_STAGES;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < SW_STAGES; ++s) {
      // the producer lane's expect_tx arrival plus one cp.async arrival per producer lane
      mbar_init(full0 + 8 * s, 1 + 32);
      mbar_init(empty0 + 8 * s, SW_CONSUMERS);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  const int total = *P.n_tiles;
  uint32_t it = 0;
  if (warp == 0) {
    // ---- producer warp: lane 0 waits and issues the weight box, every lane
    // copies up to two token rows of the stage
    bool ok = true;
    int4 na = make_int4(0, 0, 0, 0), nb = na;
    fetch_tile(P, blockIdx.x, total, na, nb);
    for (int tile = blockIdx.x; tile < total && ok; tile += gridDim.x) {
      TileInfo ti;
      unpack_tile(P, na, nb, ti);
      fetch_tile(P, tile + gridDim.x, total, na, nb);  // next descriptor in flight
      const StreamOp& op = P.op[ti.op];
      const CUtensorMap* map = op.tmaps + ti.node;
      const int rt0 = (ti.grp * ti.Ng + ti.row0) / SW_ROWS;
      const long acol = (long)ti.grp * ti.K;
      __syncwarp();  // earlier readers of xsrc are done
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int m = lane + 32 * h;
        if (m < ti.M) {
          const int row = ti.tok0 + m;
          const long r = op.gather ? op.gather[row] : row;
          xsrc[m] = op.X + r * op.ldx + acol;
        }
      }
      __syncwarp();
      const int nkb = (ti.K + SW_BOX - 1) / SW_BOX;
      for (int cb = 0; cb < ti.ncb && ok; ++cb) {
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const uint32_t s = it % SW_STAGES;
          int good = 1;
          if (lane == 0) {
            good = mbar_wait(empty0 + 8 * s, ((it / SW_STAGES) & 1) ^ 1, abort_flag) ? 1 : 0;
            if (good) mbar_expect_tx(full0 + 8 * s, SW_BOX_BYTES);
          }
          good = __shfl_sync(0xffffffffu, good, 0);
          if (!good) {
            ok = false;
            break;
          }
          const uint32_t wbox = smem_base + s * SW_STAGE_BYTES;
          if (lane == 0) tma_load_tile(wbox, map, kb, rt0 + cb, full0 + 8 * s);
          // token rows: M rows x 128 bytes as 16-byte pieces over the 32 lanes
          for (int piece = lane; piece < ti.M * 8; piece += 32) {
            const int m = piece >> 3, u = piece & 7;
            cp_async16(wbox + SW_BOX_BYTES + m * SW_XROW + u * 16, xsrc[m] + kb * SW_BOX + u * 8);
          }
          cp_async_arrive(full0 + 8 * s);
        }
      }
    }
    if (!ok && lane == 0) {
      atomicExch(P.err, LX_ERR_TIMEOUT);
      *abort_flag = 1;
      // drain: every issued stage's copies must land before the CTA exits
      const uint32_t first = it > SW_STAGES ? it - SW_STAGES : 0;
      volatile int never = 0;
      for (uint32_t j = first; j < it; ++j)
        mbar_wait(full0 + 8 * (j % SW_STAGES), (j / SW_STAGES) & 1, &never);
    }
    return;
  }
  // ---- consumers
  int4 na = make_int4(0, 0, 0, 0), nb = na;
  fetch_tile(P, blockIdx.x, total, na, nb);
  for (int tile = blockIdx.x; tile < total; tile += gridDim.x) {
    TileInfo ti;
    unpack_tile(P, na, nb, ti);
    fetch_tile(P, tile + gridDim.x, total, na, nb);
    const int nt = (ti.M + 7) / 8;
    bool ok;
    if (nt <= 1) ok = consume_tile<1>(P, ti, smem_base, full0, empty0, it, abort_flag);
    else if (nt <= 2) ok = consume_tile<2>(P, ti, smem_base, full0, empty0, it, abort_flag);
    else if (nt <= 4) ok = consume_tile<4>(P, ti, smem_base, full0, empty0, it, abort_flag);
    else ok = consume_tile<8>(P, ti, smem_base, full0, empty0, it, abort_flag);
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
  return SW_STAGES * SW_STAGE_BYTES + 2 * SW_STAGES * 8 + 16 + SW_TOK * 8 + 1024;
}

lx_status launch_stream(lx_layer* L, const StreamLaunch& P, cudaStream_t s, const char* name) {
  const int smem = stream_smem_bytes();
  static bool done[64] = {};
  LX_CUDA(smem_cap_once((const void*)k_stream_gemm, smem, L->device, done));
  ProfScope ps(L, s, name);
  k_stream_gemm<<<L->num_sms * 2, SW_THREADS, smem, s>>>(P);
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

static StreamOp make_op(lx_layer* L, int op, const __nv_bfloat16* X, long ldx, const int* gather,
                        void* out, long ldo, bool out_f32) {
  StreamOp o;
  o.shape = op_shape(L, op);
  o.tmaps = L->d_tmaps + (size_t)op * L->N;
  o.items = o.shape.on_anchors ? L->d_anchors : L->d_corrs;
  o.n_items = o.shape.on_anchors ? L->n_anchor : L->n_corr;
  o.tile_off = nullptr;
  o.node_off = L->ws.key_off;
  o.gather = gather;
  o.X = X;
  o.ldx = ldx;
  o.out = out;
  o.ldo = ldo;
  o.out_f32 = out_f32 ? 1 : 0;
  o.rank = L->d_rank;
  return o;
}

// One launch of launch group g (its tile list was built during bucketing).
static lx_status run_stream(lx_layer* L, int g, const StreamOp& o0, const StreamOp* o1,
                            cudaStream_t s, const char* name) {
  StreamLaunch P;
  P.op[0] = o0;
  P.op_id[0] = stream_group_op(g, 0);
  P.n_ops = 1;
  P.op_id[1] = -1;
  if (o1) {
    P.op[1] = *o1;
    P.op_id[1] = stream_group_op(g, 1);
    P.n_ops = 2;
  }
  if (o0.n_items == 0 && (!o1 || o1->n_items == 0)) return LX_OK;
  P.tiles = L->ws.stiles + (size_t)g * L->ws.stile_cap * 2;
  P.n_tiles = L->ws.stile_cnt + g;
  P.err = L->ws.err;
  return launch_stream(L, P, s, name);
}

// The decode forward: every touched weight byte is streamed once.
lx_status launch_fast_experts(lx_layer* L, const void* x, int T, int k, void* y, cudaStream_t s) {
  Workspace& w = L->ws;
  const long H = L->H, I = L->I, rmax = L->max_rank;
  const __nv_bfloat16* xb = static_cast<const __nv_bfloat16*>(x);
  // x-side: shared anchor gate/up, and x V of every correction
  const StreamOp up_v = make_op(L, OP_UP_V, xb, H, w.node_tok, w.Pb, 2 * rmax, false);
  LX_TRY(run_stream(L, 0, make_op(L, OP_UP_ANCHOR, xb, H, w.node_tok, w.h, 2 * I, true), &up_v,
                    s, "stream_up_anchor_V"));
  LX_TRY(run_stream(L, 1, make_op(L, OP_UP_U, w.Pb, 2 * rmax, nullptr, w.h, 2 * I, true),
                    nullptr, s, "stream_up_U"));
  LX_TRY(launch_swiglu(L, T, k, w.zb, true, s));
  // z-side: shared anchor down projection, and z Vd of every correction
  const StreamOp dn_v = make_op(L, OP_DN_V, w.zb, I, nullptr, w.Qb, rmax, false);
  LX_TRY(run_stream(L, 2, make_op(L, OP_DN_ANCHOR, w.zb, I, nullptr, w.ypart, H, true), &dn_v,
                    s, "stream_dn_anchor_V"));
  LX_TRY(run_stream(L, 3, make_op(L, OP_DN_U, w.Qb, rmax, nullptr, w.ypart, H, true), nullptr, s,
                    "stream_dn_U"));
  LX_TRY(launch_combine(L, T, k, y, s));
  return LX_OK;
}

int stream_tile_rows() { return SW_ROWS; }
int stream_tile_tokens() { return SW_TOK; }
int stream_box() { return SW_BOX; }

}  // namespace lx
