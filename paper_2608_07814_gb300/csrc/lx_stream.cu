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

#include <initializer_list>

#include "lx_internal.cuh"

namespace lx {

namespace {

constexpr int SW_ROWS = 64;         // weight rows per tile
constexpr int SW_TOK = 64;          // tokens per tile
constexpr int SW_BOX = 64;          // TMA box: 64 K x 64 rows
constexpr int SW_BOX_BYTES = SW_BOX * SW_ROWS * 2;
constexpr int SW_STAGE_BOXES = 2;   // K per stage = 128
constexpr int SW_STAGE_BYTES = SW_BOX_BYTES * SW_STAGE_BOXES;
constexpr int SW_STAGES = 4;
constexpr int SW_CONSUMERS = 2;
constexpr int SW_THREADS = 32 * (1 + SW_CONSUMERS);
constexpr unsigned long long SW_TIMEOUT_CYCLES = 4000000000ull;  // ~2 s

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
    __nanosleep(64);
  }
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint4 ldg_nc_v4(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ uint4 lds_v4(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr));
  return v;
}

struct TileInfo {
  int op, node, grp, row0, tok0, M, Ng, K;
};

__device__ __forceinline__ bool decode_tile(const StreamLaunch& P, int tile, TileInfo& ti) {
  int base = 0;
  for (int o = 0; o < P.n_ops; ++o) {
    const StreamOp& op = P.op[o];
    const int tot = op.tile_off[op.n_items];
    if (tile < base + tot) {
      const int local0 = tile - base;
      int lo = 0, hi = op.n_items;
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (op.tile_off[mid] <= local0) lo = mid; else hi = mid;
      }
      const int n = op.items[lo];
      const int local = local0 - op.tile_off[lo];
      const int r = op.rank[n];
      ti.op = o;
      ti.node = n;
      ti.Ng = op.shape.n_const + op.shape.n_rank * r;
      ti.K = op.shape.k_const + op.shape.k_rank * r;
      const int ncol = (ti.Ng + SW_ROWS - 1) / SW_ROWS;
      const int per_tb = ncol * op.shape.groups;
      const int tb = local / per_tb, rem = local % per_tb;
      ti.grp = rem / ncol;
      ti.row0 = (rem % ncol) * SW_ROWS;
      ti.tok0 = op.node_off[n] + tb * SW_TOK;
      ti.M = min(SW_TOK, op.node_off[n + 1] - ti.tok0);
      return true;
    }
    base += tot;
  }
  return false;
}

__device__ __forceinline__ int total_tiles(const StreamLaunch& P) {
  int t = 0;
  for (int o = 0; o < P.n_ops; ++o) t += P.op[o].tile_off[P.op[o].n_items];
  return t;
}

template <int NT>
__device__ __forceinline__ bool consume_tile(const StreamLaunch& P, const TileInfo& ti,
                                             uint32_t smem_base, uint32_t full0, uint32_t empty0,
                                             uint32_t& it, volatile int* abort_flag) {
  const StreamOp& op = P.op[ti.op];
  const int lane = threadIdx.x & 31, cw = (threadIdx.x >> 5) - 1;
  const int g = lane >> 2, q = lane & 3;
  float acc[2][NT][4];
#pragma unroll
  for (int i = 0; i < 2; ++i)
#pragma unroll
    for (int j = 0; j < NT; ++j)
#pragma unroll
      for (int c = 0; c < 4; ++c) acc[i][j][c] = 0.f;
  // token rows of this lane (token 8j + g of the tile)
  const __nv_bfloat16* xrow[NT];
  const long acol = (long)ti.grp * ti.K;
#pragma unroll
  for (int j = 0; j < NT; ++j) {
    const int m = 8 * j + g;
    if (m < ti.M) {
      const int row = ti.tok0 + m;
      const long src = op.gather ? op.gather[row] : row;
      xrow[j] = op.X + src * op.ldx + acol;
    } else {
      xrow[j] = nullptr;
    }
  }
  const int nkb = (ti.K + SW_BOX * SW_STAGE_BOXES - 1) / (SW_BOX * SW_STAGE_BOXES);
  const int wrow = cw * 32 + g;  // first of this lane's weight rows inside the tile
  for (int kb = 0; kb < nkb; ++kb, ++it) {
    const uint32_t s = it % SW_STAGES;
    if (!mbar_wait(full0 + 8 * s, (it / SW_STAGES) & 1, abort_flag)) return false;
    const int kstage = kb * SW_BOX * SW_STAGE_BOXES;
#pragma unroll
    for (int b = 0; b < SW_STAGE_BOXES; ++b) {
      if (kstage + b * SW_BOX >= ti.K) break;
      const uint32_t box = smem_base + s * SW_STAGE_BYTES + b * SW_BOX_BYTES;
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const int kk = kstage + b * SW_BOX + c * 32 + 8 * q;
        uint4 xv[NT];
#pragma unroll
        for (int j = 0; j < NT; ++j)
          xv[j] = (xrow[j] && kk < ti.K) ? ldg_nc_v4(xrow[j] + kk) : make_uint4(0, 0, 0, 0);
        const uint32_t unit = ((c * 4 + q) ^ g) * 16;  // 128-byte swizzle (row & 7 == g)
#pragma unroll
        for (int i = 0; i < 2; ++i) {
          const uint4 w0 = lds_v4(box + (wrow + 16 * i) * 128 + unit);
          const uint4 w1 = lds_v4(box + (wrow + 16 * i + 8) * 128 + unit);
#pragma unroll
          for (int j = 0; j < NT; ++j) {
            mma_bf16(acc[i][j], w0.x, w1.x, w0.y, w1.y, xv[j].x, xv[j].y);
            mma_bf16(acc[i][j], w0.z, w1.z, w0.w, w1.w, xv[j].z, xv[j].w);
          }
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
        const int wr = ti.row0 + wrow + 16 * i + (c >= 2 ? 8 : 0);
        const int m = 8 * j + 2 * q + (c & 1);
        if (wr < ti.Ng && m < ti.M) {
          const size_t o = (size_t)(ti.tok0 + m) * op.ldo + (size_t)ti.grp * ti.Ng + wr;
          if (op.out_f32) static_cast<float*>(op.out)[o] = acc[i][j][c];
          else static_cast<__nv_bfloat16*>(op.out)[o] = __float2bfloat16_rn(acc[i][j][c]);
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
  const uint32_t smem_base = smem_u32(smem);
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * SW_STAGES;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < SW_STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, SW_CONSUMERS);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  const int total = total_tiles(P);
  uint32_t it = 0;
  if (warp == 0) {
    if (lane != 0) return;
    // ---- producer
    bool ok = true;
    for (int tile = blockIdx.x; tile < total && ok; tile += gridDim.x) {
      TileInfo ti;
      decode_tile(P, tile, ti);
      const CUtensorMap* map = P.op[ti.op].tmaps + ti.node;
      const int y = ti.grp * ti.Ng + ti.row0;
      const int nkb = (ti.K + SW_BOX * SW_STAGE_BOXES - 1) / (SW_BOX * SW_STAGE_BOXES);
      for (int kb = 0; kb < nkb; ++kb, ++it) {
        const uint32_t s = it % SW_STAGES;
        if (!mbar_wait(empty0 + 8 * s, ((it / SW_STAGES) & 1) ^ 1, abort_flag)) {
          ok = false;
          break;
        }
        const int kstage = kb * SW_BOX * SW_STAGE_BOXES;
        const int nb = (kstage + SW_BOX < ti.K) ? 2 : 1;
        mbar_expect_tx(full0 + 8 * s, nb * SW_BOX_BYTES);
        for (int b = 0; b < nb; ++b)
          tma_load_2d(smem_base + s * SW_STAGE_BYTES + b * SW_BOX_BYTES, map, kstage + b * SW_BOX,
                      y, full0 + 8 * s);
      }
    }
    if (!ok) {
      atomicExch(P.err, LX_ERR_TIMEOUT);
      *abort_flag = 1;
      // drain: every issued stage's copy must land before the CTA exits
      const uint32_t first = it > SW_STAGES ? it - SW_STAGES : 0;
      for (uint32_t j = first; j < it; ++j) {
        const uint32_t s = j % SW_STAGES;
        volatile int never = 0;
        mbar_wait(full0 + 8 * s, (j / SW_STAGES) & 1, &never);
      }
    }
    return;
  }
  // ---- consumers
  for (int tile = blockIdx.x; tile < total; tile += gridDim.x) {
    TileInfo ti;
    decode_tile(P, tile, ti);
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

int stream_smem_bytes() { return SW_STAGES * SW_STAGE_BYTES + 2 * SW_STAGES * 8 + 16 + 1024; }

lx_status launch_stream(lx_layer* L, const StreamLaunch& P, cudaStream_t s, const char* name) {
  const int smem = stream_smem_bytes();
  LX_CUDA(cudaFuncSetAttribute(k_stream_gemm, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
  ProfScope ps(L, s, name);
  k_stream_gemm<<<L->num_sms * 3, SW_THREADS, smem, s>>>(P);
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

static StreamOp make_op(lx_layer* L, int op, const __nv_bfloat16* X, long ldx, const int* gather,
                        void* out, long ldo, bool out_f32) {
  Workspace& w = L->ws;
  StreamOp o;
  o.shape = op_shape(L, op);
  o.tmaps = L->d_tmaps + (size_t)op * L->N;
  o.items = o.shape.on_anchors ? L->d_anchors : L->d_corrs;
  o.n_items = o.shape.on_anchors ? L->n_anchor : L->n_corr;
  o.tile_off = w.tile_off + (PLAN_STREAM + op) * (op_max_items(L) + 1);
  o.node_off = w.key_off;
  o.gather = gather;
  o.X = X;
  o.ldx = ldx;
  o.out = out;
  o.ldo = ldo;
  o.out_f32 = out_f32 ? 1 : 0;
  o.rank = L->d_rank;
  return o;
}

static lx_status run_stream(lx_layer* L, std::initializer_list<StreamOp> ops, cudaStream_t s,
                            const char* name) {
  StreamLaunch P;
  P.n_ops = 0;
  P.err = L->ws.err;
  for (const StreamOp& o : ops)
    if (o.n_items > 0) P.op[P.n_ops++] = o;
  if (P.n_ops == 0) return LX_OK;
  return launch_stream(L, P, s, name);
}

// The decode forward: every touched weight byte is streamed once.
lx_status launch_fast_experts(lx_layer* L, const void* x, int T, int k, void* y, cudaStream_t s) {
  Workspace& w = L->ws;
  const long H = L->H, I = L->I, rmax = L->max_rank;
  const __nv_bfloat16* xb = static_cast<const __nv_bfloat16*>(x);
  // x-side: shared anchor gate/up, and x V of every correction
  LX_TRY(run_stream(L, {make_op(L, OP_UP_ANCHOR, xb, H, w.node_tok, w.h, 2 * I, true),
                        make_op(L, OP_UP_V, xb, H, w.node_tok, w.Pb, 2 * rmax, false)},
                    s, "stream_up_anchor_V"));
  LX_TRY(run_stream(L, {make_op(L, OP_UP_U, w.Pb, 2 * rmax, nullptr, w.h, 2 * I, true)}, s,
                    "stream_up_U"));
  LX_TRY(launch_swiglu(L, k, w.zb, true, s));
  // z-side: shared anchor down projection, and z Vd of every correction
  LX_TRY(run_stream(L, {make_op(L, OP_DN_ANCHOR, w.zb, I, nullptr, w.ypart, H, true),
                        make_op(L, OP_DN_V, w.zb, I, nullptr, w.Qb, rmax, false)},
                    s, "stream_dn_anchor_V"));
  LX_TRY(run_stream(L, {make_op(L, OP_DN_U, w.Qb, rmax, nullptr, w.ypart, H, true)}, s,
                    "stream_dn_U"));
  LX_TRY(launch_combine(L, T, k, y, s));
  return LX_OK;
}

int stream_tile_rows() { return SW_ROWS; }
int stream_tile_tokens() { return SW_TOK; }
int stream_box() { return SW_BOX; }

}  // namespace lx
