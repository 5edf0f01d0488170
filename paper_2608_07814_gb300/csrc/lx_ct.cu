// Fused member correction + SwiGLU of flat layers on the tensor cores (prefill).
//
// For a cluster c (an anchor and its members, every member a direct child),
// the member e's gate/up pre-activations are the anchor's plus the rank-r
// correction, g_e(t) = h_c(t) + P_e(t) U_{g,e}^T and u_e(t) = u_c(t) +
// P'_e(t) U_{u,e}^T with P_e = x V_{g,e}, P'_e = x V_{u,e} (Sec. 3.1, Sec. 3.2
// Stage 3 iii).  The anchor products h_c, u_c are computed once per (token,
// cluster) and shared by every selected member (Sec. 5.1).  This kernel works
// on tiles of one cluster's bucket: 128 rows (tokens of the cluster) x 64
// d_ff columns.  For each member it accumulates the correction of all 128
// rows in tensor memory (the member's P rows stored aligned to the cluster's
// rows), and the epilogue applies the SwiGLU and the gates:
//   a_e(t) = g_{t,e} silu(h_c(t) + corr_g) (u_c(t) + corr_u)   (member rows)
//   z_c(t) = g_{t,dom} silu(h_c(t)) u_c(t) + sum_e a_e(t)      (cluster rows)
// so the correction products never leave the chip and the SwiGLU is not a
// separate pass.  z_c feeds the shared down product of the anchor and a_e the
// member's down correction (by linearity of the down projection).
//
// One persistent CTA per SM, 12 warps (warp 3 has no role):
//   warp 2      scheduler: claims tiles (anchor, 128-row block, 64-column
//               chunk; chunks of a block are consecutive, so the block's P
//               rows are re-read from L2) and decodes them into a queue;
//   warp 0      producer: per member, per 64-wide K block of the rank, the
//               gate then the up half: one stage = the 128 P rows (one TMA box of the
//               cluster-aligned P buffer) and the 64 U rows of the chunk (one
//               64 x 64 box of the member's tiled [Ug;Uu]);
//   warp 1      allocates 512 TMEM columns (four member accumulators of
//               [gate 64 | up 64] columns) and issues tcgen05.mma (M=128,
//               N=64, K=16, bf16 -> fp32), one accumulator per member in turn,
//               so that the MMAs run up to four members ahead of the epilogue;
//   warps 4..11 epilogue: two warps per TMEM lane quadrant, 32 columns
//               each; a thread owns one row of the tile: it keeps the anchor's
//               gate and up values and its z columns in registers, adds every
//               member's correction (tcgen05.ld), and stores a_e and z as bf16.
// Rows of a member's slot that did not select it hold stale P values; their
// accumulator rows are never read.  Every wait is bounded (LX_ERR_TIMEOUT).
#include <algorithm>
#include <climits>

#include "lx_internal.cuh"
#include "lx_tcgen05.cuh"

namespace lx {

namespace {

using namespace tcg;

constexpr int CT_BM = 128;
constexpr int CT_BK = 64;
constexpr int CT_A_BYTES = CT_BM * CT_BK * 2;           // 16 KiB
constexpr int CT_B_BYTES = CT_CW * CT_BK * 2;           // 8 KiB
constexpr int CT_STAGE_BYTES = CT_A_BYTES + CT_B_BYTES;  // 24 KiB
constexpr int CT_STAGES = 6;
// per tile, staged by the producer (double-buffered): the anchor's gate and up
// pre-activations of the tile's 128 rows x 64 columns (two 128-row TMA boxes,
// 128-byte swizzle) and the rows' gate / child-row tables (bulk copies)
constexpr int CT_H_BYTES = 2 * CT_BM * CT_CW * 2;        // 32 KiB
constexpr int CT_TAB_STRIDE = 8;                         // max table row (4-byte words)
static_assert(CT_MAX_CH + 1 <= CT_TAB_STRIDE, "a gate row fits the staged table");
constexpr int CT_TAB_BYTES = CT_BM * CT_TAB_STRIDE * 4;  // 4 KiB per table
constexpr int CT_ACC_COLS = 2 * CT_CW;                  // [gate | up]
constexpr int CT_NBUF = 4;                              // member accumulators in flight
constexpr int CT_TMEM_COLS = CT_NBUF * CT_ACC_COLS;     // all 512 columns
constexpr int CT_EPI_WARPS = 8;                       // 2 per TMEM lane quadrant
constexpr int CT_EC = CT_CW / (CT_EPI_WARPS / 4);     // columns of an epilogue warp
constexpr int CT_THREADS = 32 * (4 + CT_EPI_WARPS);
static_assert(CT_STAGE_BYTES % 1024 == 0, "stages keep the 1024-byte swizzle alignment");
static_assert(CT_CW == 64, "one 64-row U box per stage");
static_assert(CT_EC % 16 == 0, "an epilogue warp reads 16-column groups of each half");

struct CtLaunch {
  const int* items;        // anchors
  int n_items;
  const int* tile_off;     // [n_items+1]: ceil(rows / 128) * (I / 64) tiles per anchor
  const int* node_off;
  const int* child;        // [N][CT_MAX_CH]
  const int* rank;
  const CUtensorMap* umaps;  // [N] [Ug;Uu] maps (tiled, 64 x 64 boxes)
  const CUtensorMap* pmap;   // Pal, 128-row boxes
  const CUtensorMap* hmap;   // anchor pre-activations h [R][2I], 128-row boxes
  int pslot;               // columns of a child's slot in Pal (2 rmax)
  __nv_bfloat16* z;        // [R][I]
  __nv_bfloat16* qal;      // [R][qld]: child slot j at columns j * qslot (zeroed here
  int qld, qslot;          //  where the row did not select the child)
  const float* al_g;       // [R][gstride]: dominant's gate, then the children's
  const int* al_row;       // [R][rstride]: the children's rows
  int gstride, rstride;    // multiples of 4 (16-byte rows), at most CT_TAB_STRIDE
  int nch;
  int I;
  long rows_cap;
  int* ctr;
  int* err;
  unsigned long long wait_cycles;
  int unmet_wait;
};

struct CtTile {
  int node, tok0, M, q, nch;  // node < 0: sentinel
  int ch[CT_MAX_CH];
  int rk[CT_MAX_CH];
};

// tile index -> (anchor, block, chunk) through the plan prefix (whole warp:
// one round of independent loads and ballots, as in the tensor-core GEMM)
__device__ __forceinline__ void ct_decode_warp(const CtLaunch& P, int tile, CtTile& t) {
  const int lane = threadIdx.x & 31;
  const int* to = P.tile_off;
  int cnt = 0;
  for (int i0 = 0; i0 < P.n_items; i0 += 256) {
    int v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int i = i0 + lane + 32 * j;
      v[j] = i < P.n_items ? __ldg(to + i) : INT_MAX;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) cnt += __popc(__ballot_sync(0xffffffffu, v[j] <= tile));
  }
  const int lo = cnt - 1;
  const int n = __ldg(P.items + lo);
  const int local = tile - __ldg(to + lo);
  const int nchunk = P.I / CT_CW;
  const int b0 = __ldg(P.node_off + n), b1 = __ldg(P.node_off + n + 1);
  t.node = n;
  t.q = local % nchunk;
  t.tok0 = b0 + (local / nchunk) * CT_BM;
  t.M = min(CT_BM, b1 - t.tok0);
  const int c = lane < CT_MAX_CH ? __ldg(P.child + (size_t)n * CT_MAX_CH + lane) : -1;
  const int r = c >= 0 ? __ldg(P.rank + c) : 0;
  t.nch = __popc(__ballot_sync(0xffffffffu, c >= 0));
#pragma unroll
  for (int j = 0; j < CT_MAX_CH; ++j) {
    t.ch[j] = __shfl_sync(0xffffffffu, c, j);
    t.rk[j] = __shfl_sync(0xffffffffu, r, j);
  }
}

// one lane waits (bounded), the warp follows: the result is warp-uniform, and
// __syncwarp orders the other lanes' reads after lane 0's acquire
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          unsigned long long limit) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, abort_flag, limit) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  __syncwarp();
  return ok != 0;
}

// fp32 pairs and the packed fp32x2 arithmetic of sm_100+ (each half rounded
// as the scalar operation)
struct F2 {
  float x, y;
};
__device__ __forceinline__ F2 add2(F2 a, F2 b) {
  F2 d;
  asm("{\n\t.reg .b64 ra, rb, rd;\n\tmov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}
__device__ __forceinline__ F2 mul2(F2 a, F2 b) {
  F2 d;
  asm("{\n\t.reg .b64 ra, rb, rd;\n\tmov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "mul.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}
__device__ __forceinline__ F2 fma2(F2 a, F2 b, F2 c) {
  F2 d;
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\tmov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
      "mov.b64 rc, {%6, %7};\n\tfma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}
// 1-D bulk copy global -> shared (16-byte aligned addresses, size a multiple
// of 16), counted on the mbarrier
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}
__device__ __forceinline__ float tanh_approx(float v) {
  float r;
  asm("tanh.approx.f32 %0, %1;" : "=f"(r) : "f"(v));
  return r;
}
// silu(v) = v sigmoid(v) = h + h tanh(h) with h = v / 2 (one MUFU operation
// per element; tanh.approx's error, about 2^-11 relative, is far below the
// bf16 rounding of the operands and of the stored result)
__device__ __forceinline__ F2 silu2(F2 v) {
  const F2 h = mul2(v, F2{0.5f, 0.5f});
  return fma2(h, F2{tanh_approx(h.x), tanh_approx(h.y)}, h);
}
__device__ __forceinline__ F2 bf2(uint32_t w) {
  return F2{__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u)};
}

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ uint32_t pack_bf2(float a, float b) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&v);
}

__global__ void __launch_bounds__(CT_THREADS, 1) k_ct_swiglu(const __grid_constant__ CtLaunch P) {
  constexpr int S = CT_STAGES;
  pdl_wait();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint8_t* hbuf = smem + S * CT_STAGE_BYTES;                       // [2][gate | up box]
  uint8_t* tbuf = hbuf + 2 * CT_H_BYTES;                            // [2][gate table | row table]
  uint64_t* bars = reinterpret_cast<uint64_t*>(tbuf + 4 * CT_TAB_BYTES);
  // full[S], empty[S], tfull[NBUF], tempty[NBUF], efull[2], eempty[2], qfull, qempty, drain,
  // hfull[2], hempty[2]
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * S;
  const uint32_t tfull0 = empty0 + 8 * S, tempty0 = tfull0 + 8 * CT_NBUF;
  const uint32_t efull0 = tempty0 + 8 * CT_NBUF, eempty0 = efull0 + 16;
  const uint32_t qfull = eempty0 + 16, qempty = qfull + 8, drain = qempty + 8;
  const uint32_t hfull0 = drain + 8, hempty0 = hfull0 + 16;
  constexpr int NB = 2 * S + 2 * CT_NBUF + 11;  // mbarriers
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + NB);
  uint32_t* tmem_base_s = reinterpret_cast<uint32_t*>(bars + NB + 1);
  CtTile* slot = reinterpret_cast<CtTile*>(bars + NB + 2);  // [S] tile of a tile's first stage
  CtTile* eslot = slot + S;                                      // [2] MMA -> epilogue
  CtTile* qslot = eslot + 2;                                     // [1] scheduler -> producer
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t smem_base = smem_u32(smem);
  uint32_t prod_it = 0, prod_ht = 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full0 + 8 * s, 1);   // the producer's arrival (with the stage's bytes)
      mbar_init(empty0 + 8 * s, 1);  // tcgen05.commit (or the MMA thread's arrival)
    }
    for (int b = 0; b < CT_NBUF; ++b) {
      mbar_init(tfull0 + 8 * b, 1);   // tcgen05.commit: a member's accumulator is ready
      mbar_init(tempty0 + 8 * b, CT_EPI_WARPS);  // each epilogue warp: accumulator drained
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(efull0 + 8 * b, 1);   // the MMA thread: tile handed to the epilogue
      mbar_init(eempty0 + 8 * b, CT_EPI_WARPS);  // each epilogue warp: tile read
    }
    mbar_init(qfull, 1);
    mbar_init(qempty, 1);
    mbar_init(drain, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(hfull0 + 8 * b, 1);              // the producer's arrival (with the bytes)
      mbar_init(hempty0 + 8 * b, CT_EPI_WARPS);  // each epilogue warp: tile's rows read
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_base_s)),
                 "r"(CT_TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_base_s;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    uint32_t it = 0, qi = 0, ht = 0;
    bool ok = true;
    while (ok) {
      int got = 1;
      if (lane == 0) got = mbar_wait(qfull, qi & 1, abort_flag, P.wait_cycles);
      if (!__shfl_sync(0xffffffffu, got, 0)) {
        ok = false;
        break;
      }
      __syncwarp();
      const CtTile t = *qslot;
      __syncwarp();
      if (lane == 0) mbar_arrive(qempty);
      ++qi;
      const bool sentinel = t.node < 0;
      int good = 1;
      if (lane == 0 && !sentinel) {
        // the tile's anchor rows and tables, into the buffer the epilogue
        // released two tiles ago
        const uint32_t hb = ht % 2;
        good = mbar_wait(hempty0 + 8 * hb, ((ht / 2) & 1) ^ 1, abort_flag, P.wait_cycles);
        if (good) {
          const uint32_t gbytes = (uint32_t)t.M * P.gstride * 4, rbytes = (uint32_t)t.M * P.rstride * 4;
          mbar_expect_tx(hfull0 + 8 * hb, CT_H_BYTES + gbytes + rbytes);
          const uint32_t hs = smem_u32(hbuf) + hb * CT_H_BYTES;
          tma_load_2d(hs, P.hmap, t.q * CT_CW, t.tok0, hfull0 + 8 * hb);
          tma_load_2d(hs + CT_H_BYTES / 2, P.hmap, P.I + t.q * CT_CW, t.tok0, hfull0 + 8 * hb);
          const uint32_t ts = smem_u32(tbuf) + hb * 2 * CT_TAB_BYTES;
          bulk_load(ts, P.al_g + (size_t)t.tok0 * P.gstride, gbytes, hfull0 + 8 * hb);
          bulk_load(ts + CT_TAB_BYTES, P.al_row + (size_t)t.tok0 * P.rstride, rbytes, hfull0 + 8 * hb);
          ++ht;
        }
      }
      if (lane == 0 && good) {
        int nst = 0;
        if (!sentinel)
          for (int j = 0; j < t.nch; ++j) nst += 2 * (t.rk[j] / CT_BK);
        if (nst == 0) {
          // a tile without members (or the sentinel): its header alone, in a
          // stage without copies
          const uint32_t s = it % S;
          good = mbar_wait(empty0 + 8 * s, ((it / S) & 1) ^ 1, abort_flag, P.wait_cycles);
          if (good) {
            slot[s] = t;
            mbar_arrive(full0 + 8 * s);
            ++it;
          }
        } else {
          bool first = true;
          for (int j = 0; j < t.nch && good; ++j) {
            const int kbn = t.rk[j] / CT_BK;
            for (int kb = 0; kb < kbn && good; ++kb) {
              for (int g = 0; g < 2; ++g) {
                const uint32_t s = it % S;
                good = mbar_wait(empty0 + 8 * s, ((it / S) & 1) ^ 1, abort_flag, P.wait_cycles);
                if (!good) break;
                if (first) slot[s] = t;
                first = false;
                mbar_expect_tx(full0 + 8 * s, CT_STAGE_BYTES);
                const uint32_t a_s = smem_base + s * CT_STAGE_BYTES, b_s = a_s + CT_A_BYTES;
                // the member's P (gate: columns 0..r, up: r..2r of its slot) for
                // the block's 128 cluster rows, and 64 U rows of the chunk
                tma_load_2d(a_s, P.pmap, j * P.pslot + g * t.rk[j] + kb * CT_BK, t.tok0,
                            full0 + 8 * s);
                tma_load_4d(b_s, P.umaps + t.ch[j], 0, 0, kb, g * (P.I / CT_CW) + t.q,
                            full0 + 8 * s);
                ++it;
              }
            }
          }
        }
      }
      good = __shfl_sync(0xffffffffu, good, 0);
      if (!good) {
        ok = false;
        break;
      }
      if (sentinel) break;
    }
    if (!ok && lane == 0) {
      atomicExch(P.err, LX_ERR_TIMEOUT);
      *abort_flag = 1;
    }
    prod_it = __shfl_sync(0xffffffffu, it, 0);
    prod_ht = __shfl_sync(0xffffffffu, ht, 0);
  } else if (warp == 2) {
    // ------------------------------------------------------------ scheduler
    const int total = P.tile_off[P.n_items];
    uint32_t qi = 0;
    bool ok = true;
    while (true) {
      int cur = lane == 0 ? atomicAdd(P.ctr, 1) : 0;
      cur = __shfl_sync(0xffffffffu, cur, 0);
      CtTile t;
      if (cur < total) {
        ct_decode_warp(P, cur, t);
      } else {
        t.node = -1;
        t.nch = 0;
      }
      int good = 1;
      if (lane == 0) {
        good = mbar_wait(qempty, (qi & 1) ^ 1, abort_flag, P.wait_cycles) ? 1 : 0;
        if (good) {
          *qslot = t;
          mbar_arrive(qfull);
        }
      }
      good = __shfl_sync(0xffffffffu, good, 0);
      if (!good) {
        ok = false;
        break;
      }
      ++qi;
      if (cur >= total) break;
    }
    if (!ok && lane == 0) {
      atomicExch(P.err, LX_ERR_TIMEOUT);
      *abort_flag = 1;
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      uint32_t it = 0, mc = 0, et = 0;
      bool ok = true;
      // an injected unmet wait (test hook): the drain barrier gets no arrival
      // before the abort path, so this bounded wait runs out
      if (P.unmet_wait == LX_WAIT_TC_MMA && !mbar_wait(drain, 0, abort_flag, P.wait_cycles))
        ok = false;
      const uint32_t idesc = instr_desc(CT_BM, CT_CW);
      while (ok) {
        uint32_t s = it % S;
        if (!mbar_wait(full0 + 8 * s, (it / S) & 1, abort_flag, P.wait_cycles)) {
          ok = false;
          break;
        }
        const CtTile t = slot[s];
        const uint32_t e = et % 2;
        if (!mbar_wait(eempty0 + 8 * e, ((et / 2) & 1) ^ 1, abort_flag, P.wait_cycles)) {
          ok = false;
          break;
        }
        eslot[e] = t;  // released to the epilogue by this arrival
        mbar_arrive(efull0 + 8 * e);
        ++et;
        if (t.node < 0) break;  // sentinel
        if (t.nch == 0) {       // the header stage of a tile without members
          mbar_arrive(empty0 + 8 * s);
          ++it;
          continue;
        }
        for (int j = 0; j < t.nch && ok; ++j) {
          const uint32_t b = mc % CT_NBUF;
          // this accumulator must have been drained (CT_NBUF members ago)
          if (!mbar_wait(tempty0 + 8 * b, ((mc / CT_NBUF) & 1) ^ 1, abort_flag, P.wait_cycles)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d = tmem + b * CT_ACC_COLS;
          const int kbn = t.rk[j] / CT_BK;
          // per K block, the gate and the up stage: their MMAs alternate between
          // the two accumulators, so that consecutive MMAs are independent (an
          // N = 64 MMA is shorter than the latency of accumulating into the
          // result of the previous one)
          for (int kb = 0; kb < kbn && ok; ++kb) {
            const uint32_t s0 = it % S, s1 = (it + 1) % S;
            if (!mbar_wait(full0 + 8 * s0, (it / S) & 1, abort_flag, P.wait_cycles) ||
                !mbar_wait(full0 + 8 * s1, ((it + 1) / S) & 1, abort_flag, P.wait_cycles)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t a0 = smem_base + s0 * CT_STAGE_BYTES, b0 = a0 + CT_A_BYTES;
            const uint32_t a1 = smem_base + s1 * CT_STAGE_BYTES, b1 = a1 + CT_A_BYTES;
#pragma unroll
            for (int k = 0; k < CT_BK / 16; ++k) {
              const uint32_t acc = (kb | k) != 0 ? 1u : 0u;
              tc_mma(d, smem_desc(a0 + 32 * k), smem_desc(b0 + 32 * k), idesc, acc);
              tc_mma(d + CT_CW, smem_desc(a1 + 32 * k), smem_desc(b1 + 32 * k), idesc, acc);
            }
            tc_commit(empty0 + 8 * s0);  // free the stages once these MMAs are done
            tc_commit(empty0 + 8 * s1);
            it += 2;
          }
          if (!ok) break;
          tc_commit(tfull0 + 8 * b);  // the member's accumulator is ready
          ++mc;
        }
      }
      if (!ok) {
        atomicExch(P.err, LX_ERR_TIMEOUT);
        *abort_flag = 1;
        tc_commit(drain);  // arrives once every MMA issued so far has completed
        mbar_wait(drain, 0, nullptr);
      }
    }
    __syncwarp();
  } else if (warp >= 4) {
    // ------------------------------------------------------------ epilogue
    // warp w: TMEM lanes 32 (w % 4) .. + 31 (the tile rows it may access) and
    // the tile's columns CT_EC ((w - 4) / 4) .. + CT_EC - 1
    const int ew = warp & 3, cs = (warp - 4) >> 2;
    const long I = P.I;
    uint32_t et = 0, mc = 0, nt = 0;
    bool failed = false;
    while (!failed) {
      const uint32_t e = et % 2;
      if (!warp_wait(efull0 + 8 * e, (et / 2) & 1, abort_flag, P.wait_cycles)) {
        failed = true;
        break;
      }
      const CtTile t = eslot[e];
      __syncwarp();
      if (lane == 0) mbar_arrive(eempty0 + 8 * e);
      ++et;
      if (t.node < 0) break;
      const int m = 32 * ew + lane;
      const long a = (long)t.tok0 + m;
      const bool valid = m < t.M && a < P.rows_cap;
      const long c0 = (long)t.q * CT_CW + CT_EC * cs;
      // the tile's anchor rows and tables, staged by the producer
      const uint32_t hb = nt % 2;
      if (!warp_wait(hfull0 + 8 * hb, (nt / 2) & 1, abort_flag, P.wait_cycles)) {
        failed = true;
        break;
      }
      // row m of each 128-byte-swizzled box: 16-byte unit u sits at u ^ (m % 8);
      // the anchor values are read from the staged boxes where they are used
      // (the registers go to a member's whole set of accumulator loads), and
      // the buffer is released once the tile is done
      const uint8_t* gbox = hbuf + hb * CT_H_BYTES + m * 128;
      const uint8_t* ubox = gbox + CT_H_BYTES / 2;
      auto h_unit = [&](const uint8_t* box, int i) {  // this warp's 16-byte unit i (8 columns)
        return *reinterpret_cast<const uint4*>(box + 16 * (((CT_EC / 8) * cs + i) ^ (m & 7)));
      };
      float gd = 0.f;
      float gm[CT_MAX_CH];
      int rm[CT_MAX_CH];
      {
        const float* tg = reinterpret_cast<const float*>(tbuf + hb * 2 * CT_TAB_BYTES) + m * P.gstride;
        const int* tr = reinterpret_cast<const int*>(tbuf + hb * 2 * CT_TAB_BYTES + CT_TAB_BYTES) +
                        m * P.rstride;
        gd = valid ? tg[0] : 0.f;
#pragma unroll
        for (int jj = 0; jj < CT_MAX_CH; ++jj) {
          gm[jj] = (valid && jj < t.nch) ? tg[1 + jj] : 0.f;
          rm[jj] = (valid && jj < t.nch) ? tr[jj] : -1;
        }
      }
      // the down side sums every child slot of a cluster row: the slots of
      // children this row did not select are zeroed (once, by the first chunk)
      if (t.q == 0 && cs == 0 && valid) {
#pragma unroll
        for (int jj = 0; jj < CT_MAX_CH; ++jj) {
          if (jj >= t.nch || rm[jj] >= 0) continue;
          uint4* q = reinterpret_cast<uint4*>(P.qal + (size_t)a * P.qld + (size_t)jj * P.qslot);
          for (int i = 0; i < t.rk[jj] / 8; ++i) q[i] = make_uint4(0u, 0u, 0u, 0u);
        }
      }
      // z starts with the dominant's own gated SwiGLU (if the token selected it)
      F2 zr[CT_EC / 2];
      if (__any_sync(0xffffffffu, gd != 0.f)) {
        const F2 gd2{gd, gd};
#pragma unroll
        for (int i = 0; i < CT_EC / 8; ++i) {
          const uint4 vg = h_unit(gbox, i), vu = h_unit(ubox, i);
          const uint32_t wg[4] = {vg.x, vg.y, vg.z, vg.w}, wu[4] = {vu.x, vu.y, vu.z, vu.w};
#pragma unroll
          for (int q = 0; q < 4; ++q) zr[4 * i + q] = mul2(mul2(silu2(bf2(wg[q])), bf2(wu[q])), gd2);
        }
      } else {
#pragma unroll
        for (int i = 0; i < CT_EC / 2; ++i) zr[i] = F2{0.f, 0.f};
      }
      for (int j = 0; j < t.nch; ++j) {
        const uint32_t b = mc % CT_NBUF;
        if (!warp_wait(tfull0 + 8 * b, (mc / CT_NBUF) & 1, abort_flag, P.wait_cycles)) {
          failed = true;
          break;
        }
        tc_fence_after();
        float gj = 0.f;
        int rj = -1;
#pragma unroll
        for (int jj = 0; jj < CT_MAX_CH; ++jj)
          if (jj == j) {
            gj = gm[jj];
            rj = rm[jj];
          }
        const bool use = valid && rj >= 0 && (long)rj < P.rows_cap;
        if (__any_sync(0xffffffffu, use)) {
          const uint32_t acc =
              tmem + ((uint32_t)(32 * ew) << 16) + b * CT_ACC_COLS + CT_EC * cs;
          const F2 gj2{gj, gj};
          uint4* dst = reinterpret_cast<uint4*>(P.z + (size_t)(use ? rj : 0) * I + c0);
          // all of the member's accumulator columns of this warp in flight, one wait
          uint32_t cg[CT_EC], cu[CT_EC];
#pragma unroll
          for (int q16 = 0; q16 < CT_EC / 16; ++q16) {
            tc_ld16_async(acc + 16 * q16, *reinterpret_cast<uint32_t(*)[16]>(cg + 16 * q16));
            tc_ld16_async(acc + CT_CW + 16 * q16, *reinterpret_cast<uint32_t(*)[16]>(cu + 16 * q16));
          }
          tc_wait_ld();
#pragma unroll
          for (int i = 0; i < CT_EC / 8; ++i) {  // 16-byte unit i: column pairs 4 i .. 4 i + 3
            const uint4 vg = h_unit(gbox, i), vu = h_unit(ubox, i);
            const uint32_t wg[4] = {vg.x, vg.y, vg.z, vg.w}, wu[4] = {vu.x, vu.y, vu.z, vu.w};
            uint32_t pk[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const int w = 4 * i + q;  // column pair 2 w, 2 w + 1 of this warp
              const F2 gp = add2(bf2(wg[q]), F2{__uint_as_float(cg[2 * w]), __uint_as_float(cg[2 * w + 1])});
              const F2 up = add2(bf2(wu[q]), F2{__uint_as_float(cu[2 * w]), __uint_as_float(cu[2 * w + 1])});
              const F2 av = mul2(mul2(silu2(gp), up), gj2);
              if (use) zr[w] = add2(zr[w], av);
              pk[q] = pack_bf2(av.x, av.y);
            }
            if (use) dst[i] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(tempty0 + 8 * b);
        ++mc;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(hempty0 + 8 * hb);  // this tile's staged rows are done
      ++nt;
      if (failed) break;
      if (valid) {
        uint4* dst = reinterpret_cast<uint4*>(P.z + a * I + c0);
#pragma unroll
        for (int i = 0; i < CT_EC / 8; ++i)
          dst[i] = make_uint4(pack_bf2(zr[4 * i].x, zr[4 * i].y), pack_bf2(zr[4 * i + 1].x, zr[4 * i + 1].y),
                              pack_bf2(zr[4 * i + 2].x, zr[4 * i + 2].y),
                              pack_bf2(zr[4 * i + 3].x, zr[4 * i + 3].y));
      }
    }
    if (failed && lane == 0) {
      atomicExch(P.err, LX_ERR_TIMEOUT);
      *abort_flag = 1;
    }
  }
  // all roles meet before the TMEM is released
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(CT_TMEM_COLS)
                 : "memory");
  } else if (warp == 0 && lane == 0 && *abort_flag) {
    // an aborted CTA may leave copies in flight: wait (bounded) for the last
    // stages the producer issued before shared memory goes away
    const uint32_t first = prod_it > S ? prod_it - S : 0;
    for (uint32_t j = first; j < prod_it; ++j) mbar_wait(full0 + 8 * (j % S), (j / S) & 1, nullptr);
    const uint32_t hfirst = prod_ht > 2 ? prod_ht - 2 : 0;
    for (uint32_t j = hfirst; j < prod_ht; ++j) mbar_wait(hfull0 + 8 * (j % 2), (j / 2) & 1, nullptr);
  }
}

}  // namespace

lx_status launch_ct_swiglu(lx_layer* L, cudaStream_t s) {
  Workspace& w = L->ws;
  CtLaunch P;
  P.items = L->d_anchors;
  P.n_items = L->n_anchor;
  P.tile_off = w.tile_off + (PLAN_TC + OP_UP_U) * (op_max_items(L) + 1);
  P.node_off = w.key_off;
  P.child = L->d_child;
  P.rank = L->d_rank;
  P.umaps = L->d_tmaps + (size_t)OP_UP_U * L->N;
  P.pmap = w.pamap;
  P.hmap = w.pamap + 1;
  P.pslot = 2 * std::max(1, L->max_rank);
  P.z = w.zb;
  P.qal = w.Qal;
  P.qslot = std::max(1, L->max_rank);
  P.qld = L->ct_nch * P.qslot;
  P.al_g = w.al_g;
  P.al_row = w.al_row;
  P.gstride = ct_gstride(L);
  P.rstride = ct_rstride(L);
  P.nch = L->ct_nch;
  P.I = L->I;
  P.rows_cap = w.rows_cap;
  P.ctr = w.sctr + N_STREAM_GROUPS + OP_UP_U;
  P.err = w.err;
  P.wait_cycles = wait_limit(L);
  P.unmet_wait = L->unmet_wait;
  constexpr int smem = CT_STAGES * CT_STAGE_BYTES + 2 * CT_H_BYTES + 4 * CT_TAB_BYTES +
                       8 * (2 * CT_STAGES + 2 * CT_NBUF + 13) +
                       (CT_STAGES + 3) * (int)sizeof(CtTile) + 1024;
  static_assert(smem <= 227 * 1024, "fits the shared memory of one CTA");
  static bool done[64] = {};
  LX_CUDA(smem_cap_once((const void*)k_ct_swiglu, smem, L->device, done));
  ProfScope ps(L, s, "ct_swiglu");
  launch_k(L, k_ct_swiglu, L->num_sms, CT_THREADS, smem, s, P);
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

}  // namespace lx
