// Tensor-core grouped GEMM for large token counts (prefill), sm_103a tcgen05.
//
// out[rows of node n][cols] = X[rows][K] . W_n[cols][K]^T for every active
// node, in tiles of 128 tokens (rows of the node's bucket) x BN <= 256 output
// columns over the full K -- the dense anchor and factor contractions of the
// amortised forward (Sec. 5.1), each evaluated once per (token, node).
//
// One persistent CTA per SM, 8 warps:
//   warp 2      scheduler: claims tiles from the launch's counter and
//               decodes them (plan-prefix search, bucket lookups) into a small
//               shared-memory queue ahead of the producer;
//   warp 0      producer: takes decoded tiles from the queue and loads the
//               weight boxes (64 rows x 64 K, 128B swizzle, tiled layout) and
//               the 128 token rows (one box: rows are contiguous in node-row
//               order, x rows having been gathered once) with TMA;
//   warp 1      allocates 512 TMEM columns (two 256-column accumulators, so
//               the epilogue of one tile overlaps the MMAs of the next); lane 0
//               issues tcgen05.mma (kind::f16, bf16 x bf16 -> fp32, M=128,
//               N=BN, K=16 per instruction) and commits stage releases and
//               accumulator-ready signals with tcgen05.commit;
//   warps 4..7  epilogue: tcgen05.ld (32 lanes x 32 columns per load), a
//               transpose through a per-warp shared-memory block, and stores
//               of whole 128-byte row segments.
// Every wait is bounded; a wait that gives up records LX_ERR_TIMEOUT, makes the
// other roles stop, drains the CTA's copies and MMAs in flight and frees TMEM.
#include <cuda.h>

#include <algorithm>
#include <climits>

#include "lx_internal.cuh"
#include "lx_tcgen05.cuh"

namespace lx {

namespace {

using namespace tcg;

constexpr int TC_BN = 256;          // max output columns per tile (UMMA N)
constexpr int TC_BK = 64;           // K per stage (one 128-byte swizzle row)
constexpr int TC_B_BYTES = TC_BN * TC_BK * 2;   // 32 KiB
constexpr int TC_ACC_COLS = 256;                 // one accumulator
constexpr int TC_TMEM_COLS = 2 * TC_ACC_COLS;    // double-buffered
constexpr int TC_EPI_LD = 36;                    // staging row stride (floats)
constexpr int TC_EPI_BYTES = 32 * TC_EPI_LD * 4; // per epilogue warp
constexpr int TC_QN = 1;
constexpr int TC_GATHER_WARPS = 2;  // warps gathering the A rows of a gathered product  // decoded tiles queued ahead of the producer (one, as a claim one tile ahead)

// Tile rows BM (tokens): 128 (one M = 128 MMA per K step, two TMEM
// accumulators so that a tile's epilogue overlaps the next tile's MMAs) or 256
// (two M = 128 MMAs per K step share each weight box: 1.5x the tensor work per
// byte in flight, which lifts the long-K products whose stage ring cannot
// cover the load latency; one accumulator of 2 x 256 columns, so the epilogue
// does not overlap the next tile).
// EPI: epilogue warps, 4 or 8 (two per TMEM lane quadrant, splitting the
// column passes; for the short-K factor products, whose tiles are bound by
// writing their output, with a 3-stage ring to make room for the staging).
template <int BM, int EPI>
struct TcCfg {
  static constexpr int NH = BM / 128;                    // 128-row halves of a tile
  static constexpr int A_BYTES = BM * TC_BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + TC_B_BYTES;
  static constexpr int STAGES = (NH == 1 && EPI == 4) ? 4 : 3;
  static constexpr int NBUF = NH == 1 ? 2 : 1;           // accumulators of NH x 256 columns
  static constexpr int THREADS = 32 * (4 + EPI);
  // 256-row tiles with eight epilogue warps stage 32 bf16 columns per pass:
  // two 2 KiB buffers per warp for TMA stores of 32 x 32 blocks (64-byte rows,
  // 64-byte swizzle), or 80-byte rows for the row-by-row stores
  static constexpr bool HALF = BM == 256 && EPI == 8;
  static constexpr int EPI_LD = HALF ? 20 : TC_EPI_LD;  // staging row stride (4-byte words)
  static constexpr int EPI_BYTES = HALF ? 4096 : 32 * EPI_LD * 4;
  static_assert(!HALF || 32 * EPI_LD * 4 <= EPI_BYTES, "row-by-row staging fits the buffers");
  static_assert(EPI == 4 || EPI == 8, "four or eight epilogue warps");
  static_assert(STAGE_BYTES % 1024 == 0, "stages keep the 1024-byte swizzle alignment");
  static_assert(NBUF * NH * TC_ACC_COLS <= TC_TMEM_COLS, "accumulators fit the TMEM allocation");
};

struct TcTile {
  int node, grp, row0, tok0, M, Ng, K, BN;  // BN < 0: sentinel
};

// Tile index -> (node, token block, group, column block) through the plan
// prefix, by the whole producer warp: one round of independent loads of the
// prefix and ballots count the items whose first tile is <= `tile` (the
// prefix is non-decreasing and starts at 0), instead of a chain of dependent
// loads of a binary search.
template <int BM>
__device__ __forceinline__ void tc_decode_warp(const TcLaunch& P, int tile, TcTile& t) {
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
  const int r = __ldg(P.rank + n);
  const int b0 = __ldg(P.node_off + n), b1 = __ldg(P.node_off + n + 1);
  t.Ng = P.shape.n_const + P.shape.n_rank * r;
  t.K = P.shape.k_const + P.shape.k_rank * r;
  if (P.kc_child) {
    // K concatenation: the anchor's children's rank-r products follow its own K
    const int c = lane < CT_MAX_CH ? __ldg(P.kc_child + (size_t)n * CT_MAX_CH + lane) : -1;
    int rc = c >= 0 ? __ldg(P.rank + c) : 0;
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) rc += __shfl_xor_sync(0xffffffffu, rc, o);
    t.K += rc;
  }
  const int ncol = (t.Ng + TC_BN - 1) / TC_BN;
  const int per_tb = ncol * P.shape.groups;
  const int tb = local / per_tb, rem = local % per_tb;
  t.grp = rem / ncol;
  t.row0 = (rem % ncol) * TC_BN;
  t.BN = min(TC_BN, t.Ng - t.row0);
  t.node = n;
  t.tok0 = b0 + tb * BM;
  t.M = min(BM, b1 - t.tok0);
}

// cp.async 16-byte copy global -> shared, completion tracked by cp.async groups
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}

// GATHER: warps 3 and 4 + EPI (TC_GATHER_WARPS, each half of the rows) fill
// the A stages with the tile's token rows, gathered from
// x by row -> token (16-byte cp.async, eight lanes per 128-byte row segment,
// stored in the 128-byte-swizzled K-major layout the MMA reads); a stage is
// published once its copies have landed (cp.async.wait_group) and been made
// visible to the tensor core's async proxy (fence.proxy.async), so no copy of
// the token rows in node-row order is written to memory first.
template <int BM, int EPI, bool GATHER>
__global__ void __launch_bounds__(TcCfg<BM, EPI>::THREADS + (GATHER ? 32 * (TC_GATHER_WARPS - 1) : 0), 1)
k_tc_gemm(const __grid_constant__ TcLaunch P) {
  using C = TcCfg<BM, EPI>;
  constexpr int TC_STAGES = C::STAGES, TC_STAGE_BYTES = C::STAGE_BYTES, TC_A_BYTES = C::A_BYTES;
  constexpr int NH = C::NH, NBUF = C::NBUF;
  pdl_wait();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  float* epi = reinterpret_cast<float*>(smem + TC_STAGES * TC_STAGE_BYTES);  // [EPI][32][EPI_LD]
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + TC_STAGES * TC_STAGE_BYTES + EPI * C::EPI_BYTES);
  // full[S], empty[S], tmem_full[2], tmem_empty[2], drain
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * TC_STAGES;
  const uint32_t tfull0 = empty0 + 8 * TC_STAGES, tempty0 = tfull0 + 16, drain = tempty0 + 16;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 2 * TC_STAGES + 5);
  uint32_t* tmem_base_s = reinterpret_cast<uint32_t*>(bars + 2 * TC_STAGES + 6);
  TcTile* slot = reinterpret_cast<TcTile*>(bars + 2 * TC_STAGES + 7);     // [TC_STAGES]
  TcTile* eslot = slot + TC_STAGES;                                         // [2] epilogue hand-off
  TcTile* qslot = eslot + 2;                                                // [TC_QN] decoded tiles
  uint64_t* qbars = reinterpret_cast<uint64_t*>(qslot + TC_QN);             // qfull[QN], qempty[QN]
  const uint32_t qfull0 = smem_u32(qbars), qempty0 = qfull0 + 8 * TC_QN;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t smem_base = smem_u32(smem);
  uint32_t prod_it = 0;  // stages the producer issued

  if (threadIdx.x == 0) {
    for (int s = 0; s < TC_STAGES; ++s) {
      // the producer's arrival (with the bytes) + one per lane of the producer
      // (or of every gather warp)
      mbar_init(full0 + 8 * s, 1 + 32 * (GATHER ? TC_GATHER_WARPS : 1));
      mbar_init(empty0 + 8 * s, 1);      // tcgen05.commit
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(tfull0 + 8 * b, 2);   // MMA thread's arrival (tile info written) + tcgen05.commit
      mbar_init(tempty0 + 8 * b, EPI);  // one arrival per epilogue warp
    }
    mbar_init(drain, 1);
    for (int q = 0; q < TC_QN; ++q) {
      mbar_init(qfull0 + 8 * q, 1);   // the scheduler's arrival (tile written)
      mbar_init(qempty0 + 8 * q, GATHER ? 1 + TC_GATHER_WARPS : 1);  // producer (+ gather warps)
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_base_s)),
                 "r"(TC_TMEM_COLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_base_s;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    // Tiles come decoded from the scheduler warp's queue, so that the TMA
    // issue never waits on the plan lookups.
    uint32_t it = 0, qi = 0;
    bool ok = true;
    while (ok) {
      const uint32_t q = qi % TC_QN;
      int got = 1;
      if (lane == 0) got = mbar_wait(qfull0 + 8 * q, (qi / TC_QN) & 1, abort_flag, P.wait_cycles);
      if (!__shfl_sync(0xffffffffu, got, 0)) {
        ok = false;
        break;
      }
      __syncwarp();  // lane 0's acquire orders the scheduler's write before every lane's read
      const TcTile t = qslot[q];
      __syncwarp();
      if (lane == 0) mbar_arrive(qempty0 + 8 * q);
      ++qi;
      if (t.BN < 0) break;  // no tile left
      const int nkb = (t.K + TC_BK - 1) / TC_BK;
      const int rt0 = (t.grp * t.Ng + t.row0) / 64;  // first 64-row weight tile
      const int nbox = (t.BN + 63) / 64;
      // K concatenation: k-blocks from kb_own on read child cj's k-block ckb;
      // the tile's children and their K blocks are looked up once, lane j
      // holding child j (their loads overlap the tile's first stages)
      const int kb_own = P.kc_child ? P.shape.k_const / TC_BK : nkb;
      int my_child = -1, my_nkb = 0;
      if (P.kc_child && lane < CT_MAX_CH) {
        my_child = __ldg(P.kc_child + (size_t)t.node * CT_MAX_CH + lane);
        my_nkb = my_child >= 0 ? __ldg(P.rank + my_child) / TC_BK : 0;
      }
      int cj = 0, ckb = 0;
      for (int kb = 0; kb < nkb; ++kb, ++it) {
        const uint32_t s = it % TC_STAGES;
        int cnode = -1, cnkb = 0;
        if (kb >= kb_own) {  // warp-uniform: every lane takes child cj's entry
          cnode = __shfl_sync(0xffffffffu, my_child, cj);
          cnkb = __shfl_sync(0xffffffffu, my_nkb, cj);
        }
        int good = 1;
        if (lane == 0) {
          good = mbar_wait(empty0 + 8 * s, ((it / TC_STAGES) & 1) ^ 1, abort_flag,
                           P.wait_cycles) ? 1 : 0;
          if (good) {
            if (kb == 0) slot[s] = t;
            // a 256-row tile whose rows end within its first half loads one half
            const int nh = GATHER ? 0 : ((NH == 2 && t.M > 128) ? 2 : 1);
            mbar_expect_tx(full0 + 8 * s, nbox * 8192 + nh * 128 * TC_BK * 2);
            const uint32_t a_s = smem_base + s * TC_STAGE_BYTES, b_s = a_s + TC_A_BYTES;
            if (kb < kb_own) {
              for (int b = 0; b < nbox; ++b)
                tma_load_4d(b_s + b * 8192, P.wmaps + t.node, 0, 0, kb, rt0 + b, full0 + 8 * s);
              for (int h = 0; h < nh; ++h)
                tma_load_2d(a_s + h * 128 * TC_BK * 2, P.xmap,
                            (int)(t.grp * t.K) + kb * TC_BK + P.xcol, t.tok0 + 128 * h,
                            full0 + 8 * s);
            } else {
              for (int b = 0; b < nbox; ++b)
                tma_load_4d(b_s + b * 8192, P.kc_wmaps + cnode, 0, 0, ckb, rt0 + b, full0 + 8 * s);
              for (int h = 0; h < nh; ++h)
                tma_load_2d(a_s + h * 128 * TC_BK * 2, P.kc_xmap, cj * P.kc_slot + ckb * TC_BK,
                            t.tok0 + 128 * h, full0 + 8 * s);
            }
          }
        }
        if (kb >= kb_own && ++ckb == cnkb) {  // every lane walks the children alike
          ckb = 0;
          ++cj;
        }
        good = __shfl_sync(0xffffffffu, good, 0);
        if (!good) {
          ok = false;
          break;
        }
        if (!GATHER) mbar_arrive(full0 + 8 * s);  // else the gather warp's 32 lanes arrive
      }
    }
    if (ok) {
      // sentinel stage
      const uint32_t s = it % TC_STAGES;
      int good = 1;
      if (lane == 0) {
        good = mbar_wait(empty0 + 8 * s, ((it / TC_STAGES) & 1) ^ 1, abort_flag, P.wait_cycles)
                   ? 1 : 0;
        if (good) {
          slot[s].BN = -1;
          mbar_arrive(full0 + 8 * s);
        }
      }
      good = __shfl_sync(0xffffffffu, good, 0);
      if (good) {
        if (!GATHER) mbar_arrive(full0 + 8 * s);
        ++it;
      } else {
        ok = false;
      }
    }
    if (!ok && lane == 0) {
      atomicExch(P.err, LX_ERR_TIMEOUT);
      *abort_flag = 1;
    }
    prod_it = it;
  } else if (GATHER && (warp == 3 || warp >= 4 + EPI)) {
    // ------------------------------------------------------------ gather
    // Same tiles and stages as the producer: gather warp gw takes rows
    // m = 4 i + r8 of the tile for i in its half (lanes 8 r8 .. 8 r8 + 7),
    // 16-byte unit u of the stage's 64-wide K slice; up to TC_STAGES - 1
    // stages in flight before the oldest is published (32 arrivals per warp
    // on its full barrier).
    constexpr int GR = BM / 4 / TC_GATHER_WARPS;  // row groups of a gather warp
    const int gw = warp == 3 ? 0 : warp - (4 + EPI) + 1;
    const int r8 = lane >> 3, u = lane & 7;
    uint32_t it = 0, qi = 0, pq = 0;
    int np = 0;
    bool ok = true;
    auto publish_oldest = [&]() {
      asm volatile("cp.async.wait_group %0;" ::"n"(TC_STAGES - 2) : "memory");
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      mbar_arrive(full0 + 8 * (pq & 0xffu));
      pq >>= 8;
      --np;
    };
    while (ok) {
      const uint32_t q = qi % TC_QN;
      int got = 1;
      if (lane == 0) got = mbar_wait(qfull0 + 8 * q, (qi / TC_QN) & 1, abort_flag, P.wait_cycles);
      if (!__shfl_sync(0xffffffffu, got, 0)) {
        ok = false;
        break;
      }
      __syncwarp();
      const TcTile t = qslot[q];
      __syncwarp();
      if (lane == 0) mbar_arrive(qempty0 + 8 * q);
      ++qi;
      if (t.BN < 0) break;
      // this lane's source row addresses (16-byte unit u of the row's first
      // K slice), or null past the bucket
      const __nv_bfloat16* src[GR];
#pragma unroll
      for (int i = 0; i < GR; ++i) {
        const int m = 4 * (gw * GR + i) + r8;
        const int tr = (m < t.M && (long)t.tok0 + m < P.rows_cap) ? __ldg(P.gather + t.tok0 + m) : -1;
        src[i] = tr >= 0 ? P.xsrc + (size_t)tr * P.ldx + (size_t)(t.grp * t.K) + 8 * u : nullptr;
      }
      const int nkb = (t.K + TC_BK - 1) / TC_BK;
      for (int kb = 0; kb < nkb; ++kb, ++it) {
        const uint32_t s = it % TC_STAGES;
        int good = 1;
        if (lane == 0)
          good = mbar_wait(empty0 + 8 * s, ((it / TC_STAGES) & 1) ^ 1, abort_flag, P.wait_cycles)
                     ? 1 : 0;
        good = __shfl_sync(0xffffffffu, good, 0);
        if (!good) {
          ok = false;
          break;
        }
        const uint32_t a_s = smem_base + s * TC_STAGE_BYTES;
#pragma unroll
        for (int i = 0; i < GR; ++i) {
          const int m = 4 * (gw * GR + i) + r8;
          if (src[i]) cp_async16(a_s + m * 128 + ((u ^ (m & 7)) << 4), src[i] + kb * TC_BK);
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
        pq |= s << (8 * np);
        ++np;
        if (np == TC_STAGES - 1) publish_oldest();
      }
    }
    // the stages still in flight, oldest first, then the sentinel stage
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    while (np > 0) {
      mbar_arrive(full0 + 8 * (pq & 0xffu));
      pq >>= 8;
      --np;
    }
    if (ok) {
      const uint32_t s = it % TC_STAGES;
      int good = 1;
      if (lane == 0)
        good = mbar_wait(empty0 + 8 * s, ((it / TC_STAGES) & 1) ^ 1, abort_flag, P.wait_cycles)
                   ? 1 : 0;
      good = __shfl_sync(0xffffffffu, good, 0);
      if (good) mbar_arrive(full0 + 8 * s);
      else ok = false;
    }
    if (!ok && lane == 0) {
      atomicExch(P.err, LX_ERR_TIMEOUT);
      *abort_flag = 1;
    }
  } else if (warp == 2) {
    // ------------------------------------------------------------ scheduler
    // Claims tiles from the launch's counter and decodes them (the plan-prefix
    // search and the bucket lookups: dependent global loads) into a queue of
    // TC_QN tiles ahead of the producer; a sentinel (BN < 0) ends the queue.
    const int total = P.tile_off[P.n_items];
    uint32_t qi = 0;
    bool ok = true;
    while (true) {
      int cur = lane == 0 ? atomicAdd(P.ctr, 1) : 0;
      cur = __shfl_sync(0xffffffffu, cur, 0);
      TcTile t;
      if (cur < total) tc_decode_warp<BM>(P, cur, t);
      else t.BN = -1;
      const uint32_t q = qi % TC_QN;
      int good = 1;
      if (lane == 0) {
        good = mbar_wait(qempty0 + 8 * q, ((qi / TC_QN) & 1) ^ 1, abort_flag, P.wait_cycles)
                   ? 1 : 0;
        if (good) {
          qslot[q] = t;
          mbar_arrive(qfull0 + 8 * q);
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
      uint32_t it = 0, tiles = 0;
      bool ok = true;
      // An injected unmet wait: the drain barrier gets no arrival before the
      // abort path, so this bounded wait runs out and the CTA takes that path.
      if (P.unmet_wait == LX_WAIT_TC_MMA && !mbar_wait(drain, 0, abort_flag, P.wait_cycles))
        ok = false;
      while (ok) {
        const uint32_t s = it % TC_STAGES;
        if (!mbar_wait(full0 + 8 * s, (it / TC_STAGES) & 1, abort_flag, P.wait_cycles)) {
          ok = false;
          break;
        }
        const TcTile t = slot[s];
        const uint32_t b = tiles % NBUF, u = tiles / NBUF;
        // this accumulator must have been drained by the epilogue (NBUF tiles ago)
        if (!mbar_wait(tempty0 + 8 * b, (u & 1) ^ 1, abort_flag, P.wait_cycles)) {
          ok = false;
          break;
        }
        eslot[b] = t;  // tile info for the epilogue, released by this arrival
        mbar_arrive(tfull0 + 8 * b);
        if (t.BN < 0) {  // sentinel: the second arrival completes the phase
          mbar_arrive(tfull0 + 8 * b);
          ++it;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + b * NH * TC_ACC_COLS;
        const uint32_t idesc = instr_desc(128, t.BN);
        const int nh = (NH == 2 && t.M > 128) ? 2 : 1;
        const int nkb = (t.K + TC_BK - 1) / TC_BK;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const uint32_t s2 = it % TC_STAGES;
          if (!mbar_wait(full0 + 8 * s2, (it / TC_STAGES) & 1, abort_flag, P.wait_cycles)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_s = smem_base + s2 * TC_STAGE_BYTES, b_s = a_s + TC_A_BYTES;
#pragma unroll
          for (int k = 0; k < TC_BK / 16; ++k)
            for (int h = 0; h < nh; ++h)  // the 128-row halves share the weight box
              tc_mma(d + h * TC_ACC_COLS, smem_desc(a_s + h * 128 * TC_BK * 2 + 32 * k),
                     smem_desc(b_s + 32 * k), idesc, (kb | k) != 0 ? 1u : 0u);
          tc_commit(empty0 + 8 * s2);  // frees the stage once these MMAs are done
        }
        if (!ok) break;
        tc_commit(tfull0 + 8 * b);  // accumulator ready
        ++tiles;
      }
      if (!ok) {
        atomicExch(P.err, LX_ERR_TIMEOUT);
        *abort_flag = 1;
        tc_commit(drain);  // arrives once every MMA issued so far has completed
        mbar_wait(drain, 0, nullptr);
      }
    }
    __syncwarp();
  } else if (warp >= 4 && warp < 4 + EPI) {
    // ------------------------------------------------------------ epilogue
    const int ew = warp & 3;        // TMEM lanes 32 ew .. 32 ew + 31
    const int eh = (warp - 4) >> 2; // with 8 warps: which column passes (alternate)
    constexpr int ESTEP = EPI / 4;  // passes are dealt out to ESTEP warps per quadrant
    float* stg = epi + (warp - 4) * (C::EPI_BYTES / 4);  // 1024-byte aligned
    uint32_t nstore = 0;  // TMA stores issued by this warp (lane 0), alternating buffers
    uint32_t tiles = 0;
    while (true) {
      const uint32_t b = tiles % NBUF, u = tiles / NBUF;
      if (!mbar_wait(tfull0 + 8 * b, u & 1, abort_flag, P.wait_cycles)) {
        if (lane == 0) {
          atomicExch(P.err, LX_ERR_TIMEOUT);
          *abort_flag = 1;
        }
        break;
      }
      tc_fence_after();
      const TcTile t = eslot[b];
      if (t.BN < 0) break;
      const long col0 = (long)t.grp * t.Ng + t.row0 + (P.node_col ? P.node_col[t.node] : 0);
      const bool tile_ok = t.tok0 >= 0 && col0 + t.BN <= P.ldo;
      const int cq = lane & 7;
      if constexpr (C::HALF) {
        // bf16, 32 columns per pass: one TMEM load, rows staged 64 bytes wide,
        // stored as 64-byte row segments (four lanes per row, eight rows a
        // pass).  The passes of both 128-row halves form one sequence, and the
        // next pass's TMEM load is issued before this pass's stores, so that
        // its latency is spent storing.
        const int nhh = t.M > 128 ? 2 : 1;
        const int pph = t.BN > 32 * eh ? (t.BN - 32 * eh + 32 * ESTEP - 1) / (32 * ESTEP) : 0;
        const int npass = nhh * pph;
        auto pass_taddr = [&](int p) {
          const int h = p / pph, c0 = 32 * eh + (p - h * pph) * 32 * ESTEP;
          return tmem + (b * NH + h) * TC_ACC_COLS + ((uint32_t)(32 * ew) << 16) + (uint32_t)c0;
        };
        uint32_t r0[32];
        if (npass > 0) tc_ld32_async(pass_taddr(0), r0);
        long orow_l = 0;
        int hcur = -1;
        for (int p = 0; p < npass; ++p) {
          const int h = p / pph, c0 = 32 * eh + (p - h * pph) * 32 * ESTEP;
          if (h != hcur) {
            // output rows of this warp's 32 tile rows (remapped when row_map is set)
            hcur = h;
            orow_l = (long)t.tok0 + 128 * h + 32 * ew + lane;
            if (P.row_map)
              orow_l = (32 * ew + lane + 128 * h < t.M && orow_l < P.rows_cap) ? P.row_map[orow_l] : -1;
          }
          tc_wait_ld();
          uint32_t pk[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            __nv_bfloat162 b0 = __floats2bfloat162_rn(__uint_as_float(r0[2 * e]),
                                                      __uint_as_float(r0[2 * e + 1]));
            pk[e] = *reinterpret_cast<uint32_t*>(&b0);
          }
          if (p + 1 < npass) tc_ld32_async(pass_taddr(p + 1), r0);
          // a whole 32-row block inside the tile's rows and the buffer, at a
          // 16-byte-aligned column: one TMA store from the staged block
          const long grow0 = (long)t.tok0 + 128 * h + 32 * ew;
          const int xcol = (int)(col0 + c0);
          if (P.omap && !P.row_map && tile_ok && 128 * h + 32 * ew + 32 <= t.M &&
              c0 + 32 <= t.BN && grow0 + 32 <= P.rows_cap && (xcol & 7) == 0) {
            uint8_t* tb = reinterpret_cast<uint8_t*>(stg) + (nstore & 1) * 2048;
            if (lane == 0) bulk_wait_read<1>();  // the store that used this buffer has read it
            __syncwarp();
            // row `lane`, 16-byte chunk q at q ^ ((row / 2) % 4): the 64-byte swizzle
            uint4* trow = reinterpret_cast<uint4*>(tb + lane * 64);
#pragma unroll
            for (int q = 0; q < 4; ++q)
              trow[q ^ ((lane >> 1) & 3)] = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            if (lane == 0) {
              tma_store_2d(P.omap, xcol, (int)grow0, smem_u32(tb));
              bulk_commit();
            }
            ++nstore;
            continue;
          }
          if (lane == 0) bulk_wait_read<0>();  // the staging is shared with the TMA stores
          __syncwarp();
          uint4* srow = reinterpret_cast<uint4*>(stg + lane * C::EPI_LD);
#pragma unroll
          for (int q = 0; q < 4; ++q)
            srow[q] = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
          __syncwarp();
          const int c4 = lane & 3;
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int rr = 8 * j + (lane >> 2);
            const int m = 128 * h + 32 * ew + rr;
            const long grow = __shfl_sync(0xffffffffu, orow_l, rr);
            if (tile_ok && m < t.M && grow >= 0 && grow < P.rows_cap) {
              const uint4 u4 = *reinterpret_cast<const uint4*>(stg + rr * C::EPI_LD + 4 * c4);
              *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(P.out) + (size_t)grow * P.ldo +
                                        col0 + c0 + 8 * c4) = u4;
            }
          }
          __syncwarp();
        }
      } else {
      for (int h = 0; h < NH && 128 * h < t.M; ++h) {
      const uint32_t acc = tmem + (b * NH + h) * TC_ACC_COLS;
      // output rows of this warp's 32 tile rows (remapped when row_map is set)
      long orow_l = (long)t.tok0 + 128 * h + 32 * ew + lane;
      if (P.row_map)
        orow_l = (32 * ew + lane + 128 * h < t.M && orow_l < P.rows_cap) ? P.row_map[orow_l] : -1;
      if (P.out_f32) {
        for (int c0 = 32 * eh; c0 < t.BN; c0 += 32 * ESTEP) {
          float v[32];
          tc_ld32(acc + ((uint32_t)(32 * ew) << 16) + (uint32_t)c0, v);
          // lane = accumulator row: stage the 32 x 32 block row-major
          float4* srow = reinterpret_cast<float4*>(stg + lane * TC_EPI_LD);
#pragma unroll
          for (int q = 0; q < 8; ++q)
            srow[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          __syncwarp();
          // eight lanes per row, four rows per pass: whole 128-byte segments
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int rr = 4 * j + (lane >> 3);
            const int m = 128 * h + 32 * ew + rr;
            const long grow = (long)t.tok0 + m;
            if (tile_ok && m < t.M && grow < P.rows_cap) {
              const float4 f = *reinterpret_cast<const float4*>(stg + rr * TC_EPI_LD + 4 * cq);
              *reinterpret_cast<float4*>(static_cast<float*>(P.out) + (size_t)grow * P.ldo +
                                         col0 + c0 + 4 * cq) = f;
            }
          }
          __syncwarp();
        }
      } else {
        // bf16: 64 columns per pass, converted before staging, so that a row
        // segment is again 128 bytes
        for (int c0 = 64 * eh; c0 < t.BN; c0 += 64 * ESTEP) {
          uint32_t pk[32];
          {
            // both 32-column loads of the pass in flight, one wait
            uint32_t r0[32], r1[32];
            tc_ld32_async(acc + ((uint32_t)(32 * ew) << 16) + (uint32_t)c0, r0);
            tc_ld32_async(acc + ((uint32_t)(32 * ew) << 16) + (uint32_t)(c0 + 32), r1);
            tc_wait_ld();
#pragma unroll
            for (int e = 0; e < 16; ++e) {
              __nv_bfloat162 b0 = __floats2bfloat162_rn(__uint_as_float(r0[2 * e]),
                                                        __uint_as_float(r0[2 * e + 1]));
              __nv_bfloat162 b1 = __floats2bfloat162_rn(__uint_as_float(r1[2 * e]),
                                                        __uint_as_float(r1[2 * e + 1]));
              pk[e] = *reinterpret_cast<uint32_t*>(&b0);
              pk[16 + e] = *reinterpret_cast<uint32_t*>(&b1);
            }
          }
          uint4* srow = reinterpret_cast<uint4*>(stg + lane * TC_EPI_LD);
#pragma unroll
          for (int q = 0; q < 8; ++q)
            srow[q] = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
          __syncwarp();
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int rr = 4 * j + (lane >> 3);
            const int m = 128 * h + 32 * ew + rr;
            const long grow = __shfl_sync(0xffffffffu, orow_l, rr);
            if (tile_ok && m < t.M && grow >= 0 && grow < P.rows_cap) {
              const uint4 u4 = *reinterpret_cast<const uint4*>(stg + rr * TC_EPI_LD + 4 * cq);
              *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(P.out) + (size_t)grow * P.ldo +
                                        col0 + c0 + 8 * cq) = u4;
            }
          }
          __syncwarp();
        }
      }
      }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(tempty0 + 8 * b);
      ++tiles;
    }
    // the TMA stores complete before the CTA exits
    if (lane == 0) bulk_wait_all();
    __syncwarp();
  }
  // all roles meet before the TMEM is released
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(TC_TMEM_COLS)
                 : "memory");
  } else if (warp == 0 && lane == 0 && *abort_flag) {
    // an aborted CTA may leave weight/activation copies in flight: wait (bounded)
    // for the last stages the producer issued before shared memory goes away
    const uint32_t first = prod_it > TC_STAGES ? prod_it - TC_STAGES : 0;
    for (uint32_t j = first; j < prod_it; ++j)
      mbar_wait(full0 + 8 * (j % TC_STAGES), (j / TC_STAGES) & 1, nullptr);
  }
}

}  // namespace

int tc_tile_tokens() { return 128; }
int tc_tile_cols() { return TC_BN; }
// The anchor gate/up product (anchor buckets of hundreds of rows) and, on
// flat layers, the anchor down tile with the members' corrections along K take
// 256-row tiles; the others 128 (measured at the Qwen3-shaped prefill of 8192:
// tc_up_anchor 156 -> 146 us and the down tile with the corrections 142 -> 128
// us with 256 rows; the tree layer's plain down tile is faster at 128 rows,
// 34 vs 39 us, and x V, whose member buckets are a few hundred rows, loses more
// to half-empty tiles and a single wave than it gains).
int tc_tile_rows(const lx_layer* L, int op) {
  return (op == OP_UP_ANCHOR || (op == OP_DN_ANCHOR && L->ct)) ? 256 : 128;
}

template <int BM, int EPI>
static int tc_smem_bytes_() {
  using C = TcCfg<BM, EPI>;
  return C::STAGES * C::STAGE_BYTES + EPI * C::EPI_BYTES + 8 * (2 * C::STAGES + 7) +
         (C::STAGES + 2 + TC_QN) * (int)sizeof(TcTile) + 16 * TC_QN + 1024;
}
template <int BM, int EPI>
static int tc_smem_bytes() { return tc_smem_bytes_<BM, EPI>(); }

template <int BM, int EPI, bool GATHER>
static lx_status launch_tc_cfg(lx_layer* L, const TcLaunch& P, cudaStream_t s, const char* name) {
  const int smem = tc_smem_bytes<BM, EPI>();
  static bool done[64] = {};
  LX_CUDA(smem_cap_once((const void*)k_tc_gemm<BM, EPI, GATHER>, smem, L->device, done));
  ProfScope ps(L, s, name);
  launch_k(L, k_tc_gemm<BM, EPI, GATHER>, L->num_sms,
           TcCfg<BM, EPI>::THREADS + (GATHER ? 32 * (TC_GATHER_WARPS - 1) : 0), smem, s, P);
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

lx_status launch_tc(lx_layer* L, const TcLaunch& P, cudaStream_t s, const char* name) {
  const bool g = P.gather != nullptr;
  if (g && P.kc_child) return fail(LX_ERR_STATE, "gathered A rows with a K concatenation");
  if (P.bm == 256) {
    // eight epilogue warps: the single accumulator of a 256-row tile is
    // drained while the tensor core waits, so the drain is split eight ways
    if (g || P.out_f32) return fail(LX_ERR_STATE, "256-row tiles take TMA rows and bf16 output");
    return launch_tc_cfg<256, 8, false>(L, P, s, name);
  }
  if (P.epi == 8) {
    if (g) return fail(LX_ERR_STATE, "gathered A rows need four epilogue warps");
    return launch_tc_cfg<128, 8, false>(L, P, s, name);
  }
  return g ? launch_tc_cfg<128, 4, true>(L, P, s, name) : launch_tc_cfg<128, 4, false>(L, P, s, name);
}

static TcLaunch tc_op(lx_layer* L, int op, const CUtensorMap* xmap, int xcol, void* out,
                      long ldo, bool out_f32, int counter) {
  Workspace& w = L->ws;
  TcLaunch P;
  P.shape = op_shape(L, op);
  P.bm = tc_tile_rows(L, op);
  // short-K products (the U factors, K = rank; the down side, K = d_ff): tiles
  // bound by writing their output take eight epilogue warps
  P.epi = (op == OP_UP_U || op == OP_DN_U || op == OP_DN_ANCHOR || op == OP_DN_V) ? 8 : 4;
  P.items = P.shape.on_anchors ? L->d_anchors : L->d_corrs;
  P.n_items = P.shape.on_anchors ? L->n_anchor : L->n_corr;
  P.tile_off = w.tile_off + (PLAN_TC + op) * (op_max_items(L) + 1);
  P.node_off = w.key_off;
  P.rank = L->d_rank;
  P.wmaps = L->d_tmaps + (size_t)op * L->N;
  P.xmap = xmap;
  P.xcol = xcol;
  P.out = out;
  P.ldo = ldo;
  P.out_f32 = out_f32 ? 1 : 0;
  P.ctr = w.sctr + N_STREAM_GROUPS + counter;
  P.err = w.err;
  P.wait_cycles = wait_limit(L);
  P.unmet_wait = L->unmet_wait;
  P.rows_cap = w.rows_cap;
  P.row_map = nullptr;
  P.node_col = nullptr;
  P.kc_child = nullptr;
  P.kc_wmaps = nullptr;
  P.kc_xmap = nullptr;
  P.kc_slot = 0;
  P.gather = nullptr;
  P.xsrc = nullptr;
  P.ldx = 0;
  P.omap = nullptr;
  return P;
}

namespace {

// xg[r] = x[node_tok[r]] for the anchor rows r < R of this forward (R = the
// node rows, key_off[N]; rows of correction nodes are skipped: their products
// gather their rows themselves): one warp per row, 16-byte loads and stores.
__global__ void __launch_bounds__(256)
k_gather_rows(const __nv_bfloat16* __restrict__ x, int H, const int* __restrict__ node_tok,
              const int* __restrict__ row_node, const int* __restrict__ rank,
              const int* __restrict__ rows_total, long rows_cap, __nv_bfloat16* __restrict__ xg) {
  pdl_wait();
  const long R = min((long)*rows_total, rows_cap);
  const int lane = threadIdx.x & 31;
  const long warps = (long)gridDim.x * (blockDim.x >> 5);
  const int vec = H / 8;
  constexpr int U = 8;  // 16-byte loads of a row in flight per lane before any store
  long r = (long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  int tok = r < R ? node_tok[r] : 0;
  bool anc = r < R && __ldg(rank + row_node[r]) == 0;
  for (; r < R; r += warps) {
    const uint4* src = reinterpret_cast<const uint4*>(x + (size_t)tok * H);
    uint4* dst = reinterpret_cast<uint4*>(xg + (size_t)r * H);
    const long rn = r + warps;
    const bool this_anc = anc;
    tok = rn < R ? node_tok[rn] : 0;  // the next row's token, looked up early
    anc = rn < R && __ldg(rank + row_node[rn]) == 0;
    if (!this_anc) continue;
    for (int i0 = lane; i0 < vec; i0 += 32 * U) {
      uint4 v[U];
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (i0 + 32 * u < vec) v[u] = __ldg(src + i0 + 32 * u);
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (i0 + 32 * u < vec) dst[i0 + 32 * u] = v[u];
    }
  }
}

}  // namespace

// The prefill forward: every (token, node) product on the tensor cores.
lx_status launch_tc_experts(lx_layer* L, const void* x, int T, int k, void* y, cudaStream_t s) {
  Workspace& w = L->ws;
  const long H = L->H, I = L->I, rmax = L->max_rank;
  const __nv_bfloat16* xb = static_cast<const __nv_bfloat16*>(x);
  auto run = [&](const TcLaunch& P, const char* name) -> lx_status {
    if (P.n_items == 0) return LX_OK;
    return launch_tc(L, P, s, name);
  };
  // the anchor rows in node-row order once, so that the anchor product's A
  // tiles are TMA boxes (its 256-row stages are too few to hide gathers); the
  // correction products read their rows straight from x (gathered by the
  // GEMM's gather warp)
  {
    ProfScope ps(L, s, "gather_rows");
    launch_k(L, k_gather_rows, L->num_sms * 8, 256, 0, s, xb, (int)H, w.node_tok, w.row_node,
             L->d_rank, w.key_off + L->N, w.rows_cap, w.xg);
    LX_CUDA(cudaGetLastError());
  }
  auto gathered = [&](TcLaunch P) {
    P.gather = w.node_tok;
    P.xsrc = xb;
    P.ldx = H;
    return P;
  };
  {
    TcLaunch ua = tc_op(L, OP_UP_ANCHOR, w.gmap, 0, w.hb, 2 * I, false, 0);
    ua.omap = w.omaps;  // hb (null when not encodable)
    LX_TRY(run(ua, "tc_up_anchor"));
  }
  if (L->ct) {
    // flat layers: the members' x V rows land aligned to their cluster's rows,
    // and one fused kernel adds the corrections and applies the SwiGLU
    // (the per-cluster-row gate / child-row tables come from the bucketing)
    TcLaunch pv = gathered(tc_op(L, OP_UP_V, w.gmap, 0, w.Pal, (long)L->ct_nch * 2 * rmax, false, 1));
    pv.row_map = w.rho2al;
    pv.node_col = L->d_child_col;
    LX_TRY(run(pv, "tc_up_V"));
    LX_TRY(launch_ct_swiglu(L, s));
    // the members' down corrections join their anchor's down tile along K:
    // [z | Q_1 | Q_2 | ...] . [Wd | Ud_1 | Ud_2 | ...]^T, Q stored aligned to
    // the cluster's rows (zero where a member is not selected)
    TcLaunch qv = tc_op(L, OP_DN_V, w.xmaps + 1, 0, w.Qal, (long)L->ct_nch * rmax, false, 4);
    qv.row_map = w.rho2al;
    qv.node_col = L->d_child_qcol;
    LX_TRY(run(qv, "tc_dn_V"));
    TcLaunch dn = tc_op(L, OP_DN_ANCHOR, w.xmaps + 1, 0, w.yb, H, false, 3);
    dn.kc_child = L->d_child;
    dn.kc_wmaps = L->d_tmaps + (size_t)OP_DN_U * L->N;
    dn.kc_xmap = w.pamap + 2;
    dn.kc_slot = (int)rmax;
    dn.omap = w.omaps ? w.omaps + 1 : nullptr;  // yb
    LX_TRY(run(dn, "tc_dn_anchor_U"));
    return launch_combine(L, T, k, y, true, s, SplitParts(), /*anchors_only=*/true);
  } else {
    LX_TRY(run(gathered(tc_op(L, OP_UP_V, w.gmap, 0, w.Pb, 2 * rmax, false, 1)),
               "tc_up_V"));
    LX_TRY(run(tc_op(L, OP_UP_U, w.xmaps + 0, 0, w.hb, 2 * I, false, 2),
               "tc_up_U"));
    LX_TRY(launch_swiglu(L, T, k, true, s));
  }
  LX_TRY(run(tc_op(L, OP_DN_ANCHOR, w.xmaps + 1, 0, w.yb, H, false, 3),
             "tc_dn_anchor"));
  LX_TRY(run(tc_op(L, OP_DN_V, w.xmaps + 1, 0, w.Qb, rmax, false, 4),
             "tc_dn_V"));
  LX_TRY(run(tc_op(L, OP_DN_U, w.xmaps + 2, 0, w.yb, H, false, 5),
             "tc_dn_U"));
  LX_TRY(launch_combine(L, T, k, y, true, s));
  return LX_OK;
}

}  // namespace lx
