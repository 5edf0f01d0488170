// Neuron alignment of a member to its dominant (Sec. 3.2 Stage 3 (i)).
//
// Neuron i of an expert is the vector a_i = (gate[i, :], up[i, :], down[:, i])
// of length 3H (the x W^T storage: gate/up [I][H], down [H][I]).  The matching
// cost is C[i][j] = ||a_i||^2 + ||b_j||^2 - 2 a_i . b_j (Eq. cost), the optimal
// matching minimises sum_i C[i][P(i)] (Eq. assign), and the aligned member takes
// the member's neuron P(i) as its neuron i.
//
// k_align_cost: one 64 x 64 tile of C per CTA, fp32 multiply-adds over the
// three K segments (gate rows, up rows: K-major; down columns: MN-major) staged
// through shared memory in 32-deep chunks; the tile's row norms are summed
// from the same staged chunks, so every operand byte is read once per tile.
// Tensor-core form (bf16 experts, d_model a multiple of 256): both experts'
// neuron vectors are packed K-major, cat[i] = (gate[i, :], up[i, :], down[:, i])
// (the down columns transposed through shared memory, the gate/up rows
// copies; k_align_pack, which also takes ||cat[i]||^2), one tcgen05 split-K GEMM forms the
// dot products (bf16 operands, fp32 accumulation; 256-column chunks of the
// member's neurons in one launch), and k_align_finish adds the K ranges in
// order and forms C.  k_align_cost_mma: the 64 x 64 tile form (mma.sync) for
// the other bf16 shapes.
// k_permute_rows / k_permute_cols: gathers (bit-exact copies).
// lx_lap_solve / lx_lap_solve_batch: the exact assignment on the host (Jonker
// and Volgenant: column reduction, augmenting row reduction, then shortest
// augmenting paths with dual potentials); the batch form spreads independent
// problems over host threads.
#include <algorithm>
#include <cstring>
#include <atomic>
#include <limits>
#include <thread>
#include <vector>

#include "lx_internal.cuh"

namespace lx {
namespace {

constexpr int AC_TILE = 64;     // rows (dominant neurons) and columns (member neurons) per CTA
constexpr int AC_KC = 32;       // K chunk
constexpr int AC_LD = AC_TILE + 4;
constexpr int AC_THREADS = 256;

// 8 consecutive elements starting at p (16-byte aligned for bf16, 32 for fp32)
__device__ __forceinline__ void load8(const __nv_bfloat16* p, float (&v)[8]) {
  const uint4 q = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&q);
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float2 f = __bfloat1622float2(h[e]);
    v[2 * e] = f.x;
    v[2 * e + 1] = f.y;
  }
}
__device__ __forceinline__ void load8(const float* p, float (&v)[8]) {
  const float4 a = *reinterpret_cast<const float4*>(p);
  const float4 b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

// Stages the chunk (segment seg, K offset h0, length kc <= 32) of the neuron
// vectors of rows r0 .. r0+63 into S[k][row] (zero beyond I or kc).
//   seg 0 / 1: rows of gate / up [I][H]  (element (i, h) at i*H + h)
//   seg 2:     columns of down [H][I]    (element (i, h) at h*I + i)
template <typename TW>
__device__ __forceinline__ void stage_chunk(float (*S)[AC_LD], const TW* g, const TW* u,
                                            const TW* d, int seg, int h0, int kc, int r0,
                                            int H, int I, int tid) {
  float v[8];
  if (seg < 2) {
    const TW* W = seg == 0 ? g : u;
    const int row = tid >> 2, hq = (tid & 3) * 8;  // 64 rows x 4 groups of 8
    const bool ok = r0 + row < I && hq < kc;
    if (ok) load8(W + (size_t)(r0 + row) * H + h0 + hq, v);
#pragma unroll
    for (int e = 0; e < 8; ++e) S[hq + e][row] = ok ? v[e] : 0.f;
  } else {
    const int hr = tid >> 3, iq = (tid & 7) * 8;  // 32 K rows x 8 groups of 8 neurons
    const bool ok = hr < kc && r0 + iq < I;
    if (ok) load8(d + (size_t)(h0 + hr) * I + r0 + iq, v);
#pragma unroll
    for (int e = 0; e < 8; ++e) S[hr][iq + e] = ok ? v[e] : 0.f;
  }
}

template <typename TW>
__global__ void __launch_bounds__(AC_THREADS)
k_align_cost(const TW* __restrict__ dg, const TW* __restrict__ du, const TW* __restrict__ dd,
             const TW* __restrict__ mg, const TW* __restrict__ mu, const TW* __restrict__ md,
             int H, int I, float* __restrict__ cost) {
  __shared__ __align__(16) float As[AC_KC][AC_LD];
  __shared__ __align__(16) float Bs[AC_KC][AC_LD];
  __shared__ float na[AC_TILE], nb[AC_TILE];
  const int tid = threadIdx.x;
  const int i0 = blockIdx.y * AC_TILE, j0 = blockIdx.x * AC_TILE;
  const int ty = tid >> 4, tx = tid & 15;
  float acc[4][4] = {};
  float nrm = 0.f;  // threads 0..63: |a_{i0+tid}|^2, 64..127: |b_{j0+tid-64}|^2
  for (int seg = 0; seg < 3; ++seg) {
    for (int h0 = 0; h0 < H; h0 += AC_KC) {
      const int kc = min(AC_KC, H - h0);
      stage_chunk(As, dg, du, dd, seg, h0, kc, i0, H, I, tid);
      stage_chunk(Bs, mg, mu, md, seg, h0, kc, j0, H, I, tid);
      __syncthreads();
      if (tid < 2 * AC_TILE) {
        float (*S)[AC_LD] = tid < AC_TILE ? As : Bs;
        const int c = tid & (AC_TILE - 1);
#pragma unroll 8
        for (int k = 0; k < AC_KC; ++k) nrm = fmaf(S[k][c], S[k][c], nrm);
      }
#pragma unroll 8
      for (int k = 0; k < AC_KC; ++k) {
        const float4 a = *reinterpret_cast<const float4*>(&As[k][ty * 4]);
        const float4 b = *reinterpret_cast<const float4*>(&Bs[k][tx * 4]);
        const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
        for (int r = 0; r < 4; ++r)
#pragma unroll
          for (int c = 0; c < 4; ++c) acc[r][c] = fmaf(av[r], bv[c], acc[r][c]);
      }
      __syncthreads();
    }
  }
  if (tid < AC_TILE) na[tid] = nrm;
  else if (tid < 2 * AC_TILE) nb[tid - AC_TILE] = nrm;
  __syncthreads();
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int i = i0 + ty * 4 + r;
    if (i >= I) continue;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int j = j0 + tx * 4 + c;
      if (j < I) cost[(size_t)i * I + j] = na[ty * 4 + r] + nb[tx * 4 + c] - 2.f * acc[r][c];
    }
  }
}

// Tensor-core form of the cost for bf16 experts: the same tile of C, with the
// products a_i . b_j on mma.sync m16n8k16 (bf16 inputs, fp32 accumulation:
// every product is exact, as on the CUDA-core path).  Per 64-deep K chunk the
// 64 dominant rows (A) and 64 member rows (B) are staged K-major in shared
// memory as 128-byte rows with the 128-byte XOR swizzle (unit u of row r at
// unit u ^ (r & 7)); gate/up chunks are copied as 16-byte units, down chunks
// (columns of [H][I]) are transposed in registers from 8 x 8 blocks.  Lane
// (g, q) feeds the MMA its own 16-byte K unit 2q + c of both operands, a K
// permutation shared by A and B (the sum over K is unchanged).  The next
// chunk's global loads are issued before the current chunk's MMAs (register
// double buffering).  Row norms are summed from the staged chunks.
constexpr int AM_TILE = 64;
constexpr int AM_THREADS = 256;
constexpr int AM_ROWB = 128;  // bytes per staged row (64 bf16)

__device__ __forceinline__ void am_mma(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                       uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// this thread's part of chunk (seg, h0, kc) of A (rows i0..) and B (rows j0..)
struct AmRegs {
  uint4 v[8];
};

__device__ __forceinline__ void am_load(AmRegs& R, const __nv_bfloat16* dg, const __nv_bfloat16* du,
                                        const __nv_bfloat16* dd, const __nv_bfloat16* mg,
                                        const __nv_bfloat16* mu, const __nv_bfloat16* md, int seg,
                                        int h0, int kc, int i0, int j0, int H, int I, int tid) {
  const uint4 z = make_uint4(0u, 0u, 0u, 0u);
  if (seg < 2) {
    // 2 units of A and 2 of B per thread: index q = tid + 256 v, row q / 8, unit q % 8
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      const int qi = tid + AM_THREADS * (v & 1);
      const int row = qi >> 3, u = qi & 7;
      const bool isA = v < 2;
      const int r0 = isA ? i0 : j0;
      const __nv_bfloat16* W = isA ? (seg == 0 ? dg : du) : (seg == 0 ? mg : mu);
      const bool ok = r0 + row < I && u * 8 < kc;
      R.v[v] = ok ? *reinterpret_cast<const uint4*>(W + (size_t)(r0 + row) * H + h0 + u * 8) : z;
    }
  } else if (tid < 2 * AM_TILE) {
    // one 8 x 8 block (8 K rows x 8 neurons) of the down matrix [H][I]
    const bool isA = tid < AM_TILE;
    const int b = tid & (AM_TILE - 1), hb = b >> 3, ib = b & 7;
    const __nv_bfloat16* W = isA ? dd : md;
    const int n0 = (isA ? i0 : j0) + ib * 8;
#pragma unroll
    for (int rr = 0; rr < 8; ++rr) {
      const bool ok = hb * 8 + rr < kc && n0 < I;
      R.v[rr] = ok ? *reinterpret_cast<const uint4*>(W + (size_t)(h0 + hb * 8 + rr) * I + n0) : z;
    }
  }
}

__device__ __forceinline__ void am_store(const AmRegs& R, unsigned char* As, unsigned char* Bs,
                                         int seg, int tid) {
  if (seg < 2) {
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      const int qi = tid + AM_THREADS * (v & 1);
      const int row = qi >> 3, u = qi & 7;
      unsigned char* S = v < 2 ? As : Bs;
      *reinterpret_cast<uint4*>(S + row * AM_ROWB + ((u ^ (row & 7)) << 4)) = R.v[v];
    }
  } else if (tid < 2 * AM_TILE) {
    const bool isA = tid < AM_TILE;
    const int b = tid & (AM_TILE - 1), hb = b >> 3, ib = b & 7;
    unsigned char* S = isA ? As : Bs;
    const uint32_t* w = reinterpret_cast<const uint32_t*>(R.v);  // w[rr * 4 + word]
#pragma unroll
    for (int ii = 0; ii < 8; ++ii) {
      // neuron ii: element ii of K rows rr = 0..7, packed two K values per word
      const uint32_t sel = (ii & 1) ? 0x7632u : 0x5410u;
      const int wd = ii >> 1;
      uint4 o;
      o.x = __byte_perm(w[0 * 4 + wd], w[1 * 4 + wd], sel);
      o.y = __byte_perm(w[2 * 4 + wd], w[3 * 4 + wd], sel);
      o.z = __byte_perm(w[4 * 4 + wd], w[5 * 4 + wd], sel);
      o.w = __byte_perm(w[6 * 4 + wd], w[7 * 4 + wd], sel);
      const int row = ib * 8 + ii;
      *reinterpret_cast<uint4*>(S + row * AM_ROWB + ((hb ^ (row & 7)) << 4)) = o;
    }
  }
}

__global__ void __launch_bounds__(AM_THREADS)
k_align_cost_mma(const __nv_bfloat16* __restrict__ dg, const __nv_bfloat16* __restrict__ du,
                 const __nv_bfloat16* __restrict__ dd, const __nv_bfloat16* __restrict__ mg,
                 const __nv_bfloat16* __restrict__ mu, const __nv_bfloat16* __restrict__ md,
                 int H, int I, float* __restrict__ cost) {
  __shared__ __align__(128) unsigned char sA[2][AM_TILE * AM_ROWB];
  __shared__ __align__(128) unsigned char sB[2][AM_TILE * AM_ROWB];
  __shared__ float s_norm[2][2 * AM_TILE];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int g = lane >> 2, q = lane & 3;
  const int wm = warp & 3, wn = warp >> 2;  // 16 rows x 32 columns per warp
  const int i0 = blockIdx.y * AM_TILE, j0 = blockIdx.x * AM_TILE;
  const int nch = (H + 63) / 64, total = 3 * nch;
  float acc[4][4] = {};
  float nrm = 0.f;  // row (tid & 127) of A (< 64) or B, units 4 (tid >> 7) .. +3
  AmRegs R;
  am_load(R, dg, du, dd, mg, mu, md, 0, 0, min(64, H), i0, j0, H, I, tid);
  am_store(R, sA[0], sB[0], 0, tid);
  __syncthreads();
  for (int t = 0; t < total; ++t) {
    const int buf = t & 1;
    if (t + 1 < total) {
      const int seg = (t + 1) / nch, h0 = ((t + 1) % nch) * 64;
      am_load(R, dg, du, dd, mg, mu, md, seg, h0, min(64, H - h0), i0, j0, H, I, tid);
    }
    const unsigned char* A = sA[buf];
    const unsigned char* B = sB[buf];
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      const int unit = (((q << 1) | c) ^ g) << 4;
      const int ra = 16 * wm + g;
      const uint4 w0 = *reinterpret_cast<const uint4*>(A + ra * AM_ROWB + unit);
      const uint4 w1 = *reinterpret_cast<const uint4*>(A + (ra + 8) * AM_ROWB + unit);
#pragma unroll
      for (int nj = 0; nj < 4; ++nj) {
        const uint4 xv = *reinterpret_cast<const uint4*>(B + (32 * wn + 8 * nj + g) * AM_ROWB + unit);
        am_mma(acc[nj], w0.x, w1.x, w0.y, w1.y, xv.x, xv.y);
        am_mma(acc[nj], w0.z, w1.z, w0.w, w1.w, xv.z, xv.w);
      }
    }
    {
      const int r = tid & 127, half = tid >> 7;
      const unsigned char* S = r < AM_TILE ? A : B;
      const int row = r & (AM_TILE - 1);
#pragma unroll
      for (int uu = 0; uu < 4; ++uu) {
        const int u = half * 4 + uu;
        const uint4 v = *reinterpret_cast<const uint4*>(S + row * AM_ROWB + ((u ^ (row & 7)) << 4));
        const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = __bfloat1622float2(h2[e]);
          nrm = fmaf(f.x, f.x, nrm);
          nrm = fmaf(f.y, f.y, nrm);
        }
      }
    }
    if (t + 1 < total) am_store(R, sA[buf ^ 1], sB[buf ^ 1], (t + 1) / nch, tid);
    __syncthreads();
  }
  s_norm[tid >> 7][tid & 127] = nrm;
  __syncthreads();
#pragma unroll
  for (int nj = 0; nj < 4; ++nj)
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int rl = 16 * wm + g + (c >= 2 ? 8 : 0);
      const int cl = 32 * wn + 8 * nj + 2 * q + (c & 1);
      const int i = i0 + rl, j = j0 + cl;
      if (i < I && j < I) {
        const float na = s_norm[0][rl] + s_norm[1][rl];
        const float nb = s_norm[0][AM_TILE + cl] + s_norm[1][AM_TILE + cl];
        cost[(size_t)i * I + j] = na + nb - 2.f * acc[nj][c];
      }
    }
}

// Packs one expert (blockIdx.z: 0 dominant, 1 member) for the tensor-core
// cost: cat[i] = (gate[i, :], up[i, :], down[:, i]) as K-major bf16 rows of
// 3H, and the squared norms of the pieces.  A CTA owns 32 neurons (warp w
// rows 4 w .. 4 w + 3) and one 256-wide range hb of d_model: the gate and up
// pieces are copied in 16-byte units, the down columns pass through shared
// memory in 64 (h) x 32 (i) blocks; each lane sums its squares in a fixed
// order (gate, up, then the down blocks), the 32 lane partials of a row are
// added by a shuffle tree into npart[hb][i] (the ranges are added in order
// by k_align_finish).  H is a multiple of 256.
constexpr int AP_HB = 256;
struct AlignPackArgs {
  const __nv_bfloat16* g[2];
  const __nv_bfloat16* u[2];
  const __nv_bfloat16* d[2];
  __nv_bfloat16* cat[2];
  float* npart[2];  // [H / AP_HB][I]
};
__global__ void __launch_bounds__(256) k_align_pack(const AlignPackArgs A, int H, int I) {
  __shared__ __align__(16) __nv_bfloat16 blk[64][34];
  const int x = blockIdx.z, i0 = blockIdx.x * 32, hb = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long K = 3L * H;
  const __nv_bfloat16* g = A.g[x];
  const __nv_bfloat16* u = A.u[x];
  const __nv_bfloat16* d = A.d[x];
  __nv_bfloat16* cat = A.cat[x];
  float part[4] = {0.f, 0.f, 0.f, 0.f};
  auto sq8 = [](const uint4& v, float acc) {
    const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 f = __bfloat1622float2(h2[e]);
      acc = fmaf(f.x, f.x, acc);
      acc = fmaf(f.y, f.y, acc);
    }
    return acc;
  };
  const int nq = H / 8, q = hb * (AP_HB / 8) + lane;  // this lane's 16-byte unit
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    const int i = i0 + 4 * warp + r;
    if (i >= I) continue;
    const uint4 a = reinterpret_cast<const uint4*>(g + (size_t)i * H)[q];
    const uint4 b = reinterpret_cast<const uint4*>(u + (size_t)i * H)[q];
    uint4* dst = reinterpret_cast<uint4*>(cat + (size_t)i * K);
    dst[q] = a;
    dst[nq + q] = b;
    part[r] = sq8(b, sq8(a, part[r]));
  }
  for (int h0 = hb * AP_HB; h0 < (hb + 1) * AP_HB; h0 += 64) {
    __syncthreads();
    // the 64 x 32 block d[h0 .. h0 + 63][i0 .. i0 + 31] in 4-byte pieces
    for (int e = threadIdx.x; e < 64 * 16; e += 256) {
      const int hh = e >> 4, ii = 2 * (e & 15);
      uint32_t v = 0u;
      if (i0 + ii < I) v = *reinterpret_cast<const uint32_t*>(d + (size_t)(h0 + hh) * I + i0 + ii);
      *reinterpret_cast<uint32_t*>(&blk[hh][ii]) = v;
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int il = 4 * warp + r, i = i0 + il;
      if (i >= I) continue;
      // lane l: elements h0 + 2 l, h0 + 2 l + 1 of row i's down segment
      __nv_bfloat162 pr;
      pr.x = blk[2 * lane][il];
      pr.y = blk[2 * lane + 1][il];
      *reinterpret_cast<__nv_bfloat162*>(cat + (size_t)i * K + 2L * H + h0 + 2 * lane) = pr;
      const float fa = __bfloat162float(pr.x), fb = __bfloat162float(pr.y);
      part[r] = fmaf(fb, fb, fmaf(fa, fa, part[r]));
    }
  }
#pragma unroll
  for (int r = 0; r < 4; ++r) {
    float v = part[r];
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const int i = i0 + 4 * warp + r;
    if (lane == 0 && i < I) A.npart[x][(size_t)hb * I + i] = v;
  }
}

// cost[i][j] = na[i] + nb[j] - 2 sum_s part[z][s][i][j - z Npad], z = j / Npad
// (the K ranges in ascending order), na / nb the sums of the nhb norm
// partials [nhb][I] in range order
__global__ void k_align_finish(const float* __restrict__ part, int splits, int I, int Npad,
                               const float* __restrict__ npa, const float* __restrict__ npb,
                               int nhb, float* __restrict__ cost) {
  // four consecutive columns per thread (I and Npad are multiples of 4)
  const long total = (long)I * I / 4;
  for (long e = (long)blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += (long)gridDim.x * blockDim.x) {
    const int i = (int)(4 * e / I), j = (int)(4 * e % I), z = j / Npad, jj = j % Npad;
    const float4* p = reinterpret_cast<const float4*>(part + ((size_t)z * splits * I + i) * Npad + jj);
    const size_t st = (size_t)I * Npad / 4;
    float4 dot = make_float4(0.f, 0.f, 0.f, 0.f);
    int sp = 0;
    for (; sp + 4 <= splits; sp += 4) {  // four ranges' loads in flight, added in order
      float4 v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) v[u] = p[(sp + u) * st];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        dot.x += v[u].x; dot.y += v[u].y; dot.z += v[u].z; dot.w += v[u].w;
      }
    }
    for (; sp < splits; ++sp) {
      const float4 v = p[sp * st];
      dot.x += v.x; dot.y += v.y; dot.z += v.z; dot.w += v.w;
    }
    float a = 0.f;
    float4 b = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int r = 0; r < nhb; ++r) {
      a += npa[(size_t)r * I + i];
      const float4 v = *reinterpret_cast<const float4*>(npb + (size_t)r * I + j);
      b.x += v.x; b.y += v.y; b.z += v.z; b.w += v.w;
    }
    *reinterpret_cast<float4*>(cost + (size_t)i * I + j) =
        make_float4(a + b.x - 2.f * dot.x, a + b.y - 2.f * dot.y, a + b.z - 2.f * dot.z,
                    a + b.w - 2.f * dot.w);
  }
}

// dst row i = src row perm[i] of a [rows][cols] matrix (16-byte pieces; a row
// whose perm entry is outside [0, rows) is written as zeros)
__global__ void k_permute_rows(const uint4* __restrict__ src, uint4* __restrict__ dst,
                               const int* __restrict__ perm, int rows, int pieces) {
  const int i = blockIdx.x;
  const int p = perm[i];
  const bool ok = p >= 0 && p < rows;
  for (int q = threadIdx.x; q < pieces; q += blockDim.x)
    dst[(size_t)i * pieces + q] = ok ? src[(size_t)p * pieces + q] : make_uint4(0u, 0u, 0u, 0u);
}

// dst[h][i] = src[h][perm[i]] of a [H][cols] matrix of esz-byte elements
template <typename TE>
__global__ void k_permute_cols(const TE* __restrict__ src, TE* __restrict__ dst,
                               const int* __restrict__ perm, int rows, int cols) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= cols) return;
  const int p = perm[i];
  const bool ok = p >= 0 && p < cols;
  for (int h = blockIdx.y; h < rows; h += gridDim.y)
    dst[(size_t)h * cols + i] = ok ? src[(size_t)h * cols + p] : TE(0);
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

lx_status check_expert_args(int32_t dtype, int32_t H, int32_t I) {
  if (dtype != LX_F32 && dtype != LX_BF16) return fail(LX_ERR_ARG, "unknown dtype");
  if (H < 8 || I < 8 || H % 8 || I % 8 || H > 65536 || I > 65536)
    return fail(LX_ERR_SHAPE, "d_model and d_ff must be multiples of 8 in 8..65536");
  return LX_OK;
}

}  // namespace
}  // namespace lx

namespace lx {
namespace {

// The tensor-core form of the cost (bf16, H % 256 == 0): scratch from the
// stream-ordered allocator (packed operands, norms, split-K partials), freed on
// the stream after the last kernel.
lx_status align_cost_tc(int H, int I, const void* dg, const void* du, const void* dd,
                        const void* mg, const void* mu, const void* md, float* cost,
                        cudaStream_t s) {
  using B = __nv_bfloat16;
  int dev = 0, sms = 0;
  LX_CUDA(cudaGetDevice(&dev));
  LX_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  const long K = 3L * H;
  const int nz = (I + 255) / 256;
  const int Npad = ((I + nz - 1) / nz + 15) / 16 * 16;  // chunk width (<= 256)
  auto al = [](size_t v) { return (v + 255) / 256 * 256; };
  const int nhb = H / AP_HB;
  const size_t b_cat = al((size_t)I * K * 2), b_nrm = al((size_t)nhb * I * 4);
  const size_t b_part = al((size_t)nz * RES_TC_MAX_SPLITS * I * Npad * 4);
  char* ws = nullptr;
  LX_CUDA(cudaMallocAsync((void**)&ws, 2 * b_cat + 2 * b_nrm + b_part, s));
  B* A = reinterpret_cast<B*>(ws);
  B* Bm = reinterpret_cast<B*>(ws + b_cat);
  float* na = reinterpret_cast<float*>(ws + 2 * b_cat);
  float* nb = reinterpret_cast<float*>(ws + 2 * b_cat + b_nrm);
  float* part = reinterpret_cast<float*>(ws + 2 * b_cat + 2 * b_nrm);
  lx_status st = LX_OK;
  AlignPackArgs pa;
  pa.g[0] = static_cast<const B*>(dg);
  pa.u[0] = static_cast<const B*>(du);
  pa.d[0] = static_cast<const B*>(dd);
  pa.g[1] = static_cast<const B*>(mg);
  pa.u[1] = static_cast<const B*>(mu);
  pa.d[1] = static_cast<const B*>(md);
  pa.cat[0] = A;
  pa.cat[1] = Bm;
  pa.npart[0] = na;
  pa.npart[1] = nb;
  k_align_pack<<<dim3((I + 31) / 32, nhb, 2), 256, 0, s>>>(pa, H, I);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) st = cuda_fail(e, "pack alignment operands");
  CUtensorMap ma, mb;
  std::memset(&ma, 0, sizeof(ma));
  std::memset(&mb, 0, sizeof(mb));
  if (st == LX_OK && (!encode_bf16_2d(&ma, A, K, I, 64, 128) || !encode_bf16_2d(&mb, Bm, K, I, 64, Npad)))
    st = fail(LX_ERR_CUDA, "cuTensorMapEncodeTiled(alignment operands) failed");
  int splits = 1;
  if (st == LX_OK)
    st = tc_splitk_gemm_chunks(ma, mb, I, Npad, nz, (int)K, part, RES_TC_MAX_SPLITS, &splits, sms,
                               dev, s);
  if (st == LX_OK) {
    const long total = (long)I * I;
    k_align_finish<<<(unsigned)std::min<long>((total / 4 + 255) / 256, 8L * sms), 256, 0, s>>>(
        part, splits, I, Npad, na, nb, nhb, cost);
    e = cudaGetLastError();
    if (e != cudaSuccess) st = cuda_fail(e, "alignment cost");
  }
  e = cudaFreeAsync(ws, s);
  if (st == LX_OK && e != cudaSuccess) st = cuda_fail(e, "free alignment scratch");
  return st;
}

}  // namespace
}  // namespace lx

extern "C" lx_status lx_align_cost(int32_t dtype, int32_t d_model, int32_t d_ff,
                                   const void* dom_gate, const void* dom_up, const void* dom_down,
                                   const void* mem_gate, const void* mem_up, const void* mem_down,
                                   float* cost, void* stream) {
  using namespace lx;
  LX_TRY(check_expert_args(dtype, d_model, d_ff));
  const void* ptrs[7] = {dom_gate, dom_up, dom_down, mem_gate, mem_up, mem_down, cost};
  for (const void* p : ptrs) {
    if (!p) return fail(LX_ERR_ARG, "NULL weight or cost pointer");
    if (!aligned16(p)) return fail(LX_ERR_ARG, "weights and cost must be 16-byte aligned");
  }
  const int H = d_model, I = d_ff;
  const dim3 grid((I + AC_TILE - 1) / AC_TILE, (I + AC_TILE - 1) / AC_TILE);
  cudaStream_t s = (cudaStream_t)stream;
  if (dtype == LX_BF16 && H % 256 == 0) return align_cost_tc(H, I, dom_gate, dom_up, dom_down,
                                                            mem_gate, mem_up, mem_down, cost, s);
  if (dtype == LX_BF16) {
    using B = __nv_bfloat16;
    k_align_cost_mma<<<grid, AM_THREADS, 0, s>>>((const B*)dom_gate, (const B*)dom_up,
                                                 (const B*)dom_down, (const B*)mem_gate,
                                                 (const B*)mem_up, (const B*)mem_down, H, I, cost);
  } else {
    k_align_cost<float><<<grid, AC_THREADS, 0, s>>>(
        (const float*)dom_gate, (const float*)dom_up, (const float*)dom_down,
        (const float*)mem_gate, (const float*)mem_up, (const float*)mem_down, H, I, cost);
  }
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

extern "C" lx_status lx_permute_neurons(int32_t dtype, int32_t d_model, int32_t d_ff,
                                        const int32_t* perm, const void* gate, const void* up,
                                        const void* down, void* gate_out, void* up_out,
                                        void* down_out, void* stream) {
  using namespace lx;
  LX_TRY(check_expert_args(dtype, d_model, d_ff));
  const void* ptrs[7] = {perm, gate, up, down, gate_out, up_out, down_out};
  for (const void* p : ptrs)
    if (!p) return fail(LX_ERR_ARG, "NULL pointer");
  for (int q = 1; q < 7; ++q)
    if (!aligned16(ptrs[q])) return fail(LX_ERR_ARG, "weights must be 16-byte aligned");
  const int H = d_model, I = d_ff;
  const size_t esz = dtype == LX_BF16 ? 2 : 4;
  const size_t row_bytes = (size_t)H * esz, mat = (size_t)I * H * esz;
  // the outputs may overlap no input (a gather cannot run in place)
  const char* ins[3] = {(const char*)gate, (const char*)up, (const char*)down};
  const char* outs[3] = {(const char*)gate_out, (const char*)up_out, (const char*)down_out};
  for (const char* o : outs)
    for (const char* in : ins)
      if (o < in + mat && in < o + mat) return fail(LX_ERR_ARG, "outputs overlap the inputs");
  cudaStream_t s = (cudaStream_t)stream;
  const int pieces = (int)(row_bytes / 16);
  k_permute_rows<<<I, 128, 0, s>>>((const uint4*)gate, (uint4*)gate_out, perm, I, pieces);
  k_permute_rows<<<I, 128, 0, s>>>((const uint4*)up, (uint4*)up_out, perm, I, pieces);
  const dim3 cg((I + 255) / 256, std::min(H, 4096));
  if (dtype == LX_BF16)
    k_permute_cols<unsigned short><<<cg, 256, 0, s>>>((const unsigned short*)down,
                                                      (unsigned short*)down_out, perm, H, I);
  else
    k_permute_cols<unsigned int><<<cg, 256, 0, s>>>((const unsigned int*)down,
                                                    (unsigned int*)down_out, perm, H, I);
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

// Exact linear assignment on the host: Jonker and Volgenant's column reduction
// assigns every column's cheapest row where that row is free, their augmenting
// row reduction assigns most of the rest; each remaining row is then added by
// a shortest augmenting path (Dijkstra over the columns
// on reduced costs c[i][j] - u[i] - v[j] >= 0), after which the dual
// potentials u, v are updated so that every reduced cost stays non-negative
// and those on the matching are zero -- JV's augmentation.  O(n^3), float64.
namespace {
bool costs_finite(const float* cost, long count) {
  for (long q = 0; q < count; ++q)
    if (!(cost[q] == cost[q]) || cost[q] == std::numeric_limits<float>::infinity() ||
        cost[q] == -std::numeric_limits<float>::infinity())
      return false;
  return true;
}

// The solver proper (arguments already checked); thread-safe.
void lap_solve_one(const float* cost, int32_t n, int32_t* assign, double* total) {
  const double kInf = std::numeric_limits<double>::infinity();
  // column 0 is a virtual column that holds the row being added
  std::vector<double> u(n + 1, 0.0), v(n + 1, 0.0), dist(n + 1);
  std::vector<int> row_of(n + 1, 0), prev(n + 1, 0);  // row_of[j]: row (1-based) on column j
  std::vector<char> done(n + 1), row_used(n + 1, 0);
  // JV column reduction: v_j = min_i c_ij, and column j takes its minimising
  // row when that row is still free.  Reduced costs c - u - v stay >= 0 and
  // every assigned pair is tight, so the augmentation below starts from a
  // partial optimum.
  for (int j = 1; j <= n; ++j) {
    int best_i = 1;
    double best = (double)cost[j - 1];
    for (int i = 2; i <= n; ++i) {
      const double c = (double)cost[(size_t)(i - 1) * n + (j - 1)];
      if (c < best) {
        best = c;
        best_i = i;
      }
    }
    v[j] = best;
    if (!row_used[best_i]) {
      row_used[best_i] = 1;
      row_of[j] = best_i;
    }
  }
  // JV augmenting row reduction, two passes over the free rows: a free row i
  // takes the column j1 minimising c_ij - v_j; if that beats the runner-up j2
  // strictly, v_j1 drops by the gap (so j1 and j2 tie for row i) and the row
  // that held j1, if any, is processed next; on a tie the row takes j2 when j1
  // is held, and a displaced row waits for the next pass.  Every assigned row
  // keeps a column of least c_ij - v_j (lowering a v only raises c - v), so
  // u_i = that least value makes c - u - v >= 0 with the matching tight.  A
  // step limit hands whatever is left to the augmentation below, which is exact
  // from any such state.
  std::vector<int> col_of(n + 1, 0);
  for (int j = 1; j <= n; ++j)
    if (row_of[j]) col_of[row_of[j]] = j;
  if (n > 1) {
    std::vector<int> freel, later;
    for (int i = 1; i <= n; ++i)
      if (!row_used[i]) freel.push_back(i);
    for (int pass = 0; pass < 2 && !freel.empty(); ++pass) {
      later.clear();
      size_t k = 0;
      long steps = 0;
      const long max_steps = 16L * n;
      while (k < freel.size()) {
        if (++steps > max_steps) {
          for (; k < freel.size(); ++k) later.push_back(freel[k]);
          break;
        }
        const int i = freel[k++];
        const float* ci = cost + (size_t)(i - 1) * n;
        double u1 = (double)ci[0] - v[1], u2 = kInf;
        int j1 = 1, j2 = 0;
        for (int j = 2; j <= n; ++j) {
          const double h = (double)ci[j - 1] - v[j];
          if (h < u2) {
            if (h >= u1) {
              u2 = h;
              j2 = j;
            } else {
              u2 = u1;
              u1 = h;
              j2 = j1;
              j1 = j;
            }
          }
        }
        int i0 = row_of[j1];
        const bool strict = u1 < u2;
        if (strict) {
          v[j1] -= u2 - u1;
        } else if (i0 != 0) {
          j1 = j2;
          i0 = row_of[j1];
        }
        if (i0 != 0) {
          col_of[i0] = 0;
          row_used[i0] = 0;
        }
        row_of[j1] = i;
        col_of[i] = j1;
        row_used[i] = 1;
        if (i0 != 0) {
          if (strict) freel[--k] = i0;  // the displaced row goes next
          else later.push_back(i0);
        }
      }
      freel.swap(later);
    }
    for (int i = 1; i <= n; ++i)
      if (row_used[i]) u[i] = (double)cost[(size_t)(i - 1) * n + (col_of[i] - 1)] - v[col_of[i]];
  }
  for (int r = 1; r <= n; ++r) {
    if (row_used[r]) continue;
    row_of[0] = r;
    int col = 0;
    std::fill(dist.begin(), dist.end(), kInf);
    std::fill(done.begin(), done.end(), 0);
    // grow the shortest-path tree until it reaches a free column
    while (true) {
      done[col] = 1;
      const int i = row_of[col];
      const float* ci = cost + (size_t)(i - 1) * n;
      double best = kInf;
      int next = -1;
      for (int j = 1; j <= n; ++j) {
        if (done[j]) continue;
        const double red = (double)ci[j - 1] - u[i] - v[j];
        if (red < dist[j]) {
          dist[j] = red;
          prev[j] = col;
        }
        if (dist[j] < best) {
          best = dist[j];
          next = j;
        }
      }
      // shift the potentials by the step length: tree columns keep zero
      // reduced cost along the tree, the others' tentative distances shrink
      for (int j = 0; j <= n; ++j) {
        if (done[j]) {
          u[row_of[j]] += best;
          v[j] -= best;
        } else {
          dist[j] -= best;
        }
      }
      col = next;
      if (row_of[col] == 0) break;
    }
    // augment along the path back to the virtual column
    while (col) {
      const int p = prev[col];
      row_of[col] = row_of[p];
      col = p;
    }
  }
  double sum = 0.0;
  for (int j = 1; j <= n; ++j) {
    assign[row_of[j] - 1] = j - 1;
  }
  for (int i = 0; i < n; ++i) sum += (double)cost[(size_t)i * n + assign[i]];
  if (total) *total = sum;
}
}  // namespace

extern "C" lx_status lx_lap_solve(const float* cost, int32_t n, int32_t* assign, double* total) {
  using namespace lx;
  if (n < 1 || n > 65536) return fail(LX_ERR_ARG, "n must be in 1..65536");
  if (!cost || !assign) return fail(LX_ERR_ARG, "cost or assign is NULL");
  if (!costs_finite(cost, (long)n * n)) return fail(LX_ERR_ARG, "cost holds a NaN or an infinity");
  lap_solve_one(cost, n, assign, total);
  return LX_OK;
}

extern "C" lx_status lx_lap_solve_batch(const float* costs, int32_t n, int32_t count,
                                        int32_t* assign, double* totals, int32_t threads) {
  using namespace lx;
  if (n < 1 || n > 65536) return fail(LX_ERR_ARG, "n must be in 1..65536");
  if (count < 0) return fail(LX_ERR_ARG, "count < 0");
  if (count == 0) return LX_OK;
  if (!costs || !assign) return fail(LX_ERR_ARG, "costs or assign is NULL");
  const size_t nn = (size_t)n * n;
  if (!costs_finite(costs, (long)(nn * count)))
    return fail(LX_ERR_ARG, "a cost holds a NaN or an infinity");
  int nt = threads > 0 ? threads : (int)std::thread::hardware_concurrency();
  nt = std::max(1, std::min(nt, (int)count));
  std::atomic<int> next(0);
  auto work = [&]() {
    for (int b = next.fetch_add(1); b < count; b = next.fetch_add(1))
      lap_solve_one(costs + (size_t)b * nn, n, assign + (size_t)b * n, totals ? totals + b : nullptr);
  };
  std::vector<std::thread> pool;
  for (int t = 1; t < nt; ++t) pool.emplace_back(work);
  work();
  for (auto& th : pool) th.join();
  return LX_OK;
}
