// The range finder's residual products on the tensor cores (Sec. 3.2 Stage 3
// (ii), Eq. svd): C = R X with R = W_mem - W_dom [M][K] (or R^T) and X an fp32
// [K][N] basis (the Gaussian test matrix, then the orthonormal bases of the
// power iterations).
//
// The weights are exact bf16 operands; X is split into three bf16 parts,
// X = X_hi + X_mid + X_lo (each part the bf16 rounding of what the previous
// ones leave, so the sum reproduces X to fp32 precision), and the difference
// of the two experts rides along K: one tcgen05 GEMM over the concatenation
//   [W_mem | W_mem | W_mem | W_dom | W_dom | W_dom] . [X_hi ; X_mid ; X_lo ; -X_hi ; -X_mid ; -X_lo]
// (bf16 x bf16 products are exact in the fp32 accumulator).  Every segment is
// padded to a multiple of 64 in K (zeros), so a 64-wide K block never straddles
// two segments.  M is cut into 128-row tiles and K into ranges (split-K, one
// CTA each, so that a few row tiles still fill the GPU); each CTA writes its
// fp32 partial and a second kernel adds the partials in range order.
//
// Kernels: k_split3 (X -> the transposed bf16 parts, [Npad][6 Kp]),
// k_transpose_bf16 (W^T for the R^T products), k_res_mma (TMA + tcgen05, M=128,
// N = Npad <= 256, K=16 per instruction, one accumulator in TMEM), k_sum_parts.
#include <algorithm>
#include <cstring>

#include "lx_internal.cuh"
#include "lx_tcgen05.cuh"

namespace lx {
namespace {

using namespace tcg;

constexpr int RM_BM = 128;
constexpr int RM_BK = 64;
constexpr int RM_STAGES = 4;
constexpr int RM_THREADS = 192;  // producer, MMA, four epilogue warps
constexpr int RM_A_BYTES = RM_BM * RM_BK * 2;  // 16 KiB

struct ResLaunch {
  CUtensorMap a_mem;  // [M][K] bf16, 64 x 128 boxes (W_mem or W_mem^T)
  CUtensorMap a_dom;  // [M][K] bf16 (W_dom or W_dom^T)
  CUtensorMap b;      // [Npad][6 Kp] bf16, 64 x Npad boxes
  int M, Npad, kb_seg, kb_split, n_kb;  // 64-wide K blocks: per segment, per CTA, in all
  float* part;        // [gridDim.z][splits][M][Npad]: blockIdx.z takes B rows z Npad ..
  unsigned long long wait_cycles;
};

__global__ void __launch_bounds__(RM_THREADS, 1) k_res_mma(const __grid_constant__ ResLaunch P) {
  pdl_wait();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int b_bytes = P.Npad * RM_BK * 2;
  const int stage_bytes = RM_A_BYTES + ((b_bytes + 1023) & ~1023);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + RM_STAGES * stage_bytes);
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * RM_STAGES;
  const uint32_t done = empty0 + 8 * RM_STAGES;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 2 * RM_STAGES + 1);
  uint32_t* tmem_base_s = reinterpret_cast<uint32_t*>(bars + 2 * RM_STAGES + 2);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t smem_base = smem_u32(smem);
  const int m0 = blockIdx.x * RM_BM;
  const int kb0 = blockIdx.y * P.kb_split;
  const int nkb = min(P.kb_split, P.n_kb - kb0);
  if (threadIdx.x == 0) {
    for (int s = 0; s < RM_STAGES; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    mbar_init(done, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_base_s)),
                 "r"(256)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_base_s;
  uint32_t issued = 0;

  if (warp == 0) {
    if (lane == 0) {
      for (int i = 0; i < nkb; ++i) {
        const uint32_t s = i % RM_STAGES;
        if (!mbar_wait(empty0 + 8 * s, ((i / RM_STAGES) & 1) ^ 1, abort_flag, P.wait_cycles)) {
          *abort_flag = 1;
          break;
        }
        const int kb = kb0 + i, seg = kb / P.kb_seg, kk = kb % P.kb_seg;
        mbar_expect_tx(full0 + 8 * s, RM_A_BYTES + b_bytes);
        const uint32_t a_s = smem_base + s * stage_bytes, b_s = a_s + RM_A_BYTES;
        tma_load_2d(a_s, seg < 3 ? &P.a_mem : &P.a_dom, kk * RM_BK, m0, full0 + 8 * s);
        tma_load_2d(b_s, &P.b, kb * RM_BK, (int)blockIdx.z * P.Npad, full0 + 8 * s);
        issued = i + 1;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = instr_desc(RM_BM, P.Npad);
      bool ok = true;
      for (int i = 0; i < nkb; ++i) {
        const uint32_t s = i % RM_STAGES;
        if (!mbar_wait(full0 + 8 * s, (i / RM_STAGES) & 1, abort_flag, P.wait_cycles)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a_s = smem_base + s * stage_bytes, b_s = a_s + RM_A_BYTES;
#pragma unroll
        for (int k = 0; k < RM_BK / 16; ++k)
          tc_mma(tmem, smem_desc(a_s + 32 * k), smem_desc(b_s + 32 * k), idesc,
                 (i | k) != 0 ? 1u : 0u);
        tc_commit(empty0 + 8 * s);
      }
      if (!ok) *abort_flag = 1;
      // arrives once every MMA issued has completed (also on the abort path,
      // so that no MMA is in flight when the TMEM is released)
      tc_commit(done);
    }
    __syncwarp();
  } else {
    // epilogue: warp w reads TMEM lanes 32 (w % 4) .. + 31 (tile rows)
    const int q = warp & 3;
    int ok = 1;
    if (lane == 0) ok = (mbar_wait(done, 0, abort_flag, P.wait_cycles) && !*abort_flag) ? 1 : 0;
    ok = __shfl_sync(0xffffffffu, ok, 0);  // warp-uniform: the TMEM loads are warp-wide
    __syncwarp();
    tc_fence_after();
    // 32-column blocks of the warp's 32 rows staged in shared memory (the
    // stages are free: every MMA has completed), then stored as whole 128-byte
    // row segments (eight lanes per row, four rows per store)
    float* out = P.part + (((size_t)blockIdx.z * gridDim.y + blockIdx.y) * P.M + m0 + 32 * q) * P.Npad;
    float* stg = reinterpret_cast<float*>(smem) + q * 32 * 33;
    if (ok) {
      for (int c0 = 0; c0 < P.Npad; c0 += 32) {
        const int w = min(32, P.Npad - c0);  // 16 or 32 (Npad is a multiple of 16)
        const uint32_t ta = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)c0;
        uint32_t v[32];
        tc_ld16_async(ta, *reinterpret_cast<uint32_t(*)[16]>(v));
        if (w == 32) tc_ld16_async(ta + 16, *reinterpret_cast<uint32_t(*)[16]>(v + 16));
        tc_wait_ld();
#pragma unroll
        for (int c = 0; c < 32; ++c)
          if (c < w) stg[lane * 33 + c] = __uint_as_float(v[c]);
        __syncwarp();
        const int cq = lane & 7;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int rr = 4 * j + (lane >> 3);
          if (m0 + 32 * q + rr < P.M && 4 * cq < w) {
            const float* sr = stg + rr * 33 + 4 * cq;
            *reinterpret_cast<float4*>(out + (size_t)rr * P.Npad + c0 + 4 * cq) =
                make_float4(sr[0], sr[1], sr[2], sr[3]);
          }
        }
        __syncwarp();
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(256)
                 : "memory");
  } else if (warp == 0 && lane == 0 && *abort_flag) {
    // copies still in flight land before shared memory goes away
    const uint32_t first = issued > RM_STAGES ? issued - RM_STAGES : 0;
    for (uint32_t j = first; j < issued; ++j)
      mbar_wait(full0 + 8 * (j % RM_STAGES), (j / RM_STAGES) & 1, nullptr);
  }
}

// X [K][N] fp32 (row-major) -> Bc [Npad][6 Kp] bf16: row n holds column n of
// X as hi | mid | lo | -hi | -mid | -lo, each segment Kp long (zeros past K
// and for n >= N).  hi = bf16(x), mid = bf16(x - hi), lo = bf16(x - hi - mid)
// (both differences are exact in fp32).
__global__ void k_split3(const float* __restrict__ X, int K, int N, int Kp, int Npad,
                         __nv_bfloat16* __restrict__ Bc) {
  const int n = blockIdx.y;
  for (int k = blockIdx.x * blockDim.x + threadIdx.x; k < Kp; k += gridDim.x * blockDim.x) {
    const float x = (n < N && k < K) ? X[(size_t)k * N + n] : 0.f;
    const __nv_bfloat16 hi = __float2bfloat16_rn(x);
    const float r1 = x - __bfloat162float(hi);
    const __nv_bfloat16 mid = __float2bfloat16_rn(r1);
    const __nv_bfloat16 lo = __float2bfloat16_rn(r1 - __bfloat162float(mid));
    __nv_bfloat16* row = Bc + (size_t)n * 6 * Kp + k;
    row[0] = hi;
    row[Kp] = mid;
    row[2 * (size_t)Kp] = lo;
    row[3 * (size_t)Kp] = __hneg(hi);
    row[4 * (size_t)Kp] = __hneg(mid);
    row[5 * (size_t)Kp] = __hneg(lo);
  }
}

// W [rows][cols] -> W^T [cols][rows] (bf16), 32 x 32 tiles through shared memory
__global__ void k_transpose_bf16(const __nv_bfloat16* __restrict__ W, int rows, int cols,
                                 __nv_bfloat16* __restrict__ Wt) {
  __shared__ __nv_bfloat16 tile[32][33];
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  for (int i = threadIdx.y; i < 32; i += blockDim.y) {
    const int r = r0 + i, c = c0 + threadIdx.x;
    if (r < rows && c < cols) tile[i][threadIdx.x] = W[(size_t)r * cols + c];
  }
  __syncthreads();
  for (int i = threadIdx.y; i < 32; i += blockDim.y) {
    const int c = c0 + i, r = r0 + threadIdx.x;
    if (r < rows && c < cols) Wt[(size_t)c * rows + r] = tile[threadIdx.x][i];
  }
}

// C [M][N] = sum over the K ranges s (ascending) of part[s][M][Npad]
__global__ void k_sum_parts(const float* __restrict__ part, int splits, int M, int N, int Npad,
                            float* __restrict__ C) {
  const long total = (long)M * N;
  for (long i = (long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (long)gridDim.x * blockDim.x) {
    const long m = i / N, n = i % N;
    float acc = 0.f;
    for (int s = 0; s < splits; ++s) acc += part[((size_t)s * M + m) * Npad + n];
    C[i] = acc;
  }
}

bool g_rm_cap[64] = {};

}  // namespace

size_t res_tc_workspace(long rows, long cols, long l) {
  const long Npad = (l + 15) / 16 * 16, Kp = (std::max(rows, cols) + 63) / 64 * 64;
  const long Mmax = std::max(rows, cols);
  auto al = [](size_t v) { return (v + 255) / 256 * 256; };
  return al(2 * (size_t)rows * cols * 2) + al((size_t)Npad * 6 * Kp * 2) +
         al((size_t)RES_TC_MAX_SPLITS * Mmax * Npad * 4);
}

bool res_tc_fits(long rows, long cols, long l) {
  return rows % 8 == 0 && cols % 8 == 0 && l >= 1 && (l + 15) / 16 * 16 <= 256;
}

lx_status res_gemm_tc(bool transposed, const __nv_bfloat16* Wm, const __nv_bfloat16* Wd,
                      long rows, long cols, const float* X, long N, float* C, char* ws,
                      int num_sms, int dev, cudaStream_t s) {
  auto al = [](size_t v) { return (v + 255) / 256 * 256; };
  __nv_bfloat16* Wt = reinterpret_cast<__nv_bfloat16*>(ws);  // [2][cols][rows]
  __nv_bfloat16* Bc = reinterpret_cast<__nv_bfloat16*>(ws + al(2 * (size_t)rows * cols * 2));
  const long M = transposed ? cols : rows, K = transposed ? rows : cols;
  const long Npad = (N + 15) / 16 * 16, Kp = (K + 63) / 64 * 64;
  float* part = reinterpret_cast<float*>(
      ws + al(2 * (size_t)rows * cols * 2) +
      al((size_t)Npad * 6 * ((std::max(rows, cols) + 63) / 64 * 64) * 2));
  const __nv_bfloat16* Am = Wm;
  const __nv_bfloat16* Ad = Wd;
  if (transposed) {
    const dim3 grid((unsigned)((cols + 31) / 32), (unsigned)((rows + 31) / 32));
    k_transpose_bf16<<<grid, dim3(32, 8), 0, s>>>(Wm, (int)rows, (int)cols, Wt);
    k_transpose_bf16<<<grid, dim3(32, 8), 0, s>>>(Wd, (int)rows, (int)cols,
                                                   Wt + (size_t)rows * cols);
    Am = Wt;
    Ad = Wt + (size_t)rows * cols;
  }
  k_split3<<<dim3((unsigned)((Kp + 255) / 256), (unsigned)Npad), 256, 0, s>>>(
      X, (int)K, (int)N, (int)Kp, (int)Npad, Bc);
  ResLaunch P;
  std::memset(&P, 0, sizeof(P));
  if (!encode_bf16_2d(&P.a_mem, Am, K, M, 64, RM_BM) ||
      !encode_bf16_2d(&P.a_dom, Ad, K, M, 64, RM_BM) ||
      !encode_bf16_2d(&P.b, Bc, 6 * Kp, Npad, 64, (int)Npad))
    return fail(LX_ERR_CUDA, "cuTensorMapEncodeTiled(residual product) failed");
  const int mt = (int)((M + RM_BM - 1) / RM_BM);
  P.M = (int)M;
  P.Npad = (int)Npad;
  P.kb_seg = (int)(Kp / 64);
  P.n_kb = 6 * P.kb_seg;
  // K ranges: enough CTAs to fill the GPU, at least 4 K blocks each
  int splits = std::max(1, std::min(RES_TC_MAX_SPLITS, num_sms / mt));
  splits = std::min(splits, std::max(1, P.n_kb / 4));
  P.kb_split = (P.n_kb + splits - 1) / splits;
  splits = (P.n_kb + P.kb_split - 1) / P.kb_split;
  P.part = part;
  P.wait_cycles = kDefaultWaitCycles;
  const int b_bytes = (int)Npad * 64 * 2;
  const int smem = RM_STAGES * (RM_A_BYTES + ((b_bytes + 1023) & ~1023)) + 8 * (2 * RM_STAGES + 3) + 1024;
  LX_CUDA(smem_cap_once((const void*)k_res_mma, 227 * 1024, dev, g_rm_cap));
  k_res_mma<<<dim3((unsigned)mt, (unsigned)splits), RM_THREADS, smem, s>>>(P);
  const long total = M * N;
  k_sum_parts<<<(unsigned)std::min<long>((total + 255) / 256, 4L * num_sms), 256, 0, s>>>(
      part, splits, (int)M, (int)N, (int)Npad, C);
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

// A plain split-K product on the same kernel (one K segment): part[s][M][Npad]
// = A[M][K-range s] . B[Npad][K-range s]^T, A and B given as 2-D bf16 maps of
// 64 x 128 and 64 x Npad boxes (K a multiple of 64); returns the ranges used.
lx_status tc_splitk_gemm(lx_layer* L, const CUtensorMap& a, const CUtensorMap& b, int M, int Npad,
                         int K, float* part, int max_splits, int* splits_out, cudaStream_t s,
                         const char* name) {
  ResLaunch P;
  std::memset(&P, 0, sizeof(P));
  P.a_mem = a;
  P.a_dom = a;
  P.b = b;
  const int mt = (M + RM_BM - 1) / RM_BM;
  P.M = M;
  P.Npad = Npad;
  P.kb_seg = K / 64;
  P.n_kb = P.kb_seg;  // one segment: every K block reads A from a_mem
  int splits = std::max(1, std::min(max_splits, L->num_sms / mt));
  splits = std::min(splits, std::max(1, P.n_kb / 4));
  P.kb_split = (P.n_kb + splits - 1) / splits;
  splits = (P.n_kb + P.kb_split - 1) / P.kb_split;
  P.part = part;
  P.wait_cycles = wait_limit(L);
  const int b_bytes = Npad * 64 * 2;
  const int smem = RM_STAGES * (RM_A_BYTES + ((b_bytes + 1023) & ~1023)) + 8 * (2 * RM_STAGES + 3) + 1024;
  LX_CUDA(smem_cap_once((const void*)k_res_mma, 227 * 1024, L->device, g_rm_cap));
  ProfScope ps(L, s, name);
  launch_k(L, k_res_mma, dim3((unsigned)mt, (unsigned)splits), RM_THREADS, smem, s, P);
  LX_CUDA(cudaGetLastError());
  *splits_out = splits;
  return LX_OK;
}

// The same kernel over column chunks: part[z][s][M][Npad] = A[M][K-range s] .
// B[rows z Npad ..][K-range s]^T for z < nz (one launch, grid (M tiles, ranges,
// nz)); a plain launch (no layer), for the stateless entry points.
lx_status tc_splitk_gemm_chunks(const CUtensorMap& a, const CUtensorMap& b, int M, int Npad,
                                int nz, int K, float* part, int max_splits, int* splits_out,
                                int num_sms, int dev, cudaStream_t s) {
  ResLaunch P;
  std::memset(&P, 0, sizeof(P));
  P.a_mem = a;
  P.a_dom = a;
  P.b = b;
  const int mt = (M + RM_BM - 1) / RM_BM;
  P.M = M;
  P.Npad = Npad;
  P.kb_seg = K / 64;
  P.n_kb = P.kb_seg;
  int splits = std::max(1, std::min(max_splits, num_sms / std::max(1, mt * nz)));
  splits = std::min(splits, std::max(1, P.n_kb / 4));
  P.kb_split = (P.n_kb + splits - 1) / splits;
  splits = (P.n_kb + P.kb_split - 1) / P.kb_split;
  P.part = part;
  P.wait_cycles = kDefaultWaitCycles;
  const int b_bytes = Npad * 64 * 2;
  const int smem = RM_STAGES * (RM_A_BYTES + ((b_bytes + 1023) & ~1023)) + 8 * (2 * RM_STAGES + 3) + 1024;
  LX_CUDA(smem_cap_once((const void*)k_res_mma, 227 * 1024, dev, g_rm_cap));
  k_res_mma<<<dim3((unsigned)mt, (unsigned)splits, (unsigned)nz), RM_THREADS, smem, s>>>(P);
  LX_CUDA(cudaGetLastError());
  *splits_out = splits;
  return LX_OK;
}

}  // namespace lx
