// Router profiling statistics (Sec. 3.2 Stage 1: per-layer firing counts N_e
// read from the router; Sec. 2.2: the expert co-activation graph weighted by
// normalised pointwise mutual information, whose 1 - NPMI is Stage 2's
// Coact-NPMI clustering distance).
//
// Co-activation counts are an integer histogram over the pairs of each token's
// selected set.  Up to 256 experts, every CTA accumulates its tokens' pairs in
// a shared-memory upper triangle (E(E+1)/2 32-bit counters, 128.5 KiB at
// E = 256) and adds the non-zero entries to the caller's 64-bit matrix at the
// end; above that, pairs go straight to global 64-bit atomics.  Integer
// addition is associative, so both give the same counts in any order.
#include <algorithm>

#include "lx_internal.cuh"

namespace lx {
namespace {

constexpr int CO_THREADS = 512;
constexpr int CO_WARPS = CO_THREADS / 32;
constexpr int CO_SMEM_MAX_E = 256;
constexpr int CO_MIN_TOKENS_PER_CTA = 256;  // keeps the per-CTA flush small against the work

__host__ __device__ inline int tri_size(int E) { return E * (E + 1) / 2; }
// entry (i, j), i <= j, of the row-major upper triangle
__device__ __forceinline__ int tri_index(int i, int j, int E) { return i * E - i * (i - 1) / 2 + (j - i); }

// One warp per token: lane s holds slot s's id.  A lane is selected when its id
// is in [0, E) and no lower lane holds the same id (the selected set of the
// token).  Returns the selected-lane mask; `id` is this lane's id.
__device__ __forceinline__ unsigned token_selection(const int* __restrict__ ids, int t, int k,
                                                    int E, int lane, int& id) {
  id = lane < k ? ids[(size_t)t * k + lane] : -1;
  const bool valid = id >= 0 && id < E;
  const int key = valid ? id : -1 - lane;  // invalid lanes never match another lane
  const unsigned same = __match_any_sync(0xffffffffu, key);
  const bool first = lane == __ffs(same) - 1;
  return __ballot_sync(0xffffffffu, valid && first);
}

__global__ void __launch_bounds__(CO_THREADS)
k_coact_smem(const int* __restrict__ ids, int T, int k, int E,
             unsigned long long* __restrict__ fire, unsigned long long* __restrict__ coact) {
  extern __shared__ unsigned int tri[];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int n_tri = tri_size(E);
  for (int q = tid; q < n_tri; q += CO_THREADS) tri[q] = 0u;
  __syncthreads();
  for (int t = blockIdx.x * CO_WARPS + warp; t < T; t += gridDim.x * CO_WARPS) {
    int id;
    const unsigned sel = token_selection(ids, t, k, E, lane, id);
    const bool mine = (sel >> lane) & 1u;
    for (unsigned b = sel; b; b &= b - 1) {  // warp-uniform loop over the selected lanes
      const int other = __shfl_sync(0xffffffffu, id, __ffs(b) - 1);
      if (mine && other >= id) atomicAdd(&tri[tri_index(id, other, E)], 1u);
    }
  }
  __syncthreads();
  for (int q = tid; q < E * E; q += CO_THREADS) {
    const int i = q / E, j = q - i * E;
    if (j < i) continue;
    const unsigned int c = tri[tri_index(i, j, E)];
    if (!c) continue;
    if (coact) {
      atomicAdd(&coact[(size_t)i * E + j], (unsigned long long)c);
      if (i != j) atomicAdd(&coact[(size_t)j * E + i], (unsigned long long)c);
    }
    if (i == j && fire) atomicAdd(&fire[i], (unsigned long long)c);
  }
}

__global__ void __launch_bounds__(CO_THREADS)
k_coact_global(const int* __restrict__ ids, int T, int k, int E,
               unsigned long long* __restrict__ fire, unsigned long long* __restrict__ coact) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int t = blockIdx.x * CO_WARPS + warp; t < T; t += gridDim.x * CO_WARPS) {
    int id;
    const unsigned sel = token_selection(ids, t, k, E, lane, id);
    const bool mine = (sel >> lane) & 1u;
    if (mine && fire) atomicAdd(&fire[id], 1ull);
    if (!coact) continue;
    for (unsigned b = sel; b; b &= b - 1) {
      const int other = __shfl_sync(0xffffffffu, id, __ffs(b) - 1);
      if (mine) atomicAdd(&coact[(size_t)id * E + other], 1ull);
    }
  }
}

// p_i = C_ii / n, p_ij = C_ij / n; ln(p_ij / (p_i p_j)) / (-ln p_ij) for
// 0 < p_ij < 1, -1 for p_ij = 0, +1 for p_ij = 1 (float64).
__global__ void k_npmi(const unsigned long long* __restrict__ coact, int E,
                       unsigned long long n, double* __restrict__ npmi) {
  const long q = (long)blockIdx.x * blockDim.x + threadIdx.x;
  if (q >= (long)E * E) return;
  const int i = (int)(q / E), j = (int)(q - (long)i * E);
  const unsigned long long cij = coact[q];
  double v;
  if (cij == 0ull) {
    v = -1.0;
  } else if (cij >= n) {
    v = 1.0;
  } else {
    const double nn = (double)n;
    const double p_ij = (double)cij / nn;
    const double p_i = (double)coact[(size_t)i * E + i] / nn;
    const double p_j = (double)coact[(size_t)j * E + j] / nn;
    v = log(p_ij / (p_i * p_j)) / (-log(p_ij));
  }
  npmi[q] = v;
}

bool g_co_smem_cap[64] = {};

}  // namespace
}  // namespace lx

extern "C" lx_status lx_coact_accumulate(const int32_t* topk_id, int32_t T, int32_t k, int32_t E,
                                         uint64_t* fire, uint64_t* coact, void* stream) {
  using namespace lx;
  if (T < 0) return fail(LX_ERR_ARG, "T < 0");
  if (k < 1 || k > LX_MAX_K) return fail(LX_ERR_ARG, "k must be in 1..LX_MAX_K");
  if (E < 1 || E > LX_MAX_EXPERTS) return fail(LX_ERR_ARG, "E must be in 1..LX_MAX_EXPERTS");
  if (!fire && !coact) return fail(LX_ERR_ARG, "fire and coact are both NULL");
  if (T == 0) return LX_OK;
  if (!topk_id) return fail(LX_ERR_ARG, "topk_id is NULL");
  cudaStream_t s = (cudaStream_t)stream;
  int dev = 0, sms = 0;
  LX_CUDA(cudaGetDevice(&dev));
  LX_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  const long want = ((long)T + CO_MIN_TOKENS_PER_CTA - 1) / CO_MIN_TOKENS_PER_CTA;
  const int grid = (int)std::max(1L, std::min(want, 2L * sms));
  unsigned long long* f = reinterpret_cast<unsigned long long*>(fire);
  unsigned long long* c = reinterpret_cast<unsigned long long*>(coact);
  if (E <= CO_SMEM_MAX_E) {
    const size_t smem = sizeof(unsigned int) * (size_t)tri_size(E);
    LX_CUDA(smem_cap_once((const void*)k_coact_smem, (int)(sizeof(unsigned int) * tri_size(CO_SMEM_MAX_E)),
                          dev, g_co_smem_cap));
    k_coact_smem<<<grid, CO_THREADS, smem, s>>>(topk_id, T, k, E, f, c);
  } else {
    const long g2 = std::min(((long)T + CO_WARPS - 1) / CO_WARPS, 8L * sms);
    k_coact_global<<<(int)std::max(1L, g2), CO_THREADS, 0, s>>>(topk_id, T, k, E, f, c);
  }
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

extern "C" lx_status lx_coact_npmi(const uint64_t* coact, int32_t E, int64_t n_tokens,
                                   double* npmi, void* stream) {
  using namespace lx;
  if (E < 1 || E > LX_MAX_EXPERTS) return fail(LX_ERR_ARG, "E must be in 1..LX_MAX_EXPERTS");
  if (n_tokens < 0) return fail(LX_ERR_ARG, "n_tokens < 0");
  if (!coact || !npmi) return fail(LX_ERR_ARG, "coact or npmi is NULL");
  const long n = (long)E * E;
  k_npmi<<<(unsigned)((n + 255) / 256), 256, 0, (cudaStream_t)stream>>>(
      reinterpret_cast<const unsigned long long*>(coact), E, (unsigned long long)n_tokens, npmi);
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}
