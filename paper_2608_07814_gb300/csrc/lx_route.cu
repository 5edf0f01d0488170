// Router: logits in the canonical fp32 order, top-k, softmax gates.
//
// The router is the MoE layer's own, unchanged by compression (Sec. 1, Fig. 1;
// Sec. 3.2 Stage 1).  Logit order (fixed so that the top-k decision is
// reproducible): H is cut into chunks of 8 elements, chunk q belongs to lane
// q mod 32, each lane accumulates its chunks in ascending h with fused
// multiply-adds, and the 32 lane partials are added pairwise at offsets
// 16, 8, 4, 2, 1; the bias (if any) is added last.
#include <climits>

#include "lx_internal.cuh"

namespace lx {

namespace {

constexpr int RT_TOK = 8;        // tokens per CTA
constexpr int RT_THREADS = 256;  // 8 warps

__device__ __forceinline__ void load8(const float* p, float (&v)[8]) {
  const float4 a = *reinterpret_cast<const float4*>(p);
  const float4 b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

__device__ __forceinline__ void load8(const __nv_bfloat16* p, float (&v)[8]) {
  const uint4 u = *reinterpret_cast<const uint4*>(p);
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    v[2 * i] = __uint_as_float(w[i] << 16);
    v[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

// better(v, i) than (bv, bi): larger logit, ties to the lower expert id
__device__ __forceinline__ bool better(float v, int i, float bv, int bi) {
  return v > bv || (v == bv && i < bi);
}

template <typename T>
__global__ void __launch_bounds__(RT_THREADS)
k_router(const T* __restrict__ x, const T* __restrict__ W, const float* __restrict__ bias,
         int Ttok, int E, int H, int k, int* __restrict__ topk_id, float* __restrict__ topk_w,
         float* __restrict__ logits_out) {
  extern __shared__ __align__(16) unsigned char smem[];
  T* xs = reinterpret_cast<T*>(smem);
  const size_t xbytes = ((size_t)RT_TOK * H * sizeof(T) + 15) / 16 * 16;
  float* ls = reinterpret_cast<float*>(smem + xbytes);
  const int t0 = blockIdx.x * RT_TOK;
  const int nt = min(RT_TOK, Ttok - t0);

  // stage the token tile (16-byte vectors; H*sizeof(T) is a multiple of 16)
  {
    const int vec_per_tok = H * (int)sizeof(T) / 16;
    const uint4* src = reinterpret_cast<const uint4*>(x + (size_t)t0 * H);
    uint4* dst = reinterpret_cast<uint4*>(xs);
    for (int i = threadIdx.x; i < nt * vec_per_tok; i += blockDim.x) dst[i] = src[i];
  }
  __syncthreads();

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  const int nchunk = H / 8;
  for (int e = warp; e < E; e += nw) {
    float acc[RT_TOK];
#pragma unroll
    for (int tt = 0; tt < RT_TOK; ++tt) acc[tt] = 0.f;
    const T* w = W + (size_t)e * H;
    for (int q = lane; q < nchunk; q += 32) {
      float wv[8];
      load8(w + 8 * q, wv);
#pragma unroll
      for (int tt = 0; tt < RT_TOK; ++tt) {
        if (tt < nt) {
          float xv[8];
          load8(xs + (size_t)tt * H + 8 * q, xv);
#pragma unroll
          for (int i = 0; i < 8; ++i) acc[tt] = __fmaf_rn(xv[i], wv[i], acc[tt]);
        }
      }
    }
#pragma unroll
    for (int tt = 0; tt < RT_TOK; ++tt) {
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1)
        acc[tt] = __fadd_rn(acc[tt], __shfl_down_sync(0xffffffffu, acc[tt], off));
    }
    if (lane == 0) {
      const float b = bias ? bias[e] : 0.f;
      for (int tt = 0; tt < nt; ++tt) ls[tt * E + e] = bias ? __fadd_rn(acc[tt], b) : acc[tt];
    }
  }
  __syncthreads();

  // top-k per token: one warp per token
  for (int tt = warp; tt < nt; tt += nw) {
    const float* lt = ls + tt * E;
    const size_t t = (size_t)t0 + tt;
    if (logits_out)
      for (int e = lane; e < E; e += 32) logits_out[t * E + e] = lt[e];
    uint32_t taken = 0;  // bit i <-> expert lane + 32 i
    float m = 0.f, denom = 0.f;
    float selv = 0.f;
    int seli = 0;
    for (int j = 0; j < k; ++j) {
      float bv = -INFINITY;
      int bi = INT_MAX;
      for (int i = 0, e = lane; e < E; ++i, e += 32)
        if (!((taken >> i) & 1u) && better(lt[e], e, bv, bi)) { bv = lt[e]; bi = e; }
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
        const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
        if (better(ov, oi, bv, bi)) { bv = ov; bi = oi; }
      }
      if (bi == INT_MAX) {  // only NaN left: take the lowest free id so ids stay valid
        int fi = INT_MAX;
        for (int i = 0, e = lane; e < E; ++i, e += 32)
          if (!((taken >> i) & 1u)) { fi = e; break; }
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) fi = min(fi, __shfl_xor_sync(0xffffffffu, fi, off));
        bi = fi;
        bv = lt[bi];
      }
      if ((bi & 31) == lane) taken |= 1u << (bi >> 5);
      if (j == 0) m = bv;
      const float ex = expf(bv - m);
      denom += ex;
      if (lane == j) { selv = ex; seli = bi; }
    }
    if (lane < k) {
      topk_id[t * k + lane] = seli;
      topk_w[t * k + lane] = selv / denom;
    }
  }
}

}  // namespace

lx_status launch_router(lx_layer* L, const void* x, int T, int k, int* topk_id, float* topk_w,
                        float* logits, cudaStream_t s) {
  if (reinterpret_cast<uintptr_t>(x) % 16)
    return fail(LX_ERR_ARG, "x must be 16-byte aligned");
  const size_t xbytes = ((size_t)RT_TOK * L->H * L->esz + 15) / 16 * 16;
  const size_t smem = xbytes + (size_t)RT_TOK * L->E * 4;
  if (smem > 200 * 1024) return fail(LX_ERR_SHAPE, "router tile exceeds shared memory");
  const dim3 grid((T + RT_TOK - 1) / RT_TOK);
  ProfScope ps(L, s, "router");
  if (L->dtype == LX_BF16) {
    auto kern = k_router<__nv_bfloat16>;
    LX_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    kern<<<grid, RT_THREADS, smem, s>>>((const __nv_bfloat16*)x, (const __nv_bfloat16*)L->router_w,
                                        L->router_bias, T, L->E, L->H, k, topk_id, topk_w, logits);
  } else {
    auto kern = k_router<float>;
    LX_CUDA(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
    kern<<<grid, RT_THREADS, smem, s>>>((const float*)x, (const float*)L->router_w, L->router_bias,
                                        T, L->E, L->H, k, topk_id, topk_w, logits);
  }
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

}  // namespace lx
