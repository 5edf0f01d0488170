// Router: logits in the canonical fp32 order, then top-k and softmax gates,
// in one launch.
//
// The router is the MoE layer's own, unchanged by compression (Sec. 1, Fig. 1;
// Sec. 3.2 Stage 1).  Logit order (fixed so that the top-k decision is
// reproducible): H is cut into chunks of 8 elements, chunk q belongs to lane
// q mod 32, each lane accumulates its chunks in ascending h with fused
// multiply-adds, and the 32 lane partials are added pairwise at offsets
// 16, 8, 4, 2, 1; the bias (if any) is added last.
//
// Small batches (k_router_logits): one CTA computes the logits of 4 tokens
// for a slice of the experts (one expert per warp, so that a decode batch
// still spreads the 0.5 MB router matrix over many SMs).  Each warp owns one
// expert at a time and issues its weight loads in groups of 8 independent
// 16-byte loads before using them; the first group goes out before the wait
// for the preceding kernel, since the router matrix does not depend on it.
//
// Large bf16 batches (k_router_tiled): persistent CTAs walk tiles of 8
// tokens.  A thread holds the lane partials of 8 tokens x 8 experts for its
// lane's chunks (64 accumulators), so every widened weight value serves 8
// tokens and every widened token value 8 experts; two tokens' partials of one
// expert advance by one packed fp32x2 FMA (each half rounded once, as fmaf),
// which halves the FMA instructions of this issue-bound loop; the weight
// chunks (read through L2) are software-pipelined one chunk ahead.  The 32 lane partials are
// then combined by a transpose-reduce whose pairs are those of the canonical
// order (lane l with lane l ^ 16, then ^ 8, ^ 4, ^ 2, ^ 1; IEEE addition is
// commutative, so each sum is bit-identical), leaving lane l with the logits
// of entries 2l and 2l + 1 of the 8 x 8 block.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <type_traits>

#include "lx_internal.cuh"

namespace lx {

namespace {

constexpr int RT_TOK = 4;        // tokens per CTA (measured at a decode batch of 64: 4 before 2, 8, 1)
constexpr int RT_THREADS = 256;  // 8 warps
constexpr int RT_PREF = 8;       // 16-byte weight loads in flight per lane

__device__ __forceinline__ void widen8(const uint4& u, float (&v)[8]) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    v[2 * i] = __uint_as_float(w[i] << 16);
    v[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

// acc += lo(x) lo(w), then acc += hi(x) hi(w) for the two bf16 halves of the
// packed words x and w: the mixed-precision fma (bf16 operands, fp32 addend and
// result) rounds each product-sum once, exactly as fmaf on the widened
// operands (widening bf16 to fp32 is exact), without the widening operations
__device__ __forceinline__ float fma_bf16_pair(float acc, uint32_t x, uint32_t w) {
  asm("{\n\t.reg .b16 xl, xh, wl, wh;\n\t"
      "mov.b32 {xl, xh}, %1;\n\t"
      "mov.b32 {wl, wh}, %2;\n\t"
      "fma.rn.f32.bf16 %0, xl, wl, %0;\n\t"
      "fma.rn.f32.bf16 %0, xh, wh, %0;\n\t}"
      : "+f"(acc)
      : "r"(x), "r"(w));
  return acc;
}

// 8 consecutive elements as fp32 (bf16: one 16-byte load; fp32: two)
template <typename T>
__device__ __forceinline__ void load8(const T* p, float (&v)[8]);
template <>
__device__ __forceinline__ void load8<float>(const float* p, float (&v)[8]) {
  const float4 a = *reinterpret_cast<const float4*>(p);
  const float4 b = *reinterpret_cast<const float4*>(p + 4);
  v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}
template <>
__device__ __forceinline__ void load8<__nv_bfloat16>(const __nv_bfloat16* p, float (&v)[8]) {
  widen8(*reinterpret_cast<const uint4*>(p), v);
}

template <typename T>
__global__ void __launch_bounds__(RT_THREADS)
k_router_logits(const T* __restrict__ x, const T* __restrict__ W, const float* __restrict__ bias,
                int Ttok, int E, int H, int experts_per_cta, float* __restrict__ logits,
                int* __restrict__ tile_cnt, int k, int* __restrict__ topk_id,
                float* __restrict__ topk_w) {
  extern __shared__ __align__(16) unsigned char smem[];
  T* xs = reinterpret_cast<T*>(smem);
  const int t0 = blockIdx.x * RT_TOK;
  const int nt = min(RT_TOK, Ttok - t0);
  const int e_begin = blockIdx.y * experts_per_cta;
  const int e_end = min(E, e_begin + experts_per_cta);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  const int nchunk = H / 8;
  // weight chunks q0 + 32u (u < RT_PREF) of expert e: independent 16-byte
  // loads (bf16: kept packed, multiplied by the mixed-precision fma)
  constexpr bool kBF = std::is_same<T, __nv_bfloat16>::value;
  float wv[kBF ? 1 : RT_PREF][8];
  uint4 wr[kBF ? RT_PREF : 1];
  auto load_w = [&](int e, int q0) {
#pragma unroll
    for (int u = 0; u < RT_PREF; ++u) {
      const int q = q0 + 32 * u;
      if (q < nchunk) {
        if constexpr (kBF)
          wr[u] = *reinterpret_cast<const uint4*>(W + (size_t)e * H + 8 * q);
        else
          load8(W + (size_t)e * H + 8 * q, wv[u]);
      }
    }
  };
  // The router matrix is a layer constant: the first expert's weights are
  // requested before the wait for the preceding kernel (which may write x).
  int e = e_begin + warp;
  if (e < e_end) load_w(e, lane);
  pdl_wait();
  {
    // the token tile: every 16-byte piece in flight at once
    const int vec_per_tok = H * (int)sizeof(T) / 16;
    const uint4* src = reinterpret_cast<const uint4*>(x + (size_t)t0 * H);
    uint4* dst = reinterpret_cast<uint4*>(xs);
    for (int i = threadIdx.x; i < nt * vec_per_tok; i += blockDim.x) {
      const uint32_t da = static_cast<uint32_t>(__cvta_generic_to_shared(dst + i));
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(da), "l"(src + i) : "memory");
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    asm volatile("cp.async.wait_group 0;" ::: "memory");
  }
  __syncthreads();
  for (; e < e_end; e += nw) {
    float acc[RT_TOK];
#pragma unroll
    for (int tt = 0; tt < RT_TOK; ++tt) acc[tt] = 0.f;
    for (int q0 = lane; q0 < nchunk; q0 += 32 * RT_PREF) {
      if (q0 != lane) load_w(e, q0);  // the expert's first chunks are already loaded
#pragma unroll
      for (int u = 0; u < RT_PREF; ++u) {
        const int q = q0 + 32 * u;
        if (q >= nchunk) break;
#pragma unroll
        for (int tt = 0; tt < RT_TOK; ++tt) {
          if (tt < nt) {
            if constexpr (kBF) {
              const uint4 xr = *reinterpret_cast<const uint4*>(xs + (size_t)tt * H + 8 * q);
              acc[tt] = fma_bf16_pair(acc[tt], xr.x, wr[u].x);
              acc[tt] = fma_bf16_pair(acc[tt], xr.y, wr[u].y);
              acc[tt] = fma_bf16_pair(acc[tt], xr.z, wr[u].z);
              acc[tt] = fma_bf16_pair(acc[tt], xr.w, wr[u].w);
            } else {
              float xv[8];
              load8(xs + (size_t)tt * H + 8 * q, xv);
#pragma unroll
              for (int i = 0; i < 8; ++i) acc[tt] = __fmaf_rn(xv[i], wv[u][i], acc[tt]);
            }
          }
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
      for (int tt = 0; tt < nt; ++tt)
        logits[(size_t)(t0 + tt) * E + e] = bias ? __fadd_rn(acc[tt], b) : acc[tt];
    }
    if (e + nw < e_end) load_w(e + nw, lane);  // the next expert's first chunks
  }
  // The last CTA to finish this token tile's expert slices takes its top-k
  // (no CTA waits for another; the counter is reset for the next call).
  __shared__ int s_last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    const int old = atomicAdd(&tile_cnt[blockIdx.x], 1);
    s_last = old == (int)gridDim.y - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  float* ls = reinterpret_cast<float*>(smem);  // reuse the token tile's space
  for (int i = threadIdx.x; i < nt * E; i += blockDim.x)
    ls[i] = __ldcg(logits + (size_t)t0 * E + i);
  __syncthreads();
  for (int tt = warp; tt < nt; tt += nw) {
    int id;
    float w;
    warp_topk(ls + tt * E, E, k, id, w);
    if (lane < k) {
      topk_id[(size_t)(t0 + tt) * k + lane] = id;
      topk_w[(size_t)(t0 + tt) * k + lane] = w;
    }
  }
  if (threadIdx.x == 0) tile_cnt[blockIdx.x] = 0;
}

constexpr int RTT_TOK = 8;         // tokens per tile (one token per warp in the top-k)
constexpr int RTT_THREADS = 256;   // 8 warps, each on 8-expert groups

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ uint32_t word_of(const uint4& u, int i) {
  return i == 0 ? u.x : i == 1 ? u.y : i == 2 ? u.z : u.w;
}

// (d0, d1) = (a0 * b + d0, a1 * b + d1): two fused multiply-adds, each
// rounded once (the same result as two fmaf), issued as one packed fp32x2
// instruction
__device__ __forceinline__ void fma2_rn(float& d0, float& d1, float a0, float a1, float b) {
  asm("{\n\t.reg .b64 ra, rb, rc;\n\t"
      "mov.b64 ra, {%2, %3};\n\t"
      "mov.b64 rb, {%4, %4};\n\t"
      "mov.b64 rc, {%0, %1};\n\t"
      "fma.rn.f32x2 rc, ra, rb, rc;\n\t"
      "mov.b64 {%0, %1}, rc;\n\t}"
      : "+f"(d0), "+f"(d1)
      : "f"(a0), "f"(a1), "f"(b));
}

// x tile rows [t0, t0 + nt) into shared memory (16-byte cp.async), zeros after
__device__ __forceinline__ void rtt_load_tile(const __nv_bfloat16* x, int t0, int nt, int H,
                                              __nv_bfloat16* xs) {
  const int vec_per_tok = H / 8;
  for (int i = threadIdx.x; i < RTT_TOK * vec_per_tok; i += blockDim.x) {
    const int r = i / vec_per_tok;
    uint4* d = reinterpret_cast<uint4*>(xs) + i;
    if (r < nt) {
      const uint32_t da = static_cast<uint32_t>(__cvta_generic_to_shared(d));
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(da),
                   "l"(reinterpret_cast<const uint4*>(x + (size_t)t0 * H) + i)
                   : "memory");
    } else {
      *d = make_uint4(0, 0, 0, 0);
    }
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
}

__global__ void __launch_bounds__(RTT_THREADS, 1)
k_router_tiled(const __nv_bfloat16* __restrict__ x, const __nv_bfloat16* __restrict__ W,
               const float* __restrict__ bias, int Ttok, int E, int H,
               float* __restrict__ logits, int k, int* __restrict__ topk_id,
               float* __restrict__ topk_w) {
  pdl_wait();
  extern __shared__ __align__(16) unsigned char smem[];
  __nv_bfloat16* xs0 = reinterpret_cast<__nv_bfloat16*>(smem);
  __nv_bfloat16* xs1 = xs0 + (size_t)RTT_TOK * H;
  float* ls = reinterpret_cast<float*>(xs1 + (size_t)RTT_TOK * H);  // [RTT_TOK][E]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nchunk = H / 8, nj = (nchunk + 31) / 32;
  const int ngroups = (E + 7) / 8;
  const int ntiles = (Ttok + RTT_TOK - 1) / RTT_TOK;
  int buf = 0;
  if ((int)blockIdx.x < ntiles) {
    const int t0 = blockIdx.x * RTT_TOK;
    rtt_load_tile(x, t0, min(RTT_TOK, Ttok - t0), H, xs0);
  }
  for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x, buf ^= 1) {
    const int t0 = tile * RTT_TOK, nt = min(RTT_TOK, Ttok - t0);
    const __nv_bfloat16* xs = buf ? xs1 : xs0;
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();
    // the next tile streams in while this one is computed
    const int nxt = tile + gridDim.x;
    if (nxt < ntiles) {
      const int n0 = nxt * RTT_TOK;
      rtt_load_tile(x, n0, min(RTT_TOK, Ttok - n0), H, buf ? xs0 : xs1);
    }
    for (int g = warp; g < ngroups; g += RTT_THREADS / 32) {
      // [expert ee][token tt] partials of this lane: a token pair (tt, tt + 1)
      // of one expert is an adjacent pair, updated by one packed FMA
      float acc[64];
#pragma unroll
      for (int a = 0; a < 64; ++a) acc[a] = 0.f;
      // weight chunks are software-pipelined one chunk ahead (raw bf16 in
      // registers); each token's chunk comes from shared memory as one
      // 16-byte load (lanes 16 bytes apart: conflict-free)
      uint4 wr[8];
      const int q_first = lane;
#pragma unroll
      for (int ee = 0; ee < 8; ++ee) {
        const int e = 8 * g + ee;
        wr[ee] = (e < E && q_first < nchunk)
                     ? __ldg(reinterpret_cast<const uint4*>(W + (size_t)e * H) + q_first)
                     : make_uint4(0, 0, 0, 0);
      }
      for (int j = 0; j < nj; ++j) {
        const int q = lane + 32 * j;  // this lane's chunk
        if (q >= nchunk) break;
        uint4 wn[8];
        const int qn = q + 32;
#pragma unroll
        for (int ee = 0; ee < 8; ++ee) {
          const int e = 8 * g + ee;
          wn[ee] = (e < E && qn < nchunk)
                       ? __ldg(reinterpret_cast<const uint4*>(W + (size_t)e * H) + qn)
                       : make_uint4(0, 0, 0, 0);
        }
        uint4 xr[8];
#pragma unroll
        for (int tt = 0; tt < 8; ++tt)
          xr[tt] = *reinterpret_cast<const uint4*>(xs + (size_t)tt * H + 8 * q);
#pragma unroll
        for (int el = 0; el < 8; ++el) {  // element 8 q + el of the chunk, ascending
          float xv[8], wv[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const uint32_t xw = word_of(xr[i], el >> 1), ww = word_of(wr[i], el >> 1);
            xv[i] = (el & 1) ? bf16_hi(xw) : bf16_lo(xw);
            wv[i] = (el & 1) ? bf16_hi(ww) : bf16_lo(ww);
          }
#pragma unroll
          for (int ee = 0; ee < 8; ++ee)
#pragma unroll
            for (int tp = 0; tp < 4; ++tp)
              fma2_rn(acc[ee * 8 + 2 * tp], acc[ee * 8 + 2 * tp + 1], xv[2 * tp], xv[2 * tp + 1],
                      wv[ee]);
        }
#pragma unroll
        for (int ee = 0; ee < 8; ++ee) wr[ee] = wn[ee];
      }
      // transpose-reduce: at offset o, the lane with bit o clear keeps the lower
      // half of its live entries and adds its partner's copy of them
#pragma unroll
      for (int o = 16, n = 64; o >= 1; o >>= 1, n >>= 1) {
        const bool upper = (lane & o) != 0;
#pragma unroll
        for (int a = 0; a < n / 2; ++a) {
          const float send = upper ? acc[a] : acc[a + n / 2];
          const float keep = upper ? acc[a + n / 2] : acc[a];
          acc[a] = __fadd_rn(keep, __shfl_xor_sync(0xffffffffu, send, o));
        }
      }
      // lane l now holds entries 2l, 2l + 1: expert l / 4, tokens 2 (l % 4) + {0, 1}
      const int e = 8 * g + (lane >> 2);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int tt = 2 * (lane & 3) + h;
        if (e < E) {
          const float v = bias ? __fadd_rn(acc[h], bias[e]) : acc[h];
          ls[tt * E + e] = v;
          if (tt < nt) logits[(size_t)(t0 + tt) * E + e] = v;
        }
      }
    }
    __syncthreads();
    if (warp < nt) {
      int id;
      float w;
      warp_topk(ls + warp * E, E, k, id, w);
      if (lane < k) {
        topk_id[(size_t)(t0 + warp) * k + lane] = id;
        topk_w[(size_t)(t0 + warp) * k + lane] = w;
      }
    }
    // the logits block and the x buffer are reused two tiles on
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
}

// ---------------------------------------------------------------------------
// Screened routing (large bf16 batches whose caller needs only the ids and
// gates).  The tensor cores give approximate logits a_e (bf16 products, fp32
// accumulation in the tensor core's order, K ranges added in order); their
// distance to the canonical fp32 logits l_e is at most eps = RS_EPS_REL *
// ||x_t|| * max_e ||W_r[e]|| (Cauchy-Schwarz bounds sum_h |x_h w_h| by the
// norms; RS_EPS_REL is several times a per-MMA-step bound of 2^-20 of that sum
// over H/16 steps, plus the canonical order's own 69 fp32 roundings).  If L is
// the k-th largest a_e, every expert of the exact top-k has a_e >= L - 2 eps
// (an expert with a_f > l_(k) + eps has l_f > l_(k), so at most k - 1 of them
// exceed l_(k) + eps, i.e. L <= l_(k) + eps; and a_e >= l_e - eps >= l_(k) - eps).
// So the canonical logits of the candidates {e : a_e >= L - 2 eps} decide the
// top-k exactly as all E logits would: the same warp top-k runs on them (the
// others are -inf) and gives the same ids, order and gates.  A token with more
// than RS_MAX_CAND candidates, or a non-finite value, takes all E exact logits.
// ---------------------------------------------------------------------------
constexpr float RS_EPS_REL = 1e-3f;
constexpr int RS_MAX_CAND = 32;
constexpr int RS_WARPS = 8;
constexpr int RS_U = 4;  // 16-byte weight chunks of a lane in flight per candidate (two candidates)

template <int EPL>
__global__ void __launch_bounds__(RS_WARPS * 32, 3)
k_router_screen(const float* __restrict__ part, int splits, int Epad,
                const __nv_bfloat16* __restrict__ x, const __nv_bfloat16* __restrict__ W,
                const float* __restrict__ bias, int T, int E, int H, float wmax, int k,
                int* __restrict__ topk_id, float* __restrict__ topk_w) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __nv_bfloat16* xs = reinterpret_cast<__nv_bfloat16*>(smem) + (size_t)warp * H;
  float* ls = reinterpret_cast<float*>(smem + (size_t)RS_WARPS * H * 2) + (size_t)warp * E;
  pdl_wait();
  const int t = blockIdx.x * RS_WARPS + warp;
  if (t >= T) return;
  // the token's row into shared memory, and ||x_t||^2
  const uint4* xr = reinterpret_cast<const uint4*>(x + (size_t)t * H);
  uint4* xw = reinterpret_cast<uint4*>(xs);
  float ss = 0.f;
  for (int i = lane; i < H / 8; i += 32) {
    const uint4 v = __ldg(xr + i);
    xw[i] = v;
    const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float a = __uint_as_float(w4[q] << 16), b = __uint_as_float(w4[q] & 0xFFFF0000u);
      ss = fmaf(a, a, ss);
      ss = fmaf(b, b, ss);
    }
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  // the approximate logits (K ranges in order, then the bias)
  float ap[EPL];
  bool finite = ss == ss && ss <= 3.0e38f;
#pragma unroll
  for (int i = 0; i < EPL; ++i) {
    const int e = lane + 32 * i;
    float v = 0.f;
    if (e < E) {
      for (int sp = 0; sp < splits; ++sp) v += part[((size_t)sp * T + t) * Epad + e];
      if (bias) v += bias[e];
      finite = finite && (v - v == 0.f);
      ls[e] = v;
    }
    ap[i] = v;
  }
  finite = __all_sync(0xffffffffu, finite);
  __syncwarp();
  unsigned cand[EPL];
  int ncand = E;
  if (finite) {
    // the k-th largest approximate logit
    int sid;
    float sw;
    warp_topk(ls, E, k, sid, sw);
    const float Lk = ls[__shfl_sync(0xffffffffu, sid, k - 1)];
    // both terms of the bound, with a margin for the fp32 norm itself
    const float eps = RS_EPS_REL * sqrtf(ss) * 1.001f * wmax;
    ncand = 0;
#pragma unroll
    for (int i = 0; i < EPL; ++i) {
      const int e = lane + 32 * i;
      cand[i] = __ballot_sync(0xffffffffu, e < E && ap[i] >= Lk - 2.f * eps);
      ncand += __popc(cand[i]);
    }
  }
  if (!finite || ncand > RS_MAX_CAND) {
#pragma unroll
    for (int i = 0; i < EPL; ++i) cand[i] = (lane + 32 * i) < E ? 0xffffffffu : 0u;
#pragma unroll
    for (int i = 0; i < EPL; ++i) cand[i] = __ballot_sync(0xffffffffu, lane + 32 * i < E);
  }
  __syncwarp();
  // non-candidates can never be selected
#pragma unroll
  for (int i = 0; i < EPL; ++i) {
    const int e = lane + 32 * i;
    if (e < E && !((cand[i] >> lane) & 1u)) ls[e] = -INFINITY;
  }
  __syncwarp();
  // canonical fp32 logits of the candidates: lane j accumulates the 8-element
  // chunks q = j, j + 32, ... of the dot product with fused multiply-adds in
  // ascending order; the lane partials are added at offsets 16, 8, 4, 2, 1
  // (lane j, j < off, adds lane j + off's); the bias last
  // Two candidates at a time (two independent chains sharing the x loads).
  const int nchunk = H / 8;
  auto pop = [&]() {  // the next candidate (warp-uniform), -1 when none is left
    int e = -1;
#pragma unroll
    for (int i = 0; i < EPL; ++i)
      if (e < 0 && cand[i]) {
        e = 32 * i + __ffs(cand[i]) - 1;
        cand[i] &= cand[i] - 1;
      }
    return e;
  };
  for (int e0 = pop(); e0 >= 0; e0 = pop()) {
    const int e1 = pop();
    const uint4* w0 = reinterpret_cast<const uint4*>(W + (size_t)e0 * H);
    const uint4* w1 = reinterpret_cast<const uint4*>(W + (size_t)(e1 >= 0 ? e1 : e0) * H);
    float acc0 = 0.f, acc1 = 0.f;
    for (int q0 = lane; q0 < nchunk; q0 += 32 * RS_U) {
      uint4 wv0[RS_U], wv1[RS_U];
#pragma unroll
      for (int u = 0; u < RS_U; ++u) {
        const bool in = q0 + 32 * u < nchunk;
        wv0[u] = in ? __ldg(w0 + q0 + 32 * u) : make_uint4(0u, 0u, 0u, 0u);
        wv1[u] = in && e1 >= 0 ? __ldg(w1 + q0 + 32 * u) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < RS_U; ++u) {
        if (q0 + 32 * u >= nchunk) break;
        const uint4 xv = xw[q0 + 32 * u];
        acc0 = fma_bf16_pair(acc0, xv.x, wv0[u].x);
        acc1 = fma_bf16_pair(acc1, xv.x, wv1[u].x);
        acc0 = fma_bf16_pair(acc0, xv.y, wv0[u].y);
        acc1 = fma_bf16_pair(acc1, xv.y, wv1[u].y);
        acc0 = fma_bf16_pair(acc0, xv.z, wv0[u].z);
        acc1 = fma_bf16_pair(acc1, xv.z, wv1[u].z);
        acc0 = fma_bf16_pair(acc0, xv.w, wv0[u].w);
        acc1 = fma_bf16_pair(acc1, xv.w, wv1[u].w);
      }
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) {
      acc0 = __fadd_rn(acc0, __shfl_down_sync(0xffffffffu, acc0, off));
      acc1 = __fadd_rn(acc1, __shfl_down_sync(0xffffffffu, acc1, off));
    }
    if (lane == 0) {
      ls[e0] = bias ? __fadd_rn(acc0, bias[e0]) : acc0;
      if (e1 >= 0) ls[e1] = bias ? __fadd_rn(acc1, bias[e1]) : acc1;
    }
  }
  __syncwarp();
  int id;
  float w;
  warp_topk(ls, E, k, id, w);
  if (lane < k) {
    topk_id[(size_t)t * k + lane] = id;
    topk_w[(size_t)t * k + lane] = w;
  }
}

}  // namespace

bool router_is_tiled(const lx_layer* L, int T) {
  const int tiles = (T + RTT_TOK - 1) / RTT_TOK;
  return L->dtype == LX_BF16 && tiles >= L->num_sms && L->H % 8 == 0 &&
         2 * (size_t)RTT_TOK * L->H * 2 + (size_t)RTT_TOK * L->E * 4 <= 200 * 1024;
}

lx_status launch_router(lx_layer* L, const void* x, int T, int k, float* logits, int* topk_id,
                        float* topk_w, cudaStream_t s, bool need_logits) {
  if (reinterpret_cast<uintptr_t>(x) % 16)
    return fail(LX_ERR_ARG, "x must be 16-byte aligned");
  const int tiles = (T + RT_TOK - 1) / RT_TOK;
  if (!need_logits && L->router_screen && router_is_tiled(L, T)) {
    // screened: approximate logits on the tensor cores, then the candidates'
    // canonical logits and the top-k (the logits buffer is not written)
    CUtensorMap xm;
    std::memset(&xm, 0, sizeof(xm));
    if (!encode_bf16_2d(&xm, x, L->H, T, 64, 128))
      return fail(LX_ERR_CUDA, "cuTensorMapEncodeTiled(x) failed");
    const int Epad = router_epad(L);
    int splits = 1;
    LX_TRY(tc_splitk_gemm(L, xm, L->router_map, T, Epad, L->H, L->ws.rs_part, RS_MAX_SPLITS,
                          &splits, s, "router_screen"));
    const size_t smem = (size_t)RS_WARPS * ((size_t)L->H * 2 + (size_t)L->E * 4);
    if (smem > 200 * 1024) return fail(LX_ERR_SHAPE, "router screening rows exceed shared memory");
    const unsigned grid = (unsigned)((T + RS_WARPS - 1) / RS_WARPS);
    ProfScope ps(L, s, "router_select");
    if (L->E <= 128) {
      static bool done4[64] = {};
      LX_CUDA(smem_cap_once((const void*)k_router_screen<4>, 200 * 1024, L->device, done4));
      launch_k(L, k_router_screen<4>, grid, RS_WARPS * 32, smem, s, (const float*)L->ws.rs_part,
               splits, Epad, (const __nv_bfloat16*)x, (const __nv_bfloat16*)L->router_w,
               (const float*)L->router_bias, T, L->E, L->H, L->router_wmax, k, topk_id, topk_w);
    } else {
      static bool done8[64] = {};
      LX_CUDA(smem_cap_once((const void*)k_router_screen<8>, 200 * 1024, L->device, done8));
      launch_k(L, k_router_screen<8>, grid, RS_WARPS * 32, smem, s, (const float*)L->ws.rs_part,
               splits, Epad, (const __nv_bfloat16*)x, (const __nv_bfloat16*)L->router_w,
               (const float*)L->router_bias, T, L->E, L->H, L->router_wmax, k, topk_id, topk_w);
    }
    LX_CUDA(cudaGetLastError());
    return LX_OK;
  }
  if (router_is_tiled(L, T)) {
    // large batch: persistent register-tiled kernel
    const size_t smem2 = 2 * (size_t)RTT_TOK * L->H * 2 + (size_t)RTT_TOK * L->E * 4;
    static bool done_t[64] = {};
    LX_CUDA(smem_cap_once((const void*)k_router_tiled, 200 * 1024, L->device, done_t));
    ProfScope ps(L, s, "router");
    const int grid = std::min(tiles, L->num_sms);
    launch_k(L, k_router_tiled, grid, RTT_THREADS, smem2, s, (const __nv_bfloat16*)x,
             (const __nv_bfloat16*)L->router_w, L->router_bias, T, L->E, L->H, logits, k, topk_id,
             topk_w);
    LX_CUDA(cudaGetLastError());
    return LX_OK;
  }
  const size_t smem = std::max((size_t)RT_TOK * L->H * L->esz, (size_t)RT_TOK * L->E * 4);
  if (smem > 200 * 1024) return fail(LX_ERR_SHAPE, "router token tile exceeds shared memory");
  // few token tiles: slice the experts so the router matrix spreads over the SMs
  const int per_cta = tiles >= L->num_sms ? L->E : RT_THREADS / 32;
  const dim3 grid(tiles, (L->E + per_cta - 1) / per_cta);
  ProfScope ps(L, s, "router");
  static bool done_bf16[64] = {}, done_f32[64] = {};
  if (L->dtype == LX_BF16) {
    auto kern = k_router_logits<__nv_bfloat16>;
    LX_CUDA(smem_cap_once((const void*)kern, 200 * 1024, L->device, done_bf16));
    launch_k(L, kern, grid, RT_THREADS, smem, s, (const __nv_bfloat16*)x, (const __nv_bfloat16*)L->router_w,
                                        L->router_bias, T, L->E, L->H, per_cta, logits,
                                        L->ws.tile_cnt, k, topk_id, topk_w);
  } else {
    auto kern = k_router_logits<float>;
    LX_CUDA(smem_cap_once((const void*)kern, 200 * 1024, L->device, done_f32));
    launch_k(L, kern, grid, RT_THREADS, smem, s, (const float*)x, (const float*)L->router_w, L->router_bias,
                                        T, L->E, L->H, per_cta, logits, L->ws.tile_cnt, k,
                                        topk_id, topk_w);
  }
  LX_CUDA(cudaGetLastError());
  return LX_OK;
}

int router_tile_counters(int T) { return (T + RT_TOK - 1) / RT_TOK; }

}  // namespace lx
