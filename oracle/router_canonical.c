/*
 * Oracle: canonical fp32 router logits (test infrastructure, not product code).
 *
 * The paper's router is the unchanged top-k router of the MoE layer (Sec. 1,
 * Fig. 1; Sec. 3.2 Stage 1: compression only reads it).  Its logits are the
 * plain dot products  l[t,e] = sum_h x[t,h] * W_r[e,h]  (+ b[e]).  The paper
 * fixes no summation order, so this file fixes one ("canonical") order, which
 * the CUDA router also follows, so that the top-k decision is taken on the same
 * fp32 numbers on both sides:
 *
 *   - H is split into chunks of 8 consecutive elements; chunk q belongs to
 *     lane j = q mod 32.
 *   - lane j keeps one fp32 partial p[j] = 0 and, for its chunks in ascending
 *     order and the 8 elements of each chunk in ascending order, updates
 *     p[j] = fmaf(x[h], w[h], p[j])   (one correctly rounded fused multiply-add).
 *   - the 32 partials are combined pairwise: for off = 16, 8, 4, 2, 1 and every
 *     j < off,  p[j] = p[j] + p[j + off]   (fp32 adds).
 *   - the logit is p[0], plus b[e] (one fp32 add) when a bias is given.
 *
 * Inputs are fp32 or bf16 (bit patterns, widened exactly to fp32).
 * Build with -ffp-contract=off so that the compiler adds no fusion of its own.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

static float widen(const void* base, long i, int is_bf16) {
  if (is_bf16) {
    uint32_t u = ((uint32_t)((const uint16_t*)base)[i]) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
  }
  return ((const float*)base)[i];
}

/* H must be a multiple of 8.  out is [T, E] row-major. */
int oracle_router_logits(const void* x, const void* w, const float* bias, int is_bf16,
                         int T, int E, int H, float* out) {
  if (H % 8 != 0 || T < 0 || E <= 0) return 1;
  const int nchunk = H / 8;
  for (int t = 0; t < T; ++t) {
    for (int e = 0; e < E; ++e) {
      float p[32];
      for (int j = 0; j < 32; ++j) p[j] = 0.0f;
      for (int q = 0; q < nchunk; ++q) {
        const int j = q % 32;
        for (int i = 0; i < 8; ++i) {
          const long h = 8L * q + i;
          p[j] = fmaf(widen(x, (long)t * H + h, is_bf16), widen(w, (long)e * H + h, is_bf16), p[j]);
        }
      }
      for (int off = 16; off >= 1; off /= 2)
        for (int j = 0; j < off; ++j) p[j] = p[j] + p[j + off];
      float l = p[0];
      if (bias) l = l + bias[e];
      out[(long)t * E + e] = l;
    }
  }
  return 0;
}
