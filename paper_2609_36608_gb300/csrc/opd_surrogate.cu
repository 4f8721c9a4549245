// Per-token work of token scoring and of the sampled-token surrogate
// (ActFirst-OPD Appendix B.4), one warp per token row:
//
//   lse_i  = (M + log2 S) ln 2 from the per-split base-2 statistics of the
//            single-head fused forward (M = max of split maxima, S = rescaled sum)
//   z_x    = H[i,:] . W[x_i,:]           the sampled token's logit (fp32 dot product)
//   logp_i = z_x / tau - lse_i
//
// and, for the surrogate (Eq. opd-token-advantage, opd-ratio, opd-dual-clip):
//   A_i   = logp_teacher_i - logp_old_i                  (a constant: stop-gradient)
//   rho_i = exp(clip(logp_i - logp_old_i, -c, c))
//   l_clip = -min(rho A, clip(rho, 1 - delta, 1 + delta) A)
//   l_DC  = min(l_clip, -kappa A) if A < 0 else l_clip
//   coef_i = w_i (d l_DC / d logp_i) / tau,  so that the backward emits
//   dz_i[k] = coef_i (1[k = x_i] - p_i[k]); rowc carries coef_i (1 - p_i[x_i]) for the
//   token's column, with p_i[x_i] = exp(logp_i).
#include <math_constants.h>

#include "opd_device.cuh"
#include "opd_internal.h"

namespace opd {

namespace {

__device__ __forceinline__ void merge_stats(float& m, float& s, float m2, float s2) {
  const float M = fmaxf(m, m2);
  if (M == -CUDART_INF_F) return;
  s = s * exp2f(m - M) + s2 * exp2f(m2 - M);
  m = M;
}

// Dual-clip PPO loss of one token and its slope with respect to logp (the paper's
// definitions; the unclipped product is active when rho A <= clip(rho) A, and the
// dual clip when l_clip > -kappa A).
__device__ __forceinline__ void dual_clip(float logp, float logp_old, float A, float delta, float kappa, float c,
                                          float& loss, float& slope) {
  const float r = logp - logp_old;
  const float rc = fminf(fmaxf(r, -c), c);
  const float rho = expf(rc);
  const float drho = (r > -c && r < c) ? rho : 0.f;
  const float lo = 1.f - delta, hi = 1.f + delta;
  const float rho_c = fminf(fmaxf(rho, lo), hi);
  const float mu = rho * A, mc = rho_c * A;
  float l, dl;
  if (mu <= mc) {
    l = -mu;
    dl = -A;
  } else {
    l = -mc;
    dl = (rho > lo && rho < hi) ? -A : 0.f;
  }
  if (A < 0.f) {
    const float floor_value = -kappa * A;
    if (l > floor_value) {
      l = floor_value;
      dl = 0.f;
    }
  }
  loss = l;
  slope = dl * drho;
}

__global__ void k_head_rows(const HeadRowsParams p) {
  const int lane = threadIdx.x & 31;
  const int warps = (gridDim.x * blockDim.x) >> 5;
  const int R = p.ctrl->R;
  const int n_vs = p.ctrl->n_vsplit;
  const int h0 = p.ctrl->half_tile - 1;  // first row of a half-height tile, or -1
  const size_t plane = (size_t)p.T_pad;
  for (int i = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; i < p.T; i += warps) {
    const int r = p.pos[i];
    if (r < 0) {
      if (lane == 0) {
        if (p.lse_out) p.lse_out[i] = 0.f;
        if (p.logp_out) p.logp_out[i] = 0.f;
        if (p.loss_out) p.loss_out[i] = 0.f;
      }
      continue;
    }
    float m = -CUDART_INF_F, s = 0.f;
    // in a half-height tile, columns 128-255 of each split are a second partial at row r + 128
    const bool two = h0 >= 0 && r >= h0 && r < h0 + 128;
    for (int j = lane; j < n_vs; j += 32) {
      const float* b = p.partials + (size_t)j * 5 * plane + r;
      merge_stats(m, s, b[0], b[plane]);
      if (two) merge_stats(m, s, b[128], b[plane + 128]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
      const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
      merge_stats(m, s, m2, s2);
    }
    const float lse = (m + log2f(s)) * 0.69314718055994531f;

    int x = p.tokens[i];
    const bool x_ok = x >= 0 && x < p.V;
    if (!x_ok) {
      if (lane == 0) atomicOr(&p.ctrl_rw->status, kDevBadToken);
      x = 0;
    }
    // z_x: 16-byte chunks of the gathered row and of W's row x, summed across the warp
    const uint4* hrow = reinterpret_cast<const uint4*>(p.H_g + (size_t)r * p.d);
    const uint4* wrow = reinterpret_cast<const uint4*>(p.W + (size_t)x * p.d);
    float acc = 0.f;
    for (int c = lane; c < p.d / 8; c += 32) {
      const uint4 a = hrow[c], b = wrow[c];
      const __nv_bfloat162* a2 = reinterpret_cast<const __nv_bfloat162*>(&a);
      const __nv_bfloat162* b2 = reinterpret_cast<const __nv_bfloat162*>(&b);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 fa = __bfloat1622float2(a2[e]);
        const float2 fb = __bfloat1622float2(b2[e]);
        acc = fmaf(fa.x, fb.x, acc);
        acc = fmaf(fa.y, fb.y, acc);
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    const float logp = x_ok ? acc * p.inv_tau - lse : 0.f;

    if (lane == 0) {
      if (p.lse_out) p.lse_out[i] = lse;
      if (p.logp_out) p.logp_out[i] = logp;
      if (p.surrogate) {
        const float A = p.logp_teacher[i] - p.logp_old[i];
        float loss = 0.f, slope = 0.f;
        if (x_ok) dual_clip(logp, p.logp_old[i], A, p.delta, p.kappa, p.clip, loss, slope);
        p.loss_out[i] = loss;
        const float coef = p.weights[i] * slope * p.inv_tau;
        // the backward writes -coef p everywhere and this value, coef (1 - p_x), at the token
        const float at_token = x_ok ? coef * (1.0f - expf(logp)) : 0.f;
        p.rowc[r] = make_float4(lse * 1.4426950408889634f, coef, __int_as_float(x), at_token);
      }
    }
  }
  // rows past R in the last tile: zero constants (no gradient)
  if (p.surrogate) {
    const int R_pad = (R + kRowPad - 1) / kRowPad * kRowPad;
    for (int r = R + blockIdx.x * blockDim.x + threadIdx.x; r < R_pad; r += gridDim.x * blockDim.x)
      p.rowc[r] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
}

}  // namespace

cudaError_t launch_head_rows(const HeadRowsParams& p, int n_sm, cudaStream_t s) {
  long blocks = ((long)p.T * 32 + 255) / 256;
  const long cap = (long)n_sm * 16;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  k_head_rows<<<(int)blocks, 256, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace opd
