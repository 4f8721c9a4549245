// float32 path on CUDA cores (fp32 FMA), for float32 inputs, where bf16 tensor
// cores do not apply. Same quantities as the tensor-core path (Section 3,
// Eq. reverse-kl; gradient with respect to H_s and W_s; frozen teacher), computed
// row by row: one CTA streams the vocabulary of one token context with online
// max / sum statistics, then the gradient rows and dW_s columns are plain dot
// products over the fp32 dz buffer.
#include <math_constants.h>

#include "opd_device.cuh"
#include "opd_internal.h"

namespace opd {

namespace {

constexpr int kThreads = 256;

struct Stats5 {
  float ms, Ss, A, mt, St;  // natural-log units: S = sum e^(u - m), A = sum e^(u_s - m_s)(u_s - u_t)
};

__device__ __forceinline__ Stats5 merge(const Stats5& a, const Stats5& b) {
  Stats5 r;
  r.ms = fmaxf(a.ms, b.ms);
  const float fa = a.ms == -CUDART_INF_F ? 0.f : expf(a.ms - r.ms);
  const float fb = b.ms == -CUDART_INF_F ? 0.f : expf(b.ms - r.ms);
  r.Ss = a.Ss * fa + b.Ss * fb;
  r.A = a.A * fa + b.A * fb;
  r.mt = fmaxf(a.mt, b.mt);
  const float ga = a.mt == -CUDART_INF_F ? 0.f : expf(a.mt - r.mt);
  const float gb = b.mt == -CUDART_INF_F ? 0.f : expf(b.mt - r.mt);
  r.St = a.St * ga + b.St * gb;
  return r;
}

__device__ __forceinline__ float dot(const float* __restrict__ a, const float* __restrict__ b, int d) {
  float acc = 0.f;
  for (int j = 0; j < d; ++j) acc = fmaf(a[j], b[j], acc);
  return acc;
}

// One CTA per token row i of the T rows.
__global__ void __launch_bounds__(kThreads)
    k_simt_forward(const float* __restrict__ Hs, const float* __restrict__ Ht, const float* __restrict__ Ws,
                   const float* __restrict__ Wt, int d_s, int d_t, int V, float inv_tau,
                   const int32_t* __restrict__ pos, float* __restrict__ kl_out, float* __restrict__ stats) {
  const int i = blockIdx.x;
  if (pos[i] < 0) {
    if (threadIdx.x == 0) {
      kl_out[i] = 0.f;
      stats[3 * (size_t)i] = stats[3 * (size_t)i + 1] = stats[3 * (size_t)i + 2] = 0.f;
    }
    return;
  }
  const float* hs = Hs + (size_t)i * d_s;
  const float* ht = Ht + (size_t)i * d_t;
  Stats5 st{-CUDART_INF_F, 0.f, 0.f, -CUDART_INF_F, 0.f};
  for (int k = threadIdx.x; k < V; k += kThreads) {
    const float us = dot(hs, Ws + (size_t)k * d_s, d_s) * inv_tau;
    const float ut = dot(ht, Wt + (size_t)k * d_t, d_t) * inv_tau;
    Stats5 one{us, 1.f, us - ut, ut, 1.f};
    st = merge(st, one);
  }
  __shared__ Stats5 red[kThreads];
  red[threadIdx.x] = st;
  __syncthreads();
  for (int o = kThreads / 2; o > 0; o >>= 1) {
    if (threadIdx.x < o) red[threadIdx.x] = merge(red[threadIdx.x], red[threadIdx.x + o]);
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const Stats5 s = red[0];
    const float lse_s = s.ms + logf(s.Ss);
    const float lse_t = s.mt + logf(s.St);
    const float kl = s.A / s.Ss - lse_s + lse_t;
    kl_out[i] = kl;
    stats[3 * (size_t)i] = lse_s;
    stats[3 * (size_t)i + 1] = lse_t;
    stats[3 * (size_t)i + 2] = kl;
  }
}

// dz[r, k] = (g_i / tau) p_s[k] (u_s[k] - u_t[k] - (lse_s - lse_t + KL)), r = rank of row i.
__global__ void __launch_bounds__(kThreads)
    k_simt_dz(const float* __restrict__ Hs, const float* __restrict__ Ht, const float* __restrict__ Ws,
              const float* __restrict__ Wt, int d_s, int d_t, int V, float inv_tau, const int32_t* __restrict__ pos,
              const float* __restrict__ stats, const float* __restrict__ grad_kl, float* __restrict__ dZ) {
  const int i = blockIdx.x;
  const int r = pos[i];
  if (r < 0) return;
  const float lse_s = stats[3 * (size_t)i], lse_t = stats[3 * (size_t)i + 1], kl = stats[3 * (size_t)i + 2];
  const float c = lse_s - lse_t + kl;
  const float coef = grad_kl[i] * inv_tau;
  const float* hs = Hs + (size_t)i * d_s;
  const float* ht = Ht + (size_t)i * d_t;
  for (int k = threadIdx.x; k < V; k += kThreads) {
    const float us = dot(hs, Ws + (size_t)k * d_s, d_s) * inv_tau;
    const float ut = dot(ht, Wt + (size_t)k * d_t, d_t) * inv_tau;
    dZ[(size_t)r * V + k] = coef * expf(us - lse_s) * (us - ut - c);
  }
}

// dH_s[i, :] = dz[r, :] W_s (zero for unsupervised rows).
__global__ void __launch_bounds__(kThreads)
    k_simt_dH(const float* __restrict__ dZ, const float* __restrict__ Ws, int d_s, int V,
              const int32_t* __restrict__ pos, float* __restrict__ dH) {
  const int i = blockIdx.x;
  const int r = pos[i];
  for (int j = threadIdx.x; j < d_s; j += kThreads) {
    float acc = 0.f;
    if (r >= 0)
      for (int k = 0; k < V; ++k) acc = fmaf(dZ[(size_t)r * V + k], Ws[(size_t)k * d_s + j], acc);
    dH[(size_t)i * d_s + j] = acc;
  }
}

// dW_s[k, j] (+)= sum_r dz[r, k] H_s[idx[r], j].
__global__ void __launch_bounds__(kThreads)
    k_simt_dW(const float* __restrict__ dZ, const float* __restrict__ Hs, int d_s, int V,
              const int32_t* __restrict__ idx, const Ctrl* __restrict__ ctrl, int accumulate, float* __restrict__ dW) {
  const int R = ctrl->R;
  const long total = (long)V * d_s;
  for (long e = blockIdx.x * (long)kThreads + threadIdx.x; e < total; e += (long)gridDim.x * kThreads) {
    const int k = (int)(e / d_s);
    const int j = (int)(e - (long)k * d_s);
    float acc = 0.f;
    for (int r = 0; r < R; ++r) acc = fmaf(dZ[(size_t)r * V + k], Hs[(size_t)idx[r] * d_s + j], acc);
    dW[e] = accumulate ? dW[e] + acc : acc;
  }
}

}  // namespace

cudaError_t launch_simt_forward(const float* H_s, const float* H_t, const float* W_s, const float* W_t,
                                int32_t T, int32_t d_s, int32_t d_t, int32_t V, float tau, const int32_t* idx,
                                const int32_t* pos, const Ctrl* ctrl, float* kl_out, float* stats,
                                cudaStream_t s) {
  (void)idx;
  (void)ctrl;
  if (T == 0) return cudaSuccess;
  k_simt_forward<<<T, kThreads, 0, s>>>(H_s, H_t, W_s, W_t, d_s, d_t, V, 1.0f / tau, pos, kl_out, stats);
  return cudaGetLastError();
}

cudaError_t launch_simt_backward(const float* H_s, const float* H_t, const float* W_s, const float* W_t,
                                 int32_t T, int32_t d_s, int32_t d_t, int32_t V, float tau, const int32_t* idx,
                                 const int32_t* pos, const Ctrl* ctrl, const float* stats, const float* grad_kl,
                                 float* dZ, float* dH_s, float* dW_s, int accumulate_dW, cudaStream_t s) {
  const float inv_tau = 1.0f / tau;
  if (T > 0) {
    k_simt_dz<<<T, kThreads, 0, s>>>(H_s, H_t, W_s, W_t, d_s, d_t, V, inv_tau, pos, stats, grad_kl, dZ);
    k_simt_dH<<<T, kThreads, 0, s>>>(dZ, W_s, d_s, V, pos, dH_s);
  }
  long blocks = ((long)V * d_s + kThreads - 1) / kThreads;
  if (blocks > 4096) blocks = 4096;
  k_simt_dW<<<(int)blocks, kThreads, 0, s>>>(dZ, H_s, d_s, V, idx, ctrl, accumulate_dW, dW_s);
  return cudaGetLastError();
}

}  // namespace opd
