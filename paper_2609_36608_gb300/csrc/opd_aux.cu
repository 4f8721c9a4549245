// Memory-bound steps around the tensor-core kernels:
//   compaction  mask[T] -> idx[R] (supervised rows in order), pos[T] (rank or -1)
//               (Appendix B.4: m = 1 on model-generated response tokens only)
//   gather      H_s, H_t rows -> contiguous [R_pad, d] bf16 buffers, zero rows R..R_pad-1
//   combine     per-split statistics -> lse_s, lse_t, KL per token (Eq. reverse-kl)
//   bwd_rowc    per-row constants of dz = (g/tau) p_s (log p_s - log p_t - KL)
//   zero_rows / scatter_rows   dH_s partial-sum buffer, then back to the T rows
#include <math_constants.h>

#include "opd_device.cuh"
#include "opd_internal.h"

namespace opd {

namespace {

constexpr int kCompactThreads = 1024;
constexpr int kCompactPer = 16;  // mask bytes per thread and pass (one 16-byte load when aligned)

// One CTA walks the mask in passes of kCompactThreads x 16 rows: each thread takes 16
// consecutive rows, a block-wide exclusive scan of the per-thread counts gives each
// thread its output offset, and a running total carries the offset to the next pass.
// Loads are coalesced (16-byte vectors when the mask is 16-byte aligned, bytes
// otherwise) and pos is written four rows per 16-byte store.
__global__ void __launch_bounds__(kCompactThreads)
    k_compact(const uint8_t* __restrict__ mask, int32_t T, int32_t* __restrict__ idx, int32_t* __restrict__ pos,
              Ctrl* ctrl) {
  __shared__ int32_t warp_tot[32];
  const int tid = threadIdx.x;
  const int lane = tid & 31, w = tid >> 5;
  if (tid == 0) ctrl->status = 0u;
  if (tid < 4) ctrl->work[tid] = 0;
  const bool vec = (reinterpret_cast<uintptr_t>(mask) & 15u) == 0;
  int carry = 0;  // supervised rows before this pass
  for (int base = 0; base < T; base += kCompactThreads * kCompactPer) {
    const int lo = base + tid * kCompactPer;
    uint32_t bits = 0;  // bit j: row lo + j is supervised
    if (vec && lo + kCompactPer <= T) {
      const uint4 v = *reinterpret_cast<const uint4*>(mask + lo);
      const uint32_t wv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int j = 0; j < kCompactPer; ++j) bits |= (((wv[j >> 2] >> (8 * (j & 3))) & 0xFFu) != 0u ? 1u : 0u) << j;
    } else {
#pragma unroll
      for (int j = 0; j < kCompactPer; ++j)
        if (lo + j < T && mask[lo + j] != 0) bits |= 1u << j;
    }
    const int cnt = __popc(bits);
    // inclusive warp scan, then scan of the warp totals
    int x = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    __syncthreads();  // warp_tot of the previous pass has been read
    if (lane == 31) warp_tot[w] = x;
    __syncthreads();
    if (w == 0) {
      int t = warp_tot[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, t, o);
        if (lane >= o) t += y;
      }
      warp_tot[lane] = t;  // inclusive totals
    }
    __syncthreads();
    int off = carry + x - cnt + (w > 0 ? warp_tot[w - 1] : 0);
    int pv[kCompactPer];
#pragma unroll
    for (int j = 0; j < kCompactPer; ++j) {
      if ((bits >> j) & 1u) {
        idx[off] = lo + j;
        pv[j] = off++;
      } else {
        pv[j] = -1;
      }
    }
    if (lo + kCompactPer <= T) {  // pos is 16-byte aligned (workspace) and lo a multiple of 16
#pragma unroll
      for (int j = 0; j < kCompactPer; j += 4)
        *reinterpret_cast<int4*>(pos + lo + j) = make_int4(pv[j], pv[j + 1], pv[j + 2], pv[j + 3]);
    } else {
      for (int j = 0; j < kCompactPer && lo + j < T; ++j) pos[lo + j] = pv[j];
    }
    carry += warp_tot[31];
  }
  if (tid == 0) {
    ctrl->R = carry;
    ctrl->n_vsplit = 0;
    ctrl->half_tile = 0;
  }
}

// Row gather in 16-byte vectors; rows in [R, R_pad) become zero. One block per
// gathered row at a time (no per-element division); each thread loads up to
// kGatherVec vectors of the row (H_s part, then H_t part) before storing them.
constexpr int kGatherVec = 4;

__global__ void __launch_bounds__(256) k_gather2(const uint4* __restrict__ Hs, const uint4* __restrict__ Ht,
                                                 int32_t vs, int32_t vt, const int32_t* __restrict__ idx,
                                                 const Ctrl* __restrict__ ctrl, uint4* __restrict__ Hs_g,
                                                 uint4* __restrict__ Ht_g) {
  const int R = ctrl->R;
  const int R_pad = (R + kRowPad - 1) / kRowPad * kRowPad;
  const int per_row = vs + vt;
  for (int r = blockIdx.x; r < R_pad; r += gridDim.x) {
    const bool live = r < R;
    const long src = live ? (long)idx[r] : 0;
    for (int v0 = 0; v0 < per_row; v0 += kGatherVec * blockDim.x) {
      uint4 x[kGatherVec];
#pragma unroll
      for (int k = 0; k < kGatherVec; ++k) {
        const int v = v0 + k * blockDim.x + threadIdx.x;
        x[k] = make_uint4(0u, 0u, 0u, 0u);
        if (live && v < per_row) x[k] = v < vs ? Hs[src * vs + v] : Ht[src * vt + (v - vs)];
      }
#pragma unroll
      for (int k = 0; k < kGatherVec; ++k) {
        const int v = v0 + k * blockDim.x + threadIdx.x;
        if (v < vs)
          Hs_g[(long)r * vs + v] = x[k];
        else if (v < per_row)
          Ht_g[(long)r * vt + (v - vs)] = x[k];
      }
    }
  }
}

// Merge the base-2 statistics of every vocabulary split of one row:
//   M = max_j m_j,  S = sum_j S_j 2^(m_j - M),  A likewise
// then  lse = (M + log2 S) ln 2,  KL = (A_s / S_s) ln 2 - lse_s + lse_t.
// Merge of two base-2 partial statistics (max M, sum S at M, A at M for the student;
// the teacher's max and sum) into the first.
__device__ __forceinline__ void merge_partial(float& ms, float& ss, float& as, float& mt, float& st, float ms2,
                                              float ss2, float as2, float mt2, float st2) {
  const float Ms = fmaxf(ms, ms2), Mt = fmaxf(mt, mt2);
  const float f1 = ms == -CUDART_INF_F ? 0.f : exp2f(ms - Ms), f2 = ms2 == -CUDART_INF_F ? 0.f : exp2f(ms2 - Ms);
  const float g1 = mt == -CUDART_INF_F ? 0.f : exp2f(mt - Mt), g2 = mt2 == -CUDART_INF_F ? 0.f : exp2f(mt2 - Mt);
  ss = ss * f1 + ss2 * f2;
  as = as * f1 + as2 * f2;
  st = st * g1 + st2 * g2;
  ms = Ms;
  mt = Mt;
}

// Rows in blocks of 32 consecutive gathered rows, four warps per block: warp g takes the
// vocabulary splits g, g + 4, ... of all 32 rows, so each load reads 32 consecutive floats of
// one statistics plane (the partials are laid out [split][5][row]). The four running merges
// meet in shared memory and warp 0 finishes the rows. idx maps a gathered row to its token
// row (NULL: the identity, for schedules over every token row); pos[i] != r marks a row that
// was computed but is not supervised. With weights, sum_i weights[i] KL_i is added to
// *loss_acc. Rows outside the supervised set get zeros.
constexpr int kCombineGroups = 4;
__global__ void __launch_bounds__(32 * kCombineGroups)
    k_combine(const float* __restrict__ part, const int32_t* __restrict__ pos, const int32_t* __restrict__ idx,
              const Ctrl* __restrict__ ctrl, int32_t T, int32_t T_pad, float* __restrict__ kl_out,
              float* __restrict__ stats, const float* __restrict__ weights, double* loss_acc) {
  __shared__ float sh[kCombineGroups - 1][5][32];
  const int R = ctrl->R;
  const int n_vs = ctrl->n_vsplit;
  const int h0 = ctrl->half_tile - 1;  // first row of a half-height tile, or -1
  const size_t plane = (size_t)T_pad;
  const int lane = threadIdx.x & 31;
  const int g = threadIdx.x >> 5;
  double wkl = 0.0;  // warp 0's share of sum_i w_i KL_i
  const int n_row_blocks = (R + 31) / 32;
  for (int rb = blockIdx.x; rb < n_row_blocks; rb += gridDim.x) {
    const int r = rb * 32 + lane;
    float ms = -CUDART_INF_F, ss = 0.f, as = 0.f, mt = -CUDART_INF_F, st = 0.f;
    if (r < R) {
      // in a half-height tile, columns 128-255 of each split are a second partial at row r + 128
      const bool two = h0 >= 0 && r >= h0 && r < h0 + 128;
#pragma unroll 4
      for (int j = g; j < n_vs; j += kCombineGroups) {
        const float* b = part + (size_t)j * 5 * plane + r;
        merge_partial(ms, ss, as, mt, st, b[0], b[plane], b[2 * plane], b[3 * plane], b[4 * plane]);
        if (two)
          merge_partial(ms, ss, as, mt, st, b[128], b[plane + 128], b[2 * plane + 128], b[3 * plane + 128],
                        b[4 * plane + 128]);
      }
    }
    if (g > 0) {
      sh[g - 1][0][lane] = ms;
      sh[g - 1][1][lane] = ss;
      sh[g - 1][2][lane] = as;
      sh[g - 1][3][lane] = mt;
      sh[g - 1][4][lane] = st;
    }
    __syncthreads();
    if (g == 0 && r < R) {
#pragma unroll
      for (int k = 0; k < kCombineGroups - 1; ++k)
        merge_partial(ms, ss, as, mt, st, sh[k][0][lane], sh[k][1][lane], sh[k][2][lane], sh[k][3][lane],
                      sh[k][4][lane]);
      const int i = idx ? idx[r] : r;
      if (i >= 0 && i < T && pos[i] == r) {
        float lse_s = 0.f, lse_t = 0.f, kl = 0.f;
        if (n_vs > 0) {
          const float ln2 = 0.69314718055994531f;
          lse_s = (ms + log2f(ss)) * ln2;
          lse_t = (mt + log2f(st)) * ln2;
          kl = (as / ss) * ln2 - lse_s + lse_t;
        }
        kl_out[i] = kl;
        stats[3 * (size_t)i + 0] = lse_s;
        stats[3 * (size_t)i + 1] = lse_t;
        stats[3 * (size_t)i + 2] = kl;
        if (weights) wkl += (double)weights[i] * (double)kl;
      }
    }
    __syncthreads();  // sh is rewritten by the next row block
  }
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < T; i += gridDim.x * blockDim.x) {
    if (pos[i] >= 0) continue;
    kl_out[i] = 0.f;
    stats[3 * (size_t)i + 0] = 0.f;
    stats[3 * (size_t)i + 1] = 0.f;
    stats[3 * (size_t)i + 2] = 0.f;
  }
  if (weights && g == 0) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) wkl += __shfl_xor_sync(0xffffffffu, wkl, o);
    if (lane == 0 && wkl != 0.0) atomicAdd(loss_acc, wkl);
  }
}

__global__ void k_bwd_rowc(const float* __restrict__ stats, const float* __restrict__ grad_kl,
                           const int32_t* __restrict__ idx, const Ctrl* __restrict__ ctrl, int32_t T_pad, float tau,
                           float4* __restrict__ rowc) {
  const int R = ctrl->R;
  const int R_pad = (R + kRowPad - 1) / kRowPad * kRowPad;
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < R_pad; r += gridDim.x * blockDim.x) {
    float4 c = make_float4(0.f, 0.f, 0.f, 0.f);
    if (r < R) {
      const int i = idx[r];
      const float lse_s = stats[3 * (size_t)i + 0];
      const float lse_t = stats[3 * (size_t)i + 1];
      const float kl = stats[3 * (size_t)i + 2];
      c.x = lse_s * 1.4426950408889634f;
      c.y = lse_s - lse_t + kl;
      c.z = grad_kl[i] / tau;
    }
    rowc[r] = c;
  }
}

__global__ void k_zero_rows(float4* __restrict__ buf, int32_t vec_per_row, const Ctrl* __restrict__ ctrl) {
  const int R = ctrl->R;
  const int R_pad = (R + kRowPad - 1) / kRowPad * kRowPad;
  const long total = (long)R_pad * vec_per_row;
  for (long e = blockIdx.x * (long)blockDim.x + threadIdx.x; e < total; e += (long)gridDim.x * blockDim.x)
    buf[e] = make_float4(0.f, 0.f, 0.f, 0.f);
}

// One block per token row at a time (no per-element division); each thread moves
// up to kScatterVec 16-byte vectors of the row, all loads issued before the stores.
constexpr int kScatterVec = 4;

__global__ void __launch_bounds__(256) k_scatter_rows(const float4* __restrict__ src, int32_t vec_per_row,
                                                      const int32_t* __restrict__ pos, int32_t T,
                                                      float4* __restrict__ dst) {
  for (int i = blockIdx.x; i < T; i += gridDim.x) {
    const int r = pos[i];
    const float4* s = src + (long)(r >= 0 ? r : 0) * vec_per_row;
    float4* d = dst + (long)i * vec_per_row;
    for (int v0 = 0; v0 < vec_per_row; v0 += kScatterVec * blockDim.x) {
      float4 x[kScatterVec];
#pragma unroll
      for (int k = 0; k < kScatterVec; ++k) {
        const int v = v0 + k * blockDim.x + threadIdx.x;
        x[k] = (r >= 0 && v < vec_per_row) ? s[v] : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int k = 0; k < kScatterVec; ++k) {
        const int v = v0 + k * blockDim.x + threadIdx.x;
        if (v < vec_per_row) d[v] = x[k];
      }
    }
  }
}

// Waits on an mbarrier that nothing will ever complete, to exercise the bounded
// wait: it must give up after limit_ns, flag kDevTimeout and return.
__global__ void k_selftest_timeout(Ctrl* ctrl, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    ctrl->status = 0u;
    mbar_wait(&bar, 0u, &ctrl->status, limit_ns);
  }
}

int grid_for(long work, int n_sm, int threads) {
  long g = (work + threads - 1) / threads;
  const long cap = (long)n_sm * 8;
  if (g > cap) g = cap;
  return (int)(g < 1 ? 1 : g);
}

}  // namespace

cudaError_t launch_compact(const uint8_t* mask, int32_t T, int32_t* idx, int32_t* pos, Ctrl* ctrl,
                           cudaStream_t s) {
  k_compact<<<1, kCompactThreads, 0, s>>>(mask, T, idx, pos, ctrl);
  return cudaGetLastError();
}

cudaError_t launch_gather_bf16(const void* H_s, const void* H_t, int32_t d_s, int32_t d_t, const int32_t* idx,
                               const Ctrl* ctrl, void* Hs_g, void* Ht_g, int32_t T_pad, int n_sm, cudaStream_t s) {
  const int vs = d_s / 8, vt = d_t / 8;  // 8 bf16 per 16-byte vector
  // rows are walked by blocks; R is known only on the device, so the grid covers T_pad rows
  const long blocks = (long)T_pad < (long)n_sm * 8 ? (long)T_pad : (long)n_sm * 8;
  k_gather2<<<(int)(blocks < 1 ? 1 : blocks), 256, 0, s>>>(
      static_cast<const uint4*>(H_s), static_cast<const uint4*>(H_t), vs, vt, idx, ctrl,
      static_cast<uint4*>(Hs_g), static_cast<uint4*>(Ht_g));
  return cudaGetLastError();
}

cudaError_t launch_combine(const float* partials, const int32_t* pos, const int32_t* idx, const Ctrl* ctrl,
                           int32_t T, int32_t T_pad, float* kl_out, float* stats, const float* weights,
                           double* loss_acc, int n_sm, cudaStream_t s) {
  // one block per 32 rows of T (an upper bound on the supervised rows), at most 8 per SM
  long blocks = ((long)T + 31) / 32;
  if (blocks > (long)n_sm * 8) blocks = (long)n_sm * 8;
  k_combine<<<(int)(blocks < 1 ? 1 : blocks), 32 * kCombineGroups, 0, s>>>(partials, pos, idx, ctrl, T, T_pad,
                                                                           kl_out, stats, weights, loss_acc);
  return cudaGetLastError();
}

cudaError_t launch_bwd_rowc(const float* stats, const float* grad_kl, const int32_t* idx, const Ctrl* ctrl,
                            int32_t T_pad, float tau, float4* rowc, cudaStream_t s) {
  k_bwd_rowc<<<(T_pad + 255) / 256, 256, 0, s>>>(stats, grad_kl, idx, ctrl, T_pad, tau, rowc);
  return cudaGetLastError();
}

cudaError_t launch_zero_rows(float* buf, int32_t cols, const Ctrl* ctrl, int32_t T_pad, int n_sm, cudaStream_t s) {
  k_zero_rows<<<grid_for((long)T_pad * cols / 4, n_sm, 256), 256, 0, s>>>(reinterpret_cast<float4*>(buf), cols / 4,
                                                                           ctrl);
  return cudaGetLastError();
}

cudaError_t launch_scatter_rows(const float* src_g, int32_t cols, const int32_t* pos, int32_t T, float* dst,
                                int n_sm, cudaStream_t s) {
  // blocks of 128 threads when a row has at most 512 vectors (d_s <= 2048), so each thread
  // keeps four vectors in flight; 8 blocks per SM, at most one per row
  const int vpr = cols / 4;
  const int threads = vpr <= 512 ? 128 : 256;
  const long blocks = T < (long)n_sm * 8 ? T : (long)n_sm * 8;
  k_scatter_rows<<<(int)(blocks < 1 ? 1 : blocks), threads, 0, s>>>(
      reinterpret_cast<const float4*>(src_g), vpr, pos, T, reinterpret_cast<float4*>(dst));
  return cudaGetLastError();
}

// Debug check of an output buffer: any NaN or infinity sets kDevNonFinite.
__global__ void k_check_finite(const float* __restrict__ p, size_t n, uint32_t* status) {
  bool bad = false;
  for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x)
    bad |= !isfinite(p[i]);
  if (__any_sync(0xffffffffu, bad) && (threadIdx.x & 31) == 0) atomicOr(status, kDevNonFinite);
}

cudaError_t launch_check_finite(const float* p, size_t n, Ctrl* ctrl, int n_sm, cudaStream_t s) {
  if (!p || n == 0) return cudaSuccess;
  k_check_finite<<<grid_for((long)((n + 3) / 4), n_sm, 256), 256, 0, s>>>(p, n, &ctrl->status);
  return cudaGetLastError();
}

cudaError_t launch_selftest_timeout(Ctrl* ctrl, uint64_t limit_ns, cudaStream_t s) {
  k_selftest_timeout<<<1, 32, 0, s>>>(ctrl, limit_ns);
  return cudaGetLastError();
}

}  // namespace opd
