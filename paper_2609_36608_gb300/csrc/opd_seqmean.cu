// seq-mean-token-mean on the device (ActFirst-OPD Appendix B.4, Eq. opd-surrogate):
//   L = 1/|B| sum_b ( sum_j m_bj l_bj ) / ( sum_j m_bj + eps )
// so the weight of token i is w_i = m_i / (|B| (n_seg(i) + eps)), with n_b the number of
// supervised tokens of response b and |B| the number of distinct responses (ids >= 0,
// including responses whose tokens are all masked). Three small memory-bound passes:
// a histogram of supervised tokens per response id, the count of distinct ids, then the
// weights and (optionally) sum_i w_i l_i.
//
// For a batch whose rows are spread over several processes the histogram is its own
// pass (launch_seq_counts: supervised rows and all rows per id, summable across
// processes), and the last two passes run from the summed histogram
// (launch_seq_from_counts), so every process gets the whole batch's n_b and |B|.
#include "opd_device.cuh"
#include "opd_internal.h"

namespace opd {

namespace {

// Scratch: [double acc][int32 n_resp, pad][counts n_ids][present n_ids]; the status word
// lives in a Ctrl of the caller's workspace.
__global__ void k_seq_zero(uint32_t* status, bool clear_status, int32_t* counts, int32_t* present, int32_t n_ids,
                           int32_t* n_resp, double* acc) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n_ids; i += gridDim.x * blockDim.x) {
    counts[i] = 0;
    present[i] = 0;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    if (clear_status) *status = 0u;
    *n_resp = 0;
    *acc = 0.0;
  }
}

__global__ void k_seq_zero_counts(uint32_t* status, int32_t* counts, int32_t n) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) counts[i] = 0;
  if (blockIdx.x == 0 && threadIdx.x == 0) *status = 0u;
}

// counts[b] += supervised rows of response b; present[b] = 1 (or, with count_rows, += every
// row of b, so that the planes of several processes can be summed).
__global__ void k_seq_hist(const int32_t* __restrict__ seg, const uint8_t* __restrict__ mask, int32_t T,
                           int32_t n_ids, int32_t* counts, int32_t* present, uint32_t* status, bool count_rows) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < T; i += gridDim.x * blockDim.x) {
    const int b = seg[i];
    if (b < 0) continue;
    if (b >= n_ids) {
      atomicOr(status, kDevBadToken);
      continue;
    }
    if (count_rows)
      atomicAdd(&present[b], 1);
    else
      present[b] = 1;
    if (mask[i]) atomicAdd(&counts[b], 1);
  }
}

// |B|: the ids with at least one row (present[] may hold row counts summed over processes).
__global__ void k_seq_count(const int32_t* __restrict__ present, int32_t n_ids, int32_t* n_resp) {
  int local = 0;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n_ids; i += gridDim.x * blockDim.x)
    local += present[i] != 0 ? 1 : 0;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) local += __shfl_xor_sync(0xffffffffu, local, o);
  if ((threadIdx.x & 31) == 0 && local) atomicAdd(n_resp, local);
}

__global__ void k_seq_weights(const int32_t* __restrict__ seg, const uint8_t* __restrict__ mask, int32_t T,
                              int32_t n_ids, const int32_t* __restrict__ counts, const int32_t* __restrict__ n_resp,
                              float eps, const float* __restrict__ loss_in, float* __restrict__ w_out, double* acc) {
  const double nb = (double)*n_resp;
  double part = 0.0;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < T; i += gridDim.x * blockDim.x) {
    const int b = seg[i];
    float w = 0.f;
    if (b >= 0 && b < n_ids && mask[i]) w = (float)(1.0 / (nb * ((double)counts[b] + (double)eps)));
    if (w_out) w_out[i] = w;
    if (loss_in) part += (double)w * (double)loss_in[i];
  }
  if (loss_in) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
    if ((threadIdx.x & 31) == 0 && part != 0.0) atomicAdd(acc, part);
  }
}

__global__ void k_seq_store(const double* acc, float* loss_out) { *loss_out = (float)*acc; }

}  // namespace

cudaError_t launch_store_loss(const double* acc, float* loss_out, cudaStream_t s) {
  k_seq_store<<<1, 1, 0, s>>>(acc, loss_out);
  return cudaGetLastError();
}

size_t seq_mean_token_mean_scratch_bytes(int64_t n_ids) { return 16 + 8 * (size_t)n_ids; }

double* seq_mean_token_mean_acc(void* scratch) { return static_cast<double*>(scratch); }

cudaError_t launch_seq_mean_token_mean(const int32_t* seg, const uint8_t* mask, int32_t T, int32_t n_ids, float eps,
                                       const float* loss_in, float* w_out, float* loss_out, Ctrl* ctrl,
                                       bool clear_status, void* scratch, int n_sm, cudaStream_t s) {
  double* acc = static_cast<double*>(scratch);
  int32_t* n_resp = reinterpret_cast<int32_t*>(acc + 1);
  int32_t* counts = n_resp + 2;
  int32_t* present = counts + n_ids;
  uint32_t* status = &ctrl->status;
  const int threads = 256;
  auto blocks = [&](long work) {
    long b = (work + threads - 1) / threads;
    if (b > (long)n_sm * 4) b = (long)n_sm * 4;
    return (int)(b < 1 ? 1 : b);
  };
  k_seq_zero<<<blocks(n_ids), threads, 0, s>>>(status, clear_status, counts, present, n_ids, n_resp, acc);
  k_seq_hist<<<blocks(T), threads, 0, s>>>(seg, mask, T, n_ids, counts, present, status, false);
  k_seq_count<<<blocks(n_ids), threads, 0, s>>>(present, n_ids, n_resp);
  k_seq_weights<<<blocks(T), threads, 0, s>>>(seg, mask, T, n_ids, counts, n_resp, eps, loss_in, w_out, acc);
  if (loss_out) k_seq_store<<<1, 1, 0, s>>>(acc, loss_out);
  return cudaGetLastError();
}

cudaError_t launch_seq_counts(const int32_t* seg, const uint8_t* mask, int32_t T, int32_t n_ids, int32_t* counts,
                              Ctrl* ctrl, int n_sm, cudaStream_t s) {
  const int threads = 256;
  auto blocks = [&](long work) {
    long b = (work + threads - 1) / threads;
    if (b > (long)n_sm * 4) b = (long)n_sm * 4;
    return (int)(b < 1 ? 1 : b);
  };
  // counts [2, n_ids]: supervised rows, then all rows, of each response id
  k_seq_zero_counts<<<blocks(2 * (long)n_ids), threads, 0, s>>>(&ctrl->status, counts, 2 * n_ids);
  k_seq_hist<<<blocks(T), threads, 0, s>>>(seg, mask, T, n_ids, counts, counts + n_ids, &ctrl->status, true);
  return cudaGetLastError();
}

cudaError_t launch_seq_from_counts(const int32_t* seg, const uint8_t* mask, int32_t T, int32_t n_ids,
                                   const int32_t* counts, float eps, const float* loss_in, float* w_out,
                                   float* loss_out, Ctrl* ctrl, void* scratch, int n_sm, cudaStream_t s) {
  double* acc = static_cast<double*>(scratch);
  int32_t* n_resp = reinterpret_cast<int32_t*>(acc + 1);
  const int threads = 256;
  auto blocks = [&](long work) {
    long b = (work + threads - 1) / threads;
    if (b > (long)n_sm * 4) b = (long)n_sm * 4;
    return (int)(b < 1 ? 1 : b);
  };
  k_seq_zero<<<1, threads, 0, s>>>(&ctrl->status, false, nullptr, nullptr, 0, n_resp, acc);
  k_seq_count<<<blocks(n_ids), threads, 0, s>>>(counts + n_ids, n_ids, n_resp);
  k_seq_weights<<<blocks(T), threads, 0, s>>>(seg, mask, T, n_ids, counts, n_resp, eps, loss_in, w_out, acc);
  if (loss_out) k_seq_store<<<1, 1, 0, s>>>(acc, loss_out);
  return cudaGetLastError();
}

}  // namespace opd
