// opd_kl_forward_noalloc: the forward pass for callers that cannot allocate
// device memory at all. Some host applications own every byte of the GPU (a
// serving process or plugin host with its own fixed memory pool, or a framework
// that forbids libraries from calling cudaMalloc because it would synchronise
// the device or break the host's memory accounting). Those callers can still
// pass inputs and outputs, but cannot hand the library a workspace.
//
// This entry point keeps its scratch in one file-scope device array of fixed
// size (kScratchBytes, about 5 MiB). Every GPU that loads the library holds that
// array until the process exits. It serves up to kMaxRows token rows, skips the
// row compaction and gather (which would need T x (d_s + d_t) bf16 of scratch),
// and runs the same fused forward kernel and combine kernel as opd_kl_forward
// directly over all T rows; rows with mask 0 are computed and then written as
// zeros. All calls share the one array, so calls whose kernels overlap on the
// GPU (different streams, or several host threads) race on it.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdlib>
#include <mutex>

#include "opd_device.cuh"
#include "opd_internal.h"
#include "opd_kl.h"

using namespace opd;

namespace {

constexpr int kMaxRows = OPD_KL_NOALLOC_MAX_ROWS;                          // token rows per call
constexpr size_t kCtrlBytes = 256;                                         // Ctrl block
constexpr size_t kPosBytes = (size_t)kMaxRows * 4;                         // pos[T]
constexpr int kSplits = 64;                                                 // vocabulary splits used here
constexpr size_t kPartialBytes = (size_t)kSplits * 5 * kMaxRows * 4;       // [split][5][row] floats
constexpr size_t kScratchBytes = kCtrlBytes + kPosBytes + kPartialBytes;  // 5,259,520 bytes
static_assert(sizeof(Ctrl) <= kCtrlBytes, "control block");
static_assert(kMaxRows % kRowPad == 0, "row cap is a whole number of padded row tiles");

static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

// Every row is processed in place (row r of the tile schedule is token row r):
// pos[i] = i for supervised rows, -1 otherwise, and the row count is T.
__global__ void k_noalloc_rows(const uint8_t* __restrict__ mask, int32_t T) {
  Ctrl* ctrl = reinterpret_cast<Ctrl*>(g_noalloc_scratch);
  int32_t* pos = reinterpret_cast<int32_t*>(g_noalloc_scratch + kCtrlBytes);
  for (int i = threadIdx.x; i < T; i += blockDim.x) pos[i] = mask[i] != 0 ? i : -1;
  if (threadIdx.x == 0) {
    ctrl->R = T;
    ctrl->status = 0u;
    ctrl->n_vsplit = 0;
    ctrl->half_tile = 0;
  }
  if (threadIdx.x < 4) ctrl->work[threadIdx.x] = 0;
}

// After the combine: if a bounded wait of this call ran out, every kl_out and stats
// entry becomes NaN, so that a caller who does not synchronise still cannot mistake
// partial statistics for a result (this entry point has no workspace whose status
// word the caller could read).
__global__ void k_noalloc_poison_on_timeout(float* kl_out, float* stats, int32_t T) {
  const Ctrl* ctrl = reinterpret_cast<const Ctrl*>(g_noalloc_scratch);
  if ((ctrl->status & kDevTimeout) == 0u) return;
  const float nan = __int_as_float(0x7fc00000);
  for (int i = threadIdx.x; i < T; i += blockDim.x) {
    kl_out[i] = nan;
    stats[3 * i] = nan;
    stats[3 * i + 1] = nan;
    stats[3 * i + 2] = nan;
  }
}

// Device address of the scratch array, looked up once per device (with that
// device current) and cached; host code must not use the symbol itself.
unsigned char* scratch_address(int dev) {
  static std::mutex mu;
  static unsigned char* addr[64] = {};
  if (dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (!addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
    addr[dev] = static_cast<unsigned char*>(p);
  }
  return addr[dev];
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

bool tmap_bf16(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint32_t box_inner,
               uint32_t box_outer) {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  });
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" opd_status opd_kl_forward_noalloc(const opd_problem* problem, const void* H_s, const void* H_t,
                                             const void* W_s, const void* W_t, const uint8_t* mask, float* kl_out,
                                             float* stats, void* stream) {
  if (!problem) return OPD_ERR_INVALID_ARG;
  const opd_problem p = *problem;
  if (p.T < 0 || p.d_s < 1 || p.d_t < 1 || p.V < 1 || p.V > (int64_t)0x7FFF0000 || p.d_s > (1 << 20) ||
      p.d_t > (1 << 20) || !(p.temperature > 0.0f) || !std::isfinite(p.temperature))
    return OPD_ERR_INVALID_ARG;
  if (p.dtype != OPD_DTYPE_BF16 || p.d_s % 8 != 0 || p.d_t % 8 != 0) return OPD_ERR_UNSUPPORTED;
  if (p.T > kMaxRows) return OPD_ERR_UNSUPPORTED;  // beyond the fixed scratch
  if (!W_s || !W_t || (p.T > 0 && (!H_s || !H_t || !mask || !kl_out || !stats))) return OPD_ERR_INVALID_ARG;
  if (!aligned16(H_s) || !aligned16(H_t) || !aligned16(W_s) || !aligned16(W_t)) return OPD_ERR_INVALID_ARG;
  if (p.T == 0) return OPD_OK;

  int dev = 0, sms = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return OPD_ERR_CUDA;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
    return OPD_ERR_CUDA;
  if (!(major == 10 && minor == 3)) return OPD_ERR_UNSUPPORTED;
  unsigned char* base = scratch_address(dev);
  if (!base) return OPD_ERR_CUDA;
  Ctrl* ctrl = reinterpret_cast<Ctrl*>(base);
  int32_t* pos = reinterpret_cast<int32_t*>(base + kCtrlBytes);
  float* partials = reinterpret_cast<float*>(base + kCtrlBytes + kPosBytes);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int32_t T = (int32_t)p.T;
  const int32_t T_pad = (T + kRowPad - 1) / kRowPad * kRowPad;

  CUtensorMap hs, ht, ws, wt;
  if (!tmap_bf16(&hs, H_s, (uint64_t)p.d_s, (uint64_t)T, kKBlock, kRowTile) ||
      !tmap_bf16(&ht, H_t, (uint64_t)p.d_t, (uint64_t)T, kKBlock, kRowTile) ||
      !tmap_bf16(&ws, W_s, (uint64_t)p.d_s, (uint64_t)p.V, kKBlock, fused_w_box(kFusedDefaultMode)) ||
      !tmap_bf16(&wt, W_t, (uint64_t)p.d_t, (uint64_t)p.V, kKBlock, fused_w_box(kFusedDefaultMode)))
    return OPD_ERR_CUDA;

  k_noalloc_rows<<<1, 1024, 0, s>>>(mask, T);
  if (cudaGetLastError() != cudaSuccess) return OPD_ERR_CUDA;

  FusedParams fp{};
  fp.ctrl = ctrl;
  fp.V = (int32_t)p.V;
  fp.d_s = (int32_t)p.d_s;
  fp.d_t = (int32_t)p.d_t;
  fp.T_pad = T_pad;
  fp.group_rows = 10;
  fp.k2 = (float)(1.4426950408889634 / (double)p.temperature);
  fp.inv_tau = 1.0f / p.temperature;
  fp.wait_limit_ns = 2000000000ull;
  fp.partials = partials;
  fp.max_vsplit = kSplits;
  fp.rowc = nullptr;
  fp.half_tile = 1;
  fp.vsplit = 0;
  if (launch_fused_forward(hs, ht, ws, wt, fp, sms, s) != cudaSuccess) return OPD_ERR_CUDA;
  if (launch_combine(partials, pos, nullptr, ctrl, T, T_pad, kl_out, stats, nullptr, nullptr, sms, s) != cudaSuccess)
    return OPD_ERR_CUDA;
  k_noalloc_poison_on_timeout<<<1, 1024, 0, s>>>(kl_out, stats, T);
  if (cudaGetLastError() != cudaSuccess) return OPD_ERR_CUDA;

  const char* sync = std::getenv("OPD_KL_SYNC_CHECK");
  if (sync && sync[0] && sync[0] != '0') {
    if (launch_check_finite(kl_out, (size_t)T, ctrl, sms, s) != cudaSuccess ||
        launch_check_finite(stats, 3 * (size_t)T, ctrl, sms, s) != cudaSuccess)
      return OPD_ERR_CUDA;
    uint32_t st = 0;
    if (cudaStreamSynchronize(s) != cudaSuccess) return OPD_ERR_CUDA;
    if (cudaMemcpy(&st, &ctrl->status, sizeof st, cudaMemcpyDeviceToHost) != cudaSuccess) return OPD_ERR_CUDA;
    if (st & kDevTimeout) return OPD_ERR_TIMEOUT;
    if (st & kDevNonFinite) return OPD_ERR_NONFINITE;
  }
  return OPD_OK;
}
