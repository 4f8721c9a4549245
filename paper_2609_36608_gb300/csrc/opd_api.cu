// C ABI of the OPD reverse-KL step (declared in include/opd_kl.h): argument
// validation, workspace layout, TMA tensor-map encoding and the launch sequence.
// All launches go to the caller's stream; nothing here allocates device memory.
#include <cuda.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <vector>

#include "opd_device.cuh"
#include "opd_internal.h"
#include "opd_kl.h"

using namespace opd;

namespace {

constexpr uint64_t kDefaultWaitLimitNs = 2000000000ull;  // 2 s per wait

inline size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct WsLayout {
  size_t ctrl = 0, idx = 0, pos = 0, hs_g = 0, ht_g = 0, partials = 0, rowc = 0, dz = 0, dh_g = 0, total = 0;
  size_t fwd_total = 0;  // the prefix that forward-only calls touch (no backward constants, dz or dH_g)
  int64_t T_pad = 0, Vp = 0;
};

// Workspace layout, 256-byte aligned sections. Sized for every row supervised. The
// sections a forward-only call uses come first, so a forward needs only the prefix
// [0, fwd_total) and a full workspace serves every call.
WsLayout ws_layout(const opd_problem& p) {
  WsLayout L;
  L.T_pad = (int64_t)round_up((size_t)(p.T > 0 ? p.T : 1), kRowPad);
  L.Vp = (int64_t)round_up((size_t)p.V, 64);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = round_up(off + bytes, 256);
    return o;
  };
  const size_t Tp = (size_t)L.T_pad;
  L.ctrl = take(sizeof(Ctrl));
  L.idx = take(4 * Tp);
  L.pos = take(4 * Tp);
  if (p.dtype == OPD_DTYPE_BF16) {
    L.hs_g = take(2 * Tp * (size_t)p.d_s);
    L.ht_g = take(2 * Tp * (size_t)p.d_t);
    L.partials = take(4 * (size_t)kMaxVSplit * 5 * Tp);
    L.fwd_total = off;
    L.rowc = take(16 * Tp);
    L.dz = take(2 * Tp * (size_t)L.Vp);
    L.dh_g = take(4 * Tp * (size_t)p.d_s);
  } else {
    L.fwd_total = off;
    L.dz = take(4 * Tp * (size_t)p.V);
  }
  L.total = off;
  return L;
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

opd_status check_problem(const opd_problem* p) {
  if (!p) return OPD_ERR_INVALID_ARG;
  if (p->T < 0 || p->T > (int64_t)0x7FFF0000 || p->d_s < 1 || p->d_t < 1 || p->V < 1) return OPD_ERR_INVALID_ARG;
  if (p->d_s > (1 << 20) || p->d_t > (1 << 20) || p->V > (int64_t)0x7FFF0000) return OPD_ERR_INVALID_ARG;
  if (!(p->temperature > 0.0f) || !std::isfinite(p->temperature)) return OPD_ERR_INVALID_ARG;
  if (p->dtype != OPD_DTYPE_BF16 && p->dtype != OPD_DTYPE_F32) return OPD_ERR_INVALID_ARG;
  if (p->dtype == OPD_DTYPE_BF16 && (p->d_s % 8 != 0 || p->d_t % 8 != 0)) return OPD_ERR_UNSUPPORTED;
  return OPD_OK;
}

bool env_flag(const char* name) {
  const char* v = std::getenv(name);
  return v && v[0] && v[0] != '0';
}

int env_int(const char* name, int dflt) {
  const char* v = std::getenv(name);
  if (!v || !v[0]) return dflt;
  return std::atoi(v);
}

// ------------------------------------------------------------ device info --

struct DeviceInfo {
  int sm_count = 0;
  int major = 0, minor = 0;
};

DeviceInfo device_info() {
  static std::mutex mu;
  static std::vector<DeviceInfo> cache;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return {};
  std::lock_guard<std::mutex> lock(mu);
  if ((int)cache.size() <= dev) cache.resize(dev + 1);
  if (cache[dev].sm_count == 0) {
    DeviceInfo d;
    cudaDeviceGetAttribute(&d.sm_count, cudaDevAttrMultiProcessorCount, dev);
    cudaDeviceGetAttribute(&d.major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&d.minor, cudaDevAttrComputeCapabilityMinor, dev);
    cache[dev] = d;
  }
  return cache[dev];
}

// ------------------------------------------------------------ tensor maps --

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
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
  return fn;
}

// 2-D tiled map over a row-major matrix: `inner` contiguous elements per row,
// `outer` rows, row pitch `pitch` elements; 128-byte swizzle; out-of-range
// elements read as zero and are clipped on stores.
bool tmap2d(CUtensorMap* m, CUtensorMapDataType dt, size_t esize, const void* base, uint64_t inner, uint64_t outer,
            uint64_t pitch, uint32_t box_inner, uint32_t box_outer) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {pitch * esize};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t es[2] = {1, 1};
  return fn(m, dt, 2, const_cast<void*>(base), dims, strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// ---------------------------------------------------------- kernel timing --

struct Profiler {
  std::mutex mu;
  bool on = false;
  struct Rec {
    const char* name;
    cudaEvent_t a, b;
  };
  std::vector<Rec> recs;
  std::vector<cudaEvent_t> pool;

  cudaEvent_t take() {
    if (!pool.empty()) {
      cudaEvent_t e = pool.back();
      pool.pop_back();
      return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
  }
};

Profiler& profiler() {
  static Profiler P;
  return P;
}

// Launch through `fn`, bracketed by events when timing is on.
template <class F>
cudaError_t timed(const char* name, cudaStream_t s, F&& fn) {
  Profiler& P = profiler();
  cudaEvent_t a = nullptr, b = nullptr;
  {
    std::lock_guard<std::mutex> lock(P.mu);
    if (P.on) {
      a = P.take();
      b = P.take();
    }
  }
  if (a && b) cudaEventRecord(a, s);
  const cudaError_t e = fn();
  if (a && b) {
    cudaEventRecord(b, s);
    std::lock_guard<std::mutex> lock(P.mu);
    P.recs.push_back({name, a, b});
  }
  return e;
}

// ------------------------------------------------------------- call state --

struct Call {
  opd_problem p;
  WsLayout L;
  uint8_t* ws;
  size_t ws_bytes;
  cudaStream_t s;
  DeviceInfo dev;
  Ctrl* ctrl() const { return reinterpret_cast<Ctrl*>(ws + L.ctrl); }
  int32_t* idx() const { return reinterpret_cast<int32_t*>(ws + L.idx); }
  int32_t* pos() const { return reinterpret_cast<int32_t*>(ws + L.pos); }
};

opd_status cuda_status(cudaError_t e) { return e == cudaSuccess ? OPD_OK : OPD_ERR_CUDA; }

#define OPD_TRY(expr)                         \
  do {                                        \
    const opd_status _st = (expr);            \
    if (_st != OPD_OK) return _st;            \
  } while (0)
#define OPD_CUDA(expr) OPD_TRY(cuda_status(expr))

// forward_only: the call runs no backward, so the workspace prefix of
// opd_kl_forward_workspace_size bytes is enough.
opd_status begin_call(Call& c, const opd_problem* problem, void* workspace, size_t ws_bytes, void* stream,
                      bool forward_only) {
  OPD_TRY(check_problem(problem));
  c.p = *problem;
  c.L = ws_layout(c.p);
  if (!workspace || !aligned(workspace, 256) || ws_bytes < (forward_only ? c.L.fwd_total : c.L.total))
    return OPD_ERR_INVALID_ARG;
  c.ws_bytes = ws_bytes;
  c.ws = static_cast<uint8_t*>(workspace);
  c.s = static_cast<cudaStream_t>(stream);
  c.dev = device_info();
  if (c.dev.sm_count <= 0) return OPD_ERR_CUDA;
  if (c.p.dtype == OPD_DTYPE_BF16 && !(c.dev.major == 10 && c.dev.minor == 3)) return OPD_ERR_UNSUPPORTED;
  return OPD_OK;
}

// Output buffers a call wrote (pointer, element count), checked for non-finite
// values in debug mode.
struct Outputs {
  const float* p[5] = {};
  size_t n[5] = {};
  int k = 0;
  Outputs& add(const float* q, size_t m) {
    if (q && m && k < 5) {
      p[k] = q;
      n[k++] = m;
    }
    return *this;
  }
};

opd_status finish_call(const Call& c, const Outputs& out = Outputs()) {
  if (cudaGetLastError() != cudaSuccess) return OPD_ERR_CUDA;
  if (env_flag("OPD_KL_SYNC_CHECK")) {
    for (int i = 0; i < out.k; ++i) OPD_CUDA(launch_check_finite(out.p[i], out.n[i], c.ctrl(), c.dev.sm_count, c.s));
    return opd_kl_get_status(c.ws, c.ws_bytes, c.s);
  }
  return OPD_OK;
}

opd_status check_inputs(const Call& c, const void* H_s, const void* H_t, const void* W_s, const void* W_t,
                        const uint8_t* mask) {
  if (!W_s || !W_t) return OPD_ERR_INVALID_ARG;
  if (c.p.T > 0 && (!H_s || !H_t || !mask)) return OPD_ERR_INVALID_ARG;
  const size_t a = c.p.dtype == OPD_DTYPE_BF16 ? 16 : 4;
  if (!aligned(W_s, a) || !aligned(W_t, a) || !aligned(H_s, a) || !aligned(H_t, a)) return OPD_ERR_INVALID_ARG;
  return OPD_OK;
}

// Row compaction plus (bf16) the gather of supervised rows (H_t may be null: one head).
opd_status prologue(const Call& c, const void* H_s, const void* H_t, const uint8_t* mask) {
  OPD_CUDA(timed("compact", c.s, [&] { return launch_compact(mask, (int32_t)c.p.T, c.idx(), c.pos(), c.ctrl(), c.s); }));
  if (c.p.dtype == OPD_DTYPE_BF16) {
    const int32_t d_t = H_t ? (int32_t)c.p.d_t : 0;
    OPD_CUDA(timed("gather", c.s, [&] {
      return launch_gather_bf16(H_s, H_t, (int32_t)c.p.d_s, d_t, c.idx(), c.ctrl(), c.ws + c.L.hs_g,
                                c.ws + c.L.ht_g, (int32_t)c.L.T_pad, c.dev.sm_count, c.s);
    }));
  }
  return OPD_OK;
}

struct Maps {
  CUtensorMap hs, ht, ws, wt;        // fused kernels: K-major A (rows) and B (vocab rows)
  CUtensorMap dz_store;              // fused backward: bf16 dz tiles out
  CUtensorMap dz_a_k, ws_b_mn, dhg;  // dH_s GEMM
  CUtensorMap dz_a_mn, hsg_b_mn, dw; // dW_s GEMM
};

// Gradient-GEMM tiling: CTA pairs unless OPD_KL_GEMM=cta1.
int gemm_pair_mode() {
  const char* v = std::getenv("OPD_KL_GEMM");
  return (v && std::strcmp(v, "cta1") == 0) ? 0 : 1;
}

// Fused-kernel tiling: OPD_KL_FUSED=bn256 | pair256 overrides the default.
int fused_tile_mode() {
  const char* v = std::getenv("OPD_KL_FUSED");
  if (v && std::strcmp(v, "bn256") == 0) return kFusedBN256;
  if (v && std::strcmp(v, "pair256") == 0) return kFusedPair256;
  return kFusedDefaultMode;
}

opd_status encode_maps(const Call& c, const void* W_s, const void* W_t, float* dW_s, Maps& m, bool bwd) {
  const uint32_t bn = (uint32_t)fused_w_box(fused_tile_mode());
  const auto BF = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  const auto F32 = CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
  const uint64_t Tp = (uint64_t)c.L.T_pad, ds = (uint64_t)c.p.d_s, dt = (uint64_t)c.p.d_t, V = (uint64_t)c.p.V;
  const uint64_t Vp = (uint64_t)c.L.Vp;
  bool ok = tmap2d(&m.hs, BF, 2, c.ws + c.L.hs_g, ds, Tp, ds, kKBlock, kRowTile) &&
            tmap2d(&m.ht, BF, 2, c.ws + c.L.ht_g, dt, Tp, dt, kKBlock, kRowTile) &&
            tmap2d(&m.ws, BF, 2, W_s, ds, V, ds, kKBlock, bn) &&
            tmap2d(&m.wt, BF, 2, W_t, dt, V, dt, kKBlock, bn);
  if (ok && bwd) {
    ok = tmap2d(&m.dz_store, BF, 2, c.ws + c.L.dz, V, Tp, Vp, 64, 32) &&
         tmap2d(&m.dz_a_k, BF, 2, c.ws + c.L.dz, V, Tp, Vp, kKBlock, kRowTile) &&
         tmap2d(&m.ws_b_mn, BF, 2, W_s, ds, V, ds, 64, kKBlock) &&
         tmap2d(&m.dhg, F32, 4, c.ws + c.L.dh_g, ds, Tp, ds, 32, 32) &&
         tmap2d(&m.dz_a_mn, BF, 2, c.ws + c.L.dz, V, Tp, Vp, 64, kKBlock) &&
         tmap2d(&m.hsg_b_mn, BF, 2, c.ws + c.L.hs_g, ds, Tp, ds, 64, kKBlock) &&
         tmap2d(&m.dw, F32, 4, dW_s, ds, V, ds, 32, 32);
  }
  return ok ? OPD_OK : OPD_ERR_CUDA;
}

FusedParams fused_params(const Call& c) {
  FusedParams fp{};
  fp.ctrl = c.ctrl();
  fp.V = (int32_t)c.p.V;
  fp.d_s = (int32_t)c.p.d_s;
  fp.d_t = (int32_t)c.p.d_t;
  fp.T_pad = (int32_t)c.L.T_pad;
  fp.group_rows = env_int("OPD_KL_GROUP_ROWS", 10);
  fp.k2 = (float)(1.4426950408889634 / (double)c.p.temperature);
  fp.inv_tau = 1.0f / c.p.temperature;
  fp.wait_limit_ns = kDefaultWaitLimitNs;
  fp.partials = reinterpret_cast<float*>(c.ws + c.L.partials);
  fp.rowc = reinterpret_cast<const float4*>(c.ws + c.L.rowc);
  fp.mode = fused_tile_mode();
  fp.max_vsplit = kMaxVSplit;
  fp.half_tile = env_int("OPD_KL_HALF_TILE", 1) != 0 ? 1 : 0;
  fp.vsplit = env_int("OPD_KL_VSPLIT", 0);
  return fp;
}

// The paper's batch loss over the per-token KL (Appendix B.4, seq-mean-token-mean):
// per-token weights computed on the device, then L = sum_i w_i KL_i.
struct SeqLoss {
  const int32_t* seg_id;
  int64_t n_ids;
  float eps;
  float* weights;  // [T] in the workspace; also the backward's upstream weights
  void* scratch;   // seq-mean scratch (starts with the double accumulator of L)
  float* loss_out; // [1]
};

// opd_kl_seq_mean_fwd_bwd's workspace: the reverse-KL workspace, then the per-token
// weights, then the seq-mean scratch; 256-byte aligned sections.
struct SeqLayout {
  size_t weights = 0, scratch = 0, total = 0;
};

SeqLayout seq_layout(const WsLayout& L, int64_t n_ids) {
  SeqLayout S;
  size_t off = round_up(L.total, 256);
  S.weights = off;
  off = round_up(off + 4 * (size_t)L.T_pad, 256);
  S.scratch = off;
  off = round_up(off + seq_mean_token_mean_scratch_bytes(n_ids), 256);
  S.total = off;
  return S;
}

// Fused forward and combine; with loss weights, the combine also accumulates L.
opd_status forward_body(const Call& c, const Maps& m, float* kl_out, float* stats, const SeqLoss* seq) {
  if (c.p.dtype == OPD_DTYPE_F32) return OPD_OK;  // handled by caller
  const FusedParams fp = fused_params(c);
  OPD_CUDA(timed("fused_logits_fwd", c.s,
                 [&] { return launch_fused_forward(m.hs, m.ht, m.ws, m.wt, fp, c.dev.sm_count, c.s); }));
  OPD_CUDA(timed("combine", c.s, [&] {
    return launch_combine(fp.partials, c.pos(), c.idx(), c.ctrl(), (int32_t)c.p.T, (int32_t)c.L.T_pad, kl_out, stats,
                          seq ? seq->weights : nullptr, seq ? seq_mean_token_mean_acc(seq->scratch) : nullptr,
                          c.dev.sm_count, c.s);
  }));
  return OPD_OK;
}

// dW_s is written through the tensor map m.dw (encoded over the caller's dW_s).
opd_status gradient_gemms(const Call& c, const Maps& m, float* dH_s, int accumulate_dW);

opd_status backward_body(const Call& c, const Maps& m, const float* stats, const float* grad_kl, float* dH_s,
                         int accumulate_dW) {
  FusedParams fp = fused_params(c);
  float4* rowc = reinterpret_cast<float4*>(c.ws + c.L.rowc);
  OPD_CUDA(timed("bwd_rowc", c.s, [&] {
    return launch_bwd_rowc(stats, grad_kl, c.idx(), c.ctrl(), (int32_t)c.L.T_pad, c.p.temperature, rowc, c.s);
  }));
  OPD_CUDA(timed("fused_logits_bwd", c.s, [&] {
    return launch_fused_backward(m.hs, m.ht, m.ws, m.wt, m.dz_store, fp, c.dev.sm_count, c.s);
  }));
  return gradient_gemms(c, m, dH_s, accumulate_dW);
}

// dH_s = dZ W_s (split-K partial sums, then scattered back to the T rows) and
// dW_s (+)= dZ^T H_s, from the bf16 dz the fused backward wrote.
opd_status gradient_gemms(const Call& c, const Maps& m, float* dH_s, int accumulate_dW) {
  float* dhg = reinterpret_cast<float*>(c.ws + c.L.dh_g);
  OPD_CUDA(timed("zero_rows", c.s, [&] {
    return launch_zero_rows(dhg, (int32_t)c.p.d_s, c.ctrl(), (int32_t)c.L.T_pad, c.dev.sm_count, c.s);
  }));

  GemmParams gh{};
  gh.ctrl = c.ctrl();
  gh.M = 0;
  gh.m_is_R = 1;
  gh.N = (int32_t)c.p.d_s;
  gh.K = (int32_t)c.p.V;
  gh.k_is_R = 0;
  // deterministic mode: each dH_s tile takes the whole K = V range and is stored, not
  // summed from split-K partials whose reduce-adds land in any order
  const bool deterministic = env_flag("OPD_KL_DETERMINISTIC");
  gh.max_ksplit = deterministic ? 1 : env_int("OPD_KL_MAX_KSPLIT", kMaxKSplit);
  gh.reduce = deterministic ? 0 : 1;
  gh.pair = gemm_pair_mode();
  gh.work_slot = 2;
  gh.half_tile = env_int("OPD_KL_HALF_TILE", 1) != 0 ? 1 : 0;
  gh.wait_limit_ns = kDefaultWaitLimitNs;
  OPD_CUDA(timed("gemm_dH", c.s, [&] { return launch_gemm(false, true, m.dz_a_k, m.ws_b_mn, m.dhg, gh, c.dev.sm_count, c.s); }));

  GemmParams gw{};
  gw.ctrl = c.ctrl();
  gw.M = (int32_t)c.p.V;
  gw.m_is_R = 0;
  gw.N = (int32_t)c.p.d_s;
  gw.K = 0;
  gw.k_is_R = 1;
  gw.max_ksplit = 1;
  gw.reduce = accumulate_dW ? 1 : 0;
  gw.pair = gemm_pair_mode();
  gw.work_slot = 3;
  gw.half_tile = gh.half_tile;
  gw.wait_limit_ns = kDefaultWaitLimitNs;
  OPD_CUDA(timed("gemm_dW", c.s, [&] { return launch_gemm(true, true, m.dz_a_mn, m.hsg_b_mn, m.dw, gw, c.dev.sm_count, c.s); }));

  OPD_CUDA(timed("scatter_rows", c.s, [&] { return launch_scatter_rows(dhg, (int32_t)c.p.d_s, c.pos(), (int32_t)c.p.T, dH_s, c.dev.sm_count, c.s); }));
  return OPD_OK;
}

opd_status run(const opd_problem* problem, const void* H_s, const void* H_t, const void* W_s, const void* W_t,
               const uint8_t* mask, const float* grad_kl, float* kl_out, float* stats_out, const float* stats_in,
               float* dH_s, float* dW_s, int accumulate_dW, void* workspace, size_t ws_bytes, void* stream,
               bool do_fwd, bool do_bwd, const SeqLoss* seq = nullptr) {
  Call c;
  OPD_TRY(begin_call(c, problem, workspace, ws_bytes, stream, !do_bwd));
  OPD_TRY(check_inputs(c, H_s, H_t, W_s, W_t, mask));
  const int64_t T = c.p.T;
  if (do_fwd && T > 0 && (!kl_out || !stats_out)) return OPD_ERR_INVALID_ARG;
  if (do_bwd) {
    if (!dW_s || (T > 0 && (!grad_kl || !dH_s))) return OPD_ERR_INVALID_ARG;
    if (!do_fwd && T > 0 && !stats_in) return OPD_ERR_INVALID_ARG;
    const size_t a = c.p.dtype == OPD_DTYPE_BF16 ? 16 : 4;
    if (!aligned(dW_s, a) || !aligned(dH_s, a)) return OPD_ERR_INVALID_ARG;
  }
  const float* stats = do_fwd ? stats_out : stats_in;
  Outputs outputs;
  const size_t Tn = (size_t)T;
  if (do_fwd) outputs.add(kl_out, Tn).add(stats_out, 3 * Tn);
  if (do_bwd) outputs.add(dH_s, Tn * (size_t)c.p.d_s).add(dW_s, (size_t)c.p.V * (size_t)c.p.d_s);

  OPD_TRY(prologue(c, H_s, H_t, mask));
  if (seq) {  // the upstream weights of the batch loss, after compaction cleared the status word
    OPD_CUDA(timed("seq_mean_token_mean", c.s, [&] {
      return launch_seq_mean_token_mean(seq->seg_id, mask, (int32_t)T, (int32_t)seq->n_ids, seq->eps, nullptr,
                                        seq->weights, nullptr, c.ctrl(), false, seq->scratch, c.dev.sm_count, c.s);
    }));
    outputs.add(seq->loss_out, 1);
  }
  if (c.p.dtype == OPD_DTYPE_F32) {
    const float* hs = static_cast<const float*>(H_s);
    const float* ht = static_cast<const float*>(H_t);
    const float* ws = static_cast<const float*>(W_s);
    const float* wt = static_cast<const float*>(W_t);
    if (do_fwd)
      OPD_CUDA(timed("simt_forward", c.s, [&] {
        return launch_simt_forward(hs, ht, ws, wt, (int32_t)T, (int32_t)c.p.d_s, (int32_t)c.p.d_t, (int32_t)c.p.V,
                                   c.p.temperature, c.idx(), c.pos(), c.ctrl(), kl_out, stats_out, c.s);
      }));
    if (seq)  // L from the forward's per-token KL (the CUDA-core path has no combine pass)
      OPD_CUDA(timed("seq_mean_token_mean", c.s, [&] {
        return launch_seq_mean_token_mean(seq->seg_id, mask, (int32_t)T, (int32_t)seq->n_ids, seq->eps, kl_out,
                                          nullptr, seq->loss_out, c.ctrl(), false, seq->scratch, c.dev.sm_count,
                                          c.s);
      }));
    if (do_bwd)
      OPD_CUDA(timed("simt_backward", c.s, [&] {
        return launch_simt_backward(hs, ht, ws, wt, (int32_t)T, (int32_t)c.p.d_s, (int32_t)c.p.d_t,
                                    (int32_t)c.p.V, c.p.temperature, c.idx(), c.pos(), c.ctrl(), stats, grad_kl,
                                    reinterpret_cast<float*>(c.ws + c.L.dz), dH_s, dW_s, accumulate_dW, c.s);
      }));
    return finish_call(c, outputs);
  }

  Maps m;
  OPD_TRY(encode_maps(c, W_s, W_t, dW_s, m, do_bwd));
  if (do_fwd) OPD_TRY(forward_body(c, m, kl_out, stats_out, seq));
  if (seq)
    OPD_CUDA(timed("store_loss", c.s,
                   [&] { return launch_store_loss(seq_mean_token_mean_acc(seq->scratch), seq->loss_out, c.s); }));
  if (do_bwd) OPD_TRY(backward_body(c, m, stats, grad_kl, dH_s, accumulate_dW));
  return finish_call(c, outputs);
}

// Single-head path: compaction, gather of the head's rows, fused forward statistics,
// then the per-token finish (and, for the surrogate, the student backward).
opd_status head_call(const opd_problem* problem, const void* H, const void* W, const int32_t* tokens,
                     const uint8_t* mask, float* lse_out, float* logp_out, const float* logp_old,
                     const float* logp_teacher, const float* weights, const opd_surrogate_params* sp,
                     float* loss_out, float* dH, float* dW, int accumulate_dW, void* workspace, size_t ws_bytes,
                     void* stream, bool surrogate) {
  Call c;
  OPD_TRY(begin_call(c, problem, workspace, ws_bytes, stream, !surrogate));
  if (c.p.dtype != OPD_DTYPE_BF16) return OPD_ERR_UNSUPPORTED;
  const int64_t T = c.p.T;
  if (!W || !aligned(W, 16) || !aligned(H, 16)) return OPD_ERR_INVALID_ARG;
  if (T > 0 && (!H || !tokens || !mask || !logp_out)) return OPD_ERR_INVALID_ARG;
  if (!surrogate && T > 0 && !lse_out) return OPD_ERR_INVALID_ARG;
  if (surrogate) {
    if (!dW || !aligned(dW, 16) || !aligned(dH, 16)) return OPD_ERR_INVALID_ARG;
    if (T > 0 && (!logp_old || !logp_teacher || !weights || !loss_out || !dH)) return OPD_ERR_INVALID_ARG;
    if (sp && (!(sp->delta >= 0.0f && sp->delta < 1.0f) || !(sp->kappa > 0.0f) || !(sp->log_ratio_clip > 0.0f)))
      return OPD_ERR_INVALID_ARG;
  }
  OPD_TRY(prologue(c, H, nullptr, mask));
  Maps m;
  OPD_TRY(encode_maps(c, W, W, dW, m, surrogate));
  FusedParams fp = fused_params(c);
  OPD_CUDA(timed("head_logits_fwd", c.s, [&] { return launch_head_forward(m.hs, m.ws, fp, c.dev.sm_count, c.s); }));
  HeadRowsParams hp{};
  hp.ctrl = c.ctrl();
  hp.ctrl_rw = c.ctrl();
  hp.partials = fp.partials;
  hp.T = (int32_t)T;
  hp.T_pad = (int32_t)c.L.T_pad;
  hp.V = (int32_t)c.p.V;
  hp.d = (int32_t)c.p.d_s;
  hp.pos = c.pos();
  hp.H_g = reinterpret_cast<const __nv_bfloat16*>(c.ws + c.L.hs_g);
  hp.W = static_cast<const __nv_bfloat16*>(W);
  hp.tokens = tokens;
  hp.inv_tau = 1.0f / c.p.temperature;
  hp.lse_out = lse_out;
  hp.logp_out = logp_out;
  hp.surrogate = surrogate ? 1 : 0;
  hp.logp_old = logp_old;
  hp.logp_teacher = logp_teacher;
  hp.weights = weights;
  hp.delta = sp ? sp->delta : 0.2f;
  hp.kappa = sp ? sp->kappa : 3.0f;
  hp.clip = sp ? sp->log_ratio_clip : 20.0f;
  hp.loss_out = loss_out;
  hp.rowc = reinterpret_cast<float4*>(c.ws + c.L.rowc);
  OPD_CUDA(timed("head_rows", c.s, [&] { return launch_head_rows(hp, c.dev.sm_count, c.s); }));
  if (surrogate) {
    OPD_CUDA(timed("head_logits_bwd", c.s,
                   [&] { return launch_head_backward(m.hs, m.ws, m.dz_store, fp, c.dev.sm_count, c.s); }));
    OPD_TRY(gradient_gemms(c, m, dH, accumulate_dW));
  }
  Outputs outputs;
  const size_t Tn = (size_t)T;
  outputs.add(lse_out, Tn).add(logp_out, Tn);
  if (surrogate)
    outputs.add(loss_out, Tn).add(dH, Tn * (size_t)c.p.d_s).add(dW, (size_t)c.p.V * (size_t)c.p.d_s);
  return finish_call(c, outputs);
}

}  // namespace

extern "C" {

opd_status opd_score_tokens(const opd_problem* problem, const void* H, const void* W, const int32_t* tokens,
                            const uint8_t* mask, float* lse_out, float* logp_out, void* workspace,
                            size_t workspace_bytes, void* stream) {
  return head_call(problem, H, W, tokens, mask, lse_out, logp_out, nullptr, nullptr, nullptr, nullptr, nullptr,
                   nullptr, nullptr, 0, workspace, workspace_bytes, stream, false);
}

opd_status opd_surrogate_fwd_bwd(const opd_problem* problem, const void* H_s, const void* W_s,
                                 const int32_t* tokens, const float* logp_old, const float* logp_teacher,
                                 const uint8_t* mask, const float* weights, const opd_surrogate_params* params,
                                 float* loss_out, float* logp_out, float* dH_s, float* dW_s, int accumulate_dW,
                                 void* workspace, size_t workspace_bytes, void* stream) {
  return head_call(problem, H_s, W_s, tokens, mask, nullptr, logp_out, logp_old, logp_teacher, weights, params,
                   loss_out, dH_s, dW_s, accumulate_dW, workspace, workspace_bytes, stream, true);
}

size_t opd_kl_workspace_size(const opd_problem* problem) {
  if (!problem) return 0;
  const opd_status st = check_problem(problem);
  if (st != OPD_OK) return 0;
  return ws_layout(*problem).total;
}

size_t opd_kl_forward_workspace_size(const opd_problem* problem) {
  if (!problem) return 0;
  if (check_problem(problem) != OPD_OK) return 0;
  return ws_layout(*problem).fwd_total;
}

opd_status opd_kl_forward(const opd_problem* problem, const void* H_s, const void* H_t, const void* W_s,
                          const void* W_t, const uint8_t* mask, float* kl_out, float* stats, void* workspace,
                          size_t workspace_bytes, void* stream) {
  return run(problem, H_s, H_t, W_s, W_t, mask, nullptr, kl_out, stats, nullptr, nullptr, nullptr, 0, workspace,
             workspace_bytes, stream, true, false);
}

opd_status opd_kl_backward(const opd_problem* problem, const void* H_s, const void* H_t, const void* W_s,
                           const void* W_t, const uint8_t* mask, const float* stats, const float* grad_kl,
                           float* dH_s, float* dW_s, int accumulate_dW, void* workspace, size_t workspace_bytes,
                           void* stream) {
  return run(problem, H_s, H_t, W_s, W_t, mask, grad_kl, nullptr, nullptr, stats, dH_s, dW_s, accumulate_dW,
             workspace, workspace_bytes, stream, false, true);
}

opd_status opd_kl_fwd_bwd(const opd_problem* problem, const void* H_s, const void* H_t, const void* W_s,
                          const void* W_t, const uint8_t* mask, const float* grad_kl, float* kl_out, float* stats,
                          float* dH_s, float* dW_s, int accumulate_dW, void* workspace, size_t workspace_bytes,
                          void* stream) {
  return run(problem, H_s, H_t, W_s, W_t, mask, grad_kl, kl_out, stats, nullptr, dH_s, dW_s, accumulate_dW,
             workspace, workspace_bytes, stream, true, true);
}

opd_status opd_seq_mean_token_mean_weights(const int32_t* seg_id, const uint8_t* mask, int64_t T, float eps,
                                           float* w_out) {
  if (T < 0 || !(eps >= 0.0f)) return OPD_ERR_INVALID_ARG;
  if (T > 0 && (!seg_id || !mask || !w_out)) return OPD_ERR_INVALID_ARG;
  int32_t max_id = -1;
  for (int64_t i = 0; i < T; ++i) max_id = seg_id[i] > max_id ? seg_id[i] : max_id;
  std::vector<int64_t> count((size_t)(max_id + 1), 0);
  std::vector<uint8_t> seen((size_t)(max_id + 1), 0);
  int64_t n_resp = 0;
  for (int64_t i = 0; i < T; ++i) {
    const int32_t b = seg_id[i];
    if (b < 0) continue;
    if (!seen[b]) {
      seen[b] = 1;
      ++n_resp;
    }
    if (mask[i]) ++count[b];
  }
  for (int64_t i = 0; i < T; ++i) {
    const int32_t b = seg_id[i];
    w_out[i] = (b < 0 || !mask[i]) ? 0.0f : (float)(1.0 / ((double)n_resp * ((double)count[b] + (double)eps)));
  }
  return OPD_OK;
}

size_t opd_kl_seq_mean_workspace_size(const opd_problem* problem, int64_t n_ids) {
  if (check_problem(problem) != OPD_OK || n_ids < 1 || n_ids > (int64_t)0x7FFF0000) return 0;
  return seq_layout(ws_layout(*problem), n_ids).total;
}

opd_status opd_kl_seq_mean_fwd_bwd(const opd_problem* problem, const void* H_s, const void* H_t, const void* W_s,
                                   const void* W_t, const uint8_t* mask, const int32_t* seg_id, int64_t n_ids,
                                   float eps, float* loss_out, float* kl_out, float* stats, float* dH_s, float* dW_s,
                                   int accumulate_dW, void* workspace, size_t workspace_bytes, void* stream) {
  OPD_TRY(check_problem(problem));
  if (n_ids < 1 || n_ids > (int64_t)0x7FFF0000 || !(eps >= 0.0f) || !loss_out) return OPD_ERR_INVALID_ARG;
  if (problem->T > 0 && !seg_id) return OPD_ERR_INVALID_ARG;
  const SeqLayout S = seq_layout(ws_layout(*problem), n_ids);
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < S.total) return OPD_ERR_INVALID_ARG;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  SeqLoss seq{seg_id, n_ids, eps, reinterpret_cast<float*>(ws + S.weights), ws + S.scratch, loss_out};
  return run(problem, H_s, H_t, W_s, W_t, mask, seq.weights, kl_out, stats, nullptr, dH_s, dW_s, accumulate_dW,
             workspace, workspace_bytes, stream, true, true, &seq);
}

size_t opd_seq_mean_token_mean_workspace_size(int64_t n_ids) {
  if (n_ids < 1 || n_ids > (int64_t)0x7FFF0000) return 0;
  return round_up(sizeof(Ctrl) + seq_mean_token_mean_scratch_bytes(n_ids), 256);
}

opd_status opd_seq_mean_token_mean_device(const int32_t* seg_id, const uint8_t* mask, int64_t T, int64_t n_ids,
                                          float eps, const float* loss_in, float* w_out, float* loss_out,
                                          void* workspace, size_t workspace_bytes, void* stream) {
  if (T < 0 || T > (int64_t)0x7FFF0000 || n_ids < 1 || n_ids > (int64_t)0x7FFF0000 || !(eps >= 0.0f))
    return OPD_ERR_INVALID_ARG;
  if (T > 0 && (!seg_id || !mask)) return OPD_ERR_INVALID_ARG;
  // the loss is requested by loss_out; its input may be absent only when there are no rows
  if ((loss_out && T > 0 && !loss_in) || (!w_out && !loss_out)) return OPD_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < opd_seq_mean_token_mean_workspace_size(n_ids))
    return OPD_ERR_INVALID_ARG;
  const DeviceInfo dev = device_info();
  if (dev.sm_count <= 0) return OPD_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  OPD_CUDA(timed("seq_mean_token_mean", s, [&] {
    return launch_seq_mean_token_mean(seg_id, mask, (int32_t)T, (int32_t)n_ids, eps, loss_out ? loss_in : nullptr,
                                      w_out, loss_out, static_cast<Ctrl*>(workspace), true,
                                      static_cast<uint8_t*>(workspace) + sizeof(Ctrl), dev.sm_count, s);
  }));
  if (cudaGetLastError() != cudaSuccess) return OPD_ERR_CUDA;
  if (env_flag("OPD_KL_SYNC_CHECK")) {
    Ctrl* ctrl = static_cast<Ctrl*>(workspace);
    OPD_CUDA(launch_check_finite(w_out, w_out ? (size_t)T : 0, ctrl, dev.sm_count, s));
    OPD_CUDA(launch_check_finite(loss_out, 1, ctrl, dev.sm_count, s));
    return opd_kl_get_status(workspace, workspace_bytes, stream);
  }
  return OPD_OK;
}

opd_status opd_seq_mean_token_mean_counts(const int32_t* seg_id, const uint8_t* mask, int64_t T, int64_t n_ids,
                                          int32_t* counts, void* workspace, size_t workspace_bytes, void* stream) {
  if (T < 0 || T > (int64_t)0x7FFF0000 || n_ids < 1 || n_ids > (int64_t)0x3FFF0000) return OPD_ERR_INVALID_ARG;
  if ((T > 0 && (!seg_id || !mask)) || !counts) return OPD_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < opd_seq_mean_token_mean_workspace_size(n_ids))
    return OPD_ERR_INVALID_ARG;
  const DeviceInfo dev = device_info();
  if (dev.sm_count <= 0) return OPD_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  Ctrl* ctrl = static_cast<Ctrl*>(workspace);
  OPD_CUDA(timed("seq_counts", s, [&] {
    return launch_seq_counts(seg_id, mask, (int32_t)T, (int32_t)n_ids, counts, ctrl, dev.sm_count, s);
  }));
  if (cudaGetLastError() != cudaSuccess) return OPD_ERR_CUDA;
  if (env_flag("OPD_KL_SYNC_CHECK")) return opd_kl_get_status(workspace, workspace_bytes, stream);
  return OPD_OK;
}

opd_status opd_seq_mean_token_mean_from_counts(const int32_t* seg_id, const uint8_t* mask, int64_t T, int64_t n_ids,
                                               const int32_t* counts, float eps, const float* loss_in,
                                               float* w_out, float* loss_out, void* workspace,
                                               size_t workspace_bytes, void* stream) {
  if (T < 0 || T > (int64_t)0x7FFF0000 || n_ids < 1 || n_ids > (int64_t)0x3FFF0000 || !(eps >= 0.0f))
    return OPD_ERR_INVALID_ARG;
  if ((T > 0 && (!seg_id || !mask)) || !counts) return OPD_ERR_INVALID_ARG;
  // the loss is requested by loss_out; its input may be absent only when there are no rows
  if ((loss_out && T > 0 && !loss_in) || (!w_out && !loss_out)) return OPD_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < opd_seq_mean_token_mean_workspace_size(n_ids))
    return OPD_ERR_INVALID_ARG;
  const DeviceInfo dev = device_info();
  if (dev.sm_count <= 0) return OPD_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  Ctrl* ctrl = static_cast<Ctrl*>(workspace);
  OPD_CUDA(timed("seq_from_counts", s, [&] {
    return launch_seq_from_counts(seg_id, mask, (int32_t)T, (int32_t)n_ids, counts, eps, loss_out ? loss_in : nullptr,
                                  w_out, loss_out, ctrl, static_cast<uint8_t*>(workspace) + sizeof(Ctrl),
                                  dev.sm_count, s);
  }));
  if (cudaGetLastError() != cudaSuccess) return OPD_ERR_CUDA;
  if (env_flag("OPD_KL_SYNC_CHECK")) {
    OPD_CUDA(launch_check_finite(w_out, w_out ? (size_t)T : 0, ctrl, dev.sm_count, s));
    OPD_CUDA(launch_check_finite(loss_out, 1, ctrl, dev.sm_count, s));
    return opd_kl_get_status(workspace, workspace_bytes, stream);
  }
  return OPD_OK;
}

opd_status opd_kl_get_status(void* workspace, size_t workspace_bytes, void* stream) {
  if (!workspace || workspace_bytes < sizeof(Ctrl) || !aligned(workspace, 256)) return OPD_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return OPD_ERR_CUDA;
  uint32_t st = 0;
  Ctrl* ctrl = static_cast<Ctrl*>(workspace);
  if (cudaMemcpy(&st, &ctrl->status, sizeof st, cudaMemcpyDeviceToHost) != cudaSuccess) return OPD_ERR_CUDA;
  const uint32_t zero = 0;
  if (cudaMemcpy(&ctrl->status, &zero, sizeof zero, cudaMemcpyHostToDevice) != cudaSuccess) return OPD_ERR_CUDA;
  if (st & kDevTimeout) return OPD_ERR_TIMEOUT;
  if (st & kDevBadToken) return OPD_ERR_INVALID_ARG;
  if (st & kDevBadShape) return OPD_ERR_UNSUPPORTED;
  if (st & kDevNonFinite) return OPD_ERR_NONFINITE;
  return OPD_OK;
}

opd_status opd_kl_selftest_timeout(void* workspace, size_t workspace_bytes, uint64_t limit_ns, void* stream) {
  if (!workspace || workspace_bytes < sizeof(Ctrl) || !aligned(workspace, 256)) return OPD_ERR_INVALID_ARG;
  if (limit_ns == 0 || limit_ns > 1000000000ull) return OPD_ERR_INVALID_ARG;
  OPD_CUDA(launch_selftest_timeout(static_cast<Ctrl*>(workspace), limit_ns, static_cast<cudaStream_t>(stream)));
  return opd_kl_get_status(workspace, workspace_bytes, stream);
}

opd_status opd_kl_profile_start(void) {
  Profiler& P = profiler();
  std::lock_guard<std::mutex> lock(P.mu);
  for (auto& r : P.recs) {
    P.pool.push_back(r.a);
    P.pool.push_back(r.b);
  }
  P.recs.clear();
  P.on = true;
  return OPD_OK;
}

opd_status opd_kl_profile_stop(opd_kernel_time* out, int capacity, int* n_out) {
  Profiler& P = profiler();
  std::lock_guard<std::mutex> lock(P.mu);
  P.on = false;
  std::vector<opd_kernel_time> agg;
  opd_status st = OPD_OK;
  for (auto& r : P.recs) {
    float ms = 0.f;
    if (cudaEventSynchronize(r.b) != cudaSuccess || cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess) {
      st = OPD_ERR_CUDA;
      ms = 0.f;
    }
    size_t k = 0;
    while (k < agg.size() && std::strncmp(agg[k].name, r.name, sizeof agg[k].name) != 0) ++k;
    if (k == agg.size()) {
      opd_kernel_time t{};
      std::strncpy(t.name, r.name, sizeof t.name - 1);
      agg.push_back(t);
    }
    agg[k].launches += 1;
    agg[k].total_ms += ms;
    P.pool.push_back(r.a);
    P.pool.push_back(r.b);
  }
  P.recs.clear();
  if (n_out) *n_out = (int)agg.size();
  for (int i = 0; out && i < capacity && i < (int)agg.size(); ++i) out[i] = agg[i];
  return st;
}

const char* opd_status_string(opd_status status) {
  switch (status) {
    case OPD_OK: return "OPD_OK";
    case OPD_ERR_INVALID_ARG: return "OPD_ERR_INVALID_ARG";
    case OPD_ERR_UNSUPPORTED: return "OPD_ERR_UNSUPPORTED";
    case OPD_ERR_CUDA: return "OPD_ERR_CUDA";
    case OPD_ERR_TIMEOUT: return "OPD_ERR_TIMEOUT";
    case OPD_ERR_NONFINITE: return "OPD_ERR_NONFINITE";
  }
  return "OPD_ERR_UNKNOWN";
}

}  // extern "C"
