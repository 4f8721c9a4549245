// Internal interface between the C-ABI layer (opd_api.cu) and the kernel
// translation units. Not installed; not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace opd {

struct Ctrl;

// Tile geometry shared by host and device code.
constexpr int kRowTile = 128;   // token rows per MMA tile (TMEM lanes)
constexpr int kKBlock = 64;     // bf16 elements per 128-byte swizzled row
constexpr int kMaxVSplit = 128; // vocabulary splits of the forward statistics (partials planes)
constexpr int kMaxKSplit = 16;  // K splits of the dH_s GEMM
constexpr int kRowPad = 256;    // gathered rows are zero-padded to a multiple of this
constexpr int kGemmBN = 256;    // output columns per gradient-GEMM tile

// Fused-kernel tilings: 128 x 256 tiles on one CTA, or 256 x 256 tiles on a CTA
// pair (tcgen05 cta_group::2).
enum FusedMode : int32_t { kFusedDefault = 0, kFusedBN256 = 2, kFusedPair256 = 3 };
constexpr FusedMode kFusedDefaultMode = kFusedPair256;

// Rows of W (vocabulary entries) one CTA stages per tile: the W tensor maps' box height.
constexpr int fused_w_box(int mode) { return mode == kFusedBN256 ? 256 : 128; }

struct FusedParams {
  Ctrl* ctrl;
  int32_t V, d_s, d_t;
  int32_t T_pad;        // rows of the gathered buffers (multiple of kRowPad)
  int32_t group_rows;   // row tiles walked together (L2 raster group)
  float k2;             // log2(e) / tau
  float inv_tau;
  uint64_t wait_limit_ns;
  float* partials;      // forward: [max_vsplit][5][T_pad]
  int32_t max_vsplit;   // vocabulary splits the forward may use (<= kMaxVSplit; sizes partials)
  const float4* rowc;   // backward: [T_pad] = (lse_s log2 e, lse_s - lse_t + KL, g / tau, 0)
  int32_t mode;         // FusedMode; the W tensor maps' box height must be fused_w_box(mode)
  int32_t half_tile;    // 1: on CTA pairs, a last row tile with at most 128 rows runs as M = 128 MMAs
  int32_t vsplit;       // > 0: exactly this many vocabulary splits (capped by max_vsplit); 0: searched
};

inline int fused_mode(const FusedParams& p) { return p.mode == kFusedDefault ? kFusedDefaultMode : p.mode; }

struct GemmParams {
  Ctrl* ctrl;
  int32_t M, N, K;      // sizes; M or K is replaced by the supervised row count when flagged
  int32_t m_is_R, k_is_R;
  int32_t max_ksplit;   // 1 = whole K per tile
  int32_t reduce;       // 1 = TMA reduce-add into C, 0 = TMA store
  int32_t pair;         // 1 = 256 x 256 tiles on CTA pairs (B must be MN-major), 0 = 128 x 256 on one CTA
  int32_t work_slot;    // pairs: the Ctrl::work counter this launch takes its tiles from (2 or 3)
  int32_t half_tile;    // 1: on CTA pairs, a last M tile with at most 128 rows runs as M = 128 MMAs
  uint64_t wait_limit_ns;
};

// Per-token finish of single-head scoring and of the sampled-token surrogate (opd_surrogate.cu).
struct HeadRowsParams {
  const Ctrl* ctrl;             // R and the forward's split count
  Ctrl* ctrl_rw;                // status word (bad token ids)
  const float* partials;        // [split][5][T_pad] base-2 statistics (planes 0, 1 used)
  int32_t T, T_pad, V, d;
  const int32_t* pos;           // token row -> gathered rank or -1
  const __nv_bfloat16* H_g;     // gathered rows [T_pad, d]
  const __nv_bfloat16* W;       // head [V, d]
  const int32_t* tokens;        // [T]
  float inv_tau;
  float* lse_out;               // [T] (may be null)
  float* logp_out;              // [T] (may be null)
  int32_t surrogate;            // 1: also the dual-clip loss and the backward constants
  const float* logp_old;        // [T]
  const float* logp_teacher;    // [T]
  const float* weights;         // [T] upstream weight of each token's loss
  float delta, kappa, clip;
  float* loss_out;              // [T]
  float4* rowc;                 // [T_pad] (lse log2 e, coef, token bits, 0)
};

// aux kernels (opd_aux.cu)
cudaError_t launch_compact(const uint8_t* mask, int32_t T, int32_t* idx, int32_t* pos, Ctrl* ctrl,
                           cudaStream_t s);
cudaError_t launch_gather_bf16(const void* H_s, const void* H_t, int32_t d_s, int32_t d_t, const int32_t* idx,
                               const Ctrl* ctrl, void* Hs_g, void* Ht_g, int32_t T_pad, int n_sm, cudaStream_t s);
// weights != nullptr: also adds sum_i weights[i] KL_i to *loss_acc (the batch loss, fused here).
// idx maps gathered rows to token rows; nullptr: gathered row r is token row r.
cudaError_t launch_combine(const float* partials, const int32_t* pos, const int32_t* idx, const Ctrl* ctrl,
                           int32_t T, int32_t T_pad, float* kl_out, float* stats, const float* weights,
                           double* loss_acc, int n_sm, cudaStream_t s);
cudaError_t launch_bwd_rowc(const float* stats, const float* grad_kl, const int32_t* idx, const Ctrl* ctrl,
                            int32_t T_pad, float tau, float4* rowc, cudaStream_t s);
cudaError_t launch_zero_rows(float* buf, int32_t cols, const Ctrl* ctrl, int32_t T_pad, int n_sm, cudaStream_t s);
cudaError_t launch_scatter_rows(const float* src_g, int32_t cols, const int32_t* pos, int32_t T, float* dst,
                                int n_sm, cudaStream_t s);
cudaError_t launch_selftest_timeout(Ctrl* ctrl, uint64_t limit_ns, cudaStream_t s);
// Debug mode only: sets the non-finite status bit if p[0..n) holds a NaN or infinity.
cudaError_t launch_check_finite(const float* p, size_t n, Ctrl* ctrl, int n_sm, cudaStream_t s);

// fp32 CUDA-core path (opd_simt.cu)
cudaError_t launch_simt_forward(const float* H_s, const float* H_t, const float* W_s, const float* W_t,
                                int32_t T, int32_t d_s, int32_t d_t, int32_t V, float tau, const int32_t* idx,
                                const int32_t* pos, const Ctrl* ctrl, float* kl_out, float* stats,
                                cudaStream_t s);
cudaError_t launch_simt_backward(const float* H_s, const float* H_t, const float* W_s, const float* W_t,
                                 int32_t T, int32_t d_s, int32_t d_t, int32_t V, float tau, const int32_t* idx,
                                 const int32_t* pos, const Ctrl* ctrl, const float* stats, const float* grad_kl,
                                 float* dZ, float* dH_s, float* dW_s, int accumulate_dW, cudaStream_t s);

// tcgen05 kernels (opd_fused.cu, opd_gemm.cu)
cudaError_t launch_fused_forward(const CUtensorMap& hs, const CUtensorMap& ht, const CUtensorMap& ws,
                                 const CUtensorMap& wt, const FusedParams& p, int grid, cudaStream_t s);
cudaError_t launch_fused_backward(const CUtensorMap& hs, const CUtensorMap& ht, const CUtensorMap& ws,
                                  const CUtensorMap& wt, const CUtensorMap& dz_store, const FusedParams& p,
                                  int grid, cudaStream_t s);
// Single-head variants (scoring, surrogate): the head's rows and weights come in the
// student slots; forward writes base-2 (max, sum) partials, backward writes
// dz = coef (1[k = x] - p) from rowc = (lse log2 e, coef, token bits, 0).
cudaError_t launch_head_forward(const CUtensorMap& h, const CUtensorMap& w, const FusedParams& p, int grid,
                                cudaStream_t s);
cudaError_t launch_head_backward(const CUtensorMap& h, const CUtensorMap& w, const CUtensorMap& dz_store,
                                 const FusedParams& p, int grid, cudaStream_t s);
cudaError_t launch_head_rows(const HeadRowsParams& p, int n_sm, cudaStream_t s);
// seq-mean-token-mean on the device (opd_seqmean.cu). Scratch of seq_mean_token_mean_scratch_bytes
// (starts with the double loss accumulator); bad response ids set ctrl->status, which the first
// kernel clears when clear_status is set.
size_t seq_mean_token_mean_scratch_bytes(int64_t n_ids);
double* seq_mean_token_mean_acc(void* scratch);
cudaError_t launch_seq_mean_token_mean(const int32_t* seg, const uint8_t* mask, int32_t T, int32_t n_ids, float eps,
                                       const float* loss_in, float* w_out, float* loss_out, Ctrl* ctrl,
                                       bool clear_status, void* scratch, int n_sm, cudaStream_t s);
cudaError_t launch_store_loss(const double* acc, float* loss_out, cudaStream_t s);
// The histogram pass alone, into counts [2, n_ids] (supervised rows, then all rows, per id);
// clears ctrl->status first, and bad ids set it.
cudaError_t launch_seq_counts(const int32_t* seg, const uint8_t* mask, int32_t T, int32_t n_ids, int32_t* counts,
                              Ctrl* ctrl, int n_sm, cudaStream_t s);
// Weights (and sum_i w_i loss_in[i]) from a histogram summed over processes (ctrl->status is
// left as the histogram pass set it); scratch holds
// the double accumulator and |B| (seq_mean_token_mean_scratch_bytes(0) bytes suffice).
cudaError_t launch_seq_from_counts(const int32_t* seg, const uint8_t* mask, int32_t T, int32_t n_ids,
                                   const int32_t* counts, float eps, const float* loss_in, float* w_out,
                                   float* loss_out, Ctrl* ctrl, void* scratch, int n_sm, cudaStream_t s);
// C = A * B^T with A [M, K] and B [N, K] given through tensor maps; a_mn / b_mn select
// MN-major operand tiles (the operand's contiguous dimension is M or N, not K).
cudaError_t launch_gemm(bool a_mn, bool b_mn, const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c,
                        const GemmParams& p, int grid, cudaStream_t s);

}  // namespace opd
