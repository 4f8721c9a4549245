/*
 * opd_kl.h: C ABI of the fused on-policy-distillation reverse-KL step on one
 * NVIDIA GB300 (sm_103a).
 *
 * What is computed (ActFirst-OPD, Section 3, Eq. opd-objective and
 * Eq. reverse-kl; masking and the frozen teacher from Appendix B.4):
 *
 *   for every packed token row i with mask[i] = 1 (a model-generated response
 *   token; prompts, observations, inserted thinking-budget tokens and padding
 *   have mask 0):
 *     z_s = H_s[i,:] W_s^T,  z_t = H_t[i,:] W_t^T         (length V logits)
 *     u = z / temperature,   log p = u - logsumexp(u)     (student s, teacher t)
 *     KL_i = sum_v p_s[v] (log p_s[v] - log p_t[v])       reverse KL, student || teacher
 *   and, given upstream weights g_i = dL/dKL_i,
 *     dz_i[v] = (g_i / temperature) p_s[v] (log p_s[v] - log p_t[v] - KL_i)
 *     dH_s[i,:] = dz_i W_s,    dW_s = sum_i dz_i^T H_s[i,:]
 *   Rows with mask 0 get KL_i = 0 and dH_s[i,:] = 0 and add nothing to dW_s.
 *   The teacher is frozen: no gradient for H_t or W_t.
 *
 * Layouts: every matrix is dense row-major.
 *   H_s [T, d_s], H_t [T, d_t]   hidden states at the token positions
 *   W_s [V, d_s], W_t [V, d_t]   LM heads in nn.Linear layout (z = H W^T)
 *   mask [T] uint8 (nonzero = supervised), kl_out [T] float, stats [T, 3] float
 *   (lse_s, lse_t, KL per row, natural log; zeros on unsupervised rows),
 *   grad_kl [T] float, dH_s [T, d_s] float, dW_s [V, d_s] float.
 *
 * Element types: OPD_DTYPE_BF16 runs the tcgen05 tensor-core path (bf16 inputs,
 * fp32 accumulation, fp32 outputs); it needs d_s and d_t multiples of 8 and
 * 16-byte aligned base addresses. OPD_DTYPE_F32 runs a CUDA-core fp32 path.
 *
 * Ownership: the caller owns and allocates every buffer (device memory),
 * including the workspace; the library allocates nothing, keeps no pointer
 * after a call returns, and enqueues all work on the given stream without
 * synchronising it (unless OPD_KL_SYNC_CHECK=1 is set in the environment, which
 * makes every call scan its float outputs for NaN and infinity, synchronise, and
 * report device-side errors, OPD_ERR_NONFINITE included).
 *
 * Errors: every argument is validated on the host before any launch; a bad
 * argument returns OPD_ERR_INVALID_ARG or OPD_ERR_UNSUPPORTED and launches
 * nothing. Launch failures return OPD_ERR_CUDA. Device-side failures (a bounded
 * wait that ran out) set a status word inside the workspace; read it with
 * opd_kl_get_status. Nothing ever traps the GPU.
 *
 * Streams are passed as void* and are cudaStream_t values (NULL = legacy default stream).
 * No call synchronises the host, so a sequence of calls can be captured in a CUDA graph.
 *
 * Tuning overrides, read from the environment at every call (defaults are the
 * measured best on GB300):
 *   OPD_KL_FUSED=bn256|pair256  fused-kernel tiling: 128 x 256 tiles on one CTA, or
 *                               256 x 256 tiles on a CTA pair (default)
 *   OPD_KL_GEMM=cta1|pair       gradient-GEMM tiling, same two choices (default pair)
 *   OPD_KL_GROUP_ROWS=n         row tiles walked together in L2 (default 10)
 *   OPD_KL_HALF_TILE=0|1        on CTA pairs, a last row tile with at most 128 rows runs at
 *                               half height, M = 128, in the fused kernels and GEMMs (default 1)
 *   OPD_KL_VSPLIT=n             exactly n vocabulary splits in the fused kernels (default 0:
 *                               searched)
 *   OPD_KL_MAX_KSPLIT=n         largest K split of the dH_s GEMM (default 16)
 *   OPD_KL_DETERMINISTIC=1      bit-reproducible dH_s: no split-K reduce-adds (KL, stats and
 *                               dW_s are bit-reproducible in every mode); the dH_s GEMM then
 *                               balances worse across the SMs
 */
#ifndef OPD_KL_H
#define OPD_KL_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  OPD_OK = 0,
  OPD_ERR_INVALID_ARG = 1, /* null pointer, bad size, misaligned buffer, workspace too small */
  OPD_ERR_UNSUPPORTED = 2, /* valid but not handled (e.g. bf16 with d % 8 != 0) */
  OPD_ERR_CUDA = 3,        /* a CUDA runtime call or launch failed */
  OPD_ERR_TIMEOUT = 4,     /* a device-side bounded wait ran out (see opd_kl_get_status) */
  OPD_ERR_NONFINITE = 5    /* debug mode (OPD_KL_SYNC_CHECK=1) only: an output holds NaN or infinity.
                              Inputs must be finite; outside debug mode nothing is checked */
} opd_status;

typedef enum { OPD_DTYPE_BF16 = 0, OPD_DTYPE_F32 = 1 } opd_dtype;

/* One problem: T packed token rows, hidden sizes, vocabulary size, element type
 * of H_s/H_t/W_s/W_t, and the softmax temperature applied to both policies. */
typedef struct {
  int64_t T;
  int64_t d_s;
  int64_t d_t;
  int64_t V;
  int32_t dtype;       /* opd_dtype */
  float temperature;   /* > 0 */
} opd_problem;

/* Bytes of device workspace that forward, backward and fwd_bwd need for this
 * problem (an upper bound: it assumes every row may be supervised). Returns 0
 * for an invalid problem. The workspace must be 256-byte aligned. Its largest
 * part is the bf16 dz buffer of T x V elements. To bound it, split a batch into
 * row chunks: give each chunk its rows' upstream weights (computed once for the
 * whole batch) and pass accumulate_dW = 1 after the first chunk; the results equal
 * one call over the whole batch. */
size_t opd_kl_workspace_size(const opd_problem* problem);

/* Bytes of device workspace that the forward-only calls need: opd_kl_forward and
 * opd_score_tokens. It is the leading part of the opd_kl_workspace_size layout
 * (control block, row indices, gathered rows, per-split statistics) without the
 * backward's row constants, dz buffer and dH_s partial sums, so a forward at the
 * Qwen3-1.7B shape (T = 16,384, d_s = 2,048, d_t = 4,096, V = 151,936) needs 0.24 GB
 * instead of 5.36 GB.
 * A workspace of either size serves those two calls; the backward, fwd_bwd and
 * surrogate calls need the full size. Returns 0 for an invalid problem. */
size_t opd_kl_forward_workspace_size(const opd_problem* problem);

/* Forward (Eq. reverse-kl): per-token KL and the per-row statistics the backward
 * needs. kl_out [T] and stats [T, 3] are written for every row (zeros on
 * unsupervised rows). The workspace needs opd_kl_forward_workspace_size bytes. */
opd_status opd_kl_forward(const opd_problem* problem, const void* H_s, const void* H_t, const void* W_s,
                          const void* W_t, const uint8_t* mask, float* kl_out, float* stats, void* workspace,
                          size_t workspace_bytes, void* stream);

/* Backward: given stats from opd_kl_forward on the same inputs and grad_kl [T]
 * (dL/dKL_i; entries on unsupervised rows are ignored), writes dH_s [T, d_s]
 * (zeros on unsupervised rows) and dW_s [V, d_s]; with accumulate_dW != 0 the
 * dW_s contribution is added to what dW_s already holds. */
opd_status opd_kl_backward(const opd_problem* problem, const void* H_s, const void* H_t, const void* W_s,
                           const void* W_t, const uint8_t* mask, const float* stats, const float* grad_kl,
                           float* dH_s, float* dW_s, int accumulate_dW, void* workspace, size_t workspace_bytes,
                           void* stream);

/* Forward then backward in one call (row compaction and gathering done once):
 * writes kl_out, stats, dH_s and dW_s as the two calls above would. */
opd_status opd_kl_fwd_bwd(const opd_problem* problem, const void* H_s, const void* H_t, const void* W_s,
                          const void* W_t, const uint8_t* mask, const float* grad_kl, float* kl_out, float* stats,
                          float* dH_s, float* dW_s, int accumulate_dW, void* workspace, size_t workspace_bytes,
                          void* stream);

/* The paper's aggregation of the per-token KL into one batch loss (Appendix B.4: the
 * seq-mean-token-mean of Eq. opd-surrogate, here applied to KL_i):
 *   w_i = mask_i / (|B| (n_seg(i) + eps)),   L = sum_i w_i KL_i
 * with n_b the supervised tokens of response b and |B| the distinct response ids. One call
 * computes the weights on the device (as opd_seq_mean_token_mean_device), the forward
 * with L summed inside its combine pass (in double, in no fixed order) and the backward
 * with grad_kl = w. Writes loss_out[0] = L, kl_out [T], stats [T, 3], dH_s = dL/dH_s
 * (zeros on masked rows) and dW_s = dL/dW_s (added to dW_s when accumulate_dW != 0).
 * seg_id [T] int32: each row's response id, -1 outside responses; an id >= n_ids is
 * skipped and reported by opd_kl_get_status as OPD_ERR_INVALID_ARG. The workspace holds
 * opd_kl_seq_mean_workspace_size(problem, n_ids) bytes: the reverse-KL workspace, T
 * weights and the response counters (0 for an invalid problem or n_ids < 1). */
size_t opd_kl_seq_mean_workspace_size(const opd_problem* problem, int64_t n_ids);
opd_status opd_kl_seq_mean_fwd_bwd(const opd_problem* problem, const void* H_s, const void* H_t, const void* W_s,
                                   const void* W_t, const uint8_t* mask, const int32_t* seg_id, int64_t n_ids,
                                   float eps, float* loss_out, float* kl_out, float* stats, float* dH_s,
                                   float* dW_s, int accumulate_dW, void* workspace, size_t workspace_bytes,
                                   void* stream);

/* Token scoring under one head (the frozen teacher's scores, or the student's):
 * for every row with mask[i] = 1,
 *   lse_out[i]  = logsumexp_v (H[i,:] . W[v,:]) / temperature
 *   logp_out[i] = (H[i,:] . W[tokens[i],:]) / temperature - lse_out[i]
 * (zeros on rows with mask 0). ActFirst-OPD Appendix B.4: the teacher's log-probability
 * of each generated token enters the token advantage (Eq. opd-token-advantage), the
 * student's enters the ratio (Eq. opd-ratio). H [T, d], W [V, d] bf16 with d =
 * problem->d_s (problem->d_t is not used; pass any valid value, e.g. d_s); tokens [T]
 * int32 in [0, V) (an id outside that range sets the workspace status, reported as
 * OPD_ERR_INVALID_ARG by opd_kl_get_status). The workspace needs opd_kl_forward_workspace_size
 * bytes, as for opd_kl_forward. bf16 only
 * (OPD_ERR_UNSUPPORTED otherwise). */
opd_status opd_score_tokens(const opd_problem* problem, const void* H, const void* W, const int32_t* tokens,
                            const uint8_t* mask, float* lse_out, float* logp_out, void* workspace,
                            size_t workspace_bytes, void* stream);

/* Constants of the dual-clip surrogate; NULL means the paper's values
 * (delta = 0.2, kappa = 3, log-ratio clip 20; Appendix B.4). */
typedef struct {
  float delta;           /* clipping width of the ratio, 0 <= delta < 1 */
  float kappa;           /* dual-clip constant, > 0 */
  float log_ratio_clip;  /* bound on |log ratio| before exponentiation, > 0 */
} opd_surrogate_params;

/* The sampled-token surrogate the paper optimises (Appendix B.4, Eq. opd-token-advantage,
 * opd-ratio, opd-dual-clip, opd-surrogate), forward and backward, student side:
 *   logp_i = log pi_student(tokens[i])                       (full-vocabulary softmax of H_s W_s^T / tau)
 *   A_i    = logp_teacher[i] - logp_old[i]                    (stop-gradient)
 *   rho_i  = exp(clip(logp_i - logp_old[i], -c, c))
 *   l_clip = -min(rho A, clip(rho, 1 - delta, 1 + delta) A);  l_i = min(l_clip, -kappa A) if A < 0
 *   L = sum_i weights[i] l_i   (weights: e.g. opd_seq_mean_token_mean_weights)
 * Writes loss_out[i] = l_i and logp_out[i] (zeros on rows with mask 0), dH_s [T, d_s] =
 * dL/dH_s (zeros on masked rows) and dW_s [V, d_s] = dL/dW_s (added to dW_s when
 * accumulate_dW != 0). The teacher enters only through logp_teacher (frozen). Sizes and
 * workspace as for opd_kl_fwd_bwd with d_t unused; bf16 only. Token ids as for
 * opd_score_tokens. */
opd_status opd_surrogate_fwd_bwd(const opd_problem* problem, const void* H_s, const void* W_s,
                                 const int32_t* tokens, const float* logp_old, const float* logp_teacher,
                                 const uint8_t* mask, const float* weights, const opd_surrogate_params* params,
                                 float* loss_out, float* logp_out, float* dH_s, float* dW_s, int accumulate_dW,
                                 void* workspace, size_t workspace_bytes, void* stream);

/* Largest T that opd_kl_forward_noalloc accepts. */
#define OPD_KL_NOALLOC_MAX_ROWS 4096

/* opd_kl_forward without a workspace, for callers that cannot allocate device
 * memory: hosts that own every byte of the GPU (a serving process or plugin host
 * with a fixed pool) and do not let a library call cudaMalloc. The paper has no
 * counterpart; this is a deployment convenience. Same inputs and outputs as
 * opd_kl_forward (bf16 only), same results within the parity tolerance.
 *   - Scratch is a fixed 5,259,520-byte array in the library's device memory,
 *     held by every GPU that loads the library until the process exits.
 *   - T above OPD_KL_NOALLOC_MAX_ROWS returns OPD_ERR_UNSUPPORTED (use
 *     opd_kl_forward); F32 problems also return OPD_ERR_UNSUPPORTED.
 *   - The first call on each device looks up the array's device address with
 *     that device current; make that first call before any stream capture.
 *   - All calls share the array, which keeps the last call's contents (each call
 *     resets what must start at zero), so calls whose kernels overlap on the
 *     GPU race on it: serialise them on one stream.
 *   - Rows are not compacted: unsupervised rows are computed and then written
 *     as zeros, so the tensor-core work scales with T rather than with the
 *     supervised count.
 *   - Device-side failures: there is no workspace, so opd_kl_get_status cannot
 *     report them. If a bounded wait of the call runs out, the call fills every
 *     kl_out and stats entry with NaN instead. It still returns OPD_OK, because it
 *     does not synchronise; only with OPD_KL_SYNC_CHECK=1 does it synchronise and
 *     return OPD_ERR_TIMEOUT (or OPD_ERR_NONFINITE for a non-finite output).
 * Allocates nothing: no cudaMalloc, cudaFree or allocating library call. */
opd_status opd_kl_forward_noalloc(const opd_problem* problem, const void* H_s, const void* H_t, const void* W_s,
                                  const void* W_t, const uint8_t* mask, float* kl_out, float* stats, void* stream);

/* Host helper (Appendix B.4, Eq. opd-surrogate, seq-mean-token-mean): upstream
 * weights w_i = dL/dl_i for L = 1/|B| sum_b (sum_j m_bj l_bj) / (sum_j m_bj + eps).
 * seg_id [T]: response index of row i (>= 0) or negative outside any response;
 * |B| = number of distinct non-negative ids. w_out [T] host memory; rows with
 * mask 0 or a negative id get 0. Returns OPD_ERR_INVALID_ARG on null pointers
 * (with T > 0), T < 0 or eps < 0. */
opd_status opd_seq_mean_token_mean_weights(const int32_t* seg_id, const uint8_t* mask, int64_t T, float eps,
                                           float* w_out);

/* The same weights on the device, for a training step that stays on the GPU:
 * seg_id [T] int32 and mask [T] uint8 in device memory, response ids in [0, n_ids) (ids < 0
 * mark rows outside every response; an id >= n_ids sets the workspace status, reported as
 * OPD_ERR_INVALID_ARG by opd_kl_get_status). Writes w_out [T] (device, may be NULL) and,
 * when loss_out [1] is given, loss_out[0] = sum_i w_i loss_in[i], which is the paper's L for
 * per-token losses loss_in [T] (accumulated in double; the summation order is not fixed).
 * loss_in is required with loss_out unless T = 0 (then L = 0). At least one of the two
 * outputs must be requested.
 * The workspace (device, 256-byte aligned) holds opd_seq_mean_token_mean_workspace_size(n_ids)
 * bytes; it starts with the status word opd_kl_get_status reads. */
size_t opd_seq_mean_token_mean_workspace_size(int64_t n_ids);
opd_status opd_seq_mean_token_mean_device(const int32_t* seg_id, const uint8_t* mask, int64_t T, int64_t n_ids,
                                          float eps, const float* loss_in, float* w_out, float* loss_out,
                                          void* workspace, size_t workspace_bytes, void* stream);

/* The same weights for a batch whose rows are spread over several processes (token-sharded
 * data parallelism: each process holds some rows of the batch; a response may even straddle
 * two processes). The paper's L is over the whole batch (Appendix B.4, Eq. opd-surrogate),
 * so n_b and |B| must count every process's rows. Two calls per process, with one sum over
 * processes between them:
 *   1. opd_seq_mean_token_mean_counts writes counts [2, n_ids] int32 (device): row b of the
 *      first plane is the number of this process's supervised rows of response b, of the
 *      second plane the number of all its rows of response b. An id >= n_ids is skipped and
 *      sets the workspace status (OPD_ERR_INVALID_ARG from opd_kl_get_status).
 *   2. The caller sums counts over the processes (an all-reduce of 2 n_ids int32 values).
 *   3. opd_seq_mean_token_mean_from_counts takes the summed counts and writes this process's
 *      weights w_out [T] (may be NULL) and, when loss_out [1] is given, loss_out[0] = sum over
 *      this process's rows of w_i loss_in[i] (in double, in no fixed order; loss_in [T] is
 *      required unless T = 0, where the part is 0). The sum of loss_out over the processes is
 *      the batch loss L. At least one of w_out and loss_out must be given.
 * Response ids are global ids in [0, n_ids) (ids < 0 mark rows outside every response).
 * With one process the result equals opd_seq_mean_token_mean_device. Workspaces as for
 * opd_seq_mean_token_mean_device (the status word of step 1 stays set through step 3).
 * seg_id, mask, counts, loss_in, w_out and loss_out are device memory. */
opd_status opd_seq_mean_token_mean_counts(const int32_t* seg_id, const uint8_t* mask, int64_t T, int64_t n_ids,
                                          int32_t* counts, void* workspace, size_t workspace_bytes, void* stream);
opd_status opd_seq_mean_token_mean_from_counts(const int32_t* seg_id, const uint8_t* mask, int64_t T, int64_t n_ids,
                                               const int32_t* counts, float eps, const float* loss_in,
                                               float* w_out, float* loss_out, void* workspace,
                                               size_t workspace_bytes, void* stream);

/* Reads and clears the device status word in the workspace, after
 * synchronising the stream: OPD_OK, OPD_ERR_TIMEOUT if a bounded wait in the last
 * call ran out, or OPD_ERR_INVALID_ARG if a token id was outside [0, V) (or a response
 * id outside [0, n_ids) in opd_seq_mean_token_mean_device). */
opd_status opd_kl_get_status(void* workspace, size_t workspace_bytes, void* stream);

/* Self-test of the bounded-wait machinery: launches one kernel that waits on a
 * barrier nothing completes, with the given limit (nanoseconds, at most 1e9),
 * then reads the status as opd_kl_get_status does. Returns OPD_ERR_TIMEOUT when
 * the wait gave up as designed; the CUDA context stays usable. */
opd_status opd_kl_selftest_timeout(void* workspace, size_t workspace_bytes, uint64_t limit_ns, void* stream);

/* Per-kernel timing of the library's own launches, for roofline accounting.
 * Between opd_kl_profile_start and opd_kl_profile_stop every kernel the library
 * launches is bracketed by two CUDA events recorded on the caller's stream (off
 * by default; when on it adds two event records per launch). stop() waits for
 * those events, then writes up to `capacity` entries (one per kernel name: launch
 * count and summed event time in milliseconds) to `out` (host memory), sets
 * *n_out to the number of distinct kernels, and turns timing off. */
typedef struct {
  char name[48];
  int64_t launches;
  double total_ms;
} opd_kernel_time;

opd_status opd_kl_profile_start(void);
opd_status opd_kl_profile_stop(opd_kernel_time* out, int capacity, int* n_out);

/* Human-readable name of a status code (static storage). */
const char* opd_status_string(opd_status status);

#ifdef __cplusplus
}
#endif

#endif /* OPD_KL_H */
