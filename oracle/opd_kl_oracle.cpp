// Float64 CPU oracle for the token-level OPD reverse-KL step and its gradient.
//
// TEST INFRASTRUCTURE ONLY. Nothing on the product path may link, load or call
// this file: only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline /
// --impl reference legs use it. It shares no code, header, table or helper with
// the CUDA library.
//
// What it computes (ActFirst-OPD, Section 3 "On-Policy Distillation for
// Multi-Turn Agents", Eq. opd-objective and Eq. reverse-kl; mask semantics from
// Appendix B.4 "OPD Optimization"; the teacher is frozen, same appendix):
//
//   for every supervised token context i (mask[i] == 1):
//     z_s[k] = sum_j H_s[i,j] W_s[k,j]          student logits, k over the vocab
//     z_t[k] = sum_j H_t[i,j] W_t[k,j]          teacher logits
//     u = z / tau                               temperature (reading: both sides)
//     log p = u - logsumexp(u)                  two-pass log-softmax
//     KL_i = sum_k p_s[k] (log p_s[k] - log p_t[k])      reverse KL, student || teacher
//     dz[k] = g_i / tau * p_s[k] (log p_s[k] - log p_t[k] - KL_i)   = d(g_i KL_i)/d z_s[k]
//     dH_s[i,:] = sum_k dz[k] W_s[k,:]
//   dW_s[k,:] = sum_i dz_i[k] H_s[i,:]
//   masked rows (mask[i] == 0): KL_i = 0, dz = 0, dH_s[i,:] = 0, no dW_s term.
//
// Also, for the sampled-token surrogate the paper optimises (Appendix B.4,
// Eq. opd-token-advantage, opd-ratio, opd-dual-clip, opd-surrogate):
//   log pi(x_i) = u[x_i] - logsumexp(u)                 token scoring under one head
//   A_i = sg[ log pi_teacher(x_i) - log pi_old(x_i) ]    (0 on masked rows)
//   rho_i = exp(clip(log pi_student(x_i) - log pi_old(x_i), -c, c))      c = 20
//   l_clip = -min(rho A, clip(rho, 1 - delta, 1 + delta) A)             delta = 0.2
//   l_DC = min(l_clip, -kappa A) if A < 0 else l_clip                   kappa = 3
//   L = sum_i w_i l_DC,i with w the seq-mean-token-mean weights
//   dL/dz_s[i,k] = w_i dl/drho drho/dr (1/tau) (1[k = x_i] - p_s[i,k])
//
// Everything is plain: logits are materialised, sums run in index order with
// one double accumulator, no blocking, no online rescaling. Threads only split
// independent rows (phase 1) or independent vocab rows of dW_s (phase 2).
//
// Inputs are read exactly: float32 values, or bf16 bit patterns widened to
// float32 by a 16-bit shift, then to double.

#include <cmath>
#include <cstdint>
#include <cstring>
#include <thread>
#include <vector>

namespace {

enum ElemKind { KIND_F32 = 0, KIND_BF16 = 1 };

inline double load(const void* base, int kind, int64_t index) {
  if (kind == KIND_F32) return static_cast<double>(static_cast<const float*>(base)[index]);
  uint32_t bits = static_cast<uint32_t>(static_cast<const uint16_t*>(base)[index]) << 16;
  float f;
  std::memcpy(&f, &bits, sizeof f);
  return static_cast<double>(f);
}

struct Problem {
  int64_t T, d_s, d_t, V;
  double tau;
  int kind;
  const void *H_s, *H_t, *W_s, *W_t;
  const uint8_t* mask;
  const double* g;
};

// Logits of one token context under one head: z[k] = H[i,:] . W[k,:].
void logits(const void* H, const void* W, int kind, int64_t i, int64_t d, int64_t V,
            std::vector<double>& z) {
  for (int64_t k = 0; k < V; ++k) {
    double acc = 0.0;
    for (int64_t j = 0; j < d; ++j) acc += load(H, kind, i * d + j) * load(W, kind, k * d + j);
    z[k] = acc;
  }
}

// log-sum-exp by the two-pass rule: M = max_k u[k], lse = M + log sum_k exp(u[k] - M).
double logsumexp(const std::vector<double>& u) {
  double M = u[0];
  for (double x : u) M = x > M ? x : M;
  double s = 0.0;
  for (double x : u) s += std::exp(x - M);
  return M + std::log(s);
}

// Phase 1 for one row: KL, both log-partition values, dz and the dH_s row.
void one_row(const Problem& P, int64_t i, std::vector<double>& zs, std::vector<double>& zt,
             double* kl, double* lse_s_out, double* lse_t_out, double* dz, double* dH_row) {
  logits(P.H_s, P.W_s, P.kind, i, P.d_s, P.V, zs);
  logits(P.H_t, P.W_t, P.kind, i, P.d_t, P.V, zt);
  for (int64_t k = 0; k < P.V; ++k) {
    zs[k] /= P.tau;
    zt[k] /= P.tau;
  }
  const double lse_s = logsumexp(zs);
  const double lse_t = logsumexp(zt);
  if (lse_s_out) *lse_s_out = lse_s;
  if (lse_t_out) *lse_t_out = lse_t;

  const bool supervised = P.mask[i] != 0;
  double KL = 0.0;
  if (supervised) {
    for (int64_t k = 0; k < P.V; ++k) {
      const double lp_s = zs[k] - lse_s;
      const double lp_t = zt[k] - lse_t;
      KL += std::exp(lp_s) * (lp_s - lp_t);
    }
  }
  *kl = KL;

  const double gi = supervised ? P.g[i] : 0.0;
  for (int64_t k = 0; k < P.V; ++k) {
    if (!supervised) {
      dz[k] = 0.0;
      continue;
    }
    const double lp_s = zs[k] - lse_s;
    const double lp_t = zt[k] - lse_t;
    dz[k] = gi / P.tau * std::exp(lp_s) * (lp_s - lp_t - KL);
  }
  if (dH_row) {
    for (int64_t j = 0; j < P.d_s; ++j) {
      double acc = 0.0;
      for (int64_t k = 0; k < P.V; ++k) acc += dz[k] * load(P.W_s, P.kind, k * P.d_s + j);
      dH_row[j] = acc;
    }
  }
}

template <class F>
void parallel_for(int64_t n, int n_threads, F body) {
  if (n_threads <= 1 || n <= 1) {
    for (int64_t i = 0; i < n; ++i) body(i);
    return;
  }
  std::vector<std::thread> pool;
  for (int t = 0; t < n_threads; ++t) {
    pool.emplace_back([=, &body]() {
      for (int64_t i = t; i < n; i += n_threads) body(i);
    });
  }
  for (auto& th : pool) th.join();
}

}  // namespace

extern "C" {

// Evaluate the rows listed in `rows` (n_rows entries; rows == nullptr means all
// T rows in order). Outputs are indexed by position in that list:
//   kl[n], lse_s[n], lse_t[n], dZ[n, V], dH_s[n, d_s]   (each optional: nullptr)
//   dW_s[V, d_s] = sum over the listed rows                (optional)
// `g` holds the upstream weight dL/dKL_i for every one of the T rows.
// Returns 0 on success, -1 on invalid arguments.
int opd_oracle_kl(int64_t T, int64_t d_s, int64_t d_t, int64_t V, double tau, int kind,
                  const void* H_s, const void* H_t, const void* W_s, const void* W_t,
                  const uint8_t* mask, const double* g, const int64_t* rows, int64_t n_rows,
                  double* kl, double* lse_s, double* lse_t, double* dZ, double* dH_s,
                  double* dW_s, int n_threads) {
  if (T < 0 || d_s <= 0 || d_t <= 0 || V <= 0 || !(tau > 0.0)) return -1;
  if (kind != KIND_F32 && kind != KIND_BF16) return -1;
  if (!H_s || !H_t || !W_s || !W_t || !mask || !g || !kl) return -1;
  if (!rows) n_rows = T;
  for (int64_t n = 0; rows && n < n_rows; ++n)
    if (rows[n] < 0 || rows[n] >= T) return -1;

  const Problem P{T, d_s, d_t, V, tau, kind, H_s, H_t, W_s, W_t, mask, g};
  const bool want_dz = dZ != nullptr || dW_s != nullptr;
  std::vector<double> dz_all(want_dz ? static_cast<size_t>(n_rows * V) : 0);

  // Phase 1: every listed row on its own.
  parallel_for(n_rows, n_threads, [&](int64_t n) {
    const int64_t i = rows ? rows[n] : n;
    std::vector<double> zs(V), zt(V), dz_local(want_dz ? 0 : V);
    double* dz = want_dz ? &dz_all[n * V] : dz_local.data();
    one_row(P, i, zs, zt, &kl[n], lse_s ? &lse_s[n] : nullptr, lse_t ? &lse_t[n] : nullptr, dz,
            dH_s ? &dH_s[n * d_s] : nullptr);
  });
  if (dZ) std::memcpy(dZ, dz_all.data(), sizeof(double) * n_rows * V);

  // Phase 2: dW_s[k, j] = sum over listed rows n of dz[n, k] * H_s[row_n, j].
  if (dW_s) {
    parallel_for(V, n_threads, [&](int64_t k) {
      for (int64_t j = 0; j < d_s; ++j) {
        double acc = 0.0;
        for (int64_t n = 0; n < n_rows; ++n) {
          const int64_t i = rows ? rows[n] : n;
          acc += dz_all[n * V + k] * load(H_s, kind, i * d_s + j);
        }
        dW_s[k * d_s + j] = acc;
      }
    });
  }
  return 0;
}

// seq-mean-token-mean upstream weights (Appendix B.4, Eq. opd-surrogate):
//   L = 1/|B| sum_b ( sum_j m_bj l_bj / (sum_j m_bj + eps) )
// so dL/dl_i = m_i / (|B| (sum_{j in seg(i)} m_j + eps)).
// seg_id[i] >= 0 names the response row i belongs to; seg_id[i] < 0 marks a
// row outside every response (prompt or observation). |B| counts the distinct
// non-negative ids, including responses whose tokens are all masked.
// Returns 0, or -1 on invalid arguments.
int opd_oracle_seq_mean_token_mean_weights(const int32_t* seg_id, const uint8_t* mask, int64_t T,
                                           double eps, double* w_out) {
  if (T < 0 || (T > 0 && (!seg_id || !mask || !w_out))) return -1;
  int32_t max_id = -1;
  for (int64_t i = 0; i < T; ++i) max_id = seg_id[i] > max_id ? seg_id[i] : max_id;
  std::vector<double> supervised(static_cast<size_t>(max_id + 1), 0.0);
  std::vector<char> present(static_cast<size_t>(max_id + 1), 0);
  for (int64_t i = 0; i < T; ++i) {
    if (seg_id[i] < 0) continue;
    present[seg_id[i]] = 1;
    if (mask[i]) supervised[seg_id[i]] += 1.0;
  }
  double n_responses = 0.0;
  for (char p : present) n_responses += p ? 1.0 : 0.0;
  for (int64_t i = 0; i < T; ++i) {
    if (seg_id[i] < 0 || !mask[i]) {
      w_out[i] = 0.0;
      continue;
    }
    w_out[i] = 1.0 / (n_responses * (supervised[seg_id[i]] + eps));
  }
  return 0;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Token scoring and the sampled-token surrogate (Appendix B.4).
// ---------------------------------------------------------------------------

namespace {

// Per-token dual-clip PPO loss and its derivative with respect to the student
// log-probability of the sampled token (the advantage A is a constant: stop-gradient).
//   r = logp_s - logp_old; rho = exp(clip(r, -c, c)); drho/dr = rho inside (-c, c), else 0
//   l_clip = -min(rho A, clip(rho, 1-delta, 1+delta) A); the unclipped product is the
//   active branch when rho A <= clip(rho) A, otherwise the clipped one (zero slope).
//   l_DC = min(l_clip, -kappa A) when A < 0; l_clip is active when l_clip <= -kappa A.
void dual_clip_loss(double logp_s, double logp_old, double A, double delta, double kappa, double c,
                    double* loss, double* dloss_dlogp) {
  const double r = logp_s - logp_old;
  const double rc = r < -c ? -c : (r > c ? c : r);
  const double rho = std::exp(rc);
  const double drho = (r > -c && r < c) ? rho : 0.0;
  const double lo = 1.0 - delta, hi = 1.0 + delta;
  const double rho_clipped = rho < lo ? lo : (rho > hi ? hi : rho);
  const double m_unclipped = rho * A;
  const double m_clipped = rho_clipped * A;
  double l_clip, dl_drho;
  if (m_unclipped <= m_clipped) {
    l_clip = -m_unclipped;
    dl_drho = -A;
  } else {
    l_clip = -m_clipped;
    dl_drho = (rho > lo && rho < hi) ? -A : 0.0;
  }
  double l = l_clip;
  if (A < 0.0) {
    const double floor_value = -kappa * A;
    if (l_clip > floor_value) {
      l = floor_value;
      dl_drho = 0.0;
    }
  }
  *loss = l;
  *dloss_dlogp = dl_drho * drho;
}

}  // namespace

extern "C" {

// Scoring under one head for the listed rows (rows == nullptr: all T):
//   lse[n] = logsumexp_k (H[i,:] . W[k,:]) / tau,  logp[n] = (H[i,:] . W[tokens[i],:]) / tau - lse[n]
// Every listed row is scored, whatever its mask. Returns 0, or -1 on invalid arguments.
int opd_oracle_score(int64_t T, int64_t d, int64_t V, double tau, int kind, const void* H, const void* W,
                     const int32_t* tokens, const int64_t* rows, int64_t n_rows, double* lse, double* logp,
                     int n_threads) {
  if (T < 0 || d <= 0 || V <= 0 || !(tau > 0.0) || (kind != KIND_F32 && kind != KIND_BF16)) return -1;
  if (!H || !W || !tokens || !lse || !logp) return -1;
  if (!rows) n_rows = T;
  for (int64_t n = 0; n < n_rows; ++n) {
    const int64_t i = rows ? rows[n] : n;
    if (i < 0 || i >= T || tokens[i] < 0 || tokens[i] >= V) return -1;
  }
  parallel_for(n_rows, n_threads, [&](int64_t n) {
    const int64_t i = rows ? rows[n] : n;
    std::vector<double> z(V);
    logits(H, W, kind, i, d, V, z);
    for (int64_t k = 0; k < V; ++k) z[k] /= tau;
    lse[n] = logsumexp(z);
    logp[n] = z[tokens[i]] - lse[n];
  });
  return 0;
}

// Sampled-token surrogate, student side, for the listed rows (rows == nullptr: all T).
// Inputs per token row i: tokens[i] (sampled token), logp_old[i] (behaviour policy),
// logp_teacher[i] (frozen teacher), mask[i], w[i] (upstream weight of l_DC,i, e.g. the
// seq-mean-token-mean weights), constants delta, kappa and the log-ratio clip c.
// Outputs by list position: loss[n] = l_DC (0 on masked rows), logp_s[n], adv[n] = A,
// dZ[n, V] (optional), dH_s[n, d] (optional); dW_s[V, d] sums the listed rows (optional).
// Returns 0, or -1 on invalid arguments.
int opd_oracle_surrogate(int64_t T, int64_t d, int64_t V, double tau, int kind, const void* H_s, const void* W_s,
                         const int32_t* tokens, const double* logp_old, const double* logp_teacher,
                         const uint8_t* mask, const double* w, double delta, double kappa, double clip,
                         const int64_t* rows, int64_t n_rows, double* loss, double* logp_s, double* adv,
                         double* dZ, double* dH_s, double* dW_s, int n_threads) {
  if (T < 0 || d <= 0 || V <= 0 || !(tau > 0.0) || (kind != KIND_F32 && kind != KIND_BF16)) return -1;
  if (!H_s || !W_s || !tokens || !logp_old || !logp_teacher || !mask || !w || !loss || !logp_s || !adv)
    return -1;
  if (!rows) n_rows = T;
  for (int64_t n = 0; n < n_rows; ++n) {
    const int64_t i = rows ? rows[n] : n;
    if (i < 0 || i >= T || tokens[i] < 0 || tokens[i] >= V) return -1;
  }
  const bool want_dz = dZ != nullptr || dW_s != nullptr;
  std::vector<double> dz_all(want_dz ? static_cast<size_t>(n_rows * V) : 0);

  parallel_for(n_rows, n_threads, [&](int64_t n) {
    const int64_t i = rows ? rows[n] : n;
    std::vector<double> z(V), dz_local(want_dz ? 0 : V);
    double* dz = want_dz ? &dz_all[n * V] : dz_local.data();
    logits(H_s, W_s, kind, i, d, V, z);
    for (int64_t k = 0; k < V; ++k) z[k] /= tau;
    const double lse = logsumexp(z);
    const double lp = z[tokens[i]] - lse;
    logp_s[n] = lp;
    const bool supervised = mask[i] != 0;
    const double A = supervised ? logp_teacher[i] - logp_old[i] : 0.0;
    adv[n] = A;
    double l = 0.0, dl = 0.0;
    if (supervised) dual_clip_loss(lp, logp_old[i], A, delta, kappa, clip, &l, &dl);
    loss[n] = l;
    const double coef = supervised ? w[i] * dl / tau : 0.0;
    for (int64_t k = 0; k < V; ++k) {
      const double p = std::exp(z[k] - lse);
      dz[k] = coef * ((k == tokens[i] ? 1.0 : 0.0) - p);
    }
    if (dH_s) {
      for (int64_t j = 0; j < d; ++j) {
        double acc = 0.0;
        for (int64_t k = 0; k < V; ++k) acc += dz[k] * load(W_s, kind, k * d + j);
        dH_s[n * d + j] = acc;
      }
    }
  });
  if (dZ) std::memcpy(dZ, dz_all.data(), sizeof(double) * n_rows * V);
  if (dW_s) {
    parallel_for(V, n_threads, [&](int64_t k) {
      for (int64_t j = 0; j < d; ++j) {
        double acc = 0.0;
        for (int64_t n = 0; n < n_rows; ++n) {
          const int64_t i = rows ? rows[n] : n;
          acc += dz_all[n * V + k] * load(H_s, kind, i * d + j);
        }
        dW_s[k * d + j] = acc;
      }
    });
  }
  return 0;
}

// The per-token dual-clip loss and its slope with respect to logp_s, element by element,
// for direct checks of the piecewise definition.
int opd_oracle_dual_clip(int64_t n, const double* logp_s, const double* logp_old, const double* A, double delta,
                         double kappa, double clip, double* loss, double* dloss_dlogp) {
  if (n < 0 || (n > 0 && (!logp_s || !logp_old || !A || !loss || !dloss_dlogp))) return -1;
  for (int64_t i = 0; i < n; ++i) dual_clip_loss(logp_s[i], logp_old[i], A[i], delta, kappa, clip, &loss[i],
                                                 &dloss_dlogp[i]);
  return 0;
}

}  // extern "C"
