// Fused vocabulary-tiled LM-head kernel (tcgen05 + TMEM + TMA), two variants:
//
//  forward  (Section 3, Eq. reverse-kl): for a tile of 128 supervised token rows
//           and BN vocabulary columns, the student logits z_s = H_s W_s^T and the
//           teacher logits z_t = H_t W_t^T accumulate in TMEM; the epilogue folds
//           them into per-row online statistics in base 2 (x = z log2(e) / tau):
//             m_s, S_s = sum 2^(x_s - m_s), A = sum 2^(x_s - m_s) (x_s - x_t),
//             m_t, S_t = sum 2^(x_t - m_t)
//           over the columns of one vocabulary split. Logits never reach HBM.
//  backward: recomputes the same two tiles and writes
//             dz = (g / tau) p_s (log p_s - log p_t - KL)
//           (the derivative of g KL with respect to the student logits) as bf16
//           for the two gradient GEMMs.
//
// Roles (192 threads): warp 0 issues TMA loads, warp 1 allocates TMEM and issues
// the MMAs from one thread, warps 2-5 run the epilogue (one TMEM lane = one row).
// Persistent: each CTA walks work units (row tile, vocabulary range) grid-strided.
#include "opd_device.cuh"
#include "opd_internal.h"

namespace opd {

namespace {

// BN vocabulary columns per tile; NEPI epilogue warps (4, or 8 with two warps
// per TMEM lane quadrant, each taking half of the tile's columns).
template <int BN, bool BWD, int NEPI>
struct FusedCfg {
  static constexpr int kBufs = 512 / (2 * BN);  // (student, teacher) accumulator pairs in TMEM
  static constexpr int kHalves = NEPI / 4;      // epilogue warps per lane quadrant
  static constexpr int kColsPerWarp = BN / kHalves;
  static constexpr int kThreads = 64 + 32 * NEPI;
  static constexpr int kStages = BWD ? (BN == 128 ? 5 : 3) : (BN == 128 ? 6 : 4);
  static constexpr uint32_t kABytes = kRowTile * kKBlock * 2;
  static constexpr uint32_t kBBytes = BN * kKBlock * 2;
  static constexpr uint32_t kStageBytes = kABytes + kBBytes;
  static constexpr uint32_t kStagingPerWarp = BWD ? 32 * kColsPerWarp * 2 : 0;  // bf16 dz rows of one warp
  static constexpr uint32_t kMergeBytes = (!BWD && kHalves > 1) ? 4 * 5 * 32 * 4 : 0;  // per quadrant 5 x 32
  static constexpr uint32_t kBarrierBytes = 256;
  static constexpr size_t kSmem =
      1024 + (size_t)kStages * kStageBytes + NEPI * kStagingPerWarp + kMergeBytes + kBarrierBytes;
  static_assert(kColsPerWarp % 64 == 0, "whole 64-column boxes per epilogue warp");
};

// Unit u -> (row tile, vocabulary tile range). Units are grouped by `G` row tiles
// so that CTAs running at the same time share a few hidden-state tiles and a few
// vocabulary tiles in L2.
struct FusedSchedule {
  int n_rt, n_vt, n_vs, G, n_units;

  __device__ void init(int R, int V, int BN, int grid, int G_, bool bwd) {
    n_rt = (R + kRowTile - 1) / kRowTile;
    n_vt = (V + BN - 1) / BN;
    G = G_ < 1 ? 1 : G_;
    if (bwd || n_rt == 0) {
      n_vs = bwd ? n_vt : 1;
    } else {
      // fewest tiles on the busiest CTA, then the fewest splits
      long best = -1;
      n_vs = 1;
      const int max_vs = n_vt < kMaxVSplit ? n_vt : kMaxVSplit;
      for (int s = 1; s <= max_vs; ++s) {
        const long waves = ((long)n_rt * s + grid - 1) / grid;
        const long cost = waves * ((n_vt + s - 1) / s);
        if (best < 0 || cost < best) {
          best = cost;
          n_vs = s;
        }
      }
    }
    n_units = n_rt * n_vs;
  }

  __device__ void unit(int u, int& rt, int& split, int& vt_begin, int& vt_end) const {
    const int gsize = G * n_vs;
    const int g = u / gsize;
    int rows_in_g = n_rt - g * G;
    rows_in_g = rows_in_g < G ? rows_in_g : G;
    const int rem = u - g * gsize;
    split = rem / rows_in_g;
    rt = g * G + rem % rows_in_g;
    vt_begin = (int)(((long)split * n_vt) / n_vs);
    vt_end = (int)(((long)(split + 1) * n_vt) / n_vs);
  }
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// Wait without the early exit on a raised status: used only while draining.
__device__ __forceinline__ void mbar_wait_drain(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
  const uint32_t addr = smem_u32(bar);
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t it = 0; !mbar_try_wait(addr, parity); ++it) {
    if ((it & 63u) == 63u && (globaltimer_ns() - t0 > limit_ns || it >= (1u << 28))) return;
  }
}

// Fold 32 columns (or the first nvalid of them) of one row into the running
// base-2 statistics; indices stay compile-time so the values stay in registers.
// x = z k2 with k2 = log2(e) / tau; A is kept in raw logit units (times k2 at the end).
template <bool PARTIAL>
__device__ __forceinline__ void fold_chunk(const uint32_t (&rs)[32], const uint32_t (&rt)[32], int nvalid, float k2,
                                           float& ms, float& Ss, float& A, float& mt, float& St) {
  float cms = -INFINITY, cmt = -INFINITY;
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    if (!PARTIAL || j < nvalid) {
      cms = fmaxf(cms, __uint_as_float(rs[j]));
      cmt = fmaxf(cmt, __uint_as_float(rt[j]));
    }
  }
  // k2 > 0, so the scaled maximum is the maximum of the scaled values
  const float nms = fmaxf(ms, cms * k2);
  const float nmt = fmaxf(mt, cmt * k2);
  const float scs = exp2f(ms - nms);
  Ss *= scs;
  A *= scs;
  St *= exp2f(mt - nmt);
  ms = nms;
  mt = nmt;
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    if (!PARTIAL || j < nvalid) {
      const float zs = __uint_as_float(rs[j]);
      const float zt = __uint_as_float(rt[j]);
      const float e = exp2f(fmaf(zs, k2, -ms));
      Ss += e;
      A = fmaf(e, zs - zt, A);
      St += exp2f(fmaf(zt, k2, -mt));
    }
  }
}

template <int BN, bool BWD, int NEPI>
__global__ void __launch_bounds__(64 + 32 * NEPI, 1)
    k_fused_logits(const __grid_constant__ CUtensorMap tm_hs, const __grid_constant__ CUtensorMap tm_ht,
                   const __grid_constant__ CUtensorMap tm_ws, const __grid_constant__ CUtensorMap tm_wt,
                   const __grid_constant__ CUtensorMap tm_dz, const FusedParams p) {
  using C = FusedCfg<BN, BWD, NEPI>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* stage_base = smem;
  uint8_t* staging = smem + C::kStages * C::kStageBytes;
  float* merge = reinterpret_cast<float*>(staging + NEPI * C::kStagingPerWarp);
  uint64_t* full = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(merge) + C::kMergeBytes);
  uint64_t* empty = full + C::kStages;
  uint64_t* acc_full = empty + C::kStages;
  uint64_t* acc_empty = acc_full + C::kBufs;
  uint64_t* mma_done = acc_empty + C::kBufs;
  uint64_t* merge_full = mma_done + 1;   // [4], forward with two warps per quadrant
  uint64_t* merge_empty = merge_full + 4;  // [4]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(merge_empty + 4);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  uint32_t* status = &p.ctrl->status;
  const uint64_t lim = p.wait_limit_ns;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < C::kBufs; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], NEPI);
    }
    mbar_init(mma_done, 1);
    for (int qd = 0; qd < 4; ++qd) {
      mbar_init(&merge_full[qd], 1);
      mbar_init(&merge_empty[qd], 1);
    }
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&tm_hs);
    prefetch_tmap(&tm_ht);
    prefetch_tmap(&tm_ws);
    prefetch_tmap(&tm_wt);
    if (BWD) prefetch_tmap(&tm_dz);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int R = p.ctrl->R;
  FusedSchedule sch;
  sch.init(R, p.V, BN, gridDim.x, p.group_rows, BWD);
  if (!BWD && blockIdx.x == 0 && threadIdx.x == 0) p.ctrl->n_vsplit = sch.n_vs;
  const int nks = (p.d_s + kKBlock - 1) / kKBlock;
  const int nkt = (p.d_t + kKBlock - 1) / kKBlock;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      uint32_t stage = 0, phase = 0;
      bool ok = true, any = false;
      for (int u = blockIdx.x; ok && u < sch.n_units; u += gridDim.x) {
        int rt, split, vb, ve;
        sch.unit(u, rt, split, vb, ve);
        for (int vt = vb; ok && vt < ve; ++vt) {
          for (int seg = 0; ok && seg < 2; ++seg) {
            const CUtensorMap* ta = seg ? &tm_ht : &tm_hs;
            const CUtensorMap* tb = seg ? &tm_wt : &tm_ws;
            const int nk = seg ? nkt : nks;
            for (int kb = 0; kb < nk; ++kb) {
              if (!mbar_wait(&empty[stage], phase ^ 1u, status, lim)) {
                ok = false;
                break;
              }
              uint8_t* sa = stage_base + stage * C::kStageBytes;
              mbar_arrive_expect_tx(&full[stage], C::kStageBytes);
              tma_load_2d(sa, ta, &full[stage], kb * kKBlock, rt * kRowTile);
              tma_load_2d(sa + C::kABytes, tb, &full[stage], kb * kKBlock, vt * BN);
              any = true;
              if (++stage == (uint32_t)C::kStages) {
                stage = 0;
                phase ^= 1u;
              }
            }
          }
        }
      }
      if (!ok && any) {
        // Let every copy already issued land before the CTA can exit.
        for (int s = 0; s < C::kStages; ++s) {
          const uint32_t par = ((uint32_t)s < stage) ? phase : (phase ^ 1u);
          mbar_wait_drain(&full[s], par, lim);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kRowTile, BN, false, false);
      uint32_t stage = 0, phase = 0;
      int lt = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < sch.n_units; u += gridDim.x) {
        int rt, split, vb, ve;
        sch.unit(u, rt, split, vb, ve);
        for (int vt = vb; ok && vt < ve; ++vt, ++lt) {
          const int buf = lt % C::kBufs;
          const uint32_t acc_par = (uint32_t)(lt / C::kBufs) & 1u;
          if (!mbar_wait(&acc_empty[buf], acc_par ^ 1u, status, lim)) {
            ok = false;
            break;
          }
          tc_fence_after();
          for (int seg = 0; ok && seg < 2; ++seg) {
            const uint32_t d_tmem = tmem_base + (uint32_t)((buf * 2 + seg) * BN);
            const int nk = seg ? nkt : nks;
            for (int kb = 0; kb < nk; ++kb) {
              if (!mbar_wait(&full[stage], phase, status, lim)) {
                ok = false;
                break;
              }
              tc_fence_after();
              const uint32_t sa = smem_u32(stage_base + stage * C::kStageBytes);
              const uint32_t sb = sa + C::kABytes;
#pragma unroll
              for (int k = 0; k < kKBlock / 16; ++k) {
                umma_bf16(d_tmem, sdesc_sw128(sa + k * 32, 16, 1024), sdesc_sw128(sb + k * 32, 16, 1024), idesc,
                          (kb | k) != 0);
              }
              umma_commit(&empty[stage]);
              if (++stage == (uint32_t)C::kStages) {
                stage = 0;
                phase ^= 1u;
              }
            }
          }
          if (ok) umma_commit(&acc_full[buf]);
        }
      }
      // Every MMA issued by this thread completes before TMEM is released.
      umma_commit(mma_done);
      mbar_wait_drain(mma_done, 0, lim);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int ew = warp - 2;                 // epilogue warp index
    const int q = warp & 3;                  // TMEM lane quadrant this warp may access
    const int half = ew / 4;                 // which share of the tile's columns
    const int cbase = half * C::kColsPerWarp;
    const int row_in_tile = q * 32 + lane;
    const uint32_t t_lane = (uint32_t)(q * 32) << 16;
    int lt = 0, nu = 0;
    bool ok = true;
    uint8_t* stg = staging + ew * C::kStagingPerWarp;
    for (int u = blockIdx.x; ok && u < sch.n_units; u += gridDim.x, ++nu) {
      int rt, split, vb, ve;
      sch.unit(u, rt, split, vb, ve);
      const int row = rt * kRowTile + row_in_tile;
      float ms = -INFINITY, Ss = 0.f, A = 0.f, mt = -INFINITY, St = 0.f;
      // backward row constants: p_s = 2^(z_s k2 - b1), dz = p_s ((z_s - z_t) kc - cc)
      float b1 = 0.f, kc = 0.f, cc = 0.f;
      if (BWD) {
        const float4 rc = p.rowc[row];
        b1 = rc.x;
        kc = rc.z * p.inv_tau;
        cc = rc.z * rc.y;
      }
      for (int vt = vb; vt < ve; ++vt, ++lt) {
        const int buf = lt % C::kBufs;
        const uint32_t acc_par = (uint32_t)(lt / C::kBufs) & 1u;
        // warp-uniform outcome: the TMEM loads below are .sync.aligned
        if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[buf], acc_par, status, lim))) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int col0 = vt * BN + cbase;
        const uint32_t ts = tmem_base + t_lane + (uint32_t)(buf * 2 * BN + cbase);
        const uint32_t tt = ts + BN;
#pragma unroll 1
        for (int c = 0; c < C::kColsPerWarp / 32; ++c) {
          uint32_t rs[32], rtt[32];
          tmem_ld32x2(ts + c * 32, tt + c * 32, rs, rtt);
          if (!BWD) {
            const int nvalid = p.V - (col0 + c * 32);
            if (nvalid >= 32)
              fold_chunk<false>(rs, rtt, 32, p.k2, ms, Ss, A, mt, St);
            else if (nvalid > 0)
              fold_chunk<true>(rs, rtt, nvalid, p.k2, ms, Ss, A, mt, St);
          } else {
            const int h = c >> 1;  // 64-column box of this warp's staging tile
            if ((c & 1) == 0) {
              if (lane == 0) bulk_wait_read<C::kColsPerWarp / 64 - 1>();
              __syncwarp();
            }
            uint32_t w[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) {
              float dz2[2];
#pragma unroll
              for (int e = 0; e < 2; ++e) {
                const float zs = __uint_as_float(rs[2 * j + e]);
                const float zt = __uint_as_float(rtt[2 * j + e]);
                const float ps = exp2f(fmaf(zs, p.k2, -b1));
                dz2[e] = ps * fmaf(zs - zt, kc, -cc);
              }
              w[j] = pack_bf16x2(dz2[0], dz2[1]);
            }
            const uint32_t box = smem_u32(stg + h * 4096);
            const uint32_t jb = (uint32_t)(c & 1) * 4u;
#pragma unroll
            for (int jj = 0; jj < 4; ++jj) {
              st_shared_v4(box + sw128_offset((uint32_t)lane, jb + jj), w[4 * jj], w[4 * jj + 1], w[4 * jj + 2],
                           w[4 * jj + 3]);
            }
            if (c & 1) {
              fence_proxy_async_smem();
              __syncwarp();
              if (lane == 0) {
                tma_store_2d(&tm_dz, stg + h * 4096, col0 + h * 64, rt * kRowTile + q * 32);
                bulk_commit();
              }
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acc_empty[buf]);
      }
      if (!BWD && ok) {
        A *= p.k2;  // A was accumulated in raw logit units
        if (C::kHalves > 1) {
          // the two warps of a quadrant fold their column shares: half 1 hands its
          // statistics to half 0 through shared memory
          float* mb = merge + q * 5 * 32;
          if (half == 1) {
            if (nu > 0 && !__all_sync(0xffffffffu, mbar_wait(&merge_empty[q], (uint32_t)(nu - 1) & 1u, status, lim))) {
              ok = false;
              break;
            }
            mb[0 * 32 + lane] = ms;
            mb[1 * 32 + lane] = Ss;
            mb[2 * 32 + lane] = A;
            mb[3 * 32 + lane] = mt;
            mb[4 * 32 + lane] = St;
            __syncwarp();
            if (lane == 0) mbar_arrive(&merge_full[q]);
            continue;
          }
          if (!__all_sync(0xffffffffu, mbar_wait(&merge_full[q], (uint32_t)nu & 1u, status, lim))) {
            ok = false;
            break;
          }
          const float ms1 = mb[0 * 32 + lane], Ss1 = mb[1 * 32 + lane], A1 = mb[2 * 32 + lane];
          const float mt1 = mb[3 * 32 + lane], St1 = mb[4 * 32 + lane];
          __syncwarp();
          if (lane == 0) mbar_arrive(&merge_empty[q]);
          const float Ms = fmaxf(ms, ms1), Mt = fmaxf(mt, mt1);
          const float f0 = exp2f(ms - Ms), f1 = exp2f(ms1 - Ms);
          Ss = Ss * f0 + Ss1 * f1;
          A = A * f0 + A1 * f1;
          St = St * exp2f(mt - Mt) + St1 * exp2f(mt1 - Mt);
          ms = Ms;
          mt = Mt;
        }
        const size_t plane = (size_t)p.T_pad;
        float* base = p.partials + (size_t)split * 5 * plane + row;
        base[0 * plane] = ms;
        base[1 * plane] = Ss;
        base[2 * plane] = A;
        base[3 * plane] = mt;
        base[4 * plane] = St;
      }
    }
    if (BWD && lane == 0) bulk_wait_all<0>();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, 512);
  }
}

template <int BN, bool BWD, int NEPI>
cudaError_t launch_fused_impl(const CUtensorMap& hs, const CUtensorMap& ht, const CUtensorMap& ws,
                              const CUtensorMap& wt, const CUtensorMap& dz, const FusedParams& p, int grid,
                              cudaStream_t s) {
  using C = FusedCfg<BN, BWD, NEPI>;
  static_assert(C::kSmem <= 232448, "shared memory budget");
  auto kern = k_fused_logits<BN, BWD, NEPI>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::kSmem);
  if (e != cudaSuccess) return e;
  kern<<<grid, C::kThreads, C::kSmem, s>>>(hs, ht, ws, wt, dz, p);
  return cudaGetLastError();
}

template <bool BWD>
cudaError_t launch_fused_bn(const CUtensorMap& hs, const CUtensorMap& ht, const CUtensorMap& ws,
                            const CUtensorMap& wt, const CUtensorMap& dz, const FusedParams& p, int grid,
                            cudaStream_t s) {
  switch (fused_bn(p)) {
    case 128: return launch_fused_impl<128, BWD, 4>(hs, ht, ws, wt, dz, p, grid, s);
    case 256: return launch_fused_impl<256, BWD, 8>(hs, ht, ws, wt, dz, p, grid, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_fused_forward(const CUtensorMap& hs, const CUtensorMap& ht, const CUtensorMap& ws,
                                 const CUtensorMap& wt, const FusedParams& p, int grid, cudaStream_t s) {
  return launch_fused_bn<false>(hs, ht, ws, wt, hs, p, grid, s);
}

cudaError_t launch_fused_backward(const CUtensorMap& hs, const CUtensorMap& ht, const CUtensorMap& ws,
                                  const CUtensorMap& wt, const CUtensorMap& dz_store, const FusedParams& p,
                                  int grid, cudaStream_t s) {
  return launch_fused_bn<true>(hs, ht, ws, wt, dz_store, p, grid, s);
}

}  // namespace opd
