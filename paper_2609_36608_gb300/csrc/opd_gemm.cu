// Gradient GEMMs of the OPD reverse-KL step on tcgen05 (bf16 in, fp32 out):
//
//   dH_s = dZ W_s      M = supervised rows, N = d_s, K = V   (A K-major, B MN-major)
//   dW_s = dZ^T H_s    M = V, N = d_s, K = supervised rows   (A and B MN-major)
//
// dZ is the bf16 gradient of the weighted per-token KL with respect to the
// student logits, written by the fused backward kernel. The teacher is frozen
// (Appendix B.4), so there is no teacher gradient.
//
// Tiles: 128 x 256 fp32 accumulators in TMEM (two buffers = 512 columns), 64-deep
// K blocks staged by TMA with 128-byte swizzle, one thread issuing MMAs, four
// epilogue warps draining TMEM through swizzled shared memory into TMA stores
// (or TMA reduce-adds, for split-K partial sums and for accumulating into dW_s).
//
// PAIR = true runs 256 x 256 tiles on a CTA pair (tcgen05 cta_group::2): each CTA
// stages its own 128 rows of A and 128 of the 256 columns of B, holds its 128 x 256
// accumulator in its own TMEM and stores it; the even CTA issues the MMAs. Per
// byte staged from L2 this does 1.5 times the MMA work of the single-CTA tile.
// Pairs take tiles in increasing order from a global counter (single CTAs walk a
// fixed stride), so the pairs that read the same A rows run them at the same time.
#include "opd_device.cuh"
#include "opd_internal.h"

namespace opd {

namespace {

constexpr int kBN = kGemmBN;
constexpr uint32_t kChunkBytes = 32 * 32 * 4;         // one 32x32 fp32 staging box
constexpr uint32_t kStagingPerWarp = 2 * kChunkBytes;

template <bool PAIR>
struct GemmCfg {
  static constexpr int kTileRows = PAIR ? 2 * kRowTile : kRowTile;  // M rows per tile (whole pair)
  static constexpr int kBCols = PAIR ? kBN / 2 : kBN;               // N columns of B one CTA stages
  static constexpr uint32_t kABytes = kRowTile * kKBlock * 2;       // 16 KB
  static constexpr uint32_t kBBytes = kBCols * kKBlock * 2;         // 32 KB (16 KB in a pair)
  static constexpr uint32_t kStageBytes = kABytes + kBBytes;
  static constexpr size_t kFixed = 1024 + 4 * kStagingPerWarp + 512;
  static constexpr int kStages = (int)((232448 - kFixed) / kStageBytes) > 6 ? 6 : (int)((232448 - kFixed) / kStageBytes);
  static constexpr size_t kSmem = kFixed + (size_t)kStages * kStageBytes;
  static_assert(kStages >= 4, "pipeline depth");
  static_assert(kSmem <= 232448, "shared memory budget");
};

struct GemmSchedule {
  int n_mt, n_nt, nkb, n_ks, n_units;
  int half_mt;  // M tile run at half height (M = 128 on a pair), or -1

  // allow_half: on a CTA pair, a last M tile with at most half of its rows in range runs
  // as M = 128 MMAs (64 rows per CTA). The split search still counts it as a full tile:
  // counting it as half picks more K splits (16 instead of 9 for dH_s at the 1.7B size),
  // whose extra reduce-adds cost more than the better balance gains (measured).
  __device__ void init(int M, int N, int K, int tile_rows, int grid, int max_ks, bool allow_half) {
    n_mt = (M + tile_rows - 1) / tile_rows;
    n_nt = (N + kBN - 1) / kBN;
    nkb = (K + kKBlock - 1) / kKBlock;
    half_mt = (allow_half && n_mt > 0 && M - (n_mt - 1) * tile_rows <= tile_rows / 2) ? n_mt - 1 : -1;
    n_ks = 1;
    if (max_ks > 1 && n_mt > 0 && nkb > 1) {
      long best = -1;
      const int lim = max_ks < nkb ? max_ks : nkb;
      for (int s = 1; s <= lim; ++s) {
        const long waves = ((long)n_mt * n_nt * s + grid - 1) / grid;
        const long cost = waves * ((nkb + s - 1) / s);
        if (best < 0 || cost < best) {
          best = cost;
          n_ks = s;
        }
      }
    }
    n_units = n_mt * n_nt * n_ks;
  }

  __device__ void unit(int u, int& mt, int& nt, int& kb0, int& kb1) const {
    nt = u % n_nt;
    const int r = u / n_nt;
    mt = r % n_mt;
    const int ks = r / n_mt;
    kb0 = (int)(((long)ks * nkb) / n_ks);
    kb1 = (int)(((long)(ks + 1) * nkb) / n_ks);
  }
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

template <bool A_MN, bool B_MN, bool PAIR>
__global__ void __launch_bounds__(192, 1)
    k_umma_gemm(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
                const __grid_constant__ CUtensorMap tm_c, const GemmParams p) {
  using C = GemmCfg<PAIR>;
  constexpr int kStages = C::kStages;
  constexpr uint32_t kABytes = C::kABytes;
  constexpr uint32_t kStageBytes = C::kStageBytes;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* stage_base = smem;
  uint8_t* staging = smem + kStages * kStageBytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(staging + 4 * kStagingPerWarp);
  uint64_t* empty = full + kStages;
  uint64_t* acc_full = empty + kStages;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* mma_done = acc_empty + 2;
  uint64_t* unit_full = mma_done + 1;  // [kUnitRing] (pairs)
  uint64_t* unit_empty = unit_full + kUnitRing;
  int32_t* units = reinterpret_cast<int32_t*>(unit_empty + kUnitRing);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(units + kUnitRing);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  uint32_t* status = &p.ctrl->status;
  const uint64_t lim = p.wait_limit_ns;
  const uint32_t rank = PAIR ? cluster_ctarank() : 0u;  // CTA rank within the pair
  const int worker = PAIR ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
  const int n_workers = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;
  int32_t* counter = &p.ctrl->work[p.work_slot];

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], PAIR ? 8 : 4);  // epilogue warps of the pair
    }
    mbar_init(mma_done, 1);
    // readers of each unit slot: MMA issuer and epilogue warps of the even CTA, producer
    // and epilogue warps of the odd one
    for (int i = 0; i < kUnitRing; ++i) {
      mbar_init(&unit_full[i], 1);
      mbar_init(&unit_empty[i], 2 * 5);
    }
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&tm_a);
    prefetch_tmap(&tm_b);
    prefetch_tmap(&tm_c);
  }
  if (warp == 1) {
    if (PAIR) {
      tmem_alloc_pair(tmem_slot, 512);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(tmem_slot, 512);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  if (PAIR)
    cluster_sync_all();  // barriers of both CTAs initialised before any remote use
  else
    __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int R = p.ctrl->R;
  const int M = p.m_is_R ? R : p.M;
  const int K = p.k_is_R ? R : p.K;
  GemmSchedule sch;
  sch.init(M, p.N, K, C::kTileRows, n_workers, p.max_ksplit, PAIR && p.half_tile != 0);

  if (warp == 0) {
    if (lane == 0) {
      uint32_t stage = 0, phase = 0;
      bool ok = true, any = false;
      // a pair counts both CTAs' bytes on the leader's full barriers
      const uint32_t full_leader = PAIR ? mapa_shared(smem_u32(full), 0u) : smem_u32(full);
      int next = (PAIR && rank == 0) ? atomicAdd(counter, 1) : 0;
      for (uint32_t k = 0; ok; ++k) {
        int u;
        if (!PAIR) {
          u = worker + (int)k * n_workers;
        } else if (rank == 0) {
          u = next;
          if (!publish_unit<true>(k, u, unit_full, unit_empty, units, status, lim))
            u = -1;
          else if (u < sch.n_units)
            next = atomicAdd(counter, 1);  // claimed now, used by the next iteration
        } else {
          u = take_unit<true>(k, unit_full, unit_empty, units, true, status, lim);
        }
        if (u < 0) {
          ok = false;
          break;
        }
        if (u >= sch.n_units) break;
        int mt, nt, kb0, kb1;
        sch.unit(u, mt, nt, kb0, kb1);
        // this CTA's 128 rows of A (64 used in a half-height tile) and (pair) its half of B's columns
        const int m0 = mt * C::kTileRows + (int)rank * (mt == sch.half_mt ? kRowTile / 2 : kRowTile);
        const int n0 = nt * kBN + (int)rank * (kBN - C::kBCols);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, status, lim)) {
            ok = false;
            break;
          }
          uint8_t* sa = stage_base + stage * kStageBytes;
          uint8_t* sb = sa + kABytes;
          const int k0 = kb * kKBlock;
          if (!PAIR) {
            mbar_arrive_expect_tx(&full[stage], kStageBytes);
          } else if (rank == 0) {
            mbar_arrive_expect_tx(&full[stage], 2 * kStageBytes);
          }
          const uint32_t fb = full_leader + stage * 8u;
          auto load = [&](void* dst, const CUtensorMap* m, int32_t c0, int32_t c1) {
            if (PAIR)
              tma_load_2d_pair(dst, m, fb, c0, c1);
            else
              tma_load_2d(dst, m, &full[stage], c0, c1);
          };
          if (A_MN) {
            load(sa, &tm_a, m0, k0);
            load(sa + 8192, &tm_a, m0 + 64, k0);
          } else {
            load(sa, &tm_a, k0, m0);
          }
          if (B_MN) {
#pragma unroll
            for (int i = 0; i < C::kBCols / 64; ++i) load(sb + 8192 * i, &tm_b, n0 + 64 * i, k0);
          } else {
            load(sb, &tm_b, k0, n0);
          }
          any = true;
          if (++stage == (uint32_t)kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok && any && rank == 0) {
        // let every copy already issued land before the CTA can exit (in a pair,
        // the leader's barriers also count the peer's copies)
        for (int s = 0; s < kStages; ++s) {
          const uint32_t par = ((uint32_t)s < stage) ? phase : (phase ^ 1u);
          mbar_wait_drain(&full[s], par, lim);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc_full = idesc_bf16_f32(C::kTileRows, kBN, A_MN, B_MN);
      constexpr uint32_t idesc_half = idesc_bf16_f32(C::kTileRows / 2, kBN, A_MN, B_MN);
      uint32_t stage = 0, phase = 0;
      int lt = 0;
      bool ok = true;
      for (uint32_t k = 0; ok; ++k, ++lt) {
        const int u = PAIR ? take_unit<true>(k, unit_full, unit_empty, units, false, status, lim)
                           : worker + (int)k * n_workers;
        if (u < 0) {
          ok = false;
          break;
        }
        if (u >= sch.n_units) break;
        int mt, nt, kb0, kb1;
        sch.unit(u, mt, nt, kb0, kb1);
        const uint32_t idesc = mt == sch.half_mt ? idesc_half : idesc_full;
        const int buf = lt & 1;
        const uint32_t acc_par = (uint32_t)(lt >> 1) & 1u;
        if (!mbar_wait(&acc_empty[buf], acc_par ^ 1u, status, lim)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(buf * kBN);
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait(&full[stage], phase, status, lim)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(stage_base + stage * kStageBytes);
          const uint32_t sb = sa + kABytes;
#pragma unroll
          for (int k = 0; k < kKBlock / 16; ++k) {
            // K-major: the 16-wide K slice starts 32 bytes further along each 128-byte row.
            // MN-major: it starts 16 rows (2048 bytes) further down; 64-wide MN blocks are 8 KB apart.
            const uint64_t ad = A_MN ? sdesc_sw128(sa + k * 2048, 8192, 1024) : sdesc_sw128(sa + k * 32, 16, 1024);
            const uint64_t bd = B_MN ? sdesc_sw128(sb + k * 2048, 8192, 1024) : sdesc_sw128(sb + k * 32, 16, 1024);
            if (PAIR)
              umma_bf16_pair(d_tmem, ad, bd, idesc, (kb != kb0 || k != 0) ? 1u : 0u);
            else
              umma_bf16(d_tmem, ad, bd, idesc, (kb != kb0 || k != 0) ? 1u : 0u);
          }
          if (PAIR)
            umma_commit_pair_mc(&empty[stage], 0x3);
          else
            umma_commit(&empty[stage]);
          if (++stage == (uint32_t)kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (ok) {
          if (PAIR)
            umma_commit_pair_mc(&acc_full[buf], 0x3);
          else
            umma_commit(&acc_full[buf]);
        }
      }
      // every MMA issued by this thread completes before TMEM is released
      if (PAIR)
        umma_commit_pair_mc(mma_done, 0x1);
      else
        umma_commit(mma_done);
      mbar_wait_drain(mma_done, 0, lim);
    }
  } else {
    const int q = warp & 3;
    const uint32_t t_lane = (uint32_t)(q * 32) << 16;
    uint8_t* stg = staging + q * kStagingPerWarp;
    int lt = 0;
    int nchunk = 0;
    // the MMA issuer (in the pair's leader) waits for every epilogue warp of the pair
    const uint32_t acc_empty_leader = PAIR ? mapa_shared(smem_u32(acc_empty), 0u) : smem_u32(acc_empty);
    for (uint32_t k = 0;; ++k, ++lt) {
      const int u = PAIR ? take_unit_warp<true>(k, unit_full, unit_empty, units, rank != 0, status, lim)
                         : worker + (int)k * n_workers;
      if (u < 0 || u >= sch.n_units) break;
      int mt, nt, kb0, kb1;
      sch.unit(u, mt, nt, kb0, kb1);
      const int buf = lt & 1;
      const uint32_t acc_par = (uint32_t)(lt >> 1) & 1u;
      // warp-uniform outcome: the TMEM loads below are .sync.aligned
      if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[buf], acc_par, status, lim))) break;
      tc_fence_after();
      const bool empty_k = kb1 <= kb0;
      // Full tile: this CTA's rows 32q.. over all 256 columns. Half-height tile: the CTA's
      // 64 rows sit in lanes 0-63 with columns 0-127 and in lanes 64-127 with columns
      // 128-255, all in TMEM columns 0-127.
      const bool hm = mt == sch.half_mt;
      const int m0 = mt * C::kTileRows + (hm ? (int)rank * (kRowTile / 2) + (q & 1) * 32 : (int)rank * kRowTile + q * 32);
      const int n0 = nt * kBN + (hm ? (q >> 1) * (kBN / 2) : 0);
      const int n_chunks = hm ? kBN / 64 : kBN / 32;
      // rows of the last tile past M (a pair's odd CTA can hold none) are not stored
      if (!(empty_k && p.reduce) && m0 < M) {
#pragma unroll 1
        for (int c = 0; c < n_chunks; ++c) {
          if (n0 + c * 32 >= p.N) break;
          uint32_t r[32];
          if (!empty_k) {
            tmem_ld32(tmem_base + t_lane + (uint32_t)(buf * kBN + c * 32), r);
          } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) r[j] = 0u;
          }
          uint8_t* box = stg + (nchunk & 1) * kChunkBytes;
          if (lane == 0) bulk_wait_read<1>();
          __syncwarp();
          const uint32_t bx = smem_u32(box);
#pragma unroll
          for (int j = 0; j < 8; ++j)
            st_shared_v4(bx + sw128_offset((uint32_t)lane, (uint32_t)j), r[4 * j], r[4 * j + 1], r[4 * j + 2],
                         r[4 * j + 3]);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            if (p.reduce)
              tma_reduce_add_2d(&tm_c, box, n0 + c * 32, m0);
            else
              tma_store_2d(&tm_c, box, n0 + c * 32, m0);
            bulk_commit();
          }
          ++nchunk;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (PAIR)
          mbar_arrive_cluster(acc_empty_leader + (uint32_t)buf * 8u);
        else
          mbar_arrive(&acc_empty[buf]);
      }
    }
    if (lane == 0) bulk_wait_all<0>();
  }

  tc_fence_before();
  if (PAIR)
    cluster_sync_all();  // the pair's MMAs and both epilogues are done with TMEM
  else
    __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    if (PAIR)
      tmem_dealloc_pair(tmem_base, 512);
    else
      tmem_dealloc(tmem_base, 512);
  }
}

template <bool A_MN, bool B_MN, bool PAIR>
cudaError_t launch_impl(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c, const GemmParams& p,
                        int grid, cudaStream_t s) {
  constexpr size_t smem = GemmCfg<PAIR>::kSmem;
  auto kern = k_umma_gemm<A_MN, B_MN, PAIR>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  if (!PAIR) {
    kern<<<grid, 192, smem, s>>>(a, b, c, p);
    return cudaGetLastError();
  }
  // one CTA pair per two SMs, no more pairs than can be resident at once
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(192, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3((unsigned)(grid & ~1), 1, 1);
  int max_clusters = 0;
  e = cudaOccupancyMaxActiveClusters(&max_clusters, kern, &cfg);
  if (e != cudaSuccess) return e;
  if (max_clusters < 1) return cudaErrorInvalidConfiguration;
  const int pairs = (grid / 2) < max_clusters ? (grid / 2) : max_clusters;
  cfg.gridDim = dim3((unsigned)(2 * pairs), 1, 1);
  e = cudaLaunchKernelEx(&cfg, kern, a, b, c, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

// The pair tiling stages B as 64-column MN-major boxes only: a K-major B would need
// a 128-row tensor-map box, which the maps of this library do not provide.
cudaError_t launch_gemm(bool a_mn, bool b_mn, const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c,
                        const GemmParams& p, int grid, cudaStream_t s) {
  if (p.pair) {
    if (!b_mn) return cudaErrorInvalidValue;
    return a_mn ? launch_impl<true, true, true>(a, b, c, p, grid, s) : launch_impl<false, true, true>(a, b, c, p, grid, s);
  }
  if (!a_mn && !b_mn) return launch_impl<false, false, false>(a, b, c, p, grid, s);
  if (!a_mn && b_mn) return launch_impl<false, true, false>(a, b, c, p, grid, s);
  if (a_mn && !b_mn) return launch_impl<true, false, false>(a, b, c, p, grid, s);
  return launch_impl<true, true, false>(a, b, c, p, grid, s);
}

}  // namespace opd
