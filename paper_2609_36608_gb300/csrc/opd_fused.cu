// Fused vocabulary-tiled LM-head kernel (tcgen05 + TMEM + TMA), two variants:
//
//  forward  (Section 3, Eq. reverse-kl): for a tile of supervised token rows and
//           256 vocabulary columns, the teacher logits z_t = H_t W_t^T and the
//           student logits z_s = H_s W_s^T accumulate in TMEM; the epilogue folds
//           them into per-row online statistics in base 2 (x = z log2(e) / tau):
//             m_s, S_s = sum 2^(x_s - m_s), A = sum 2^(x_s - m_s) (x_s - x_t),
//             m_t, S_t = sum 2^(x_t - m_t)
//           over the columns of one vocabulary split. Logits never reach HBM.
//  backward: recomputes the same two tiles and writes
//             dz = (g / tau) p_s (log p_s - log p_t - KL)
//           (the derivative of g KL with respect to the student logits) as bf16
//           for the two gradient GEMMs.
//
// Roles: warp 0 issues TMA loads, warp 1 allocates TMEM and issues the MMAs from
// one thread, eight epilogue warps drain TMEM (TMEM lane = tile row; the two
// warps of each lane quadrant take 128 columns each). Persistent: work units (row
// tile, vocabulary range) are taken in order from a global counter.
//
// TMEM holds one tile: teacher accumulator in columns [0,256), student in
// [256,512). Each tile computes the teacher segment first and signals it on its
// own barrier. While the student segment runs, the epilogue copies the teacher
// columns to registers and releases them, so the next tile's teacher GEMM (d_t of
// the d_s + d_t reduction) follows this tile's student GEMM without a gap and
// overlaps this tile's epilogue; the student columns are released as soon as they
// have been read, well before the next tile's student GEMM starts.
//
// PAIR = true runs each tile on a CTA pair (2-CTA cluster, tcgen05 cta_group::2):
// 256 rows per tile, 128 in each CTA's TMEM; each CTA stages its own 128 rows of
// H and 128 of the 256 rows of W, the even-ranked CTA issues the MMAs, and both
// CTAs' TMA completions are counted on the leader's barriers. Per byte staged
// from L2 this does 1.5 times the MMA work of a single-CTA 128 x 256 tile (each
// CTA stages half of W's rows).
//
// Half-height last tile: when the last row tile of a pair schedule holds at most
// 128 supervised rows, its MMAs run with M = 128 (64 rows from each CTA), half the
// tensor work. Each CTA's TMEM then holds its 64 rows twice: lanes 0-63 with
// vocabulary columns 0-127 of the tile and lanes 64-127 with columns 128-255, in
// TMEM columns 0-127. The forward stores the statistics of columns 128-255 of row r
// as a second partial at row r + 128 (a padding row), which the readers merge.
#include "opd_device.cuh"
#include "opd_internal.h"

namespace opd {

namespace {

constexpr int kBN = 256;   // vocabulary columns per tile (MMA N)
constexpr int kNEpi = 8;   // epilogue warps
constexpr int kColsPerWarp = kBN / 2;
constexpr int kThreads = 64 + 32 * kNEpi;
// Backward: 64-column bf16 dz staging boxes per epilogue warp (4 KB each). With one box
// the warp waits for each TMA store to read it before refilling it, and the 32 KB saved
// buy a sixth pipeline stage: the backward ran 2.2% faster than with two boxes and five
// stages (the single-head backward 4.9%).
constexpr int kDzBoxes = 1;

template <bool BWD, bool PAIR, int HEADS>
struct FusedCfg {
  static constexpr int kTileRows = PAIR ? 2 * kRowTile : kRowTile;  // rows per tile (whole pair)
  static constexpr int kBRows = PAIR ? kBN / 2 : kBN;              // W rows staged by one CTA
  static constexpr uint32_t kABytes = kRowTile * kKBlock * 2;
  static constexpr uint32_t kBBytes = kBRows * kKBlock * 2;
  static constexpr uint32_t kStageBytes = kABytes + kBBytes;
  static constexpr uint32_t kStagingPerWarp = BWD ? 32 * 64 * 2 * kDzBoxes : 0;  // bf16 dz boxes of one warp
  static constexpr uint32_t kMergeBytes = BWD ? 0 : 4 * 5 * 32 * 4;             // per quadrant 5 x 32
  static constexpr uint32_t kBarrierBytes = 512;
  static constexpr size_t kFixed = 1024 + (size_t)kNEpi * kStagingPerWarp + kMergeBytes + kBarrierBytes;
  static constexpr int kStagesFit = (int)((232448 - kFixed) / kStageBytes);
  static constexpr int kStages = kStagesFit > 8 ? 8 : kStagesFit;
  static constexpr size_t kSmem = kFixed + (size_t)kStages * kStageBytes;
  static constexpr int kFreeCount = PAIR ? 2 * kNEpi : kNEpi;  // epilogue warps that release TMEM
  static_assert(kStages >= 3, "pipeline depth");
  static_assert(HEADS == 1 || HEADS == 2, "one head (scoring, surrogate) or two (reverse KL)");
};

// Unit u -> (row tile, vocabulary tile range). Units are grouped by `G` row tiles
// so that CTAs (or CTA pairs) running at the same time share a few hidden-state
// tiles and a few vocabulary tiles in L2. Workers take units in increasing order
// from a global counter (not a fixed stride), so the workers that share a
// vocabulary range start it together and stay together however their speeds differ.
struct FusedSchedule {
  int n_rt, n_vt, n_vs, G, n_units;
  int half_rt;  // row tile run at half height (M = 128 on a pair), or -1

  // Both passes walk the same units; only the forward keeps per-split statistics.
  // allow_half: on a CTA pair, a last row tile with at most half of its rows
  // supervised runs as M = 128 MMAs (64 rows per CTA), half the tensor work.
  __device__ void init(int R, int V, int tile_rows, int workers, int G_, int max_split, bool allow_half,
                       int force_split) {
    n_rt = (R + tile_rows - 1) / tile_rows;
    n_vt = (V + kBN - 1) / kBN;
    half_rt = (allow_half && n_rt > 0 && R - (n_rt - 1) * tile_rows <= tile_rows / 2) ? n_rt - 1 : -1;
    // groups of at most G_ row tiles, as equal in size as possible
    G = G_ < 1 ? 1 : G_;
    if (n_rt > 0) {
      const int n_groups = (n_rt + G - 1) / G;
      G = (n_rt + n_groups - 1) / n_groups;
    }
    const int cap = max_split < 1 ? 1 : (max_split > kMaxVSplit ? kMaxVSplit : max_split);
    const int max_vs = n_vt < cap ? n_vt : cap;
    if (n_rt == 0) {
      n_vs = 1;
    } else if (force_split > 0) {
      n_vs = force_split < max_vs ? force_split : max_vs;
    } else {
      // fewest tiles on the busiest worker, then the fewest splits; at least enough
      // splits that the units running at once span one raster group of row tiles, so
      // the group's hidden-state tiles stay in L2 (with fewer splits every worker
      // streams the whole vocabulary against its own row tile and H leaves L2).
      // A half-height tile still counts as a full one here: counted as half, the search
      // at the 1.7B size picks 75 splits instead of 33, whose unequal unit lengths break
      // the lockstep of the pairs sharing a range and cost more DRAM reads than the
      // balance gains (measured).
      long best = -1;
      int min_vs = (workers + G - 1) / G;
      min_vs = min_vs < 1 ? 1 : (min_vs > max_vs ? max_vs : min_vs);
      n_vs = min_vs;
      for (int s = min_vs; s <= max_vs; ++s) {
        const long waves = ((long)n_rt * s + workers - 1) / workers;
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

// Maximum of the 32 values of one chunk (three-input max, 16 instructions).
__device__ __forceinline__ float chunk_max(const uint32_t* v) {
  float m = fmaxf(__uint_as_float(v[0]), __uint_as_float(v[1]));
#pragma unroll
  for (int j = 2; j < 32; j += 2) m = fmax3(m, __uint_as_float(v[j]), __uint_as_float(v[j + 1]));
  return m;
}

// Fold 32 columns (or the first nvalid of them) of one row into the running
// base-2 statistics: student logits in rs, teacher logits in tv[OFF..OFF+31].
// Indices stay compile-time so the values stay in registers. x = z k2 with
// k2 = log2(e) / tau; A is kept in raw logit units (times k2 at the end). A full
// chunk runs on paired fp32 instructions, two columns per instruction.
template <bool PARTIAL, int OFF>
__device__ __forceinline__ void fold_chunk(const uint32_t (&rs)[32], const uint32_t (&tv)[kColsPerWarp], int nvalid,
                                           float k2, float& ms, float& Ss, float& A, float& mt, float& St) {
  if constexpr (!PARTIAL) {
    const float nms = fmaxf(ms, chunk_max(rs) * k2);  // k2 > 0: max of scaled = scaled max
    const float nmt = fmaxf(mt, chunk_max(tv + OFF) * k2);
    const float scs = ex2_ftz(ms - nms);
    Ss *= scs;
    A *= scs;
    St *= ex2_ftz(mt - nmt);
    ms = nms;
    mt = nmt;
    const uint64_t k22 = f2_pack(k2, k2), nms2 = f2_pack(-ms, -ms), nmt2 = f2_pack(-mt, -mt);
    uint64_t S2 = f2_pack(0.f, 0.f), A2 = S2, T2 = S2;
#pragma unroll
    for (int j = 0; j < 32; j += 2) {
      const uint64_t zs = f2_pack(__uint_as_float(rs[j]), __uint_as_float(rs[j + 1]));
      const uint64_t zt = f2_pack(__uint_as_float(tv[OFF + j]), __uint_as_float(tv[OFF + j + 1]));
      float a, b;
      f2_unpack(f2_fma(zs, k22, nms2), a, b);
      const uint64_t e = f2_pack(ex2_ftz(a), ex2_ftz(b));
      S2 = f2_add(S2, e);
      A2 = f2_fma(e, f2_sub(zs, zt), A2);
      f2_unpack(f2_fma(zt, k22, nmt2), a, b);
      T2 = f2_add(T2, f2_pack(ex2_ftz(a), ex2_ftz(b)));
    }
    float lo, hi;
    f2_unpack(S2, lo, hi);
    Ss += lo + hi;
    f2_unpack(A2, lo, hi);
    A += lo + hi;
    f2_unpack(T2, lo, hi);
    St += lo + hi;
    return;
  }
  float cms = -INFINITY, cmt = -INFINITY;
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    if (!PARTIAL || j < nvalid) {
      cms = fmaxf(cms, __uint_as_float(rs[j]));
      cmt = fmaxf(cmt, __uint_as_float(tv[OFF + j]));
    }
  }
  // k2 > 0, so the scaled maximum is the maximum of the scaled values
  const float nms = fmaxf(ms, cms * k2);
  const float nmt = fmaxf(mt, cmt * k2);
  const float scs = ex2_ftz(ms - nms);
  Ss *= scs;
  A *= scs;
  St *= ex2_ftz(mt - nmt);
  ms = nms;
  mt = nmt;
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    if (!PARTIAL || j < nvalid) {
      const float zs = __uint_as_float(rs[j]);
      const float zt = __uint_as_float(tv[OFF + j]);
      const float e = ex2_ftz(fmaf(zs, k2, -ms));
      Ss += e;
      A = fmaf(e, zs - zt, A);
      St += ex2_ftz(fmaf(zt, k2, -mt));
    }
  }
}

// Forward: 32 student columns of one row folded with the matching teacher columns.
template <int C>
__device__ __forceinline__ void fwd_chunk(uint32_t ts, const uint32_t (&tv)[kColsPerWarp], int nvalid_base,
                                          float k2, float& ms, float& Ss, float& A, float& mt, float& St) {
  uint32_t rs[32];
  tmem_ld32(ts + C * 32, rs);
  const int nvalid = nvalid_base - C * 32;
  if (nvalid >= 32)
    fold_chunk<false, C * 32>(rs, tv, 32, k2, ms, Ss, A, mt, St);
  else if (nvalid > 0)
    fold_chunk<true, C * 32>(rs, tv, nvalid, k2, ms, Ss, A, mt, St);
}

// Backward: dz for 32 columns of one row, packed to bf16 into this warp's
// 128B-swizzled staging box (64 columns per box; chunk C fills half of box C/2).
template <int C>
__device__ __forceinline__ void bwd_chunk(uint32_t ts, const uint32_t (&tv)[kColsPerWarp], float k2, float b1,
                                          float kc, float cc, uint32_t stg, int lane) {
  uint32_t rs[32];
  tmem_ld32(ts + C * 32, rs);
  uint32_t w[16];
  // scalar: with the 128 teacher registers live, paired operands cost more moves and
  // spills than they save here (measured)
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    float dz2[2];
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const float zs = __uint_as_float(rs[2 * j + e]);
      const float zt = __uint_as_float(tv[C * 32 + 2 * j + e]);
      const float ps = ex2_ftz(fmaf(zs, k2, -b1));
      dz2[e] = ps * fmaf(zs - zt, kc, -cc);
    }
    w[j] = pack_bf16x2(dz2[0], dz2[1]);
  }
  const uint32_t box = stg + (uint32_t)((C >> 1) % kDzBoxes) * 4096u;
  const uint32_t jb = (uint32_t)(C & 1) * 4u;
#pragma unroll
  for (int jj = 0; jj < 4; ++jj)
    st_shared_v4(box + sw128_offset((uint32_t)lane, jb + jj), w[4 * jj], w[4 * jj + 1], w[4 * jj + 2],
                 w[4 * jj + 3]);
}

// One head: 32 columns of one row folded into the running base-2 (max, sum).
template <bool PARTIAL>
__device__ __forceinline__ void fold_chunk1(const uint32_t (&rs)[32], int nvalid, float k2, float& m, float& S) {
  if constexpr (!PARTIAL) {
    const float nm = fmaxf(m, chunk_max(rs) * k2);
    S *= ex2_ftz(m - nm);
    m = nm;
    const uint64_t k22 = f2_pack(k2, k2), nm2 = f2_pack(-m, -m);
    uint64_t S2 = f2_pack(0.f, 0.f);
#pragma unroll
    for (int j = 0; j < 32; j += 2) {
      float a, b;
      f2_unpack(f2_fma(f2_pack(__uint_as_float(rs[j]), __uint_as_float(rs[j + 1])), k22, nm2), a, b);
      S2 = f2_add(S2, f2_pack(ex2_ftz(a), ex2_ftz(b)));
    }
    float lo, hi;
    f2_unpack(S2, lo, hi);
    S += lo + hi;
    return;
  }
  float cm = -INFINITY;
#pragma unroll
  for (int j = 0; j < 32; ++j)
    if (!PARTIAL || j < nvalid) cm = fmaxf(cm, __uint_as_float(rs[j]));
  const float nm = fmaxf(m, cm * k2);
  S *= ex2_ftz(m - nm);
  m = nm;
#pragma unroll
  for (int j = 0; j < 32; ++j)
    if (!PARTIAL || j < nvalid) S += ex2_ftz(fmaf(__uint_as_float(rs[j]), k2, -m));
}

template <int C>
__device__ __forceinline__ void fwd_chunk1(uint32_t ts, int nvalid_base, float k2, float& m, float& S) {
  uint32_t rs[32];
  tmem_ld32(ts + C * 32, rs);
  const int nvalid = nvalid_base - C * 32;
  if (nvalid >= 32)
    fold_chunk1<false>(rs, 32, k2, m, S);
  else if (nvalid > 0)
    fold_chunk1<true>(rs, nvalid, k2, m, S);
}

// One head, backward of a loss on the sampled token's log-probability:
// dz = coef (1[col = x] - p), p = 2^(z k2 - b1), into the warp's staging box. This writes
// -coef p in every column; token_fixup() then puts coef (1 - p_x) in the token's column.
template <int C>
__device__ __forceinline__ void bwd_chunk1(uint32_t ts, float k2, float b1, float coef, uint32_t stg, int lane) {
  uint32_t rs[32];
  tmem_ld32(ts + C * 32, rs);
  uint32_t w[16];
  const uint64_t k22 = f2_pack(k2, k2), nb2 = f2_pack(-b1, -b1), ncoef2 = f2_pack(-coef, -coef);
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    // two columns per instruction: -coef 2^(z k2 - b1)
    float a, b;
    f2_unpack(f2_fma(f2_pack(__uint_as_float(rs[2 * j]), __uint_as_float(rs[2 * j + 1])), k22, nb2), a, b);
    f2_unpack(f2_mul(ncoef2, f2_pack(ex2_ftz(a), ex2_ftz(b))), a, b);
    w[j] = pack_bf16x2(a, b);
  }
  const uint32_t box = stg + (uint32_t)((C >> 1) % kDzBoxes) * 4096u;
  const uint32_t jb = (uint32_t)(C & 1) * 4u;
#pragma unroll
  for (int jj = 0; jj < 4; ++jj)
    st_shared_v4(box + sw128_offset((uint32_t)lane, jb + jj), w[4 * jj], w[4 * jj + 1], w[4 * jj + 2],
                 w[4 * jj + 3]);
}

// The token's column of one row in a 64-column staging box (128-byte swizzled rows,
// one row per lane): overwritten with the bf16 of `value` when the token lies in it.
__device__ __forceinline__ void token_fixup(uint32_t box, int lane, int col_in_box, float value) {
  if (col_in_box < 0 || col_in_box >= 64) return;
  const uint32_t addr = box + sw128_offset((uint32_t)lane, (uint32_t)(col_in_box >> 3)) + (uint32_t)(col_in_box & 7) * 2u;
  const __nv_bfloat16 h = __float2bfloat16_rn(value);
  asm volatile("st.shared.b16 [%0], %1;" ::"r"(addr), "h"(*reinterpret_cast<const unsigned short*>(&h)) : "memory");
}

template <bool BWD, bool PAIR, int HEADS>
__global__ void __launch_bounds__(kThreads, 1)
    k_fused_logits(const __grid_constant__ CUtensorMap tm_hs, const __grid_constant__ CUtensorMap tm_ht,
                   const __grid_constant__ CUtensorMap tm_ws, const __grid_constant__ CUtensorMap tm_wt,
                   const __grid_constant__ CUtensorMap tm_dz, const FusedParams p) {
  using C = FusedCfg<BWD, PAIR, HEADS>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* stage_base = smem;
  uint8_t* staging = smem + C::kStages * C::kStageBytes;
  float* merge = reinterpret_cast<float*>(staging + kNEpi * C::kStagingPerWarp);
  uint64_t* full = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(merge) + C::kMergeBytes);
  uint64_t* empty = full + C::kStages;
  // Two heads: acc_full[1] completes when a tile's teacher segment is computed,
  // acc_full[0] when its student segment is. One head: acc_full[slot] for TMEM slot 0 / 1
  // (columns 0-255 / 256-511, alternate tiles). Each barrier runs at most one phase ahead
  // of the epilogue that waits on it.
  uint64_t* acc_full = empty + C::kStages;
  // Two heads: teacher / student columns read by every epilogue warp. One head: slot 0 /
  // slot 1 read by every epilogue warp.
  uint64_t* t_free = acc_full + 2;
  uint64_t* s_free = t_free + 1;
  uint64_t* mma_done = s_free + 1;
  uint64_t* merge_full = mma_done + 1;      // [4]
  uint64_t* merge_empty = merge_full + 4;   // [4]
  uint64_t* unit_full = merge_empty + 4;    // [kUnitRing]
  uint64_t* unit_empty = unit_full + kUnitRing;
  int32_t* units = reinterpret_cast<int32_t*>(unit_empty + kUnitRing);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(units + kUnitRing);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  uint32_t* status = &p.ctrl->status;
  const uint64_t lim = p.wait_limit_ns;
  const uint32_t rank = PAIR ? cluster_ctarank() : 0u;  // CTA rank within the pair
  const int n_workers = PAIR ? (int)(gridDim.x >> 1) : (int)gridDim.x;
  int32_t* counter = &p.ctrl->work[BWD ? 1 : 0];

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(&acc_full[0], 1);
    mbar_init(&acc_full[1], 1);
    mbar_init(t_free, C::kFreeCount);
    mbar_init(s_free, C::kFreeCount);
    mbar_init(mma_done, 1);
    for (int qd = 0; qd < 4; ++qd) {
      mbar_init(&merge_full[qd], 1);
      mbar_init(&merge_empty[qd], 1);
    }
    // readers of each ring slot: the MMA issuer and the epilogue warps of the even
    // CTA, plus the odd CTA's producer and epilogue warps in a pair
    for (int i = 0; i < kUnitRing; ++i) {
      mbar_init(&unit_full[i], 1);
      mbar_init(&unit_empty[i], PAIR ? 2 * (1 + kNEpi) : 1 + kNEpi);
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
  const uint32_t tmem_t = tmem_base;        // teacher accumulator columns
  const uint32_t tmem_s = tmem_base + kBN;  // student accumulator columns

  const int R = p.ctrl->R;
  FusedSchedule sch;
  sch.init(R, p.V, C::kTileRows, n_workers, p.group_rows, p.max_vsplit, PAIR && p.half_tile != 0, p.vsplit);
  if (!BWD && blockIdx.x == 0 && threadIdx.x == 0) {
    p.ctrl->n_vsplit = sch.n_vs;
    p.ctrl->half_tile = sch.half_rt >= 0 ? sch.half_rt * C::kTileRows + 1 : 0;
  }
  const int nks = (p.d_s + kKBlock - 1) / kKBlock;
  const int nkt = (p.d_t + kKBlock - 1) / kKBlock;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      uint32_t stage = 0, phase = 0;
      bool ok = true, any = false;
      // a pair counts both CTAs' bytes on the leader's full barriers
      const uint32_t full_leader = PAIR ? mapa_shared(smem_u32(full), 0u) : smem_u32(full);
      int next = rank == 0 ? atomicAdd(counter, 1) : 0;
      for (uint32_t k = 0; ok; ++k) {
        int u = -1;
        if (rank == 0) {
          u = next;
          if (!publish_unit<PAIR>(k, u, unit_full, unit_empty, units, status, lim)) u = -1;
          if (u >= 0 && u < sch.n_units) next = atomicAdd(counter, 1);  // used by the next iteration
        } else {
          u = take_unit<PAIR>(k, unit_full, unit_empty, units, true, status, lim);
        }
        if (u < 0) {
          ok = false;
          break;
        }
        if (u >= sch.n_units) break;
        int rt, split, vb, ve;
        sch.unit(u, rt, split, vb, ve);
        // a half-height tile takes 64 rows from each CTA (the MMA reads the first 64 staged)
        const int row0 = rt * C::kTileRows + (int)rank * (rt == sch.half_rt ? kRowTile / 2 : kRowTile);
        for (int vt = vb; ok && vt < ve; ++vt) {
          const int wrow0 = vt * kBN + (int)rank * C::kBRows;
          for (int seg = 2 - HEADS; ok && seg < 2; ++seg) {  // teacher (two heads), then student
            const CUtensorMap* ta = seg ? &tm_hs : &tm_ht;
            const CUtensorMap* tb = seg ? &tm_ws : &tm_wt;
            const int nk = seg ? nks : nkt;
            for (int kb = 0; kb < nk; ++kb) {
              if (!mbar_wait(&empty[stage], phase ^ 1u, status, lim)) {
                ok = false;
                break;
              }
              uint8_t* sa = stage_base + stage * C::kStageBytes;
              if (PAIR) {
                if (rank == 0) mbar_arrive_expect_tx(&full[stage], 2 * C::kStageBytes);
                const uint32_t fb = full_leader + stage * 8u;
                tma_load_2d_pair(sa, ta, fb, kb * kKBlock, row0);
                tma_load_2d_pair(sa + C::kABytes, tb, fb, kb * kKBlock, wrow0);
              } else {
                mbar_arrive_expect_tx(&full[stage], C::kStageBytes);
                tma_load_2d(sa, ta, &full[stage], kb * kKBlock, row0);
                tma_load_2d(sa + C::kABytes, tb, &full[stage], kb * kKBlock, wrow0);
              }
              any = true;
              if (++stage == (uint32_t)C::kStages) {
                stage = 0;
                phase ^= 1u;
              }
            }
          }
        }
      }
      if (!ok && any && rank == 0) {
        // Let every copy already issued land before the CTA can exit (in a pair,
        // the leader's barriers also count the peer's copies).
        for (int s = 0; s < C::kStages; ++s) {
          const uint32_t par = ((uint32_t)s < stage) ? phase : (phase ^ 1u);
          mbar_wait_drain(&full[s], par, lim);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc_full = idesc_bf16_f32(C::kTileRows, kBN, false, false);
      constexpr uint32_t idesc_half = idesc_bf16_f32(C::kTileRows / 2, kBN, false, false);
      uint32_t stage = 0, phase = 0;
      int lt = 0;
      bool ok = true;
      for (uint32_t k = 0; ok; ++k) {
        const int u = take_unit<PAIR>(k, unit_full, unit_empty, units, false, status, lim);
        if (u < 0) {
          ok = false;
          break;
        }
        if (u >= sch.n_units) break;
        int rt, split, vb, ve;
        sch.unit(u, rt, split, vb, ve);
        const uint32_t idesc = rt == sch.half_rt ? idesc_half : idesc_full;
        for (int vt = vb; ok && vt < ve; ++vt, ++lt) {
          for (int seg = 2 - HEADS; ok && seg < 2; ++seg) {
            // two heads: each segment reuses its columns every tile; one head: the
            // tile alternates between two column slots
            const int slot = HEADS == 2 ? seg : (lt & 1);
            const uint32_t free_par = HEADS == 2 ? (((uint32_t)lt & 1u) ^ 1u) : ((((uint32_t)lt >> 1) & 1u) ^ 1u);
            if (!mbar_wait(slot ? s_free : t_free, free_par, status, lim)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t d_tmem = slot ? tmem_s : tmem_t;
            const int nk = seg ? nks : nkt;
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
                const uint64_t ad = sdesc_sw128(sa + k * 32, 16, 1024);
                const uint64_t bd = sdesc_sw128(sb + k * 32, 16, 1024);
                if (PAIR)
                  umma_bf16_pair(d_tmem, ad, bd, idesc, (kb | k) != 0);
                else
                  umma_bf16(d_tmem, ad, bd, idesc, (kb | k) != 0);
              }
              if (PAIR)
                umma_commit_pair_mc(&empty[stage], 0x3);
              else
                umma_commit(&empty[stage]);
              if (++stage == (uint32_t)C::kStages) {
                stage = 0;
                phase ^= 1u;
              }
            }
            // two heads: the teacher segment is signalled on its own, so the epilogue
            // can drain and release its columns while the student segment runs
            if (HEADS == 2 && seg == 0 && ok) {
              if (PAIR)
                umma_commit_pair_mc(&acc_full[1], 0x3);
              else
                umma_commit(&acc_full[1]);
            }
          }
          if (ok) {
            uint64_t* af = HEADS == 2 ? &acc_full[0] : &acc_full[lt & 1];
            if (PAIR)
              umma_commit_pair_mc(af, 0x3);
            else
              umma_commit(af);
          }
        }
      }
      // Every MMA issued by this thread completes before TMEM is released.
      if (PAIR)
        umma_commit_pair_mc(mma_done, 0x1);
      else
        umma_commit(mma_done);
      mbar_wait_drain(mma_done, 0, lim);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int ew = warp - 2;                 // epilogue warp index
    const int q = warp & 3;                  // TMEM lane quadrant this warp may access
    const int half = ew / 4;                 // which half of the accumulator's TMEM columns
    const uint32_t t_lane = (uint32_t)(q * 32) << 16;
    // the MMA issuer (in the pair's leader) waits for every epilogue warp of the pair
    const uint32_t t_free_addr = PAIR ? mapa_shared(smem_u32(t_free), 0u) : smem_u32(t_free);
    const uint32_t s_free_addr = PAIR ? mapa_shared(smem_u32(s_free), 0u) : smem_u32(s_free);
    int lt = 0, nu = 0;
    bool ok = true;
    bool one_box = false;  // backward: the last tile stored only staging box 0
    const uint32_t stg = smem_u32(staging + ew * C::kStagingPerWarp);
    for (uint32_t k = 0; ok; ++k, ++nu) {
      const int u = take_unit_warp<PAIR>(k, unit_full, unit_empty, units, PAIR && rank != 0, status, lim);
      if (u < 0) {
        ok = false;
        break;
      }
      if (u >= sch.n_units) break;
      int rt, split, vb, ve;
      sch.unit(u, rt, split, vb, ve);
      // Full tile: this CTA's 128 rows, lane quadrant q = rows 32q.., and this warp's
      // 128 of the 256 columns. Half-height tile (M = 128 on the pair): this CTA's 64
      // rows sit in lanes 0-63 with columns 0-127 and again in lanes 64-127 with columns
      // 128-255, all in TMEM columns 0-127; this warp takes 64 of those columns.
      const bool hm = rt == sch.half_rt;
      const int drow0 = rt * C::kTileRows + (hm ? (int)rank * (kRowTile / 2) + (q & 1) * 32
                                                : (int)rank * kRowTile + q * 32);
      const int row = drow0 + lane;  // token row of this lane (rowc, dz)
      float ms = -INFINITY, Ss = 0.f, A = 0.f, mt = -INFINITY, St = 0.f;
      // backward row constants. Two heads: p_s = 2^(z_s k2 - b1), dz = p_s ((z_s - z_t) kc - cc).
      // One head: dz = coef (1[col = x] - p_s) with coef = rowc.y, token x = rowc.z (bits) and
      // the token column's value coef (1 - p_x) = rowc.w.
      float b1 = 0.f, kc = 0.f, cc = 0.f, at_token = 0.f;
      int x_tok = -1;
      if (BWD) {
        const float4 rc = p.rowc[row];
        b1 = rc.x;
        if (HEADS == 2) {
          kc = rc.z * p.inv_tau;
          cc = rc.z * rc.y;
        } else {
          kc = rc.y;
          x_tok = __float_as_int(rc.z);
          at_token = rc.w;
        }
      }
      for (int vt = vb; vt < ve; ++vt, ++lt) {
        // warp-uniform outcome: the TMEM loads below are .sync.aligned. Two heads wait
        // first for the teacher segment (acc_full[1]), one head for its slot's tile.
        uint64_t* af = HEADS == 2 ? &acc_full[1] : &acc_full[lt & 1];
        const uint32_t af_par = HEADS == 2 ? ((uint32_t)lt & 1u) : (((uint32_t)lt >> 1) & 1u);
        if (!__all_sync(0xffffffffu, mbar_wait(af, af_par, status, lim))) {
          ok = false;
          break;
        }
        tc_fence_after();
        // TMEM column offset and tile column offset of this warp's columns
        const int tcol = hm ? half * (kColsPerWarp / 2) : half * kColsPerWarp;
        const int dcol = hm ? (q >> 1) * (kBN / 2) + tcol : tcol;
        if (HEADS == 1) {
          const int slot = lt & 1;
          const int col0 = vt * kBN + dcol;
          const uint32_t ts = (slot ? tmem_s : tmem_t) + t_lane + (uint32_t)tcol;
          if (!BWD) {
            const int nv = p.V - col0;
            fwd_chunk1<0>(ts, nv, p.k2, ms, Ss);
            fwd_chunk1<1>(ts, nv, p.k2, ms, Ss);
            if (!hm) {
              fwd_chunk1<2>(ts, nv, p.k2, ms, Ss);
              fwd_chunk1<3>(ts, nv, p.k2, ms, Ss);
            }
          } else {
            const int x_rel = x_tok - col0;  // the token's column within this warp's columns
            // staging box 0 is rewritten once its previous store has been read
            if (lane == 0) {
              if (one_box || kDzBoxes == 1)
                bulk_wait_read<0>();
              else
                bulk_wait_read<1>();
            }
            __syncwarp();
            bwd_chunk1<0>(ts, p.k2, b1, kc, stg, lane);
            bwd_chunk1<1>(ts, p.k2, b1, kc, stg, lane);
            token_fixup(stg, lane, x_rel, at_token);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              tma_store_2d(&tm_dz, staging + ew * C::kStagingPerWarp, col0, drow0);
              bulk_commit();
              if (!hm) bulk_wait_read<kDzBoxes - 1>();
            }
            __syncwarp();
            if (!hm) {
              constexpr uint32_t box1 = kDzBoxes > 1 ? 4096u : 0u;
              bwd_chunk1<2>(ts, p.k2, b1, kc, stg, lane);
              bwd_chunk1<3>(ts, p.k2, b1, kc, stg, lane);
              token_fixup(stg + box1, lane, x_rel - 64, at_token);
              fence_proxy_async_smem();
              __syncwarp();
              if (lane == 0) {
                tma_store_2d(&tm_dz, staging + ew * C::kStagingPerWarp + box1, col0 + 64, drow0);
                bulk_commit();
              }
            }
            one_box = hm;
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            uint64_t* fb = slot ? s_free : t_free;
            if (PAIR)
              mbar_arrive_cluster(slot ? s_free_addr : t_free_addr);
            else
              mbar_arrive(fb);
          }
          continue;
        }
        // teacher columns to registers, then release them to the next tile's MMAs
        uint32_t tv[kColsPerWarp];  // a half-height tile uses the first 64
        tmem_ld128(tmem_t + t_lane + (uint32_t)tcol, tv);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (PAIR)
            mbar_arrive_cluster(t_free_addr);
          else
            mbar_arrive(t_free);
        }
        // then the student segment (committed after the teacher's, same tile parity)
        if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[0], (uint32_t)lt & 1u, status, lim))) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int col0 = vt * kBN + dcol;
        const uint32_t ts = tmem_s + t_lane + (uint32_t)tcol;
        if (!BWD) {
          const int nv = p.V - col0;
          fwd_chunk<0>(ts, tv, nv, p.k2, ms, Ss, A, mt, St);
          fwd_chunk<1>(ts, tv, nv, p.k2, ms, Ss, A, mt, St);
          if (!hm) {
            fwd_chunk<2>(ts, tv, nv, p.k2, ms, Ss, A, mt, St);
            fwd_chunk<3>(ts, tv, nv, p.k2, ms, Ss, A, mt, St);
          }
        } else {
          // staging box h of this warp is rewritten only after its previous TMA
          // store has finished reading it (box 0 was the last store after a
          // half-height tile, the second-to-last otherwise)
          if (lane == 0) {
            if (one_box || kDzBoxes == 1)
              bulk_wait_read<0>();
            else
              bulk_wait_read<1>();
          }
          __syncwarp();
          bwd_chunk<0>(ts, tv, p.k2, b1, kc, cc, stg, lane);
          bwd_chunk<1>(ts, tv, p.k2, b1, kc, cc, stg, lane);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_store_2d(&tm_dz, staging + ew * C::kStagingPerWarp, col0, drow0);
            bulk_commit();
            if (!hm) bulk_wait_read<kDzBoxes - 1>();
          }
          __syncwarp();
          if (!hm) {
            constexpr uint32_t box1 = kDzBoxes > 1 ? 4096u : 0u;
            bwd_chunk<2>(ts, tv, p.k2, b1, kc, cc, stg, lane);
            bwd_chunk<3>(ts, tv, p.k2, b1, kc, cc, stg, lane);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              tma_store_2d(&tm_dz, staging + ew * C::kStagingPerWarp + box1, col0 + 64, drow0);
              bulk_commit();
            }
          }
          one_box = hm;
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (PAIR)
            mbar_arrive_cluster(s_free_addr);
          else
            mbar_arrive(s_free);
        }
      }
      if (!BWD && ok) {
        A *= p.k2;  // A was accumulated in raw logit units
        // the two warps of a quadrant fold their column shares: half 1 hands its
        // statistics to half 0 through shared memory
        float* mb = merge + q * 5 * 32;
        if (half == 1) {
          if (nu > 0 &&
              !__all_sync(0xffffffffu, mbar_wait(&merge_empty[q], (uint32_t)(nu - 1) & 1u, status, lim))) {
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
        // In a half-height tile both warps of a quadrant may own no column of the unit's
        // vocabulary range (its last tile, past V): the statistics then stay empty.
        const float Ms = fmaxf(ms, ms1);
        const bool any = Ms != -INFINITY;
        const float f0 = any ? ex2_ftz(ms - Ms) : 0.f, f1 = any ? ex2_ftz(ms1 - Ms) : 0.f;
        Ss = Ss * f0 + Ss1 * f1;
        ms = Ms;
        const size_t plane = (size_t)p.T_pad;
        // a half-height tile keeps the statistics of columns 128-255 at row + 128
        const int srow = hm ? row + (q >> 1) * 128 : row;
        float* base = p.partials + (size_t)split * 5 * plane + srow;
        base[0 * plane] = ms;
        base[1 * plane] = Ss;
        if (HEADS == 2) {
          const float Mt = fmaxf(mt, mt1);
          A = A * f0 + A1 * f1;
          St = any ? St * ex2_ftz(mt - Mt) + St1 * ex2_ftz(mt1 - Mt) : 0.f;
          mt = Mt;
          base[2 * plane] = A;
          base[3 * plane] = mt;
          base[4 * plane] = St;
        }
      }
    }
    if (BWD && lane == 0) bulk_wait_all<0>();
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

template <bool BWD, bool PAIR, int HEADS>
cudaError_t launch_fused_impl(const CUtensorMap& hs, const CUtensorMap& ht, const CUtensorMap& ws,
                              const CUtensorMap& wt, const CUtensorMap& dz, const FusedParams& p, int grid,
                              cudaStream_t s) {
  using C = FusedCfg<BWD, PAIR, HEADS>;
  static_assert(C::kSmem <= 232448, "shared memory budget");
  auto kern = k_fused_logits<BWD, PAIR, HEADS>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::kSmem);
  if (e != cudaSuccess) return e;
  if (!PAIR) {
    kern<<<grid, kThreads, C::kSmem, s>>>(hs, ht, ws, wt, dz, p);
    return cudaGetLastError();
  }
  // One CTA pair per two SMs, no more pairs than can be resident at once.
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = C::kSmem;
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
  e = cudaLaunchKernelEx(&cfg, kern, hs, ht, ws, wt, dz, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <bool BWD, int HEADS>
cudaError_t launch_fused_mode(const CUtensorMap& hs, const CUtensorMap& ht, const CUtensorMap& ws,
                              const CUtensorMap& wt, const CUtensorMap& dz, const FusedParams& p, int grid,
                              cudaStream_t s) {
  switch (fused_mode(p)) {
    case kFusedBN256: return launch_fused_impl<BWD, false, HEADS>(hs, ht, ws, wt, dz, p, grid, s);
    case kFusedPair256: return launch_fused_impl<BWD, true, HEADS>(hs, ht, ws, wt, dz, p, grid, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_fused_forward(const CUtensorMap& hs, const CUtensorMap& ht, const CUtensorMap& ws,
                                 const CUtensorMap& wt, const FusedParams& p, int grid, cudaStream_t s) {
  return launch_fused_mode<false, 2>(hs, ht, ws, wt, hs, p, grid, s);
}

cudaError_t launch_fused_backward(const CUtensorMap& hs, const CUtensorMap& ht, const CUtensorMap& ws,
                                  const CUtensorMap& wt, const CUtensorMap& dz_store, const FusedParams& p,
                                  int grid, cudaStream_t s) {
  return launch_fused_mode<true, 2>(hs, ht, ws, wt, dz_store, p, grid, s);
}

cudaError_t launch_head_forward(const CUtensorMap& h, const CUtensorMap& w, const FusedParams& p, int grid,
                                cudaStream_t s) {
  return launch_fused_mode<false, 1>(h, h, w, w, h, p, grid, s);
}

cudaError_t launch_head_backward(const CUtensorMap& h, const CUtensorMap& w, const CUtensorMap& dz_store,
                                 const FusedParams& p, int grid, cudaStream_t s) {
  return launch_fused_mode<true, 1>(h, h, w, w, dz_store, p, grid, s);
}

}  // namespace opd
