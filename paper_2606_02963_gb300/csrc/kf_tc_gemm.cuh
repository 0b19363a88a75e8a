// kf_tc_gemm.cuh -- persistent, warp-specialised tcgen05 GEMM with the tail-op
// chain fused into its epilogue (sm_103a).
//
// One CTA per SM, 6 warps:
//   warp 0      TMA producer: streams 128x64 A tiles and BNx64 B tiles (bf16,
//               128-byte swizzle) into a STAGES-deep shared-memory ring.
//   warp 1      owns the tensor memory (alloc/dealloc) and, from one thread,
//               issues tcgen05.mma (M=128, N=BN, K=16) into one of two TMEM
//               accumulators; tcgen05.commit frees ring slots / publishes tiles.
//   warps 2..5  epilogue: warp w reads TMEM lanes 32*(w%4).. (one output row per
//               thread), applies the op chain in fp32 registers and writes the
//               result once (Sec. IV-B: layer-wise fusion -- the matmul result is
//               read once and the output written once; mixed precision -- bf16
//               operands, fp32 accumulation and post-processing).
// Row reductions run per thread over its row: the row log-sum-exp keeps an
// online (max, sum exp) pair per tile and a second tiny kernel combines tiles
// (Sec. IV-B: streaming online reduction); GroupNorm computes each group's
// mean and variance from the accumulator in TMEM (exact two-pass per tile,
// Chan's pairwise merge across the two 256-column halves of a 512-wide group).
//
// Every mbarrier wait is bounded (wall-time limit); a wait that runs out raises
// a CTA-wide abort flag and an error bit, the producer waits (bounded) for its
// in-flight TMA copies, the MMA thread for its in-flight MMAs, TMEM is freed and
// the CTA returns.
#pragma once
#include "kf_common.cuh"
#include "kf_ptx.cuh"

namespace kf {

template <class P>
struct IsBiasProg {
  static constexpr bool value = false;
};
template <>
struct IsBiasProg<Prog<KF_OP_BIAS>> {
  static constexpr bool value = true;
};

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kEpiWarps = 8;  // epilogue warps of the variants without a residual tile
constexpr int kThreads = 64 + 32 * kEpiWarps;  // TMA warp, MMA warp, epilogue warps
constexpr int kABytes = kBM * kBK * 2;

__host__ __device__ constexpr int pow2_at_least(int x) {
  return x <= 32 ? 32 : x <= 64 ? 64 : x <= 128 ? 128 : x <= 256 ? 256 : 512;
}

// Cluster layouts (CL): kClOne = single CTA, 128-row tiles; kClPair = a CTA
// pair (cluster of 2) computing 256-row tiles with tcgen05.mma.cta_group::2;
// kClQuad = a cluster of two such pairs whose tiles are the two 256-column
// halves of one 512-column unit (GroupNorm: one group per unit).
constexpr int kClOne = 0;
constexpr int kClPair = 1;
constexpr int kClQuad = 2;
// kClCouple = CTA pairs (clusters of 2) of one cooperative grid taken two at a
// time: the pairs of a couple hold the two 256-column halves of one 512-column
// unit and swap per-row statistics through global memory (GroupNorm).
constexpr int kClCouple = 3;

// Residual tile: dense CTA-pair store kernels whose compiled chain adds a bf16
// residual stage the unit's residual tile in shared memory by TMA, in the two
// ring slots that follow the unit's last k-block (the producer loads them, the
// MMA skips them), add it from there, write the bf16 result in place and send
// each 32 x 32 block out with one TMA store; the last epilogue warp to finish
// frees the two slots.
template <int MODE, bool GROUPED, int CL, class PRE>
constexpr bool kResTileFor = MODE == kModeStore && !GROUPED && CL == kClPair && PRE::kHasRes;
// The residual-tile variants need few registers per thread (no operands staged
// in registers), so they run 12 epilogue warps (3 per TMEM lane quadrant) in
// 448 threads; the others 8 (2 per quadrant) in 320.
template <int MODE, bool GROUPED, int CL, class PRE>
constexpr int kThreadsFor = 64 + 32 * (kResTileFor<MODE, GROUPED, CL, PRE> ? 12 : kEpiWarps);

// AR: rows of an A ring slot.  128 (the MMA's M) except for grouped GEMMs whose
// groups are known to hold at most AR rows (the MoE at decode): the TMA box
// then brings AR rows, and the MMA's 128-row read of a slot runs on into the
// next slot (or, from the last one, into the epilogue buffers that follow the
// ring) -- those rows feed accumulator rows that are never stored.
template <int BN, int STAGES, int MODE, bool GROUPED, int CL, bool RT = false, int AR = kBM>
struct TcCfg {
  static constexpr bool CTA2 = CL != kClOne;  // tcgen05 CTA-pair MMAs
  static constexpr int kEpiW = RT ? 12 : kEpiWarps;  // epilogue warps
  static constexpr int kH = kEpiW / 4;               // epilogue warps per TMEM lane quadrant
  static constexpr int kThr = 64 + 32 * kEpiW;
  static constexpr bool kQuad = CL == kClQuad;
  static_assert(BN % 32 == 0 && BN >= 64 && BN <= 256, "BN");
  static_assert(!(GROUPED && CTA2), "grouped GEMMs use single-CTA tiles");
  static_assert(!kQuad || (MODE == kModeGroupNorm && BN == 256), "quad clusters split 512-column groups");
  static_assert(CL != kClCouple || (MODE == kModeGroupNorm && BN == 256), "couples split 512-column groups");
  static_assert(!RT || (MODE == kModeStore && !GROUPED && CL == kClPair), "residual tile: dense CTA-pair store");
  static_assert(MODE != kModeRope || (kEpiW == 8 && !GROUPED), "QKV tail: two warps per lane quadrant, dense");
  static constexpr int kOutN = (MODE == kModeSwiglu) ? BN / 2 : BN;  // output columns of a (sub)tile
  // With CTA pairs each CTA stages its own 128 rows of A and half of the BN rows of B.
  static constexpr int kBRows = CTA2 ? BN / 2 : BN;
  static constexpr int kBBytes = kBRows * kBK * 2;
  static constexpr int kASlot = AR * kBK * 2;
  static_assert(AR == kBM || (GROUPED && !CTA2 && AR % 8 == 0 && AR < kBM), "short A slots: grouped, single CTA");
  static constexpr int kStageBytes = kASlot + kBBytes;
  static constexpr uint32_t kTxBytes = (CTA2 ? 2 : 1) * kStageBytes;  // bytes landing per stage on the leader's barrier
  static constexpr int kRowsPerUnit = CTA2 ? 2 * kBM : kBM;
  // accumulator buffer b starts at TMEM column b * kAccStride
  static constexpr int kAccStride = pow2_at_least(BN);
  static constexpr int kTmemCols = 2 * kAccStride;
  static constexpr int kBarBytes = (8 * (2 * STAGES + 7 + kEpiW) + 63) / 64 * 64;  // keeps what follows 64-B aligned
  // per-warp 1 KB tile buffers (1 KB aligned, right after the stages): two for
  // the asynchronous TMA stores, plus (store mode) one for the residual
  // transposition, which must not reuse a buffer a TMA store may still read
  // (residual tile: 256 B per warp, the bias of its chunks; scatter-add: 64 B
  // per lane, the row segment a bulk reduction adds to the destination row)
  static constexpr int kWarpStaging = RT ? 256 : (MODE == kModeStore) ? 3072 : (MODE == kModeRope) ? 0 : 2048;
  // residual tile: BN / 32 chunks x 4 row blocks of 32 x 32 bf16 (2 KB, 64-byte
  // swizzle), placed in the A then B regions of two ring slots
  static constexpr int kResTileBytes = 0;
  static constexpr int kResBlocksA = kASlot / 2048;
  static constexpr int kResBlocksPerSlot = kASlot / 2048 + kBBytes / 2048;
  static_assert(!RT || 2 * kResBlocksPerSlot >= (BN / 32) * 4, "residual tile fits two ring slots");
  static_assert(!RT || STAGES >= 3, "residual tile needs two slots beside an operand slot");
  static constexpr int kStagingBytes = kEpiW * kWarpStaging;
  static_assert(kStagingBytes >= kABytes - kASlot, "the MMA's read past the last short A slot stays in the CTA");
  // GroupNorm: per-warp cache of bias / gamma / beta for 4 chunks of 32 columns
  static constexpr int kGnCacheBytes = (MODE == kModeGroupNorm) ? kEpiW * 3 * 4 * 32 * 4 : 0;
  // flags + row-statistics exchange between the two warps of a quadrant (2 KB)
  // + (quad) the other pair's per-row statistics, two slots (2 KB)
  static constexpr int kMiscBytes = 64 + 2 * kBM * 8 + (kQuad ? 2 * kBM * 8 : 0);
  static constexpr int kTableBytes = GROUPED ? 8 * (kMaxGroups + 1) : 0;
  static constexpr int kSmemUse =
      STAGES * kStageBytes + kResTileBytes + kStagingBytes + kGnCacheBytes + kBarBytes + kMiscBytes + kTableBytes;
  // pad to > half of the SM's shared memory so that at most one such CTA is
  // resident per SM (tensor-memory allocation then never has to wait)
  static constexpr int kSmemBytes = 1024 + (kSmemUse > 120 * 1024 ? kSmemUse : 120 * 1024);
  static constexpr uint32_t kIdesc = idesc_bf16_f32(CTA2 ? 2 * kBM : kBM, BN);
  static_assert(kSmemBytes <= 232448, "shared memory");
  static_assert(kBBytes % 1024 == 0 && (BN / 2) % 8 == 0, "B stage alignment");
};

struct UnitInfo {
  int32_t m0, m_end, n0, g, n_blk;
};

// PRE / POST: compiled op programs (Prog<...>) for the chain before / after the
// reduction, or Interp for arbitrary chains.
template <int BN, int STAGES, int MODE, bool GROUPED, int CL, class PRE = Interp, class POST = Interp, int AR = kBM>
__global__ void __launch_bounds__(kThreadsFor<MODE, GROUPED, CL, PRE>, 1)
    kf_tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                      const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmR,
                      const __grid_constant__ TcParams p, const int32_t sub_tiles) {
  constexpr bool RT = kResTileFor<MODE, GROUPED, CL, PRE>;
  using Cfg = TcCfg<BN, STAGES, MODE, GROUPED, CL, RT, AR>;
  constexpr bool CTA2 = Cfg::CTA2;
  constexpr bool QUAD = Cfg::kQuad;
  constexpr bool COUPLE = CL == kClCouple;
  constexpr bool PRE_IS_BIAS = IsBiasProg<PRE>::value;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* smB = sm;                                // B stages first: any over-read stays inside the CTA
  uint8_t* smA = sm + STAGES * Cfg::kBBytes;
  uint8_t* staging = sm + STAGES * Cfg::kStageBytes;           // epilogue tile buffers
  float* gn_cache = reinterpret_cast<float*>(staging + Cfg::kStagingBytes);
  uint64_t* bars = reinterpret_cast<uint64_t*>(staging + Cfg::kStagingBytes + Cfg::kGnCacheBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* accf = bars + 2 * STAGES;
  uint64_t* acce = bars + 2 * STAGES + 2;
  uint64_t* drain = bars + 2 * STAGES + 4;
  uint64_t* xbar = bars + 2 * STAGES + 5;  // quad: the other pair's statistics have landed (2 slots)
  uint64_t* rbar = bars + 2 * STAGES + 7;  // residual tile: warp ew's rows have landed (one per epilogue warp)
  uint32_t* misc = reinterpret_cast<uint32_t*>(reinterpret_cast<uint8_t*>(bars) + Cfg::kBarBytes);
  uint32_t* tmem_slot = misc;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 1);
  int32_t* total_s = reinterpret_cast<int32_t*>(misc + 2);
  volatile int* zero_flag = reinterpret_cast<volatile int*>(misc + 3);
  // residual tile: epilogue warps done with the unit's slots, one counter per
  // accumulator parity (a warp runs at most one unit ahead of the slowest: the
  // unit after next reuses this unit's accumulator, freed only after this count)
  int* rdone = reinterpret_cast<int*>(misc + 4);
  int32_t* off_s = reinterpret_cast<int32_t*>(reinterpret_cast<uint8_t*>(misc) + Cfg::kMiscBytes);
  int32_t* ustart_s = off_s + (kMaxGroups + 1);

  // The CTA-pair instructions address the peer CTA of the cluster, and the
  // unit / couple arithmetic assumes the grid the host sized: refuse any other
  // launch shape (all threads alike, before any barrier, TMEM or copy).
  {
    constexpr uint32_t kCluster = QUAD ? 4u : (CTA2 ? 2u : 1u);
    constexpr uint32_t kGridMult = COUPLE ? 4u : kCluster;
    const uint32_t ncl = CTA2 ? cluster_nctarank() : 1u;
    if (ncl != kCluster || blockDim.x != static_cast<uint32_t>(Cfg::kThr) || gridDim.x % kGridMult != 0 ||
        gridDim.y != 1 || gridDim.z != 1) {
      if (threadIdx.x == 0) raise_err(p.err, p.err_dev, kErrLaunchShape);
      return;
    }
  }
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // CTA pairs are the cluster ranks that differ in bit 0; the even rank leads
  // (issues the MMAs, owns the barriers both CTAs' copies complete on)
  const uint32_t rank = CTA2 ? cluster_ctarank() : 0u;
  const uint32_t prank = rank & 1u;       // position in the pair: 128-row half
  const uint32_t lead_rank = rank & ~1u;  // cluster rank of the pair's leader
  const uint16_t pair_mask = static_cast<uint16_t>(0x3u << (rank & 2u));
  const bool leader = prank == 0;
  constexpr int kUnitShift = QUAD ? 2 : (CTA2 ? 1 : 0);
  int32_t unit0 = static_cast<int32_t>(blockIdx.x >> kUnitShift);
  int32_t unit_step = static_cast<int32_t>(gridDim.x >> kUnitShift);
  uint32_t chalf = 0;  // couples: which 256-column half of the unit this pair holds
  if constexpr (COUPLE) {
    // pair i and pair i + couples form couple i (grid = 4 x couples CTAs)
    const int32_t pi = static_cast<int32_t>(blockIdx.x >> 1), ncpl = static_cast<int32_t>(gridDim.x >> 2);
    unit0 = pi % ncpl;
    unit_step = ncpl;
    chalf = static_cast<uint32_t>(pi / ncpl);
  }

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&accf[a], 1);
      mbar_init(&acce[a], Cfg::kEpiW * (CTA2 ? 2 : 1));
    }
    mbar_init(drain, 1);
    if constexpr (QUAD) {
      mbar_init(&xbar[0], kBM);  // one arrival per row of the other pair's CTA
      mbar_init(&xbar[1], kBM);
    }
    if constexpr (RT)
      for (int w = 0; w < Cfg::kEpiW; ++w) mbar_init(&rbar[w], 1);
    *abort_flag = 0;
    *zero_flag = 0;
    rdone[0] = 0;
    rdone[1] = 0;
    *total_s = GROUPED ? 0 : p.total_units;
    fence_mbarrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    if constexpr (RT) tma_prefetch_desc(&tmR);
    if constexpr (MODE == kModeRope) {
      // the QKV projection at decode sizes streams its weights: this CTA's first
      // weight tile goes to L2 while a preceding kernel may still run (a
      // prefetch reads memory without changing it, and L2 is where that
      // kernel's writes land, so the loads after the dependency wait below see
      // current values either way)
      if (p.M <= kBM && unit0 < p.total_units) {
        const int32_t nb0 = (unit0 / p.tiles_m) * Cfg::kOutN + static_cast<int32_t>(prank) * Cfg::kBRows;
        for (int32_t kb = 0; kb < p.num_kb; ++kb) tma_prefetch_3d(&tmB, kb * kBK, nb0, 0);
      }
    }
  }
  if (warp == 1) {
    __syncwarp();
    if constexpr (CTA2) {
      tmem_alloc_pair(tmem_slot, Cfg::kTmemCols);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(tmem_slot, Cfg::kTmemCols);
      tmem_relinquish();
    }
  }
  // Everything above is independent of other kernels' results; when this grid
  // follows another of this library's kernels as a programmatic dependent (the
  // MoE chain), wait for it here, before the group table, operands or epilogue
  // inputs are read.  Without such a dependency the wait returns at once.
  griddep_wait();
  griddep_launch_dependents();
  if constexpr (GROUPED) {
    if (threadIdx.x == 64) {
      // Group table: validate the device-resident offsets and count work units
      // (ceil(rows/128) row tiles x tiles_n column tiles per group).
      bool ok = p.G >= 1 && p.G <= kMaxGroups;
      int32_t units = 0;
      int32_t prev = 0;
      for (int g = 0; ok && g <= p.G; ++g) {
        int32_t o = p.group_offsets[g];
        if (o < prev || o > p.M) ok = false;
        off_s[g] = o;
        if (g > 0) {
          ustart_s[g - 1] = units;
          units += ((o - prev + kBM - 1) / kBM) * p.tiles_n;
        }
        prev = o;
      }
      if (!ok) {
        raise_err(p.err, p.err_dev, kErrBounds);
        units = 0;
      }
      if (ok) ustart_s[p.G] = units;
      *total_s = units;
    }
  }
  tc_fence_before();
  // __syncthreads is an aligned barrier: every warp must reach it converged,
  // or a warp whose lanes arrive at different times is counted too early
  __syncwarp();
  __syncthreads();
  if constexpr (CTA2) cluster_sync();  // peer barriers initialised, TMEM allocated in both CTAs
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int32_t total = *total_s;

  // residual block (chunk c, row block q) of a unit whose residual sits in ring
  // slots s0, s1
  auto res_block = [&](int s0, int s1, int c, int qq) -> uint8_t* {
    const int bi = c * 4 + qq;
    const int sl = bi < Cfg::kResBlocksPerSlot ? s0 : s1;
    const int j = bi % Cfg::kResBlocksPerSlot;
    return j < Cfg::kResBlocksA ? smA + sl * Cfg::kASlot + j * 2048 : smB + sl * Cfg::kBBytes + (j - Cfg::kResBlocksA) * 2048;
  };

  auto decode = [&](int32_t u) -> UnitInfo {
    UnitInfo r;
    if constexpr (GROUPED) {
      int lo = 0, hi = p.G - 1;  // last g with ustart_s[g] <= u
      while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (ustart_s[mid] <= u) lo = mid; else hi = mid - 1;
      }
      // skip empty groups that share the same start
      int g = lo;
      while (g + 1 < p.G && ustart_s[g + 1] <= u) ++g;
      const int32_t rows = off_s[g + 1] - off_s[g];
      const int32_t tm = (rows + kBM - 1) / kBM;
      const int32_t local = u - ustart_s[g];
      const int32_t mb = local % tm;
      r.n_blk = local / tm;
      r.g = g;
      r.m0 = off_s[g] + mb * kBM;
      r.m_end = min(off_s[g + 1], r.m0 + kBM);
      r.n0 = r.n_blk * Cfg::kOutN;
    } else {
      const int32_t mb = u % p.tiles_m;
      r.n_blk = u / p.tiles_m;
      r.g = 0;
      r.m0 = mb * Cfg::kRowsPerUnit + static_cast<int32_t>(prank) * kBM;  // this CTA's 128 rows
      r.m_end = min(p.M, r.m0 + kBM);
      if constexpr (QUAD)
        r.n0 = r.n_blk * 2 * BN + static_cast<int32_t>(rank >> 1) * BN;  // this pair's 256 columns
      else if constexpr (COUPLE)
        r.n0 = r.n_blk * 2 * BN + static_cast<int32_t>(chalf) * BN;
      else
        r.n0 = r.n_blk * Cfg::kOutN * sub_tiles;
    }
    return r;
  };

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int32_t it = 0, rt_units = 0;
      bool ok = true;
      for (int32_t u = unit0; ok && u < total; u += unit_step) {
        const UnitInfo ui = decode(u);
        for (int s = 0; ok && s < sub_tiles; ++s) {
          const int32_t nb0 = ui.n0 + s * BN + static_cast<int32_t>(prank) * Cfg::kBRows;
          for (int32_t kb = 0; kb < p.num_kb; ++kb) {
            const int st = it % STAGES;
            const uint32_t ph = (it / STAGES) & 1;
            if (!mbar_wait(&empty[st], ph ^ 1, abort_flag, p.wait_ns)) {
              *abort_flag = 1;
              raise_err(p.err, p.err_dev, kErrWaitProducer);
              ok = false;
              break;
            }
            uint8_t* a = smA + st * Cfg::kASlot;
            uint8_t* b = smB + st * Cfg::kBBytes;
            if constexpr (CTA2) {
              // both CTAs' copies complete on the leader's full barrier
              if (leader) mbar_arrive_expect_tx(&full[st], Cfg::kTxBytes);
              const uint32_t fb = mapa_shared(smem_u32(&full[st]), lead_rank);
              tma_load_2d_pair(a, &tmA, fb, kb * kBK, ui.m0);
              tma_load_3d_pair(b, &tmB, fb, kb * kBK, nb0, ui.g);
            } else {
              mbar_arrive_expect_tx(&full[st], Cfg::kTxBytes);
              tma_load_2d(a, &tmA, &full[st], kb * kBK, ui.m0);
              if constexpr (MODE == kModeSwiglu) {
                tma_load_3d(b, &tmB, &full[st], kb * kBK, ui.n0, ui.g);
                tma_load_3d(b + Cfg::kOutN * 128, &tmB, &full[st], kb * kBK, p.b_rows + ui.n0, ui.g);
              } else {
                tma_load_3d(b, &tmB, &full[st], kb * kBK, nb0, ui.g);
              }
            }
            ++it;
          }
          if constexpr (RT) {
            // the unit's residual tile into the next two slots; each epilogue
            // warp's blocks complete on its own barrier
            int sr[2] = {0, 0};
            for (int r = 0; ok && r < 2; ++r) {
              const int st = it % STAGES;
              const uint32_t ph = (it / STAGES) & 1;
              if (!mbar_wait(&empty[st], ph ^ 1, abort_flag, p.wait_ns)) {
                *abort_flag = 1;
                raise_err(p.err, p.err_dev, kErrWaitProducer);
                ok = false;
                break;
              }
              if (leader) mbar_arrive(&full[st]);  // one phase per slot use, as for operand slots
              sr[r] = st;
              ++it;
            }
            if (!ok) break;
            for (int w = 0; w < Cfg::kEpiW; ++w) {
              uint32_t bytes = 0;
              for (int c = w >> 2; c < Cfg::kOutN / 32; c += Cfg::kH)
                if (ui.n0 + c * 32 < p.N) bytes += 2048;
              mbar_arrive_expect_tx(&rbar[w], bytes);
            }
            for (int c = 0; c < Cfg::kOutN / 32 && ui.n0 + c * 32 < p.N; ++c)
              for (int qq = 0; qq < 4; ++qq)
                tma_load_2d(res_block(sr[0], sr[1], c, qq), &tmR, &rbar[(c % Cfg::kH) * 4 + ((qq + 2) & 3)], ui.n0 + c * 32,
                            ui.m0 + qq * 32);
            ++rt_units;
          }
        }
      }
      if (!ok) {
        if constexpr (RT) {
          // residual copies still in flight land before the CTA exits
          if (rt_units > 0)
            for (int w = 0; w < Cfg::kEpiW; ++w) mbar_wait(&rbar[w], (rt_units - 1) & 1, zero_flag, p.drain_ns);
        }
        if (!CTA2 || leader) {
          // wait (bounded) for the copies still in flight before the CTA exits
          for (int32_t j = (it > STAGES ? it - STAGES : 0); j < it; ++j)
            mbar_wait(&full[j % STAGES], (j / STAGES) & 1, zero_flag, p.drain_ns);
        } else {
          // the peer's copies complete on the leader's barrier: give them time to land
          const uint64_t t0 = globaltimer_ns();
          while (globaltimer_ns() - t0 < 100000ull) {
          }
        }
      }
    }
  } else if (warp == 1) {
    // ----------------------------------------------------------------- MMA
    if (lane == 0 && leader) {
      int32_t it = 0, tl = 0;
      bool ok = true;
      // operand format of kind::f16: bf16 (as compiled) or fp16 (A and B alike)
      const uint32_t idesc = p.ab_f16 ? (Cfg::kIdesc & ~((7u << 7) | (7u << 10))) : Cfg::kIdesc;
      for (int32_t u = unit0; ok && u < total; u += unit_step) {
        for (int s = 0; ok && s < sub_tiles; ++s) {
          const int acc = tl & 1;
          if (!mbar_wait(&acce[acc], ((tl >> 1) & 1) ^ 1, abort_flag, p.wait_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d = tmem + acc * Cfg::kAccStride;
          for (int32_t kb = 0; kb < p.num_kb; ++kb) {
            const int st = it % STAGES;
            const uint32_t ph = (it / STAGES) & 1;
            if (!mbar_wait(&full[st], ph, abort_flag, p.wait_ns)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t a0 = smem_u32(smA + st * Cfg::kASlot);
            const uint32_t b0 = smem_u32(smB + st * Cfg::kBBytes);
#pragma unroll
            for (int kk = 0; kk < kBK / 16; ++kk) {
              const uint64_t ad = desc_sw128_kmajor(a0 + kk * 32), bd = desc_sw128_kmajor(b0 + kk * 32);
              const uint32_t accum = (kb | kk) != 0 ? 1u : 0u;
              if constexpr (CTA2)
                tc_mma_bf16_pair(d, ad, bd, idesc, accum);
              else
                tc_mma_bf16(d, ad, bd, idesc, accum);
            }
            if constexpr (CTA2)
              tc_commit_pair_mc(&empty[st], pair_mask);  // frees the slot in both CTAs
            else
              tc_commit(&empty[st]);
            ++it;
          }
          if (!ok) break;
          if constexpr (CTA2)
            tc_commit_pair_mc(&accf[acc], pair_mask);
          else
            tc_commit(&accf[acc]);
          if constexpr (RT) it += 2;  // the unit's residual slots are the epilogue's
          ++tl;
        }
      }
      if (!ok) {
        *abort_flag = 1;
        raise_err(p.err, p.err_dev, kErrWaitMma);
        // arrives once every MMA issued so far has completed
        if constexpr (CTA2)
          tc_commit_pair(drain);
        else
          tc_commit(drain);
        mbar_wait(drain, 0, zero_flag, p.drain_ns);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    // 8 warps: warp w reads TMEM lane quadrant q = w % 4 (rows 32q..32q+31, one
    // row per thread); the two warps of a quadrant (half h = 0, 1) take
    // alternate 32-column chunks and exchange row statistics through shared
    // memory where a reduction needs the whole row / group.
    const int ew = warp - 2;
    const int q = warp & 3;
    const int h = ew >> 2;
    const int32_t row_in_tile = q * 32 + lane;
    if constexpr (GROUPED && MODE == kModeSwiglu) {
      if (p.zero_ptr) {
        // this CTA's share of the scatter target, 16 bytes per thread and step
        const int64_t n16 = p.zero_bytes >> 4;
        const int64_t per = (n16 + gridDim.x - 1) / gridDim.x;
        const int64_t z0 = static_cast<int64_t>(blockIdx.x) * per, z1 = min(n16, z0 + per);
        uint4* zp = static_cast<uint4*>(p.zero_ptr);
        for (int64_t i = z0 + ew * 32 + lane; i < z1; i += 32 * Cfg::kEpiW) zp[i] = make_uint4(0u, 0u, 0u, 0u);
      }
    }
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    const bool fast = p.fast != 0;
    float2* xch = reinterpret_cast<float2*>(misc + 16);  // [2 halves][128 rows]
    float2* xs = xch + 2 * kBM;                           // quad: [2 slots][128 rows] from CTA rank ^ 2
    uint8_t* stage = staging + ew * Cfg::kWarpStaging;  // this warp's 1 KB tile buffers
    uint8_t* rstage = stage + 2048;                     // store mode: residual transposition
    float* gcache = gn_cache + ew * (3 * 4 * 32);  // GroupNorm: [bias | gamma | beta][4 chunks][32]
    const bool res_staged = MODE == kModeStore && p.res_op >= 0;
    const bool vec_staged = MODE == kModeStore && p.vec_op >= 0;
    const bool c_tiles = p.c_dtype == KF_BF16 && p.c_vec_ok != 0;
    const bool c_tma = p.c_tma != 0;
    int32_t tl = 0;
    bool ok = true;
    // residual tile state: the warp's bias cache, the bias vector and the phase
    // of the warp's residual barrier
    uint8_t* bcache = staging + ew * Cfg::kWarpStaging;
    const __nv_bfloat16* rt_bias_ptr =
        RT ? reinterpret_cast<const __nv_bfloat16*>(p.pre[p.vec_op < 0 ? 0 : p.vec_op].p0) : nullptr;
    uint32_t rt_phase = 0;

    auto wait_acc = [&](int32_t t) -> bool {
      bool w = mbar_wait(&accf[t & 1], (t >> 1) & 1, abort_flag, p.wait_ns);
      w = __all_sync(0xffffffffu, w);
      if (!w) {
        *abort_flag = 1;
        if (lane == 0) raise_err(p.err, p.err_dev, kErrWaitEpilogue);
        return false;
      }
      tc_fence_after();
      return true;
    };
    auto release_acc = [&](int32_t t) {
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (CTA2 && !leader)
          mbar_arrive_remote(mapa_shared(smem_u32(&acce[t & 1]), lead_rank));
        else
          mbar_arrive(&acce[t & 1]);
      }
    };
    // the two warps of this quadrant meet here (named barrier 1 + q, 64 threads)
    auto pair_sync = [&]() { asm volatile("bar.sync %0, %1;" ::"r"(1 + q), "r"(64) : "memory"); };
    // both warps of the quadrant vote; true only if both passed.  Used right
    // after an accumulator wait in the modes that exchange data, so the pair
    // always takes the same abort decision before meeting at pair_sync.
    auto pair_vote = [&](bool mine) -> bool {
      uint32_t r;
      asm volatile(
          "{\n\t.reg .pred pi, po;\n\t"
          "setp.ne.u32 pi, %1, 0;\n\t"
          "bar.red.and.pred po, %2, 64, pi;\n\t"
          "selp.u32 %0, 1, 0, po;\n\t}\n"
          : "=r"(r)
          : "r"(mine ? 1u : 0u), "r"(1 + q)
          : "memory");
      return r != 0;
    };
    // grouped GEMMs: add the unit's group bias (bf16) to 32 accumulator columns
    auto add_gbias = [&](float (&x)[32], int32_t g, int64_t col, int nvalid) {
      if (!p.gbias) return;
      float b[32];
      ld32(p.gbias, KF_BF16, static_cast<int64_t>(g) * p.gbias_ld + col, nvalid, true, b);
#pragma unroll
      for (int j = 0; j < 32; ++j) x[j] += b[j];
    };
    // Chan's pairwise merge of (count, mean, M2) moments
    auto chan = [](float na, float ma, float qa, float nb, float mb, float qb, float& n, float& m, float& qq) {
      n = na + nb;
      if (n == 0.0f) { m = 0.0f; qq = 0.0f; return; }
      const float d = mb - ma;
      m = ma + d * (nb / n);
      qq = qa + qb + d * d * (na * nb / n);
    };

    for (int32_t u = unit0; ok && u < total; u += unit_step) {
      const UnitInfo ui = decode(u);
      const int32_t grow = ui.m0 + row_in_tile;
      const bool row_ok = grow < ui.m_end;
      const int32_t wrow0 = ui.m0 + q * 32;                      // first row of this warp's 32
      const int wrows = max(0, min(32, ui.m_end - wrow0));       // rows of them that exist
      // pull this unit's residual rows toward L2 while its mainloop runs
      if (!RT && res_staged && row_ok) {
        const DevOp& ro = p.pre[p.res_op];
        const __nv_bfloat16* rp = reinterpret_cast<const __nv_bfloat16*>(ro.p0) + static_cast<int64_t>(grow) * ro.ld;
        for (int c = h + 2; c < Cfg::kOutN / 32; c += 2)
          if (ui.n0 + c * 32 < p.N) prefetch_l2(rp + ui.n0 + c * 32);
      }

      if constexpr (MODE == kModeStore || MODE == kModeSwiglu || MODE == kModeScatter) {
        // loads of the residual / bias chunk next in line (in flight across the wait)
        uint4 rq[4], bq[4];
        auto issue_chunk = [&](int c) {
          const int32_t col0 = ui.n0 + c * 32;
          if (c >= Cfg::kOutN / 32 || p.N - col0 < 32) return;
          if (res_staged) {
            const DevOp& ro = p.pre[p.res_op];
            tile32_issue(reinterpret_cast<const __nv_bfloat16*>(ro.p0) + static_cast<int64_t>(wrow0) * ro.ld + col0,
                         ro.ld, wrows, lane, rq);
          }
          if (vec_staged) vec32_issue(p.pre[p.vec_op].p0, col0, bq);
        };
        // residual tile: this warp's chunks of the bias (one 16-byte unit per lane
        // 0..15) are requested before the wait; the producer loads the residual
        uint4 rt_bias = make_uint4(0u, 0u, 0u, 0u);
        if constexpr (RT) {
          if (lane < 16) {
            const int c = h + Cfg::kH * (lane >> 2);
            const int32_t col = ui.n0 + c * 32 + (lane & 3) * 8;
            if (c < Cfg::kOutN / 32 && col + 8 <= p.N) rt_bias = ldg_v4_pinned(rt_bias_ptr + col);
          }
        } else if constexpr (MODE == kModeStore) {
          issue_chunk(h);
        }
        if (!wait_acc(tl)) { ok = false; break; }
        if constexpr (RT) {
          if (lane < 16) *reinterpret_cast<uint4*>(bcache + (lane >> 2) * 64 + (lane & 3) * 16) = rt_bias;
          bool got = mbar_wait(&rbar[ew], rt_phase, abort_flag, p.wait_ns);
          got = __all_sync(0xffffffffu, got);
          if (!got) {
            *abort_flag = 1;
            if (lane == 0) raise_err(p.err, p.err_dev, kErrWaitEpilogue);
            ok = false;
            break;
          }
          rt_phase ^= 1u;
          __syncwarp();
        }
        // ring slots holding this unit's residual tile (after its k-blocks)
        const int32_t rt_pos = tl * (p.num_kb + 2) + p.num_kb;
        const int rt_s0 = rt_pos % STAGES, rt_s1 = (rt_pos + 1) % STAGES;
        const uint32_t tb = tmem + lane_off + (tl & 1) * Cfg::kAccStride;
        float rs = 0.0f;
        int32_t dst = 0;
        bool wr = row_ok;
        if constexpr (MODE == kModeScatter) {
          if (row_ok) {
            rs = p.row_scale[grow];
            dst = p.row_dst[grow];
            if (dst < 0 || dst >= p.dst_rows) {
              raise_err(p.err, p.err_dev, kErrBounds);
              wr = false;
            }
          }
        }
        for (int c = h; c < Cfg::kOutN / 32; c += Cfg::kH) {
          const int32_t col0 = ui.n0 + c * 32;
          const int nvalid = min(32, p.N - col0);
          if (nvalid <= 0) break;  // uniform across the warp
          __syncwarp();
          float v[32];
          if constexpr (RT) {
            // residual from the tile (64-byte swizzle, row = lane), bias from the
            // warp's cache; the result overwrites the residual in place
            uint8_t* blk = res_block(rt_s0, rt_s1, c, q);
            const uint4* bc = reinterpret_cast<const uint4*>(bcache + ((c - h) / Cfg::kH) * 64);
            Staged32 sg;
            sg.use_res = true;
            sg.vec_idx = p.vec_op;
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const uint4 r = *reinterpret_cast<const uint4*>(blk + sw64_off(lane, u));
              const uint4 b = bc[u];
              sg.res[4 * u] = r.x;
              sg.res[4 * u + 1] = r.y;
              sg.res[4 * u + 2] = r.z;
              sg.res[4 * u + 3] = r.w;
              sg.vec[4 * u] = b.x;
              sg.vec[4 * u + 1] = b.y;
              sg.vec[4 * u + 2] = b.z;
              sg.vec[4 * u + 3] = b.w;
            }
            tmem_ld32(tb + c * 32, v);
            run_chain<PRE>(fast, p.pre, p.n_pre, v, grow, col0, nvalid, row_ok, sg);
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              uint4 w;
              w.x = pack_bf16x2(v[8 * u + 0], v[8 * u + 1]);
              w.y = pack_bf16x2(v[8 * u + 2], v[8 * u + 3]);
              w.z = pack_bf16x2(v[8 * u + 4], v[8 * u + 5]);
              w.w = pack_bf16x2(v[8 * u + 6], v[8 * u + 7]);
              *reinterpret_cast<uint4*>(blk + sw64_off(lane, u)) = w;
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              tma_store_2d(&tmC, blk, col0, wrow0);  // rows / columns outside Y are clipped
              bulk_commit_group();
            }
          } else if constexpr (MODE == kModeStore) {
            // operands of this chunk were issued one chunk ahead; issue the next
            Staged32 sg;
            sg.use_res = res_staged && nvalid == 32;
            sg.vec_idx = (vec_staged && nvalid == 32) ? p.vec_op : -1;
            if (sg.use_res) tile32_finish(rstage, lane, rq, sg.res);
            if (sg.vec_idx >= 0) pack16(bq, sg.vec);
            issue_chunk(c + 2);
            tmem_ld32(tb + c * 32, v);
            if constexpr (GROUPED) add_gbias(v, ui.g, col0, nvalid);
            run_chain<PRE>(fast, p.pre, p.n_pre, v, grow, col0, nvalid, row_ok, sg);
          } else if constexpr (MODE == kModeSwiglu) {
            float gt[32];
            tmem_ld32(tb + c * 32, gt);
            tmem_ld32(tb + Cfg::kOutN + c * 32, v);
            if (p.gbias) {
              add_gbias(gt, ui.g, col0, nvalid);
              add_gbias(v, ui.g, p.b_rows + col0, nvalid);
            }
            if (p.sw_ext) {
              // gated expert: gate clamped from above, linear branch on both sides
              const float L = p.sw_limit, al = p.sw_alpha, c1 = p.sw_c;
#pragma unroll
              for (int j = 0; j < 32; ++j) {
                float g1 = gt[j], u1 = v[j];
                if (L > 0.0f) {
                  g1 = fminf(g1, L);
                  u1 = fminf(fmaxf(u1, -L), L);
                }
                v[j] = g1 * (fast ? f_sigmoid_fast(al * g1) : f_sigmoid(al * g1)) * (u1 + c1);
              }
            } else if (fast) {
              // fp32 hardware tanh: h feeds the down GEMM, which sums 2880 of
              // them, so it keeps more precision than a direct bf16 output needs
#pragma unroll
              for (int j = 0; j < 32; ++j) v[j] = gt[j] * f_sigmoid_fast(gt[j]) * v[j];
            } else {
#pragma unroll
              for (int j = 0; j < 32; ++j) v[j] = gt[j] * f_sigmoid(gt[j]) * v[j];
            }
            run_chain<POST>(fast, p.post, p.n_post, v, grow, col0, nvalid, row_ok);
          } else {
            tmem_ld32(tb + c * 32, v);
            if constexpr (GROUPED) add_gbias(v, ui.g, col0, nvalid);
            run_chain<PRE>(fast, p.pre, p.n_pre, v, grow, col0, nvalid, row_ok);
          }
          if constexpr (RT) {
            // stored above
          } else if constexpr (MODE == kModeScatter) {
            float* dstp = reinterpret_cast<float*>(p.C) + static_cast<int64_t>(dst) * p.ldc + col0;
            if (nvalid == 32 && p.c_vec_ok) {
              // row = lane: the scaled row segment passes through this lane's
              // 64 bytes of the warp buffer, 16 columns at a time, and the TMA
              // unit adds it to the destination row
              float4* sb = reinterpret_cast<float4*>(stage) + lane * 4;
#pragma unroll
              for (int hf = 0; hf < 2; ++hf) {
                bulk_wait_group_read<0>();  // this lane's previous segment has been read
#pragma unroll
                for (int u = 0; u < 4; ++u)
                  sb[u] = make_float4(v[16 * hf + 4 * u] * rs, v[16 * hf + 4 * u + 1] * rs,
                                      v[16 * hf + 4 * u + 2] * rs, v[16 * hf + 4 * u + 3] * rs);
                fence_proxy_async_smem();
                if (wr) {
                  bulk_reduce_add_f32(dstp + 16 * hf, sb, 64);
                  bulk_commit_group();
                }
              }
            } else if (wr) {
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (j < nvalid) atomicAdd(dstp + j, v[j] * rs);
            }
          } else if (c_tma) {
            store_tile32_tma(stage, lane, v, &tmC, col0, wrow0);
          } else if (c_tiles && nvalid == 32) {
            store_tile32_bf16(stage, lane, v,
                              reinterpret_cast<__nv_bfloat16*>(p.C) + static_cast<int64_t>(wrow0) * p.ldc + col0, p.ldc,
                              wrows);
          } else {
            if (row_ok) st32(p.C, p.c_dtype, static_cast<int64_t>(grow) * p.ldc + col0, nvalid, p.c_vec_ok != 0, v);
          }
        }
        if constexpr (RT) {
          // this warp's stores have read its blocks: the last warp to get here
          // frees the unit's two residual slots
          if (lane == 0) {
            bulk_wait_group_read<0>();
            __threadfence_block();
            if (atomicAdd(&rdone[tl & 1], 1) == Cfg::kEpiW - 1) {
              rdone[tl & 1] = 0;
              __threadfence_block();
              mbar_arrive(&empty[rt_s0]);
              mbar_arrive(&empty[rt_s1]);
            }
          }
        }
        release_acc(tl);
        ++tl;
      } else if constexpr (MODE == kModeRope) {
        // this row's table row and cache row, requested before the wait
        int32_t pos = 0, crow = 0;
        if (row_ok) {
          pos = p.rope_pos[grow];
          crow = p.row_dst[grow];
        }
        if (!wait_acc(tl)) { ok = false; break; }
        bool wr = row_ok;
        if (row_ok && (pos < 0 || pos >= p.rope_max_pos || crow < 0 || crow >= p.dst_rows)) {
          raise_err(p.err, p.err_dev, kErrBounds);
          wr = false;
        }
        const uint32_t tb = tmem + lane_off + (tl & 1) * Cfg::kAccStride;
        // rotation pairs: chunk lo of a head's first half with chunk lo + hh of
        // its second half (hh chunks of 32 columns per half head); the tile
        // holds whole heads (BN a multiple of rope_d, tiles start on a head).
        // Pair j of the tile: head j / hh, chunk j % hh of its first half.
        const int hc = p.rope_d >> 5;
        const int hh = hc >> 1;
        const int half = p.rope_d >> 1;
        auto pair_col = [&](int j) -> int32_t { return ui.n0 + ((j / hh) * hc + j % hh) * 32; };
        // bias chain, rotation (query and key heads) and the store of one pair
        auto finish = [&](float (&a)[32], float (&b)[32], int32_t col_lo) {
          const int32_t col_hi = col_lo + half;
          run_chain<PRE>(fast, p.pre, p.n_pre, a, grow, col_lo, 32, row_ok);
          run_chain<PRE>(fast, p.pre, p.n_pre, b, grow, col_hi, 32, row_ok);
          const int32_t hcol = col_lo - (col_lo % p.rope_d);  // first column of the head
          if (wr && hcol < p.rope_rot_cols) {
            const int32_t i0 = col_lo - hcol;  // index of the pair within the half head
            const float4* cp = reinterpret_cast<const float4*>(p.rope_cos + static_cast<int64_t>(pos) * half + i0);
            const float4* sp = reinterpret_cast<const float4*>(p.rope_sin + static_cast<int64_t>(pos) * half + i0);
            float4 c4[8], s4[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              c4[u] = __ldg(cp + u);
              s4[u] = __ldg(sp + u);
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              const float cc[4] = {c4[u].x, c4[u].y, c4[u].z, c4[u].w};
              const float ss[4] = {s4[u].x, s4[u].y, s4[u].z, s4[u].w};
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float x0 = a[4 * u + e], x1 = b[4 * u + e];
                a[4 * u + e] = fmaf(x0, cc[e], -x1 * ss[e]);
                b[4 * u + e] = fmaf(x1, cc[e], x0 * ss[e]);
              }
            }
          }
          if (wr) {
            if (hcol < p.rope_q_cols) {
              const int64_t base = static_cast<int64_t>(grow) * p.ldc;
              st32(p.C, p.c_dtype, base + col_lo, 32, p.c_vec_ok != 0, a);
              st32(p.C, p.c_dtype, base + col_hi, 32, p.c_vec_ok != 0, b);
            } else {
              const bool is_k = hcol < p.rope_rot_cols;
              void* cache = is_k ? p.k_cache : p.v_cache;
              const int64_t base = static_cast<int64_t>(crow) * p.ld_cache - (is_k ? p.rope_q_cols : p.rope_rot_cols);
              st32(cache, p.c_dtype, base + col_lo, 32, p.kv_vec_ok != 0, a);
              st32(cache, p.c_dtype, base + col_hi, 32, p.kv_vec_ok != 0, b);
            }
          }
        };
        for (int j = h; j < Cfg::kOutN / 64; j += Cfg::kH) {
          const int32_t col_lo = pair_col(j);
          if (col_lo >= p.N) break;  // N is whole heads: the partner exists too
          const int clo = (col_lo - ui.n0) >> 5;
          float a[32], b[32];
          tmem_ld32(tb + clo * 32, a);
          tmem_ld32(tb + (clo + hh) * 32, b);
          finish(a, b, col_lo);
        }
        release_acc(tl);
        ++tl;
      } else if constexpr (MODE == kModeLse) {
        if (!pair_vote(wait_acc(tl))) { ok = false; break; }
        const uint32_t tb = tmem + lane_off + (tl & 1) * Cfg::kAccStride;
        const bool rsum = p.red_sum != 0;  // row sum (s only) instead of (max, sum exp)
        float m = -INFINITY, s = 0.0f;
        for (int c = h; c < BN / 32; c += 2) {
          const int32_t col0 = ui.n0 + c * 32;
          const int nvalid = min(32, p.N - col0);
          if (nvalid <= 0) break;
          __syncwarp();
          float v[32];
          tmem_ld32(tb + c * 32, v);
          run_chain<PRE>(false, p.pre, p.n_pre, v, grow, col0, nvalid, row_ok);
          if (rsum) {
            float add = 0.0f;
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (j < nvalid) add += v[j];
            s += add;
            continue;
          }
          float cm = -INFINITY;
#pragma unroll
          for (int j = 0; j < 32; ++j)
            if (j < nvalid) cm = fmaxf(cm, v[j]);
          const float nm = fmaxf(m, cm);
          float add = 0.0f;
#pragma unroll
          for (int j = 0; j < 32; ++j)
            if (j < nvalid) add += __expf(v[j] - nm);
          s = (m == -INFINITY ? 0.0f : s * __expf(m - nm)) + add;
          m = nm;
        }
        release_acc(tl);
        ++tl;
        // merge the two halves of the row: half 1 hands (m, s) to half 0
        if (h == 1) xch[row_in_tile] = make_float2(m, s);
        pair_sync();
        if (h == 0) {
          const float2 o = xch[row_in_tile];
          float2 part;
          if (rsum) {
            part = make_float2(0.0f, s + o.y);  // half 0's columns, then half 1's
          } else {
            const float nm = fmaxf(m, o.x);
            float ss = 0.0f;
            if (nm != -INFINITY)
              ss = (m == -INFINITY ? 0.f : s * __expf(m - nm)) + (o.x == -INFINITY ? 0.f : o.y * __expf(o.x - nm));
            part = make_float2(nm, ss);
          }
          if (row_ok) p.lse_part[static_cast<int64_t>(grow) * p.tiles_n + ui.n_blk] = part;
        }
        pair_sync();  // xch is reused by the next tile
      } else if constexpr (MODE == kModeGroupNorm) {
        const int32_t gs = p.norm.groups;  // group size (columns), multiple of 32
        const float eps = p.norm.eps;
        // a row sum after the post chain (red_sum): each thread adds up the
        // chunks it finishes instead of storing them; the quadrant's two warps
        // then merge (half 0 first) and write one partial per 256-column block
        const bool gn_sum = p.red_sum != 0;
        float rsum = 0.0f;
        auto emit_sum = [&](int32_t col_base, int blocks) {
          xch[h * kBM + row_in_tile] = make_float2(rsum, 0.0f);
          pair_sync();
          if (h == 0 && row_ok) {
            const float tot = rsum + xch[kBM + row_in_tile].x;
            float2* dst = p.lse_part + static_cast<int64_t>(grow) * p.red_parts + col_base / 256;
            dst[0] = make_float2(0.0f, tot);
            for (int b = 1; b < blocks && col_base / 256 + b < p.red_parts; ++b) dst[b] = make_float2(0.0f, 0.0f);
          }
          pair_sync();  // xch is reused by the next unit
        };
        // normalise + affine + post chain + store one 32-column chunk
        // bias / gamma / beta of this warp's chunks of one accumulator, loaded
        // once into the warp's cache (coalesced, lane j = column j) so the
        // normalize pass reads them from shared memory
        const bool pre_bias = PRE_IS_BIAS;  // compiled program: the pre-chain is one bias op
        // the vectors of the warp's 4 chunks c0, c0 + step, ... (lane j = column j
        // of each chunk) are loaded into registers first, all at once, and
        // parked in the cache later: one memory round trip instead of twelve
        // (raw bits: the conversions wait for the loads only in park_vecs)
        uint32_t vb[4], vg[4], vt[4];
        auto issue_vecs = [&](int32_t colbase, int c0, int c1, int step) {
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int c = c0 + i * step;
            const int32_t col = colbase + c * 32 + lane;
            const bool in = c < c1;
            vb[i] = (in && pre_bias) ? ld_raw(p.pre[0].p0, p.pre[0].p_dtype, col) : 0u;
            vg[i] = (in && p.norm.p0) ? ld_raw(p.norm.p0, p.norm.p_dtype, col) : 0u;
            vt[i] = (in && p.norm.p1) ? ld_raw(p.norm.p1, p.norm.p_dtype, col) : 0u;
          }
        };
        auto park_vecs = [&]() {
          const int bdt = pre_bias ? p.pre[0].p_dtype : KF_F32, ndt = p.norm.p_dtype;
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            gcache[i * 32 + lane] = pre_bias ? cvt_raw(vb[i], bdt) : 0.0f;
            gcache[(4 + i) * 32 + lane] = p.norm.p0 ? cvt_raw(vg[i], ndt) : 1.0f;
            gcache[(8 + i) * 32 + lane] = p.norm.p1 ? cvt_raw(vt[i], ndt) : 0.0f;
          }
          __syncwarp();
        };
        auto fill_cache = [&](int32_t colbase, int c0, int c1, int step) {
          __syncwarp();  // the previous chunks' reads of the cache are done
          issue_vecs(colbase, c0, c1, step);
          park_vecs();
        };
        auto finish_chunk = [&](uint32_t taddr, int32_t col0, float mean, float rstd, int slot) {
          float v[32];
          tmem_ld32(taddr, v);
          const float4* cb = reinterpret_cast<const float4*>(gcache + slot * 32);
          const float4* cg = reinterpret_cast<const float4*>(gcache + (4 + slot) * 32);
          const float4* ct = reinterpret_cast<const float4*>(gcache + (8 + slot) * 32);
          if (pre_bias) {
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              const float4 b = cb[k];
              v[4 * k] += b.x;
              v[4 * k + 1] += b.y;
              v[4 * k + 2] += b.z;
              v[4 * k + 3] += b.w;
            }
          } else {
            run_chain<PRE>(false, p.pre, p.n_pre, v, grow, col0, 32, row_ok);
          }
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const float4 g = cg[k], t = ct[k];
            v[4 * k] = (v[4 * k] - mean) * rstd * g.x + t.x;
            v[4 * k + 1] = (v[4 * k + 1] - mean) * rstd * g.y + t.y;
            v[4 * k + 2] = (v[4 * k + 2] - mean) * rstd * g.z + t.z;
            v[4 * k + 3] = (v[4 * k + 3] - mean) * rstd * g.w + t.w;
          }
          run_chain<POST>(fast, p.post, p.n_post, v, grow, col0, 32, row_ok);
          if (gn_sum) {
            float add = 0.0f;
#pragma unroll
            for (int j = 0; j < 32; ++j) add += v[j];
            rsum += add;
            return;
          }
          if (c_tma)
            store_tile32_tma(stage, lane, v, &tmC, col0, wrow0);
          else if (c_tiles)
            store_tile32_bf16(stage, lane, v,
                              reinterpret_cast<__nv_bfloat16*>(p.C) + static_cast<int64_t>(wrow0) * p.ldc + col0, p.ldc,
                              wrows);
          else if (row_ok)
            st32(p.C, p.c_dtype, static_cast<int64_t>(grow) * p.ldc + col0, 32, p.c_vec_ok != 0, v);
        };
        // (count, mean, M2) of this thread's chunks c0, c0+step, ... < c1 in one pass over
        // TMEM: exact two-pass moments of each 32-value chunk in registers, merged
        // chunk by chunk with Chan's formula.
        // With `cached`, a bias pre-chain reads the chunks' bias from the cache
        // (parked for chunks c0, c0 + step, ... in order).
        auto moments = [&](uint32_t tb, int32_t colbase, int c0, int c1, int step, float& n, float& mean, float& m2,
                           bool cached) {
          n = 0.0f;
          mean = 0.0f;
          m2 = 0.0f;
          int slot = 0;
          for (int c = c0; c < c1; c += step, ++slot) {
            __syncwarp();
            float v[32];
            tmem_ld32(tb + c * 32, v);
            if (cached && pre_bias) {
              const float4* cb = reinterpret_cast<const float4*>(gcache + slot * 32);
#pragma unroll
              for (int k = 0; k < 8; ++k) {
                const float4 b = cb[k];
                v[4 * k] += b.x;
                v[4 * k + 1] += b.y;
                v[4 * k + 2] += b.z;
                v[4 * k + 3] += b.w;
              }
            } else {
              run_chain<PRE>(false, p.pre, p.n_pre, v, grow, colbase + c * 32, 32, row_ok);
            }
            float sum = 0.0f;
#pragma unroll
            for (int j = 0; j < 32; ++j) sum += v[j];
            const float cmean = sum * (1.0f / 32.0f);
            float cq = 0.0f;
#pragma unroll
            for (int j = 0; j < 32; ++j) cq += (v[j] - cmean) * (v[j] - cmean);
            chan(n, mean, m2, 32.0f, cmean, cq, n, mean, m2);
          }
        };
        if (QUAD || COUPLE || (gs == BN && sub_tiles == 1)) {
          // One accumulator holds this CTA's columns of the group: the whole
          // group (gs = BN), or (quad) one 256-column half of a 512-column group
          // whose other half CTA rank ^ 2 holds for the same rows.  The
          // quadrant's two warps split the chunks and merge their moments; with
          // quad, half 0 then sends (mean, M2) of this CTA's 256 columns to the
          // other CTA through distributed shared memory, and both CTAs merge the
          // two column halves in the same order (the lower half first), so both
          // normalise with identical statistics.  Slot tl & 1 is written for tile
          // tl only after the other CTA has passed tile tl - 1, which it reached
          // after reading slot tl & 1 for tile tl - 2.
          issue_vecs(ui.n0, h, BN / 32, 2);  // in flight across the wait
          if (!pair_vote(wait_acc(tl))) { ok = false; break; }
          park_vecs();
          const uint32_t tb = tmem + lane_off + (tl & 1) * Cfg::kAccStride;
          float n, mean, m2;
          moments(tb, ui.n0, h, BN / 32, 2, n, mean, m2, true);
          xch[h * kBM + row_in_tile] = make_float2(mean, m2);
          pair_sync();
          const float2 o = xch[(h ^ 1) * kBM + row_in_tile];
          pair_sync();
          float tn, tm, tq;
          if (h == 0)
            chan(n, mean, m2, n, o.x, o.y, tn, tm, tq);
          else
            chan(n, o.x, o.y, n, mean, m2, tn, tm, tq);
          if constexpr (QUAD) {
            const float cn = tn, cm = tm, cq = tq;
            const int slot = tl & 1;
            const uint32_t other = rank ^ 2u;
            if (h == 0) {
              st_cluster_f2(mapa_shared(smem_u32(xs + slot * kBM + row_in_tile), other), cm, cq);
              mbar_arrive_remote(mapa_shared(smem_u32(&xbar[slot]), other));
            }
            bool got = mbar_wait_cluster(&xbar[slot], (tl >> 1) & 1, abort_flag, p.wait_ns);
            got = __all_sync(0xffffffffu, got);
            if (!pair_vote(got)) {
              *abort_flag = 1;
              if (lane == 0) raise_err(p.err, p.err_dev, kErrWaitEpilogue);
              ok = false;
              break;
            }
            const float2 r = xs[slot * kBM + row_in_tile];
            if ((rank >> 1) == 0)
              chan(cn, cm, cq, cn, r.x, r.y, tn, tm, tq);
            else
              chan(cn, r.x, r.y, cn, cm, cq, tn, tm, tq);
          } else if constexpr (COUPLE) {
            // the same through global memory: half 0 writes (mean, M2) of its rows,
            // fences, and one lane publishes the warp's 32 rows with a release
            // store of (epoch, tile + 1) to the rows' flag; the other pair's warps
            // of the same rows wait for that exact value (acquire), then read.
            // Slots alternate with the tile as above.
            const float cn = tn, cm = tm, cq = tq;
            const size_t slot = static_cast<size_t>(tl & 1);
            const size_t mine = (static_cast<size_t>(unit0) * 2 + slot) * 2 + chalf;
            const size_t other = (static_cast<size_t>(unit0) * 2 + slot) * 2 + (chalf ^ 1u);
            const int32_t row_u = static_cast<int32_t>(prank) * kBM + row_in_tile;  // row within the unit
            const int fl = static_cast<int>(prank) * 4 + q;                         // the warp's 32 rows
            const unsigned long long want =
                (static_cast<unsigned long long>(p.gx_epoch) << 32) | static_cast<uint32_t>(tl + 1);
            if (h == 0) {
              p.gx_data[mine * 256 + row_u] = make_float2(cm, cq);
              __threadfence();
              __syncwarp();
              if (lane == 0) st_release_gpu_u64(p.gx_flag + mine * 8 + fl, want);
            }
            bool got = flag_wait_gpu(p.gx_flag + other * 8 + fl, want, abort_flag, p.wait_ns);
            got = __all_sync(0xffffffffu, got);
            if (!pair_vote(got)) {
              *abort_flag = 1;
              if (lane == 0) raise_err(p.err, p.err_dev, kErrWaitEpilogue);
              ok = false;
              break;
            }
            const float2 r = ld_relaxed_gpu_f2(p.gx_data + other * 256 + row_u);
            if (chalf == 0)
              chan(cn, cm, cq, cn, r.x, r.y, tn, tm, tq);
            else
              chan(cn, r.x, r.y, cn, cm, cq, tn, tm, tq);
          }
          const float rstd = rsqrtf(tq / tn + eps);
          int cs = 0;
          for (int c = h; c < BN / 32; c += 2, ++cs) {
            __syncwarp();
            finish_chunk(tb + c * 32, ui.n0 + c * 32, tm, rstd, cs);
          }
          __syncwarp();
          release_acc(tl);
          ++tl;
          if (gn_sum) emit_sum(ui.n0, 1);
        } else if (gs < BN) {
          // several whole groups per tile: half h takes groups h, h+2, ...
          // (a row sum merges the halves after the tile: both vote first)
          bool got = wait_acc(tl);
          if (gn_sum) got = pair_vote(got);
          if (!got) { ok = false; break; }
          const uint32_t tb = tmem + lane_off + (tl & 1) * Cfg::kAccStride;
          const int nch = gs / 32;
          for (int gi = h; gi < BN / gs; gi += 2) {
            const int32_t g0 = ui.n0 + gi * gs;
            if (g0 >= p.N) break;
            float n, mean, m2;
            moments(tb + gi * gs, g0, 0, nch, 1, n, mean, m2, false);
            const float rstd = rsqrtf(m2 / n + eps);
            fill_cache(g0, 0, nch, 1);
            for (int c = 0; c < nch; ++c) {
              __syncwarp();
              finish_chunk(tb + gi * gs + c * 32, g0 + c * 32, mean, rstd, c);
            }
            __syncwarp();
          }
          release_acc(tl);
          ++tl;
          if (gn_sum) emit_sum(ui.n0, 1);
        } else {
          // one group spans sub_tiles (1 or 2) accumulators of BN columns; the two
          // halves split its chunks and merge their moments through shared memory
          float n = 0.f, mean = 0.f, m2 = 0.f;
          for (int st = 0; st < sub_tiles; ++st) {
            if (!pair_vote(wait_acc(tl + st))) { ok = false; break; }
            const uint32_t tb = tmem + lane_off + ((tl + st) & 1) * Cfg::kAccStride;
            float nb, mb, qb;
            moments(tb, ui.n0 + st * BN, h, BN / 32, 2, nb, mb, qb, false);
            chan(n, mean, m2, nb, mb, qb, n, mean, m2);
          }
          if (!ok) break;
          // the two halves hold equally many columns: only (mean, M2) travel
          xch[h * kBM + row_in_tile] = make_float2(mean, m2);
          pair_sync();
          const float2 o = xch[(h ^ 1) * kBM + row_in_tile];
          pair_sync();
          // both halves merge in the same order (half 0 first) -> identical stats
          float tn, tm, tq;
          if (h == 0)
            chan(n, mean, m2, n, o.x, o.y, tn, tm, tq);
          else
            chan(n, o.x, o.y, n, mean, m2, tn, tm, tq);
          const float rstd = rsqrtf(tq / tn + eps);
          for (int st = 0; st < sub_tiles; ++st) {
            const uint32_t tb = tmem + lane_off + ((tl + st) & 1) * Cfg::kAccStride;
            fill_cache(ui.n0 + st * BN, h, BN / 32, 2);
            int slot = 0;
            for (int c = h; c < BN / 32; c += 2, ++slot) {
              __syncwarp();
              finish_chunk(tb + c * 32, ui.n0 + st * BN + c * 32, tm, rstd, slot);
            }
            __syncwarp();
            release_acc(tl + st);
          }
          tl += sub_tiles;
          if (gn_sum) emit_sum(ui.n0, sub_tiles);
        }
      }
    }
  }

  // ---------------------------------------------------------------- teardown
  if (warp >= 2 && (lane == 0 || MODE == kModeScatter)) bulk_wait_group_all();  // this warp's bulk copies have completed
  tc_fence_before();
  __syncwarp();  // lane 0 of the producer / MMA warps arrives after lanes 1-31
  __syncthreads();
  if constexpr (CTA2) cluster_sync();  // no remote access to this CTA remains
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    if constexpr (CTA2)
      tmem_dealloc_pair(tmem, Cfg::kTmemCols);
    else
      tmem_dealloc(tmem, Cfg::kTmemCols);
  }
}

}  // namespace kf
