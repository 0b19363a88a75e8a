// kf_tc_qkv_decode.cu -- the QKV projection tail for decode-sized calls (at most
// 64 tokens): bias + rotary embedding + key / value cache rows, with the K
// dimension split over the CTAs of a cluster and the partial sums reduced
// through distributed shared memory (the gpt-oss decode kernel "Bias + RoPE +
// KV update" of Sec. IV-A, here fused with its GEMM).
//
// A decode GEMM reads each weight once; one 256-column tile per CTA over the
// whole K would keep only N / 256 SMs busy and pay 4 MMAs per 64-wide k-block
// for all of K.  Here a cluster of S CTAs shares one 256-column tile (four
// 64-column heads): CTA r multiplies the k-blocks [r K / S, (r + 1) K / S),
// writes the T token rows of its 128 x 256 fp32 partial from TMEM into its own
// shared memory (the operand ring, free by then), and after a cluster barrier the epilogue warps
// of all S CTAs take the tile's (token, head) items in turn: a warp sums the S
// partials of its item (lane j: columns j and j + d/2 of the head, read from
// each CTA's shared memory through DSMEM), adds the bias, rotates query and key
// heads and stores the row to q_out or to the token's cache row.  No global
// workspace, no atomics, no waits between CTAs other than the two hardware
// cluster barriers.  While the MMAs run, the epilogue warps already load what
// their first items need besides the sums (positions, cache rows, bias, the
// table rows of the positions), so that after the barrier only the partial sums
// are read.
//
// Token rows are staged in boxes of ROWS = 32 (six-stage ring) or 64 rows
// (five stages): the box is what limits the tokens of a call.
//
// Warp roles: warp 0 TMA producer, warp 1 MMA issuer, warps 2-9 epilogue.
#include "kf_internal.h"

namespace kf {
namespace {

constexpr int kDcThreads = 320;
constexpr int kDcBM = 128;          // rows of the MMA (only the first T are tokens)
constexpr int kDcBK = 64;           // K elements per 128-byte row
constexpr int kDcBN = 256;          // tile columns
constexpr int kDcPartStride = 257;  // floats per partial row (odd: conflict-free row-per-lane stores)

template <int ROWS, int STAGES>
struct DcCfg {
  // A: ROWS token rows per k-block (4 or 8 KB).  The MMA reads 128 rows from
  // there; the ones past the box are the next stages' bytes and feed only
  // accumulator rows past T, which are never stored (A stages come first, so
  // the reads stay in the ring).
  static_assert(ROWS == 32 || ROWS == 64, "token box");
  static constexpr int kABytes = ROWS * kDcBK * 2;
  static constexpr int kBBytes = kDcBN * kDcBK * 2;    // 32 KB
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr uint32_t kTxBytes = kStageBytes;
  static constexpr int kPartBytes = ROWS * kDcPartStride * 4;
  static constexpr int kRingBytes = STAGES * kStageBytes;
  static_assert(kPartBytes <= kRingBytes, "the partial fits the ring");
  static_assert(STAGES * kABytes + kBBytes >= kDcBM * kDcBK * 2, "the MMA's 128-row reads stay in the ring");
  static constexpr int kBarBytes = 8 * (2 * STAGES + 2);
  static constexpr int kSmemBytes = 1024 + kRingBytes + kBarBytes + 64;
  static constexpr uint32_t kIdesc = idesc_bf16_f32(kDcBM, kDcBN);
  static_assert(kSmemBytes <= 232448, "shared memory");
};

__device__ __forceinline__ float ld_cluster_f32(uint32_t addr) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(addr) : "memory");
  return v;
}

// Operands of one (token, head) item that do not depend on the sums: lane j
// holds pairs j + 32 m of the head (d / 2 <= 128: m < 4).
constexpr int kBatch = 4, kMaxPl = 4;
struct DcItem {
  int32_t t, hcol, pos, crow;
  bool live, ok, rotate;
  float b0[kMaxPl], b1[kMaxPl], c[kMaxPl], s[kMaxPl];
};

// Items it = base + stride j (j < kBatch) of a tile: token it / heads, head
// it % heads.  All loads are issued before any is used.  A position or cache row
// out of range clears `ok` (the item is then reported and skipped, and no table
// row is read for it).
__device__ __forceinline__ void dc_load_items(const QkvDecodeParams& p, int32_t n0, int32_t base, int32_t stride,
                                              int32_t items, int heads, int lane, DcItem (&it)[kBatch]) {
  const int d = p.rope_d, half = d >> 1, npl = half >> 5;
#pragma unroll
  for (int j = 0; j < kBatch; ++j) {
    const int32_t idx = base + stride * j;
    const int32_t hl = idx % heads;
    it[j].t = idx / heads;
    it[j].hcol = n0 + hl * d;
    it[j].live = idx < items && it[j].hcol < p.N;
    it[j].pos = it[j].live ? p.positions[it[j].t] : 0;
    it[j].crow = it[j].live ? p.cache_rows[it[j].t] : 0;
  }
#pragma unroll
  for (int j = 0; j < kBatch; ++j) {
    it[j].ok = it[j].live && it[j].pos >= 0 && it[j].pos < p.max_pos && it[j].crow >= 0 && it[j].crow < p.rows;
    it[j].rotate = it[j].hcol < p.rot_cols;
#pragma unroll
    for (int m = 0; m < kMaxPl; ++m) {
      const int i = lane + 32 * m;
      const bool use = it[j].ok && m < npl;
      it[j].b0[m] = use && p.bias ? ld_elem(p.bias, p.bias_dtype, it[j].hcol + i) : 0.0f;
      it[j].b1[m] = use && p.bias ? ld_elem(p.bias, p.bias_dtype, it[j].hcol + i + half) : 0.0f;
      const bool tab = use && it[j].rotate;
      it[j].c[m] = tab ? __ldg(p.cos_t + static_cast<int64_t>(it[j].pos) * half + i) : 1.0f;
      it[j].s[m] = tab ? __ldg(p.sin_t + static_cast<int64_t>(it[j].pos) * half + i) : 0.0f;
    }
  }
}

template <int ROWS, int STAGES>
__global__ void __launch_bounds__(kDcThreads, 1)
    kf_qkv_decode_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                         const __grid_constant__ QkvDecodeParams p) {
  using Cfg = DcCfg<ROWS, STAGES>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* smA = sm;                                   // A stages first (see DcCfg)
  uint8_t* smB = sm + STAGES * Cfg::kABytes;
  float* part = reinterpret_cast<float*>(sm);          // after the mainloop: [ROWS][257] fp32
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + Cfg::kRingBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* accf = bars + 2 * STAGES;
  uint64_t* drain = bars + 2 * STAGES + 1;
  uint32_t* misc = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 2);
  uint32_t* tmem_slot = misc;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 1);
  volatile int* zero_flag = reinterpret_cast<volatile int*>(misc + 2);

  // the split count is the cluster size; refuse any other launch shape before
  // any barrier, TMEM allocation or copy
  const uint32_t S = cluster_nctarank();
  if (S != static_cast<uint32_t>(p.splits) || blockDim.x != kDcThreads || gridDim.x % S != 0 || gridDim.y != 1 ||
      gridDim.z != 1 || p.T > ROWS) {
    if (threadIdx.x == 0) atomicOr(p.err, kErrLaunchShape);
    return;
  }
  const uint32_t r = cluster_ctarank();
  const int32_t tile = static_cast<int32_t>(blockIdx.x / S);
  const int32_t n0 = tile * kDcBN;
  const int32_t kb0 = static_cast<int32_t>(r) * p.num_kb / static_cast<int32_t>(S);
  const int32_t kb1 = static_cast<int32_t>(r + 1) * p.num_kb / static_cast<int32_t>(S);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // (token, head) items of the tile go to the cluster's epilogue warps in turn;
  // a warp takes up to kBatch items at a time
  const int heads = kDcBN / p.rope_d;
  const int32_t items = p.T * heads;
  const int32_t stride = static_cast<int32_t>(S) * 8;
  const int32_t first = static_cast<int32_t>(r) + static_cast<int32_t>(S) * (warp - 2);
  DcItem batch[kBatch];  // the epilogue warp's current items

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accf, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    *zero_flag = 0;
    fence_mbarrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    // this CTA's weights into L2 while a preceding kernel may still run: a
    // prefetch reads memory without changing it and L2 is where that kernel's
    // writes land, so the loads after the dependency wait below see current
    // values either way; the weights are the bytes this kernel is bound by
    for (int32_t kb = kb0; kb < kb1; ++kb) tma_prefetch_3d(&tmB, kb * kDcBK, n0, 0);
  }
  if (warp == 1) {
    __syncwarp();
    tmem_alloc(tmem_slot, kDcBN);
    tmem_relinquish();
  }
  // launched as a programmatic dependent of the previous kernel in the stream:
  // wait for it before any operand, position or table is read
  griddep_wait();
  griddep_launch_dependents();
  tc_fence_before();
  __syncwarp();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  bool ok = true;

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      int32_t it = 0;
      for (int32_t kb = kb0; kb < kb1; ++kb, ++it) {
        const int st = it % STAGES;
        if (!mbar_wait(&empty[st], ((it / STAGES) & 1) ^ 1, abort_flag, p.wait_ns)) {
          *abort_flag = 1;
          atomicOr(p.err, kErrWaitProducer);
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&full[st], Cfg::kTxBytes);
        tma_load_2d(smA + st * Cfg::kABytes, &tmA, &full[st], kb * kDcBK, 0);
        tma_load_3d(smB + st * Cfg::kBBytes, &tmB, &full[st], kb * kDcBK, n0, 0);
      }
      if (!ok)  // copies still in flight land before the ring is reused or the CTA exits
        for (int32_t j = (it > STAGES ? it - STAGES : 0); j < it; ++j)
          mbar_wait(&full[j % STAGES], (j / STAGES) & 1, zero_flag, p.drain_ns);
    }
  } else if (warp == 1) {
    // --------------------------------------------------------------------- MMA
    if (lane == 0) {
      const uint32_t idesc = p.ab_f16 ? (Cfg::kIdesc & ~((7u << 7) | (7u << 10))) : Cfg::kIdesc;
      int32_t it = 0;
      for (int32_t kb = kb0; kb < kb1; ++kb, ++it) {
        const int st = it % STAGES;
        if (!mbar_wait(&full[st], (it / STAGES) & 1, abort_flag, p.wait_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a0 = smem_u32(smA + st * Cfg::kABytes);
        const uint32_t b0 = smem_u32(smB + st * Cfg::kBBytes);
#pragma unroll
        for (int kk = 0; kk < kDcBK / 16; ++kk)
          tc_mma_bf16(tmem, desc_sw128_kmajor(a0 + kk * 32), desc_sw128_kmajor(b0 + kk * 32), idesc,
                      (kb != kb0 || kk != 0) ? 1u : 0u);
        tc_commit(&empty[st]);
      }
      if (ok) {
        tc_commit(accf);
      } else {
        *abort_flag = 1;
        atomicOr(p.err, kErrWaitMma);
        tc_commit(drain);  // arrives once every MMA issued so far has completed
        mbar_wait(drain, 0, zero_flag, p.drain_ns);
      }
    }
  } else {
    // ------------------------------------- epilogue part 1: partial -> own smem
    const int ew = warp - 2;
    const int q = warp & 3;                      // TMEM lane quadrant
    const int hh = ew >> 2;                      // column half: [128 hh, 128 hh + 128)
    const int32_t row = q * 32 + lane;
    // the first batch's operands load while the MMAs run
    if (first < items) dc_load_items(p, n0, first, stride, items, heads, lane, batch);
    bool w = mbar_wait(accf, 0, abort_flag, p.wait_ns);
    w = __all_sync(0xffffffffu, w);
    if (!w) {
      *abort_flag = 1;
      if (lane == 0) atomicOr(p.err, kErrWaitEpilogue);
    } else {
      tc_fence_after();
      fence_proxy_async_smem();  // the ring's last copies were async-proxy writes
      const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
      if (q * 32 < p.T) {  // quadrants past the last token have nothing to keep
        for (int c = 0; c < 4; ++c) {
          float v[32];
          tmem_ld32(tmem + lane_off + hh * 128 + c * 32, v);
          if (row < p.T) {
            float* dst = part + row * kDcPartStride + hh * 128 + c * 32;
#pragma unroll
            for (int j = 0; j < 32; ++j) dst[j] = v[j];
          }
        }
      }
    }
  }
  // every CTA's partial is in its shared memory (the ring is idle: all copies
  // landed and all MMAs completed before the accumulator was signalled)
  tc_fence_before();
  __syncwarp();
  cluster_sync();

  if (warp >= 2 && !*abort_flag) {
    // --------------------- epilogue part 2: reduce S partials, bias, rotate, store
    // A warp issues the DSMEM loads of all its batch's partial sums before any
    // arithmetic or store, so their latencies overlap; the other operands of
    // the first batch are in registers already.
    const int d = p.rope_d, half = d >> 1, npl = half >> 5;
    const uint32_t part_base = smem_u32(part);
    for (int32_t base = first; base < items; base += stride * kBatch) {
      if (base != first) dc_load_items(p, n0, base, stride, items, heads, lane, batch);
      float a[kBatch][kMaxPl], b[kBatch][kMaxPl];
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
#pragma unroll
        for (int m = 0; m < kMaxPl; ++m) {
          a[j][m] = 0.0f;
          b[j][m] = 0.0f;
          if (batch[j].ok && m < npl) {
            const int i = lane + 32 * m;
            const uint32_t off = static_cast<uint32_t>((batch[j].t * kDcPartStride + (batch[j].hcol - n0) + i) * 4);
            // all 2S loads in flight before the first add (their round trips
            // overlap), then the sums in CTA-rank order
            float va[8], vb[8];
#pragma unroll
            for (uint32_t s2 = 0; s2 < 8; ++s2) {
              if (s2 < S) {
                const uint32_t bs = mapa_shared(part_base, s2);
                va[s2] = ld_cluster_f32(bs + off);
                vb[s2] = ld_cluster_f32(bs + off + static_cast<uint32_t>(half * 4));
              }
            }
#pragma unroll
            for (uint32_t s2 = 0; s2 < 8; ++s2) {
              if (s2 < S) {
                a[j][m] += va[s2];
                b[j][m] += vb[s2];
              }
            }
          }
        }
      }
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        if (!batch[j].live) continue;
        if (!batch[j].ok) {
          if (lane == 0) atomicOr(p.err, kErrBounds);
          continue;
        }
        const int32_t hcol = batch[j].hcol;
        void* dst;
        int64_t dst0;
        if (hcol < p.q_cols) {
          dst = p.q_out;
          dst0 = static_cast<int64_t>(batch[j].t) * p.ldq + hcol;
        } else {
          dst = batch[j].rotate ? p.k_cache : p.v_cache;
          dst0 = static_cast<int64_t>(batch[j].crow) * p.ld_cache + hcol - (batch[j].rotate ? p.q_cols : p.rot_cols);
        }
#pragma unroll
        for (int m = 0; m < kMaxPl; ++m) {
          if (m >= npl) break;
          const int i = lane + 32 * m;
          float x0 = a[j][m] + batch[j].b0[m], x1 = b[j][m] + batch[j].b1[m];
          if (batch[j].rotate) {
            const float c = batch[j].c[m], sn = batch[j].s[m];
            const float y0 = fmaf(x0, c, -x1 * sn), y1 = fmaf(x1, c, x0 * sn);
            x0 = y0;
            x1 = y1;
          }
          if (p.out_dtype == KF_F32) {
            reinterpret_cast<float*>(dst)[dst0 + i] = x0;
            reinterpret_cast<float*>(dst)[dst0 + i + half] = x1;
          } else if (p.out_dtype == KF_BF16) {
            reinterpret_cast<__nv_bfloat16*>(dst)[dst0 + i] = __float2bfloat16_rn(x0);
            reinterpret_cast<__nv_bfloat16*>(dst)[dst0 + i + half] = __float2bfloat16_rn(x1);
          } else {
            reinterpret_cast<__half*>(dst)[dst0 + i] = __float2half_rn(x0);
            reinterpret_cast<__half*>(dst)[dst0 + i + half] = __float2half_rn(x1);
          }
        }
      }
    }
  }
  // no CTA leaves while another may still read its shared memory
  cluster_sync();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kDcBN);
  }
}

template <int ROWS, int STAGES>
cudaError_t launch_dc(const CUtensorMap& a, const CUtensorMap& b, const QkvDecodeParams& p, int tiles,
                      cudaStream_t s) {
  using Cfg = DcCfg<ROWS, STAGES>;
  auto kern = kf_qkv_decode_kernel<ROWS, STAGES>;
  static std::atomic<bool> configured[64];
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(tiles * p.splits, 1, 1);
  cfg.blockDim = dim3(kDcThreads, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmemBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.splits;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // a programmatic dependent of the previous kernel in the stream (the kernel
  // waits for it before reading anything it may have written)
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, a, b, p);
}

// co-resident clusters of `splits` CTAs of one variant on the current device
template <int ROWS, int STAGES>
cudaError_t clusters_dc(int splits, int* out) {
  using Cfg = DcCfg<ROWS, STAGES>;
  auto kern = kf_qkv_decode_kernel<ROWS, STAGES>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(splits, 1, 1);
  cfg.blockDim = dim3(kDcThreads, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmemBytes;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = splits;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaOccupancyMaxActiveClusters(out, kern, &cfg);
}

}  // namespace

// token boxes of 32 rows (six stages) up to 32 tokens, of 64 rows (five) above
cudaError_t qkv_decode_launch(const CUtensorMap& a, const CUtensorMap& b, const QkvDecodeParams& p, int tiles,
                              cudaStream_t s) {
  if (p.splits < 1 || p.splits > 8 || p.T < 1 || p.T > kQkvDecodeMaxRows) return cudaErrorInvalidValue;
  return p.T <= 32 ? launch_dc<32, 6>(a, b, p, tiles, s) : launch_dc<64, 5>(a, b, p, tiles, s);
}

int qkv_decode_box_rows(int64_t T) { return T <= 32 ? 32 : 64; }

// co-resident clusters of `splits` CTAs for the decode kernel variant that
// serves T tokens (queried once per device, variant and cluster size)
cudaError_t qkv_decode_clusters(int64_t T, int splits, int* out) {
  static std::atomic<int> cache[64][2][9];  // 0: not yet queried
  if (splits < 1 || splits > 8 || T < 1 || T > kQkvDecodeMaxRows) return cudaErrorInvalidValue;
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  const int v = T <= 32 ? 0 : 1;
  if (cache[dev][v][splits] == 0) {
    int nc = 0;
    cudaError_t e = v == 0 ? clusters_dc<32, 6>(splits, &nc) : clusters_dc<64, 5>(splits, &nc);
    if (e != cudaSuccess) return e;
    cache[dev][v][splits] = nc > 0 ? nc : -1;
  }
  const int c = cache[dev][v][splits].load();
  *out = c > 0 ? c : 0;
  return cudaSuccess;
}

}  // namespace kf
