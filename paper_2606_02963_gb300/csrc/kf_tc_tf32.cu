// kf_tc_tf32.cu -- fp32 GEMM + element-wise tail on the tensor cores as three
// tf32 products (3xTF32).  Each fp32 operand x is split into a tf32 high part
// h = rna_tf32(x) and the remainder l = rna_tf32(x - h) (x - h is exact in
// fp32); X W^T is then Xh Wh^T + Xh Wl^T + Xl Wh^T in fp32,
// dropping only Xl Wl^T (relative size ~2^-22), so the result stays within fp32
// accuracy while the products run on tcgen05 (kind::tf32) instead of FFMA.
//
// Warp roles (one CTA per SM, persistent over 128 x BN output tiles):
//   warp 0      TMA producer: fp32 A [128 x 32] and B [BN x 32] boxes (128-byte
//               rows, 128-byte swizzle) into the raw buffers of a ring stage
//   warp 1      MMA issuer: per 32-wide k-block, 4 k-steps of 8 x 3 products
//   warps 2-5   splitters: raw -> high part in place, low part into the
//               stage's second buffer (same swizzled offsets), then release
//               the stage to the MMA warp
//   warps 6-9   epilogue: one per TMEM lane quadrant; tcgen05.ld 32 columns,
//               the op chain, fp32 / bf16 / fp16 stores
// Two TMEM accumulators let a tile's epilogue overlap the next tile's
// mainloop.  Every wait is bounded (error word, no trap).
#include "kf_internal.h"

namespace kf {
namespace {

constexpr int kTfBM = 128;
constexpr int kTfBK = 32;                     // fp32 elements per 128-byte row
constexpr int kTfThreads = 320;
constexpr int kTfRowBytes = kTfBK * 4;        // 128

__host__ __device__ constexpr uint32_t idesc_tf32_f32(uint32_t M, uint32_t N) {
  // D fp32 (bits 4-5 = 1), A and B tf32 (bits 7-9 = 2, bits 10-12 = 2), both
  // K-major, N >> 3 at bits 17-22, M >> 4 at bits 24-28
  return (1u << 4) | (2u << 7) | (2u << 10) | ((N >> 3) << 17) | ((M >> 4) << 24);
}

__device__ __forceinline__ void tc_mma_tf32(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ float rna_tf32(float x) {
  uint32_t r;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(r) : "f"(x));
  return __uint_as_float(r);
}

template <int BN, int STAGES>
struct Tf32Cfg {
  static constexpr int kABytes = kTfBM * kTfRowBytes;  // 16 KB
  static constexpr int kBBytes = BN * kTfRowBytes;
  // stage: A high | A low | B high | B low (each 1 KB aligned)
  static constexpr int kStageBytes = 2 * kABytes + 2 * kBBytes;
  static constexpr uint32_t kTxBytes = kABytes + kBBytes;  // the raw boxes
  static constexpr int kAccStride = BN;                     // TMEM columns per accumulator
  static constexpr int kTmemCols = 2 * BN;
  static constexpr int kBarBytes = 8 * (3 * STAGES + 5);
  static constexpr int kSmemBytes = 1024 + STAGES * kStageBytes + kBarBytes + 64;
  static constexpr uint32_t kIdesc = idesc_tf32_f32(kTfBM, BN);
  static_assert(BN % 32 == 0 && BN >= 64 && BN <= 256 && (BN & (BN - 1)) == 0, "BN");
  static_assert(kSmemBytes <= 232448, "shared memory");
};

template <int BN, int STAGES>
__global__ void __launch_bounds__(kTfThreads, 1)
    kf_tf32x3_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                          const __grid_constant__ Tf32Params p) {
  using Cfg = Tf32Cfg<BN, STAGES>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + STAGES * Cfg::kStageBytes);
  uint64_t* full = bars;                 // raw boxes landed (TMA)
  uint64_t* split = bars + STAGES;       // high / low parts written (4 splitter warps)
  uint64_t* empty = bars + 2 * STAGES;   // MMAs done with the stage
  uint64_t* accf = bars + 3 * STAGES;    // accumulator ready (2)
  uint64_t* acce = bars + 3 * STAGES + 2;  // accumulator drained (2)
  uint64_t* drain = bars + 3 * STAGES + 4;  // MMA abort: every issued MMA has completed
  uint32_t* misc = reinterpret_cast<uint32_t*>(bars + 3 * STAGES + 5);
  uint32_t* tmem_slot = misc;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 1);
  volatile int* zero_flag = reinterpret_cast<volatile int*>(misc + 2);
  auto a_hi = [&](int s) { return sm + s * Cfg::kStageBytes; };
  auto a_lo = [&](int s) { return sm + s * Cfg::kStageBytes + Cfg::kABytes; };
  auto b_hi = [&](int s) { return sm + s * Cfg::kStageBytes + 2 * Cfg::kABytes; };
  auto b_lo = [&](int s) { return sm + s * Cfg::kStageBytes + 2 * Cfg::kABytes + Cfg::kBBytes; };

  if (blockDim.x != kTfThreads || gridDim.y != 1 || gridDim.z != 1) {
    if (threadIdx.x == 0) raise_err(p.err, p.err_dev, kErrLaunchShape);
    return;
  }
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&split[s], 4);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&accf[a], 1);
      mbar_init(&acce[a], 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    *zero_flag = 0;
    fence_mbarrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    __syncwarp();
    tmem_alloc(tmem_slot, Cfg::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncwarp();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int32_t total = p.tiles_m * p.tiles_n;
  const int32_t unit0 = static_cast<int32_t>(blockIdx.x), step = static_cast<int32_t>(gridDim.x);

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      int32_t it = 0;
      bool ok = true;
      for (int32_t u = unit0; ok && u < total; u += step) {
        const int32_t m0 = (u % p.tiles_m) * kTfBM, n0 = (u / p.tiles_m) * BN;
        for (int32_t kb = 0; kb < p.num_kb; ++kb, ++it) {
          const int st = it % STAGES;
          if (!mbar_wait(&empty[st], ((it / STAGES) & 1) ^ 1, abort_flag, p.wait_ns)) {
            *abort_flag = 1;
            raise_err(p.err, p.err_dev, kErrWaitProducer);
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[st], Cfg::kTxBytes);
          tma_load_2d(a_hi(st), &tmA, &full[st], kb * kTfBK, m0);
          tma_load_2d(b_hi(st), &tmB, &full[st], kb * kTfBK, n0);
        }
      }
      if (!ok)  // copies still in flight land before the CTA exits
        for (int32_t j = (it > STAGES ? it - STAGES : 0); j < it; ++j)
          mbar_wait(&full[j % STAGES], (j / STAGES) & 1, zero_flag, p.drain_ns);
    }
  } else if (warp == 1) {
    // --------------------------------------------------------------------- MMA
    if (lane == 0) {
      int32_t it = 0, tl = 0;
      bool ok = true;
      for (int32_t u = unit0; ok && u < total; u += step, ++tl) {
        const int acc = tl & 1;
        if (!mbar_wait(&acce[acc], ((tl >> 1) & 1) ^ 1, abort_flag, p.wait_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + acc * Cfg::kAccStride;
        for (int32_t kb = 0; kb < p.num_kb; ++kb, ++it) {
          const int st = it % STAGES;
          if (!mbar_wait(&split[st], (it / STAGES) & 1, abort_flag, p.wait_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t ah = smem_u32(a_hi(st)), al = smem_u32(a_lo(st));
          const uint32_t bh = smem_u32(b_hi(st)), bl = smem_u32(b_lo(st));
#pragma unroll
          for (int kk = 0; kk < kTfBK / 8; ++kk) {
            // K = 8 tf32 per instruction: 32 bytes along the swizzled row
            const uint64_t dah = desc_sw128_kmajor(ah + kk * 32), dal = desc_sw128_kmajor(al + kk * 32);
            const uint64_t dbh = desc_sw128_kmajor(bh + kk * 32), dbl = desc_sw128_kmajor(bl + kk * 32);
            tc_mma_tf32(d, dal, dbh, Cfg::kIdesc, (kb | kk) != 0 ? 1u : 0u);  // small terms first
            tc_mma_tf32(d, dah, dbl, Cfg::kIdesc, 1u);
            tc_mma_tf32(d, dah, dbh, Cfg::kIdesc, 1u);
          }
          tc_commit(&empty[st]);
        }
        if (!ok) break;
        tc_commit(&accf[acc]);
      }
      if (!ok) {
        *abort_flag = 1;
        raise_err(p.err, p.err_dev, kErrWaitMma);
        tc_commit(drain);  // arrives once every MMA issued so far has completed
        mbar_wait(drain, 0, zero_flag, p.drain_ns);
      }
    }
  } else if (warp < 6) {
    // --------------------------------------------------------------- splitters
    const int t = threadIdx.x - 64;  // 0..127
    int32_t it = 0;
    bool ok = true;
    for (int32_t u = unit0; ok && u < total; u += step) {
      for (int32_t kb = 0; kb < p.num_kb; ++kb, ++it) {
        const int st = it % STAGES;
        bool w = mbar_wait(&full[st], (it / STAGES) & 1, abort_flag, p.wait_ns);
        w = __all_sync(0xffffffffu, w);
        if (!w) {
          *abort_flag = 1;
          if (lane == 0) raise_err(p.err, p.err_dev, kErrWaitEpilogue);
          ok = false;
          break;
        }
        // 16-byte units of the A and B boxes (positions are the same in the
        // high and low buffers, so the swizzle needs no decoding)
        float4* ha = reinterpret_cast<float4*>(a_hi(st));
        float4* la = reinterpret_cast<float4*>(a_lo(st));
        for (int i = t; i < Cfg::kABytes / 16; i += 128) {
          const float4 x = ha[i];
          float4 h, l;
          h.x = rna_tf32(x.x); h.y = rna_tf32(x.y); h.z = rna_tf32(x.z); h.w = rna_tf32(x.w);
          l.x = rna_tf32(x.x - h.x); l.y = rna_tf32(x.y - h.y);
          l.z = rna_tf32(x.z - h.z); l.w = rna_tf32(x.w - h.w);
          ha[i] = h;
          la[i] = l;
        }
        float4* hb = reinterpret_cast<float4*>(b_hi(st));
        float4* lb = reinterpret_cast<float4*>(b_lo(st));
        for (int i = t; i < Cfg::kBBytes / 16; i += 128) {
          const float4 x = hb[i];
          float4 h, l;
          h.x = rna_tf32(x.x); h.y = rna_tf32(x.y); h.z = rna_tf32(x.z); h.w = rna_tf32(x.w);
          l.x = rna_tf32(x.x - h.x); l.y = rna_tf32(x.y - h.y);
          l.z = rna_tf32(x.z - h.z); l.w = rna_tf32(x.w - h.w);
          hb[i] = h;
          lb[i] = l;
        }
        fence_proxy_async_smem();  // generic-proxy writes before the tensor core reads them
        __syncwarp();
        if (lane == 0) mbar_arrive(&split[st]);
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue
    const int q = warp & 3;  // TMEM lane quadrant this warp may access
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    int32_t tl = 0;
    for (int32_t u = unit0; u < total; u += step, ++tl) {
      const int32_t m0 = (u % p.tiles_m) * kTfBM, n0 = (u / p.tiles_m) * BN;
      const int acc = tl & 1;
      bool w = mbar_wait(&accf[acc], (tl >> 1) & 1, abort_flag, p.wait_ns);
      w = __all_sync(0xffffffffu, w);
      if (!w) {
        *abort_flag = 1;
        if (lane == 0) raise_err(p.err, p.err_dev, kErrWaitEpilogue);
        break;
      }
      tc_fence_after();
      const int32_t grow = m0 + q * 32 + lane;
      const bool row_ok = grow < p.M;
      for (int c = 0; c < BN / 32; ++c) {
        const int32_t col0 = n0 + c * 32;
        const int nvalid = min(32, p.N - col0);
        if (nvalid <= 0) break;
        float v[32];
        tmem_ld32(tmem + lane_off + acc * Cfg::kAccStride + c * 32, v);
        run_chain<Interp>(false, p.ops, p.n_ops, v, grow, col0, nvalid, row_ok);
        if (row_ok) st32(p.Y, p.y_dtype, static_cast<int64_t>(grow) * p.ldy + col0, nvalid, p.y_vec_ok != 0, v);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acce[acc]);
    }
  }

  // ---------------------------------------------------------------- teardown
  tc_fence_before();
  __syncwarp();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, Cfg::kTmemCols);
  }
}

template <int BN, int STAGES>
cudaError_t launch_tf32(const CUtensorMap& a, const CUtensorMap& b, const Tf32Params& p, int grid, cudaStream_t s) {
  using Cfg = Tf32Cfg<BN, STAGES>;
  auto kern = kf_tf32x3_gemm_kernel<BN, STAGES>;
  static std::atomic<bool> configured[64];
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  kern<<<grid, kTfThreads, Cfg::kSmemBytes, s>>>(a, b, p);
  return cudaGetLastError();
}

}  // namespace

// Compiled variants: BN -> stages (a stage holds the raw / high and low copies
// of both operands: 64 KB at BN = 128, 96 KB at BN = 256)
bool tf32x3_has(int bn) { return bn == 128 || bn == 256; }

cudaError_t tf32x3_launch(int bn, const CUtensorMap& a, const CUtensorMap& b, const Tf32Params& p, int grid,
                          cudaStream_t s) {
  if (bn == 128) return launch_tf32<128, 3>(a, b, p, grid, s);
  if (bn == 256) return launch_tf32<256, 2>(a, b, p, grid, s);
  return cudaErrorInvalidValue;
}

}  // namespace kf
