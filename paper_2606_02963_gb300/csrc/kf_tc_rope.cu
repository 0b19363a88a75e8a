// kf_tc_rope.cu -- instantiations of the tcgen05 fused GEMM for the QKV
// projection tail (bias, rotary embedding of query / key heads, key / value
// cache rows; the gpt-oss decode kernel "Bias + RoPE + KV update", Sec. IV-A).
// Tiles hold whole heads, so each rotation pair (column i and i + d/2 of a
// head) sits in one thread's row of the accumulator.  Decode-sized problems
// (one 128-row tile) take single CTAs with tiles narrow enough to spread the
// weight stream over the SMs; larger ones take CTA pairs (256-row tiles).
#include <cstring>

#include "kf_internal.h"
#include "kf_tc_gemm.cuh"

namespace kf {
namespace {

template <int BN, int STAGES, int CL>
cudaError_t launch_rope(const CUtensorMap& a, const CUtensorMap& b, const TcParams& p, int grid, cudaStream_t s) {
  using Cfg = TcCfg<BN, STAGES, kModeRope, false, CL>;
  auto kern = kf_tc_gemm_kernel<BN, STAGES, kModeRope, false, CL>;
  static std::atomic<bool> configured[64];  // the attribute is per device
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  if (CL == kClPair && grid % 2 != 0) return cudaErrorInvalidValue;
  CUtensorMap unused;
  std::memset(&unused, 0, sizeof(unused));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(Cfg::kThr, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmemBytes;
  cfg.stream = s;
  // a programmatic dependent of the previous kernel in the stream (the kernel
  // waits for it before reading anything it may have written)
  cudaLaunchAttribute attr[2];
  int na = 0;
  attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[na].val.programmaticStreamSerializationAllowed = 1;
  ++na;
  if (CL == kClPair) {
    attr[na].id = cudaLaunchAttributeClusterDimension;
    attr[na].val.clusterDim.x = 2;
    attr[na].val.clusterDim.y = 1;
    attr[na].val.clusterDim.z = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, kern, a, b, unused, unused, p, static_cast<int32_t>(1));
}

}  // namespace

// Compiled variants: (BN, stages, cluster layout)
#define KF_ROPE_VARIANTS(X) \
  X(64, 8, kClOne)          \
  X(128, 6, kClOne)         \
  X(256, 4, kClOne)         \
  X(128, 8, kClPair)        \
  X(256, 6, kClPair)

bool tc_rope_has(int bn, bool cta2) {
#define X(B_, S_, C_) \
  if (bn == B_ && cta2 == (C_ == kClPair)) return true;
  KF_ROPE_VARIANTS(X)
#undef X
  return false;
}

cudaError_t tc_rope_launch(int bn, bool cta2, const CUtensorMap& a, const CUtensorMap& b, const TcParams& p, int grid,
                           cudaStream_t s) {
#define X(B_, S_, C_) \
  if (bn == B_ && cta2 == (C_ == kClPair)) return launch_rope<B_, S_, C_>(a, b, p, grid, s);
  KF_ROPE_VARIANTS(X)
#undef X
  return cudaErrorInvalidValue;
}

}  // namespace kf
