// kf_tc_dense.cu -- dense single-CTA instantiations of the tcgen05 fused GEMM
// (128-row tiles): element-wise chains (store), row log-sum-exp partials,
// GroupNorm.  Used when M <= 128; larger problems take the CTA-pair variants
// in kf_tc_dense2.cu.
#include "kf_internal.h"
#include "kf_tc_gemm.cuh"

namespace kf {
namespace {

template <int BN, int STAGES, int MODE>
cudaError_t launch_one(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c, const CUtensorMap& r,
                       const TcParams& p, int sub, int grid, cudaStream_t s) {
  using Cfg = TcCfg<BN, STAGES, MODE, false, kClOne>;
  auto kern = kf_tc_gemm_kernel<BN, STAGES, MODE, false, kClOne>;
  static std::atomic<bool> configured[64];  // the attribute is per device
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  // a programmatic dependent of the previous kernel in the stream (see the
  // CTA-pair launcher): set-up overlaps a preceding call's tail
  return launch_k(kern, dim3(grid), dim3(Cfg::kThr), Cfg::kSmemBytes, s, true, a, b, c, r, p, static_cast<int32_t>(sub));
}

}  // namespace

// Compiled variants: (mode, BN) -> stages
#define KF_DENSE_VARIANTS(X) \
  X(kModeStore, 128, 6)      \
  X(kModeStore, 192, 4)      \
  X(kModeStore, 224, 4)      \
  X(kModeStore, 256, 4)      \
  X(kModeLse, 128, 6)        \
  X(kModeLse, 224, 4)        \
  X(kModeLse, 256, 4)        \
  X(kModeGroupNorm, 256, 4)

bool tc_dense_has(int mode, int bn, bool cta2) {
  if (cta2) return tc_dense2_has(mode, bn);
#define X(M_, B_, S_) \
  if (mode == M_ && bn == B_) return true;
  KF_DENSE_VARIANTS(X)
#undef X
  return false;
}

cudaError_t tc_dense_launch(int mode, int bn, bool cta2, int sig, const CUtensorMap& a, const CUtensorMap& b,
                            const CUtensorMap& c, const CUtensorMap& r, const TcParams& p, int sub, int grid,
                            cudaStream_t s) {
  if (cta2) return tc_dense2_launch(mode, bn, sig, a, b, c, r, p, sub, grid, s);
#define X(M_, B_, S_) \
  if (mode == M_ && bn == B_) return launch_one<B_, S_, M_>(a, b, c, r, p, sub, grid, s);
  KF_DENSE_VARIANTS(X)
#undef X
  return cudaErrorInvalidValue;
}

}  // namespace kf
