// kf_tc_grouped.cu -- grouped (per-expert) instantiations of the tcgen05 fused
// GEMM: SwiGLU gate/up, routing-weight scale + scatter-add down, plain store.
#include "kf_internal.h"
#include "kf_tc_gemm.cuh"

namespace kf {
namespace {

template <int BN, int STAGES, int MODE>
cudaError_t launch_one(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c, const TcParams& p, int grid, cudaStream_t s,
                       bool pdl) {
  using Cfg = TcCfg<BN, STAGES, MODE, true, kClOne>;
  auto kern = kf_tc_gemm_kernel<BN, STAGES, MODE, true, kClOne>;
  static std::atomic<bool> configured[64];  // the attribute is per device
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  static const CUtensorMap none = {};  // grouped variants stage no residual tile
  return launch_k(kern, dim3(grid), dim3(Cfg::kThr), Cfg::kSmemBytes, s, pdl, a, b, c, none, p, static_cast<int32_t>(1));
}

}  // namespace

#define KF_GROUPED_VARIANTS(X) \
  X(kModeSwiglu, 128, 6)       \
  X(kModeSwiglu, 192, 5)       \
  X(kModeSwiglu, 256, 4)       \
  X(kModeScatter, 128, 6)      \
  X(kModeScatter, 192, 5)      \
  X(kModeScatter, 256, 4)      \
  X(kModeStore, 128, 6)        \
  X(kModeStore, 192, 4)        \
  X(kModeStore, 256, 4)

bool tc_grouped_has(int mode, int bn) {
#define X(M_, B_, S_) \
  if (mode == M_ && bn == B_) return true;
  KF_GROUPED_VARIANTS(X)
#undef X
  return false;
}

cudaError_t tc_grouped_launch(int mode, int bn, const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c, const TcParams& p,
                              int grid, cudaStream_t s, bool pdl) {
#define X(M_, B_, S_) \
  if (mode == M_ && bn == B_) return launch_one<B_, S_, M_>(a, b, c, p, grid, s, pdl);
  KF_GROUPED_VARIANTS(X)
#undef X
  return cudaErrorInvalidValue;
}

}  // namespace kf
