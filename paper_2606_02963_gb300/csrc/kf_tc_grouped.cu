// kf_tc_grouped.cu -- grouped (per-expert) instantiations of the tcgen05 fused
// GEMM: SwiGLU gate/up, routing-weight scale + scatter-add down, plain store.
#include "kf_internal.h"
#include "kf_tc_gemm.cuh"

namespace kf {
namespace {

template <int BN, int STAGES, int MODE, int AR>
cudaError_t launch_one(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c, const TcParams& p, int grid, cudaStream_t s,
                       bool pdl) {
  using Cfg = TcCfg<BN, STAGES, MODE, true, kClOne, false, AR>;
  auto kern = kf_tc_gemm_kernel<BN, STAGES, MODE, true, kClOne, Interp, Interp, AR>;
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

// (mode, BN, stages, rows of an A slot).  The 64-row variants serve groups of
// at most 64 rows (the MoE at decode): the shared memory an A slot no longer
// needs holds more stages, i.e. more weight bytes in flight.
#define KF_GROUPED_VARIANTS(X)  \
  X(kModeSwiglu, 128, 6, 128)   \
  X(kModeSwiglu, 192, 5, 128)   \
  X(kModeSwiglu, 256, 4, 128)   \
  X(kModeSwiglu, 256, 5, 64)    \
  X(kModeScatter, 128, 6, 128)  \
  X(kModeScatter, 192, 5, 128)  \
  X(kModeScatter, 256, 4, 128)  \
  X(kModeScatter, 128, 8, 64)   \
  X(kModeStore, 128, 6, 128)    \
  X(kModeStore, 192, 4, 128)    \
  X(kModeStore, 256, 4, 128)    \
  X(kModeStore, 128, 8, 64)

bool tc_grouped_has(int mode, int bn, int ar) {
#define X(M_, B_, S_, R_) \
  if (mode == M_ && bn == B_ && ar == R_) return true;
  KF_GROUPED_VARIANTS(X)
#undef X
  return false;
}

cudaError_t tc_grouped_launch(int mode, int bn, int ar, const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c,
                              const TcParams& p, int grid, cudaStream_t s, bool pdl) {
#define X(M_, B_, S_, R_) \
  if (mode == M_ && bn == B_ && ar == R_) return launch_one<B_, S_, M_, R_>(a, b, c, p, grid, s, pdl);
  KF_GROUPED_VARIANTS(X)
#undef X
  return cudaErrorInvalidValue;
}

}  // namespace kf
