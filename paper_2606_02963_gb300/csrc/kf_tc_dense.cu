// kf_tc_dense.cu -- dense instantiations of the tcgen05 fused GEMM: element-wise
// chains (store), row log-sum-exp partials, GroupNorm.
#include "kf_internal.h"
#include "kf_tc_gemm.cuh"

namespace kf {
namespace {

template <int BN, int STAGES, int MODE>
cudaError_t launch_one(const CUtensorMap& a, const CUtensorMap& b, const TcParams& p, int sub, int grid,
                       cudaStream_t s) {
  using Cfg = TcCfg<BN, STAGES, MODE, false>;
  auto kern = kf_tc_gemm_kernel<BN, STAGES, MODE, false>;
  static int configured_dev = -1;  // attribute is per device; re-set when the device changes
  int dev = 0;
  cudaGetDevice(&dev);
  if (configured_dev != dev) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
    if (e != cudaSuccess) return e;
    configured_dev = dev;
  }
  kern<<<grid, kThreads, Cfg::kSmemBytes, s>>>(a, b, p, sub);
  return cudaGetLastError();
}

template <int BN, int STAGES, int MODE>
int smem_one() {
  return TcCfg<BN, STAGES, MODE, false>::kSmemBytes;
}

}  // namespace

// Compiled variants: (mode, BN) -> stages
#define KF_DENSE_VARIANTS(X)      \
  X(kModeStore, 128, 6)           \
  X(kModeStore, 192, 5)           \
  X(kModeStore, 224, 4)           \
  X(kModeStore, 256, 4)           \
  X(kModeLse, 128, 6)             \
  X(kModeLse, 224, 4)             \
  X(kModeLse, 256, 4)             \
  X(kModeGroupNorm, 256, 4)

bool tc_dense_has(int mode, int bn) {
#define X(M_, B_, S_) \
  if (mode == M_ && bn == B_) return true;
  KF_DENSE_VARIANTS(X)
#undef X
  return false;
}

int tc_dense_smem(int mode, int bn) {
#define X(M_, B_, S_) \
  if (mode == M_ && bn == B_) return smem_one<B_, S_, M_>();
  KF_DENSE_VARIANTS(X)
#undef X
  return 0;
}

cudaError_t tc_dense_launch(int mode, int bn, const CUtensorMap& a, const CUtensorMap& b, const TcParams& p,
                            int sub, int grid, cudaStream_t s) {
#define X(M_, B_, S_) \
  if (mode == M_ && bn == B_) return launch_one<B_, S_, M_>(a, b, p, sub, grid, s);
  KF_DENSE_VARIANTS(X)
#undef X
  return cudaErrorInvalidValue;
}

}  // namespace kf
