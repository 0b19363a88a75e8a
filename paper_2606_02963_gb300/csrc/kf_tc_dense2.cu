// kf_tc_dense2.cu -- dense CTA-pair instantiations of the tcgen05 fused GEMM:
// a cluster of two CTAs computes a 256-row tile with tcgen05.mma.cta_group::2
// (each CTA stages its own 128 rows of A and half of the B rows), which halves
// the operand bytes each SM streams per MMA and lets a 6-8 stage ring cover the
// TMA round trip.  GroupNorm over 512-column groups also runs on clusters of
// two such pairs, one 256-column half of the group each.
#include <algorithm>

#include "kf_internal.h"
#include "kf_tc_gemm.cuh"

namespace kf {
namespace {

template <int BN, int STAGES, int MODE, class PRE = Interp, class POST = Interp>
cudaError_t launch_pair(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c, const CUtensorMap& r,
                        const TcParams& p, int sub, int grid, cudaStream_t s) {
  using Cfg = TcCfg<BN, STAGES, MODE, false, kClPair, kResTileFor<MODE, false, kClPair, PRE>>;
  auto kern = kf_tc_gemm_kernel<BN, STAGES, MODE, false, kClPair, PRE, POST>;
  static std::atomic<bool> configured[64];
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  if (grid % 2 != 0) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(Cfg::kThr, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmemBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // a programmatic dependent of the previous kernel in the stream: when that
  // one is also a launch of this library (back-to-back calls), this grid's
  // barrier set-up and tensor-memory allocation overlap its tail; the kernel
  // waits for it to complete (griddepcontrol.wait) before any global access.
  // After any other kernel this is an ordinary stream-ordered launch.
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, a, b, c, r, p, static_cast<int32_t>(sub));
}

// Cluster of four (two CTA pairs).  The persistent grid holds as many clusters
// as can be resident at once (a cluster needs four free SMs of one GPC), at
// most one per unit.
template <int BN, int STAGES, int MODE, class PRE = Interp, class POST = Interp>
cudaError_t launch_quad(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c, const TcParams& p,
                        cudaStream_t s) {
  using Cfg = TcCfg<BN, STAGES, MODE, false, kClQuad>;
  auto kern = kf_tc_gemm_kernel<BN, STAGES, MODE, false, kClQuad, PRE, POST>;
  static std::atomic<int> max_clusters[64];  // per device; 0 = not yet queried
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(Cfg::kThr, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmemBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 4;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (max_clusters[dev] == 0) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
    if (e != cudaSuccess) return e;
    int nc = 0;
    cfg.gridDim = dim3(4, 1, 1);
    e = cudaOccupancyMaxActiveClusters(&nc, kern, &cfg);
    if (e != cudaSuccess) return e;
    if (nc < 1) return cudaErrorInvalidConfiguration;
    max_clusters[dev] = nc;
  }
  const int clusters = std::min(p.total_units, max_clusters[dev].load());
  if (clusters < 1) return cudaSuccess;
  cfg.gridDim = dim3(4 * clusters, 1, 1);
  static const CUtensorMap none = {};  // GroupNorm stages no residual tile
  return cudaLaunchKernelEx(&cfg, kern, a, b, c, none, p, static_cast<int32_t>(1));
}

// Couples of CTA pairs (clusters of 2) in one cooperative grid: the pairs of a
// couple wait on each other's statistics, so every CTA must be resident at once,
// which the cooperative launch guarantees (it fails rather than oversubscribe).
template <int BN, int STAGES, int MODE, class PRE = Interp, class POST = Interp>
cudaError_t launch_couple(const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c, const TcParams& p_in,
                          int max_couples, cudaStream_t s) {
  using Cfg = TcCfg<BN, STAGES, MODE, false, kClCouple>;
  auto kern = kf_tc_gemm_kernel<BN, STAGES, MODE, false, kClCouple, PRE, POST>;
  static std::atomic<int> max_pairs[64];  // per device; 0 = not yet queried
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(Cfg::kThr, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmemBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeCooperative;
  attr[1].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (max_pairs[dev] == 0) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
    if (e != cudaSuccess) return e;
    int nc = 0;
    cfg.gridDim = dim3(2, 1, 1);
    e = cudaOccupancyMaxActiveClusters(&nc, kern, &cfg);
    if (e != cudaSuccess) return e;
    if (nc < 2) return cudaErrorInvalidConfiguration;
    max_pairs[dev] = nc;
  }
  const int couples = std::min(std::min(p_in.total_units, max_pairs[dev].load() / 2), max_couples);
  if (couples < 1) return cudaSuccess;
  TcParams p = p_in;
  p.gx_couples = couples;
  cfg.gridDim = dim3(4 * couples, 1, 1);
  cfg.numAttrs = 2;
  static const CUtensorMap none = {};
  return cudaLaunchKernelEx(&cfg, kern, a, b, c, none, p, static_cast<int32_t>(1));
}

}  // namespace

bool tc_couple_has(int mode, int bn) { return mode == kModeGroupNorm && bn == 256; }

cudaError_t tc_couple_launch(int mode, int bn, int sig, const CUtensorMap& a, const CUtensorMap& b,
                             const CUtensorMap& c, const TcParams& p, int max_couples, cudaStream_t s) {
  if (mode != kModeGroupNorm || bn != 256) return cudaErrorInvalidValue;
  if (sig == kSigBiasNormSilu)
    return launch_couple<256, 6, kModeGroupNorm, ProgBias, ProgSilu>(a, b, c, p, max_couples, s);
  return launch_couple<256, 6, kModeGroupNorm>(a, b, c, p, max_couples, s);  // any other chain: interpreter
}

bool tc_dense4_has(int mode, int bn) { return mode == kModeGroupNorm && bn == 256; }

cudaError_t tc_dense4_launch(int mode, int bn, int sig, const CUtensorMap& a, const CUtensorMap& b,
                             const CUtensorMap& c, const TcParams& p, cudaStream_t s) {
  if (mode != kModeGroupNorm || bn != 256) return cudaErrorInvalidValue;
  if (sig == kSigBiasNormSilu) return launch_quad<256, 6, kModeGroupNorm, ProgBias, ProgSilu>(a, b, c, p, s);
  return launch_quad<256, 6, kModeGroupNorm>(a, b, c, p, s);  // any other chain: interpreter
}

// Compiled CTA-pair variants: (mode, BN) -> stages
#define KF_DENSE2_VARIANTS(X) \
  X(kModeStore, 128, 8)       \
  X(kModeStore, 192, 7)       \
  X(kModeStore, 224, 6)       \
  X(kModeStore, 256, 6)       \
  X(kModeLse, 128, 8)         \
  X(kModeLse, 224, 6)         \
  X(kModeLse, 256, 6)         \
  X(kModeGroupNorm, 256, 6)

bool tc_dense2_has(int mode, int bn) {
#define X(M_, B_, S_) \
  if (mode == M_ && bn == B_) return true;
  KF_DENSE2_VARIANTS(X)
#undef X
  return false;
}

// Chain-program variants: (mode, BN, stages, signature, PRE, POST)
// (the residual-tile variants keep the residual in two ring slots and need
// only small per-warp buffers, so their rings are as deep as shared memory allows)
#define KF_DENSE2_PROG_VARIANTS(X)                                              \
  X(kModeStore, 128, 9, kSigBiasGeluScaleRes, ProgGeluChain, Interp)            \
  X(kModeStore, 192, 7, kSigBiasGeluScaleRes, ProgGeluChain, Interp)            \
  X(kModeStore, 224, 7, kSigBiasGeluScaleRes, ProgGeluChain, Interp)            \
  X(kModeStore, 256, 6, kSigBiasGeluScaleRes, ProgGeluChain, Interp)            \
  X(kModeGroupNorm, 256, 6, kSigBiasNormSilu, ProgBias, ProgSilu)               \
  X(kModeLse, 224, 6, kSigScaleLse, ProgScale, Interp)                          \
  X(kModeLse, 256, 6, kSigScaleLse, ProgScale, Interp)

bool tc_dense2_has_prog(int mode, int bn, int sig) {
#define Y(M_, B_, S_, G_, PRE_, POST_) \
  if (mode == M_ && bn == B_ && sig == G_) return true;
  KF_DENSE2_PROG_VARIANTS(Y)
#undef Y
  return false;
}

cudaError_t tc_dense2_launch(int mode, int bn, int sig, const CUtensorMap& a, const CUtensorMap& b, const CUtensorMap& c,
                             const CUtensorMap& r, const TcParams& p, int sub, int grid, cudaStream_t s) {
#define Y(M_, B_, S_, G_, PRE_, POST_) \
  if (mode == M_ && bn == B_ && sig == G_) return launch_pair<B_, S_, M_, PRE_, POST_>(a, b, c, r, p, sub, grid, s);
  KF_DENSE2_PROG_VARIANTS(Y)
#undef Y
#define X(M_, B_, S_) \
  if (mode == M_ && bn == B_) return launch_pair<B_, S_, M_>(a, b, c, r, p, sub, grid, s);
  KF_DENSE2_VARIANTS(X)
#undef X
  return cudaErrorInvalidValue;
}

}  // namespace kf
