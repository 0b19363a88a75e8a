// kf_internal.h -- host-side declarations shared by the library's translation
// units (kernel launchers); not part of the public ABI.
#pragma once
#include <atomic>
#include <cuda.h>
#include <cuda_runtime.h>

#include <utility>

#include "kf_common.cuh"

namespace kf {

// Launch `kern` on `s`; with `pdl` as a programmatic dependent of the previous
// kernel in the stream (one of this library's): it may be scheduled while that
// kernel finishes and waits for it with griddepcontrol.wait before reading its
// results.
template <typename... KArgs, typename... Args>
cudaError_t launch_k(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, bool pdl,
                     Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// Compiled chain programs selectable by signature id (0 = interpreter).
using ProgGeluChain = Prog<KF_OP_BIAS, KF_OP_GELU_TANH, KF_OP_SCALE, KF_OP_RESIDUAL_ADD>;  // bias, GELU, scale, +R
using ProgBias = Prog<KF_OP_BIAS>;
using ProgSilu = Prog<KF_OP_SILU>;
using ProgScale = Prog<KF_OP_SCALE>;
enum ChainSig : int {
  kSigGeneric = 0,
  kSigBiasGeluScaleRes = 1,  // store:      pre = ProgGeluChain (CTA pairs: residual tile)
  kSigBiasNormSilu = 2,      // GroupNorm:  pre = ProgBias, post = ProgSilu
  kSigScaleLse = 3,          // row LSE:    pre = ProgScale, post = none
};

// Tensor-core GEMM launchers.  `bn` selects the tile width among the compiled
// variants; returns cudaErrorInvalidValue for a variant that is not built.
// `cta2` selects the CTA-pair variants (256-row tiles, cluster of 2, grid even).
// `sig` selects a compiled chain program when one is built for (mode, bn,
// cta2), else the interpreter variant runs.
bool tc_dense_has(int mode, int bn, bool cta2);
bool tc_dense2_has(int mode, int bn);
bool tc_dense2_has_prog(int mode, int bn, int sig);  // a compiled chain program for (mode, bn, sig)
// ar: rows of an A ring slot (128, or 64 for groups known to hold at most 64 rows)
bool tc_grouped_has(int mode, int bn, int ar = 128);
// fp32 GEMM + element-wise chain as three tf32 tensor-core products (3xTF32)
struct Tf32Params {
  int32_t M, N, K;
  int32_t tiles_m, tiles_n, num_kb;
  int32_t n_ops;
  DevOp ops[kMaxOps];
  void* Y;
  int64_t ldy;
  int32_t y_dtype;
  int32_t y_vec_ok;
  uint32_t* err;        // the call's error word (its workspace's header, else the device word)
  uint32_t* err_dev;    // the per-device error word
  uint64_t wait_ns;
  uint64_t drain_ns;
};
bool tf32x3_has(int bn);
// QKV projection tail for <= 128 tokens: K split over the CTAs of a cluster,
// partials reduced through distributed shared memory
struct QkvDecodeParams {
  int32_t T, N, K, num_kb;
  int32_t splits;        // CTAs per cluster = K splits of a 256-column tile
  int32_t ab_f16;
  const void* bias;      // [N] or null
  int32_t bias_dtype;
  const float* cos_t;
  const float* sin_t;
  const int32_t* positions;
  const int32_t* cache_rows;
  int32_t max_pos, rows;
  int32_t rope_d, q_cols, rot_cols;
  void* q_out;
  int64_t ldq;
  void* k_cache;
  void* v_cache;
  int64_t ld_cache;
  int32_t out_dtype;
  uint32_t* err;
  uint64_t wait_ns;
  uint64_t drain_ns;
};
// few-token QKV tail: at most this many tokens; A boxes of qkv_decode_box_rows(T) rows
constexpr int kQkvDecodeMaxRows = 64;
cudaError_t qkv_decode_launch(const CUtensorMap& a, const CUtensorMap& b, const QkvDecodeParams& p, int tiles,
                              cudaStream_t s);
int qkv_decode_box_rows(int64_t T);
cudaError_t qkv_decode_clusters(int64_t T, int splits, int* out);
cudaError_t tf32x3_launch(int bn, const CUtensorMap& a, const CUtensorMap& b, const Tf32Params& p, int grid,
                          cudaStream_t s);
// QKV projection tail (kModeRope): single CTAs or CTA pairs; no output map
bool tc_rope_has(int bn, bool cta2);
cudaError_t tc_rope_launch(int bn, bool cta2, const CUtensorMap& a, const CUtensorMap& b, const TcParams& p, int grid,
                           cudaStream_t s);
// `c` is the output map of the TMA stores, `r` the residual map of the
// residual-tile variants (unused by the others).
cudaError_t tc_dense_launch(int mode, int bn, bool cta2, int sig, const CUtensorMap& a, const CUtensorMap& b,
                            const CUtensorMap& c, const CUtensorMap& r, const TcParams& p, int sub_tiles, int grid,
                            cudaStream_t s);
cudaError_t tc_dense2_launch(int mode, int bn, int sig, const CUtensorMap& a, const CUtensorMap& b,
                             const CUtensorMap& c, const CUtensorMap& r, const TcParams& p, int sub_tiles, int grid,
                             cudaStream_t s);
cudaError_t tc_grouped_launch(int mode, int bn, int ar, const CUtensorMap& a, const CUtensorMap& b,
                              const CUtensorMap& c, const TcParams& p, int grid, cudaStream_t s, bool pdl);
// GroupNorm over 512-column groups on clusters of two CTA pairs (one 256-column
// half of the group per pair); units = 256-row x 512-column blocks, the grid is
// sized inside from the number of co-resident clusters.
// GroupNorm over 512-column groups on couples of CTA pairs (cooperative grid):
// the same split as the clusters of four, with the statistics exchanged through
// global memory (p.gx_data / p.gx_flag, room for `max_couples` couples), so all
// co-resident pairs work.
bool tc_couple_has(int mode, int bn);
cudaError_t tc_couple_launch(int mode, int bn, int sig, const CUtensorMap& a, const CUtensorMap& b,
                             const CUtensorMap& c, const TcParams& p, int max_couples, cudaStream_t s);
bool tc_dense4_has(int mode, int bn);
cudaError_t tc_dense4_launch(int mode, int bn, int sig, const CUtensorMap& a, const CUtensorMap& b,
                             const CUtensorMap& c, const TcParams& p, cudaStream_t s);

// SIMT kernels.
struct SimtParams {
  const float* X;
  const float* W;
  float* Y;
  int64_t ldx, ldw, ldy;
  int32_t M, N, K;
  int32_t n_ops;
  DevOp ops[kMaxOps];
};
cudaError_t simt_gemm_f32_launch(const SimtParams& p, cudaStream_t s);

struct LseCombineParams {
  const float2* part;
  int32_t M;
  int32_t parts;
  void* out;
  int32_t out_dtype;
  int32_t red_sum;      // partials are row sums (.y): add them instead of the (max, sum exp) merge
  int32_t n_post;
  DevOp post[kMaxOps];
};
cudaError_t lse_combine_launch(const LseCombineParams& p, cudaStream_t s, bool pdl);

cudaError_t route_topk_launch(const float* logits, int32_t T, int32_t E, int32_t k, int32_t* ids, float* w,
                              cudaStream_t s);
cudaError_t route_sort_launch(const int32_t* ids, const float* w, int32_t T, int32_t E, int32_t k,
                              int32_t* offsets, int32_t* sorted_token, float* sorted_w, int32_t* pair_pos,
                              cudaStream_t s, bool pdl);
// Multi-block stable sort (same order), for many pairs: `counts` is scratch of
// route_sort_mb_blocks(T k) x E int32
cudaError_t route_sort_mb_launch(const int32_t* ids, const float* w, int32_t T, int32_t E, int32_t k,
                                 int32_t* offsets, int32_t* sorted_token, float* sorted_w, int32_t* pair_pos,
                                 int32_t* counts, cudaStream_t s, bool pdl);
int32_t route_sort_mb_blocks(int32_t P);
cudaError_t moe_finalize_launch(const float* Yp, const int32_t* pair_pos, int64_t T, int32_t k, int64_t H, void* Y,
                                cudaStream_t s, bool pdl);
// MoE block tail: R_out = bf16(R + y), Y = bf16(rmsnorm(R_out) * gamma) per token;
// y from the fp32 accumulator `yacc`, or (yacc == nullptr) the slot-order sum of
// the per-row outputs `yp` through `pair_pos`.  H % 4 == 0, H <= 8192.
constexpr int64_t kAddRmsNormMaxH = 8192;
cudaError_t moe_add_rmsnorm_launch(const float* yacc, const float* yp, const int32_t* pair_pos, int32_t k, int64_t T,
                                   int64_t H, const void* R, const void* gamma, float eps, void* R_out, void* Y,
                                   cudaStream_t s, bool pdl);
cudaError_t gather_rows_launch(const void* A, int64_t lda, int64_t a_rows, const int32_t* idx, int64_t rows,
                               int64_t K, void* out, uint32_t* err, uint32_t* err_dev, cudaStream_t s, bool pdl);
cudaError_t cvt_f32_bf16_launch(const float* in, void* out, int64_t n, cudaStream_t s, bool pdl);

}  // namespace kf
