/*
 * kf.h -- C ABI of the GB300 (sm_103a) fused GEMM + tail-op library.
 *
 * The library computes the work that the KForge paper's generated kernels
 * speed up (arXiv 2606.02963):
 *   - a dense GEMM whose post-GEMM op chain (bias, activation, scale, residual,
 *     row log-sum-exp, GroupNorm) runs in the GEMM's epilogue, reading the
 *     matmul result once and writing once ("layer-wise fusion", Sec. IV-B),
 *     with 16-bit operands and fp32 accumulation / post-processing
 *     ("mixed-precision execution", Sec. IV-B);
 *   - the routed MoE expert FFN of the gpt-oss decode path (Sec. IV-A): top-k
 *     routing, a grouped gate/up GEMM with a SwiGLU epilogue, and a grouped down
 *     GEMM whose epilogue applies the routing weight and scatter-adds rows into
 *     the output (the "MoE finalize" step of Table 1).
 *
 * Conventions shared by every call
 *   - Matrices are row-major.  X is [M x K], W is [N x K] (the nn.Linear layout,
 *     so both GEMM operands are K-major) and Y = chain(X W^T) is [M x N].
 *   - Every pointer except host-side descriptors (kf_epilogue and its op array)
 *     is a DEVICE pointer on the current CUDA device.  The caller owns all of
 *     them, including the workspace; query its size with the *_workspace call.
 *     The library allocates and frees nothing and keeps no pointer after return.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  Every call is
 *     asynchronous on it; results are valid once the stream reaches that point.
 *   - Arguments are checked on the host before anything is launched; a bad
 *     argument returns a status and launches nothing.  A failed launch returns
 *     KF_ERR_CUDA.  No call aborts, exits or throws.
 *   - Device-side waits are bounded.  A kernel whose wait runs out (or that finds
 *     bad device-resident indices) records error bits and returns early.  The
 *     bits go to the error word of the call's workspace when it was given one
 *     (the first 32-bit word of the workspace's KF_WORKSPACE_HEADER_BYTES
 *     header; kf_check_device_error reads and clears it), and always to a
 *     per-device error word (kf_get_device_error reads and clears that one; it
 *     collects the errors of every call on the device, so a check there by one
 *     thread can consume another thread's error).
 *   - Workspaces: a call that takes a workspace and is given one (16-byte
 *     aligned, at least KF_WORKSPACE_HEADER_BYTES) uses its first
 *     KF_WORKSPACE_HEADER_BYTES bytes as the header and the rest as scratch.
 *     The *_workspace size queries include the header.  The header must be zero
 *     before the workspace's first use (kf_workspace_init, or a zero-filled
 *     allocation); calls only OR bits into it, kf_check_device_error clears it.
 *   - Calls on distinct streams may run concurrently if they use distinct
 *     workspaces and outputs; each then checks its own errors with
 *     kf_check_device_error on its own workspace.
 */
#ifndef KF_H_
#define KF_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum kf_status {
  KF_OK = 0,
  KF_ERR_INVALID_ARG = 1,    /* null pointer, bad size, bad op chain            */
  KF_ERR_UNSUPPORTED = 2,    /* dtype combination or chain this build lacks    */
  KF_ERR_MISALIGNED = 3,     /* TMA needs 16-byte aligned bases and row strides */
  KF_ERR_WORKSPACE = 4,      /* workspace missing or smaller than required     */
  KF_ERR_CUDA = 5,           /* a CUDA runtime/driver call or launch failed    */
  KF_ERR_DEVICE_TIMEOUT = 6, /* a device-side bounded wait ran out             */
  KF_ERR_DEVICE_BOUNDS = 7   /* device-resident indices/offsets out of range   */
} kf_status;

typedef enum kf_dtype { KF_F32 = 0, KF_BF16 = 1, KF_I32 = 2, KF_F16 = 3 } kf_dtype;

/* Bytes at the start of every workspace reserved for its header (error word). */
#define KF_WORKSPACE_HEADER_BYTES 256

/* Tail ops, applied in list order to the fp32 accumulator (Sec. IV-B: the
 * post-GEMM sequence of operations, fused into one kernel). */
typedef enum kf_op_kind {
  KF_OP_BIAS = 0,          /* v += p0[col]                           (p0: [N])        */
  KF_OP_SCALE = 1,         /* v *= scalar                                              */
  KF_OP_RELU = 2,          /* max(v, 0)                                                */
  KF_OP_GELU_TANH = 3,     /* 0.5 v (1 + tanh(sqrt(2/pi)(v + 0.044715 v^3)))           */
  KF_OP_SILU = 4,          /* v * sigmoid(v)  (Swish)                                  */
  KF_OP_SIGMOID = 5,       /* 1 / (1 + exp(-v))                                        */
  KF_OP_RESIDUAL_ADD = 6,  /* v += p0[row * ld + col]               (p0: [M x ld])    */
  KF_OP_ROW_LOGSUMEXP = 7, /* row -> max_j v_j + log sum_j exp(v_j - max); Y is [M].
                              Only scalar ops (SCALE, RELU, GELU_TANH, SILU, SIGMOID,
                              MISH, LEAKY_RELU) may follow it.                        */
  KF_OP_GROUPNORM = 8,     /* per row, `groups` contiguous column groups of N/groups:
                              (v - mean) / sqrt(biased var + eps) * p0[col] + p1[col];
                              p0 (gamma) / p1 (beta) may be NULL (1 / 0).  Group size
                              must be a multiple of 32 and at most 512.              */
  KF_OP_SWIGLU = 9,        /* grouped GEMM only: B holds 2N rows per group (gate rows
                              0..N-1, then up rows N..2N-1); C = silu(gate) * up      */
  KF_OP_ROW_SCALE_SCATTER_ADD = 10, /* grouped GEMM only, last op: C[p1[r], :] +=
                              p0[r] * v  with p0 fp32 [rows_total] (row scale) and
                              p1 int32 [rows_total] (destination row); `ld` = rows of
                              C (a destination outside [0, ld) is skipped and sets
                              KF_ERR_DEVICE_BOUNDS); C is fp32 and must be
                              initialised by the caller (atomic adds, so the order
                              of the fp32 additions is not fixed).                     */
  KF_OP_MISH = 11,         /* v * tanh(log(1 + exp(v)))                                */
  KF_OP_LEAKY_RELU = 12,   /* v > 0 ? v : scalar * v                                   */
  KF_OP_MUL = 13,          /* v *= p0[col]                          (p0: [N])        */
  KF_OP_ROW_SCALE = 14,    /* v *= p0[row]                 (p0: fp32, one per row)     */
  KF_OP_ROW_SUM = 15       /* row -> sum_j v_j; Y is [M] (fp32, bf16 or fp16).  Ends a
                              chain of pointwise ops, or follows GROUPNORM (pointwise
                              ops may sit between); only scalar ops (as after
                              ROW_LOGSUMEXP) may follow it.  Needs a workspace.  The
                              "Sum" that ends the paper's Table 3 chains (Sec. IV-B),
                              read as a reduction over each row.                      */
} kf_op_kind;

typedef struct kf_epilogue_op {
  int32_t kind;       /* kf_op_kind                                          */
  float scalar;       /* SCALE factor, LEAKY_RELU slope                      */
  float eps;          /* GROUPNORM epsilon                                   */
  int32_t groups;     /* GROUPNORM group count                               */
  const void* p0;     /* op operand (device pointer), see kf_op_kind         */
  const void* p1;     /* second operand (GROUPNORM beta, scatter rows)       */
  int32_t p_dtype;    /* kf_dtype of p0 (and of p1 for GROUPNORM)            */
  int64_t ld;         /* leading dimension of a matrix operand (RESIDUAL_ADD);
                         destination row count (ROW_SCALE_SCATTER_ADD)        */
} kf_epilogue_op;

typedef struct kf_epilogue {
  int32_t num_ops;    /* 0..8 */
  const kf_epilogue_op* ops;
} kf_epilogue;

/*
 * kf_fused_gemm -- Y = chain(X W^T)                    (Sec. IV-B, Table 3)
 *
 *   X [M x K] (row stride ldx), W [N x K] (row stride ldw), Y [M x N] (row
 *   stride ldy), or Y [M] (fp32, bf16 or fp16) when the chain holds
 *   ROW_LOGSUMEXP or ROW_SUM.
 *   Operand dtypes: both KF_BF16 or both KF_F16 (tcgen05 tensor-core path, fp32
 *   accumulation in tensor memory; Y bf16, fp16 or fp32; the paper's B580
 *   kernels ran their matmuls in fp16, Sec. IV-B), or both KF_F32 (element-wise
 *   chains only): problems below 2^30 FLOP (2 M N K) take the exact fp32 FFMA
 *   path (Y fp32); larger ones run on the tensor cores as three tf32 products
 *   (3xTF32: each operand split into a tf32 high part and an fp32 remainder,
 *   X W^T = Xh Wh^T + Xh Wl^T + Xl Wh^T accumulated in fp32; Y fp32, bf16 or
 *   fp16; needs X, W 16-byte aligned and ldx, ldw multiples of 4, else the
 *   FFMA path runs) -- kf_fused_gemm_ex chooses explicitly.
 *   bf16 path: X, W must be 16-byte aligned with ldx, ldw multiples of 8, else
 *   KF_ERR_MISALIGNED.  M == 0 or N == 0 is a no-op; K must be >= 1.
 *   workspace: kf_fused_gemm_workspace() bytes.  Required for a row
 *   log-sum-exp or row sum (per-tile row partials live there).  Optional for
 *   GroupNorm over 512-column groups with M > 128 and no row sum: with it, pairs
 *   of CTA pairs exchange per-row statistics through it (all SMs work; the
 *   launch is cooperative); with a smaller or no workspace, clusters of four CTAs
 *   exchange them on chip (fewer SMs can be used).  Same results either way.  0
 *   otherwise (a KF_WORKSPACE_HEADER_BYTES workspace may still be passed, for
 *   its error word).  Calls that share one workspace must not overlap on the GPU.
 *   Y must not alias X or W; a RESIDUAL_ADD operand may alias Y (in place).
 */
kf_status kf_fused_gemm(const void* X, int32_t x_dtype, int64_t ldx, const void* W, int32_t w_dtype,
                        int64_t ldw, void* Y, int32_t y_dtype, int64_t ldy, int64_t M, int64_t N, int64_t K,
                        const kf_epilogue* epi, void* workspace, size_t workspace_bytes, void* stream);
size_t kf_fused_gemm_workspace(int64_t M, int64_t N, int64_t K, const kf_epilogue* epi);

/* kf_fused_gemm with flags for fp32 operands: KF_GEMM_F32_FFMA keeps the exact
 * FFMA path at any size; KF_GEMM_F32_TF32X3 takes the 3xTF32 tensor-core path
 * at any size (KF_ERR_MISALIGNED if X, W or ldx, ldw do not allow its 16-byte
 * TMA boxes).  Both at once, or an unknown bit: KF_ERR_INVALID_ARG.  flags = 0
 * is kf_fused_gemm.  No effect on bf16 / fp16 operands. */
#define KF_GEMM_F32_FFMA 1u
#define KF_GEMM_F32_TF32X3 2u
kf_status kf_fused_gemm_ex(const void* X, int32_t x_dtype, int64_t ldx, const void* W, int32_t w_dtype,
                           int64_t ldw, void* Y, int32_t y_dtype, int64_t ldy, int64_t M, int64_t N, int64_t K,
                           const kf_epilogue* epi, void* workspace, size_t workspace_bytes, uint32_t flags,
                           void* stream);

/*
 * kf_moe_route -- top-k routing of T tokens over E experts  (Sec. IV-A, decode path)
 *
 *   logits fp32 [T x E].  For each token the k experts with the largest logits
 *   (ties -> lower expert index), in descending order, go to topk_ids int32
 *   [T x k]; topk_w fp32 [T x k] is the softmax over those k logits (sums to 1).
 *   The T*k (token, slot) pairs are then sorted by expert with a stable
 *   counting sort (pair p = t*k + slot keeps increasing p within an expert):
 *   expert_offsets int32 [E + 1] (offsets[e]..offsets[e+1] are expert e's rows),
 *   sorted_token int32 [T*k] (token of each sorted row), sorted_w fp32 [T*k]
 *   (its routing weight).  1 <= k <= E <= 256.  T == 0 writes offsets only.
 */
kf_status kf_moe_route(const float* logits, int64_t T, int32_t E, int32_t k, int32_t* topk_ids, float* topk_w,
                       int32_t* expert_offsets, int32_t* sorted_token, float* sorted_w, void* stream);

/*
 * kf_grouped_gemm -- per-group C rows = chain(A rows B[g]^T)  (Sec. IV-A, MoE experts)
 *
 *   Row group g owns rows r in [group_offsets[g], group_offsets[g+1]) of the
 *   rows_total output rows; group_offsets is a DEVICE int32 array [G + 1]
 *   (non-decreasing, ending at <= rows_total; read on the device, so routing
 *   never needs a host sync).  Row r of the GEMM input is A[a_row_index[r]]
 *   when a_row_index (device int32 [rows_total]) is given (gather; a_rows is
 *   A's row count, for bounds), else A[r].  B[g] = B + g*b_group_stride
 *   elements, rows of K with stride ldb: N rows, or 2N rows with SWIGLU.
 *   C is [rows_total x N] (stride ldc), bf16 or fp32; with
 *   ROW_SCALE_SCATTER_ADD C is the fp32 scatter target instead.
 *   A, B bf16; alignment rules as kf_fused_gemm (also b_group_stride % 8 == 0).
 *   workspace: kf_grouped_gemm_workspace() bytes (the gathered rows live there;
 *   0 without a gather).  Bad device-side offsets/indices set
 *   KF_ERR_DEVICE_BOUNDS in the error words.
 */
kf_status kf_grouped_gemm(const void* A, int32_t a_dtype, int64_t lda, int64_t a_rows, const int32_t* a_row_index,
                          const void* B, int32_t b_dtype, int64_t ldb, int64_t b_group_stride,
                          const int32_t* group_offsets, int32_t G, int64_t rows_total, int64_t N, int64_t K,
                          void* C, int32_t c_dtype, int64_t ldc, const kf_epilogue* epi, void* workspace,
                          size_t workspace_bytes, void* stream);
size_t kf_grouped_gemm_workspace(int64_t rows_total, int64_t N, int64_t K, int32_t G, int32_t gathered,
                                 const kf_epilogue* epi);

/*
 * kf_moe_ffn -- routed MoE expert FFN, end to end           (Sec. IV-A, Table 1)
 *
 *   Y_t = sum_j topk_w[t,j] * W_down[e] (silu(W_gate[e] x_t) * (W_up[e] x_t)),
 *   e = topk_ids[t,j], with the intermediate h rounded to bf16 (the down GEMM's
 *   input dtype).  X bf16 [T x H]; logits fp32 [T x E]; W_gu bf16 [E x 2I x H]
 *   (gate rows 0..I-1, up rows I..2I-1 per expert); W_down bf16 [E x H x I];
 *   Y bf16 [T x H].  Runs kf_moe_route, the gathered gate/up grouped GEMM with
 *   the SwiGLU epilogue, and the down grouped GEMM with the routing-weight
 *   scale + scatter-add epilogue, then converts the fp32 sum to bf16.
 *   H and I multiples of 8.  workspace: kf_moe_ffn_workspace() bytes.
 *   If topk_ids_out / topk_w_out are non-NULL the routing is copied there.
 */
kf_status kf_moe_ffn(const void* X, const float* logits, const void* W_gu, const void* W_down, void* Y, int64_t T,
                     int64_t H, int64_t I, int32_t E, int32_t k, void* workspace, size_t workspace_bytes,
                     int32_t* topk_ids_out, float* topk_w_out, void* stream);
size_t kf_moe_ffn_workspace(int64_t T, int64_t H, int64_t I, int32_t E, int32_t k);

/* kf_moe_ffn with flags.  KF_MOE_DETERMINISTIC: the down GEMM writes each routed
 * row's weighted output (fp32 [T*k x H], in the workspace) and a finalize kernel
 * sums each token's k rows in slot order, so Y is bit-identical from run to run
 * (the default scatter-add uses fp32 atomics, whose summation order is not
 * fixed).  Needs kf_moe_ffn_workspace_ex(..., flags) bytes. */
#define KF_MOE_DETERMINISTIC 1u
kf_status kf_moe_ffn_ex(const void* X, const float* logits, const void* W_gu, const void* W_down, void* Y, int64_t T,
                        int64_t H, int64_t I, int32_t E, int32_t k, uint32_t flags, void* workspace,
                        size_t workspace_bytes, int32_t* topk_ids_out, float* topk_w_out, void* stream);
size_t kf_moe_ffn_workspace_ex(int64_t T, int64_t H, int64_t I, int32_t E, int32_t k, uint32_t flags);

/*
 * kf_moe_ffn_act -- kf_moe_ffn_ex with the gated-expert activation and biases of
 *                   the gpt-oss expert MLP (the model of the paper's B200 decode
 *                   study, Sec. IV-A; the paper itself gives no formula)
 *
 *   g = x W_gate[e]^T + bg[e],  u = x W_up[e]^T + bu[e]     (fp32 accumulators)
 *   g' = min(g, limit), u' = clamp(u, -limit, limit)        (when limit > 0)
 *   h  = bf16(g' * sigmoid(alpha * g') * (u' + linear_offset))
 *   Y[t] = sum_j w_tj * (h W_down[e_tj]^T + bd[e_tj])
 *   {alpha 1, limit 0, linear_offset 0, no biases} is the plain SwiGLU of
 *   kf_moe_ffn_ex; gpt-oss uses alpha 1.702, limit 7, linear_offset 1 and both
 *   biases.  Gate and up rows stay the concatenated halves of W_gu[e] (a model
 *   that interleaves them is permuted once when its weights are loaded).
 *   b_gu: bf16 [E x 2I] (gate bias then up bias of each expert), b_down: bf16
 *   [E x H]; either may be NULL; both 16-byte aligned (KF_ERR_MISALIGNED).
 *   alpha, limit, linear_offset finite and limit >= 0 (KF_ERR_INVALID_ARG).
 *   Everything else (arguments, flags, workspace, errors) as kf_moe_ffn_ex.
 */
typedef struct kf_moe_act {
  float alpha;
  float limit;
  float linear_offset;
  const void* b_gu;
  const void* b_down;
} kf_moe_act;
kf_status kf_moe_ffn_act(const void* X, const float* logits, const void* W_gu, const void* W_down,
                         const kf_moe_act* act, void* Y, int64_t T, int64_t H, int64_t I, int32_t E, int32_t k,
                         uint32_t flags, void* workspace, size_t workspace_bytes, int32_t* topk_ids_out,
                         float* topk_w_out, void* stream);

/*
 * kf_moe_ffn_add_rmsnorm -- the MoE block tail fused into the MoE finalize
 *                          (Sec. IV-A: the gpt-oss decode kernels "Fused Add +
 *                          RMSNorm" and "MoE finalize"; Sec. V: optimising the
 *                          kernels of one block together)
 *
 *   The routed expert FFN of kf_moe_ffn_ex (same arguments and flags), whose
 *   finalize, instead of writing the FFN output, adds it to the residual stream
 *   and normalises the result:
 *     R_out[t,:] = bf16(R[t,:] + MoE(X)[t,:])                (new residual stream)
 *     Y[t,j]     = bf16(R_out[t,j] / sqrt(mean_j R_out[t,j]^2 + eps) * gamma[j])
 *   The norm reads the stored bf16 residual, as the next layer would.  R, R_out,
 *   Y bf16 [T x H] (row stride H), gamma bf16 [H], all 16-byte aligned
 *   (KF_ERR_MISALIGNED otherwise); R may be R_out (in place).  H <= 8192
 *   (KF_ERR_UNSUPPORTED above), eps >= 0 (KF_ERR_INVALID_ARG otherwise).
 *   workspace: kf_moe_ffn_workspace_ex(T, H, I, E, k, flags) bytes, owned by the
 *   caller like every buffer here; calls sharing it must not overlap on the GPU.
 */
kf_status kf_moe_ffn_add_rmsnorm(const void* X, const float* logits, const void* W_gu, const void* W_down,
                                 const void* R, const void* gamma, float eps, void* R_out, void* Y, int64_t T,
                                 int64_t H, int64_t I, int32_t E, int32_t k, uint32_t flags, void* workspace,
                                 size_t workspace_bytes, int32_t* topk_ids_out, float* topk_w_out, void* stream);

/*
 * kf_qkv_rope_kv -- the attention input projection with its tail fused into the
 *                   GEMM's epilogue (Sec. IV-A and Table 1: the gpt-oss decode
 *                   kernel "Bias + RoPE + KV update"; here it runs on the
 *                   projection's accumulator instead of a second pass)
 *
 *   s[t,:] = X[t,:] W^T + bias, N = (nq + 2 nkv) d columns: nq query heads, then
 *   nkv key heads, then nkv value heads of d columns each.  Query and key heads
 *   are rotated by the half-split rotary embedding of token t's position p_t:
 *     (s_i, s_{i+d/2}) -> (s_i c - s_{i+d/2} v, s_{i+d/2} c + s_i v),
 *     c = cos_t[p_t][i], v = sin_t[p_t][i], i < d/2
 *   (any frequency scaling lives in the caller's tables).  Queries go to
 *   q_out[t,:] (nq d columns); keys and values to row cache_rows[t] of k_cache /
 *   v_cache (nkv d columns each).  Only the named cache rows are written; two
 *   tokens naming one row leave either token's values there.
 *   X, W: both bf16 or both fp16 (KF_BF16 / KF_F16 in xw_dtype), X [T x H] row
 *     stride ldx, W [N x H] row stride ldw (K-major), 16-byte aligned, ldx and
 *     ldw multiples of 8 (KF_ERR_MISALIGNED otherwise).
 *   bias: [N] of bias_dtype (KF_BF16, KF_F16 or KF_F32), or NULL.
 *   positions, cache_rows: int32 [T] on the device.  A position outside
 *     [0, max_pos) or a cache row outside [0, cache_rows_n) skips that token's
 *     writes and sets the bounds bit of the device error word
 *     (kf_get_device_error).
 *   cos_t, sin_t: fp32 [max_pos x d/2], row stride d/2, 16-byte aligned.
 *   q_out [T x ldq], k_cache / v_cache [cache_rows_n x ld_cache]: out_dtype
 *     (KF_BF16, KF_F16 or KF_F32); ldq >= nq d, ld_cache >= nkv d.
 *   d: a multiple of 64, at most 256 (KF_ERR_UNSUPPORTED otherwise); nq, nkv >= 1.
 *   Calls of at most 64 tokens with d dividing 256 run as clusters of CTAs
 *   that split K over each 256-column tile and add their partial sums in
 *   shared memory in a fixed order; larger calls run as tensor-core tiles over
 *   the whole K.  Either way repeated calls are bitwise identical.
 *   T = 0 writes nothing.  All buffers are the caller's; nothing is allocated.
 */
kf_status kf_qkv_rope_kv(const void* X, const void* W, int32_t xw_dtype, int64_t ldx, int64_t ldw, const void* bias,
                         int32_t bias_dtype, const int32_t* positions, const int32_t* cache_rows, const float* cos_t,
                         const float* sin_t, int64_t max_pos, int64_t T, int64_t H, int32_t nq, int32_t nkv,
                         int32_t d, void* q_out, int64_t ldq, void* k_cache, void* v_cache, int64_t ld_cache,
                         int64_t cache_rows_n, int32_t out_dtype, void* stream);

/*
 * kf_fused_gemm_lse_noalloc -- kf_fused_gemm for row log-sum-exp chains, without
 * a workspace argument.  The paper has no counterpart: this entry point exists for
 * callers that cannot allocate device memory -- e.g. code hosted by another
 * runtime that owns all device memory and exposes no allocator to it, or
 * latency-critical loops that must not call cudaMalloc because it can
 * synchronize the device.  The caller still passes X, W and Y (as for
 * kf_fused_gemm, with Y the fp32 or bf16 [M] result; the chain must hold
 * KF_OP_ROW_LOGSUMEXP, else KF_ERR_INVALID_ARG).
 *   Scratch: the per-tile row partials live in one fixed device array of
 *   kf_fused_gemm_lse_noalloc_max_bytes() bytes (4 MiB) compiled into the
 *   library; every GPU that loads the library holds it until the process exits.
 *   Problems needing more (M x ceil(N/128) x 8 bytes) return KF_ERR_WORKSPACE and
 *   launch nothing.  This call never allocates or frees device memory.
 *   The first call on a device looks up the array's device address (with that
 *   device current) and caches it; make that first call before any stream
 *   capture.  Every call shares the one array: calls whose executions overlap
 *   on the GPU (different streams, or different host threads) race on it and
 *   must be serialized by the caller.  Each call overwrites every partial it
 *   reads, so no clearing is needed between calls.  Operands bf16 or fp16, as
 *   for kf_fused_gemm.  Device-side errors go to the per-device error word
 *   (kf_get_device_error).
 */
kf_status kf_fused_gemm_lse_noalloc(const void* X, int32_t x_dtype, int64_t ldx, const void* W, int32_t w_dtype,
                                    int64_t ldw, void* Y, int32_t y_dtype, int64_t M, int64_t N, int64_t K,
                                    const kf_epilogue* epi, void* stream);
size_t kf_fused_gemm_lse_noalloc_max_bytes(void);

/* Synchronize `stream`, read and clear this device's error word (the errors of
 * every call on the device).  Returns KF_OK, KF_ERR_DEVICE_TIMEOUT or
 * KF_ERR_DEVICE_BOUNDS (KF_ERR_CUDA for a launch-shape error); *raw (if non-NULL)
 * receives the raw bit set (1 = producer wait, 2 = MMA wait, 4 = epilogue wait,
 * 8 = bounds, 16 = launch shape). */
kf_status kf_get_device_error(void* stream, uint32_t* raw);

/* The same for the error word in `workspace`'s header: only the calls that were
 * given this workspace write it, so threads that use distinct workspaces see
 * only their own errors.  `workspace` is the pointer the calls were given
 * (device memory, 16-byte aligned; KF_ERR_INVALID_ARG otherwise).  Synchronizes
 * `stream`, which must be the stream of those calls (or one ordered after them).
 * Returns and reports as kf_get_device_error. */
kf_status kf_check_device_error(void* workspace, void* stream, uint32_t* raw);

/* Zero `workspace`'s header (cudaMemsetAsync of KF_WORKSPACE_HEADER_BYTES bytes
 * on `stream`): needed once before a workspace's first use unless it was
 * allocated zero-filled.  `bytes` >= KF_WORKSPACE_HEADER_BYTES and a 16-byte
 * aligned pointer, else KF_ERR_INVALID_ARG.  Allocates nothing. */
kf_status kf_workspace_init(void* workspace, size_t bytes, void* stream);

/* Wall-time limit of every device-side wait, in ns, for later launches
 * (0 restores the default of 2 s).  A short limit makes a kernel give up early
 * and report KF_ERR_DEVICE_TIMEOUT; used by the failure-detection test. */
kf_status kf_set_wait_timeout_ns(uint64_t ns);

const char* kf_status_string(int32_t status);
int32_t kf_abi_version(void);

#ifdef __cplusplus
}
#endif
#endif /* KF_H_ */
