// kf_simt.cu -- CUDA-core kernels of the path:
//   * exact fp32 FFMA GEMM + element-wise chain (fp32 operands; no TF32, since a
//     silent downcast is exactly what the paper's candidate guardrails ban, Sec. III-D),
//   * cross-tile combine of the row log-sum-exp partials (Sec. IV-B, online LSE),
//   * MoE routing: per-token top-k + softmax, then a deterministic stable
//     counting sort of the (token, slot) pairs by expert (Sec. IV-A, gpt-oss),
//   * row gather of routed tokens, fp32 -> bf16 conversion of the MoE output.
#include <cuda_bf16.h>

#include <algorithm>

#include "kf_internal.h"

namespace kf {

// Scalar form of the chain for one element (fp32 path).
__device__ __forceinline__ float apply_chain1(const DevOp* ops, int n, float v, int64_t row, int64_t col) {
  for (int o = 0; o < n; ++o) {
    const DevOp& op = ops[o];
    switch (op.kind) {
      case KF_OP_BIAS: v += ld_elem(op.p0, op.p_dtype, col); break;
      case KF_OP_MUL: v *= ld_elem(op.p0, op.p_dtype, col); break;
      case KF_OP_RESIDUAL_ADD: v += ld_elem(op.p0, op.p_dtype, row * op.ld + col); break;
      case KF_OP_ROW_SCALE: v *= reinterpret_cast<const float*>(op.p0)[row]; break;
      default: v = apply_scalar_op(op, v); break;
    }
  }
  return v;
}

// ------------------------------------------------------------------ fp32 GEMM
// 16 x 16 output tile per 256-thread block; the four warp pairs take a quarter
// of each 128-wide K chunk each (2 x 2 outputs per thread), and the quarters
// are added in a fixed order at the end.  Chunks are double-buffered: the next
// chunk's loads are in flight while the current one is multiplied, so a small
// problem (the launch-bound sizes this path serves) pays about one memory round
// trip instead of one per chunk, and 16 x 16 tiles give many blocks.
constexpr int kFT = 16;    // output tile edge
constexpr int kFK = 128;   // K chunk
constexpr int kFPad = 129; // shared row stride (floats): distinct banks per row
__device__ __forceinline__ void f32_chunk_load(const float* __restrict__ src, int64_t ld, int32_t rows, int32_t r0,
                                               int32_t K, int32_t k0, bool vec, int t, float (&r)[8]) {
  // 16 rows x 128 columns = 512 groups of 4 columns; thread t takes groups t, t + 256
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int gi = t + 256 * h;
    const int row = gi >> 5, kq = (gi & 31) * 4;
    const int32_t gr = r0 + row, gk = k0 + kq;
    const float* q = src + static_cast<int64_t>(gr) * ld + gk;
    if (gr < rows && vec && gk + 3 < K) {
      const float4 v = __ldg(reinterpret_cast<const float4*>(q));
      r[4 * h] = v.x;
      r[4 * h + 1] = v.y;
      r[4 * h + 2] = v.z;
      r[4 * h + 3] = v.w;
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j) r[4 * h + j] = (gr < rows && gk + j < K) ? __ldg(q + j) : 0.0f;
    }
  }
}
__device__ __forceinline__ void f32_chunk_store(float (*dst)[kFPad], int t, const float (&r)[8]) {
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int gi = t + 256 * h;
    const int row = gi >> 5, kq = (gi & 31) * 4;
#pragma unroll
    for (int j = 0; j < 4; ++j) dst[row][kq + j] = r[4 * h + j];
  }
}

__global__ void __launch_bounds__(256) simt_gemm_f32_kernel(const __grid_constant__ SimtParams p) {
  __shared__ float xs[2][kFT][kFPad];
  __shared__ float ws[2][kFT][kFPad];
  const int t = threadIdx.x;
  const int kq = t >> 6;            // K quarter of each chunk
  const int o = t & 63;
  const int om = (o >> 3) * 2, on = (o & 7) * 2;
  const int32_t m0 = blockIdx.y * kFT, n0 = blockIdx.x * kFT;
  const bool xvec = (reinterpret_cast<uintptr_t>(p.X) & 15) == 0 && (p.ldx & 3) == 0;
  const bool wvec = (reinterpret_cast<uintptr_t>(p.W) & 15) == 0 && (p.ldw & 3) == 0;
  const int nchunks = (p.K + kFK - 1) / kFK;
  float rx[8], rw[8];
  f32_chunk_load(p.X, p.ldx, p.M, m0, p.K, 0, xvec, t, rx);
  f32_chunk_load(p.W, p.ldw, p.N, n0, p.K, 0, wvec, t, rw);
  f32_chunk_store(xs[0], t, rx);
  f32_chunk_store(ws[0], t, rw);
  __syncthreads();
  float acc[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
  for (int c = 0; c < nchunks; ++c) {
    const int b = c & 1;
    const bool more = c + 1 < nchunks;
    if (more) {  // next chunk in flight during this one's products
      f32_chunk_load(p.X, p.ldx, p.M, m0, p.K, (c + 1) * kFK, xvec, t, rx);
      f32_chunk_load(p.W, p.ldw, p.N, n0, p.K, (c + 1) * kFK, wvec, t, rw);
    }
#pragma unroll 8
    for (int k = kq * 32; k < kq * 32 + 32; ++k) {
      const float a0 = xs[b][om][k], a1 = xs[b][om + 1][k];
      const float b0 = ws[b][on][k], b1 = ws[b][on + 1][k];
      acc[0][0] = fmaf(a0, b0, acc[0][0]);
      acc[0][1] = fmaf(a0, b1, acc[0][1]);
      acc[1][0] = fmaf(a1, b0, acc[1][0]);
      acc[1][1] = fmaf(a1, b1, acc[1][1]);
    }
    if (more) {
      f32_chunk_store(xs[b ^ 1], t, rx);
      f32_chunk_store(ws[b ^ 1], t, rw);
    }
    __syncthreads();
  }
  // the four quarters' partial sums, added in quarter order by quarter 0
  float* red = &xs[0][0][0];  // [4][16 x 16] after the last chunk
#pragma unroll
  for (int i = 0; i < 2; ++i)
#pragma unroll
    for (int j = 0; j < 2; ++j) red[kq * 256 + (om + i) * kFT + on + j] = acc[i][j];
  __syncthreads();
  if (kq == 0) {
#pragma unroll
    for (int i = 0; i < 2; ++i)
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const int e = (om + i) * kFT + on + j;
        const float v = ((red[e] + red[256 + e]) + red[512 + e]) + red[768 + e];
        const int32_t gm = m0 + om + i, gn = n0 + on + j;
        if (gm < p.M && gn < p.N) p.Y[static_cast<int64_t>(gm) * p.ldy + gn] = apply_chain1(p.ops, p.n_ops, v, gm, gn);
      }
  }
}

cudaError_t simt_gemm_f32_launch(const SimtParams& p, cudaStream_t s) {
  dim3 grid((p.N + kFT - 1) / kFT, (p.M + kFT - 1) / kFT);
  simt_gemm_f32_kernel<<<grid, 256, 0, s>>>(p);
  return cudaGetLastError();
}

// ------------------------------------------------------- row log-sum-exp combine
// (m, s) (+) (m', s') = (M, s e^{m-M} + s' e^{m'-M}),  out = M + log S.
__global__ void lse_combine_kernel(const __grid_constant__ LseCombineParams p) {
  griddep_wait();  // after the library kernel this one follows (programmatic launch)
  griddep_launch_dependents();
  const int warps = blockDim.x >> 5;
  const int row = blockIdx.x * warps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= p.M) return;
  const float2* part = p.part + static_cast<int64_t>(row) * p.parts;
  if (p.red_sum) {
    // row sum: the partials' sums, lane-strided then a fixed butterfly (the
    // same order on every call)
    float s = 0.f;
    for (int i = lane; i < p.parts; i += 32) s += part[i].y;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) {
      float v = s;
      for (int o = 0; o < p.n_post; ++o) v = apply_scalar_op(p.post[o], v);
      if (p.out_dtype == KF_BF16)
        reinterpret_cast<__nv_bfloat16*>(p.out)[row] = __float2bfloat16_rn(v);
      else if (p.out_dtype == KF_F16)
        reinterpret_cast<__half*>(p.out)[row] = __float2half_rn(v);
      else
        reinterpret_cast<float*>(p.out)[row] = v;
    }
    return;
  }
  float m = -INFINITY, s = 0.f;
  for (int i = lane; i < p.parts; i += 32) {
    const float2 q = part[i];
    const float nm = fmaxf(m, q.x);
    if (nm != -INFINITY) {
      s = (m == -INFINITY ? 0.f : s * expf(m - nm)) + (q.x == -INFINITY ? 0.f : q.y * expf(q.x - nm));
      m = nm;
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    const float om = __shfl_xor_sync(0xffffffffu, m, off);
    const float os = __shfl_xor_sync(0xffffffffu, s, off);
    const float nm = fmaxf(m, om);
    if (nm != -INFINITY) {
      s = (m == -INFINITY ? 0.f : s * expf(m - nm)) + (om == -INFINITY ? 0.f : os * expf(om - nm));
      m = nm;
    }
  }
  if (lane == 0) {
    float v = (m == -INFINITY) ? -INFINITY : m + logf(s);
    for (int o = 0; o < p.n_post; ++o) v = apply_scalar_op(p.post[o], v);
    if (p.out_dtype == KF_BF16)
      reinterpret_cast<__nv_bfloat16*>(p.out)[row] = __float2bfloat16_rn(v);
    else if (p.out_dtype == KF_F16)
      reinterpret_cast<__half*>(p.out)[row] = __float2half_rn(v);
    else
      reinterpret_cast<float*>(p.out)[row] = v;
  }
}

cudaError_t lse_combine_launch(const LseCombineParams& p, cudaStream_t s, bool pdl) {
  const int warps = 8;
  return launch_k(lse_combine_kernel, dim3((p.M + warps - 1) / warps), dim3(warps * 32), 0, s, pdl, p);
}

// ------------------------------------------------------------------- routing
// One warp per token; expert e lives in lane e % 32, slot e / 32 (E <= 256).
// Selection order: larger logit first, ties -> lower expert index.
constexpr int kMaxExperts = 256;
__global__ void route_topk_kernel(const float* __restrict__ logits, int32_t T, int32_t E, int32_t k,
                                  int32_t* __restrict__ ids, float* __restrict__ w) {
  griddep_wait();  // after the library kernel this one follows (programmatic launch)
  griddep_launch_dependents();
  const int warps = blockDim.x >> 5;
  const int t = blockIdx.x * warps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (t >= T) return;
  float val[kMaxExperts / 32];
  uint32_t taken = 0;
#pragma unroll
  for (int i = 0; i < kMaxExperts / 32; ++i) {
    const int e = i * 32 + lane;
    val[i] = e < E ? logits[static_cast<int64_t>(t) * E + e] : -INFINITY;
    if (e >= E) taken |= 1u << i;
  }
  float sel_v = 0.f, vmax = 0.f, den = 0.f;
  int sel_e = 0;
  for (int j = 0; j < k; ++j) {
    float bv = -INFINITY;
    int be = 0x7fffffff;
#pragma unroll
    for (int i = 0; i < kMaxExperts / 32; ++i) {
      const int e = i * 32 + lane;
      if (!(taken >> i & 1u) && (val[i] > bv || (val[i] == bv && e < be))) {
        bv = val[i];
        be = e;
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
      const int oe = __shfl_xor_sync(0xffffffffu, be, off);
      if (ov > bv || (ov == bv && oe < be)) {
        bv = ov;
        be = oe;
      }
    }
    if ((be & 31) == lane) taken |= 1u << (be >> 5);
    if (j == 0) vmax = bv;
    const float ex = expf(bv - vmax);
    den += ex;
    if (lane == j) {  // lane j keeps slot j (k <= 32 handled below)
      sel_v = ex;
      sel_e = be;
    }
    if (k > 32 && lane == 0) {
      ids[static_cast<int64_t>(t) * k + j] = be;
      w[static_cast<int64_t>(t) * k + j] = ex;  // normalised in a second pass below
    }
  }
  if (k <= 32) {
    if (lane < k) {
      ids[static_cast<int64_t>(t) * k + lane] = sel_e;
      w[static_cast<int64_t>(t) * k + lane] = sel_v / den;
    }
  } else if (lane == 0) {
    for (int j = 0; j < k; ++j) w[static_cast<int64_t>(t) * k + j] /= den;
  }
}

cudaError_t route_topk_launch(const float* logits, int32_t T, int32_t E, int32_t k, int32_t* ids, float* w,
                              cudaStream_t s) {
  if (T == 0) return cudaSuccess;
  const int warps = 8;
  route_topk_kernel<<<(T + warps - 1) / warps, warps * 32, 0, s>>>(logits, T, E, k, ids, w);
  return cudaGetLastError();
}

// Stable counting sort of P = T*k pairs by expert, one 1024-thread block.
// Warp w owns the contiguous pair range [w*chunk, (w+1)*chunk); counts per
// (warp, expert), scanned expert-major then warp-minor, give each warp's first
// slot per expert; a second in-order walk ranks equal experts within each
// 32-pair batch with __match_any_sync.  Output order = increasing pair index
// within each expert (bit-identical to a sequential stable sort).
constexpr int kSortWarps = 32;
__global__ void __launch_bounds__(kSortWarps * 32) route_sort_kernel(const int32_t* __restrict__ ids,
                                                                     const float* __restrict__ w, int32_t P,
                                                                     int32_t E, int32_t k, int32_t* offsets,
                                                                     int32_t* sorted_token, float* sorted_w,
                                                                     int32_t* pair_pos) {
  griddep_wait();  // after the library kernel this one follows (programmatic launch)
  griddep_launch_dependents();
  extern __shared__ int32_t cnt[];  // [kSortWarps][E]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = threadIdx.x; i < kSortWarps * E; i += blockDim.x) cnt[i] = 0;
  __syncthreads();
  const int32_t chunk = (P + kSortWarps - 1) / kSortWarps;
  const int32_t beg = min(P, warp * chunk), end = min(P, beg + chunk);
  for (int32_t p = beg + lane; p < end; p += 32) atomicAdd(&cnt[warp * E + ids[p]], 1);
  __syncthreads();
  // Scan the (expert, warp) counts in expert-major, warp-minor order.  Thread e
  // sums its expert's column; warp 0 scans the E totals (lane l owns experts
  // l*per .. l*per+per-1, then a shuffle scan across lanes); thread e then turns
  // its column into each warp's first slot for expert e.
  __shared__ int32_t tot[kMaxExperts];
  if (threadIdx.x < E) {
    int32_t t = 0;
    for (int ww = 0; ww < kSortWarps; ++ww) t += cnt[ww * E + threadIdx.x];
    tot[threadIdx.x] = t;
  }
  __syncthreads();
  if (warp == 0) {
    const int per = (E + 31) / 32;
    int32_t local = 0;
    for (int i = 0; i < per; ++i) {
      const int e = lane * per + i;
      if (e < E) local += tot[e];
    }
    int32_t incl = local;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int32_t o = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += o;
    }
    int32_t run = incl - local;  // exclusive prefix of this lane's first expert
    for (int i = 0; i < per; ++i) {
      const int e = lane * per + i;
      if (e < E) {
        const int32_t t = tot[e];
        tot[e] = run;
        offsets[e] = run;
        run += t;
      }
    }
    if (lane == 31) offsets[E] = run;
  }
  __syncthreads();
  if (threadIdx.x < E) {
    int32_t run = tot[threadIdx.x];
    for (int ww = 0; ww < kSortWarps; ++ww) {
      const int32_t c = cnt[ww * E + threadIdx.x];
      cnt[ww * E + threadIdx.x] = run;  // first slot of (warp ww, expert e)
      run += c;
    }
  }
  __syncthreads();
  const uint32_t lt_mask = (1u << lane) - 1u;
  for (int32_t b = beg; b < end; b += 32) {
    const int32_t p = b + lane;
    const bool valid = p < end;
    const int32_t e = valid ? ids[p] : E + lane;  // invalid lanes never match a real expert
    const uint32_t peers = __match_any_sync(0xffffffffu, e);
    const int rank = __popc(peers & lt_mask);
    if (valid) {
      const int32_t pos = cnt[warp * E + e] + rank;
      sorted_token[pos] = p / k;
      sorted_w[pos] = w[p];
      if (pair_pos) pair_pos[p] = pos;
    }
    __syncwarp();
    if (valid && rank == 0) cnt[warp * E + e] += __popc(peers);
    __syncwarp();
  }
}

cudaError_t route_sort_launch(const int32_t* ids, const float* w, int32_t T, int32_t E, int32_t k,
                              int32_t* offsets, int32_t* sorted_token, float* sorted_w, int32_t* pair_pos,
                              cudaStream_t s, bool pdl) {
  const int32_t P = T * k;
  const size_t smem = sizeof(int32_t) * kSortWarps * E;
  return launch_k(route_sort_kernel, dim3(1), dim3(kSortWarps * 32), smem, s, pdl, ids, w, P, E, k, offsets,
                  sorted_token, sorted_w, pair_pos);
}

// Multi-block form of the same stable counting sort, for many pairs (one SM
// issuing every scattered store of the one-block kernel takes ~24 us at 16 K
// pairs).  Pairs go in chunks of kSortChunk, one chunk per block:
//   route_count_kernel    per-block expert histogram -> counts[b][e]
//   route_scatter_kernel  block b's first slot of expert e = (pairs of experts
//                         < e) + (pairs of expert e in blocks < b); within the
//                         block, warps hold 32 consecutive pairs each, ranked by
//                         __match_any_sync and offset by the earlier warps' counts.
// The order is the one-block kernel's (increasing pair index within an expert).
constexpr int kSortChunk = 256;  // pairs per block = threads per block

__global__ void __launch_bounds__(kSortChunk) route_count_kernel(const int32_t* __restrict__ ids, int32_t P,
                                                                 int32_t E, int32_t* __restrict__ counts) {
  griddep_wait();  // after the routing kernel (programmatic launch)
  griddep_launch_dependents();
  __shared__ int32_t cnt[kMaxExperts];
  for (int e = threadIdx.x; e < E; e += blockDim.x) cnt[e] = 0;
  __syncthreads();
  const int32_t p = blockIdx.x * kSortChunk + threadIdx.x;
  if (p < P) atomicAdd(&cnt[ids[p]], 1);
  __syncthreads();
  for (int e = threadIdx.x; e < E; e += blockDim.x) counts[static_cast<int64_t>(blockIdx.x) * E + e] = cnt[e];
}

__global__ void __launch_bounds__(kSortChunk) route_scatter_kernel(const int32_t* __restrict__ ids,
                                                                   const float* __restrict__ w, int32_t P,
                                                                   int32_t E, int32_t k,
                                                                   const int32_t* __restrict__ counts,
                                                                   int32_t* offsets, int32_t* sorted_token,
                                                                   float* sorted_w, int32_t* pair_pos) {
  griddep_wait();  // after the count kernel (programmatic launch)
  griddep_launch_dependents();
  constexpr int kW = kSortChunk / 32;
  __shared__ int32_t base[kMaxExperts];   // this block's first slot per expert
  __shared__ int32_t tot[kMaxExperts];
  __shared__ int32_t wcnt[kW][kMaxExperts];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int32_t nb = gridDim.x, b = blockIdx.x;
  for (int e = threadIdx.x; e < E; e += blockDim.x) {
    int32_t before = 0, all = 0;
    for (int32_t bb = 0; bb < nb; ++bb) {
      const int32_t c = counts[static_cast<int64_t>(bb) * E + e];
      if (bb < b) before += c;
      all += c;
    }
    base[e] = before;
    tot[e] = all;
  }
  for (int i = threadIdx.x; i < kW * E; i += blockDim.x) wcnt[i / E][i % E] = 0;
  __syncthreads();
  if (warp == 0) {
    // exclusive scan of the expert totals (lane l owns experts l*per .. l*per+per-1)
    const int per = (E + 31) / 32;
    int32_t local = 0;
    for (int i = 0; i < per; ++i) {
      const int e = lane * per + i;
      if (e < E) local += tot[e];
    }
    int32_t incl = local;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int32_t o = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += o;
    }
    int32_t run = incl - local;
    for (int i = 0; i < per; ++i) {
      const int e = lane * per + i;
      if (e < E) {
        base[e] += run;
        if (b == 0) offsets[e] = run;
        run += tot[e];
      }
    }
    if (b == 0 && lane == 31) offsets[E] = run;
  }
  // ranks within the warp's 32 pairs, and the warp's count per expert
  const int32_t p = b * kSortChunk + threadIdx.x;
  const bool valid = p < P;
  const int32_t e = valid ? ids[p] : E + lane;  // invalid lanes never match a real expert
  const uint32_t peers = __match_any_sync(0xffffffffu, e);
  const int rank = __popc(peers & ((1u << lane) - 1u));
  if (valid && rank == 0) wcnt[warp][e] = __popc(peers);
  __syncthreads();
  if (valid) {
    int32_t pos = base[e] + rank;
    for (int ww = 0; ww < warp; ++ww) pos += wcnt[ww][e];
    sorted_token[pos] = p / k;
    sorted_w[pos] = w[p];
    if (pair_pos) pair_pos[p] = pos;
  }
}

cudaError_t route_sort_mb_launch(const int32_t* ids, const float* w, int32_t T, int32_t E, int32_t k,
                                 int32_t* offsets, int32_t* sorted_token, float* sorted_w, int32_t* pair_pos,
                                 int32_t* counts, cudaStream_t s, bool pdl) {
  const int32_t P = T * k;
  const int nb = (P + kSortChunk - 1) / kSortChunk;
  cudaError_t e = launch_k(route_count_kernel, dim3(nb), dim3(kSortChunk), 0, s, pdl, ids, P, E, counts);
  if (e != cudaSuccess) return e;
  return launch_k(route_scatter_kernel, dim3(nb), dim3(kSortChunk), 0, s, true, ids, w, P, E, k,
                  static_cast<const int32_t*>(counts), offsets, sorted_token, sorted_w, pair_pos);
}
int32_t route_sort_mb_blocks(int32_t P) { return (P + kSortChunk - 1) / kSortChunk; }

// ------------------------------------------------ deterministic MoE finalize
// Y[t, :] = bf16( sum_{j = 0..k-1} Yp[pair_pos[t*k + j], :] ), slot order fixed.
__global__ void moe_finalize_kernel(const float4* __restrict__ Yp, const int32_t* __restrict__ pair_pos, int64_t T,
                                    int32_t k, int64_t h4, uint2* __restrict__ Y) {
  griddep_wait();  // after the library kernel this one follows (programmatic launch)
  griddep_launch_dependents();
  const int64_t total = T * h4;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t t = i / h4, c = i % h4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int32_t j = 0; j < k; ++j) {
      const float4 y = Yp[static_cast<int64_t>(pair_pos[t * k + j]) * h4 + c];
      acc.x += y.x;
      acc.y += y.y;
      acc.z += y.z;
      acc.w += y.w;
    }
    uint2 o;
    o.x = pack_bf16x2(acc.x, acc.y);
    o.y = pack_bf16x2(acc.z, acc.w);
    Y[i] = o;
  }
}

cudaError_t moe_finalize_launch(const float* Yp, const int32_t* pair_pos, int64_t T, int32_t k, int64_t H, void* Y,
                                cudaStream_t s, bool pdl) {
  if (T == 0) return cudaSuccess;
  const int64_t h4 = H / 4, total = T * h4;
  const int blocks = static_cast<int>(std::min<int64_t>((total + 255) / 256, 148 * 8));
  return launch_k(moe_finalize_kernel, dim3(blocks), dim3(256), 0, s, pdl, reinterpret_cast<const float4*>(Yp),
                  pair_pos, T, k, h4, reinterpret_cast<uint2*>(Y));
}

// ------------------------------------------- MoE block tail: add + RMSNorm
// One block per token t (Sec. IV-A: Fused Add + RMSNorm and MoE finalize of the
// gpt-oss decode path, fused): y = the token's MoE output (the fp32 accumulator,
// or in slot order the sum of its k per-row outputs), R_out = bf16(R + y) (the
// new residual stream), Y = bf16(R_out * rsqrt(mean(R_out^2) + eps) * gamma).
// Each thread keeps its (up to kArnMaxV) 4-column groups of R_out in registers
// between the sum of squares and the normalisation.  R may alias R_out.
constexpr int kArnThreads = 256;
constexpr int kArnMaxV = 8;  // H <= 4 * 256 * 8 = 8192
__global__ void __launch_bounds__(kArnThreads)
    moe_add_rmsnorm_kernel(const float4* __restrict__ yacc, const float4* __restrict__ yp,
                           const int32_t* __restrict__ pair_pos, int32_t k, int64_t h4, const uint2* R,
                           const uint2* __restrict__ gamma, float eps, uint2* R_out, uint2* __restrict__ Y) {
  griddep_wait();  // after the library kernel this one follows (programmatic launch)
  griddep_launch_dependents();
  const int64_t t = blockIdx.x;
  float4 hv[kArnMaxV];
  float ss = 0.0f;
#pragma unroll
  for (int v = 0; v < kArnMaxV; ++v) {
    const int64_t c = threadIdx.x + static_cast<int64_t>(v) * kArnThreads;
    if (c < h4) {
      float4 y;
      if (yacc) {
        y = yacc[t * h4 + c];
      } else {
        y = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int32_t j = 0; j < k; ++j) {
          const float4 q = yp[static_cast<int64_t>(pair_pos[t * k + j]) * h4 + c];
          y.x += q.x;
          y.y += q.y;
          y.z += q.z;
          y.w += q.w;
        }
      }
      const uint2 r = R[t * h4 + c];
      uint2 o;
      o.x = pack_bf16x2(bf16lo(r.x) + y.x, bf16hi(r.x) + y.y);
      o.y = pack_bf16x2(bf16lo(r.y) + y.z, bf16hi(r.y) + y.w);
      R_out[t * h4 + c] = o;
      const float4 h = make_float4(bf16lo(o.x), bf16hi(o.x), bf16lo(o.y), bf16hi(o.y));  // the stored residual
      hv[v] = h;
      ss += h.x * h.x + h.y * h.y + h.z * h.z + h.w * h.w;
    }
  }
  __shared__ float part[kArnThreads / 32];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = ss;
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = threadIdx.x < kArnThreads / 32 ? part[threadIdx.x] : 0.0f;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    if (threadIdx.x == 0) part[0] = v;
  }
  __syncthreads();
  const float inv = rsqrtf(part[0] / static_cast<float>(4 * h4) + eps);
#pragma unroll
  for (int v = 0; v < kArnMaxV; ++v) {
    const int64_t c = threadIdx.x + static_cast<int64_t>(v) * kArnThreads;
    if (c < h4) {
      const uint2 g = gamma[c];
      uint2 o;
      o.x = pack_bf16x2(hv[v].x * inv * bf16lo(g.x), hv[v].y * inv * bf16hi(g.x));
      o.y = pack_bf16x2(hv[v].z * inv * bf16lo(g.y), hv[v].w * inv * bf16hi(g.y));
      Y[t * h4 + c] = o;
    }
  }
}

cudaError_t moe_add_rmsnorm_launch(const float* yacc, const float* yp, const int32_t* pair_pos, int32_t k, int64_t T,
                                   int64_t H, const void* R, const void* gamma, float eps, void* R_out, void* Y,
                                   cudaStream_t s, bool pdl) {
  if (T == 0) return cudaSuccess;
  if (H % 4 != 0 || H / 4 > static_cast<int64_t>(kArnThreads) * kArnMaxV) return cudaErrorInvalidValue;
  return launch_k(moe_add_rmsnorm_kernel, dim3(static_cast<unsigned>(T)), dim3(kArnThreads), 0, s, pdl,
                  reinterpret_cast<const float4*>(yacc), reinterpret_cast<const float4*>(yp), pair_pos, k, H / 4,
                  reinterpret_cast<const uint2*>(R), reinterpret_cast<const uint2*>(gamma), eps,
                  reinterpret_cast<uint2*>(R_out), reinterpret_cast<uint2*>(Y));
}

// ----------------------------------------------------------------- row gather
// out[r, :] = A[idx[r], :] (16-byte vectors; K % 8 == 0 bf16).  An index out of
// range writes a zero row and sets the bounds bit of the error word.
__global__ void gather_rows_kernel(const uint4* __restrict__ A, int64_t lda_v, int64_t a_rows,
                                   const int32_t* __restrict__ idx, int64_t rows, int64_t kv,
                                   uint4* __restrict__ out, uint32_t* err, uint32_t* err_dev) {
  griddep_wait();  // after the library kernel this one follows (programmatic launch)
  griddep_launch_dependents();
  const int64_t total = rows * kv;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t r = i / kv, c = i % kv;
    const int32_t src = idx[r];
    uint4 v = make_uint4(0, 0, 0, 0);
    if (src >= 0 && src < a_rows)
      v = __ldg(A + src * lda_v + c);
    else if (c == 0)
      raise_err(err, err_dev, kErrBounds);
    out[i] = v;
  }
}

cudaError_t gather_rows_launch(const void* A, int64_t lda, int64_t a_rows, const int32_t* idx, int64_t rows,
                               int64_t K, void* out, uint32_t* err, uint32_t* err_dev, cudaStream_t s, bool pdl) {
  if (rows == 0) return cudaSuccess;
  const int64_t kv = K / 8, total = rows * kv;
  int blocks = static_cast<int>(std::min<int64_t>((total + 255) / 256, 148 * 16));
  return launch_k(gather_rows_kernel, dim3(blocks), dim3(256), 0, s, pdl, reinterpret_cast<const uint4*>(A), lda / 8,
                  a_rows, idx, rows, kv, reinterpret_cast<uint4*>(out), err, err_dev);
}

// ------------------------------------------------------------ fp32 -> bf16
__global__ void cvt_f32_bf16_kernel(const float4* __restrict__ in, uint2* __restrict__ out, int64_t n4) {
  griddep_wait();  // after the library kernel this one follows (programmatic launch)
  griddep_launch_dependents();
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n4;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const float4 f = in[i];
    uint2 o;
    o.x = pack_bf16x2(f.x, f.y);
    o.y = pack_bf16x2(f.z, f.w);
    out[i] = o;
  }
}
__global__ void cvt_f32_bf16_tail_kernel(const float* in, __nv_bfloat16* out, int64_t beg, int64_t n) {
  griddep_wait();  // after the library kernel this one follows (programmatic launch)
  griddep_launch_dependents();
  const int64_t i = beg + threadIdx.x;
  if (i < n) out[i] = __float2bfloat16_rn(in[i]);
}

cudaError_t cvt_f32_bf16_launch(const float* in, void* out, int64_t n, cudaStream_t s, bool pdl) {
  const int64_t n4 = n / 4;
  if (n4 > 0) {
    int blocks = static_cast<int>(std::min<int64_t>((n4 + 255) / 256, 148 * 8));
    cudaError_t e = launch_k(cvt_f32_bf16_kernel, dim3(blocks), dim3(256), 0, s, pdl,
                             reinterpret_cast<const float4*>(in), reinterpret_cast<uint2*>(out), n4);
    if (e != cudaSuccess) return e;
    pdl = true;  // the tail follows the main kernel
  }
  if (n % 4)
    return launch_k(cvt_f32_bf16_tail_kernel, dim3(1), dim3(4), 0, s, pdl, in,
                    reinterpret_cast<__nv_bfloat16*>(out), n4 * 4, n);
  return cudaSuccess;
}

}  // namespace kf
