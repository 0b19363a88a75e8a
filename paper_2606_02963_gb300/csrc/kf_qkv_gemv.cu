// kf_qkv_gemv.cu -- the QKV projection tail for up to eight tokens (decode),
// as a weight stream: bias + rotary embedding + key / value cache rows (the
// gpt-oss decode kernel "Bias + RoPE + KV update" of Sec. IV-A, here fused with
// its projection).
//
// With a few tokens the projection reads every weight once and each weight byte
// feeds one to eight multiply-adds: the time is HBM time, and HBM only streams
// at full rate with most of the matrix in flight at once (Little's law at a
// loaded latency of several microseconds).  So the rotation pairs of all heads
// (rows i and i + d/2 of a head; a pair's two rows and its bias, rotation and
// stores belong together) are dealt out in contiguous runs to one CTA per SM,
// and every CTA requests all of its weight rows into shared memory at once, one
// bulk copy per row: for gpt-oss-20b 17 pairs, 34 rows, 196 KB per SM, the whole
// 29.5 MB in flight.  The dot products run on the warp-level
// mma.sync.m16n8k16 (tokens as the 16-row operand, eight weight rows as the
// 8-column one): a tcgen05.mma costs the same whatever share of its 128 rows
// hold tokens (~160 SM cycles per K = 16 step at any N up to 256), which would
// make the tensor pipe, not HBM, the bound here, while the warp MMA costs a few
// instructions per 256 weights and reads plain row-major rows.  The bias, the
// rotation and the stores follow in the same CTA: no partial sums leave the SM,
// no cluster barrier, no second pass.
//
// Stages of 8 rows complete on their own mbarriers (the last stage of a CTA
// reads the last 8 rows, so it may repeat rows of the one before).  Compute
// warp w takes k-steps [w nks / 8, (w + 1) nks / 8) of every stage (nks = K / 16
// rounded up) with its tokens' fragments in registers and writes its fp32
// partial of the stage's 8 rows x tokens to shared memory; after the last stage
// the partials of the 8 warps are added in warp order (repeated calls are
// bitwise identical).
#include <algorithm>

#include "kf_internal.h"

namespace kf {
namespace {

constexpr int kGvCompute = 8;                      // compute warps
constexpr int kGvThreads = 32 * (kGvCompute + 1);  // + one producer warp
constexpr int kGvRows = 8;                         // weight rows per stage (the MMA's N)
constexpr int kGvMaxKs = 32;                       // k-steps of 16 per warp: K <= 4096
constexpr int kGvMaxPl = 4;                        // <= 128 rotation pairs per CTA

// Bulk copy of `bytes` (a multiple of 16; both addresses 16-byte aligned) from
// global memory into this CTA's shared memory, completing on `bar`.
__device__ __forceinline__ void bulk_copy_g2s(void* smem_dst, const void* gsrc, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(smem_dst)),
               "l"(reinterpret_cast<uint64_t>(gsrc)), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

// Four 8x8 16-bit matrices from shared memory (lane l addresses row l % 8 of
// matrix l / 8); r[i] is this lane's fragment of matrix i.
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}

// D (16 x 8, fp32) += A (16 x 16) B (16 x 8), 16-bit operands (bf16 or fp16).
template <bool F16>
__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  if constexpr (F16)
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
  else
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

template <bool F16>
__global__ void __launch_bounds__(kGvThreads, 1) kf_qkv_gemv_kernel(const __grid_constant__ QkvGemvParams g) {
  const QkvDecodeParams& p = g.q;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~uintptr_t(127));
  uint8_t* wrows = sm;                                                            // [buf_rows][stride]
  float2* red = reinterpret_cast<float2*>(wrows + static_cast<size_t>(g.buf_rows) * g.stride);  // [stages][warps][32]
  float4* eop = reinterpret_cast<float4*>(red + static_cast<size_t>(g.max_stages) * kGvCompute * 32);  // [T][pairs]
  uint64_t* full = reinterpret_cast<uint64_t*>(eop + static_cast<size_t>(kQkvGemvMaxT) * g.max_pairs);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(full + g.max_stages);
  volatile int* zero_flag = abort_flag + 1;
  int32_t* tok = const_cast<int32_t*>(reinterpret_cast<volatile int32_t*>(abort_flag + 2));  // [T][3]: pos, crow, ok

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // this CTA's rotation pairs: [pa, pb) of all heads' pairs
  const int32_t pa = static_cast<int32_t>(static_cast<int64_t>(blockIdx.x) * g.pairs / g.ctas);
  const int32_t pb = static_cast<int32_t>(static_cast<int64_t>(blockIdx.x + 1) * g.pairs / g.ctas);
  const int np = pb - pa;
  const int rows = 2 * np;  // local row r < np: pair pa + r's first row, else pair pa + r - np's second
  const int stages = (rows + kGvRows - 1) / kGvRows;
  // refuse any other launch shape before any barrier or copy
  if (blockDim.x != kGvThreads || gridDim.x != static_cast<uint32_t>(g.ctas) || gridDim.y != 1 || gridDim.z != 1 ||
      p.T < 1 || p.T > kQkvGemvMaxT || p.K > 16 * kGvMaxKs * kGvCompute || np < 1 || np > 32 * kGvMaxPl ||
      np > g.max_pairs || stages > g.max_stages || max(rows, kGvRows) > g.buf_rows) {
    if (threadIdx.x == 0) atomicOr(p.err, kErrLaunchShape);
    return;
  }
  const int d = p.rope_d, half = d >> 1;
  auto pair_col = [&](int32_t pr) -> int32_t { return (pr / half) * d + pr % half; };  // the pair's first column
  auto w_row = [&](int r) -> const uint8_t* {
    const int32_t n = r < np ? pair_col(pa + r) : pair_col(pa + r - np) + half;
    return static_cast<const uint8_t*>(g.W) + static_cast<int64_t>(n) * g.ldw * 2;
  };
  const uint32_t row_bytes = static_cast<uint32_t>(p.K) * 2;

  if (threadIdx.x == 0) {
    for (int i = 0; i < stages; ++i) mbar_init(&full[i], 1);
    *abort_flag = 0;
    *zero_flag = 0;
    fence_mbarrier_init();
  }
  // the row padding past K is read by the last k-steps: zero (the copies write
  // only the first 2K bytes of a row)
  {
    const int pad16 = (g.stride - static_cast<int>(row_bytes)) >> 4;
    for (int i = threadIdx.x; i < g.buf_rows * pad16; i += kGvThreads) {
      const int rr = i / pad16, j = i - rr * pad16;
      *reinterpret_cast<uint4*>(wrows + static_cast<size_t>(rr) * g.stride + row_bytes + 16 * j) = make_uint4(0, 0, 0, 0);
    }
  }
  __syncthreads();
  // launched as a programmatic dependent of the previous kernel in the stream:
  // wait for it before any operand, position or table is read
  griddep_wait();
  griddep_launch_dependents();

  if (warp == kGvCompute) {
    // ------------------------------------------------ producer: every row at once
    // (the token rows' positions and cache rows are requested first: the
    // epilogue operands below depend on them)
    int32_t tp = 0, tc = 0;
    if (lane < p.T) {
      tp = p.positions[lane];
      tc = p.cache_rows[lane];
    }
    if (lane == 0) {
      for (int s = 0; s < stages; ++s) {
        const int r0 = s * kGvRows, r1 = min(rows, r0 + kGvRows);
        mbar_arrive_expect_tx(&full[s], static_cast<uint32_t>(r1 - r0) * row_bytes);
        for (int r = r0; r < r1; ++r)
          bulk_copy_g2s(wrows + static_cast<size_t>(r) * g.stride, w_row(r), row_bytes, &full[s]);
      }
    }
    // then, while the weights stream, the epilogue operands: per token its
    // position and cache row, per (token, pair) the bias pair and the table
    // entries of the rotation.  Behind the copies in the memory queues these
    // loads take about as long as the stream, so each lane issues all of its
    // items' loads before it uses any.
    int32_t tk = 0;
    if (lane < p.T) {
      tk = (tp >= 0 && tp < p.max_pos && tc >= 0 && tc < p.rows) ? 1 : 0;
      tok[3 * lane] = tp;
      tok[3 * lane + 1] = tc;
      tok[3 * lane + 2] = tk;
    }
    constexpr int kIt = 8;  // items per lane per round
    for (int base = 0; base < p.T * np; base += 32 * kIt) {
      float4 e[kIt];
#pragma unroll
      for (int u = 0; u < kIt; ++u) {
        const int it = base + lane + 32 * u;
        const int t = it / np, lp = it - t * np;
        const int32_t pos = __shfl_sync(0xffffffffu, tp, t & 31);
        const int ok = __shfl_sync(0xffffffffu, tk, t & 31);
        e[u] = make_float4(0.0f, 0.0f, 1.0f, 0.0f);
        if (it < p.T * np) {
          const int32_t c0 = pair_col(pa + lp);
          const bool rot = ok && c0 < p.rot_cols;
          const int i = (pa + lp) % half;
          if (p.bias) {
            e[u].x = ld_elem(p.bias, p.bias_dtype, c0);
            e[u].y = ld_elem(p.bias, p.bias_dtype, c0 + half);
          }
          if (rot) {
            e[u].z = __ldg(p.cos_t + static_cast<int64_t>(pos) * half + i);
            e[u].w = __ldg(p.sin_t + static_cast<int64_t>(pos) * half + i);
          }
        }
      }
#pragma unroll
      for (int u = 0; u < kIt; ++u) {
        const int it = base + lane + 32 * u;
        if (it < p.T * np) eop[(it / np) * g.max_pairs + it % np] = e[u];
      }
    }
  } else {
    // ----------------------------------------------------------------- compute
    // token fragments of this warp's k-steps (A of the MMA: row = token g =
    // lane / 4, k pairs 2 (lane % 4) and 2 (lane % 4) + 8; tokens past T and k
    // past K are zero)
    const int nks = (p.K + 15) >> 4;
    const int ks0 = warp * nks / kGvCompute, ks1 = (warp + 1) * nks / kGvCompute;
    const int tg = lane >> 2, tq = lane & 3;
    uint32_t xa[kGvMaxKs][2];
#pragma unroll
    for (int j = 0; j < kGvMaxKs; ++j) {
      xa[j][0] = 0u;
      xa[j][1] = 0u;
      const int k = 16 * (ks0 + j) + 2 * tq;
      if (ks0 + j < ks1 && tg < p.T) {
        const uint32_t* xr = reinterpret_cast<const uint32_t*>(static_cast<const uint8_t*>(g.X) +
                                                               static_cast<int64_t>(tg) * g.ldx * 2);
        if (k < p.K) xa[j][0] = __ldg(xr + (k >> 1));
        if (k + 8 < p.K) xa[j][1] = __ldg(xr + ((k + 8) >> 1));
      }
    }
    // ldmatrix rows: lane l reads row l % 8 of the stage, k-step (l / 8) / 2 of
    // the pair of k-steps, half (l / 8) % 2
    const uint32_t lrow = static_cast<uint32_t>(lane & 7) * static_cast<uint32_t>(g.stride);
    const uint32_t lcol = static_cast<uint32_t>(((lane >> 3) >> 1) * 32 + ((lane >> 3) & 1) * 16);
    const uint32_t base0 = smem_u32(wrows) + lrow + lcol + static_cast<uint32_t>(ks0) * 32u;
    for (int s = 0; s < stages; ++s) {
      bool got = mbar_wait(&full[s], 0u, abort_flag, p.wait_ns);
      got = __all_sync(0xffffffffu, got);  // the warp leaves the loop together
      if (!got) {
        if (lane == 0) {
          *abort_flag = 1;
          atomicOr(p.err, kErrWaitEpilogue);
        }
        break;
      }
      const int r0 = max(0, min(s * kGvRows, rows - kGvRows));  // the stage's 8 rows
      const uint32_t base = base0 + static_cast<uint32_t>(r0) * static_cast<uint32_t>(g.stride);
      float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
      for (int j = 0; j < kGvMaxKs; j += 2) {
        if (ks0 + j < ks1) {
          uint32_t b[4];
          ldsm_x4(base + static_cast<uint32_t>(j) * 32u, b);  // k-steps j and j + 1 (zero padding past K)
          mma16816<F16>(acc, xa[j][0], 0u, xa[j][1], 0u, b[0], b[1]);
          if (ks0 + j + 1 < ks1) mma16816<F16>(acc, xa[j + 1][0], 0u, xa[j + 1][1], 0u, b[2], b[3]);
        }
      }
      // D: token lane / 4, rows r0 + 2 (lane % 4) and r0 + 2 (lane % 4) + 1
      red[(static_cast<size_t>(s) * kGvCompute + warp) * 32 + lane] = make_float2(acc[0], acc[1]);
    }
  }
  __syncthreads();
  if (*abort_flag) {
    // after a timeout: the copies land (bounded) before the CTA exits
    if (warp == kGvCompute && lane == 0)
      for (int s = 0; s < stages; ++s) mbar_wait(&full[s], 0u, zero_flag, p.drain_ns);
    return;
  }
  const int t = warp;
  if (t >= p.T) return;

  // --------------------------- bias, rotation and stores of token `warp`
  if (!tok[3 * t + 2]) {
    if (lane == 0) atomicOr(p.err, kErrBounds);
    return;
  }
  const int32_t crow = tok[3 * t + 1];
  // y of local row r for token t: the 8 warps' partials, in warp order
  auto y_of = [&](int r) -> float {
    const int s = min(r / kGvRows, stages - 1);
    const int rr = r - max(0, min(s * kGvRows, rows - kGvRows));
    const float2* q = red + static_cast<size_t>(s) * kGvCompute * 32 + t * 4 + (rr >> 1);
    float v = 0.0f;
#pragma unroll
    for (int w = 0; w < kGvCompute; ++w) {
      const float2 x = q[w * 32];
      v += (rr & 1) ? x.y : x.x;
    }
    return v;
  };
#pragma unroll
  for (int m = 0; m < kGvMaxPl; ++m) {
    const int lp = lane + 32 * m;
    if (lp >= np) break;
    const int32_t c0 = pair_col(pa + lp);
    const float4 e = eop[t * g.max_pairs + lp];
    float x0 = y_of(lp) + e.x, x1 = y_of(np + lp) + e.y;
    if (c0 < p.rot_cols) {
      const float y0 = fmaf(x0, e.z, -x1 * e.w), y1 = fmaf(x1, e.z, x0 * e.w);
      x0 = y0;
      x1 = y1;
    }
    void* dst;
    int64_t o;
    if (c0 < p.q_cols) {
      dst = p.q_out;
      o = static_cast<int64_t>(t) * p.ldq + c0;
    } else {
      dst = c0 < p.rot_cols ? p.k_cache : p.v_cache;
      o = static_cast<int64_t>(crow) * p.ld_cache + c0 - (c0 < p.rot_cols ? p.q_cols : p.rot_cols);
    }
    if (p.out_dtype == KF_F32) {
      reinterpret_cast<float*>(dst)[o] = x0;
      reinterpret_cast<float*>(dst)[o + half] = x1;
    } else if (p.out_dtype == KF_BF16) {
      reinterpret_cast<__nv_bfloat16*>(dst)[o] = __float2bfloat16_rn(x0);
      reinterpret_cast<__nv_bfloat16*>(dst)[o + half] = __float2bfloat16_rn(x1);
    } else {
      reinterpret_cast<__half*>(dst)[o] = __float2half_rn(x0);
      reinterpret_cast<__half*>(dst)[o + half] = __float2half_rn(x1);
    }
  }
}

template <bool F16>
cudaError_t launch_gv(const QkvGemvParams& g, size_t smem, cudaStream_t s) {
  auto kern = kf_qkv_gemv_kernel<F16>;
  // the attribute is per device; the largest request so far is remembered
  static std::atomic<size_t> configured[64];
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (configured[dev] < smem) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    configured[dev] = smem;
  }
  return launch_k(kern, dim3(g.ctas), dim3(kGvThreads), smem, s, true, g);
}

}  // namespace

bool qkv_gemv_plan(int64_t T, int64_t H, int32_t heads, int32_t d, int nsm, QkvGemvParams* g, size_t* smem) {
  if (T < 1 || T > kQkvGemvMaxT || H < 8 || H % 8 != 0 || H > 16 * kGvMaxKs * kGvCompute || d < 64 || d % 64 != 0 ||
      d > 256 || nsm < 1)
    return false;
  const int64_t pairs = static_cast<int64_t>(heads) * (d / 2);
  const int64_t ctas = std::min<int64_t>(nsm, pairs);
  const int64_t np_max = (pairs + ctas - 1) / ctas;
  if (np_max > 32 * kGvMaxPl) return false;
  const int64_t rows_max = 2 * np_max;
  const int64_t max_stages = (rows_max + kGvRows - 1) / kGvRows;
  // row stride: the 2H bytes and the k-step an ldmatrix may read past the last
  // one (32 bytes, zero), rounded up to 128, + 16, so that the rows of an
  // ldmatrix start 4 banks apart
  const int64_t stride = (H * 2 + 32 + 127) / 128 * 128 + 16;
  const int64_t buf_rows = std::max<int64_t>(rows_max, kGvRows);
  const int64_t bytes = 128 + buf_rows * stride + max_stages * (kGvCompute * 32 * 8 + 8) +
                        static_cast<int64_t>(kQkvGemvMaxT) * np_max * 16 + 16 + 4 * 3 * kQkvGemvMaxT + 64;
  if (bytes > 232448) return false;  // the CTA's rows do not fit at once
  g->ctas = static_cast<int32_t>(ctas);
  g->pairs = static_cast<int32_t>(pairs);
  g->max_stages = static_cast<int32_t>(max_stages);
  g->max_pairs = static_cast<int32_t>(np_max);
  g->buf_rows = static_cast<int32_t>(buf_rows);
  g->stride = static_cast<int32_t>(stride);
  *smem = static_cast<size_t>(bytes);
  return true;
}

cudaError_t qkv_gemv_launch(const QkvGemvParams& g, size_t smem, cudaStream_t s) {
  if (g.q.T < 1 || g.q.T > kQkvGemvMaxT) return cudaErrorInvalidValue;
  return g.q.ab_f16 ? launch_gv<true>(g, smem, s) : launch_gv<false>(g, smem, s);
}

}  // namespace kf
