// kf_common.cuh -- device-side structures shared by the kernels: the decoded
// epilogue op list, the tcgen05 GEMM parameter block, and the register-level
// tail-op interpreter that applies the chain to 32 accumulator columns of one
// row (Sec. IV-B: the post-GEMM op chain is applied to the matmul result while it
// is still on chip, in fp32).
#pragma once
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cstdint>

#include "../../include/kf.h"
#include "kf_ptx.cuh"

namespace kf {

constexpr int kMaxOps = 8;
constexpr int kMaxGroups = 512;   // grouped GEMM: row groups (experts)

// error-word bits
constexpr uint32_t kErrWaitProducer = 1u;
constexpr uint32_t kErrWaitMma = 2u;
constexpr uint32_t kErrWaitEpilogue = 4u;
constexpr uint32_t kErrBounds = 8u;
constexpr uint32_t kErrLaunchShape = 16u;  // grid or cluster shape not the variant's

// Record error bits in the call's error word and in the device-wide word (the
// same word when the call has no workspace).
__device__ __forceinline__ void raise_err(uint32_t* call_word, uint32_t* dev_word, uint32_t bits) {
  atomicOr(call_word, bits);
  if (dev_word != nullptr && dev_word != call_word) atomicOr(dev_word, bits);
}

struct DevOp {
  int32_t kind;
  float scalar;
  float eps;
  int32_t groups;   // GROUPNORM: group size in columns (not the count)
  const void* p0;
  const void* p1;
  int32_t p_dtype;
  int32_t vec_ok;   // p0 (and p1) allow 16-byte vector access for 32-column chunks
  int64_t ld;
};

// Modes of the tcgen05 GEMM kernel (what its epilogue does with a tile).
enum TcMode : int {
  kModeStore = 0,    // chain of element-wise ops -> store C tile
  kModeLse = 1,      // element-wise pre-ops -> per-tile row (max, sum exp) partials
  kModeGroupNorm = 2,// pre-ops -> GroupNorm -> post-ops -> store
  kModeSwiglu = 3,   // gate/up halves -> silu(g) * u -> post-ops -> store
  kModeScatter = 4,  // chain -> * row scale -> atomic add into C[dst row]
  kModeRope = 5,     // QKV projection: chain (bias) -> rotary embedding of query / key
                     // heads -> queries to C[row], keys / values to cache row row_dst[row]
};

struct TcParams {
  int32_t M;            // dense: rows of X;  grouped: rows_total
  int32_t N;            // output columns
  int32_t K;
  int32_t tiles_m;      // dense only
  int32_t tiles_n;      // output-column tiles (units for GroupNorm)
  int32_t num_kb;       // K blocks of 64
  int32_t total_units;  // dense: number of work units (tiles or GN units)
  int32_t G;            // grouped: number of groups (0 = dense)
  const int32_t* group_offsets;
  int32_t b_rows;       // grouped: rows of B per group used for the N offset of up rows (= N)
  int32_t n_pre;        // ops applied before the reduction / norm / store
  int32_t n_post;       // ops applied after it
  DevOp pre[kMaxOps];
  DevOp post[kMaxOps];
  DevOp norm;           // GROUPNORM op (group size in .groups)
  void* C;
  int64_t ldc;
  int32_t c_dtype;
  int32_t c_vec_ok;
  float2* lse_part;     // [M x tiles_n] (max, sum exp) partials
  const float* row_scale;   // scatter
  const int32_t* row_dst;   // scatter
  int32_t dst_rows;         // scatter: rows of C (bounds)
  uint32_t* err;        // error word of the call: its workspace's header, else the device word
  uint32_t* err_dev;    // the per-device error word (also written, for the device-wide view)
  uint64_t wait_ns;
  uint64_t drain_ns;
  // row sum instead of a row log-sum-exp (kModeLse), or after the GroupNorm's
  // post chain (kModeGroupNorm): per-tile row partials go to lse_part, red_parts
  // per row (kModeGroupNorm: one per 256-column block), nothing else is stored
  int32_t red_sum;
  int32_t red_parts;
  int32_t fast;         // reduced-precision activations (result stored as bf16)
  int32_t res_op;       // index in pre[] of a bf16 RESIDUAL_ADD staged by coalesced loads, or -1
  int32_t vec_op;       // index in pre[] of a bf16 BIAS / MUL whose vector is loaded ahead, or -1
  int32_t c_tma;        // output tiles leave through TMA stores (dense, bf16, aligned)
  int32_t ab_f16;       // A and B are fp16 (else bf16): the MMA's operand format
  // GroupNorm on couples of CTA pairs: per-row statistics exchanged through
  // global memory (workspace) -- [couples][2 slots][2 halves][256 rows] float2,
  // then [couples][2 slots][2 halves][8 row blocks] uint64 flags tagged with
  // (epoch << 32 | tile sequence + 1)
  float2* gx_data;
  unsigned long long* gx_flag;
  uint32_t gx_epoch;
  int32_t gx_couples;
  // QKV tail: heads of rope_d columns; columns [0, rope_q_cols) are queries,
  // [rope_q_cols, rope_rot_cols) keys (both rotated), the rest values.  Row r
  // turns by the angles of table row rope_pos[r] (cos / sin fp32 [rope_max_pos x
  // rope_d / 2]); its keys and values go to row row_dst[r] of k_cache / v_cache
  // (row stride ld_cache, dst_rows rows, element type c_dtype).
  const float* rope_cos;
  const float* rope_sin;
  const int32_t* rope_pos;
  int32_t rope_max_pos;
  int32_t rope_d;
  int32_t rope_q_cols;
  int32_t rope_rot_cols;
  void* k_cache;
  void* v_cache;
  int64_t ld_cache;
  int32_t kv_vec_ok;    // caches allow 16-byte stores of 32-column chunks
  // grouped GEMMs: bf16 bias of the unit's group added to the accumulator
  // before anything else (column j of group g at gbias[g * gbias_ld + j]; for
  // SwiGLU the up half's bias follows at + b_rows), or null
  const void* gbias;
  int64_t gbias_ld;
  // SwiGLU with the gated-expert extension (sw_ext != 0): h = g' sigmoid(sw_alpha
  // g') (u' + sw_c), g' = min(g, sw_limit), u' = clamp(u, -sw_limit, sw_limit)
  // when sw_limit > 0; otherwise the plain silu(g) * u
  int32_t sw_ext;
  float sw_alpha;
  float sw_limit;
  float sw_c;
  // grouped SwiGLU (the MoE gate/up GEMM): zero_bytes (a multiple of 16) at
  // zero_ptr are cleared by the epilogue warps while the first unit's mainloop
  // runs -- the down GEMM's fp32 scatter target, which that GEMM only touches
  // after this grid has completed
  void* zero_ptr;
  int64_t zero_bytes;
};

// ---------------------------------------------------------------- loads/stores
// One element's raw bits (a 32-bit load for fp32, a 16-bit load for bf16 / fp16:
// predicated, no branch) and their conversion, kept apart so that a run of loads
// issues back to back before any conversion waits on one.
__device__ __forceinline__ uint32_t ld_raw(const void* p, int dt, int64_t i) {
  return dt == KF_F32 ? reinterpret_cast<const uint32_t*>(p)[i]
                      : static_cast<uint32_t>(reinterpret_cast<const uint16_t*>(p)[i]);
}
__device__ __forceinline__ float cvt_raw(uint32_t b, int dt) {
  if (dt == KF_F32) return __uint_as_float(b);
  if (dt == KF_BF16) return __uint_as_float(b << 16);
  return __half2float(__ushort_as_half(static_cast<unsigned short>(b)));
}
__device__ __forceinline__ float ld_elem(const void* p, int dt, int64_t i) { return cvt_raw(ld_raw(p, dt, i), dt); }
__device__ __forceinline__ float2 f16x2_to_f2(uint32_t w) {
  return __half22float2(*reinterpret_cast<const __half2*>(&w));
}
__device__ __forceinline__ uint32_t pack_f16x2(float a, float b) {
  __half2 h = __floats2half2_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

// Load 32 consecutive elements starting at element index i0 (first `nvalid`
// are in bounds; the rest read as 0).  Vector path when the whole chunk is in
// bounds and the caller guaranteed 16-byte alignment.
__device__ __forceinline__ void ld32(const void* p, int dt, int64_t i0, int nvalid, bool vec_ok, float (&o)[32]) {
  if (nvalid >= 32 && vec_ok) {
    if (dt == KF_BF16) {
      const uint4* q = reinterpret_cast<const uint4*>(reinterpret_cast<const __nv_bfloat16*>(p) + i0);
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        uint4 u = __ldg(q + v);
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int h = 0; h < 4; ++h) {
          o[v * 8 + 2 * h] = __uint_as_float(w[h] << 16);
          o[v * 8 + 2 * h + 1] = __uint_as_float(w[h] & 0xFFFF0000u);
        }
      }
    } else if (dt == KF_F16) {
      const uint4* q = reinterpret_cast<const uint4*>(reinterpret_cast<const __half*>(p) + i0);
#pragma unroll
      for (int v = 0; v < 4; ++v) {
        uint4 u = __ldg(q + v);
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int h = 0; h < 4; ++h) {
          const float2 f = f16x2_to_f2(w[h]);
          o[v * 8 + 2 * h] = f.x;
          o[v * 8 + 2 * h + 1] = f.y;
        }
      }
    } else {
      const float4* q = reinterpret_cast<const float4*>(reinterpret_cast<const float*>(p) + i0);
#pragma unroll
      for (int v = 0; v < 8; ++v) {
        float4 f = __ldg(q + v);
        o[4 * v] = f.x;
        o[4 * v + 1] = f.y;
        o[4 * v + 2] = f.z;
        o[4 * v + 3] = f.w;
      }
    }
  } else {
#pragma unroll
    for (int j = 0; j < 32; ++j) o[j] = (j < nvalid) ? ld_elem(p, dt, i0 + j) : 0.0f;
  }
}

// 8 consecutive elements (16-byte vector loads when vec_ok; all in bounds).
__device__ __forceinline__ void ld8(const void* p, int dt, int64_t i0, bool vec_ok, float (&o)[8]) {
  if (vec_ok && dt == KF_BF16) {
    uint4 u = __ldg(reinterpret_cast<const uint4*>(reinterpret_cast<const __nv_bfloat16*>(p) + i0));
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int h = 0; h < 4; ++h) {
      o[2 * h] = __uint_as_float(w[h] << 16);
      o[2 * h + 1] = __uint_as_float(w[h] & 0xFFFF0000u);
    }
  } else if (vec_ok && dt == KF_F16) {
    uint4 u = __ldg(reinterpret_cast<const uint4*>(reinterpret_cast<const __half*>(p) + i0));
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int h = 0; h < 4; ++h) {
      const float2 f = f16x2_to_f2(w[h]);
      o[2 * h] = f.x;
      o[2 * h + 1] = f.y;
    }
  } else if (vec_ok) {
    const float4* q = reinterpret_cast<const float4*>(reinterpret_cast<const float*>(p) + i0);
    const float4 a = __ldg(q), b = __ldg(q + 1);
    o[0] = a.x; o[1] = a.y; o[2] = a.z; o[3] = a.w;
    o[4] = b.x; o[5] = b.y; o[6] = b.z; o[7] = b.w;
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j) o[j] = ld_elem(p, dt, i0 + j);
  }
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

__device__ __forceinline__ void st32(void* p, int dt, int64_t i0, int nvalid, bool vec_ok, const float (&v)[32]) {
  if (nvalid >= 32 && vec_ok) {
    if (dt == KF_BF16) {
      uint4* q = reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(p) + i0);
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        uint4 u;
        u.x = pack_bf16x2(v[8 * c + 0], v[8 * c + 1]);
        u.y = pack_bf16x2(v[8 * c + 2], v[8 * c + 3]);
        u.z = pack_bf16x2(v[8 * c + 4], v[8 * c + 5]);
        u.w = pack_bf16x2(v[8 * c + 6], v[8 * c + 7]);
        q[c] = u;
      }
    } else if (dt == KF_F16) {
      uint4* q = reinterpret_cast<uint4*>(reinterpret_cast<__half*>(p) + i0);
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        uint4 u;
        u.x = pack_f16x2(v[8 * c + 0], v[8 * c + 1]);
        u.y = pack_f16x2(v[8 * c + 2], v[8 * c + 3]);
        u.z = pack_f16x2(v[8 * c + 4], v[8 * c + 5]);
        u.w = pack_f16x2(v[8 * c + 6], v[8 * c + 7]);
        q[c] = u;
      }
    } else {
      float4* q = reinterpret_cast<float4*>(reinterpret_cast<float*>(p) + i0);
#pragma unroll
      for (int c = 0; c < 8; ++c) q[c] = make_float4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
    }
  } else {
    if (dt == KF_BF16) {
      __nv_bfloat16* q = reinterpret_cast<__nv_bfloat16*>(p) + i0;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (j < nvalid) q[j] = __float2bfloat16_rn(v[j]);
    } else if (dt == KF_F16) {
      __half* q = reinterpret_cast<__half*>(p) + i0;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (j < nvalid) q[j] = __float2half_rn(v[j]);
    } else {
      float* q = reinterpret_cast<float*>(p) + i0;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (j < nvalid) q[j] = v[j];
    }
  }
}

// ------------------------------------------- warp-cooperative 32x32 bf16 tiles
// A warp owns 32 rows (one per lane) x 32 columns.  Global traffic is made
// coalesced by passing the tile through a 1 KB shared buffer, 16 columns (32 B
// per row) at a time: for global accesses lane t handles 16 bytes of row
// 16i + t/2 (two lanes per 32-byte row segment, one full sector); for
// registers lane r owns row r.  The 16-byte unit u of row r is stored at unit
// u ^ ((r >> 2) & 1) of that row, which makes both access patterns free of
// shared-memory bank conflicts.
__device__ __forceinline__ uint32_t xpose_off(int row, int unit) {
  return static_cast<uint32_t>(row * 32 + ((unit ^ ((row >> 2) & 1)) << 4));
}
// 64-byte-swizzled block of 32 bf16 columns (64 B per row): the 16-byte unit u
// of row r sits at unit u ^ ((r >> 1) & 3), the layout TMA's SWIZZLE_64B mode
// reads and writes.  One row per lane: each 16-byte access of a warp touches
// every bank group once per 8 rows (no conflicts beyond the 4 wavefronts that
// 512 bytes need).
__device__ __forceinline__ uint32_t sw64_off(int row, int unit) {
  return static_cast<uint32_t>(row * 64 + ((unit ^ ((row >> 1) & 3)) << 4));
}

// Store the lane's 32 values (row `lane`) as bf16 to rows [0, rows) of the
// 32 x 32 block at `gbase` (row stride ld elements).
__device__ __forceinline__ void store_tile32_bf16(uint8_t* stage, int lane, const float (&v)[32], void* gbase,
                                                  int64_t ld, int rows) {
  const int u = lane & 1;
#pragma unroll
  for (int half = 0; half < 2; ++half) {
#pragma unroll
    for (int uu = 0; uu < 2; ++uu) {
      const int c = 16 * half + 8 * uu;
      uint4 w;
      w.x = pack_bf16x2(v[c + 0], v[c + 1]);
      w.y = pack_bf16x2(v[c + 2], v[c + 3]);
      w.z = pack_bf16x2(v[c + 4], v[c + 5]);
      w.w = pack_bf16x2(v[c + 6], v[c + 7]);
      *reinterpret_cast<uint4*>(stage + xpose_off(lane, uu)) = w;
    }
    __syncwarp();
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int r = 16 * i + (lane >> 1);
      const uint4 w = *reinterpret_cast<const uint4*>(stage + xpose_off(r, u));
      if (r < rows)
        *reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(gbase) + r * ld + 16 * half + 8 * u) = w;
    }
    __syncwarp();
  }
}

// Store the lane's 32 values (row `lane`) as bf16 through TMA: each 16-column
// half goes into one of the warp's two 1 KB buffers (the 32-byte-swizzle layout
// of xpose_off, which is what the tensor map's SWIZZLE_32B expects) and leaves
// as a {16 x 32} box at (x + 16*half, y).  Rows/columns outside the tensor are
// clipped by TMA.  A buffer is rewritten only after the store that last read it
// has finished reading (at most one other group in flight).
__device__ __forceinline__ void store_tile32_tma(uint8_t* stage2, int lane, const float (&v)[32], const CUtensorMap* map,
                                                 int32_t x, int32_t y) {
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    uint8_t* buf = stage2 + half * 1024;
    if (lane == 0) bulk_wait_group_read<1>();
    __syncwarp();
#pragma unroll
    for (int uu = 0; uu < 2; ++uu) {
      const int c = 16 * half + 8 * uu;
      uint4 w;
      w.x = pack_bf16x2(v[c + 0], v[c + 1]);
      w.y = pack_bf16x2(v[c + 2], v[c + 3]);
      w.z = pack_bf16x2(v[c + 4], v[c + 5]);
      w.w = pack_bf16x2(v[c + 6], v[c + 7]);
      *reinterpret_cast<uint4*>(buf + xpose_off(lane, uu)) = w;
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      tma_store_2d(map, buf, x + 16 * half, y);
      bulk_commit_group();
    }
  }
}

// 16-byte read-only load issued where it is written: volatile, so the compiler
// cannot sink it past the accumulator wait that follows (the point of issuing
// it early is to overlap its latency with that wait).
__device__ __forceinline__ uint4 ldg_v4_pinned(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(reinterpret_cast<uint64_t>(p)));
  return r;
}

// Issue the coalesced loads of rows [0, rows) of a 32 x 32 bf16 block into
// registers: q[2*half + i] is 16 bytes of row 16i + t/2, columns
// 16*half + 8*(t&1) ..; rows >= `rows` read as 0.
__device__ __forceinline__ void tile32_issue(const void* gbase, int64_t ld, int rows, int lane, uint4 (&q)[4]) {
  const int u = lane & 1;
#pragma unroll
  for (int half = 0; half < 2; ++half)
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int r = 16 * i + (lane >> 1);
      q[2 * half + i] = make_uint4(0, 0, 0, 0);
      if (r < rows)
        q[2 * half + i] = ldg_v4_pinned(reinterpret_cast<const __nv_bfloat16*>(gbase) + r * ld + 16 * half + 8 * u);
    }
}
// Pass loaded blocks through the shared buffer; row `lane` comes back as 16
// packed bf16 pairs (element 2k in the low half of o[k]).
__device__ __forceinline__ void tile32_finish(uint8_t* stage, int lane, const uint4 (&q)[4], uint32_t (&o)[16]) {
  const int u = lane & 1;
#pragma unroll
  for (int half = 0; half < 2; ++half) {
#pragma unroll
    for (int i = 0; i < 2; ++i)
      *reinterpret_cast<uint4*>(stage + xpose_off(16 * i + (lane >> 1), u)) = q[2 * half + i];
    __syncwarp();
#pragma unroll
    for (int uu = 0; uu < 2; ++uu) {
      const uint4 w = *reinterpret_cast<const uint4*>(stage + xpose_off(lane, uu));
      o[8 * half + 4 * uu] = w.x;
      o[8 * half + 4 * uu + 1] = w.y;
      o[8 * half + 4 * uu + 2] = w.z;
      o[8 * half + 4 * uu + 3] = w.w;
    }
    __syncwarp();
  }
}
__device__ __forceinline__ float bf16lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
// 32 consecutive bf16 of a per-column vector (same for every lane)
__device__ __forceinline__ void vec32_issue(const void* p, int64_t i0, uint4 (&q)[4]) {
  const __nv_bfloat16* a = reinterpret_cast<const __nv_bfloat16*>(p) + i0;
#pragma unroll
  for (int i = 0; i < 4; ++i) q[i] = ldg_v4_pinned(a + 8 * i);
}
__device__ __forceinline__ void pack16(const uint4 (&q)[4], uint32_t (&o)[16]) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    o[4 * i] = q[i].x;
    o[4 * i + 1] = q[i].y;
    o[4 * i + 2] = q[i].z;
    o[4 * i + 3] = q[i].w;
  }
}

// Operands of one 32-column chunk that the caller loaded ahead of time: the
// row's residual chunk (for pre[res_op]) and a per-column vector (for pre[vec_op]).
struct Staged32 {
  uint32_t res[16];  // packed bf16 pairs
  uint32_t vec[16];  // packed bf16 pairs
  bool use_res;
  int vec_idx;  // op index whose operand is vec[], or -1
};

// ------------------------------------------------------------ element-wise ops
// The accurate forms (fp32 results) are kept out of line: the op interpreter is
// unrolled over 32 columns at several call sites, and inlining the library
// transcendentals there would multiply the kernel's code size.
static __device__ __noinline__ float f_sigmoid(float x) { return 1.0f / (1.0f + expf(-x)); }
static __device__ __noinline__ float f_gelu_tanh(float x) {
  const float c = 0.7978845608028654f;  // sqrt(2/pi)
  return 0.5f * x * (1.0f + tanhf(c * (x + 0.044715f * x * x * x)));
}
static __device__ __noinline__ float f_mish(float x) {
  float sp = x > 20.0f ? x : log1pf(expf(x));
  return x * tanhf(sp);
}

// Reduced-precision forms, used only when the result is rounded to bf16 (8
// significant bits): the hardware tanh (tanh.approx.f32, relative error about
// 2^-11) and sigmoid(x) = (1 + tanh(x/2)) / 2.
__device__ __forceinline__ float tanh_fast(float x) {
  float y;
  asm("tanh.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float f_sigmoid_fast(float x) { return fmaf(0.5f, tanh_fast(0.5f * x), 0.5f); }
// Two tanh values with one instruction (tanh.approx.f16x2: relative error about
// 2^-11, inputs rounded to fp16; |arguments| beyond the fp16 range saturate to
// +-1, which is tanh's value there to fp16 precision).
__device__ __forceinline__ void tanh2_fast(float a, float b, float& ta, float& tb) {
  uint32_t hin, hout;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(hin) : "f"(b), "f"(a));
  asm("tanh.approx.f16x2 %0, %1;" : "=r"(hout) : "r"(hin));
  const __half2 h2 = *reinterpret_cast<const __half2*>(&hout);
  ta = __low2float(h2);
  tb = __high2float(h2);
}
// GELU_tanh of two values in packed half precision, for results stored as
// bf16: g = h + h tanh(x (c0 + c1 x^2)), h = x / 2, c0 = sqrt(2/pi),
// c1 = 0.044715 c0 -- each step one f16x2 instruction.  f16 keeps 11
// significant bits (bf16 keeps 8).  Past |x| ~ 150 the tanh argument overflows
// to +-inf and tanh saturates at +-1, which is the function's limit.
// Inputs beyond fp16's range: the conversion saturates to +-65504 (never
// +-inf, so x < -65504 gives h + h * (-1) = 0, not inf - inf), and the result
// is max(g, x - 1/2): x - gelu(x) lies in [0, 0.17] for x >= 0 and x - 1/2 <
// gelu(x) for x < 0, so below 65504 this keeps g, and above it (where g stops
// at 65504) it gives x - 1/2, which bf16 cannot tell from gelu(x) = x.
__device__ __forceinline__ void gelu2_f16(float& a, float& b) {
  uint32_t x, g;
  asm("cvt.rn.satfinite.f16x2.f32 %0, %1, %2;" : "=r"(x) : "f"(b), "f"(a));
  asm("{\n\t.reg .b32 u, p, q, t, h;\n\t"
      "mul.rn.f16x2 u, %1, %1;\n\t"
      "fma.rn.f16x2 p, u, %2, %3;\n\t"
      "mul.rn.f16x2 q, %1, p;\n\t"
      "tanh.approx.f16x2 t, q;\n\t"
      "mul.rn.f16x2 h, %1, %4;\n\t"
      "fma.rn.f16x2 %0, h, t, h;\n\t}"
      : "=r"(g)
      : "r"(x), "r"(0x28912891u), "r"(0x3a623a62u), "r"(0x38003800u));  // c1, c0, 1/2 (f16 pairs)
  const __half2 h2 = *reinterpret_cast<const __half2*>(&g);
  a = fmaxf(__low2float(h2), a - 0.5f);
  b = fmaxf(__high2float(h2), b - 0.5f);
}
__device__ __forceinline__ float f_gelu_tanh_fast(float x) {
  const float c = 0.7978845608028654f;
  const float hx = 0.5f * x;
  return fmaf(hx, tanh_fast(c * fmaf(0.044715f * x, x * x, x)), hx);
}
static __device__ __noinline__ float f_mish_fast(float x) {
  float sp = x > 15.0f ? x : __logf(1.0f + __expf(x));
  return x * tanh_fast(sp);
}

template <bool FAST>
__device__ __forceinline__ float sigm(float x) { return FAST ? f_sigmoid_fast(x) : f_sigmoid(x); }

__device__ __forceinline__ float apply_scalar_op(const DevOp& op, float x) {
  switch (op.kind) {
    case KF_OP_SCALE: return x * op.scalar;
    case KF_OP_RELU: return fmaxf(x, 0.0f);
    case KF_OP_GELU_TANH: return f_gelu_tanh(x);
    case KF_OP_SILU: return x * f_sigmoid(x);
    case KF_OP_SIGMOID: return f_sigmoid(x);
    case KF_OP_MISH: return f_mish(x);
    case KF_OP_LEAKY_RELU: return x > 0.0f ? x : op.scalar * x;
    default: return x;
  }
}

// Apply ops[0..n) to the 32 values of row `row` starting at column col0 (the
// first `nvalid` columns exist).  Operands of rows that do not exist are not
// read (row_ok == false).  FAST selects the reduced-precision activations (for
// chains whose result is stored as bf16).
// `st` holds operands the caller loaded ahead of time: the RESIDUAL_ADD op uses
// st.res when st.use_res, and op st.vec_idx uses st.vec as its per-column vector;
// other operands are loaded here.
template <bool FAST>
__device__ __forceinline__ void apply_chain32(const DevOp* ops, int n, float (&v)[32], int64_t row, int64_t col0,
                                              int nvalid, bool row_ok, const Staged32& st) {
  for (int o = 0; o < n; ++o) {
    const DevOp& op = ops[o];
    switch (op.kind) {
      case KF_OP_BIAS:
      case KF_OP_MUL: {
        float b[32];
        if (o == st.vec_idx) {
#pragma unroll
          for (int k = 0; k < 16; ++k) {
            b[2 * k] = bf16lo(st.vec[k]);
            b[2 * k + 1] = bf16hi(st.vec[k]);
          }
        } else {
          ld32(op.p0, op.p_dtype, col0, nvalid, op.vec_ok != 0, b);
        }
        if (op.kind == KF_OP_BIAS) {
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] += b[j];
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] *= b[j];
        }
      } break;
      case KF_OP_RESIDUAL_ADD: {
        if (st.use_res) {
#pragma unroll
          for (int k = 0; k < 16; ++k) {
            v[2 * k] += bf16lo(st.res[k]);
            v[2 * k + 1] += bf16hi(st.res[k]);
          }
        } else if (row_ok) {
          float r[32];
          ld32(op.p0, op.p_dtype, row * op.ld + col0, nvalid, op.vec_ok != 0, r);
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] += r[j];
        }
      } break;
      case KF_OP_SCALE: {
        const float s = op.scalar;
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] *= s;
      } break;
      case KF_OP_ROW_SCALE: {
        const float s = row_ok ? reinterpret_cast<const float*>(op.p0)[row] : 0.0f;
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] *= s;
      } break;
      case KF_OP_RELU: {
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = fmaxf(v[j], 0.0f);
      } break;
      case KF_OP_GELU_TANH: {
        if (FAST) {
#pragma unroll
          for (int j = 0; j < 32; j += 2) gelu2_f16(v[j], v[j + 1]);
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = f_gelu_tanh(v[j]);
        }
      } break;
      case KF_OP_SILU:
      case KF_OP_SIGMOID: {
        if (FAST) {
          // sigmoid(x) = (1 + tanh(x / 2)) / 2
#pragma unroll
          for (int j = 0; j < 32; j += 2) {
            float t0, t1;
            tanh2_fast(0.5f * v[j], 0.5f * v[j + 1], t0, t1);
            const float s0 = fmaf(0.5f, t0, 0.5f), s1 = fmaf(0.5f, t1, 0.5f);
            v[j] = op.kind == KF_OP_SILU ? v[j] * s0 : s0;
            v[j + 1] = op.kind == KF_OP_SILU ? v[j + 1] * s1 : s1;
          }
        } else {
#pragma unroll
          for (int j = 0; j < 32; ++j) v[j] = op.kind == KF_OP_SILU ? v[j] * f_sigmoid(v[j]) : f_sigmoid(v[j]);
        }
      } break;
      case KF_OP_MISH: {
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = FAST ? f_mish_fast(v[j]) : f_mish(v[j]);
      } break;
      case KF_OP_LEAKY_RELU: {
        const float s = op.scalar;
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = v[j] > 0.0f ? v[j] : s * v[j];
      } break;
      default: break;
    }
  }
}

__device__ __forceinline__ void apply_chain32_rt(bool fast, const DevOp* ops, int n, float (&v)[32], int64_t row,
                                                 int64_t col0, int nvalid, bool row_ok, const Staged32& st) {
  if (n <= 0) return;
  if (fast)
    apply_chain32<true>(ops, n, v, row, col0, nvalid, row_ok, st);
  else
    apply_chain32<false>(ops, n, v, row, col0, nvalid, row_ok, st);
}
__device__ __forceinline__ void apply_chain32_rt(bool fast, const DevOp* ops, int n, float (&v)[32], int64_t row,
                                                 int64_t col0, int nvalid, bool row_ok) {
  Staged32 none;
  none.use_res = false;
  none.vec_idx = -1;
  apply_chain32_rt(fast, ops, n, v, row, col0, nvalid, row_ok, none);
}

// ------------------------------------------------------ compiled op programs
// A chain whose op kinds match a compiled program runs as straight-line code:
// operand fields are read at constant offsets and there is no per-op dispatch.
// Prog<> is the empty chain; Interp runs any chain through apply_chain32.
template <int KIND, bool FAST>
__device__ __forceinline__ void prog_op(const DevOp& op, float (&v)[32], int64_t row, int64_t col0, int nvalid,
                                        bool row_ok, const Staged32& st, bool staged_vec) {
  if constexpr (KIND == KF_OP_BIAS || KIND == KF_OP_MUL) {
    float b[32];
    if (staged_vec) {
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        b[2 * k] = bf16lo(st.vec[k]);
        b[2 * k + 1] = bf16hi(st.vec[k]);
      }
    } else {
      ld32(op.p0, op.p_dtype, col0, nvalid, op.vec_ok != 0, b);
    }
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = KIND == KF_OP_BIAS ? v[j] + b[j] : v[j] * b[j];
  } else if constexpr (KIND == KF_OP_RESIDUAL_ADD) {
    if (st.use_res) {
#pragma unroll
      for (int k = 0; k < 16; ++k) {
        v[2 * k] += bf16lo(st.res[k]);
        v[2 * k + 1] += bf16hi(st.res[k]);
      }
    } else if (row_ok) {
      float r[32];
      ld32(op.p0, op.p_dtype, row * op.ld + col0, nvalid, op.vec_ok != 0, r);
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] += r[j];
    }
  } else if constexpr (KIND == KF_OP_SCALE) {
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] *= op.scalar;
  } else if constexpr (KIND == KF_OP_GELU_TANH) {
    if constexpr (FAST) {
#pragma unroll
      for (int j = 0; j < 32; j += 2) gelu2_f16(v[j], v[j + 1]);
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] = f_gelu_tanh(v[j]);
    }
  } else if constexpr (KIND == KF_OP_SILU) {
    if constexpr (FAST) {
#pragma unroll
      for (int j = 0; j < 32; j += 2) {
        float t0, t1;
        tanh2_fast(0.5f * v[j], 0.5f * v[j + 1], t0, t1);
        v[j] *= fmaf(0.5f, t0, 0.5f);
        v[j + 1] *= fmaf(0.5f, t1, 0.5f);
      }
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] *= f_sigmoid(v[j]);
    }
  } else {
    static_assert(KIND == KF_OP_BIAS, "op kind has no compiled form");
  }
}

template <int... KINDS>
struct Prog {
  static constexpr int kLen = sizeof...(KINDS);
  static constexpr bool kGeneric = false;
  static constexpr bool kHasRes = ((KINDS == KF_OP_RESIDUAL_ADD) || ... || false);
  template <bool FAST>
  __device__ __forceinline__ static void run(const DevOp* ops, float (&v)[32], int64_t row, int64_t col0, int nvalid,
                                             bool row_ok, const Staged32& st) {
    int i = 0;
    ((prog_op<KINDS, FAST>(ops[i], v, row, col0, nvalid, row_ok, st, i == st.vec_idx), ++i), ...);
  }
  // does a runtime op list match this program?
  __host__ static bool matches(const DevOp* ops, int n) {
    const int kinds[] = {KINDS..., -1};
    if (n != kLen) return false;
    for (int i = 0; i < n; ++i)
      if (ops[i].kind != kinds[i]) return false;
    return true;
  }
};
struct Interp {
  static constexpr bool kGeneric = true;
  static constexpr bool kHasRes = false;
  template <bool FAST>
  __device__ __forceinline__ static void run(const DevOp* ops, int n, float (&v)[32], int64_t row, int64_t col0,
                                             int nvalid, bool row_ok, const Staged32& st) {
    apply_chain32<FAST>(ops, n, v, row, col0, nvalid, row_ok, st);
  }
};

// Apply chain `ops[0..n)` with program P (the interpreter when P is Interp).
template <class P>
__device__ __forceinline__ void run_chain(bool fast, const DevOp* ops, int n, float (&v)[32], int64_t row, int64_t col0,
                                          int nvalid, bool row_ok, const Staged32& st) {
  if constexpr (P::kGeneric) {
    if (n <= 0) return;
    if (fast)
      P::template run<true>(ops, n, v, row, col0, nvalid, row_ok, st);
    else
      P::template run<false>(ops, n, v, row, col0, nvalid, row_ok, st);
  } else {
    if (fast)
      P::template run<true>(ops, v, row, col0, nvalid, row_ok, st);
    else
      P::template run<false>(ops, v, row, col0, nvalid, row_ok, st);
  }
}
template <class P>
__device__ __forceinline__ void run_chain(bool fast, const DevOp* ops, int n, float (&v)[32], int64_t row, int64_t col0,
                                          int nvalid, bool row_ok) {
  Staged32 none;
  none.use_res = false;
  none.vec_idx = -1;
  run_chain<P>(fast, ops, n, v, row, col0, nvalid, row_ok, none);
}

}  // namespace kf
