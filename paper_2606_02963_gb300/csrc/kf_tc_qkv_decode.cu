// kf_tc_qkv_decode.cu -- the QKV projection tail for decode-sized calls (at most
// 64 tokens): bias + rotary embedding + key / value cache rows, with the K
// dimension split over the CTAs of a cluster and the partial sums reduced
// through distributed shared memory (the gpt-oss decode kernel "Bias + RoPE +
// KV update" of Sec. IV-A, here fused with its GEMM).
//
// A decode GEMM reads each weight once; one 256-column tile per CTA over the
// whole K would keep only N / 256 SMs busy and pay 4 MMAs per 64-wide k-block
// for all of K.  Here a cluster of S CTAs shares one 256-column tile (four
// 64-column heads): CTA r multiplies the k-blocks [r K / S, (r + 1) K / S).
// The tile's T token rows are dealt out to the cluster's CTAs in runs of
// RPO = ceil(T / S) rows; each CTA sends every row of its 128 x 256 fp32
// partial to the shared memory of the row's owner as 16-byte DSMEM stores,
// which need no reply and overlap the other CTAs' mainloops: up to 32 tokens
// straight from TMEM (lane = row), above that staged in its operand ring (free
// by then) and sent as whole 512-byte warp stores by all ten warps.  After one
// cluster barrier an owner's epilogue warps reduce its rows from local shared
// memory alone (its own rows from its ring): a warp sums the S partials of a
// row in CTA-rank order (lane j: the four rotation pairs 4j .. 4j + 3 of the
// tile), adds the bias, rotates query and key heads and stores the row's heads
// to q_out or to the token's cache row.  No global workspace, no atomics, no
// waits between CTAs other than the hardware cluster barriers (one that every
// CTA has started before any DSMEM store, one after the stores), and no CTA
// waits for the others to exit.  While the MMAs run, the epilogue warps already
// load what their rows need besides the sums (bias, positions, cache rows, the
// first two rows' table entries).
//
// Token rows are staged in boxes of ROWS = 32 (five-stage ring) or 64 rows
// (four stages): the box is what limits the tokens of a call.
//
// Warp roles: warp 0 TMA producer, warp 1 MMA issuer, warps 2-9 epilogue.
#include "kf_internal.h"

namespace kf {
namespace {

constexpr int kDcThreads = 320;
constexpr int kDcBM = 128;          // rows of the MMA (only the first T are tokens)
constexpr int kDcBK = 64;           // K elements per 128-byte row
constexpr int kDcBN = 256;          // tile columns
constexpr int kDcDirectMaxT = 32;  // up to this many tokens partial rows leave TMEM for their owners directly
constexpr int kDcPartStride = 260;  // floats per partial row (4 banks apart: conflict-free 16-byte row-per-lane stores)

template <int ROWS, int STAGES>
struct DcCfg {
  // A: ROWS token rows per k-block (4 or 8 KB).  The MMA reads 128 rows from
  // there; the ones past the box are the next stages' bytes and feed only
  // accumulator rows past T, which are never stored (A stages come first, so
  // the reads stay in the ring).
  static_assert(ROWS == 32 || ROWS == 64, "token box");
  static constexpr int kABytes = ROWS * kDcBK * 2;
  static constexpr int kBBytes = kDcBN * kDcBK * 2;    // 32 KB
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr uint32_t kTxBytes = kStageBytes;
  static constexpr int kRingBytes = STAGES * kStageBytes;
  // after the mainloop the ring holds the CTA's own partial of the rows it
  // owns; the other CTAs' partials of those rows land in a region of their own
  // (written while this CTA may still be in its mainloop): (S - 1) ceil(T / S)
  // rows, at most 60 (ROWS = 64) or 30 (ROWS = 32) for S <= 8
  static constexpr int kRecvRows = ROWS == 64 ? 60 : 30;
  static constexpr int kRowBytes = kDcPartStride * 4;
  static_assert(ROWS * kRowBytes <= kRingBytes, "the own partial fits the ring");
  static_assert(STAGES * kABytes + kBBytes >= kDcBM * kDcBK * 2, "the MMA's 128-row reads stay in the ring");
  static constexpr int kBarBytes = 256;  // 2 STAGES + 2 barriers and three words
  static_assert(8 * (2 * STAGES + 2) + 16 <= kBarBytes, "barrier block");
  static constexpr int kRecvOff = kRingBytes + kBarBytes;
  static constexpr int kSmemBytes = 1024 + kRecvOff + kRecvRows * kRowBytes;
  static constexpr uint32_t kIdesc = idesc_bf16_f32(kDcBM, kDcBN);
  static_assert(kSmemBytes <= 232448, "shared memory");
};

// A tile row (one token, 256 columns) is reduced by one warp: lane j takes the
// rotation pairs 4j .. 4j + 3 of the tile, i.e. four consecutive columns of one
// head's first half and the four that pair with them in its second half (a
// head's half is a multiple of 32 columns, so the four never straddle heads).
// These operands of the lane do not depend on the token.
struct DcLane {
  int32_t hcol;  // first column of the lane's head
  int32_t i;     // first of the lane's four pair indices within the head
  bool live, rotate;
  float b0[4], b1[4];
};
// The token-dependent operands of a row.
struct DcRow {
  int32_t pos, crow;
  bool ok;
  float c[4], s[4];
};

// A 16-byte load of read-only data issued exactly here: a plain __ldg may be
// moved to its first use (read-only loads are free to move), which would put
// its latency back after the cluster barrier that this prefetch is meant to
// hide it behind.
__device__ __forceinline__ float4 ldg_f4_here(const float* ptr) {
  float4 v;
  asm volatile("ld.global.nc.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "l"(ptr));
  return v;
}
// one bias element (fp32, bf16 or fp16), issued exactly here likewise
__device__ __forceinline__ float ld_bias_here(const void* ptr, int dt, int64_t i) {
  uint32_t b;
  if (dt == KF_F32) {
    asm volatile("ld.global.nc.b32 %0, [%1];" : "=r"(b) : "l"(static_cast<const uint32_t*>(ptr) + i));
  } else {
    uint16_t h;
    asm volatile("ld.global.nc.b16 %0, [%1];" : "=h"(h) : "l"(static_cast<const uint16_t*>(ptr) + i));
    b = h;
  }
  return cvt_raw(b, dt);
}

__device__ __forceinline__ void dc_lane(const QkvDecodeParams& p, int32_t n0, int lane, DcLane& L) {
  const int d = p.rope_d, half = d >> 1;
  const int pr = 4 * lane;
  L.hcol = n0 + (pr / half) * d;
  L.i = pr % half;
  L.live = L.hcol < p.N;
  L.rotate = L.hcol < p.rot_cols;
#pragma unroll
  for (int m = 0; m < 4; ++m) {
    const bool use = L.live && p.bias;
    L.b0[m] = use ? ld_bias_here(p.bias, p.bias_dtype, L.hcol + L.i + m) : 0.0f;
    L.b1[m] = use ? ld_bias_here(p.bias, p.bias_dtype, L.hcol + L.i + m + half) : 0.0f;
  }
}

// 16 bytes of this CTA's shared memory (explicit state space: the partial
// buffers are addressed through an aligned integer, which a plain pointer
// access would turn into a generic load or store)
__device__ __forceinline__ float4 lds_f4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(addr));
  return v;
}
__device__ __forceinline__ void sts_f4(uint32_t addr, float a, float b, float c, float d) {
  asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "f"(a), "f"(b), "f"(c), "f"(d) : "memory");
}

// A position or cache row out of range clears `ok` (the row is then reported
// and skipped, and no table row is read for it).
__device__ __forceinline__ void dc_row(const QkvDecodeParams& p, const DcLane& L, int32_t pos, int32_t crow,
                                       DcRow& R) {
  const int half = p.rope_d >> 1;
  R.pos = pos;
  R.crow = crow;
  R.ok = pos >= 0 && pos < p.max_pos && crow >= 0 && crow < p.rows;
  // the tables start on 16 bytes and half and i are multiples of 4: one
  // 16-byte load per table
  float4 c = make_float4(1.0f, 1.0f, 1.0f, 1.0f), s = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
  if (R.ok && L.live && L.rotate) {
    const int64_t o = static_cast<int64_t>(pos) * half + L.i;
    c = ldg_f4_here(p.cos_t + o);
    s = ldg_f4_here(p.sin_t + o);
  }
  R.c[0] = c.x;
  R.c[1] = c.y;
  R.c[2] = c.z;
  R.c[3] = c.w;
  R.s[0] = s.x;
  R.s[1] = s.y;
  R.s[2] = s.z;
  R.s[3] = s.w;
}

// four consecutive outputs from element o on: one vector store where o and the
// base allow it, else four scalar stores
__device__ __forceinline__ void dc_store4(void* dst, int dt, int64_t o, float x0, float x1, float x2, float x3) {
  const uintptr_t base = reinterpret_cast<uintptr_t>(dst);
  if (dt == KF_F32) {
    float* d = reinterpret_cast<float*>(dst) + o;
    if ((o & 3) == 0 && (base & 15) == 0) {
      *reinterpret_cast<float4*>(d) = make_float4(x0, x1, x2, x3);
    } else {
      d[0] = x0;
      d[1] = x1;
      d[2] = x2;
      d[3] = x3;
    }
  } else {
    uint32_t w0, w1;
    if (dt == KF_BF16) {
      w0 = pack_bf16x2(x0, x1);
      w1 = pack_bf16x2(x2, x3);
    } else {
      w0 = pack_f16x2(x0, x1);
      w1 = pack_f16x2(x2, x3);
    }
    uint16_t* d = reinterpret_cast<uint16_t*>(dst) + o;
    if ((o & 3) == 0 && (base & 7) == 0) {
      *reinterpret_cast<uint2*>(d) = make_uint2(w0, w1);
    } else {
      d[0] = static_cast<uint16_t>(w0);
      d[1] = static_cast<uint16_t>(w0 >> 16);
      d[2] = static_cast<uint16_t>(w1);
      d[3] = static_cast<uint16_t>(w1 >> 16);
    }
  }
}

template <int ROWS, int STAGES>
__global__ void __launch_bounds__(kDcThreads, 1)
    kf_qkv_decode_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                         const __grid_constant__ QkvDecodeParams p) {
  using Cfg = DcCfg<ROWS, STAGES>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* smA = sm;                                   // A stages first (see DcCfg)
  uint8_t* smB = sm + STAGES * Cfg::kABytes;
  float* part = reinterpret_cast<float*>(sm);          // after the mainloop: own partial, [RPO][260] fp32
  float* recv = reinterpret_cast<float*>(sm + Cfg::kRecvOff);  // other CTAs' partials, [S - 1][RPO][260]
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + Cfg::kRingBytes);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* accf = bars + 2 * STAGES;
  uint64_t* drain = bars + 2 * STAGES + 1;
  uint32_t* misc = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 2);
  uint32_t* tmem_slot = misc;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 1);
  volatile int* zero_flag = reinterpret_cast<volatile int*>(misc + 2);

  // the split count is the cluster size; refuse any other launch shape before
  // any barrier, TMEM allocation or copy
  const uint32_t S = cluster_nctarank();
  if (S != static_cast<uint32_t>(p.splits) || blockDim.x != kDcThreads || gridDim.x % S != 0 || gridDim.y != 1 ||
      gridDim.z != 1 || p.T < 1 || p.T > ROWS ||
      (static_cast<int32_t>(S) - 1) * ((p.T + static_cast<int32_t>(S) - 1) / static_cast<int32_t>(S)) > Cfg::kRecvRows) {
    if (threadIdx.x == 0) atomicOr(p.err, kErrLaunchShape);
    return;
  }
  const uint32_t r = cluster_ctarank();
  const int32_t tile = static_cast<int32_t>(blockIdx.x / S);
  const int32_t n0 = tile * kDcBN;
  const int32_t kb0 = static_cast<int32_t>(r) * p.num_kb / static_cast<int32_t>(S);
  const int32_t kb1 = static_cast<int32_t>(r + 1) * p.num_kb / static_cast<int32_t>(S);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // CTA o of the cluster owns the token rows [o RPO, (o + 1) RPO) of the tile
  // and reduces them; its epilogue warp ew takes the owned rows ew, ew + 8, ...
  const int32_t rpo = (p.T + static_cast<int32_t>(S) - 1) / static_cast<int32_t>(S);
  const int32_t own0 = static_cast<int32_t>(r) * rpo;
  const int32_t nown = max(0, min(rpo, p.T - own0));
  const int32_t nrows = warp >= 2 && warp - 2 < nown ? (nown - (warp - 2) + 7) / 8 : 0;
  DcLane L;       // the epilogue lane's columns and bias
  DcRow cur, nxt;  // the warp's current and next row
  int32_t my_pos = 0, my_crow = 0;  // lane k < nrows: row k's position and cache row

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accf, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    *zero_flag = 0;
    fence_mbarrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
    // this CTA's weights into L2 while a preceding kernel may still run: a
    // prefetch reads memory without changing it and L2 is where that kernel's
    // writes land, so the loads after the dependency wait below see current
    // values either way; the weights are the bytes this kernel is bound by
    for (int32_t kb = kb0; kb < kb1; ++kb) tma_prefetch_3d(&tmB, kb * kDcBK, n0, 0);
  }
  if (warp == 1) {
    __syncwarp();
    tmem_alloc(tmem_slot, kDcBN);
    tmem_relinquish();
  }
  // launched as a programmatic dependent of the previous kernel in the stream:
  // wait for it before any operand, position or table is read
  griddep_wait();
  griddep_launch_dependents();
  tc_fence_before();
  __syncwarp();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  bool ok = true;
  bool acc_ok = false;  // epilogue warps: the accumulator is complete
  // this CTA has started: the other CTAs of the cluster may write its shared
  // memory once every CTA has arrived here
  cluster_arrive_relaxed();

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      int32_t it = 0;
      for (int32_t kb = kb0; kb < kb1; ++kb, ++it) {
        const int st = it % STAGES;
        if (!mbar_wait(&empty[st], ((it / STAGES) & 1) ^ 1, abort_flag, p.wait_ns)) {
          *abort_flag = 1;
          atomicOr(p.err, kErrWaitProducer);
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&full[st], Cfg::kTxBytes);
        tma_load_2d(smA + st * Cfg::kABytes, &tmA, &full[st], kb * kDcBK, 0);
        tma_load_3d(smB + st * Cfg::kBBytes, &tmB, &full[st], kb * kDcBK, n0, 0);
      }
      if (!ok)  // copies still in flight land before the ring is reused or the CTA exits
        for (int32_t j = (it > STAGES ? it - STAGES : 0); j < it; ++j)
          mbar_wait(&full[j % STAGES], (j / STAGES) & 1, zero_flag, p.drain_ns);
    }
  } else if (warp == 1) {
    // --------------------------------------------------------------------- MMA
    if (lane == 0) {
      const uint32_t idesc = p.ab_f16 ? (Cfg::kIdesc & ~((7u << 7) | (7u << 10))) : Cfg::kIdesc;
      int32_t it = 0;
      for (int32_t kb = kb0; kb < kb1; ++kb, ++it) {
        const int st = it % STAGES;
        if (!mbar_wait(&full[st], (it / STAGES) & 1, abort_flag, p.wait_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a0 = smem_u32(smA + st * Cfg::kABytes);
        const uint32_t b0 = smem_u32(smB + st * Cfg::kBBytes);
#pragma unroll
        for (int kk = 0; kk < kDcBK / 16; ++kk)
          tc_mma_bf16(tmem, desc_sw128_kmajor(a0 + kk * 32), desc_sw128_kmajor(b0 + kk * 32), idesc,
                      (kb != kb0 || kk != 0) ? 1u : 0u);
        tc_commit(&empty[st]);
      }
      if (ok) {
        tc_commit(accf);
      } else {
        *abort_flag = 1;
        atomicOr(p.err, kErrWaitMma);
        tc_commit(drain);  // arrives once every MMA issued so far has completed
        mbar_wait(drain, 0, zero_flag, p.drain_ns);
      }
    }
  } else {
    // ------------------ epilogue: operands while the MMAs run, the accumulator
    // the lane's bias, the positions and cache rows of all the warp's rows (at
    // most 8: T <= 64 and 8 warps), the first two rows' table entries
    dc_lane(p, n0, lane, L);
    if (lane < nrows) {
      my_pos = p.positions[own0 + warp - 2 + 8 * lane];
      my_crow = p.cache_rows[own0 + warp - 2 + 8 * lane];
    }
    if (nrows > 0)
      dc_row(p, L, __shfl_sync(0xffffffffu, my_pos, 0), __shfl_sync(0xffffffffu, my_crow, 0), cur);
    if (nrows > 1)
      dc_row(p, L, __shfl_sync(0xffffffffu, my_pos, 1), __shfl_sync(0xffffffffu, my_crow, 1), nxt);
    bool w = mbar_wait(accf, 0, abort_flag, p.wait_ns);
    acc_ok = __all_sync(0xffffffffu, w);
    if (!acc_ok) {
      *abort_flag = 1;
      if (lane == 0) atomicOr(p.err, kErrWaitEpilogue);
    }
  }
  // every CTA of the cluster has started
  cluster_wait();
  // Few rows go straight from TMEM to their owners (lane = row: the warps of
  // the token quadrants alone send); more rows are staged in this CTA's ring
  // first and sent by all ten warps as whole 512-byte warp stores, which the
  // DSMEM path moves much faster.
  const bool direct = p.T <= kDcDirectMaxT;
  if (warp >= 2 && acc_ok) {
    // -------------------------------- epilogue part 1: partial rows out of TMEM
    // Own rows (all rows when staging) go to the ring (idle: all copies landed
    // and all MMAs completed before the accumulator was signalled), row t at
    // t * 260 floats; the others to slot r (r - 1 past the owner's rank) of the
    // owner's receive region.  DSMEM stores need no reply.
    const int ew = warp - 2;
    const int q = warp & 3;  // TMEM lane quadrant
    const int hh = ew >> 2;  // column half: [128 hh, 128 hh + 128)
    const int32_t row = q * 32 + lane;
    tc_fence_after();
    fence_proxy_async_smem();  // the ring's last copies were async-proxy writes
    const uint32_t lane_off = static_cast<uint32_t>(q * 32) << 16;
    if (q * 32 < p.T) {  // quadrants past the last token have nothing to keep
      const int32_t rr = min(row, p.T - 1);  // lanes past the last token store nothing
      const uint32_t o = static_cast<uint32_t>(rr / rpo);
      uint32_t dst = smem_u32(part) + static_cast<uint32_t>(rr * Cfg::kRowBytes);
      if (direct && o != r) {
        const uint32_t slot = r < o ? r : r - 1;
        const int32_t lr = rr - static_cast<int32_t>(o) * rpo;
        dst = mapa_shared(smem_u32(recv), o) + static_cast<uint32_t>((slot * rpo + lr) * Cfg::kRowBytes);
      }
      dst += static_cast<uint32_t>((hh * 128) * 4);
      for (int c = 0; c < 4; ++c) {
        float v[32];
        tmem_ld32(tmem + lane_off + hh * 128 + c * 32, v);
        // sent directly: one store path for the warp's own and remote rows
        // alike (splitting the lanes over two paths costs more than it saves)
        if (row < p.T && direct) {
#pragma unroll
          for (int j = 0; j < 8; ++j)
            st_cluster_f4(dst + static_cast<uint32_t>((c * 32 + 4 * j) * 4), v[4 * j], v[4 * j + 1], v[4 * j + 2],
                          v[4 * j + 3]);
        } else if (row < p.T) {
#pragma unroll
          for (int j = 0; j < 8; ++j)
            sts_f4(dst + static_cast<uint32_t>((c * 32 + 4 * j) * 4), v[4 * j], v[4 * j + 1], v[4 * j + 2],
                   v[4 * j + 3]);
        }
      }
    }
  }
  if (!direct) {
    __syncthreads();
    if (!*abort_flag) {
      // ----------- epilogue part 2: staged rows other CTAs own -> their shared memory
      // warp w sends rows w, w + 10, ... (a row is 1 KB: two 512-byte warp
      // stores, lane j: 16 bytes)
      for (int32_t t = warp; t < p.T; t += kDcThreads / 32) {
        const uint32_t o = static_cast<uint32_t>(t / rpo);
        if (o == r) continue;  // reduced in place
        const uint32_t slot = r < o ? r : r - 1;
        const int32_t lr = t - static_cast<int32_t>(o) * rpo;
        const uint32_t dst =
            mapa_shared(smem_u32(recv), o) + static_cast<uint32_t>((slot * rpo + lr) * Cfg::kRowBytes);
        const uint32_t src = smem_u32(part) + static_cast<uint32_t>(t * Cfg::kRowBytes);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const float4 v = lds_f4(src + static_cast<uint32_t>((h * 128 + 4 * lane) * 4));
          st_cluster_f4(dst + static_cast<uint32_t>((h * 128 + 4 * lane) * 4), v.x, v.y, v.z, v.w);
        }
      }
    }
  }
  // every partial row is in its owner's shared memory; after this barrier no
  // CTA touches another's shared memory, so none waits for the others to exit
  tc_fence_before();
  __syncwarp();
  cluster_sync();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kDcBN);
  }

  if (warp >= 2 && !*abort_flag) {
    // ---------- epilogue part 3: reduce the S partials of the owned rows, bias,
    // rotate, store (all from this CTA's shared memory); the table entries of
    // the row after the next load meanwhile
    const int half = p.rope_d >> 1;
    for (int32_t k = 0; k < nrows; ++k) {
      const int32_t lr = warp - 2 + 8 * k;
      const int32_t t = own0 + lr;
      DcRow nn = nxt;  // the row after the next one, loaded while this one is reduced
      if (k + 2 < nrows)
        dc_row(p, L, __shfl_sync(0xffffffffu, my_pos, k + 2), __shfl_sync(0xffffffffu, my_crow, k + 2), nn);
      if (!cur.ok) {
        if (lane == 0) atomicOr(p.err, kErrBounds);
      } else if (L.live) {
        const int32_t c0 = L.hcol - n0 + L.i;
        float4 va[8], vb[8];
#pragma unroll
        for (uint32_t s2 = 0; s2 < 8; ++s2) {
          if (s2 < S) {
            // rank s2's partial: the ring for this CTA's own, else its slot
            const uint32_t src =
                s2 == r ? smem_u32(part) + static_cast<uint32_t>(t * Cfg::kRowBytes)
                        : smem_u32(recv) + static_cast<uint32_t>(((s2 < r ? s2 : s2 - 1) * rpo + lr) * Cfg::kRowBytes);
            va[s2] = lds_f4(src + static_cast<uint32_t>(c0 * 4));
            vb[s2] = lds_f4(src + static_cast<uint32_t>((c0 + half) * 4));
          }
        }
        // the sums in CTA-rank order
        float a[4] = {0.0f, 0.0f, 0.0f, 0.0f}, b[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
        for (uint32_t s2 = 0; s2 < 8; ++s2) {
          if (s2 < S) {
            a[0] += va[s2].x;
            a[1] += va[s2].y;
            a[2] += va[s2].z;
            a[3] += va[s2].w;
            b[0] += vb[s2].x;
            b[1] += vb[s2].y;
            b[2] += vb[s2].z;
            b[3] += vb[s2].w;
          }
        }
        float y0[4], y1[4];
#pragma unroll
        for (int m = 0; m < 4; ++m) {
          float x0 = a[m] + L.b0[m], x1 = b[m] + L.b1[m];
          if (L.rotate) {
            const float c = cur.c[m], sn = cur.s[m];
            const float r0 = fmaf(x0, c, -x1 * sn), r1 = fmaf(x1, c, x0 * sn);
            x0 = r0;
            x1 = r1;
          }
          y0[m] = x0;
          y1[m] = x1;
        }
        void* dst;
        int64_t dst0;
        if (L.hcol < p.q_cols) {
          dst = p.q_out;
          dst0 = static_cast<int64_t>(t) * p.ldq + L.hcol;
        } else {
          dst = L.rotate ? p.k_cache : p.v_cache;
          dst0 = static_cast<int64_t>(cur.crow) * p.ld_cache + L.hcol - (L.rotate ? p.q_cols : p.rot_cols);
        }
        dc_store4(dst, p.out_dtype, dst0 + L.i, y0[0], y0[1], y0[2], y0[3]);
        dc_store4(dst, p.out_dtype, dst0 + L.i + half, y1[0], y1[1], y1[2], y1[3]);
      }
      cur = nxt;
      nxt = nn;
    }
  }
}

template <int ROWS, int STAGES>
cudaError_t launch_dc(const CUtensorMap& a, const CUtensorMap& b, const QkvDecodeParams& p, int tiles,
                      cudaStream_t s) {
  using Cfg = DcCfg<ROWS, STAGES>;
  auto kern = kf_qkv_decode_kernel<ROWS, STAGES>;
  static std::atomic<bool> configured[64];
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!configured[dev]) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(tiles * p.splits, 1, 1);
  cfg.blockDim = dim3(kDcThreads, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmemBytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = p.splits;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  // a programmatic dependent of the previous kernel in the stream (the kernel
  // waits for it before reading anything it may have written)
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, a, b, p);
}

// co-resident clusters of `splits` CTAs of one variant on the current device
template <int ROWS, int STAGES>
cudaError_t clusters_dc(int splits, int* out) {
  using Cfg = DcCfg<ROWS, STAGES>;
  auto kern = kf_qkv_decode_kernel<ROWS, STAGES>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(splits, 1, 1);
  cfg.blockDim = dim3(kDcThreads, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmemBytes;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = splits;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaOccupancyMaxActiveClusters(out, kern, &cfg);
}

}  // namespace

// token boxes of 32 rows (five stages) up to 32 tokens, of 64 rows (four) above
cudaError_t qkv_decode_launch(const CUtensorMap& a, const CUtensorMap& b, const QkvDecodeParams& p, int tiles,
                              cudaStream_t s) {
  if (p.splits < 1 || p.splits > 8 || p.T < 1 || p.T > kQkvDecodeMaxRows) return cudaErrorInvalidValue;
  return p.T <= 32 ? launch_dc<32, 5>(a, b, p, tiles, s) : launch_dc<64, 4>(a, b, p, tiles, s);
}

int qkv_decode_box_rows(int64_t T) { return T <= 32 ? 32 : 64; }

// co-resident clusters of `splits` CTAs for the decode kernel variant that
// serves T tokens (queried once per device, variant and cluster size)
cudaError_t qkv_decode_clusters(int64_t T, int splits, int* out) {
  static std::atomic<int> cache[64][2][9];  // 0: not yet queried
  if (splits < 1 || splits > 8 || T < 1 || T > kQkvDecodeMaxRows) return cudaErrorInvalidValue;
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  const int v = T <= 32 ? 0 : 1;
  if (cache[dev][v][splits] == 0) {
    int nc = 0;
    cudaError_t e = v == 0 ? clusters_dc<32, 5>(splits, &nc) : clusters_dc<64, 4>(splits, &nc);
    if (e != cudaSuccess) return e;
    cache[dev][v][splits] = nc > 0 ? nc : -1;
  }
  const int c = cache[dev][v][splits].load();
  *out = c > 0 ? c : 0;
  return cudaSuccess;
}

}  // namespace kf
