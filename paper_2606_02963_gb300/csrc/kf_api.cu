// kf_api.cu -- the C ABI declared in include/kf.h: host-side argument checks,
// tail-chain planning, TMA tensor-map encoding and kernel dispatch.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <atomic>
#include <chrono>
#include <cstring>
#include <mutex>

#include "kf_internal.h"
#include "kf_tc_gemm.cuh"

// Per-device error word written by the kernels' bounded waits / bounds checks.
__device__ uint32_t g_kf_err;

namespace kf {
namespace {

constexpr uint64_t kDefaultWaitNs = 2000000000ull;  // 2 s
std::atomic<uint64_t> g_wait_ns{kDefaultWaitNs};

struct DevInfo {
  bool init = false;
  int nsm = 0;
  uint32_t* err = nullptr;
};
constexpr int kMaxDevices = 64;
DevInfo g_dev[kMaxDevices];
std::mutex g_mu;

kf_status cuda_status(cudaError_t e) { return e == cudaSuccess ? KF_OK : KF_ERR_CUDA; }

kf_status device_info(DevInfo* out) {
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= kMaxDevices) return KF_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  DevInfo& di = g_dev[d];
  if (!di.init) {
    if (cudaDeviceGetAttribute(&di.nsm, cudaDevAttrMultiProcessorCount, d) != cudaSuccess) return KF_ERR_CUDA;
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_kf_err) != cudaSuccess) return KF_ERR_CUDA;
    di.err = static_cast<uint32_t*>(p);
    di.init = true;
  }
  *out = di;
  return KF_OK;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// bf16 (or fp16) tensor map, 128-byte swizzle, box = 64 (K) x box_rows (x 1).
// Rank 2 for A operands ([rows, K]); rank 3 for B operands ([groups, rows, K]),
// which the kernel always loads with 3-D coordinates (groups = 1 for dense calls).
kf_status make_map(CUtensorMap* m, const void* base, uint64_t k, uint64_t rows, uint64_t row_stride_bytes,
                   uint64_t groups, uint64_t group_stride_bytes, uint32_t box_rows, cuuint32_t rank,
                   CUtensorMapDataType dt = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16) {
  auto fn = encode_fn();
  if (!fn) return KF_ERR_CUDA;
  std::memset(m, 0, sizeof(*m));
  cuuint64_t dims[3] = {k, rows, groups};
  cuuint64_t strides[2] = {row_stride_bytes, group_stride_bytes};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(kBK), box_rows, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(m, dt, rank, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? KF_OK : KF_ERR_CUDA;
}

// fp32 operand map for the 3xTF32 path: [rows, K], box 32 (K, 128 bytes) x
// box_rows, 128-byte swizzle.
kf_status make_map_f32(CUtensorMap* m, const void* base, uint64_t k, uint64_t rows, uint64_t row_stride_bytes,
                       uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) return KF_ERR_CUDA;
  std::memset(m, 0, sizeof(*m));
  cuuint64_t dims[2] = {k, rows};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {32, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? KF_OK : KF_ERR_CUDA;
}

// Output tensor map for the epilogue's TMA stores: bf16 [rows x cols] (row
// stride in bytes), box 16 columns x 32 rows, 32-byte swizzle (the layout of the
// epilogue's tile buffers).
kf_status make_map_out(CUtensorMap* m, void* base, uint64_t cols, uint64_t rows, uint64_t row_stride_bytes) {
  auto fn = encode_fn();
  if (!fn) return KF_ERR_CUDA;
  std::memset(m, 0, sizeof(*m));
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {16, 32};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  CU_TENSOR_MAP_SWIZZLE_32B, CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? KF_OK : KF_ERR_CUDA;
}

// bf16 [rows x cols] map with 32 x 32 boxes in the 64-byte swizzle: the
// residual-tile kernels load the residual and store the output through it.
kf_status make_map_blk64(CUtensorMap* m, const void* base, uint64_t cols, uint64_t rows, uint64_t row_stride_bytes) {
  auto fn = encode_fn();
  if (!fn) return KF_ERR_CUDA;
  std::memset(m, 0, sizeof(*m));
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? KF_OK : KF_ERR_CUDA;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
int elt_size(int dt) { return (dt == KF_BF16 || dt == KF_F16) ? 2 : 4; }
bool float_dtype(int dt) { return dt == KF_F32 || dt == KF_BF16 || dt == KF_F16; }

bool is_scalar_op(int k) {
  return k == KF_OP_SCALE || k == KF_OP_RELU || k == KF_OP_GELU_TANH || k == KF_OP_SILU || k == KF_OP_SIGMOID ||
         k == KF_OP_MISH || k == KF_OP_LEAKY_RELU;
}
bool is_pointwise_op(int k) {
  return is_scalar_op(k) || k == KF_OP_BIAS || k == KF_OP_MUL || k == KF_OP_RESIDUAL_ADD || k == KF_OP_ROW_SCALE;
}

struct ChainPlan {
  int mode = kModeStore;
  int n_pre = 0, n_post = 0;
  DevOp pre[kMaxOps];
  DevOp post[kMaxOps];
  // a row reduction's result ([M]): row sum instead of log-sum-exp (kModeLse),
  // or a row sum after the GroupNorm's post chain (kModeGroupNorm); the scalar
  // ops after the reduction run in the combine kernel (fin)
  bool red_sum = false;
  int n_fin = 0;
  DevOp fin[kMaxOps];
  DevOp norm;
  int gs = 0;
  const float* row_scale = nullptr;
  const int32_t* row_dst = nullptr;
  int64_t dst_rows = 0;
};

kf_status to_devop(const kf_epilogue_op& o, int64_t N, DevOp* d) {
  std::memset(d, 0, sizeof(*d));
  d->kind = o.kind;
  d->scalar = o.scalar;
  d->eps = o.eps;
  d->p0 = o.p0;
  d->p1 = o.p1;
  d->p_dtype = o.p_dtype;
  d->ld = o.ld;
  switch (o.kind) {
    case KF_OP_BIAS:
    case KF_OP_MUL:
      if (!o.p0 || !float_dtype(o.p_dtype)) return KF_ERR_INVALID_ARG;
      d->vec_ok = aligned16(o.p0);
      return KF_OK;
    case KF_OP_ROW_SCALE:
      if (!o.p0 || o.p_dtype != KF_F32) return KF_ERR_INVALID_ARG;
      return KF_OK;
    case KF_OP_RESIDUAL_ADD:
      if (!o.p0 || !float_dtype(o.p_dtype) || o.ld < N) return KF_ERR_INVALID_ARG;
      d->vec_ok = aligned16(o.p0) && (o.ld * elt_size(o.p_dtype)) % 16 == 0;
      return KF_OK;
    default:
      return is_scalar_op(o.kind) ? KF_OK : KF_ERR_INVALID_ARG;
  }
}

kf_status plan_chain(const kf_epilogue* epi, int64_t N, bool grouped, ChainPlan* pl) {
  const int n = epi ? epi->num_ops : 0;
  if (n < 0 || n > kMaxOps || (n > 0 && !epi->ops)) return KF_ERR_INVALID_ARG;
  // one reduction / special op per chain, except that a row sum may end a
  // GroupNorm chain (GroupNorm, pointwise ops, row sum, scalar ops)
  int special = -1, gn_sum = -1;
  for (int i = 0; i < n; ++i) {
    const int k = epi->ops[i].kind;
    if (k == KF_OP_ROW_LOGSUMEXP || k == KF_OP_GROUPNORM || k == KF_OP_SWIGLU || k == KF_OP_ROW_SCALE_SCATTER_ADD ||
        k == KF_OP_ROW_SUM) {
      if (special >= 0) {
        if (epi->ops[special].kind == KF_OP_GROUPNORM && k == KF_OP_ROW_SUM && gn_sum < 0) {
          gn_sum = i;
          continue;
        }
        return KF_ERR_UNSUPPORTED;
      }
      special = i;
    } else if (!is_pointwise_op(k)) {
      return KF_ERR_INVALID_ARG;
    }
  }
  const int sk = special >= 0 ? epi->ops[special].kind : -1;
  if (!grouped && (sk == KF_OP_SWIGLU || sk == KF_OP_ROW_SCALE_SCATTER_ADD)) return KF_ERR_INVALID_ARG;
  if (grouped && (sk == KF_OP_ROW_LOGSUMEXP || sk == KF_OP_GROUPNORM || sk == KF_OP_ROW_SUM)) return KF_ERR_UNSUPPORTED;
  const bool row_red = sk == KF_OP_ROW_LOGSUMEXP || sk == KF_OP_ROW_SUM;
  const int split = special >= 0 ? special : n;
  const int post_end = gn_sum >= 0 ? gn_sum : n;  // ops the kernel applies after the special op
  pl->n_pre = split;
  pl->n_post = special >= 0 ? post_end - special - 1 : 0;
  for (int i = 0; i < split; ++i) {
    kf_status st = to_devop(epi->ops[i], N, &pl->pre[i]);
    if (st != KF_OK) return st;
  }
  for (int i = 0; i < pl->n_post; ++i) {
    const kf_epilogue_op& o = epi->ops[special + 1 + i];
    if (row_red && !is_scalar_op(o.kind)) return KF_ERR_INVALID_ARG;
    kf_status st = to_devop(o, N, &pl->post[i]);
    if (st != KF_OK) return st;
  }
  // scalar ops after a row reduction run on the combined value
  pl->red_sum = sk == KF_OP_ROW_SUM || gn_sum >= 0;
  if (row_red) {
    pl->n_fin = pl->n_post;
    for (int i = 0; i < pl->n_post; ++i) pl->fin[i] = pl->post[i];
  } else if (gn_sum >= 0) {
    pl->n_fin = n - gn_sum - 1;
    for (int i = 0; i < pl->n_fin; ++i) {
      const kf_epilogue_op& o = epi->ops[gn_sum + 1 + i];
      if (!is_scalar_op(o.kind)) return KF_ERR_INVALID_ARG;
      kf_status st = to_devop(o, N, &pl->fin[i]);
      if (st != KF_OK) return st;
    }
  }
  switch (sk) {
    case -1: pl->mode = kModeStore; break;
    case KF_OP_ROW_LOGSUMEXP:
    case KF_OP_ROW_SUM: pl->mode = kModeLse; break;
    case KF_OP_SWIGLU:
      pl->mode = kModeSwiglu;
      if (pl->n_pre != 0) return KF_ERR_UNSUPPORTED;  // SwiGLU acts on the raw gate/up accumulators
      break;
    case KF_OP_ROW_SCALE_SCATTER_ADD: {
      const kf_epilogue_op& o = epi->ops[special];
      if (pl->n_post != 0) return KF_ERR_INVALID_ARG;  // must be last
      if (!o.p0 || !o.p1 || o.ld <= 0) return KF_ERR_INVALID_ARG;
      pl->mode = kModeScatter;
      pl->row_scale = static_cast<const float*>(o.p0);
      pl->row_dst = static_cast<const int32_t*>(o.p1);
      pl->dst_rows = o.ld;
    } break;
    case KF_OP_GROUPNORM: {
      const kf_epilogue_op& o = epi->ops[special];
      if (o.groups < 1 || N % o.groups != 0) return KF_ERR_INVALID_ARG;
      if ((o.p0 || o.p1) && !float_dtype(o.p_dtype)) return KF_ERR_INVALID_ARG;
      if (!(o.eps >= 0.0f)) return KF_ERR_INVALID_ARG;
      const int64_t gs = N / o.groups;
      if (gs % 32 != 0 || !(256 % gs == 0 || gs == 512)) return KF_ERR_UNSUPPORTED;
      pl->mode = kModeGroupNorm;
      pl->gs = static_cast<int>(gs);
      std::memset(&pl->norm, 0, sizeof(pl->norm));
      pl->norm.kind = KF_OP_GROUPNORM;
      pl->norm.eps = o.eps;
      pl->norm.groups = static_cast<int32_t>(gs);
      pl->norm.p0 = o.p0;
      pl->norm.p1 = o.p1;
      pl->norm.p_dtype = o.p_dtype;
      pl->norm.vec_ok = (!o.p0 || aligned16(o.p0)) && (!o.p1 || aligned16(o.p1));
    } break;
    default: return KF_ERR_INVALID_ARG;
  }
  return KF_OK;
}

void fill_params_common(TcParams& p, const ChainPlan& pl, uint32_t* err, uint32_t* err_dev) {
  // a single bf16 residual operand in the pre-chain is staged through shared
  // memory with coalesced loads (a second one would need its own buffer)
  int nres = 0, ires = -1;
  for (int i = 0; i < pl.n_pre; ++i)
    if (pl.pre[i].kind == KF_OP_RESIDUAL_ADD) {
      ++nres;
      ires = i;
    }
  p.res_op = (nres == 1 && pl.pre[ires].p_dtype == KF_BF16 && pl.pre[ires].vec_ok) ? ires : -1;
  // the first bf16 per-column vector (bias / mul) of the pre-chain is loaded ahead
  p.vec_op = -1;
  for (int i = 0; i < pl.n_pre && p.vec_op < 0; ++i)
    if ((pl.pre[i].kind == KF_OP_BIAS || pl.pre[i].kind == KF_OP_MUL) && pl.pre[i].p_dtype == KF_BF16 &&
        pl.pre[i].vec_ok)
      p.vec_op = i;
  p.n_pre = pl.n_pre;
  p.n_post = pl.n_post;
  for (int i = 0; i < pl.n_pre; ++i) p.pre[i] = pl.pre[i];
  for (int i = 0; i < pl.n_post; ++i) p.post[i] = pl.post[i];
  p.norm = pl.norm;
  p.red_sum = pl.red_sum ? 1 : 0;
  p.err = err;
  p.err_dev = err_dev;
  p.wait_ns = g_wait_ns.load();
  p.drain_ns = std::max<uint64_t>(p.wait_ns, 1000000000ull);
}

// Tile width for the dense store / LSE variants: the fewest tiles per CTA (or
// CTA pair) of the persistent grid, weighted by the tile width (+ a fixed
// per-tile cost).
int pick_dense_bn(int mode, int64_t M, int64_t N, int nsm, bool cta2) {
  static const int cand[] = {256, 224, 192, 128};
  int best = 0;
  int64_t best_cost = INT64_MAX;
  const int64_t rows = cta2 ? 2 * kBM : kBM;
  const int64_t workers = cta2 ? nsm / 2 : nsm;
  const int64_t tm = (M + rows - 1) / rows;
  for (int bn : cand) {
    if (!tc_dense_has(mode, bn, cta2)) continue;
    const int64_t tiles = tm * ((N + bn - 1) / bn);
    const int64_t per = (tiles + workers - 1) / workers;
    const int64_t cost = per * (bn + 48);
    if (cost < best_cost) {
      best_cost = cost;
      best = bn;
    }
  }
  return best;
}

// Output-column tile for the grouped variants.  Decode-like problems (at most
// one 128-row tile per group on average) stream each group's weights once and
// are bound by how evenly the tiles fall on the SMs: take the width with the
// fewest tile-widths of weights on the busiest SM (+ a small fixed cost per
// tile).  Otherwise the fewest tiles: a tcgen05.mma of K = 16 takes the same
// time for any N up to 256 on this GPU (measured: ~0.33 us per 64-wide k-block
// at N = 128, 192 and 256, with or without the operand loads), so a tile's
// mainloop costs the same whatever its width and the widest tile does the most
// work per MMA; its epilogue adds a little per column.
int pick_grouped_outn(int mode, int64_t N, int64_t rows_total, int32_t G, int nsm) {
  static const int cand[] = {256, 192, 128};
  int best = 0;
  if (G > 0 && rows_total <= static_cast<int64_t>(G) * kBM && nsm > 0) {
    const int64_t row_tiles = std::min<int64_t>(G, rows_total);  // one tile per touched group
    int64_t best_cost = INT64_MAX;
    for (int bn : cand) {
      if (!tc_grouped_has(mode, bn)) continue;
      const int outn = mode == kModeSwiglu ? bn / 2 : bn;
      const int64_t units = row_tiles * ((N + outn - 1) / outn);
      const int64_t cost = ((units + nsm - 1) / nsm) * (bn + 16);
      if (cost < best_cost) {
        best_cost = cost;
        best = bn;
      }
    }
    return best;
  }
  int64_t best_cost = INT64_MAX;
  for (int bn : cand) {
    if (!tc_grouped_has(mode, bn)) continue;
    const int outn = mode == kModeSwiglu ? bn / 2 : bn;
    const int64_t cost = ((N + outn - 1) / outn) * (1024 + outn);
    if (cost < best_cost) {
      best_cost = cost;
      best = bn;
    }
  }
  return best;
}

// rows of one B box: the whole tile, or each of the gate / up halves for SwiGLU
uint32_t mode_box(int mode, int bn) { return mode == kModeSwiglu ? bn / 2 : bn; }

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// A workspace starts with a header whose first 32-bit word is the error word of
// the calls given that workspace; the call's scratch (payload) follows it.
constexpr size_t kWsHeader = KF_WORKSPACE_HEADER_BYTES;
struct WsView {
  uint32_t* err = nullptr;  // the header's error word (null: no usable workspace)
  void* payload = nullptr;
  size_t bytes = 0;         // payload bytes
};
WsView split_ws(void* ws, size_t bytes) {
  WsView v;
  if (ws && aligned16(ws) && bytes >= kWsHeader) {
    v.err = static_cast<uint32_t*>(ws);
    v.payload = static_cast<char*>(ws) + kWsHeader;
    v.bytes = bytes - kWsHeader;
  }
  return v;
}
size_t with_header(size_t payload) { return payload ? kWsHeader + payload : 0; }

// GroupNorm couples: statistics exchange area for up to kMaxCouples couples
// ([couples][2 slots][2 halves][256 rows] float2, then [couples][2][2][8] flags)
constexpr int kMaxCouples = 128;
constexpr size_t kCoupleDataBytes = 2 * 2 * 256 * sizeof(float) * 2;
constexpr size_t kCoupleFlagBytes = 2 * 2 * 8 * sizeof(unsigned long long);
int couple_slots(int64_t M, int64_t N) {
  const int64_t units = ((M + 255) / 256) * (N / 512);
  return static_cast<int>(std::min<int64_t>(units, kMaxCouples));
}
size_t couple_ws_bytes(int64_t M, int64_t N) {
  return align_up(static_cast<size_t>(couple_slots(M, N)) * (kCoupleDataBytes + kCoupleFlagBytes), 256);
}
// True when the chain normalises 512-column groups and M spans CTA pairs: the
// case the couples (with a workspace) and clusters of four (without) serve.
bool gn512_pairs(const kf_epilogue* epi, int64_t M, int64_t N) {
  if (M <= 128 || !epi || !epi->ops) return false;
  for (int i = 0; i < epi->num_ops; ++i)
    if (epi->ops[i].kind == KF_OP_GROUPNORM)
      return epi->ops[i].groups > 0 && N % epi->ops[i].groups == 0 && N / epi->ops[i].groups == 512;
  return false;
}
// Per-call tag of the couples' flags: unique within the process, and seeded from
// the clock so that flags left in reused memory by another process do not match.
uint32_t next_epoch() {
  static std::atomic<uint32_t> ctr{static_cast<uint32_t>(
      std::chrono::steady_clock::now().time_since_epoch().count() * 2654435761ull)};
  uint32_t e = ctr.fetch_add(1);
  return e == 0 ? ctr.fetch_add(1) : e;
}

size_t lse_ws_bytes(int64_t M, int64_t N) {
  // upper bound over all tile widths (narrowest tile = most partials per row)
  return align_up(static_cast<size_t>(M) * static_cast<size_t>((N + 127) / 128) * sizeof(float2), 256);
}

// -------------------------------------------------------------- grouped core
struct GroupedArgs {
  const void* A;
  int64_t lda;
  int64_t a_rows;
  const int32_t* a_row_index;
  const void* B;
  int64_t ldb;
  int64_t b_group_stride;
  const int32_t* offsets;
  int32_t G;
  int64_t rows_total, N, K;
  void* C;
  int32_t c_dtype;
  int64_t ldc;
};

size_t grouped_ws_bytes(int64_t rows_total, int64_t K, bool gathered) {
  return gathered ? align_up(static_cast<size_t>(rows_total) * static_cast<size_t>(K) * 2, 256) : 0;
}

// Per-group bias and the gated SwiGLU of the MoE path (see TcParams).
struct GroupExtras {
  const void* gbias = nullptr;  // bf16, group stride gbias_ld
  int64_t gbias_ld = 0;
  bool sw_ext = false;
  float sw_alpha = 1.0f, sw_limit = 0.0f, sw_c = 0.0f;
  void* zero_ptr = nullptr;  // SwiGLU: cleared while its first units run (see TcParams)
  int64_t zero_bytes = 0;
  int64_t max_group_rows = 0;  // an upper bound on every group's rows, when the caller knows one (0: none)
};

// `pdl`: the previous kernel in the stream is one of this library's (MoE chain),
// so the launches here may be programmatic dependents of it.
// `ws`: the payload the gathered rows go to; `werr`: the call's error word.
kf_status grouped_core(const GroupedArgs& g, const ChainPlan& pl, void* ws, uint32_t* werr, cudaStream_t s,
                       const DevInfo& di, bool pdl, const GroupExtras* ex = nullptr) {
  const void* A = g.A;
  int64_t lda = g.lda;
  if (g.a_row_index) {
    kf_status st = cuda_status(
        gather_rows_launch(g.A, g.lda, g.a_rows, g.a_row_index, g.rows_total, g.K, ws, werr, di.err, s, pdl));
    if (st != KF_OK) return st;
    A = ws;
    lda = g.K;
  }
  const int bn = pick_grouped_outn(pl.mode, g.N, g.rows_total, g.G, di.nsm);
  if (bn == 0) return KF_ERR_UNSUPPORTED;
  const int outn = pl.mode == kModeSwiglu ? bn / 2 : bn;
  const int64_t nb = pl.mode == kModeSwiglu ? 2 * g.N : g.N;
  // groups known to hold at most 64 rows take the variant with 64-row A slots
  // (and a deeper ring), where there is one
  const int ar = ex && ex->max_group_rows > 0 && ex->max_group_rows <= 64 && tc_grouped_has(pl.mode, bn, 64) ? 64 : kBM;
  CUtensorMap ma, mb;
  kf_status st = make_map(&ma, A, g.K, g.rows_total, lda * 2, 1, 0, ar, 2);
  if (st != KF_OK) return st;
  st = make_map(&mb, g.B, g.K, nb, g.ldb * 2, g.G, g.b_group_stride * 2, mode_box(pl.mode, bn), 3);
  if (st != KF_OK) return st;
  TcParams p;
  std::memset(&p, 0, sizeof(p));
  p.M = static_cast<int32_t>(g.rows_total);
  p.N = static_cast<int32_t>(g.N);
  p.K = static_cast<int32_t>(g.K);
  p.tiles_n = static_cast<int32_t>((g.N + outn - 1) / outn);
  p.num_kb = static_cast<int32_t>((g.K + kBK - 1) / kBK);
  p.G = g.G;
  p.group_offsets = g.offsets;
  p.b_rows = static_cast<int32_t>(g.N);
  p.C = g.C;
  p.ldc = g.ldc;
  p.c_dtype = g.c_dtype;
  p.c_vec_ok = aligned16(g.C) && (g.ldc * elt_size(g.c_dtype)) % 16 == 0;
  p.row_scale = pl.row_scale;
  p.row_dst = pl.row_dst;
  p.dst_rows = static_cast<int32_t>(pl.dst_rows);
  fill_params_common(p, pl, werr, di.err);
  p.fast = g.c_dtype == KF_BF16 && pl.mode != kModeScatter;
  if (ex) {
    p.gbias = ex->gbias;
    p.gbias_ld = ex->gbias_ld;
    p.sw_ext = ex->sw_ext ? 1 : 0;
    p.sw_alpha = ex->sw_alpha;
    p.sw_limit = ex->sw_limit;
    p.sw_c = ex->sw_c;
    p.zero_ptr = ex->zero_ptr;
    p.zero_bytes = ex->zero_bytes;
  }
  const int64_t ub = ((g.rows_total + kBM - 1) / kBM + g.G) * p.tiles_n;
  const int grid = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(ub, di.nsm)));
  CUtensorMap mc;  // grouped outputs are masked per group: plain stores, no TMA map
  std::memset(&mc, 0, sizeof(mc));
  // after the gather (when there is one) the GEMM follows a library kernel
  return cuda_status(tc_grouped_launch(pl.mode, bn, ar, ma, mb, mc, p, grid, s, pdl || g.a_row_index != nullptr));
}

}  // namespace
}  // namespace kf

using namespace kf;

extern "C" {

const char* kf_status_string(int32_t s) {
  switch (s) {
    case KF_OK: return "ok";
    case KF_ERR_INVALID_ARG: return "invalid argument";
    case KF_ERR_UNSUPPORTED: return "unsupported dtype combination or op chain";
    case KF_ERR_MISALIGNED: return "misaligned pointer or stride (TMA needs 16-byte alignment)";
    case KF_ERR_WORKSPACE: return "workspace missing or too small";
    case KF_ERR_CUDA: return "CUDA error";
    case KF_ERR_DEVICE_TIMEOUT: return "device-side wait timed out";
    case KF_ERR_DEVICE_BOUNDS: return "device-resident index or offset out of range";
    default: return "unknown status";
  }
}

int32_t kf_abi_version(void) { return 2; }

kf_status kf_set_wait_timeout_ns(uint64_t ns) {
  g_wait_ns.store(ns == 0 ? kDefaultWaitNs : ns);
  return KF_OK;
}

}  // extern "C"

namespace {
// Synchronize `stream`, then read and clear the error word `word` (device memory).
kf_status read_clear_error(uint32_t* word, void* stream, uint32_t* raw) {
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return KF_ERR_CUDA;
  uint32_t v = 0, z = 0;
  if (cudaMemcpy(&v, word, sizeof(v), cudaMemcpyDeviceToHost) != cudaSuccess) return KF_ERR_CUDA;
  if (v && cudaMemcpy(word, &z, sizeof(z), cudaMemcpyHostToDevice) != cudaSuccess) return KF_ERR_CUDA;
  if (raw) *raw = v;
  if (v & (kErrWaitProducer | kErrWaitMma | kErrWaitEpilogue)) return KF_ERR_DEVICE_TIMEOUT;
  if (v & kErrBounds) return KF_ERR_DEVICE_BOUNDS;
  if (v & kErrLaunchShape) return KF_ERR_CUDA;
  return KF_OK;
}
}  // namespace

extern "C" {

kf_status kf_get_device_error(void* stream, uint32_t* raw) {
  DevInfo di;
  kf_status st = device_info(&di);
  if (st != KF_OK) return st;
  return read_clear_error(di.err, stream, raw);
}

kf_status kf_check_device_error(void* workspace, void* stream, uint32_t* raw) {
  if (!workspace || !aligned16(workspace)) return KF_ERR_INVALID_ARG;
  return read_clear_error(static_cast<uint32_t*>(workspace), stream, raw);
}

kf_status kf_workspace_init(void* workspace, size_t bytes, void* stream) {
  if (!workspace || !aligned16(workspace) || bytes < kWsHeader) return KF_ERR_INVALID_ARG;
  return cuda_status(cudaMemsetAsync(workspace, 0, kWsHeader, static_cast<cudaStream_t>(stream)));
}

size_t kf_fused_gemm_workspace(int64_t M, int64_t N, int64_t K, const kf_epilogue* epi) {
  (void)K;
  if (!epi || M <= 0 || N <= 0) return 0;
  for (int i = 0; i < epi->num_ops && epi->ops; ++i)
    if (epi->ops[i].kind == KF_OP_ROW_LOGSUMEXP || epi->ops[i].kind == KF_OP_ROW_SUM)
      return with_header(lse_ws_bytes(M, N));
  if (gn512_pairs(epi, M, N)) return with_header(couple_ws_bytes(M, N));  // optional: enables the couples
  return 0;
}

kf_status kf_fused_gemm(const void* X, int32_t xt, int64_t ldx, const void* W, int32_t wt, int64_t ldw, void* Y,
                        int32_t yt, int64_t ldy, int64_t M, int64_t N, int64_t K, const kf_epilogue* epi,
                        void* workspace, size_t ws_bytes, void* stream) {
  return kf_fused_gemm_ex(X, xt, ldx, W, wt, ldw, Y, yt, ldy, M, N, K, epi, workspace, ws_bytes, 0u, stream);
}

}  // extern "C"

namespace {
// kf_fused_gemm_ex on a split workspace: `payload` / `ws_bytes` is the scratch
// (row partials, GroupNorm exchange area), `werr` the call's error word (null:
// the device word only).
kf_status fused_gemm_impl(const void* X, int32_t xt, int64_t ldx, const void* W, int32_t wt, int64_t ldw, void* Y,
                          int32_t yt, int64_t ldy, int64_t M, int64_t N, int64_t K, const kf_epilogue* epi,
                          void* workspace, size_t ws_bytes, uint32_t* werr, uint32_t flags, void* stream) {
  if (flags & ~(KF_GEMM_F32_FFMA | KF_GEMM_F32_TF32X3)) return KF_ERR_INVALID_ARG;
  if ((flags & KF_GEMM_F32_FFMA) && (flags & KF_GEMM_F32_TF32X3)) return KF_ERR_INVALID_ARG;
  if (M < 0 || N < 0 || K < 1) return KF_ERR_INVALID_ARG;
  if (M > INT32_MAX || N > INT32_MAX || K > INT32_MAX) return KF_ERR_INVALID_ARG;
  if (M == 0 || N == 0) return KF_OK;  // empty problem: nothing to read or write
  if (!X || !W || !Y) return KF_ERR_INVALID_ARG;
  if (ldx < K || ldw < K) return KF_ERR_INVALID_ARG;
  if (!float_dtype(xt) || !float_dtype(wt) || !float_dtype(yt)) return KF_ERR_INVALID_ARG;
  ChainPlan pl;
  kf_status st = plan_chain(epi, N, false, &pl);
  if (st != KF_OK) return st;
  if (pl.mode != kModeLse && !pl.red_sum && ldy < N) return KF_ERR_INVALID_ARG;
  const bool f32_path = xt == KF_F32 && wt == KF_F32;
  // fp32 operands: FFMA for small problems, three tf32 tensor-core products for
  // large ones (>= 2^30 FLOP), or as the flags say
  bool tf32x3 = false;
  if (f32_path) {
    if (pl.mode != kModeStore) return KF_ERR_UNSUPPORTED;  // element-wise chains only
    const bool big = 2.0 * static_cast<double>(M) * static_cast<double>(N) * static_cast<double>(K) >= 1073741824.0;
    tf32x3 = (flags & KF_GEMM_F32_TF32X3) || (big && !(flags & KF_GEMM_F32_FFMA));
    if (tf32x3) {
      if (!aligned16(X) || !aligned16(W) || ldx % 4 != 0 || ldw % 4 != 0) {
        if (flags & KF_GEMM_F32_TF32X3) return KF_ERR_MISALIGNED;
        tf32x3 = false;  // automatic choice: the FFMA path takes any layout
      }
    }
    if (!tf32x3 && yt != KF_F32) return KF_ERR_UNSUPPORTED;
  } else {
    // tensor-core path: A and B both bf16 or both fp16 (one operand format per MMA)
    if (xt != wt || (xt != KF_BF16 && xt != KF_F16)) return KF_ERR_UNSUPPORTED;
    if (!aligned16(X) || !aligned16(W) || ldx % 8 != 0 || ldw % 8 != 0) return KF_ERR_MISALIGNED;
    if ((pl.mode == kModeLse || pl.red_sum) &&
        (!workspace || !aligned16(workspace) || ws_bytes < lse_ws_bytes(M, N)))
      return KF_ERR_WORKSPACE;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  DevInfo di;
  st = device_info(&di);
  if (st != KF_OK) return st;
  if (!werr) werr = di.err;

  if (tf32x3) {
    // tile width: 256 columns (each MMA does twice the work of a 128-wide one
    // for the same issue cost) when that still gives every SM a tile
    const int64_t tm = (M + 127) / 128;
    const int bn = (tm * ((N + 255) / 256) >= di.nsm && tf32x3_has(256)) ? 256 : 128;
    CUtensorMap ma, mb;
    st = make_map_f32(&ma, X, K, M, ldx * 4, 128);
    if (st != KF_OK) return st;
    st = make_map_f32(&mb, W, K, N, ldw * 4, bn);
    if (st != KF_OK) return st;
    Tf32Params tp;
    std::memset(&tp, 0, sizeof(tp));
    tp.M = static_cast<int32_t>(M);
    tp.N = static_cast<int32_t>(N);
    tp.K = static_cast<int32_t>(K);
    tp.tiles_m = static_cast<int32_t>(tm);
    tp.tiles_n = static_cast<int32_t>((N + bn - 1) / bn);
    tp.num_kb = static_cast<int32_t>((K + 31) / 32);
    tp.n_ops = pl.n_pre;
    for (int i = 0; i < pl.n_pre; ++i) tp.ops[i] = pl.pre[i];
    tp.Y = Y;
    tp.ldy = ldy;
    tp.y_dtype = yt;
    tp.y_vec_ok = aligned16(Y) && (ldy * elt_size(yt)) % 16 == 0;
    tp.err = werr;
    tp.err_dev = di.err;
    tp.wait_ns = g_wait_ns.load();
    tp.drain_ns = std::max<uint64_t>(tp.wait_ns, 1000000000ull);
    const int64_t tiles = static_cast<int64_t>(tp.tiles_m) * tp.tiles_n;
    const int grid = static_cast<int>(std::min<int64_t>(tiles, di.nsm));
    return cuda_status(tf32x3_launch(bn, ma, mb, tp, grid, s));
  }
  if (f32_path) {
    SimtParams sp;
    std::memset(&sp, 0, sizeof(sp));
    sp.X = static_cast<const float*>(X);
    sp.W = static_cast<const float*>(W);
    sp.Y = static_cast<float*>(Y);
    sp.ldx = ldx;
    sp.ldw = ldw;
    sp.ldy = ldy;
    sp.M = static_cast<int32_t>(M);
    sp.N = static_cast<int32_t>(N);
    sp.K = static_cast<int32_t>(K);
    sp.n_ops = pl.n_pre;
    for (int i = 0; i < pl.n_pre; ++i) sp.ops[i] = pl.pre[i];
    return cuda_status(simt_gemm_f32_launch(sp, s));
  }

  // CTA pairs (256-row tiles, tcgen05.mma.cta_group::2) unless one 128-row
  // tile already covers M
  const bool cta2 = M > kBM && di.nsm >= 2;
  // GroupNorm over 512-column groups: clusters of two CTA pairs, one 256-column
  // half of each group per pair, so each CTA double-buffers its accumulators
  const bool quad = cta2 && pl.mode == kModeGroupNorm && pl.gs == 512 && di.nsm >= 4 && tc_dense4_has(pl.mode, 256);
  // with a workspace for the statistics exchange: couples of CTA pairs instead
  // (all co-resident pairs work; clusters of four leave SMs idle)
  const bool couple = quad && !pl.red_sum && tc_couple_has(pl.mode, 256) && workspace && aligned16(workspace) &&
                      ws_bytes >= couple_ws_bytes(M, N);
  int bn = 0, sub = 1;
  int64_t tiles_n = 0;
  if (quad) {
    bn = 256;
    tiles_n = N / 512;
  } else if (pl.mode == kModeGroupNorm) {
    bn = 256;
    sub = pl.gs == 512 ? 2 : 1;
    tiles_n = (N + bn * sub - 1) / (bn * sub);
  } else {
    bn = pick_dense_bn(pl.mode, M, N, di.nsm, cta2);
    if (bn == 0) return KF_ERR_UNSUPPORTED;
    tiles_n = (N + bn - 1) / bn;
  }
  CUtensorMap ma, mb;
  const CUtensorMapDataType op_dt = xt == KF_F16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  st = make_map(&ma, X, K, M, ldx * 2, 1, 0, kBM, 2, op_dt);
  if (st != KF_OK) return st;
  st = make_map(&mb, W, K, N, ldw * 2, 1, static_cast<uint64_t>(N) * ldw * 2, cta2 ? bn / 2 : bn, 3, op_dt);
  if (st != KF_OK) return st;
  TcParams p;
  std::memset(&p, 0, sizeof(p));
  p.M = static_cast<int32_t>(M);
  p.N = static_cast<int32_t>(N);
  p.K = static_cast<int32_t>(K);
  p.tiles_m = static_cast<int32_t>((M + (cta2 ? 2 * kBM : kBM) - 1) / (cta2 ? 2 * kBM : kBM));
  p.tiles_n = static_cast<int32_t>(tiles_n);
  p.num_kb = static_cast<int32_t>((K + kBK - 1) / kBK);
  p.total_units = p.tiles_m * p.tiles_n;
  p.C = Y;
  p.ldc = ldy;
  p.c_dtype = yt;
  p.c_vec_ok = aligned16(Y) && (ldy * elt_size(yt)) % 16 == 0;
  if (pl.mode == kModeLse || pl.red_sum) p.lse_part = static_cast<float2*>(workspace);
  // GroupNorm + row sum: one partial per 256-column block of a row
  p.red_parts = pl.mode == kModeGroupNorm ? static_cast<int32_t>((N + 255) / 256) : p.tiles_n;
  fill_params_common(p, pl, werr, di.err);
  CUtensorMap mc;
  std::memset(&mc, 0, sizeof(mc));
  if ((pl.mode == kModeStore || pl.mode == kModeGroupNorm) && !pl.red_sum && yt == KF_BF16 && p.c_vec_ok) {
    st = make_map_out(&mc, Y, static_cast<uint64_t>(N), static_cast<uint64_t>(M), static_cast<uint64_t>(ldy) * 2);
    if (st != KF_OK) return st;
    p.c_tma = 1;
  }
  // 16-bit results: reduced-precision activations suffice (not under a row
  // reduction: its sum of thousands of values needs each term at fp32)
  p.fast = (yt == KF_BF16 || yt == KF_F16) && pl.mode != kModeLse && !pl.red_sum;
  p.ab_f16 = xt == KF_F16;
  const int grid = cta2 ? 2 * std::min(p.total_units, di.nsm / 2) : std::min(p.total_units, di.nsm);
  // a compiled chain program, if the chain matches one (bf16 operands staged)
  int sig = kSigGeneric;
  CUtensorMap mr;
  std::memset(&mr, 0, sizeof(mr));
  // bias-GELU-scale-residual on CTA pairs: the residual tile goes through shared
  // memory (TMA in, in-place result, TMA out) -- needs TMA-able residual and
  // output and whole 8-column bias units
  if (pl.mode == kModeStore && ProgGeluChain::matches(pl.pre, pl.n_pre) && p.vec_op == 0 && p.res_op == 3 && cta2 &&
      p.c_tma && N % 8 == 0 && tc_dense2_has_prog(pl.mode, bn, kSigBiasGeluScaleRes)) {
    sig = kSigBiasGeluScaleRes;
    const DevOp& ro = pl.pre[3];
    st = make_map_blk64(&mr, ro.p0, static_cast<uint64_t>(N), static_cast<uint64_t>(M), static_cast<uint64_t>(ro.ld) * 2);
    if (st != KF_OK) return st;
    st = make_map_blk64(&mc, Y, static_cast<uint64_t>(N), static_cast<uint64_t>(M), static_cast<uint64_t>(ldy) * 2);
    if (st != KF_OK) return st;
  }
  else if (pl.mode == kModeGroupNorm && ProgBias::matches(pl.pre, pl.n_pre) && ProgSilu::matches(pl.post, pl.n_post))
    sig = kSigBiasNormSilu;
  else if (pl.mode == kModeLse && ProgScale::matches(pl.pre, pl.n_pre))
    sig = kSigScaleLse;
  if (couple) {
    const int slots = couple_slots(M, N);
    p.gx_data = static_cast<float2*>(workspace);
    p.gx_flag = reinterpret_cast<unsigned long long*>(static_cast<char*>(workspace) + slots * kCoupleDataBytes);
    p.gx_epoch = next_epoch();
    st = cuda_status(tc_couple_launch(pl.mode, bn, sig, ma, mb, mc, p, slots, s));
  } else if (quad)
    st = cuda_status(tc_dense4_launch(pl.mode, bn, sig, ma, mb, mc, p, s));
  else
    st = cuda_status(tc_dense_launch(pl.mode, bn, cta2, sig, ma, mb, mc, mr, p, sub, grid, s));
  if (st != KF_OK || (pl.mode != kModeLse && !pl.red_sum)) return st;
  LseCombineParams cp;
  std::memset(&cp, 0, sizeof(cp));
  cp.part = p.lse_part;
  cp.M = p.M;
  cp.parts = p.red_parts;
  cp.out = Y;
  cp.out_dtype = yt;
  cp.red_sum = pl.red_sum ? 1 : 0;
  cp.n_post = pl.n_fin;
  for (int i = 0; i < pl.n_fin; ++i) cp.post[i] = pl.fin[i];
  return cuda_status(lse_combine_launch(cp, s, true));
}
}  // namespace

extern "C" {

kf_status kf_fused_gemm_ex(const void* X, int32_t xt, int64_t ldx, const void* W, int32_t wt, int64_t ldw, void* Y,
                           int32_t yt, int64_t ldy, int64_t M, int64_t N, int64_t K, const kf_epilogue* epi,
                           void* workspace, size_t ws_bytes, uint32_t flags, void* stream) {
  const WsView v = split_ws(workspace, ws_bytes);
  return fused_gemm_impl(X, xt, ldx, W, wt, ldw, Y, yt, ldy, M, N, K, epi, v.payload, v.bytes, v.err, flags, stream);
}

kf_status kf_moe_route(const float* logits, int64_t T, int32_t E, int32_t k, int32_t* topk_ids, float* topk_w,
                       int32_t* offsets, int32_t* sorted_token, float* sorted_w, void* stream) {
  if (T < 0 || E < 1 || E > 256 || k < 1 || k > E) return KF_ERR_INVALID_ARG;
  if (T * k > INT32_MAX) return KF_ERR_INVALID_ARG;
  if (!offsets || (T > 0 && (!logits || !topk_ids || !topk_w || !sorted_token || !sorted_w)))
    return KF_ERR_INVALID_ARG;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  kf_status st = cuda_status(route_topk_launch(logits, static_cast<int32_t>(T), E, k, topk_ids, topk_w, s));
  if (st != KF_OK) return st;
  return cuda_status(route_sort_launch(topk_ids, topk_w, static_cast<int32_t>(T), E, k, offsets, sorted_token,
                                       sorted_w, nullptr, s, true));
}

size_t kf_grouped_gemm_workspace(int64_t rows_total, int64_t N, int64_t K, int32_t G, int32_t gathered,
                                 const kf_epilogue* epi) {
  (void)N;
  (void)G;
  (void)epi;
  if (rows_total <= 0 || K <= 0) return 0;
  return with_header(grouped_ws_bytes(rows_total, K, gathered != 0));
}

kf_status kf_grouped_gemm(const void* A, int32_t at, int64_t lda, int64_t a_rows, const int32_t* a_row_index,
                          const void* B, int32_t bt, int64_t ldb, int64_t b_group_stride, const int32_t* offsets,
                          int32_t G, int64_t rows_total, int64_t N, int64_t K, void* C, int32_t ct, int64_t ldc,
                          const kf_epilogue* epi, void* workspace, size_t ws_bytes, void* stream) {
  if (rows_total < 0 || N < 1 || K < 1 || G < 1 || G > kMaxGroups) return KF_ERR_INVALID_ARG;
  if (rows_total > INT32_MAX || N > INT32_MAX || K > INT32_MAX) return KF_ERR_INVALID_ARG;
  if (rows_total == 0) return KF_OK;  // no rows: nothing to read or write
  if (!A || !B || !C || !offsets) return KF_ERR_INVALID_ARG;
  if (lda < K || ldb < K || ldc < N || b_group_stride < 0) return KF_ERR_INVALID_ARG;
  if (a_row_index && a_rows < 1) return KF_ERR_INVALID_ARG;
  if (at != KF_BF16 || bt != KF_BF16) return KF_ERR_UNSUPPORTED;
  if (!float_dtype(ct)) return KF_ERR_INVALID_ARG;
  ChainPlan pl;
  kf_status st = plan_chain(epi, N, true, &pl);
  if (st != KF_OK) return st;
  if (pl.mode == kModeScatter && ct != KF_F32) return KF_ERR_UNSUPPORTED;
  const int64_t nb = pl.mode == kModeSwiglu ? 2 * N : N;
  if (G > 1 && b_group_stride < nb * ldb) return KF_ERR_INVALID_ARG;
  if (!aligned16(A) || !aligned16(B) || lda % 8 != 0 || ldb % 8 != 0 || b_group_stride % 8 != 0)
    return KF_ERR_MISALIGNED;
  if (a_row_index && K % 8 != 0) return KF_ERR_MISALIGNED;
  const WsView v = split_ws(workspace, ws_bytes);
  if (a_row_index && (!v.payload || v.bytes < grouped_ws_bytes(rows_total, K, true))) return KF_ERR_WORKSPACE;
  DevInfo di;
  st = device_info(&di);
  if (st != KF_OK) return st;
  GroupedArgs g{A, lda, a_row_index ? a_rows : rows_total, a_row_index, B, ldb,
                G > 1 ? b_group_stride : nb * ldb, offsets, G, rows_total, N, K, C, ct, ldc};
  return grouped_core(g, pl, v.payload, v.err ? v.err : di.err, static_cast<cudaStream_t>(stream), di, false);
}

// Workspace layout of kf_moe_ffn (each region 256-byte aligned):
//   topk_ids i32 [T k] | topk_w f32 [T k] | offsets i32 [E+1] | sorted_token i32 [T k]
//   | sorted_w f32 [T k] | Xg bf16 [T k, H] | h bf16 [T k, I] | Yacc f32 [T, H]
struct MoeLayout {
  size_t ids, w, off, st, sw, cnt, xg, h, yacc, pos, yp, total;
};
// pairs from which the routing sort runs on many blocks
constexpr int64_t kSortMultiBlockPairs = 2048;
// deterministic mode adds: pair_pos i32 [T k] | Yp f32 [T k, H]
static MoeLayout moe_layout(int64_t T, int64_t H, int64_t I, int32_t E, int32_t k, uint32_t flags = 0) {
  MoeLayout L;
  const size_t P = static_cast<size_t>(T) * static_cast<size_t>(k);
  size_t o = 0;
  auto take = [&](size_t bytes) {
    size_t at = o;
    o = align_up(o + bytes, 256);
    return at;
  };
  L.ids = take(P * 4);
  L.w = take(P * 4);
  L.off = take(static_cast<size_t>(E + 1) * 4);
  L.st = take(P * 4);
  L.sw = take(P * 4);
  L.cnt = take(static_cast<size_t>(route_sort_mb_blocks(static_cast<int32_t>(P))) * static_cast<size_t>(E) * 4);
  L.xg = take(P * static_cast<size_t>(H) * 2);
  L.h = take(P * static_cast<size_t>(I) * 2);
  L.yacc = take(static_cast<size_t>(T) * static_cast<size_t>(H) * 4);
  L.pos = L.yp = 0;
  if (flags & KF_MOE_DETERMINISTIC) {
    L.pos = take(P * 4);
    L.yp = take(P * static_cast<size_t>(H) * 4);
  }
  L.total = o;
  return L;
}

size_t kf_moe_ffn_workspace(int64_t T, int64_t H, int64_t I, int32_t E, int32_t k) {
  return kf_moe_ffn_workspace_ex(T, H, I, E, k, 0);
}

size_t kf_moe_ffn_workspace_ex(int64_t T, int64_t H, int64_t I, int32_t E, int32_t k, uint32_t flags) {
  if (T < 0 || H < 1 || I < 1 || E < 1 || k < 1) return 0;
  return kWsHeader + moe_layout(T, H, I, E, k, flags).total;
}

kf_status kf_moe_ffn(const void* X, const float* logits, const void* W_gu, const void* W_down, void* Y, int64_t T,
                     int64_t H, int64_t I, int32_t E, int32_t k, void* workspace, size_t ws_bytes,
                     int32_t* topk_ids_out, float* topk_w_out, void* stream) {
  return kf_moe_ffn_ex(X, logits, W_gu, W_down, Y, T, H, I, E, k, 0, workspace, ws_bytes, topk_ids_out, topk_w_out,
                       stream);
}

}  // extern "C"

namespace {
// Residual add + RMSNorm that replaces the MoE finalize's plain bf16 output.
struct BlockTail {
  const void* R;
  const void* gamma;
  float eps;
  void* R_out;
};

kf_status moe_ffn_impl(const void* X, const float* logits, const void* W_gu, const void* W_down, void* Y, int64_t T,
                       int64_t H, int64_t I, int32_t E, int32_t k, uint32_t flags, void* workspace, size_t ws_bytes,
                       int32_t* topk_ids_out, float* topk_w_out, void* stream, const BlockTail* tail,
                       const kf_moe_act* act = nullptr) {
  if (flags & ~KF_MOE_DETERMINISTIC) return KF_ERR_INVALID_ARG;
  if (act && (!std::isfinite(act->alpha) || !(act->limit >= 0.0f) || !std::isfinite(act->limit) ||
              !std::isfinite(act->linear_offset)))
    return KF_ERR_INVALID_ARG;
  if (act && ((act->b_gu && !aligned16(act->b_gu)) || (act->b_down && !aligned16(act->b_down))))
    return KF_ERR_MISALIGNED;
  const bool det = (flags & KF_MOE_DETERMINISTIC) != 0;
  if (T < 0 || H < 1 || I < 1 || E < 1 || E > 256 || k < 1 || k > E) return KF_ERR_INVALID_ARG;
  if (T * k > INT32_MAX || H > INT32_MAX || I > INT32_MAX) return KF_ERR_INVALID_ARG;
  if (!X || !logits || !W_gu || !W_down || !Y) return KF_ERR_INVALID_ARG;
  if (!aligned16(X) || !aligned16(W_gu) || !aligned16(W_down) || !aligned16(Y) || H % 8 != 0 || I % 8 != 0)
    return KF_ERR_MISALIGNED;
  if (det && H % 4 != 0) return KF_ERR_MISALIGNED;
  if (T == 0) return KF_OK;
  const MoeLayout L = moe_layout(T, H, I, E, k, flags);
  const WsView v = split_ws(workspace, ws_bytes);
  if (!v.payload || v.bytes < L.total) return KF_ERR_WORKSPACE;
  DevInfo di;
  kf_status st = device_info(&di);
  if (st != KF_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* ws = static_cast<char*>(v.payload);
  uint32_t* werr = v.err;
  auto* ids = reinterpret_cast<int32_t*>(ws + L.ids);
  auto* w = reinterpret_cast<float*>(ws + L.w);
  auto* off = reinterpret_cast<int32_t*>(ws + L.off);
  auto* stok = reinterpret_cast<int32_t*>(ws + L.st);
  auto* sw = reinterpret_cast<float*>(ws + L.sw);
  void* xg = ws + L.xg;
  void* h = ws + L.h;
  auto* yacc = reinterpret_cast<float*>(ws + L.yacc);
  const int64_t P = T * k;

  int32_t* pos = det ? reinterpret_cast<int32_t*>(ws + L.pos) : nullptr;
  // the fp32 scatter target is cleared by the gate/up GEMM's epilogue warps
  // while its first units run (the down GEMM starts after that grid completes),
  // so no separate pass over it and the kernels of the chain follow one another
  // directly (each a programmatic dependent of the last)
  st = cuda_status(route_topk_launch(logits, static_cast<int32_t>(T), E, k, ids, w, s));
  if (st != KF_OK) return st;
  if (P >= kSortMultiBlockPairs)
    st = cuda_status(route_sort_mb_launch(ids, w, static_cast<int32_t>(T), E, k, off, stok, sw, pos,
                                          reinterpret_cast<int32_t*>(ws + L.cnt), s, true));
  else
    st = cuda_status(route_sort_launch(ids, w, static_cast<int32_t>(T), E, k, off, stok, sw, pos, s, true));
  if (st != KF_OK) return st;
  // a token's k experts are distinct, so no expert holds more than T rows
  // gate/up: h = silu(Xg W_gate[e]^T) * (Xg W_up[e]^T), rows gathered by token
  {
    kf_epilogue_op op{};
    op.kind = KF_OP_SWIGLU;
    kf_epilogue epi{1, &op};
    ChainPlan pl;
    st = plan_chain(&epi, I, true, &pl);
    if (st != KF_OK) return st;
    GroupedArgs g{X, H, T, stok, W_gu, H, 2 * I * H, off, E, P, I, H, h, KF_BF16, I};
    GroupExtras ex;
    ex.max_group_rows = T;
    if (!det) {
      ex.zero_ptr = yacc;
      ex.zero_bytes = T * H * 4;
    }
    if (act) {
      ex.gbias = act->b_gu;
      ex.gbias_ld = 2 * I;
      ex.sw_ext = true;
      ex.sw_alpha = act->alpha;
      ex.sw_limit = act->limit;
      ex.sw_c = act->linear_offset;
    }
    st = grouped_core(g, pl, xg, werr, s, di, true, &ex);
    if (st != KF_OK) return st;
  }
  if (det) {
    // down: Yp[r] = w_r * (h_r W_down[e]^T), then a fixed-order sum per token
    kf_epilogue_op op{};
    op.kind = KF_OP_ROW_SCALE;
    op.p0 = sw;
    op.p_dtype = KF_F32;
    kf_epilogue epi{1, &op};
    ChainPlan pl;
    st = plan_chain(&epi, H, true, &pl);
    if (st != KF_OK) return st;
    float* yp = reinterpret_cast<float*>(ws + L.yp);
    GroupedArgs g{h, I, P, nullptr, W_down, I, H * I, off, E, P, H, I, yp, KF_F32, H};
    GroupExtras ex;
    ex.max_group_rows = T;
    if (act) {
      ex.gbias = act->b_down;
      ex.gbias_ld = H;
    }
    st = grouped_core(g, pl, nullptr, werr, s, di, true, &ex);
    if (st != KF_OK) return st;
    if (tail)
      st = cuda_status(moe_add_rmsnorm_launch(nullptr, yp, pos, k, T, H, tail->R, tail->gamma, tail->eps, tail->R_out, Y,
                                              s, true));
    else
      st = cuda_status(moe_finalize_launch(yp, pos, T, k, H, Y, s, true));
    if (st != KF_OK) return st;
  } else {
    // down: Yacc[token] += w * (h W_down[e]^T), then bf16
    kf_epilogue_op op{};
    op.kind = KF_OP_ROW_SCALE_SCATTER_ADD;
    op.p0 = sw;
    op.p1 = stok;
    op.p_dtype = KF_F32;
    op.ld = T;
    kf_epilogue epi{1, &op};
    ChainPlan pl;
    st = plan_chain(&epi, H, true, &pl);
    if (st != KF_OK) return st;
    GroupedArgs g{h, I, P, nullptr, W_down, I, H * I, off, E, P, H, I, yacc, KF_F32, H};
    GroupExtras ex;
    ex.max_group_rows = T;
    if (act) {
      ex.gbias = act->b_down;
      ex.gbias_ld = H;
    }
    st = grouped_core(g, pl, nullptr, werr, s, di, true, &ex);
    if (st != KF_OK) return st;
    if (tail)
      st = cuda_status(moe_add_rmsnorm_launch(yacc, nullptr, nullptr, k, T, H, tail->R, tail->gamma, tail->eps,
                                              tail->R_out, Y, s, true));
    else
      st = cuda_status(cvt_f32_bf16_launch(yacc, Y, T * H, s, true));
    if (st != KF_OK) return st;
  }
  if (topk_ids_out &&
      cudaMemcpyAsync(topk_ids_out, ids, static_cast<size_t>(P) * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return KF_ERR_CUDA;
  if (topk_w_out &&
      cudaMemcpyAsync(topk_w_out, w, static_cast<size_t>(P) * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return KF_ERR_CUDA;
  return KF_OK;
}
}  // namespace

extern "C" {

kf_status kf_moe_ffn_ex(const void* X, const float* logits, const void* W_gu, const void* W_down, void* Y, int64_t T,
                        int64_t H, int64_t I, int32_t E, int32_t k, uint32_t flags, void* workspace, size_t ws_bytes,
                        int32_t* topk_ids_out, float* topk_w_out, void* stream) {
  return moe_ffn_impl(X, logits, W_gu, W_down, Y, T, H, I, E, k, flags, workspace, ws_bytes, topk_ids_out, topk_w_out,
                      stream, nullptr);
}

kf_status kf_moe_ffn_act(const void* X, const float* logits, const void* W_gu, const void* W_down,
                         const kf_moe_act* act, void* Y, int64_t T, int64_t H, int64_t I, int32_t E, int32_t k,
                         uint32_t flags, void* workspace, size_t ws_bytes, int32_t* topk_ids_out, float* topk_w_out,
                         void* stream) {
  if (!act) return KF_ERR_INVALID_ARG;
  return moe_ffn_impl(X, logits, W_gu, W_down, Y, T, H, I, E, k, flags, workspace, ws_bytes, topk_ids_out, topk_w_out,
                      stream, nullptr, act);
}

kf_status kf_moe_ffn_add_rmsnorm(const void* X, const float* logits, const void* W_gu, const void* W_down,
                                 const void* R, const void* gamma, float eps, void* R_out, void* Y, int64_t T,
                                 int64_t H, int64_t I, int32_t E, int32_t k, uint32_t flags, void* workspace,
                                 size_t ws_bytes, int32_t* topk_ids_out, float* topk_w_out, void* stream) {
  if (!(eps >= 0.0f) || eps > 1e30f) return KF_ERR_INVALID_ARG;
  if (T > 0 && (!R || !gamma || !R_out)) return KF_ERR_INVALID_ARG;
  if (H > kAddRmsNormMaxH) return KF_ERR_UNSUPPORTED;
  if (T > 0 && (!aligned16(R) || !aligned16(gamma) || !aligned16(R_out))) return KF_ERR_MISALIGNED;
  const BlockTail tail{R, gamma, eps, R_out};
  return moe_ffn_impl(X, logits, W_gu, W_down, Y, T, H, I, E, k, flags, workspace, ws_bytes, topk_ids_out, topk_w_out,
                      stream, &tail);
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free variant of the row log-sum-exp GEMM.  Its per-tile row
// partials live in a fixed file-scope device array instead of a caller
// workspace, for callers that cannot allocate device memory themselves.
// ---------------------------------------------------------------------------
namespace kf {
namespace {

constexpr size_t kNoAllocScratchBytes = size_t(4) << 20;  // 4 MiB, resident on every device that loads the library
static __device__ __align__(256) float2 g_kf_noalloc_scratch[kNoAllocScratchBytes / sizeof(float2)];

struct NoAllocScratch {
  bool init = false;
  void* ptr = nullptr;
};
NoAllocScratch g_noalloc[kMaxDevices];
std::mutex g_noalloc_mu;

// Device address of the scratch array on the current device.  The symbol's
// name is only a host-side handle; the address is looked up once per device
// (with that device current) and cached.
kf_status noalloc_scratch(void** out) {
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= kMaxDevices) return KF_ERR_CUDA;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  NoAllocScratch& s = g_noalloc[d];
  if (!s.init) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_kf_noalloc_scratch) != cudaSuccess || p == nullptr) return KF_ERR_CUDA;
    s.ptr = p;
    s.init = true;
  }
  *out = s.ptr;
  return KF_OK;
}

}  // namespace
}  // namespace kf

extern "C" size_t kf_fused_gemm_lse_noalloc_max_bytes(void) { return kf::kNoAllocScratchBytes; }

extern "C" kf_status kf_fused_gemm_lse_noalloc(const void* X, int32_t xt, int64_t ldx, const void* W, int32_t wt,
                                               int64_t ldw, void* Y, int32_t yt, int64_t M, int64_t N, int64_t K,
                                               const kf_epilogue* epi, void* stream) {
  bool has_lse = false;
  if (epi && epi->ops)
    for (int i = 0; i < epi->num_ops && i < kf::kMaxOps; ++i) has_lse |= epi->ops[i].kind == KF_OP_ROW_LOGSUMEXP;
  if (!has_lse) return KF_ERR_INVALID_ARG;  // this variant is the row log-sum-exp GEMM only
  if (M < 0 || N < 0) return KF_ERR_INVALID_ARG;
  if (M == 0 || N == 0) return KF_OK;
  const size_t need = kf::lse_ws_bytes(M, N);
  if (need > kf::kNoAllocScratchBytes) return KF_ERR_WORKSPACE;  // problem exceeds the fixed scratch
  void* scratch = nullptr;
  kf_status st = kf::noalloc_scratch(&scratch);
  if (st != KF_OK) return st;
  // the whole array holds row partials; device-side errors go to the device word
  return fused_gemm_impl(X, xt, ldx, W, wt, ldw, Y, yt, 1, M, N, K, epi, scratch, kf::kNoAllocScratchBytes, nullptr,
                         0u, stream);
}

namespace kf {
namespace {

// Tile width of the QKV projection: whole heads per tile (a multiple of d),
// then the fewest tile-widths on the busiest SM (or CTA pair) + a fixed cost
// per tile, as for the dense store variants.
// Calls of at most this many tokens (the decode kernel's largest token box) take
// the cluster-split decode kernel; with both kernels launched as programmatic
// dependents that prefetch their weights, it is the faster one up to there
// (gpt-oss-20b shape, back to back: 56 tokens 17.0 against 18.8 us, 64 tokens
// 17.1 against 19.0 us)
constexpr int64_t kQkvClusterMaxT = 64;
static_assert(kQkvClusterMaxT <= kQkvDecodeMaxRows, "the decode kernel's token box");

int pick_rope_bn(int64_t M, int64_t N, int d, int nsm, bool cta2) {
  static const int cand[] = {256, 128, 64};
  int best = 0;
  int64_t best_cost = INT64_MAX;
  const int64_t rows = cta2 ? 2 * kBM : kBM;
  const int64_t workers = cta2 ? nsm / 2 : nsm;
  const int64_t tm = (M + rows - 1) / rows;
  for (int bn : cand) {
    if (bn % d != 0 || !tc_rope_has(bn, cta2)) continue;
    const int64_t tiles = tm * ((N + bn - 1) / bn);
    const int64_t cost = ((tiles + workers - 1) / workers) * (bn + 48);
    if (cost < best_cost) {
      best_cost = cost;
      best = bn;
    }
  }
  return best;
}

}  // namespace
}  // namespace kf

extern "C" kf_status kf_qkv_rope_kv(const void* X, const void* W, int32_t xw_dtype, int64_t ldx, int64_t ldw,
                                    const void* bias, int32_t bias_dtype, const int32_t* positions,
                                    const int32_t* cache_rows, const float* cos_t, const float* sin_t,
                                    int64_t max_pos, int64_t T, int64_t H, int32_t nq, int32_t nkv, int32_t d,
                                    void* q_out, int64_t ldq, void* k_cache, void* v_cache, int64_t ld_cache,
                                    int64_t cache_rows_n, int32_t out_dtype, void* stream) {
  using namespace kf;
  if (T < 0 || H < 1 || nq < 1 || nkv < 1 || d < 1 || max_pos < 1 || cache_rows_n < 1) return KF_ERR_INVALID_ARG;
  if (T > INT32_MAX || H > INT32_MAX || max_pos > INT32_MAX || cache_rows_n > INT32_MAX) return KF_ERR_INVALID_ARG;
  if (d % 64 != 0 || d > 256) return KF_ERR_UNSUPPORTED;
  const int64_t N = (static_cast<int64_t>(nq) + 2 * static_cast<int64_t>(nkv)) * d;
  if (N > INT32_MAX) return KF_ERR_INVALID_ARG;
  if (xw_dtype != KF_BF16 && xw_dtype != KF_F16) return KF_ERR_UNSUPPORTED;
  if (!float_dtype(out_dtype) || (bias && !float_dtype(bias_dtype))) return KF_ERR_INVALID_ARG;
  if (ldx < H || ldw < H || ldq < static_cast<int64_t>(nq) * d || ld_cache < static_cast<int64_t>(nkv) * d)
    return KF_ERR_INVALID_ARG;
  if (T == 0) return KF_OK;  // nothing to read or write
  if (!X || !W || !positions || !cache_rows || !cos_t || !sin_t || !q_out || !k_cache || !v_cache)
    return KF_ERR_INVALID_ARG;
  if (!aligned16(X) || !aligned16(W) || ldx % 8 != 0 || ldw % 8 != 0 || !aligned16(cos_t) || !aligned16(sin_t))
    return KF_ERR_MISALIGNED;
  // the bias is the chain before the rotation
  kf_epilogue_op bop;
  std::memset(&bop, 0, sizeof(bop));
  bop.kind = KF_OP_BIAS;
  bop.p0 = bias;
  bop.p_dtype = bias_dtype;
  kf_epilogue epi = {bias ? 1 : 0, &bop};
  ChainPlan pl;
  kf_status st = plan_chain(&epi, N, false, &pl);
  if (st != KF_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  DevInfo di;
  st = device_info(&di);
  if (st != KF_OK) return st;
  const bool cta2 = T > kBM && di.nsm >= 2;
  const int64_t num_kb = (H + kBK - 1) / kBK;
  if (T <= kQkvClusterMaxT && 256 % d == 0) {
    // few tokens: clusters of S CTAs split K over one 256-column tile and
    // reduce through distributed shared memory; S as large as keeps every
    // cluster of the call resident at once
    const int64_t tiles = (N + 255) / 256;
    int S = 1;
    for (int cand : {8, 6, 4, 2}) {
      int nc = 0;
      if (cand <= num_kb && qkv_decode_clusters(T, cand, &nc) == cudaSuccess && nc >= tiles) {
        S = cand;
        break;
      }
    }
    const CUtensorMapDataType dt = xw_dtype == KF_F16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    CUtensorMap ma, mb;
    st = make_map(&ma, X, H, T, ldx * 2, 1, 0, qkv_decode_box_rows(T), 2, dt);  // token boxes of 32 or 64 rows
    if (st != KF_OK) return st;
    st = make_map(&mb, W, H, N, ldw * 2, 1, static_cast<uint64_t>(N) * ldw * 2, 256, 3, dt);
    if (st != KF_OK) return st;
    QkvDecodeParams dp;
    std::memset(&dp, 0, sizeof(dp));
    dp.T = static_cast<int32_t>(T);
    dp.N = static_cast<int32_t>(N);
    dp.K = static_cast<int32_t>(H);
    dp.num_kb = static_cast<int32_t>(num_kb);
    dp.ab_f16 = xw_dtype == KF_F16;
    dp.bias = bias;
    dp.bias_dtype = bias_dtype;
    dp.cos_t = cos_t;
    dp.sin_t = sin_t;
    dp.positions = positions;
    dp.cache_rows = cache_rows;
    dp.max_pos = static_cast<int32_t>(max_pos);
    dp.rows = static_cast<int32_t>(cache_rows_n);
    dp.rope_d = d;
    dp.q_cols = nq * d;
    dp.rot_cols = (nq + nkv) * d;
    dp.q_out = q_out;
    dp.ldq = ldq;
    dp.k_cache = k_cache;
    dp.v_cache = v_cache;
    dp.ld_cache = ld_cache;
    dp.out_dtype = out_dtype;
    dp.err = di.err;
    dp.wait_ns = g_wait_ns.load();
    dp.drain_ns = std::max<uint64_t>(dp.wait_ns, 1000000000ull);
    dp.splits = S;
    return cuda_status(qkv_decode_launch(ma, mb, dp, static_cast<int>(tiles), s));
  }
  const int bn = pick_rope_bn(T, N, d, di.nsm, cta2);
  if (bn == 0) return KF_ERR_UNSUPPORTED;
  const CUtensorMapDataType op_dt =
      xw_dtype == KF_F16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  CUtensorMap ma, mb;
  st = make_map(&ma, X, H, T, ldx * 2, 1, 0, kBM, 2, op_dt);
  if (st != KF_OK) return st;
  st = make_map(&mb, W, H, N, ldw * 2, 1, static_cast<uint64_t>(N) * ldw * 2, cta2 ? bn / 2 : bn, 3, op_dt);
  if (st != KF_OK) return st;
  TcParams p;
  std::memset(&p, 0, sizeof(p));
  p.M = static_cast<int32_t>(T);
  p.N = static_cast<int32_t>(N);
  p.K = static_cast<int32_t>(H);
  p.tiles_m = static_cast<int32_t>((T + (cta2 ? 2 * kBM : kBM) - 1) / (cta2 ? 2 * kBM : kBM));
  p.tiles_n = static_cast<int32_t>((N + bn - 1) / bn);  // whole heads per tile; the last may hold fewer
  p.num_kb = static_cast<int32_t>(num_kb);
  p.total_units = p.tiles_m * p.tiles_n;
  p.C = q_out;
  p.ldc = ldq;
  p.c_dtype = out_dtype;
  p.c_vec_ok = aligned16(q_out) && (ldq * elt_size(out_dtype)) % 16 == 0;
  fill_params_common(p, pl, di.err, di.err);
  p.res_op = -1;
  p.vec_op = -1;
  p.fast = 0;
  p.ab_f16 = xw_dtype == KF_F16;
  p.row_dst = cache_rows;
  p.dst_rows = static_cast<int32_t>(cache_rows_n);
  p.rope_cos = cos_t;
  p.rope_sin = sin_t;
  p.rope_pos = positions;
  p.rope_max_pos = static_cast<int32_t>(max_pos);
  p.rope_d = d;
  p.rope_q_cols = nq * d;
  p.rope_rot_cols = (nq + nkv) * d;
  p.k_cache = k_cache;
  p.v_cache = v_cache;
  p.ld_cache = ld_cache;
  p.kv_vec_ok = aligned16(k_cache) && aligned16(v_cache) && (ld_cache * elt_size(out_dtype)) % 16 == 0;
  const int grid = cta2 ? 2 * std::min(p.total_units, di.nsm / 2) : std::min(p.total_units, di.nsm);
  return cuda_status(tc_rope_launch(bn, cta2, ma, mb, p, grid, s));
}
