/*
 * kf_oracle.c -- plain, slow, fp64 CPU oracle of the fused GEMM + tail path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path links, loads or calls
 * this file; only the tests, the smoke check and the benchmark's CPU-baseline
 * leg do.  It shares no code, header, table or constant with the CUDA library.
 *
 * What it computes is the plain definition of each step, in double precision:
 *   - operands are read at their stored values (bf16 bits widened exactly, or
 *     fp32 widened exactly) -- the "mixed precision" of the paper (Sec. IV-B,
 *     discussion of Table 3: 16-bit matmul inputs, wider accumulation and
 *     post-processing) means the fused kernel must reach the result of the
 *     unfused chain; the oracle is that result in exact-as-possible arithmetic;
 *   - the GEMM is a triple loop, s_ij = sum_k x_ik w_jk (both operands K-major);
 *   - each tail op of the chain is applied in list order by its formula
 *     ("layer-wise fusion", Sec. IV-B: the post-GEMM sequence of operations);
 *   - row log-sum-exp and GroupNorm are the plain two-pass definitions (the
 *     paper's single-pass/online forms, Sec. IV-B, reach the same value up to
 *     rounding order); the row sum (one reading of the "Sum" that ends the
 *     chains of Table 3, Sec. IV-B) is the plain sum over the row's columns;
 *   - the MoE expert FFN (gpt-oss decode path, Sec. IV-A) is written per token as
 *     Y_t = sum_j w_tj * W_down[e_tj] (silu(W_gate[e_tj] x_t) * (W_up[e_tj] x_t)),
 *     with the intermediate h rounded to bf16 (the down GEMM consumes bf16 h);
 *     the "MoE finalize" kernel of Table 1 is the routing-weighted sum over j.
 *   - the block tail after the MoE FFN (Sec. IV-A: "Fused Add + RMSNorm" and
 *     "MoE finalize" of the gpt-oss decode path; Sec. V: fusing kernels of one
 *     block) is the residual add and RMS normalisation of the new residual
 *     stream: R_out = bf16(R + Y), normed_j = R_out_j / sqrt(mean(R_out^2) + eps)
 *     * gamma_j -- the norm reads the stored (bf16) residual, as the next layer
 *     would;
 *   - the attention input projection with its tail (the Bias + RoPE + KV update
 *     kernel of the gpt-oss decode path, Sec. IV-A and Table 1, here as the tail
 *     of the QKV GEMM; the paper gives no formula, this is the standard
 *     half-split rotary embedding) is
 *     s = X W^T + b split into nq query, nkv key and nkv value heads of d columns;
 *     query and key heads are rotated pairwise, (s_i, s_{i+d/2}) ->
 *     (s_i c - s_{i+d/2} v, s_{i+d/2} c + s_i v) with c = cos[pos][i],
 *     v = sin[pos][i] from the caller's tables; queries go to q_out[t], keys and
 *     values to row cache_rows[t] of the key / value caches.
 *
 * Threads (pthreads) split independent rows / tokens; each row is computed by
 * one thread in a fixed order, so results do not depend on the thread count.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <unistd.h>

/* dtype codes of this oracle's own interface */
enum { ORC_F32 = 0, ORC_BF16 = 1, ORC_F16 = 2 };

/* tail-op codes of this oracle's own interface */
enum {
  ORC_BIAS = 0,          /* s_j += p0[j]                                  */
  ORC_SCALE = 1,         /* s_j *= scalar                                 */
  ORC_RELU = 2,          /* max(0, s)                                     */
  ORC_GELU_TANH = 3,     /* 0.5 s (1 + tanh(sqrt(2/pi) (s + 0.044715 s^3))) */
  ORC_SILU = 4,          /* s * sigmoid(s)  (Swish)                       */
  ORC_SIGMOID = 5,       /* 1 / (1 + exp(-s))                             */
  ORC_RESIDUAL_ADD = 6,  /* s_ij += p0[i*ld + j]                          */
  ORC_ROW_LOGSUMEXP = 7, /* row -> max_j s_j + log sum_j exp(s_j - max)   */
  ORC_GROUPNORM = 8,     /* per row, per contiguous column group          */
  ORC_SWIGLU = 9,        /* row of 2N -> silu(s[0:N]) * s[N:2N]           */
  ORC_ROW_SCALE_SCATTER_ADD = 10, /* out[p1[i]] += p0[i] * row          */
  ORC_MISH = 11,         /* s * tanh(log(1 + exp(s)))                     */
  ORC_LEAKY_RELU = 12,   /* s > 0 ? s : scalar * s                        */
  ORC_MUL = 13,          /* s_j *= p0[j]                                  */
  ORC_ROW_SCALE = 14,    /* s_ij *= p0[i]                                 */
  ORC_ROW_SUM = 15,      /* row -> sum_j s_j                              */
};

typedef struct {
  int32_t kind;
  int32_t groups;
  double scalar;
  double eps;
  const void *p0;
  const void *p1;
  int32_t p_dtype; /* dtype of p0 (and p1 where it is a vector) */
  int32_t pad_;
  int64_t ld;      /* leading dimension of a matrix operand (residual)   */
} orc_op;

/* Bytes of one stored element: fp32 is 4, the two 16-bit formats 2. */
static size_t orc_elt_size(int dt) { return dt == ORC_F32 ? 4 : 2; }

/* Widen one stored element to double.  bf16 is the top half of an IEEE
 * binary32 with the low 16 mantissa bits zero, so the widening is exact. */
static double orc_load(const void *p, int dt, int64_t i) {
  if (dt == ORC_F16) {
    /* IEEE binary16: 1 sign bit, 5 exponent bits (bias 15), 10 fraction bits;
     * exponent 0 holds the subnormals m 2^-24, exponent 31 inf / nan */
    const uint16_t b = ((const uint16_t *)p)[i];
    const int sign = b >> 15, ex = (b >> 10) & 31, fr = b & 1023;
    double v;
    if (ex == 0)
      v = ldexp((double)fr, -24);
    else if (ex == 31)
      v = fr ? NAN : INFINITY;
    else
      v = ldexp((double)(1024 + fr), ex - 25);
    return sign ? -v : v;
  }
  if (dt == ORC_BF16) {
    uint32_t bits = (uint32_t)((const uint16_t *)p)[i] << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
  }
  return (double)((const float *)p)[i];
}

/* Round a double to the nearest bfloat16 value (ties to even), returned as a
 * double.  bf16 keeps 8 significant bits: for |x| in [2^(e-1), 2^e) the spacing
 * is 2^(e-8); below the smallest normal 2^-126 the spacing is fixed at 2^-133. */
double orc_round_bf16(double x) {
  if (x == 0.0 || !isfinite(x)) return x;
  int e;
  frexp(x, &e); /* |x| = m 2^e, 0.5 <= m < 1 */
  if (e < -125) e = -125;
  double q = ldexp(1.0, e - 8);
  double r = nearbyint(x / q) * q; /* default rounding mode: nearest, ties even */
  if (fabs(r) > 3.3895313892515355e38) r = copysign(INFINITY, x);
  return r;
}

static double orc_sigmoid(double v) { return 1.0 / (1.0 + exp(-v)); }

static double orc_gelu_tanh(double v) {
  const double c = sqrt(2.0 / M_PI);
  return 0.5 * v * (1.0 + tanh(c * (v + 0.044715 * v * v * v)));
}

static double orc_softplus(double v) { return v > 30.0 ? v + log1p(exp(-v)) : log1p(exp(v)); }

/* Apply one elementwise op to a value at (row i, column j). */
static double orc_pointwise(const orc_op *op, double v, int64_t i, int64_t j) {
  switch (op->kind) {
    case ORC_BIAS: return v + orc_load(op->p0, op->p_dtype, j);
    case ORC_SCALE: return v * op->scalar;
    case ORC_RELU: return v > 0.0 ? v : 0.0;
    case ORC_GELU_TANH: return orc_gelu_tanh(v);
    case ORC_SILU: return v * orc_sigmoid(v);
    case ORC_SIGMOID: return orc_sigmoid(v);
    case ORC_RESIDUAL_ADD: return v + orc_load(op->p0, op->p_dtype, i * op->ld + j);
    case ORC_MISH: return v * tanh(orc_softplus(v));
    case ORC_LEAKY_RELU: return v > 0.0 ? v : op->scalar * v;
    case ORC_MUL: return v * orc_load(op->p0, op->p_dtype, j);
    case ORC_ROW_SCALE: return v * orc_load(op->p0, op->p_dtype, i);
    default: return NAN;
  }
}

static int orc_is_pointwise(int kind) {
  return kind == ORC_BIAS || kind == ORC_SCALE || kind == ORC_RELU || kind == ORC_GELU_TANH ||
         kind == ORC_SILU || kind == ORC_SIGMOID || kind == ORC_RESIDUAL_ADD || kind == ORC_MISH ||
         kind == ORC_LEAKY_RELU || kind == ORC_MUL || kind == ORC_ROW_SCALE;
}

/* GroupNorm of one row (PyTorch convention: biased variance, contiguous groups
 * of n/groups columns, per-column affine gamma = p0, beta = p1). */
static void orc_groupnorm_row(const orc_op *op, double *s, int64_t n) {
  int64_t gs = n / op->groups;
  for (int64_t g = 0; g < op->groups; ++g) {
    double *z = s + g * gs;
    double mean = 0.0;
    for (int64_t j = 0; j < gs; ++j) mean += z[j];
    mean /= (double)gs;
    double var = 0.0;
    for (int64_t j = 0; j < gs; ++j) var += (z[j] - mean) * (z[j] - mean);
    var /= (double)gs;
    double inv = 1.0 / sqrt(var + op->eps);
    for (int64_t j = 0; j < gs; ++j) {
      int64_t col = g * gs + j;
      double gam = op->p0 ? orc_load(op->p0, op->p_dtype, col) : 1.0;
      double bet = op->p1 ? orc_load(op->p1, op->p_dtype, col) : 0.0;
      z[j] = (z[j] - mean) * inv * gam + bet;
    }
  }
}

/* Row log-sum-exp, two-pass: m = max_j s_j, then m + log sum_j exp(s_j - m). */
static double orc_row_lse(const double *s, int64_t n) {
  double m = -INFINITY;
  for (int64_t j = 0; j < n; ++j) m = s[j] > m ? s[j] : m;
  if (m == -INFINITY) return -INFINITY;
  double acc = 0.0;
  for (int64_t j = 0; j < n; ++j) acc += exp(s[j] - m);
  return m + log(acc);
}

/* Row sum: the plain left-to-right sum of the row's n values. */
static double orc_row_sum(const double *s, int64_t n) {
  double acc = 0.0;
  for (int64_t j = 0; j < n; ++j) acc += s[j];
  return acc;
}

/* Apply the chain ops[first..n_ops) to the row vector s (length n) of row i.
 * Returns the number of live columns after the chain (1 after a row
 * log-sum-exp or a row sum, n/2 after SwiGLU).  A scatter op is not applied here. */
static int64_t orc_apply_chain(const orc_op *ops, int n_ops, double *s, int64_t n, int64_t i) {
  for (int o = 0; o < n_ops; ++o) {
    const orc_op *op = &ops[o];
    if (orc_is_pointwise(op->kind)) {
      for (int64_t j = 0; j < n; ++j) s[j] = orc_pointwise(op, s[j], i, j);
    } else if (op->kind == ORC_ROW_LOGSUMEXP) {
      s[0] = orc_row_lse(s, n);
      n = 1;
      /* ops after the reduction act on the scalar (column index 0) */
    } else if (op->kind == ORC_ROW_SUM) {
      s[0] = orc_row_sum(s, n);
      n = 1;
    } else if (op->kind == ORC_GROUPNORM) {
      orc_groupnorm_row(op, s, n);
    } else if (op->kind == ORC_SWIGLU) {
      int64_t h = n / 2;
      for (int64_t j = 0; j < h; ++j) {
        double g = s[j], u = s[h + j];
        s[j] = g * orc_sigmoid(g) * u;
      }
      n = h;
    } else if (op->kind == ORC_ROW_SCALE_SCATTER_ADD) {
      /* handled by the caller */
    } else {
      for (int64_t j = 0; j < n; ++j) s[j] = NAN;
    }
  }
  return n;
}

/* ------------------------------------------------------------------------- */
/* Dense fused GEMM: Y = chain(X W^T).  X [M x K] (ld ldx), W [N x K] (ld ldw). */
/* Output: double Y[M x ldy]; after a row log-sum-exp Y has one value per row   */
/* or a row sum (stored at Y[i*ldy]).                                          */
/* ------------------------------------------------------------------------- */
typedef struct {
  const void *X; int xt; int64_t ldx;
  const void *W; int wt; int64_t ldw;
  int64_t M, N, K;
  const orc_op *ops; int n_ops;
  double *Y; int64_t ldy;
  const int64_t *rows; /* optional subset of row indices (output row r <- X row rows[r]) */
  int64_t n_rows;
  int64_t next;        /* work counter */
  pthread_mutex_t mu;
} orc_dense_job;

static void *orc_dense_worker(void *arg) {
  orc_dense_job *jb = (orc_dense_job *)arg;
  double *xr = (double *)malloc(sizeof(double) * (size_t)(jb->K > 0 ? jb->K : 1));
  double *s = (double *)malloc(sizeof(double) * (size_t)(jb->N > 0 ? jb->N : 1));
  for (;;) {
    pthread_mutex_lock(&jb->mu);
    int64_t r = jb->next++;
    pthread_mutex_unlock(&jb->mu);
    if (r >= jb->n_rows) break;
    int64_t i = jb->rows ? jb->rows[r] : r;
    for (int64_t k = 0; k < jb->K; ++k) xr[k] = orc_load(jb->X, jb->xt, i * jb->ldx + k);
    for (int64_t j = 0; j < jb->N; ++j) {
      double acc = 0.0;
      for (int64_t k = 0; k < jb->K; ++k) acc += xr[k] * orc_load(jb->W, jb->wt, j * jb->ldw + k);
      s[j] = acc;
    }
    int64_t n = orc_apply_chain(jb->ops, jb->n_ops, s, jb->N, i);
    for (int64_t j = 0; j < n; ++j) jb->Y[r * jb->ldy + j] = s[j];
  }
  free(xr);
  free(s);
  return NULL;
}

static int orc_threads(int nthreads) {
  if (nthreads > 0) return nthreads;
  long c = sysconf(_SC_NPROCESSORS_ONLN);
  return c > 0 ? (int)c : 1;
}

static void orc_run(void *(*fn)(void *), void *job, int nthreads) {
  int nt = orc_threads(nthreads);
  if (nt == 1) { fn(job); return; }
  pthread_t *th = (pthread_t *)malloc(sizeof(pthread_t) * (size_t)nt);
  for (int t = 0; t < nt; ++t) pthread_create(&th[t], NULL, fn, job);
  for (int t = 0; t < nt; ++t) pthread_join(th[t], NULL);
  free(th);
}

int orc_fused_gemm(const void *X, int xt, int64_t ldx, const void *W, int wt, int64_t ldw,
                   int64_t M, int64_t N, int64_t K, const orc_op *ops, int n_ops,
                   const int64_t *rows, int64_t n_rows, double *Y, int64_t ldy, int nthreads) {
  orc_dense_job jb;
  memset(&jb, 0, sizeof jb);
  jb.X = X; jb.xt = xt; jb.ldx = ldx; jb.W = W; jb.wt = wt; jb.ldw = ldw;
  jb.M = M; jb.N = N; jb.K = K; jb.ops = ops; jb.n_ops = n_ops; jb.Y = Y; jb.ldy = ldy;
  jb.rows = rows; jb.n_rows = rows ? n_rows : M; jb.next = 0;
  pthread_mutex_init(&jb.mu, NULL);
  orc_run(orc_dense_worker, &jb, nthreads);
  pthread_mutex_destroy(&jb.mu);
  return 0;
}

/* ------------------------------------------------------------------------- */
/* MoE routing (gpt-oss decode path, Sec. IV-A): for each token, the k experts  */
/* with the largest logits (ties -> lower expert index), weights = softmax over */
/* the k selected logits (they sum to 1), then a stable counting sort of the    */
/* T*k (token, slot) pairs by expert: pairs of one expert keep increasing pair  */
/* index p = t*k + slot.                                                        */
/* ------------------------------------------------------------------------- */
int orc_moe_route(const float *logits, int64_t T, int32_t E, int32_t k, int32_t *topk_ids,
                  double *topk_w, int32_t *offsets, int32_t *sorted_token, double *sorted_w,
                  int32_t *sorted_pair) {
  if (k < 1 || k > E) return 1;
  char *taken = (char *)malloc((size_t)E);
  for (int64_t t = 0; t < T; ++t) {
    memset(taken, 0, (size_t)E);
    const float *l = logits + t * E;
    for (int32_t j = 0; j < k; ++j) {
      int32_t best = -1;
      for (int32_t e = 0; e < E; ++e) {
        if (taken[e]) continue;
        if (best < 0 || l[e] > l[best]) best = e; /* strict '>' keeps the lower index on ties */
      }
      taken[best] = 1;
      topk_ids[t * k + j] = best;
    }
    double mx = (double)l[topk_ids[t * k]];
    double den = 0.0;
    for (int32_t j = 0; j < k; ++j) den += exp((double)l[topk_ids[t * k + j]] - mx);
    for (int32_t j = 0; j < k; ++j) topk_w[t * k + j] = exp((double)l[topk_ids[t * k + j]] - mx) / den;
  }
  free(taken);
  int64_t P = T * k;
  int64_t *cnt = (int64_t *)calloc((size_t)E + 1, sizeof(int64_t));
  for (int64_t p = 0; p < P; ++p) cnt[topk_ids[p]]++;
  offsets[0] = 0;
  for (int32_t e = 0; e < E; ++e) offsets[e + 1] = offsets[e] + (int32_t)cnt[e];
  int64_t *fill = (int64_t *)calloc((size_t)E, sizeof(int64_t));
  for (int64_t p = 0; p < P; ++p) {
    int32_t e = topk_ids[p];
    int64_t pos = offsets[e] + fill[e]++;
    sorted_token[pos] = (int32_t)(p / k);
    sorted_w[pos] = topk_w[p];
    if (sorted_pair) sorted_pair[pos] = (int32_t)p;
  }
  free(cnt);
  free(fill);
  return 0;
}

/* ------------------------------------------------------------------------- */
/* MoE expert FFN, written per token (the plain definition):                   */
/*   g = W_gu[e, 0:I, :] x_t + bg[e],  u = W_gu[e, I:2I, :] x_t + bu[e],        */
/*   h = bf16(act(g, u))         (or unrounded when round_h == 0),              */
/*   Y_t = sum_j w_tj * (W_down[e_tj] h + bd[e_tj]).                            */
/* act(g, u) = g' * sigmoid(alpha g') * (u' + c) with g' = min(g, L) and       */
/* u' = clamp(u, -L, L) when L > 0 (else g' = g, u' = u): the plain SwiGLU is   */
/* alpha = 1, L = 0, c = 0 and no biases; the gpt-oss expert activation adds    */
/* the clamp, a sigmoid slope, the +1 on the linear branch and per-expert       */
/* biases (b_gu [E x 2I]: gate then up; b_down [E x H]; bf16, or NULL).        */
/* X [T x H] bf16, W_gu [E x 2I x H] bf16, W_down [E x H x I] bf16.            */
/* Only tokens listed in `tokens` (n_tok of them) are computed; output row r    */
/* of Y (double, [n_tok x H]) belongs to token tokens[r].                      */
/* ------------------------------------------------------------------------- */
typedef struct {
  const uint16_t *X, *Wgu, *Wd, *bgu, *bd;
  double alpha, limit, c;
  const int32_t *ids;
  const double *w;
  int64_t H, I;
  int32_t k;
  const int64_t *tokens;
  int64_t n_tok;
  int round_h;
  double *Y;
  int64_t next;
  pthread_mutex_t mu;
} orc_moe_job;

static void *orc_moe_worker(void *arg) {
  orc_moe_job *jb = (orc_moe_job *)arg;
  int64_t H = jb->H, I = jb->I;
  double *x = (double *)malloc(sizeof(double) * (size_t)H);
  double *h = (double *)malloc(sizeof(double) * (size_t)I);
  for (;;) {
    pthread_mutex_lock(&jb->mu);
    int64_t r = jb->next++;
    pthread_mutex_unlock(&jb->mu);
    if (r >= jb->n_tok) break;
    int64_t t = jb->tokens[r];
    for (int64_t c = 0; c < H; ++c) x[c] = orc_load(jb->X, ORC_BF16, t * H + c);
    double *y = jb->Y + r * H;
    for (int64_t c = 0; c < H; ++c) y[c] = 0.0;
    for (int32_t j = 0; j < jb->k; ++j) {
      int64_t e = jb->ids[t * jb->k + j];
      double wt = jb->w[t * jb->k + j];
      const uint16_t *wg = jb->Wgu + e * 2 * I * H;
      for (int64_t n = 0; n < I; ++n) {
        double g = 0.0, u = 0.0;
        for (int64_t c = 0; c < H; ++c) {
          g += x[c] * orc_load(wg, ORC_BF16, n * H + c);
          u += x[c] * orc_load(wg, ORC_BF16, (I + n) * H + c);
        }
        if (jb->bgu) {
          g += orc_load(jb->bgu, ORC_BF16, e * 2 * I + n);
          u += orc_load(jb->bgu, ORC_BF16, e * 2 * I + I + n);
        }
        if (jb->limit > 0.0) {
          g = fmin(g, jb->limit);
          u = fmax(fmin(u, jb->limit), -jb->limit);
        }
        double hv = g * orc_sigmoid(jb->alpha * g) * (u + jb->c);
        h[n] = jb->round_h ? orc_round_bf16(hv) : hv;
      }
      const uint16_t *wd = jb->Wd + e * H * I;
      for (int64_t c = 0; c < H; ++c) {
        double acc = 0.0;
        for (int64_t n = 0; n < I; ++n) acc += h[n] * orc_load(wd, ORC_BF16, c * I + n);
        if (jb->bd) acc += orc_load(jb->bd, ORC_BF16, e * H + c);
        y[c] += wt * acc;
      }
    }
  }
  free(x);
  free(h);
  return NULL;
}

int orc_moe_ffn(const uint16_t *X, const uint16_t *W_gu, const uint16_t *W_down,
                const int32_t *topk_ids, const double *topk_w, int64_t H, int64_t I, int32_t k,
                const int64_t *tokens, int64_t n_tok, int round_h, double *Y, int nthreads,
                const uint16_t *b_gu, const uint16_t *b_down, double alpha, double limit, double c) {
  orc_moe_job jb;
  memset(&jb, 0, sizeof jb);
  jb.X = X; jb.Wgu = W_gu; jb.Wd = W_down; jb.ids = topk_ids; jb.w = topk_w;
  jb.bgu = b_gu; jb.bd = b_down; jb.alpha = alpha; jb.limit = limit; jb.c = c;
  jb.H = H; jb.I = I; jb.k = k; jb.tokens = tokens; jb.n_tok = n_tok; jb.round_h = round_h;
  jb.Y = Y; jb.next = 0;
  pthread_mutex_init(&jb.mu, NULL);
  orc_run(orc_moe_worker, &jb, nthreads);
  pthread_mutex_destroy(&jb.mu);
  return 0;
}

/* ------------------------------------------------------------------------- */
/* Grouped GEMM over row groups: for group g, rows r in [off[g], off[g+1]):     */
/*   a_r = A[row_index ? row_index[r] : r],  s = a_r B[g]^T (B[g] = B + g*bgs), */
/*   v = chain(s);  then either out[r] = v, or (scatter op present)             */
/*   out[p1[r]] += p0[r] * v.                                                   */
/* A [* x K] (ld lda), B rows of length K (ld ldb).  out is double with ld ldo. */
/* Single-threaded over rows when scattering (fixed summation order).           */
/* ------------------------------------------------------------------------- */
/* Residual add + RMSNorm per row (see the header): R, gamma read at their stored
 * dtype, Y in double; R_out (double, holding bf16 values) and normed (double). */
int orc_add_rmsnorm(const double *Y, const void *R, int rt, const void *gamma, int gt, double eps, int64_t T,
                    int64_t H, double *R_out, double *normed) {
  if (T < 0 || H < 1 || !(eps >= 0.0)) return 1;
  for (int64_t t = 0; t < T; ++t) {
    double ss = 0.0;
    for (int64_t j = 0; j < H; ++j) {
      const double h = orc_round_bf16(orc_load(R, rt, t * H + j) + Y[t * H + j]);
      R_out[t * H + j] = h;
      ss += h * h;
    }
    const double inv = 1.0 / sqrt(ss / (double)H + eps);
    for (int64_t j = 0; j < H; ++j) normed[t * H + j] = R_out[t * H + j] * inv * orc_load(gamma, gt, j);
  }
  return 0;
}

/* Bias + RoPE + KV-cache update of the QKV projection (see the header).  X
 * [T x H], W [(nq + 2 nkv) d x H], bias [(nq + 2 nkv) d] or NULL,
 * positions / cache_rows int32 [T], cos / sin fp32 [max_pos x d/2]; q_out
 * double [T x nq d]; k_cache / v_cache double [rows x nkv d] (only the rows
 * named by cache_rows are written).  xt: element type of X and W, bt: of the
 * bias (ORC_BF16 / ORC_F16 / ORC_F32 codes). */
int orc_qkv_rope_kv(const void *X, const void *W, int xt, const void *bias, int bt, const int32_t *positions,
                    const int32_t *cache_rows, const float *cos_t, const float *sin_t, int64_t max_pos, int64_t T,
                    int64_t H, int32_t nq, int32_t nkv, int32_t d, int64_t rows, double *q_out, double *k_cache,
                    double *v_cache) {
  if (T < 0 || H < 1 || nq < 1 || nkv < 1 || d < 2 || d % 2) return 1;
  const int64_t N = (int64_t)(nq + 2 * nkv) * d, half = d / 2;
  double *s = (double *)malloc(sizeof(double) * (size_t)N);
  if (!s) return 2;
  for (int64_t t = 0; t < T; ++t) {
    const int32_t pos = positions[t], row = cache_rows[t];
    if (pos < 0 || pos >= max_pos || row < 0 || row >= rows) { free(s); return 3; }
    for (int64_t n = 0; n < N; ++n) {
      double acc = bias ? orc_load(bias, bt, n) : 0.0;
      for (int64_t k = 0; k < H; ++k) acc += orc_load(X, xt, t * H + k) * orc_load(W, xt, n * H + k);
      s[n] = acc;
    }
    for (int32_t hd = 0; hd < nq + 2 * nkv; ++hd) {
      double *h = s + (int64_t)hd * d;
      if (hd < nq + nkv) /* query and key heads: rotate the pairs */
        for (int64_t i = 0; i < half; ++i) {
          const double c = (double)cos_t[pos * half + i], v = (double)sin_t[pos * half + i];
          const double a = h[i], b = h[i + half];
          h[i] = a * c - b * v;
          h[i + half] = b * c + a * v;
        }
      double *dst = hd < nq ? q_out + t * (int64_t)nq * d + (int64_t)hd * d
                  : hd < nq + nkv ? k_cache + (int64_t)row * nkv * d + (int64_t)(hd - nq) * d
                                  : v_cache + (int64_t)row * nkv * d + (int64_t)(hd - nq - nkv) * d;
      for (int32_t i = 0; i < d; ++i) dst[i] = h[i];
    }
  }
  free(s);
  return 0;
}

int orc_grouped_gemm(const void *A, int at, int64_t lda, const int32_t *row_index, const void *B,
                     int bt, int64_t ldb, int64_t b_group_stride, const int32_t *offsets, int32_t G,
                     int64_t N, int64_t K, const orc_op *ops, int n_ops, double *out, int64_t ldo) {
  int scatter = -1;
  int64_t nb = N; /* rows of B per group used by the GEMM */
  for (int o = 0; o < n_ops; ++o) {
    if (ops[o].kind == ORC_ROW_SCALE_SCATTER_ADD) scatter = o;
    if (ops[o].kind == ORC_SWIGLU) nb = 2 * N;
  }
  double *a = (double *)malloc(sizeof(double) * (size_t)(K > 0 ? K : 1));
  double *s = (double *)malloc(sizeof(double) * (size_t)(nb > 0 ? nb : 1));
  for (int32_t g = 0; g < G; ++g) {
    const char *Bg = (const char *)B + (size_t)g * (size_t)b_group_stride * orc_elt_size(bt);
    for (int64_t r = offsets[g]; r < offsets[g + 1]; ++r) {
      int64_t src = row_index ? row_index[r] : r;
      for (int64_t k = 0; k < K; ++k) a[k] = orc_load(A, at, src * lda + k);
      for (int64_t j = 0; j < nb; ++j) {
        double acc = 0.0;
        for (int64_t k = 0; k < K; ++k) acc += a[k] * orc_load(Bg, bt, j * ldb + k);
        s[j] = acc;
      }
      int64_t n = orc_apply_chain(ops, n_ops, s, nb, r);
      if (scatter >= 0) {
        const orc_op *sc = &ops[scatter];
        double w = orc_load(sc->p0, sc->p_dtype, r);
        int64_t dst = ((const int32_t *)sc->p1)[r];
        for (int64_t j = 0; j < n; ++j) out[dst * ldo + j] += w * s[j];
      } else {
        for (int64_t j = 0; j < n; ++j) out[r * ldo + j] = s[j];
      }
    }
  }
  free(a);
  free(s);
  return 0;
}
