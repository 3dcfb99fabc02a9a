/*
 * Direct Quantized Training (DQT) -- CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, obviously-correct
 * statement of what the DQT BitLinear training step computes.  Only the test
 * suite, the smoke check and the CPU-baseline leg of the benchmark may load
 * it.  The CUDA library never includes, links or calls it, and it includes
 * nothing from the CUDA library.
 *
 * Paper: "Direct Quantized Training of Language Models with Stochastic
 * Rounding" (Zhao et al., ACML 2025, arXiv 2412.04787).
 *
 *   Eq. 1   stochastic rounding SR(x)                     -> dqt_oracle_sr
 *   Eq. 2-4 AbsMean grid, scale and initial codes         -> dqt_oracle_absmean_init
 *   Sec 3.2 8-bit activation quantisation (BitNet style)  -> dqt_oracle_act_quant
 *   Sec 3.2 BitLinear forward on the quantised operands   -> dqt_oracle_fwd
 *   Sec 3.2 backward w.r.t. the low-bit weight (no STE)   -> dqt_oracle_bwd_dx / _bwd_dw
 *   Sec 4.1/4.3 the same with X_tilde held in bf16        -> dqt_oracle_bwd_dw_bf16x
 *   Sec 4.1 AdamW producing the dense target W'           -> dqt_oracle_adamw_x
 *           (its textbook evaluation order, for the pins)   -> dqt_oracle_adamw_x_textbook
 *   Eq. 5   W_hat = SR(W'), kept on the n-bit grid        -> dqt_oracle_update
 *           on one data-parallel shard of the weight        -> dqt_oracle_update_shard
 *   Sec 5.1 absmax / round-to-nearest ablation            -> round_mode = 1
 *   Sec 4.1/4.3 FP8 environment: E4M3 activations and      -> dqt_oracle_act_quant_fp8
 *               the forward on E4M3 operands                -> dqt_oracle_fwd_fp8
 *   Sec 1       2-bit packed ternary storage                -> dqt_oracle_pack_ternary
 *   Sec 4.3     Adafactor (factored second moment) + SR     -> dqt_oracle_adafactor_*
 *               (the printed rank-one form, for the pins)   -> dqt_oracle_adafactor_u_textbook
 *
 * Readings where the paper is silent, taken here:
 *   - ternary ("1.58 bit") means the grid [-1, 1] with s = 1 / AbsMean;
 *     integer n uses Q_n = -2^(n-1), Q_p = 2^(n-1) - 1 literally;
 *   - the scale s is fixed at initialisation and SR acts on the code domain
 *     x = W' * s, followed by a clamp to [Q_n, Q_p];
 *   - Round() is round-half-to-even;
 *   - activations: per-token absmax, s_x = 127 / max(amax, 1e-5),
 *     q = clamp(rint(x * s_x), -128, 127);
 *   - the RNG is Philox4x32-10 (Salmon et al., SC'11) keyed by the seed, with
 *     the counter (element/4, step, tensor id) and word element%4; a uniform
 *     U = (word >> 8) * 2^-24 rounds up when U < x - floor(x);
 *   - FP8 environment: the 8-bit activation is E4M3 with the per-token scale
 *     448 / max(amax, 1e-5), rounded to nearest-even with saturation; the
 *     forward accumulates exactly and rounds Y as the integer path does.
 *
 * Arithmetic: the reductions of the GEMMs are exact (int64) or fp64; the
 * AdamW + SR step is a fixed sequence of individually rounded IEEE fp32
 * operations (build with -ffp-contract=off so that no FMA is formed).
 *
 * Parity of every function here is pinned by tests/test_oracle_*.py against
 * facts fixed by the paper and by mathematics (hand-worked examples, closed
 * forms, exact enumeration, published Philox known-answer vectors).
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* bf16 <-> fp32 (IEEE round-to-nearest-even on the dropped 16 bits).        */
/* ------------------------------------------------------------------------ */
static float bf16_to_f32(uint16_t h) {
  uint32_t u = (uint32_t)h << 16;
  float f;
  memcpy(&f, &u, 4);
  return f;
}

static uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  if ((u & 0x7f800000u) == 0x7f800000u && (u & 0x007fffffu) != 0)
    return (uint16_t)((u >> 16) | 0x0040u); /* quiet NaN */
  uint32_t lsb = (u >> 16) & 1u;
  u += 0x7fffu + lsb;
  return (uint16_t)(u >> 16);
}

uint16_t dqt_oracle_f32_to_bf16(float f) { return f32_to_bf16_rne(f); }

/* ------------------------------------------------------------------------ */
/* Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as   */
/* easy as 1, 2, 3", SC'11).  One round: two 32x32->64 multiplications of    */
/* counter words 0 and 2 by the Philox multipliers, then a permutation that  */
/* xors the high halves with the other counter words and the round key.      */
/* The key is bumped by the Weyl constants between rounds.                   */
/* ------------------------------------------------------------------------ */
#define PHILOX_M0 0xD2511F53u
#define PHILOX_M1 0xCD9E8D57u
#define PHILOX_W0 0x9E3779B9u
#define PHILOX_W1 0xBB67AE85u

void dqt_oracle_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2],
                              uint32_t out[4]) {
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += PHILOX_W0;
      k1 += PHILOX_W1;
    }
    uint64_t p0 = (uint64_t)PHILOX_M0 * (uint64_t)c0;
    uint64_t p1 = (uint64_t)PHILOX_M1 * (uint64_t)c2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t n0 = hi1 ^ c1 ^ k0;
    uint32_t n1 = lo1;
    uint32_t n2 = hi0 ^ c3 ^ k1;
    uint32_t n3 = lo0;
    c0 = n0; c1 = n1; c2 = n2; c3 = n3;
  }
  out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* The uniform variate that drives the rounding of element e (flat row-major
 * index into the weight tensor) at a given (seed, step, tensor id).  Returns
 * the raw 32-bit word; the uniform is (word >> 8) * 2^-24. */
uint32_t dqt_oracle_sr_word(uint64_t seed, int64_t step, uint32_t tensor_id,
                            int64_t e) {
  uint64_t blk = (uint64_t)e >> 2;
  uint32_t ctr[4] = {(uint32_t)blk, (uint32_t)(blk >> 32), (uint32_t)step,
                     tensor_id};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  uint32_t out[4];
  dqt_oracle_philox4x32_10(ctr, key, out);
  return out[e & 3];
}

float dqt_oracle_uniform_from_word(uint32_t w) {
  return (float)(w >> 8) * (1.0f / 16777216.0f);
}

/* ------------------------------------------------------------------------ */
/* Eq. 1: SR(x) = floor(x) with probability ceil(x) - x, otherwise ceil(x).  */
/* With r = x - floor(x) the value rounds up exactly when the uniform u < r, */
/* which happens with probability r = 1 - (ceil(x) - x).  An integer x has   */
/* r = 0 and never moves.                                                    */
/* ------------------------------------------------------------------------ */
int32_t dqt_oracle_sr(float x, float u) {
  float f = floorf(x);
  float r = x - f;
  return (int32_t)f + (u < r ? 1 : 0);
}

void dqt_oracle_sr_batch(const float* x, const float* u, int32_t* out,
                         int64_t n) {
  for (int64_t i = 0; i < n; ++i) out[i] = dqt_oracle_sr(x[i], u[i]);
}

static int32_t clamp_i32(int32_t v, int32_t lo, int32_t hi) {
  return v < lo ? lo : (v > hi ? hi : v);
}

/* ------------------------------------------------------------------------ */
/* Eq. 3 grid.  bits_x100 = 158 selects ternary; otherwise n = bits_x100/100 */
/* with 2 <= n <= 8 gives Q_n = -2^(n-1), Q_p = 2^(n-1) - 1.                 */
/* ------------------------------------------------------------------------ */
int dqt_oracle_grid(int32_t bits_x100, int32_t* qmin, int32_t* qmax) {
  if (bits_x100 == 158) {
    *qmin = -1;
    *qmax = 1;
    return 0;
  }
  if (bits_x100 % 100 != 0) return 1;
  int32_t n = bits_x100 / 100;
  if (n < 2 || n > 8) return 1;
  *qmin = -(1 << (n - 1));
  *qmax = (1 << (n - 1)) - 1;
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Eq. 4 alone: codes = Clip[Round(W * s), Q_n, Q_p] for a given fp32 scale  */
/* s: one fp32 multiplication, Round() half-to-even, then the clip.          */
/* ------------------------------------------------------------------------ */
void dqt_oracle_quantize_weights(const float* W, int64_t numel, float s, int32_t qmin,
                                 int32_t qmax, int8_t* codes) {
  for (int64_t i = 0; i < numel; ++i) {
    float p = W[i] * s;
    float r = rintf(p);
    int32_t c;
    if (r >= (float)qmax) c = qmax;
    else if (r <= (float)qmin) c = qmin;
    else c = (int32_t)r;
    codes[i] = (int8_t)c;
  }
}

/* ------------------------------------------------------------------------ */
/* Eq. 2-4: AbsMean(W) = (1/k) sum |w_i|;  s = Q_p / AbsMean(W);             */
/* codes = Clip[Round(W * s), Q_n, Q_p].  The sum runs in fp64 in index      */
/* order; s is rounded once to fp32; W * s is one fp32 multiplication and    */
/* Round() is round-half-to-even.                                            */
/* ------------------------------------------------------------------------ */
int dqt_oracle_absmean_init(const float* W0, int64_t numel, int32_t qmin,
                            int32_t qmax, int8_t* codes, float* s_w,
                            double* absmean_out) {
  if (numel <= 0) return 1;
  double acc = 0.0;
  for (int64_t i = 0; i < numel; ++i) acc += fabs((double)W0[i]);
  double absmean = acc / (double)numel;
  if (absmean_out) *absmean_out = absmean;
  if (!(absmean > 0.0)) return 2;
  float s = (float)((double)qmax / absmean);
  *s_w = s;
  dqt_oracle_quantize_weights(W0, numel, s, qmin, qmax, codes);
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Sec 3.2: 8-bit activation quantisation following BitNet: per token t,     */
/* amax = max_k |x|, s_x = 127 / max(amax, 1e-5), q = Clip[Round(x s_x),     */
/* -128, 127].  Also returns the two bf16 operand images the GPU path feeds  */
/* its tensor cores: the codes themselves (exact in bf16) and the            */
/* dequantised activation bf16(q / s_x).  Either image pointer may be NULL.  */
/* ------------------------------------------------------------------------ */
void dqt_oracle_act_quant(const uint16_t* X, int64_t T, int64_t K, int8_t* q,
                          float* s_x, uint16_t* q_img, uint16_t* xdq) {
  for (int64_t t = 0; t < T; ++t) {
    const uint16_t* row = X + t * K;
    float amax = 0.0f;
    for (int64_t k = 0; k < K; ++k) {
      float a = fabsf(bf16_to_f32(row[k]));
      if (a > amax) amax = a;
    }
    float denom = amax > 1e-5f ? amax : 1e-5f;
    float s = 127.0f / denom;
    s_x[t] = s;
    for (int64_t k = 0; k < K; ++k) {
      float p = bf16_to_f32(row[k]) * s;
      float r = rintf(p);
      int32_t v;
      if (r >= 127.0f) v = 127;
      else if (r <= -128.0f) v = -128;
      else v = (int32_t)r;
      q[t * K + k] = (int8_t)v;
      if (q_img) q_img[t * K + k] = f32_to_bf16_rne((float)v);
      if (xdq) xdq[t * K + k] = f32_to_bf16_rne((float)v / s);
    }
  }
}

/* ------------------------------------------------------------------------ */
/* Sec 3.2 forward: Y = X_tilde W_tilde^T on the quantised operands.         */
/* acc[t,n] = sum_k q[t,k] c[n,k]  (exact, int64; must fit int32)            */
/* Y[t,n]   = bf16( float(acc) * (1 / (s_x[t] * s_w)) )                      */
/* Returns 1 if an accumulator does not fit int32.                           */
/* ------------------------------------------------------------------------ */
int dqt_oracle_fwd(const int8_t* q, const float* s_x, const int8_t* c,
                   float s_w, int64_t T, int64_t K, int64_t N, uint16_t* Y,
                   int32_t* acc_out) {
  int overflow = 0;
  for (int64_t t = 0; t < T; ++t) {
    float a_t = 1.0f / (s_x[t] * s_w);
    for (int64_t n = 0; n < N; ++n) {
      int64_t acc = 0;
      for (int64_t k = 0; k < K; ++k)
        acc += (int64_t)q[t * K + k] * (int64_t)c[n * K + k];
      if (acc > INT32_MAX || acc < INT32_MIN) overflow = 1;
      if (acc_out) acc_out[t * N + n] = (int32_t)acc;
      if (Y) Y[t * N + n] = f32_to_bf16_rne((float)acc * a_t);
    }
  }
  return overflow;
}

/* ------------------------------------------------------------------------ */
/* Backward w.r.t. the input (no STE on the weight, straight-through on the  */
/* activation quantiser): dX[t,k] = sum_n dY[t,n] W_tilde[n,k]               */
/*                                = (sum_n dY[t,n] c[n,k]) / s_w,  fp64.     */
/* ------------------------------------------------------------------------ */
void dqt_oracle_bwd_dx(const uint16_t* dY, const int8_t* c, float s_w,
                       int64_t T, int64_t N, int64_t K, double* dX) {
  for (int64_t t = 0; t < T; ++t)
    for (int64_t k = 0; k < K; ++k) {
      double acc = 0.0;
      for (int64_t n = 0; n < N; ++n)
        acc += (double)bf16_to_f32(dY[t * N + n]) * (double)c[n * K + k];
      dX[t * K + k] = acc / (double)s_w;
    }
}

/* ------------------------------------------------------------------------ */
/* Backward w.r.t. the low-bit weight W_tilde = c / s_w (Sec 3.2):           */
/* dW[n,k] = sum_t dY[t,n] X_tilde[t,k],  X_tilde = q / s_x,  fp64.          */
/* rows (length Nr) selects which output rows n to compute; dW is [Nr, K].   */
/* ------------------------------------------------------------------------ */
void dqt_oracle_bwd_dw(const uint16_t* dY, const int8_t* q, const float* s_x,
                       int64_t T, int64_t N, int64_t K, const int64_t* rows,
                       int64_t Nr, double* dW) {
  for (int64_t i = 0; i < Nr; ++i) {
    int64_t n = rows[i];
    for (int64_t k = 0; k < K; ++k) dW[i * K + k] = 0.0;
    for (int64_t t = 0; t < T; ++t) {
      double g = (double)bf16_to_f32(dY[t * N + n]);
      double inv = 1.0 / (double)s_x[t];
      for (int64_t k = 0; k < K; ++k)
        dW[i * K + k] += g * ((double)q[t * K + k] * inv);
    }
  }
}

/* ------------------------------------------------------------------------ */
/* The same weight gradient with X_tilde held in bf16 (the BF16 training     */
/* environment of Sec 4.1/4.3): dW[n,k] = sum_t dY[t,n] bf16(q/s_x)[t,k],    */
/* fp64.  xdq is the bf16 image that dqt_oracle_act_quant returns.           */
/* ------------------------------------------------------------------------ */
void dqt_oracle_bwd_dw_bf16x(const uint16_t* dY, const uint16_t* xdq, int64_t T,
                             int64_t N, int64_t K, const int64_t* rows, int64_t Nr,
                             double* dW) {
  for (int64_t i = 0; i < Nr; ++i) {
    int64_t n = rows[i];
    for (int64_t k = 0; k < K; ++k) dW[i * K + k] = 0.0;
    for (int64_t t = 0; t < T; ++t) {
      double g = (double)bf16_to_f32(dY[t * N + n]);
      for (int64_t k = 0; k < K; ++k)
        dW[i * K + k] += g * (double)bf16_to_f32(xdq[t * K + k]);
    }
  }
}

/* ------------------------------------------------------------------------ */
/* AdamW (Loshchilov & Hutter; the optimiser of Sec 4.1) in the code domain. */
/* AdamW moves W by -lr * m_hat / (sqrt(v_hat) + eps) - lr * wd * W with     */
/* m_hat = m'/bc1, v_hat = v'/bc2.  Multiplying through by bc1 gives the same */
/* step with a single division:                                              */
/*   m_hat / (sqrt(v_hat) + eps) = m' / (sqrt(v') * k1 + k2),                 */
/*   k1 = bc1 / sqrt(bc2),  k2 = bc1 * eps.                                  */
/* Host-side constants, from the hyper-parameters in fp64, each rounded once */
/* to fp32:  omb1 = 1 - b1, omb2 = 1 - b2, bc = 1 - b^step,                  */
/*   k1, k2 as above, decay = 1 - lr * wd, lrs = lr * s_w.                   */
/* Per element, each a separately rounded fp32 operation:                    */
/*   m' = b1 m + omb1 g ;  v' = b2 v + omb2 (g g)                            */
/*   u  = m' / (sqrt(v') k1 + k2)                                            */
/*   x  = c decay - lrs u          (= W' s_w, the dense target in codes)     */
/* ------------------------------------------------------------------------ */
typedef struct {
  float b1, b2, omb1, omb2, k1, k2, decay, lrs, pad;
} oracle_adamw_consts;

void dqt_oracle_adamw_consts(float lr, float b1, float b2, float eps, float wd,
                             int64_t step, float s_w, float* out9) {
  double bc1 = 1.0 - pow((double)b1, (double)step);
  double bc2 = 1.0 - pow((double)b2, (double)step);
  out9[0] = b1;
  out9[1] = b2;
  out9[2] = (float)(1.0 - (double)b1);
  out9[3] = (float)(1.0 - (double)b2);
  out9[4] = (float)(bc1 / sqrt(bc2));
  out9[5] = (float)(bc1 * (double)eps);
  out9[6] = (float)(1.0 - (double)lr * (double)wd);
  out9[7] = (float)((double)lr * (double)s_w);
  out9[8] = 0.0f;
}

static float adamw_x(const oracle_adamw_consts* h, float g, int8_t c, float* m,
                     float* v) {
  float m1 = h->b1 * *m;
  float m2 = h->omb1 * g;
  float mn = m1 + m2;
  float v1 = h->b2 * *v;
  float gg = g * g;
  float v2 = h->omb2 * gg;
  float vn = v1 + v2;
  *m = mn;
  *v = vn;
  float sv = sqrtf(vn);
  float den = sv * h->k1 + h->k2;
  float u = mn / den;
  float cd = (float)c * h->decay;
  float du = h->lrs * u;
  return cd - du;
}

/* Dense target only (no rounding): x, m', v' for n elements. */
void dqt_oracle_adamw_x(const float* g, const int8_t* c, float* m, float* v,
                        const float* consts9, int64_t n, float* x) {
  oracle_adamw_consts h;
  memcpy(&h, consts9, sizeof(h));
  for (int64_t i = 0; i < n; ++i) x[i] = adamw_x(&h, g[i], c[i], &m[i], &v[i]);
}

/* ------------------------------------------------------------------------ */
/* The same AdamW step in the textbook order of Loshchilov & Hutter's         */
/* algorithm, each a separately rounded fp32 operation:                      */
/*   m' = b1 m + omb1 g ;  v' = b2 v + omb2 (g g)                            */
/*   m_hat = m' / bc1 ;  v_hat = v' / bc2                                    */
/*   u = m_hat / (sqrt(v_hat) + eps)                                         */
/*   x = c decay - lrs u                                                     */
/* Host constants, fp64 rounded once to fp32: b1, b2, omb1 = 1 - b1,          */
/* omb2 = 1 - b2, bc1 = 1 - b1^step, bc2 = 1 - b2^step, eps,                  */
/* decay = 1 - lr wd, lrs = lr s_w.  The restated one-division form above is  */
/* the same quantity multiplied through by bc1; the two are compared          */
/* elementwise by the pins.                                                  */
/* ------------------------------------------------------------------------ */
typedef struct {
  float b1, b2, omb1, omb2, bc1, bc2, eps, decay, lrs;
} oracle_adamw_textbook_consts;

void dqt_oracle_adamw_textbook_consts(float lr, float b1, float b2, float eps, float wd,
                                      int64_t step, float s_w, float* out9) {
  out9[0] = b1;
  out9[1] = b2;
  out9[2] = (float)(1.0 - (double)b1);
  out9[3] = (float)(1.0 - (double)b2);
  out9[4] = (float)(1.0 - pow((double)b1, (double)step));
  out9[5] = (float)(1.0 - pow((double)b2, (double)step));
  out9[6] = eps;
  out9[7] = (float)(1.0 - (double)lr * (double)wd);
  out9[8] = (float)((double)lr * (double)s_w);
}

static float adamw_x_textbook(const oracle_adamw_textbook_consts* h, float g, int8_t c,
                              float* m, float* v) {
  float m1 = h->b1 * *m;
  float m2 = h->omb1 * g;
  float mn = m1 + m2;
  float v1 = h->b2 * *v;
  float gg = g * g;
  float v2 = h->omb2 * gg;
  float vn = v1 + v2;
  *m = mn;
  *v = vn;
  float mh = mn / h->bc1;
  float vh = vn / h->bc2;
  float sv = sqrtf(vh);
  float den = sv + h->eps;
  float u = mh / den;
  float cd = (float)c * h->decay;
  float du = h->lrs * u;
  return cd - du;
}

void dqt_oracle_adamw_x_textbook(const float* g, const int8_t* c, float* m, float* v,
                                 const float* tconsts9, int64_t n, float* x) {
  oracle_adamw_textbook_consts h;
  memcpy(&h, tconsts9, sizeof(h));
  for (int64_t i = 0; i < n; ++i) x[i] = adamw_x_textbook(&h, g[i], c[i], &m[i], &v[i]);
}

/* ------------------------------------------------------------------------ */
/* Eq. 5: W_hat = SR(W'), clamped to [Q_n, Q_p], written over the codes.     */
/* g, c, m, v are [Nr, K] row blocks of an [N, K] weight; rows[i] is the      */
/* global row of block row i, so element (rows[i], k) draws the uniform of   */
/* flat index rows[i]*K + k.  rows == NULL means rows[i] = i.                */
/* round_mode 0 = stochastic (Eq. 1); 1 = round-to-nearest (Sec 5.1          */
/* ablation).  Returns the number of codes that changed.                     */
/* ------------------------------------------------------------------------ */
static int64_t update_impl(int textbook, const float* g, int8_t* c, float* m, float* v,
                           const float* consts9, int32_t qmin, int32_t qmax,
                           uint64_t seed, int64_t step, uint32_t tensor_id,
                           int32_t round_mode, const int64_t* rows, int64_t Nr,
                           int64_t K, int64_t elem0) {
  oracle_adamw_consts h;
  oracle_adamw_textbook_consts ht;
  memcpy(&h, consts9, sizeof(h));
  memcpy(&ht, consts9, sizeof(ht));
  int64_t changed = 0;
  for (int64_t i = 0; i < Nr; ++i) {
    int64_t n = rows ? rows[i] : i;
    for (int64_t k = 0; k < K; ++k) {
      int64_t j = i * K + k;
      float x = textbook ? adamw_x_textbook(&ht, g[j], c[j], &m[j], &v[j])
                         : adamw_x(&h, g[j], c[j], &m[j], &v[j]);
      int32_t r;
      if (round_mode == 1) {
        r = (int32_t)rintf(x);
      } else {
        uint32_t w = dqt_oracle_sr_word(seed, step, tensor_id, elem0 + n * K + k);
        r = dqt_oracle_sr(x, dqt_oracle_uniform_from_word(w));
      }
      r = clamp_i32(r, qmin, qmax);
      if ((int8_t)r != c[j]) ++changed;
      c[j] = (int8_t)r;
    }
  }
  return changed;
}

int64_t dqt_oracle_update(const float* g, int8_t* c, float* m, float* v,
                          const float* consts9, int32_t qmin, int32_t qmax,
                          uint64_t seed, int64_t step, uint32_t tensor_id,
                          int32_t round_mode, const int64_t* rows, int64_t Nr,
                          int64_t K) {
  return update_impl(0, g, c, m, v, consts9, qmin, qmax, seed, step, tensor_id, round_mode,
                     rows, Nr, K, 0);
}

/* Eq. 5 on a flat shard of a weight tensor: element i of the n given is    */
/* global element elem0 + i and draws that element's uniform, so updating  */
/* the shards of a partition one by one gives the codes of the whole-tensor */
/* update (the data-parallel form: each rank updates its shard).           */
int64_t dqt_oracle_update_shard(const float* g, int8_t* c, float* m, float* v,
                                const float* consts9, int32_t qmin, int32_t qmax,
                                uint64_t seed, int64_t step, uint32_t tensor_id,
                                int32_t round_mode, int64_t elem0, int64_t n) {
  return update_impl(0, g, c, m, v, consts9, qmin, qmax, seed, step, tensor_id, round_mode,
                     NULL, 1, n, elem0);
}

/* Eq. 5 with the textbook-order AdamW (tconsts9 from                        */
/* dqt_oracle_adamw_textbook_consts); otherwise identical to the above.      */
int64_t dqt_oracle_update_textbook(const float* g, int8_t* c, float* m, float* v,
                                   const float* tconsts9, int32_t qmin, int32_t qmax,
                                   uint64_t seed, int64_t step, uint32_t tensor_id,
                                   int32_t round_mode, const int64_t* rows, int64_t Nr,
                                   int64_t K) {
  return update_impl(1, g, c, m, v, tconsts9, qmin, qmax, seed, step, tensor_id, round_mode,
                     rows, Nr, K, 0);
}

/* ======================================================================== */
/* FP8 environment (Sec. 4.1 hardware paragraph, Sec. 4.3): the BitLinear    */
/* forward with 8-bit floating-point operands.  The 8-bit activation is an   */
/* E4M3 value with a per-token absmax scale instead of an int8 code; the     */
/* weight codes (integers of magnitude at most 16) are exact E4M3 values.    */
/* ======================================================================== */

/* E4M3 ("e4m3fn" of the OCP 8-bit floating point format): sign bit, four   */
/* exponent bits with bias 7, three mantissa bits.  Exponent field 0 holds   */
/* the subnormals m * 2^-9; every other field is (1 + m/8) * 2^(e-7); the    */
/* single magnitude pattern 1111.111 is NaN and there are no infinities, so  */
/* the largest finite magnitude is 1.75 * 2^8 = 448.                          */
double dqt_oracle_e4m3_value(uint8_t b) {
  int e = (b >> 3) & 0xF;
  int m = b & 0x7;
  double mag;
  if (e == 0xF && m == 0x7) return NAN;
  if (e == 0) mag = ldexp((double)m, -9);
  else mag = ldexp(1.0 + (double)m / 8.0, e - 7);
  return (b & 0x80) ? -mag : mag;
}

/* Round-to-nearest-even onto the finite E4M3 values with saturation: the    */
/* finite magnitude nearest to |p| (all 127 are tried), a tie going to the   */
/* even code (the code's last bit is the mantissa's), anything beyond 448    */
/* giving 448.  The sign is p's own, so values that round to zero keep it.   */
uint8_t dqt_oracle_e4m3_from_f32(float p) {
  if (isnan(p)) return 0x7F;
  double a = fabs((double)p);
  if (a > 448.0) return (uint8_t)(0x7E | (signbit(p) ? 0x80 : 0));
  int best = 0;
  double bd = a;
  for (int b = 1; b < 0x7F; ++b) {
    double d = fabs(a - dqt_oracle_e4m3_value((uint8_t)b));
    if (d < bd || (d == bd && (b & 1) == 0 && (best & 1) == 1)) {
      bd = d;
      best = b;
    }
  }
  return (uint8_t)(best | (signbit(p) ? 0x80 : 0));
}

void dqt_oracle_codes_to_e4m3(const int8_t* c, int64_t numel, uint8_t* out) {
  for (int64_t i = 0; i < numel; ++i) out[i] = dqt_oracle_e4m3_from_f32((float)c[i]);
}

/* 8-bit activations as E4M3: per token t, amax = max_k |x|,                 */
/* s8 = 448 / max(amax, 1e-5) (fp32 division), q8 = E4M3(x * s8) with the    */
/* product one fp32 multiplication.  xdq (optional) is the dequantised       */
/* activation bf16(value(q8) / s8) that the weight gradient reads.           */
void dqt_oracle_act_quant_fp8(const uint16_t* X, int64_t T, int64_t K, uint8_t* q8,
                              float* s8, uint16_t* xdq) {
  for (int64_t t = 0; t < T; ++t) {
    const uint16_t* row = X + t * K;
    float amax = 0.0f;
    for (int64_t k = 0; k < K; ++k) {
      float a = fabsf(bf16_to_f32(row[k]));
      if (a > amax) amax = a;
    }
    float s = 448.0f / (amax > 1e-5f ? amax : 1e-5f);
    s8[t] = s;
    for (int64_t k = 0; k < K; ++k) {
      float p = bf16_to_f32(row[k]) * s;
      uint8_t b = dqt_oracle_e4m3_from_f32(p);
      q8[t * K + k] = b;
      if (xdq) xdq[t * K + k] = f32_to_bf16_rne((float)dqt_oracle_e4m3_value(b) / s);
    }
  }
}

/* FP8 forward: acc[t,n] = sum_k value(q8[t,k]) * c[n,k], exact in fp64      */
/* (every term is a multiple of 2^-9 below 2^13), and                        */
/* Y[t,n] = bf16( float(acc) * (1 / (s8[t] * s_w)) ).                        */
/* Returns 1 if a code is outside [-16, 16] (not exact in E4M3).            */
int dqt_oracle_fwd_fp8(const uint8_t* q8, const float* s8, const int8_t* c, float s_w,
                       int64_t T, int64_t K, int64_t N, uint16_t* Y, double* acc_out) {
  /* acc = sum_k value(q8) * c for any int8 code: codes beyond 16 in magnitude
   * reach the E4M3 tensor cores as two exact terms, 16 (c >> 4) and c & 15,
   * whose products add up to the same sum */
  for (int64_t t = 0; t < T; ++t) {
    float a_t = 1.0f / (s8[t] * s_w);
    for (int64_t n = 0; n < N; ++n) {
      double acc = 0.0;
      for (int64_t k = 0; k < K; ++k)
        acc += dqt_oracle_e4m3_value(q8[t * K + k]) * (double)c[n * K + k];
      if (acc_out) acc_out[t * N + n] = acc;
      if (Y) Y[t * N + n] = f32_to_bf16_rne((float)acc * a_t);
    }
  }
  return 0;
}

/* ======================================================================== */
/* 2-bit packed ternary codes (the ternary storage of Sec. 1: about 0.2 GB    */
/* for a 1B-parameter model).  Code e of a flat tensor lives in byte e / 4,  */
/* bits 2 (e % 4) .. 2 (e % 4) + 1, as a 2-bit two's-complement number       */
/* (-1 = 0b11, 0 = 0b00, +1 = 0b01).  Unused bits of the last byte are 0.    */
/* ======================================================================== */
void dqt_oracle_pack_ternary(const int8_t* c, int64_t n, uint8_t* out) {
  for (int64_t i = 0; i < (n + 3) / 4; ++i) out[i] = 0;
  for (int64_t e = 0; e < n; ++e)
    out[e / 4] |= (uint8_t)(((unsigned)c[e] & 3u) << (2 * (e % 4)));
}

void dqt_oracle_unpack_ternary(const uint8_t* p, int64_t n, int8_t* c) {
  for (int64_t e = 0; e < n; ++e) {
    int v = (p[e / 4] >> (2 * (e % 4))) & 3;
    c[e] = (int8_t)(v >= 2 ? v - 4 : v);
  }
}

/* ======================================================================== */
/* Adafactor with stochastic rounding (Sec. 4.3: DQT trained with the memory- */
/* efficient Adafactor optimiser).  Adafactor is Shazeer & Stern, "Adafactor:  */
/* Adaptive Learning Rates with Sublinear Memory Cost" (ICML 2018): the second */
/* moment of an N x K gradient is kept as its row means R [N] and column      */
/* means C [K] (factored), updates are clipped to RMS d, and the step size    */
/* may be relative to the parameter's RMS.  Here without first moment (beta1 */
/* = 0), the configuration that stores no per-weight state at all.           */
/*                                                                          */
/* Per step t (host constants, fp64 -> fp32 once):                          */
/*   b2 = 1 - t^decay_rate,  omb2 = t^decay_rate                             */
/*   rho = relative_step ? min(warmup_init ? 1e-6 t : 1e-2, 1/sqrt(t)) : lr  */
/* Statistics (fp64 sums, state rounded to fp32):                            */
/*   R[n] <- b2 R[n] + omb2 mean_k(g^2 + eps1)                                */
/*   C[k] <- b2 C[k] + omb2 mean_n(g^2 + eps1)                                */
/*   Rbar = mean_n R[n]   (rounded once to fp32)                             */
/* The estimate V[n,k] = R[n] C[k] / Rbar is rank one, so its inverse square */
/* root is a row factor times a column factor, each an fp32 value made by    */
/* two correctly rounded operations:                                         */
/*   a[n] = 1 / sqrt(R[n] / Rbar),   b[k] = 1 / sqrt(C[k])                   */
/*   u[n,k] = (g a[n]) b[k]           (two fp32 multiplications)             */
/*   rms_u = sqrt(mean u^2) (fp64 over the fp32 u);  rms_x = sqrt(mean (c/s_w)^2) */
/*   alpha = rho * (scale_parameter ? max(eps2, rms_x) : 1)                  */
/*   step  = s_w alpha / max(1, rms_u / d)        (code-domain step, fp32)   */
/*   decay = 1 - weight_decay alpha                (fp32)                     */
/* Per element (dqt_oracle_adafactor_apply), separately rounded fp32 ops:    */
/*   u = (g a[n]) b[k];  x = c decay - step u;  c' = Clip[SR(x), Q_n, Q_p]    */
/* with the same Philox stream as AdamW.                                      */
/* ======================================================================== */
void dqt_oracle_adafactor_consts(int64_t t, float lr, float decay_rate, int32_t relative_step,
                                 int32_t warmup_init, float* b2, float* omb2, float* rho) {
  double p = pow((double)t, (double)decay_rate);
  *b2 = (float)(1.0 - p);
  *omb2 = (float)p;
  if (relative_step) {
    double cap = warmup_init ? 1e-6 * (double)t : 1e-2;
    double inv = 1.0 / sqrt((double)t);
    *rho = (float)(cap < inv ? cap : inv);
  } else {
    *rho = lr;
  }
}

static float adafactor_u(float g, float an, float bk) {
  float ga = g * an;
  return ga * bk;
}

/* Shazeer & Stern's update in its printed form: the rank-one estimate      */
/* V[n,k] = R[n] C[k] / Rbar, then u = g / sqrt(V), each a separately        */
/* rounded fp32 operation.  The factored form above computes the same        */
/* quantity; the pins compare the two elementwise.  (The printed form         */
/* underflows fp32 once R[n] C[k] drops below the smallest normal float; the  */
/* factored form does not.)                                                  */
void dqt_oracle_adafactor_u_textbook(const float* g, const float* R, const float* C, float rbar,
                                     int64_t N, int64_t K, float* u) {
  for (int64_t n = 0; n < N; ++n)
    for (int64_t k = 0; k < K; ++k) {
      float rc = R[n] * C[k];
      float vv = rc / rbar;
      float sq = sqrtf(vv);
      u[n * K + k] = g[n * K + k] / sq;
    }
}

/* The factored form's u for every element (a, b from the statistics).       */
void dqt_oracle_adafactor_u(const float* g, const float* a, const float* b, int64_t N, int64_t K,
                            float* u) {
  for (int64_t n = 0; n < N; ++n)
    for (int64_t k = 0; k < K; ++k) u[n * K + k] = adafactor_u(g[n * K + k], a[n], b[k]);
}

/* R, C updated in place; a [N], b [K] the inverse-square-root factors.     */
/* out4 = {Rbar (fp32 value), rms_u, rms_x, alpha}; step and decay above.   */
void dqt_oracle_adafactor_stats(const float* g, const int8_t* c, int64_t N, int64_t K,
                                float s_w, float* R, float* C, float b2, float omb2,
                                float rho, float eps1, float eps2, float clip_d,
                                int32_t scale_parameter, float weight_decay, float* a,
                                float* b, double* out4, float* step_out, float* decay_out) {
  for (int64_t n = 0; n < N; ++n) {
    double acc = 0.0;
    for (int64_t k = 0; k < K; ++k) {
      double gv = (double)g[n * K + k];
      acc += gv * gv + (double)eps1;
    }
    R[n] = (float)((double)b2 * (double)R[n] + (double)omb2 * (acc / (double)K));
  }
  for (int64_t k = 0; k < K; ++k) {
    double acc = 0.0;
    for (int64_t n = 0; n < N; ++n) {
      double gv = (double)g[n * K + k];
      acc += gv * gv + (double)eps1;
    }
    C[k] = (float)((double)b2 * (double)C[k] + (double)omb2 * (acc / (double)N));
  }
  double rsum = 0.0;
  for (int64_t n = 0; n < N; ++n) rsum += (double)R[n];
  float rbar = (float)(rsum / (double)N);
  for (int64_t n = 0; n < N; ++n) a[n] = 1.0f / sqrtf(R[n] / rbar);
  for (int64_t k = 0; k < K; ++k) b[k] = 1.0f / sqrtf(C[k]);
  double usq = 0.0, xsq = 0.0;
  for (int64_t n = 0; n < N; ++n)
    for (int64_t k = 0; k < K; ++k) {
      double u = (double)adafactor_u(g[n * K + k], a[n], b[k]);
      usq += u * u;
      double w = (double)c[n * K + k] / (double)s_w;
      xsq += w * w;
    }
  double rms_u = sqrt(usq / ((double)N * (double)K));
  double rms_x = sqrt(xsq / ((double)N * (double)K));
  double alpha = (double)rho * (scale_parameter ? (rms_x > (double)eps2 ? rms_x : (double)eps2) : 1.0);
  double div = rms_u / (double)clip_d;
  if (div < 1.0) div = 1.0;
  out4[0] = (double)rbar;
  out4[1] = rms_u;
  out4[2] = rms_x;
  out4[3] = alpha;
  *step_out = (float)((double)s_w * alpha / div);
  *decay_out = (float)(1.0 - (double)weight_decay * alpha);
}

static float adafactor_x(float g, int8_t c, float an, float bk, float step, float decay) {
  float u = adafactor_u(g, an, bk);
  float cd = (float)c * decay;
  float du = step * u;
  return cd - du;
}

/* Dense code-domain target only (no rounding), N x K. */
void dqt_oracle_adafactor_x(const float* g, const int8_t* c, const float* a, const float* b,
                            float step, float decay, int64_t N, int64_t K, float* x) {
  for (int64_t n = 0; n < N; ++n)
    for (int64_t k = 0; k < K; ++k)
      x[n * K + k] = adafactor_x(g[n * K + k], c[n * K + k], a[n], b[k], step, decay);
}

/* Per-element Adafactor + SR over an N x K weight, given the factors a, b,  */
/* the code-domain step and decay.  Returns the number of codes changed.     */
int64_t dqt_oracle_adafactor_apply(const float* g, int8_t* c, const float* a, const float* b,
                                   float step, float decay, int64_t N, int64_t K, int32_t qmin,
                                   int32_t qmax, uint64_t seed, int64_t t, uint32_t tensor_id,
                                   int32_t round_mode) {
  int64_t changed = 0;
  for (int64_t n = 0; n < N; ++n)
    for (int64_t k = 0; k < K; ++k) {
      int64_t e = n * K + k;
      float x = adafactor_x(g[e], c[e], a[n], b[k], step, decay);
      int32_t r;
      if (round_mode == 1) {
        r = (int32_t)rintf(x);
      } else {
        uint32_t w = dqt_oracle_sr_word(seed, t, tensor_id, e);
        r = dqt_oracle_sr(x, dqt_oracle_uniform_from_word(w));
      }
      r = clamp_i32(r, qmin, qmax);
      if ((int8_t)r != c[e]) ++changed;
      c[e] = (int8_t)r;
    }
  return changed;
}
