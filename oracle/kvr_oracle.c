/*
 * kvr_oracle.c -- plain, slow, fp64 CPU oracle for the KV-reuse attention path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product library links, includes or
 * calls this file; only the test suite, the smoke check and the CPU-baseline leg
 * of the benchmark load it (through oracle/__init__.py).  It shares no header,
 * helper, table or constant generator with the CUDA path.
 *
 * What it computes (paper: "Can I Buy Your KV Cache?", arXiv 2606.13361):
 *   - Sec. 3 "Setup and notation": a decoder layer keeps per-position keys and
 *     values; the entry of position i depends only on x_{1:i} (causal).
 *   - Sec. 3.2 / Algorithm 2: continuation tokens take positions L, L+1, ...
 *     (so RoPE matches a from-scratch pass) and attend over the full span of
 *     L+|q| cached positions.
 *   - Sec. 3.3, Claim 1: reuse rows equal the matching rows of a prefill over
 *     prefix||suffix.  Here every row is computed from its own visible keys in
 *     one fixed order, so the identity holds bit for bit in fp64.
 *   The paper is silent on the layer internals; the readings taken (Qwen3-style
 *   per-head RMSNorm on q and k, rotate-half RoPE with theta = 1e6, GQA head
 *   h -> kv head floor(h / G), softmax scale 1/sqrt(d), bf16 rounding of the
 *   cached k and of the roped q) are listed with the design notes.
 *
 * Every routine is the plain definition written out in fp64, no blocking, no
 * online softmax, no fusion.  bf16 values are decoded exactly to fp64.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ---- bf16 encode/decode (IEEE-754 binary32 truncated to its top 16 bits) ---- */

static double bf16_decode(uint16_t h) {
  uint32_t u = (uint32_t)h << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

/* Round an fp64 value to the nearest bf16 value, ties to even, straight from
 * fp64 (8 significant bits; exponent range of binary32; subnormal quantum
 * 2^-133; overflow to infinity past the largest finite bf16). */
static uint16_t bf16_encode_rne(double x) {
  if (isnan(x)) return (uint16_t)0x7fc0;
  uint16_t sign = signbit(x) ? (uint16_t)0x8000 : (uint16_t)0;
  double a = fabs(x);
  if (a == 0.0) return sign;
  if (isinf(a)) return (uint16_t)(sign | 0x7f80);
  int ex;
  (void)frexp(a, &ex);                 /* a = m * 2^ex, m in [0.5, 1) */
  int qexp = ex - 8;                   /* quantum for 8 significant bits */
  if (qexp < -133) qexp = -133;        /* subnormal range */
  double r = ldexp(nearbyint(ldexp(a, -qexp)), qexp); /* default mode: ties-to-even */
  const double max_bf16 = 3.3895313892515355e38;     /* (2 - 2^-7) * 2^127 */
  if (r > max_bf16) return (uint16_t)(sign | 0x7f80);
  float f = (float)r;                  /* exact: r has <= 8 significant bits */
  uint32_t u;
  memcpy(&u, &f, sizeof u);
  return (uint16_t)(sign | (uint16_t)((u >> 16) & 0x7fff));
}

void kvro_bf16_encode(const double* x, int64_t n, uint16_t* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = bf16_encode_rne(x[i]);
}

void kvro_bf16_decode(const uint16_t* h, int64_t n, double* out) {
  for (int64_t i = 0; i < n; ++i) out[i] = bf16_decode(h[i]);
}

/* ---- RMSNorm over one head vector (Qwen3 QK-norm reading) ----
 * y_i = x_i / sqrt(mean_j x_j^2 + eps) * w_i */
static void rmsnorm(const double* x, const double* w, int d, double eps, double* y) {
  double ss = 0.0;
  for (int i = 0; i < d; ++i) ss += x[i] * x[i];
  double inv = 1.0 / sqrt(ss / (double)d + eps);
  for (int i = 0; i < d; ++i) y[i] = x[i] * inv * w[i];
}

void kvro_rmsnorm(int64_t n_vec, int d, const double* x, const double* w, double eps, double* y) {
  for (int64_t v = 0; v < n_vec; ++v) rmsnorm(x + v * d, w, d, eps, y + v * d);
}

/* ---- RoPE, rotate-half pairing (i, i + d/2), angle pos * theta^(-2i/d) ----
 * Sec. 3.2: position ids of continuation tokens are L, L+1, ... */
static void rope(double* x, int d, int64_t pos, double theta) {
  int h = d / 2;
  for (int i = 0; i < h; ++i) {
    double ang = (double)pos * pow(theta, -2.0 * (double)i / (double)d);
    double c = cos(ang), s = sin(ang);
    double a = x[i], b = x[i + h];
    x[i] = a * c - b * s;
    x[i + h] = b * c + a * s;
  }
}

void kvro_rope(int64_t n_vec, int d, const int64_t* pos, double theta, double* x) {
  for (int64_t v = 0; v < n_vec; ++v) rope(x + v * d, d, pos[v], theta);
}

/* ---- Per-token preparation of new tokens (the append step) ----
 * For token t at position pos[t]:
 *   q'_{t,h} = RoPE(RMSNorm(q_{t,h}; wq), pos[t])        h < Hq
 *   k'_{t,g} = RoPE(RMSNorm(k_{t,g}; wk), pos[t])        g < Hkv
 * Outputs are fp64 (unrounded) and bf16 (rounded once, ties to even): the
 * cache holds bf16 by definition and attention consumes the rounded q. */
void kvro_qk_prep(int64_t T, int Hq, int Hkv, int d, const int64_t* pos,
                  const double* q_pre, const double* k_pre, const double* wq,
                  const double* wk, double theta, double eps,
                  double* q_f64, double* k_f64, uint16_t* q_bf16, uint16_t* k_bf16) {
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < T; ++t) {
    for (int h = 0; h < Hq; ++h) {
      const double* x = q_pre + (t * Hq + h) * d;
      double* y = q_f64 + (t * Hq + h) * d;
      rmsnorm(x, wq, d, eps, y);
      rope(y, d, pos[t], theta);
      for (int i = 0; i < d; ++i) q_bf16[(t * Hq + h) * d + i] = bf16_encode_rne(y[i]);
    }
    for (int g = 0; g < Hkv; ++g) {
      const double* x = k_pre + (t * Hkv + g) * d;
      double* y = k_f64 + (t * Hkv + g) * d;
      rmsnorm(x, wk, d, eps, y);
      rope(y, d, pos[t], theta);
      for (int i = 0; i < d; ++i) k_bf16[(t * Hkv + g) * d + i] = bf16_encode_rne(y[i]);
    }
  }
}

/* ---- Causal GQA softmax attention, plain definition ----
 * Rows r = 0..n_rows-1 (query heads h = 0..Hq-1); keys c = 0..n_keys-1 at
 * positions c.  Row r sees key c iff c <= row_pos[r] (causal mask; Sec. 3,
 * Alg. 2's full mask over the cached span).  Query head h reads kv head
 * floor(h / G), G = Hq / Hkv.
 *   s_c = <q_{r,h}, k_{c,g}> / sqrt(d)
 *   O_{r,h} = sum_c softmax(s)_c v_{c,g},   lse_{r,h} = log sum_c exp(s_c)
 * Masked keys are left out of the sums (not given a large negative score).
 * A row with no visible key gets O = 0 and lse = -inf.
 * q: [n_rows][Hq][d], k, v: [n_keys][Hkv][d], o: [n_rows][Hq][d], lse: [n_rows][Hq]. */
void kvro_attention(int64_t n_rows, int Hq, int Hkv, int d, const double* q,
                    const int64_t* row_pos, int64_t n_keys, const double* k,
                    const double* v, double* o, double* lse) {
  const int G = Hq / Hkv;
  const double scale = 1.0 / sqrt((double)d);
#pragma omp parallel
  {
    double* s = (double*)malloc(sizeof(double) * (size_t)(n_keys > 0 ? n_keys : 1));
#pragma omp for schedule(dynamic, 1)
    for (int64_t rh = 0; rh < n_rows * Hq; ++rh) {
      int64_t r = rh / Hq;
      int h = (int)(rh % Hq);
      int g = h / G;
      const double* qr = q + (r * Hq + h) * d;
      double* orow = o + (r * Hq + h) * d;
      int64_t nvis = row_pos[r] + 1;
      if (nvis > n_keys) nvis = n_keys;
      if (nvis < 0) nvis = 0;
      for (int i = 0; i < d; ++i) orow[i] = 0.0;
      if (nvis == 0) {
        lse[r * Hq + h] = -INFINITY;
        continue;
      }
      double mx = -INFINITY;
      for (int64_t c = 0; c < nvis; ++c) {
        const double* kc = k + (c * Hkv + g) * d;
        double acc = 0.0;
        for (int i = 0; i < d; ++i) acc += qr[i] * kc[i];
        s[c] = acc * scale;
        if (s[c] > mx) mx = s[c];
      }
      double den = 0.0;
      for (int64_t c = 0; c < nvis; ++c) {
        s[c] = exp(s[c] - mx);
        den += s[c];
      }
      for (int64_t c = 0; c < nvis; ++c) {
        const double* vc = v + (c * Hkv + g) * d;
        double p = s[c] / den;
        for (int i = 0; i < d; ++i) orow[i] += p * vc[i];
      }
      lse[r * Hq + h] = mx + log(den);
    }
    free(s);
  }
}

int kvro_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
