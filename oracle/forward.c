/*
 * CPU ORACLE -- test infrastructure only.  Only tests/, the smoke entry
 * point and bench.py's CPU-baseline leg may load this file.  It shares no
 * code with the CUDA path.
 *
 * Plain fp32 forward pass of a Llama-style decoder (the LLaMA3 / Qwen
 * families the paper evaluates, Section 4.1), used by the PARD draft pass
 * (Eq. 6), the target verification pass (Section 2.2) and autoregressive
 * greedy decoding (Eq. 2).
 *
 * Weights are bf16 bit patterns, widened exactly to fp32 when read.  The
 * paper runs its models in bf16 (Table 3), so the KV cache stores bf16
 * values: with kv_bf16 set, each key and value is rounded to bf16
 * (round-to-nearest-even) when it enters the cache.  All arithmetic is fp32, compiled with -ffp-contract=off (no fused multiply-add),
 * so results are identical on every IEEE host.  Every dot product is summed
 * in the same order whatever the number of rows computed together, so a row
 * computed inside a batch is bitwise equal to the same row computed alone.
 *
 * Model (per layer, for every new row t at position pos_t):
 *   x   = h * (mean(h^2) + eps)^-1/2 * g_attn
 *   q,k,v = x Wq^T, x Wk^T, x Wv^T
 *   q,k rotated by RoPE (rotate-half pairs (j, j+hd/2), angle pos*theta^(-2j/hd))
 *   k,v stored in the cache at pos_t; query head h reads kv head h / (Hq/Hkv)
 *   o   = softmax(q k^T / sqrt(hd)) v over cached positions <= pos_t
 *   h  += o Wo^T
 *   x   = h * (mean(h^2) + eps)^-1/2 * g_mlp
 *   h  += (silu(x Wg^T) * (x Wu^T)) Wd^T,  silu(z) = z / (1 + e^-z)
 * then logits = rmsnorm(h) * g_final  Wlm^T.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
  int32_t n_layers, d, hq, hkv, hd, ffn, vocab;
  float theta, eps;
} ocfg;

/* per layer: attn_norm, wq, wk, wv, wo, mlp_norm, wg, wu, wd */
enum { T_ATTN_NORM, T_WQ, T_WK, T_WV, T_WO, T_MLP_NORM, T_WG, T_WU, T_WD, T_PER_LAYER };

typedef struct {
  const uint16_t* embed;
  const uint16_t* final_norm;
  const uint16_t* lm_head;
  const uint16_t* const* layers; /* n_layers * T_PER_LAYER pointers */
} oweights;

static inline float bf16_to_f32(uint16_t b) {
  union { uint32_t u; float f; } v;
  v.u = (uint32_t)b << 16;
  return v.f;
}

/* fp32 -> nearest bf16 (ties to even), returned widened to fp32 */
static inline float round_bf16(float f) {
  union { float f; uint32_t u; } v;
  v.f = f;
  if ((v.u & 0x7F800000u) == 0x7F800000u) return f;
  v.u += 0x7FFFu + ((v.u >> 16) & 1u);
  v.u &= 0xFFFF0000u;
  return v.f;
}

static void widen(const uint16_t* src, float* dst, int64_t n) {
  for (int64_t i = 0; i < n; ++i) dst[i] = bf16_to_f32(src[i]);
}

/* Dot product summed in eight interleaved partial sums (lane j takes the
 * terms k = j mod 8 in increasing k), then combined pairwise.  The order
 * depends only on n. */
static float dot(const float* x, const float* w, int64_t n) {
  float acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  int64_t k = 0;
  for (; k + 8 <= n; k += 8)
    for (int j = 0; j < 8; ++j) acc[j] += x[k + j] * w[k + j];
  for (; k < n; ++k) acc[k & 7] += x[k] * w[k];
  return ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
}

/* Y[i][n] = sum_k X[i][k] * W[n][k] for i < m, n < N.  W is bf16 [N][K]. */
void oracle_matmul(const float* X, int32_t m, int32_t K, const uint16_t* W, int32_t N, float* Y) {
  const int32_t MB = 32; /* rows per pass: keeps a block of X cache-resident */
  for (int32_t i0 = 0; i0 < m; i0 += MB) {
    int32_t i1 = i0 + MB < m ? i0 + MB : m;
#pragma omp parallel
    {
      float* wrow = (float*)malloc(sizeof(float) * (size_t)K);
#pragma omp for schedule(static)
      for (int32_t n = 0; n < N; ++n) {
        widen(W + (int64_t)n * K, wrow, K);
        for (int32_t i = i0; i < i1; ++i) Y[(int64_t)i * N + n] = dot(X + (int64_t)i * K, wrow, K);
      }
      free(wrow);
    }
  }
}

/* Selected outputs only: Y[i][j] = X[i] . W[cols[j]] (for sampled checks). */
void oracle_matmul_cols(const float* X, int32_t m, int32_t K, const uint16_t* W,
                        const int32_t* cols, int32_t ncols, float* Y) {
#pragma omp parallel
  {
    float* wrow = (float*)malloc(sizeof(float) * (size_t)K);
#pragma omp for schedule(static)
    for (int32_t j = 0; j < ncols; ++j) {
      widen(W + (int64_t)cols[j] * K, wrow, K);
      for (int32_t i = 0; i < m; ++i) Y[(int64_t)i * ncols + j] = dot(X + (int64_t)i * K, wrow, K);
    }
    free(wrow);
  }
}

/* RMSNorm of one row: out = x * (mean(x^2) + eps)^-1/2 * g */
void oracle_rmsnorm(const float* x, const uint16_t* g, int32_t d, float eps, float* out) {
  float ss = 0.0f;
  for (int32_t i = 0; i < d; ++i) ss += x[i] * x[i];
  float r = 1.0f / sqrtf(ss / (float)d + eps);
  for (int32_t i = 0; i < d; ++i) out[i] = (x[i] * r) * bf16_to_f32(g[i]);
}

/* RoPE, rotate-half convention, one head vector of length hd at position pos.
 * Angles and their cosines are computed in double and rounded to fp32. */
void oracle_rope(float* v, int32_t hd, int32_t pos, float theta) {
  int32_t half = hd / 2;
  for (int32_t j = 0; j < half; ++j) {
    double inv_freq = pow((double)theta, -2.0 * (double)j / (double)hd);
    double ang = (double)pos * inv_freq;
    float c = (float)cos(ang), s = (float)sin(ang);
    float a = v[j], b = v[j + half];
    v[j] = a * c - b * s;
    v[j + half] = a * s + b * c;
  }
}

/* One query vector against cached positions 0..pos (inclusive).
 * kc/vc point at this layer's cache [max_pos][hkv][hd] and kvh selects the
 * kv head.  scores = q.k / sqrt(hd); softmax; out = sum p v. */
void oracle_attend(const float* q, const float* kc, const float* vc, int32_t hkv, int32_t hd,
                   int32_t kvh, int32_t pos, float* scratch, float* out) {
  const float scale = (float)(1.0 / sqrt((double)hd));
  float mx = -INFINITY;
  for (int32_t j = 0; j <= pos; ++j) {
    scratch[j] = dot(q, kc + ((int64_t)j * hkv + kvh) * hd, hd) * scale;
    if (scratch[j] > mx) mx = scratch[j];
  }
  float sum = 0.0f;
  for (int32_t j = 0; j <= pos; ++j) {
    scratch[j] = expf(scratch[j] - mx);
    sum += scratch[j];
  }
  for (int32_t e = 0; e < hd; ++e) out[e] = 0.0f;
  for (int32_t j = 0; j <= pos; ++j) {
    const float p = scratch[j] / sum;
    const float* v = vc + ((int64_t)j * hkv + kvh) * hd;
    for (int32_t e = 0; e < hd; ++e) out[e] += p * v[e];
  }
}

static inline float silu(float z) { return z / (1.0f + expf(-z)); }

/*
 * Forward m new rows of one sequence.
 *   tokens[m], pos[m]: ids and absolute positions of the new rows.
 *   kc, vc: this sequence's cache, [n_layers][max_pos][hkv][hd] fp32 each;
 *           every position <= max(pos) must be cached or among the new rows.
 *   out_rows[n_out]: rows whose logits are written to logits[n_out][vocab]
 *   hidden (optional): final-norm input h, [m][d].
 *   kv_bf16: store keys and values rounded to bf16 (else as fp32).
 */
int oracle_forward(const ocfg* c, const oweights* w, float* kc, float* vc, int32_t max_pos,
                   const int32_t* tokens, int32_t m, const int32_t* pos,
                   const int32_t* out_rows, int32_t n_out, float* logits, float* hidden, int32_t kv_bf16) {
  const int32_t d = c->d, hq = c->hq, hkv = c->hkv, hd = c->hd, ffn = c->ffn;
  const int32_t qd = hq * hd, kvd = hkv * hd, group = hq / hkv;
  for (int32_t i = 0; i < m; ++i) {
    if (pos[i] < 0 || pos[i] >= max_pos) return -1;
    if (tokens[i] < 0 || tokens[i] >= c->vocab) return -2;
  }
  float* h = (float*)malloc(sizeof(float) * (size_t)m * d);
  float* x = (float*)malloc(sizeof(float) * (size_t)m * d);
  float* q = (float*)malloc(sizeof(float) * (size_t)m * qd);
  float* k = (float*)malloc(sizeof(float) * (size_t)m * kvd);
  float* v = (float*)malloc(sizeof(float) * (size_t)m * kvd);
  float* o = (float*)malloc(sizeof(float) * (size_t)m * qd);
  float* t = (float*)malloc(sizeof(float) * (size_t)m * d);
  float* g = (float*)malloc(sizeof(float) * (size_t)m * ffn);
  float* u = (float*)malloc(sizeof(float) * (size_t)m * ffn);

  for (int32_t i = 0; i < m; ++i) widen(w->embed + (int64_t)tokens[i] * d, h + (int64_t)i * d, d);

  for (int32_t l = 0; l < c->n_layers; ++l) {
    const uint16_t* const* W = w->layers + (int64_t)l * T_PER_LAYER;
    float* kl = kc + (int64_t)l * max_pos * kvd;
    float* vl = vc + (int64_t)l * max_pos * kvd;

    for (int32_t i = 0; i < m; ++i) oracle_rmsnorm(h + (int64_t)i * d, W[T_ATTN_NORM], d, c->eps, x + (int64_t)i * d);
    oracle_matmul(x, m, d, W[T_WQ], qd, q);
    oracle_matmul(x, m, d, W[T_WK], kvd, k);
    oracle_matmul(x, m, d, W[T_WV], kvd, v);
    for (int32_t i = 0; i < m; ++i) {
      for (int32_t hh = 0; hh < hq; ++hh) oracle_rope(q + (int64_t)i * qd + hh * hd, hd, pos[i], c->theta);
      for (int32_t hh = 0; hh < hkv; ++hh) oracle_rope(k + (int64_t)i * kvd + hh * hd, hd, pos[i], c->theta);
      for (int32_t e = 0; e < kvd; ++e) {
        const float ke = k[(int64_t)i * kvd + e], ve = v[(int64_t)i * kvd + e];
        kl[(int64_t)pos[i] * kvd + e] = kv_bf16 ? round_bf16(ke) : ke;
        vl[(int64_t)pos[i] * kvd + e] = kv_bf16 ? round_bf16(ve) : ve;
      }
    }
#pragma omp parallel
    {
      float* scratch = (float*)malloc(sizeof(float) * (size_t)max_pos);
#pragma omp for schedule(dynamic) collapse(2)
      for (int32_t i = 0; i < m; ++i)
        for (int32_t hh = 0; hh < hq; ++hh)
          oracle_attend(q + (int64_t)i * qd + hh * hd, kl, vl, hkv, hd, hh / group, pos[i], scratch,
                        o + (int64_t)i * qd + hh * hd);
      free(scratch);
    }
    oracle_matmul(o, m, qd, W[T_WO], d, t);
    for (int64_t e = 0; e < (int64_t)m * d; ++e) h[e] += t[e];

    for (int32_t i = 0; i < m; ++i) oracle_rmsnorm(h + (int64_t)i * d, W[T_MLP_NORM], d, c->eps, x + (int64_t)i * d);
    oracle_matmul(x, m, d, W[T_WG], ffn, g);
    oracle_matmul(x, m, d, W[T_WU], ffn, u);
    for (int64_t e = 0; e < (int64_t)m * ffn; ++e) g[e] = silu(g[e]) * u[e];
    oracle_matmul(g, m, ffn, W[T_WD], d, t);
    for (int64_t e = 0; e < (int64_t)m * d; ++e) h[e] += t[e];
  }

  if (hidden) memcpy(hidden, h, sizeof(float) * (size_t)m * d);
  if (n_out > 0) {
    for (int32_t j = 0; j < n_out; ++j) {
      if (out_rows[j] < 0 || out_rows[j] >= m) { n_out = -1; break; }
      oracle_rmsnorm(h + (int64_t)out_rows[j] * d, w->final_norm, d, c->eps, x + (int64_t)j * d);
    }
    if (n_out > 0) oracle_matmul(x, n_out, d, w->lm_head, c->vocab, logits);
  }
  free(h); free(x); free(q); free(k); free(v); free(o); free(t); free(g); free(u);
  return n_out < 0 ? -3 : 0;
}
