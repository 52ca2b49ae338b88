/*
 * CPU ORACLE -- test infrastructure only.
 *
 * A plain, slow, obviously correct fp32 forward of the Llama-style decoder
 * whose prefill the restore path serves, over an explicit KV state.  Only the
 * tests, the smoke check and the benchmark's CPU-baseline leg use it; the
 * product library never calls, links or loads it, and it shares no code with
 * the CUDA path.
 *
 * What it computes (the paper's Sec. 2.1 prefill: every token's K/V are
 * computed per layer and stored as the KV cache; first-token generation then
 * touches every weight and every cached K/V, Sec. 7), with the model details
 * the paper leaves open fixed as follows (Llama-style, Sec. 6.1 models are
 * decoder-only transformers):
 *   x      = E[token]                                 (embedding row, fp32)
 *   per layer:
 *     h    = RMSNorm(x) * g_attn                      (eps from the shape)
 *     q,k,v= h Wq^T, h Wk^T, h Wv^T                   (W stored [out][in])
 *     q,k  = RoPE(q,k; position)                      (half-split pairs (i, i+hd/2))
 *     K[pos],V[pos] = round_kv(k), round_kv(v)        (stored after RoPE)
 *     a    = softmax(q K[0..pos]^T / sqrt(hd)) V[0..pos]   per query head,
 *            query head h reads KV head h / (Hq/Hkv)   (grouped-query attention)
 *     x   += a Wo^T
 *     h    = RMSNorm(x) * g_ffn
 *     x   += (silu(h Wgate^T) * (h Wup^T)) Wdown^T
 *   logits = RMSNorm(x_last) * g_final  Wlm^T
 *
 * Numerics: fp32 throughout; weights are bf16 bit patterns widened exactly;
 * every dot product sums in increasing index order; softmax is the two-pass
 * max-subtracted form over keys in increasing position.  Each row is computed
 * on its own, so the result does not depend on how rows are batched or on
 * the thread count (chunked prefill equals full prefill bit for bit).
 * K and V are rounded to the KV storage type (bf16, fp16 or kept fp32) when
 * stored, the one rounding point the method itself fixes (FP16 KV chunks,
 * Sec. 4.3 footnote).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_KV_BF16 0
#define ORC_KV_FP16 1
#define ORC_KV_F32 2

typedef struct {
  int32_t n_layers, d_model, n_q_heads, n_kv_heads, head_dim, ffn_dim, vocab;
  float rope_theta, rms_eps;
  int32_t kv_dtype;
} orc_shape;

typedef struct {
  const uint16_t *wq, *wk, *wv, *wo, *w_gate, *w_up, *w_down; /* bf16 [out][in] */
  const float *attn_norm, *ffn_norm;                          /* [d_model] */
} orc_layer;

/* ---- scalar conversions ------------------------------------------------ */

static inline float bf16_to_f32(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, 4);
  return f;
}

/* fp32 -> bf16, round to nearest, ties to even (finite inputs). */
uint16_t orc_f32_to_bf16(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

/* fp32 -> IEEE binary16, round to nearest, ties to even; overflow -> inf. */
uint16_t orc_f32_to_f16(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  uint32_t sign = (u >> 16) & 0x8000u;
  uint32_t absu = u & 0x7FFFFFFFu;
  if (absu >= 0x7F800000u) return (uint16_t)(sign | (absu > 0x7F800000u ? 0x7E00u : 0x7C00u));
  int32_t e = (int32_t)(absu >> 23) - 127; /* unbiased exponent */
  uint32_t mant = (absu & 0x7FFFFFu) | 0x800000u;
  if (absu == 0) return (uint16_t)sign;
  if (e > 15) return (uint16_t)(sign | 0x7C00u);
  int32_t shift; /* bits of the 24-bit significand to drop */
  uint32_t base;
  if (e >= -14) { /* normal half: keep 11 significant bits */
    shift = 13;
    base = (uint32_t)(e + 15) << 10;
    mant &= 0x7FFFFFu; /* implicit bit handled by the exponent field */
  } else {          /* subnormal half: value = m * 2^-24 */
    shift = 13 + (-14 - e);
    if (shift > 24) return (uint16_t)sign; /* below half of the smallest subnormal */
    base = 0;
  }
  uint32_t q = mant >> shift;
  uint32_t rem = mant & ((1u << shift) - 1u);
  uint32_t half = 1u << (shift - 1);
  if (rem > half || (rem == half && (q & 1u))) q += 1u;
  return (uint16_t)(sign | (base + q)); /* a carry out of the mantissa bumps the exponent */
}

static float f16_to_f32(uint16_t h) {
  uint32_t sign = (uint32_t)(h & 0x8000u) << 16;
  int32_t e = (h >> 10) & 0x1F;
  uint32_t m = h & 0x3FFu;
  float v;
  if (e == 0) v = ldexpf((float)m, -24);
  else if (e == 31) v = m ? NAN : INFINITY;
  else v = ldexpf((float)(m | 0x400u), e - 25);
  uint32_t u;
  memcpy(&u, &v, 4);
  u |= sign;
  memcpy(&v, &u, 4);
  return v;
}

float orc_round_kv(float x, int32_t kv_dtype) {
  if (kv_dtype == ORC_KV_BF16) return bf16_to_f32(orc_f32_to_bf16(x));
  if (kv_dtype == ORC_KV_FP16) return f16_to_f32(orc_f32_to_f16(x));
  return x;
}

/* ---- per-row operations (each is the plain definition) ------------------ */

/* y = x / sqrt(mean(x^2) + eps) * g   (RMSNorm, Zhang & Sennrich 2019) */
void orc_rmsnorm_row(const float* x, const float* g, int32_t d, float eps, float* y) {
  float ss = 0.0f;
  for (int32_t k = 0; k < d; ++k) ss += x[k] * x[k];
  float r = 1.0f / sqrtf(ss / (float)d + eps);
  for (int32_t k = 0; k < d; ++k) y[k] = x[k] * r * g[k];
}

/* y[j] = sum_k x[k] * W[j][k], k increasing; W bf16 [n_out][n_in]. */
void orc_linear_row(const float* x, const uint16_t* w, int32_t n_in, int32_t n_out, float* y) {
  for (int32_t j = 0; j < n_out; ++j) {
    const uint16_t* wr = w + (int64_t)j * n_in;
    float acc = 0.0f;
    for (int32_t k = 0; k < n_in; ++k) acc += x[k] * bf16_to_f32(wr[k]);
    y[j] = acc;
  }
}

/* Rotary table: angle(pos, i) = pos * theta^(-2i/hd), evaluated in double and
 * rounded to fp32 (RoFormer, Su et al. 2021).  cos/sin are [n_pos][hd/2]. */
void orc_rope_table(int64_t n_pos, int32_t hd, double theta, float* cos_out, float* sin_out) {
  int32_t half = hd / 2;
  for (int64_t p = 0; p < n_pos; ++p)
    for (int32_t i = 0; i < half; ++i) {
      double inv = pow(theta, -2.0 * (double)i / (double)hd);
      double a = (double)p * inv;
      cos_out[p * half + i] = (float)cos(a);
      sin_out[p * half + i] = (float)sin(a);
    }
}

/* Rotate one head vector in place with pairs (i, i + hd/2). */
void orc_rope_head(float* x, const float* cs, const float* sn, int32_t hd) {
  int32_t half = hd / 2;
  for (int32_t i = 0; i < half; ++i) {
    float x1 = x[i], x2 = x[i + half];
    x[i] = x1 * cs[i] - x2 * sn[i];
    x[i + half] = x2 * cs[i] + x1 * sn[i];
  }
}

/* Causal attention of one query head over keys 0..pos of one KV head.
 * k_base/v_base point at position 0 of that KV head; consecutive positions are
 * `pos_stride` floats apart.  Two-pass softmax, scale 1/sqrt(hd). */
void orc_attend_head(const float* q, const float* k_base, const float* v_base, int64_t pos_stride,
                     int64_t pos, int32_t hd, float* scores /* pos+1 */, float* out) {
  float scale = 1.0f / sqrtf((float)hd);
  float m = -INFINITY;
  for (int64_t j = 0; j <= pos; ++j) {
    const float* kj = k_base + j * pos_stride;
    float s = 0.0f;
    for (int32_t c = 0; c < hd; ++c) s += q[c] * kj[c];
    s *= scale;
    scores[j] = s;
    if (s > m) m = s;
  }
  float denom = 0.0f;
  for (int64_t j = 0; j <= pos; ++j) {
    scores[j] = expf(scores[j] - m);
    denom += scores[j];
  }
  for (int32_t c = 0; c < hd; ++c) out[c] = 0.0f;
  for (int64_t j = 0; j <= pos; ++j) {
    const float* vj = v_base + j * pos_stride;
    float p = scores[j];
    for (int32_t c = 0; c < hd; ++c) out[c] += p * vj[c];
  }
  for (int32_t c = 0; c < hd; ++c) out[c] /= denom;
}

static inline float silu(float g) { return g / (1.0f + expf(-g)); }

/* ---- the forward --------------------------------------------------------- */

/*
 * Process rows (tokens[i] at position pos[i]) through every layer over the KV
 * state k_cache/v_cache ([n_layers][max_ctx][n_kv_heads][head_dim] fp32,
 * already holding the stored values of every other position the rows attend
 * to).  Writes the rows' K/V into the cache and, if `logits` is not NULL, the
 * logits of the LAST row.  If `x_out` is not NULL it receives the final
 * residual stream [n_rows][d_model] (before the final norm).
 * Rows may come in any order; row i attends to every cached position <= pos[i],
 * including rows of this call.  Returns 0, or -1 on a bad argument.
 */
int orc_forward(const orc_shape* s, const uint16_t* embed, const uint16_t* lm_head,
                const float* final_norm, const orc_layer* layers, float* k_cache,
                float* v_cache, int64_t max_ctx, const int32_t* tokens, const int64_t* pos,
                int64_t n_rows, float* logits, float* x_out) {
  const int32_t d = s->d_model, hq = s->n_q_heads, hkv = s->n_kv_heads, hd = s->head_dim;
  const int32_t f = s->ffn_dim, group = hq / hkv;
  if (hkv <= 0 || hq % hkv != 0 || hd % 2 != 0 || n_rows < 0) return -1;
  int64_t max_pos = -1;
  for (int64_t i = 0; i < n_rows; ++i) {
    if (pos[i] < 0 || pos[i] >= max_ctx || tokens[i] < 0 || tokens[i] >= s->vocab) return -1;
    if (pos[i] > max_pos) max_pos = pos[i];
  }
  if (n_rows == 0) return 0;
  const int32_t half = hd / 2;
  float* cosT = (float*)malloc(sizeof(float) * (size_t)(max_pos + 1) * half);
  float* sinT = (float*)malloc(sizeof(float) * (size_t)(max_pos + 1) * half);
  orc_rope_table(max_pos + 1, hd, (double)s->rope_theta, cosT, sinT);

  float* x = (float*)malloc(sizeof(float) * (size_t)n_rows * d);
  float* q = (float*)malloc(sizeof(float) * (size_t)n_rows * hq * hd);
  for (int64_t i = 0; i < n_rows; ++i)
    for (int32_t c = 0; c < d; ++c) x[i * d + c] = bf16_to_f32(embed[(int64_t)tokens[i] * d + c]);

  const int64_t kv_pos_stride = (int64_t)hkv * hd;
  const int64_t kv_layer_stride = max_ctx * kv_pos_stride;

  for (int32_t l = 0; l < s->n_layers; ++l) {
    const orc_layer* w = &layers[l];
    float* Kl = k_cache + l * kv_layer_stride;
    float* Vl = v_cache + l * kv_layer_stride;
    /* 1) norm, projections, rotary, KV store -- every row before any attention */
#pragma omp parallel
    {
      float* h = (float*)malloc(sizeof(float) * d);
      float* kv = (float*)malloc(sizeof(float) * 2 * hkv * hd);
#pragma omp for schedule(dynamic)
      for (int64_t i = 0; i < n_rows; ++i) {
        orc_rmsnorm_row(x + i * d, w->attn_norm, d, s->rms_eps, h);
        orc_linear_row(h, w->wq, d, hq * hd, q + i * hq * hd);
        orc_linear_row(h, w->wk, d, hkv * hd, kv);
        orc_linear_row(h, w->wv, d, hkv * hd, kv + hkv * hd);
        const float* cs = cosT + pos[i] * half;
        const float* sn = sinT + pos[i] * half;
        for (int32_t a = 0; a < hq; ++a) orc_rope_head(q + (i * hq + a) * hd, cs, sn, hd);
        for (int32_t a = 0; a < hkv; ++a) orc_rope_head(kv + a * hd, cs, sn, hd);
        for (int32_t c = 0; c < hkv * hd; ++c) {
          Kl[pos[i] * kv_pos_stride + c] = orc_round_kv(kv[c], s->kv_dtype);
          Vl[pos[i] * kv_pos_stride + c] = orc_round_kv(kv[hkv * hd + c], s->kv_dtype);
        }
      }
      free(h);
      free(kv);
    }
    /* 2) attention, output projection, MLP -- row by row */
#pragma omp parallel
    {
      float* sc = (float*)malloc(sizeof(float) * (size_t)(max_pos + 1));
      float* att = (float*)malloc(sizeof(float) * hq * hd);
      float* o = (float*)malloc(sizeof(float) * d);
      float* h = (float*)malloc(sizeof(float) * d);
      float* g = (float*)malloc(sizeof(float) * f);
      float* u = (float*)malloc(sizeof(float) * f);
#pragma omp for schedule(dynamic)
      for (int64_t i = 0; i < n_rows; ++i) {
        for (int32_t a = 0; a < hq; ++a) {
          int32_t kvh = a / group;
          orc_attend_head(q + (i * hq + a) * hd, Kl + kvh * hd, Vl + kvh * hd, kv_pos_stride,
                          pos[i], hd, sc, att + a * hd);
        }
        orc_linear_row(att, w->wo, hq * hd, d, o);
        for (int32_t c = 0; c < d; ++c) x[i * d + c] += o[c];
        orc_rmsnorm_row(x + i * d, w->ffn_norm, d, s->rms_eps, h);
        orc_linear_row(h, w->w_gate, d, f, g);
        orc_linear_row(h, w->w_up, d, f, u);
        for (int32_t c = 0; c < f; ++c) g[c] = silu(g[c]) * u[c];
        orc_linear_row(g, w->w_down, f, d, o);
        for (int32_t c = 0; c < d; ++c) x[i * d + c] += o[c];
      }
      free(sc); free(att); free(o); free(h); free(g); free(u);
    }
  }
  if (x_out) memcpy(x_out, x, sizeof(float) * (size_t)n_rows * d);
  if (logits) {
    float* h = (float*)malloc(sizeof(float) * d);
    orc_rmsnorm_row(x + (n_rows - 1) * d, final_norm, d, s->rms_eps, h);
    /* one dot product per vocabulary entry; split across threads by entry */
#pragma omp parallel for schedule(static)
    for (int32_t j = 0; j < s->vocab; ++j) orc_linear_row(h, lm_head + (int64_t)j * d, d, 1, logits + j);
    free(h);
  }
  free(x); free(q); free(cosT); free(sinT);
  return 0;
}

/* ---- single operations, for kernel-level parity ------------------------- */

void orc_rmsnorm(const float* x, const float* g, int64_t n, int32_t d, float eps, float* y) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) orc_rmsnorm_row(x + i * d, g, d, eps, y + i * d);
}

/* Y[n][n_out] = X[n][n_in] W^T, W bf16 [n_out][n_in]; parallel over (row, out). */
void orc_linear(const float* x, const uint16_t* w, int64_t n, int32_t n_in, int32_t n_out, float* y) {
#pragma omp parallel for collapse(2) schedule(static)
  for (int64_t i = 0; i < n; ++i)
    for (int32_t j = 0; j < n_out; ++j)
      orc_linear_row(x + i * n_in, w + (int64_t)j * n_in, n_in, 1, y + i * n_out + j);
}

/* silu(g) * u elementwise */
void orc_swiglu(const float* g, const float* u, int64_t n, float* y) {
  for (int64_t i = 0; i < n; ++i) y[i] = silu(g[i]) * u[i];
}

/* Rotate x[n][n_heads][hd] in place by positions pos[n]. */
void orc_rope(float* x, const int64_t* pos, int64_t n, int32_t n_heads, int32_t hd, double theta) {
  int32_t half = hd / 2;
  int64_t mp = 0;
  for (int64_t i = 0; i < n; ++i) if (pos[i] > mp) mp = pos[i];
  float* cs = (float*)malloc(sizeof(float) * (size_t)(mp + 1) * half);
  float* sn = (float*)malloc(sizeof(float) * (size_t)(mp + 1) * half);
  orc_rope_table(mp + 1, hd, theta, cs, sn);
  for (int64_t i = 0; i < n; ++i)
    for (int32_t a = 0; a < n_heads; ++a)
      orc_rope_head(x + (i * n_heads + a) * hd, cs + pos[i] * half, sn + pos[i] * half, hd);
  free(cs); free(sn);
}

/* Causal GQA attention: q[n][hq][hd] at positions pos[n] over cache
 * k/v[ctx][hkv][hd] (fp32, stored values) -> out[n][hq][hd]. */
void orc_attention(const float* q, const int64_t* pos, int64_t n, int32_t hq, int32_t hkv,
                   int32_t hd, const float* k, const float* v, int64_t ctx, float* out) {
  int32_t group = hq / hkv;
#pragma omp parallel
  {
    float* sc = (float*)malloc(sizeof(float) * (size_t)ctx);
#pragma omp for collapse(2) schedule(dynamic)
    for (int64_t i = 0; i < n; ++i)
      for (int32_t a = 0; a < hq; ++a)
        orc_attend_head(q + (i * hq + a) * hd, k + (a / group) * hd, v + (a / group) * hd,
                        (int64_t)hkv * hd, pos[i], hd, sc, out + (i * hq + a) * hd);
    free(sc);
  }
}

void orc_round_kv_array(const float* x, int64_t n, int32_t kv_dtype, float* y) {
  for (int64_t i = 0; i < n; ++i) y[i] = orc_round_kv(x[i], kv_dtype);
}

void orc_f32_to_f16_array(const float* x, int64_t n, uint16_t* y) {
  for (int64_t i = 0; i < n; ++i) y[i] = orc_f32_to_f16(x[i]);
}

void orc_f32_to_bf16_array(const float* x, int64_t n, uint16_t* y) {
  for (int64_t i = 0; i < n; ++i) y[i] = orc_f32_to_bf16(x[i]);
}

/* ---- 8-bit swap codec ------------------------------------------------------
 * The paper keeps swapped KV compressed, with 8-bit quantization as the
 * default codec (Sec. 5), and notes that it is idempotent: compressing the
 * decompressed values again gives the same result (Sec. 6.5).  The format is
 * not given; reading used here: asymmetric min/max quantization over groups
 * of 64 consecutive values (one group = 64 head_dim entries of one K or V
 * row), fp32 minimum and step, step = (max - min) / 255,
 *   code  = round-half-even((x - min) / step), clamped to [0, 255]
 *           (0 for every value of a constant group, step == 0),
 *   value = code * step + min   (two fp32 roundings, no fused multiply-add).
 */
void orc_q8_encode(const float* x, int64_t n_groups, uint8_t* codes, float* mn_out,
                   float* step_out) {
  for (int64_t g = 0; g < n_groups; ++g) {
    const float* v = x + g * 64;
    float mn = v[0], mx = v[0];
    for (int i = 1; i < 64; ++i) {
      if (v[i] < mn) mn = v[i];
      if (v[i] > mx) mx = v[i];
    }
    const float step = (mx - mn) / 255.0f;
    for (int i = 0; i < 64; ++i) {
      uint8_t c = 0;
      if (step > 0.0f) {
        const float q = rintf((v[i] - mn) / step);
        c = q <= 0.0f ? 0 : (q >= 255.0f ? 255 : (uint8_t)q);
      }
      codes[g * 64 + i] = c;
    }
    mn_out[g] = mn;
    step_out[g] = step;
  }
}

void orc_q8_decode(const uint8_t* codes, const float* mn, const float* step, int64_t n_groups,
                   float* out) {
  for (int64_t g = 0; g < n_groups; ++g)
    for (int i = 0; i < 64; ++i) {
      const float prod = (float)codes[g * 64 + i] * step[g];
      out[g * 64 + i] = prod + mn[g];
    }
}

int orc_num_threads(void) {
#ifdef _OPENMP
  extern int omp_get_max_threads(void);
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/* Sets the OpenMP thread count of later calls (n >= 1); timing only. */
void orc_set_num_threads(int n) {
#ifdef _OPENMP
  extern void omp_set_num_threads(int);
  if (n >= 1) omp_set_num_threads(n);
#else
  (void)n;
#endif
}
