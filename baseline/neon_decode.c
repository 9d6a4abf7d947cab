/*
 * neon_decode.c — the paper's own method on one host core, as a timing
 * baseline for the benchmark (not the parity reference, which is the oracle,
 * and not part of the GPU library; the two share nothing).
 *
 * One float32 decode step of a Llama-2-architecture decoder (§2.1) in which
 * the matrix-vector products and RMSNorm run on 128-bit NEON vectors:
 *   - GEMV (§6.1): each output row is one dot product over float32x4 lanes;
 *     §11.1: four independent vector accumulators, so that consecutive fused
 *     multiply-adds of a row do not wait on each other; the four are added
 *     and reduced across lanes at the end of the row.
 *   - RMSNorm (§11.2): the sum of squares on vectors, one scalar reciprocal
 *     square root of (sum / n + eps), then (x * g) * r on vectors.
 * RoPE, attention and the SwiGLU gate are plain scalar float loops, as the
 * paper leaves them. On hosts without NEON (not aarch64) the same loops run
 * with four scalar accumulators of four lanes each in plain C.
 *
 * Weights are borrowed: the caller passes one pointer per tensor (float32,
 * row-major [rows x cols]) and keeps them alive; the handle owns the KV cache
 * and the activations.
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>

#if defined(__aarch64__)
#include <arm_neon.h>
#define NB_NEON 1
#else
#define NB_NEON 0
#endif

typedef struct {
  int dim, hidden, n_layers, n_heads, n_kv_heads, vocab, max_seq;
  float rope_theta, eps;
  const float* E;
  const float* g_final;
  const float* Wcls;
  /* per layer, n_layers entries each */
  const float* const* g_att;
  const float* const* Wq;
  const float* const* Wk;
  const float* const* Wv;
  const float* const* Wo;
  const float* const* g_ffn;
  const float* const* W1;
  const float* const* W3;
  const float* const* W2;
} nb_weights;

typedef struct {
  nb_weights w;
  int hd, kvd;
  float *x, *xb, *q, *k, *v, *o, *y, *a, *b, *h, *att, *kc, *vc;
} nb_model;

int nb_has_neon(void) { return NB_NEON; }

/* y[i] = W[i] . x for rows i < M of W [M x K]. */
static void nb_gemv(const float* W, const float* x, float* y, int M, int K) {
  for (int i = 0; i < M; ++i) {
    const float* w = W + (size_t)i * K;
    int j = 0;
#if NB_NEON
    float32x4_t s0 = vdupq_n_f32(0.f), s1 = s0, s2 = s0, s3 = s0;
    for (; j + 16 <= K; j += 16) {
      s0 = vfmaq_f32(s0, vld1q_f32(w + j), vld1q_f32(x + j));
      s1 = vfmaq_f32(s1, vld1q_f32(w + j + 4), vld1q_f32(x + j + 4));
      s2 = vfmaq_f32(s2, vld1q_f32(w + j + 8), vld1q_f32(x + j + 8));
      s3 = vfmaq_f32(s3, vld1q_f32(w + j + 12), vld1q_f32(x + j + 12));
    }
    for (; j + 4 <= K; j += 4) s0 = vfmaq_f32(s0, vld1q_f32(w + j), vld1q_f32(x + j));
    float acc = vaddvq_f32(vaddq_f32(vaddq_f32(s0, s1), vaddq_f32(s2, s3)));
#else
    float s[4][4] = {{0}};
    for (; j + 16 <= K; j += 16)
      for (int u = 0; u < 4; ++u)
        for (int l = 0; l < 4; ++l) s[u][l] += w[j + 4 * u + l] * x[j + 4 * u + l];
    for (; j + 4 <= K; j += 4)
      for (int l = 0; l < 4; ++l) s[0][l] += w[j + l] * x[j + l];
    float acc = 0.f;
    for (int l = 0; l < 4; ++l) acc += (s[0][l] + s[1][l]) + (s[2][l] + s[3][l]);
#endif
    for (; j < K; ++j) acc += w[j] * x[j];
    y[i] = acc;
  }
}

/* out = (x * g) * 1/sqrt(mean(x^2) + eps). */
static void nb_rmsnorm(const float* x, const float* g, float* out, int n, float eps) {
  int j = 0;
  float ss;
#if NB_NEON
  float32x4_t v = vdupq_n_f32(0.f);
  for (; j + 4 <= n; j += 4) {
    const float32x4_t t = vld1q_f32(x + j);
    v = vfmaq_f32(v, t, t);
  }
  ss = vaddvq_f32(v);
#else
  float l4[4] = {0, 0, 0, 0};
  for (; j + 4 <= n; j += 4)
    for (int l = 0; l < 4; ++l) l4[l] += x[j + l] * x[j + l];
  ss = (l4[0] + l4[1]) + (l4[2] + l4[3]);
#endif
  for (; j < n; ++j) ss += x[j] * x[j];
  const float r = 1.0f / sqrtf(ss / (float)n + eps);
  j = 0;
#if NB_NEON
  const float32x4_t vr = vdupq_n_f32(r);
  for (; j + 4 <= n; j += 4)
    vst1q_f32(out + j, vmulq_f32(vmulq_f32(vld1q_f32(x + j), vld1q_f32(g + j)), vr));
#endif
  for (; j < n; ++j) out[j] = (x[j] * g[j]) * r;
}

/* Adjacent pairs of each head turn by pos * theta^(-2i/hd). */
static void nb_rope(float* v, int n, int hd, int pos, float theta) {
  for (int i = 0; i < n; i += 2) {
    const int j = i % hd;
    const float ang = (float)pos * powf(theta, -(float)j / (float)hd);
    const float c = cosf(ang), s = sinf(ang);
    const float a = v[i], b = v[i + 1];
    v[i] = a * c - b * s;
    v[i + 1] = a * s + b * c;
  }
}

void nb_free(void* hp) {
  nb_model* m = (nb_model*)hp;
  if (!m) return;
  free(m->x);
  free(m->kc);
  free(m->vc);
  free(m);
}

void* nb_new(const nb_weights* w) {
  if (!w || w->dim <= 0 || w->n_heads <= 0 || w->n_kv_heads <= 0 || w->max_seq <= 0) return 0;
  nb_model* m = (nb_model*)calloc(1, sizeof(nb_model));
  if (!m) return 0;
  m->w = *w;
  const int d = w->dim, F = w->hidden, L = w->n_layers > 0 ? w->n_layers : 1;
  m->hd = d / w->n_heads;
  m->kvd = w->n_kv_heads * m->hd;
  const size_t acts = (size_t)6 * d + 3 * (size_t)m->kvd + 3 * (size_t)F + (size_t)w->max_seq;
  m->x = (float*)calloc(acts, sizeof(float));
  m->kc = (float*)calloc((size_t)L * w->max_seq * m->kvd, sizeof(float));
  m->vc = (float*)calloc((size_t)L * w->max_seq * m->kvd, sizeof(float));
  if (!m->x || !m->kc || !m->vc) {
    nb_free(m);
    return 0;
  }
  float* p = m->x;
  m->xb = p += d;
  m->q = p += d;
  m->o = p += d;
  m->y = p += d;
  m->k = p += d;
  m->v = p += m->kvd;
  m->a = p += m->kvd;
  m->b = p += F;
  m->h = p += F;
  m->att = p += F;
  return m;
}

int nb_forward(void* hp, int token, int pos, float* logits) {
  nb_model* m = (nb_model*)hp;
  const nb_weights* w = &m->w;
  const int d = w->dim, F = w->hidden, hd = m->hd, kvd = m->kvd, S = w->max_seq;
  if (token < 0 || token >= w->vocab || pos < 0 || pos >= S) return 6;
  memcpy(m->x, w->E + (size_t)token * d, sizeof(float) * d);
  const int group = w->n_heads / w->n_kv_heads;
  const float scale = 1.0f / sqrtf((float)hd);
  for (int l = 0; l < w->n_layers; ++l) {
    nb_rmsnorm(m->x, w->g_att[l], m->xb, d, w->eps);
    nb_gemv(w->Wq[l], m->xb, m->q, d, d);
    nb_gemv(w->Wk[l], m->xb, m->k, kvd, d);
    nb_gemv(w->Wv[l], m->xb, m->v, kvd, d);
    nb_rope(m->q, d, hd, pos, w->rope_theta);
    nb_rope(m->k, kvd, hd, pos, w->rope_theta);
    float* Kc = m->kc + (size_t)l * S * kvd;
    float* Vc = m->vc + (size_t)l * S * kvd;
    memcpy(Kc + (size_t)pos * kvd, m->k, sizeof(float) * kvd);
    memcpy(Vc + (size_t)pos * kvd, m->v, sizeof(float) * kvd);
    for (int hh = 0; hh < w->n_heads; ++hh) {
      const float* qh = m->q + hh * hd;
      const int kh = hh / group;
      float mx = -INFINITY;
      for (int t = 0; t <= pos; ++t) {
        const float* kr = Kc + (size_t)t * kvd + kh * hd;
        float s = 0.f;
        for (int j = 0; j < hd; ++j) s += qh[j] * kr[j];
        m->att[t] = s * scale;
        if (m->att[t] > mx) mx = m->att[t];
      }
      float z = 0.f;
      for (int t = 0; t <= pos; ++t) {
        m->att[t] = expf(m->att[t] - mx);
        z += m->att[t];
      }
      float* oh = m->o + hh * hd;
      for (int j = 0; j < hd; ++j) oh[j] = 0.f;
      for (int t = 0; t <= pos; ++t) {
        const float e = m->att[t] / z;
        const float* vr = Vc + (size_t)t * kvd + kh * hd;
        for (int j = 0; j < hd; ++j) oh[j] += e * vr[j];
      }
    }
    nb_gemv(w->Wo[l], m->o, m->y, d, d);
    for (int j = 0; j < d; ++j) m->x[j] += m->y[j];
    nb_rmsnorm(m->x, w->g_ffn[l], m->xb, d, w->eps);
    nb_gemv(w->W1[l], m->xb, m->a, F, d);
    nb_gemv(w->W3[l], m->xb, m->b, F, d);
    for (int i = 0; i < F; ++i) m->h[i] = (m->a[i] / (1.0f + expf(-m->a[i]))) * m->b[i];
    nb_gemv(w->W2[l], m->h, m->y, d, F);
    for (int j = 0; j < d; ++j) m->x[j] += m->y[j];
  }
  nb_rmsnorm(m->x, w->g_final, m->xb, d, w->eps);
  nb_gemv(w->Wcls, m->xb, logits, w->vocab, d);
  return 0;
}
