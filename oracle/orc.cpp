// orc.cpp — CPU oracle of the batch-1 Llama-2 decode step (test infrastructure).
//
// Only tests/, __graft_entry__.smoke() and the bench's CPU-baseline and
// reference arms load this library. It shares no code, header, table or
// constant with the CUDA path; the two meet only at the packed weight blob
// that the seeded generator writes.
//
// What is computed, and where the paper fixes it (Kilictas & Alpay,
// "Bare-Metal Tensor Virtualization", arXiv 2601.03324):
//   * y = W x, one dot product per output row          — §3.1 (Roofline, GEMV
//     data movement) and §6.1 (GEMV listing).
//   * RMSNorm: ss = sum x^2; ss = ss/n + 1e-5; r = 1/sqrt(ss); o = (x*g)*r
//                                                      — §2.1, §11.2 listing.
//   * SwiGLU FFN with three matrices W1, W2, W3        — §2.1.
//   * RoPE, rotating q and k "in the complex plane"    — §2.1.
//   * Attention over a KV cache, one new token per step— §1 (decode is GEMV
//     bound, every weight read once per token) and §2.1 (Llama 2 decoder).
//   * Classifier tied to the token embedding when the file is short — §5.1.
//   * Weight-only 8-bit codes with one scale per output row: a reading of
//     the quantization the paper leaves to future work (§ Future Work:
//     Quantization, which names 4-bit weights unpacked on the fly).
// Where the paper is silent, the readings taken are the standard Llama-2
// ones and are listed where they are used.
//
// Acc is the accumulator and activation type: double is the parity truth,
// float is the "scalar C++" analogue of Table 1. No SIMD, no threads, no
// reordering of any sum: every loop runs in index order.
#include "orc.h"

#include <cfenv>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

namespace {

int64_t align128(int64_t b) { return (b + 127) / 128 * 128; }

// Packed layout (the paper names a "Tensor Virtualization Layout" but does
// not define it; §4.1 only fixes that weights are pointers at offsets into
// one mapped file). Reading used here: float32 tensors, row-major
// [rows x cols], each starting at a 128-byte-aligned offset, in the order
//   E[V x d]; per layer: g_att[d], Wq[d x d], Wk[kvd x d], Wv[kvd x d],
//   Wo[d x d], g_ffn[d], W1[F x d], W3[F x d], W2[d x F]; g_final[d];
//   Wcls[V x d] unless tied.
struct Layout {
  int64_t E = 0, g_final = 0, Wcls = -1, total = 0;
  std::vector<int64_t> g_att, Wq, Wk, Wv, Wo, g_ffn, W1, W3, W2;
};

bool config_ok(const orc_config* c) {
  if (!c) return false;
  if (c->dim <= 0 || c->hidden_dim <= 0 || c->n_layers < 0 || c->n_heads <= 0 ||
      c->n_kv_heads <= 0 || c->vocab_size <= 0 || c->max_seq <= 0)
    return false;
  if (c->dim % c->n_heads != 0) return false;
  if (c->n_heads % c->n_kv_heads != 0) return false;
  if ((c->dim / c->n_heads) % 2 != 0) return false;  // RoPE rotates pairs
  return true;
}

Layout make_layout(const orc_config* c, bool tied) {
  Layout L;
  const int64_t d = c->dim, F = c->hidden_dim, V = c->vocab_size;
  const int64_t kvd = (int64_t)c->n_kv_heads * (d / c->n_heads);
  int64_t off = 0;
  auto take = [&](int64_t nfloats) {
    int64_t at = off;
    off = align128(off + nfloats * 4);
    return at;
  };
  L.E = take(V * d);
  for (int l = 0; l < c->n_layers; ++l) {
    L.g_att.push_back(take(d));
    L.Wq.push_back(take(d * d));
    L.Wk.push_back(take(kvd * d));
    L.Wv.push_back(take(kvd * d));
    L.Wo.push_back(take(d * d));
    L.g_ffn.push_back(take(d));
    L.W1.push_back(take(F * d));
    L.W3.push_back(take(F * d));
    L.W2.push_back(take(d * F));
  }
  L.g_final = take(d);
  if (!tied) L.Wcls = take(V * d);
  L.total = off;
  return L;
}

// ---- primitives ------------------------------------------------------------

// y[i] = sum_j W[i][j] * x[j]; W row-major [M x K] (§6.1 GEMV listing: one
// dot product per output row; the sum runs over j in index order here).
template <class Acc>
void gemv(const float* W, const Acc* x, Acc* y, int64_t M, int64_t K) {
  for (int64_t i = 0; i < M; ++i) {
    const float* w = W + i * K;
    Acc s = 0;
    for (int64_t j = 0; j < K; ++j) s += (Acc)w[j] * x[j];
    y[i] = s;
  }
}

// Weight-only codes with qmax levels on each side of zero (127 for 8-bit
// codes, 7 for 4-bit ones), one float32 scale per output row. Every decision
// is taken in float32, so that any implementation of the same definition
// finds the same codes: a_r = max_j |W_rj|; s_r = a_r / qmax; q_rj = the
// integer nearest to W_rj / s_r (ties to even), which lies in [-qmax, qmax];
// an all-zero row has s_r = 0 and codes 0. The weight a code stands for is
// s_r * q_rj.
void quantize_rows_levels(const float* W, int64_t M, int64_t K, float qmax, int8_t* q, float* s) {
  for (int64_t i = 0; i < M; ++i) {
    const float* w = W + i * K;
    float a = 0.0f;
    for (int64_t j = 0; j < K; ++j) a = std::fmax(a, std::fabs(w[j]));
    const float sc = a / qmax;
    s[i] = sc;
    for (int64_t j = 0; j < K; ++j) {
      float c = 0.0f;
      if (sc != 0.0f) {
        c = std::nearbyint(w[j] / sc);  // default rounding: nearest, ties to even
        if (c > qmax) c = qmax;
        if (c < -qmax) c = -qmax;
      }
      q[i * K + j] = (int8_t)c;
    }
  }
}

void quantize_rows(const float* W, int64_t M, int64_t K, int8_t* q, float* s) {
  quantize_rows_levels(W, M, K, 127.0f, q, s);
}

// y[i] = sum_j (s_i q_ij) x[j]: the GEMV of the weights the codes stand for.
template <class Acc>
void gemv_q8(const int8_t* q, const float* s, const Acc* x, Acc* y, int64_t M, int64_t K) {
  for (int64_t i = 0; i < M; ++i) {
    const int8_t* c = q + i * K;
    Acc acc = 0;
    for (int64_t j = 0; j < K; ++j) acc += ((Acc)s[i] * (Acc)c[j]) * x[j];
    y[i] = acc;
  }
}

// RMSNorm, §11.2 listing: mean of squares, plus epsilon, reciprocal square
// root, then the product (x * g) * r in that order.
template <class Acc>
void rmsnorm(const Acc* x, const float* g, Acc* out, int64_t n, Acc eps) {
  Acc ss = 0;
  for (int64_t j = 0; j < n; ++j) ss += x[j] * x[j];
  ss = ss / (Acc)n;
  ss = ss + eps;
  const Acc r = (Acc)1 / std::sqrt(ss);
  for (int64_t j = 0; j < n; ++j) out[j] = (x[j] * (Acc)g[j]) * r;
}

// RoPE (§2.1 names it; the formula is Su et al.'s): within each head of
// length hd, the pair (v[2i], v[2i+1]) is rotated by the angle
// pos * theta^(-2i/hd). Reading taken: adjacent pairs, the original Llama-2
// convention. The angle, cos and sin are computed in double and, for a
// float oracle, rounded once to float.
template <class Acc>
void rope(Acc* v, int64_t n, int64_t hd, int32_t pos, double theta) {
  for (int64_t i = 0; i < n; i += 2) {
    const int64_t j = i % hd;  // 2 * (pair index within the head)
    const double omega = std::pow(theta, -(double)j / (double)hd);
    const double angle = (double)pos * omega;
    const Acc c = (Acc)std::cos(angle), s = (Acc)std::sin(angle);
    const Acc a = v[i], b = v[i + 1];
    v[i] = a * c - b * s;
    v[i + 1] = a * s + b * c;
  }
}

// Softmax with the maximum subtracted first (reading: the standard stable form).
template <class Acc>
void softmax(Acc* s, int64_t n) {
  Acc m = s[0];
  for (int64_t i = 1; i < n; ++i)
    if (s[i] > m) m = s[i];
  Acc z = 0;
  for (int64_t i = 0; i < n; ++i) {
    s[i] = std::exp(s[i] - m);
    z += s[i];
  }
  for (int64_t i = 0; i < n; ++i) s[i] = s[i] / z;
}

// SiLU gate of SwiGLU (§2.1; Shazeer's GLU variants): z * sigmoid(z).
template <class Acc>
Acc silu(Acc z) { return z / ((Acc)1 + std::exp(-z)); }

// One head of causal attention for the newest token: scores q.k/sqrt(hd)
// over positions 0..npos-1 (reading: scale 1/sqrt(hd), causal, inclusive of
// the current position), softmax, then the weighted sum of V rows.
template <class Acc>
void attention_head(const Acc* q, const Acc* K, const Acc* V, int64_t npos, int64_t hd,
                    int64_t stride, Acc* out, Acc* scratch) {
  const Acc scale = (Acc)1 / std::sqrt((Acc)hd);
  for (int64_t t = 0; t < npos; ++t) {
    Acc s = 0;
    for (int64_t j = 0; j < hd; ++j) s += q[j] * K[t * stride + j];
    scratch[t] = s * scale;
  }
  softmax(scratch, npos);
  for (int64_t j = 0; j < hd; ++j) out[j] = 0;
  for (int64_t t = 0; t < npos; ++t)
    for (int64_t j = 0; j < hd; ++j) out[j] += scratch[t] * V[t * stride + j];
}

// ---- model -----------------------------------------------------------------

struct ModelBase {
  virtual ~ModelBase() {}
  virtual int forward(int32_t token, int32_t pos, double* logits) = 0;
  bool tied = false;
};

// One weight matrix as codes (qmax levels on each side of zero: 127 for
// 8-bit rows, 7 for 4-bit ones) and row scales.
struct QMat {
  std::vector<int8_t> q;
  std::vector<float> s;
  void make(const float* W, int64_t M, int64_t K, float qmax) {
    q.resize((size_t)(M * K));
    s.resize((size_t)M);
    quantize_rows_levels(W, M, K, qmax, q.data(), s.data());
  }
};

template <class Acc>
struct Model : ModelBase {
  orc_config c;
  const char* blob;
  Layout L;
  bool q8 = false;  // weight matrices as 8-bit or 4-bit codes (gains stay float32)
  std::vector<QMat> qWq, qWk, qWv, qWo, qW1, qW3, qW2;
  QMat qE, qWcls;
  int64_t d, F, V, H, Hkv, hd, kvd, S;
  std::vector<Acc> x, xb, q, k, v, o, a, b, hb, y, att, logit;
  Acc* kcache = nullptr;  // [L][S][kvd]
  Acc* vcache = nullptr;

  ~Model() override {
    std::free(kcache);
    std::free(vcache);
  }
  const float* T(int64_t off) const { return (const float*)(blob + off); }

  bool init() {
    d = c.dim; F = c.hidden_dim; V = c.vocab_size; H = c.n_heads; Hkv = c.n_kv_heads;
    hd = d / H; kvd = Hkv * hd; S = c.max_seq;
    x.resize(d); xb.resize(d); q.resize(d); k.resize(kvd); v.resize(kvd); o.resize(d);
    a.resize(F); b.resize(F); hb.resize(F); y.resize(d > F ? d : F); att.resize(S);
    logit.resize(V);
    // calloc: pages never written are never committed.
    const size_t n = (size_t)(c.n_layers > 0 ? c.n_layers : 1) * S * kvd;
    kcache = (Acc*)std::calloc(n, sizeof(Acc));
    vcache = (Acc*)std::calloc(n, sizeof(Acc));
    return kcache && vcache;
  }

  // Codes of every weight matrix (the embedding table too; it is also the
  // classifier when tied), qmax levels on each side of zero.
  void quantize_all(float qmax) {
    q8 = true;
    const int nl = c.n_layers;
    qWq.resize(nl); qWk.resize(nl); qWv.resize(nl); qWo.resize(nl);
    qW1.resize(nl); qW3.resize(nl); qW2.resize(nl);
    for (int l = 0; l < nl; ++l) {
      qWq[l].make(T(L.Wq[l]), d, d, qmax);
      qWk[l].make(T(L.Wk[l]), kvd, d, qmax);
      qWv[l].make(T(L.Wv[l]), kvd, d, qmax);
      qWo[l].make(T(L.Wo[l]), d, d, qmax);
      qW1[l].make(T(L.W1[l]), F, d, qmax);
      qW3[l].make(T(L.W3[l]), F, d, qmax);
      qW2[l].make(T(L.W2[l]), d, F, qmax);
    }
    qE.make(T(L.E), V, d, qmax);
    if (!tied) qWcls.make(T(L.Wcls), V, d, qmax);
  }
  void mv(const std::vector<QMat>& qm, const std::vector<int64_t>& off, int l, const Acc* xin,
          Acc* yout, int64_t M, int64_t K) {
    if (q8) gemv_q8(qm[l].q.data(), qm[l].s.data(), xin, yout, M, K);
    else gemv(T(off[l]), xin, yout, M, K);
  }

  int forward(int32_t token, int32_t pos, double* logits) override {
    if (token < 0 || token >= V || pos < 0 || pos >= S) return 6;
    const Acc eps = (Acc)c.norm_eps;
    // token embedding row (§4.1: weights are pointers at offsets in the blob)
    if (q8) {
      const int8_t* qe = qE.q.data() + (size_t)token * d;
      for (int64_t j = 0; j < d; ++j) x[j] = (Acc)qE.s[token] * (Acc)qe[j];
    } else {
      const float* e = T(L.E) + (int64_t)token * d;
      for (int64_t j = 0; j < d; ++j) x[j] = (Acc)e[j];
    }

    for (int l = 0; l < c.n_layers; ++l) {
      // attention block
      rmsnorm(x.data(), T(L.g_att[l]), xb.data(), d, eps);
      mv(qWq, L.Wq, l, xb.data(), q.data(), d, d);
      mv(qWk, L.Wk, l, xb.data(), k.data(), kvd, d);
      mv(qWv, L.Wv, l, xb.data(), v.data(), kvd, d);
      rope(q.data(), d, hd, pos, c.rope_theta);
      rope(k.data(), kvd, hd, pos, c.rope_theta);
      Acc* Kc = kcache + (size_t)l * S * kvd;
      Acc* Vc = vcache + (size_t)l * S * kvd;
      for (int64_t j = 0; j < kvd; ++j) {
        Kc[(size_t)pos * kvd + j] = k[j];
        Vc[(size_t)pos * kvd + j] = v[j];
      }
      // grouped heads: query head h reads key/value head h / (H / Hkv)
      const int64_t group = H / Hkv;
      for (int64_t h = 0; h < H; ++h) {
        const int64_t kvh = h / group;
        attention_head(q.data() + h * hd, Kc + kvh * hd, Vc + kvh * hd, (int64_t)pos + 1, hd,
                       kvd, o.data() + h * hd, att.data());
      }
      mv(qWo, L.Wo, l, o.data(), y.data(), d, d);
      for (int64_t j = 0; j < d; ++j) x[j] = x[j] + y[j];

      // feed-forward block: W2 (silu(W1 xb) * (W3 xb))
      rmsnorm(x.data(), T(L.g_ffn[l]), xb.data(), d, eps);
      mv(qW1, L.W1, l, xb.data(), a.data(), F, d);
      mv(qW3, L.W3, l, xb.data(), b.data(), F, d);
      for (int64_t i = 0; i < F; ++i) hb[i] = silu(a[i]) * b[i];
      mv(qW2, L.W2, l, hb.data(), y.data(), d, F);
      for (int64_t j = 0; j < d; ++j) x[j] = x[j] + y[j];
    }
    rmsnorm(x.data(), T(L.g_final), xb.data(), d, eps);
    // classifier; §5.1: W_cls is the embedding table when tied
    if (q8) {
      const QMat& qc = tied ? qE : qWcls;
      gemv_q8(qc.q.data(), qc.s.data(), xb.data(), logit.data(), V, d);
    } else {
      gemv(T(tied ? L.E : L.Wcls), xb.data(), logit.data(), V, d);
    }
    for (int64_t i = 0; i < V; ++i) logits[i] = (double)logit[i];
    return 0;
  }
};

}  // namespace

extern "C" {

int64_t orc_blob_bytes(const orc_config* cfg, int tied) {
  if (!config_ok(cfg)) return -1;
  return make_layout(cfg, tied != 0).total;
}

int64_t orc_tensor_offset(const orc_config* cfg, int tied, int which, int layer) {
  if (!config_ok(cfg)) return -1;
  Layout L = make_layout(cfg, tied != 0);
  if (which == 0) return L.E;
  if (which == 10) return L.g_final;
  if (which == 11) return L.Wcls;
  if (layer < 0 || layer >= cfg->n_layers) return -1;
  switch (which) {
    case 1: return L.g_att[layer];
    case 2: return L.Wq[layer];
    case 3: return L.Wk[layer];
    case 4: return L.Wv[layer];
    case 5: return L.Wo[layer];
    case 6: return L.g_ffn[layer];
    case 7: return L.W1[layer];
    case 8: return L.W3[layer];
    case 9: return L.W2[layer];
  }
  return -1;
}

void* orc_model_new(const orc_config* cfg, const void* blob, size_t blob_bytes, int acc_bits,
                    int* err) {
  return orc_model_new_fmt(cfg, blob, blob_bytes, acc_bits, 0, err);
}

void* orc_model_new_fmt(const orc_config* cfg, const void* blob, size_t blob_bytes, int acc_bits,
                        int weight_bits, int* err) {
  int dummy;
  if (!err) err = &dummy;
  *err = 0;
  if (!config_ok(cfg) || !blob || (acc_bits != 32 && acc_bits != 64) ||
      (weight_bits != 0 && weight_bits != 8 && weight_bits != 4)) {
    *err = 1;
    return nullptr;
  }
  // §5.1 weight tying: a blob one classifier short means W_cls == W_emb.
  bool tied;
  const int64_t tied_bytes = make_layout(cfg, true).total;
  const int64_t untied_bytes = make_layout(cfg, false).total;
  if (cfg->shared_classifier == 1) tied = true;
  else if (cfg->shared_classifier == 0) tied = false;
  else if (cfg->shared_classifier == -1) tied = ((int64_t)blob_bytes < untied_bytes);
  else { *err = 1; return nullptr; }
  if ((int64_t)blob_bytes != (tied ? tied_bytes : untied_bytes)) {
    *err = 2;
    return nullptr;
  }
  ModelBase* m = nullptr;
  if (acc_bits == 64) {
    auto* mm = new (std::nothrow) Model<double>();
    if (mm) { mm->c = *cfg; mm->blob = (const char*)blob; mm->L = make_layout(cfg, tied); }
    if (mm && !mm->init()) { delete mm; mm = nullptr; }
    m = mm;
  } else {
    auto* mm = new (std::nothrow) Model<float>();
    if (mm) { mm->c = *cfg; mm->blob = (const char*)blob; mm->L = make_layout(cfg, tied); }
    if (mm && !mm->init()) { delete mm; mm = nullptr; }
    m = mm;
  }
  if (!m) { *err = 4; return nullptr; }
  m->tied = tied;
  if (weight_bits != 0) {
    const float qmax = weight_bits == 8 ? 127.0f : 7.0f;
    if (acc_bits == 64) static_cast<Model<double>*>(m)->quantize_all(qmax);
    else static_cast<Model<float>*>(m)->quantize_all(qmax);
  }
  return m;
}

int orc_forward(void* model, int32_t token, int32_t pos, double* logits) {
  if (!model || !logits) return 1;
  return ((ModelBase*)model)->forward(token, pos, logits);
}

int orc_model_tied(const void* model) { return model ? (int)((const ModelBase*)model)->tied : -1; }

void orc_model_free(void* model) { delete (ModelBase*)model; }

void orc_quantize_rows_q8(const float* W, int64_t M, int64_t K, int8_t* q, float* s) {
  quantize_rows(W, M, K, q, s);
}

void orc_gemv_q8_f64(const int8_t* q, const float* s, const double* x, double* y, int64_t M,
                     int64_t K) {
  gemv_q8<double>(q, s, x, y, M, K);
}

void orc_quantize_rows_q4(const float* W, int64_t M, int64_t K, int8_t* q, float* s) {
  quantize_rows_levels(W, M, K, 7.0f, q, s);
}

void orc_gemv_f64(const float* W, const double* x, double* y, int64_t M, int64_t K) {
  gemv<double>(W, x, y, M, K);
}
void orc_gemv_f32(const float* W, const float* x, float* y, int64_t M, int64_t K) {
  gemv<float>(W, x, y, M, K);
}
void orc_rmsnorm_f64(const double* x, const float* g, double* out, int64_t n, double eps) {
  rmsnorm<double>(x, g, out, n, eps);
}
void orc_rope_f64(double* v, int64_t n, int64_t head_dim, int32_t pos, double theta) {
  rope<double>(v, n, head_dim, pos, theta);
}
void orc_softmax_f64(double* s, int64_t n) { softmax<double>(s, n); }
double orc_silu_f64(double z) { return silu<double>(z); }
void orc_attention_head_f64(const double* q, const double* K, const double* V, int64_t npos,
                            int64_t hd, int64_t stride, double* out) {
  std::vector<double> scratch((size_t)npos);
  attention_head<double>(q, K, V, npos, hd, stride, out, scratch.data());
}

}  // extern "C"
