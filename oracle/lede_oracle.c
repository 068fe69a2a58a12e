/*
 * lede_oracle.c -- TEST INFRASTRUCTURE: plain, slow fp64 CPU reference of
 * LEDE's self-speculative decoding loop ("Experience-Driven Dynamic Exits for
 * LLMs with Reinforcement Learning").  Only tests/, __graft_entry__.smoke() and
 * bench.py's cpu_baseline / reference leg may load it.
 *
 * What it computes (paper sections in brackets):
 *   - a Llama-style decoder with an early exit after any layer l, whose next
 *     token distribution P_t^(l) comes from the shared final RMSNorm and LM head
 *     (§2.2 and §3.1.1: LayerSkip-trained models exit through the model's own
 *     head; the state is computed from the hidden state at layer l);
 *   - the state features C^l_k (k = 5), H^l and C_trace (T = 20) (§3.1.1);
 *   - the Q-network MLP and its greedy action, continue = 0 / exit = 1, with a
 *     forced exit at the last candidate layer (§3.1.2, §3.2 "Target Q network");
 *   - one speculation round: the layer-wise walk over candidate exit layers,
 *     adaptive drafting at l*, one full-model verification pass over the k + 1
 *     positions, greedy prefix-match acceptance and KV-cache rollback (§3.3;
 *     greedy decoding with speculative acceptance, §4.1 Evaluation Setup);
 *   - plain autoregressive decoding (the AR baseline) and the static (E, d)
 *     policy (the LayerSkip baseline) (§4.1, Baselines).
 * Parity unpinned: the paper gives no trained Q-network weights, so the policy's
 * absolute behaviour (E, d, acceptance) is that of the seeded Q-network.
 */
#include "lede_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#include "../synth/synth.h"

typedef struct {
  float* f;
  uint16_t* b;
  int64_t n;
} tensor;

struct orc_model {
  orc_cfg c;
  tensor embed, lm_head;
  tensor *wqkv, *wo, *wgu, *wdown; /* per layer, row-major [rows][cols] */
  double *attn_norm, *ffn_norm;    /* [L][d] */
  double* final_norm;              /* [d] */
};

struct orc_sess {
  const orc_model* m;
  int max_seq;
  double* kv; /* [L][2][Hkv][max_seq][hd] */
  int kv_len; /* positions [0, kv_len) are valid */
  int x;      /* pending token (input of the next round), at position kv_len */
  int have_x;
  double* trace; /* pushed max-probabilities, oldest first, capacity trace_cap */
  int trace_n, trace_cap;
};

/* ------------------------------------------------------------------ weights */

static inline double tget(const tensor* t, int64_t i) {
  return t->b ? (double)synth_bf16_to_f32(t->b[i]) : (double)t->f[i];
}

static int talloc(tensor* t, int64_t n, int bf16) {
  t->n = n;
  t->f = NULL;
  t->b = NULL;
  if (bf16)
    t->b = (uint16_t*)calloc((size_t)n, sizeof(uint16_t));
  else
    t->f = (float*)calloc((size_t)n, sizeof(float));
  return (t->b || t->f) ? 0 : -1;
}

static void tfree(tensor* t) {
  free(t->f);
  free(t->b);
  t->f = NULL;
  t->b = NULL;
}

static void tfill(tensor* t, uint32_t seed, uint32_t tid, double sigma) {
  int64_t n = t->n;
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    float v = synth_weight_f32(seed, tid, (uint64_t)i, sigma);
    if (t->b)
      t->b[i] = synth_f32_to_bf16(v);
    else
      t->f[i] = v;
  }
}

static int64_t qkv_rows(const orc_cfg* c) {
  return (int64_t)(c->n_heads + 2 * c->n_kv_heads) * c->head_dim;
}

orc_model* orc_model_create(const orc_cfg* cfg) {
  const orc_cfg* c = cfg;
  if (c->n_layers < 1 || c->d_model < 1 || c->n_heads < 1 || c->n_kv_heads < 1 ||
      c->head_dim < 2 || (c->head_dim % 2) || c->n_heads % c->n_kv_heads || c->ffn_dim < 1 ||
      c->vocab < 2)
    return NULL;
  orc_model* m = (orc_model*)calloc(1, sizeof(orc_model));
  if (!m) return NULL;
  m->c = *c;
  int L = c->n_layers, d = c->d_model, bf = c->bf16 != 0;
  int64_t qd = (int64_t)c->n_heads * c->head_dim;
  int err = 0;
  m->wqkv = (tensor*)calloc(L, sizeof(tensor));
  m->wo = (tensor*)calloc(L, sizeof(tensor));
  m->wgu = (tensor*)calloc(L, sizeof(tensor));
  m->wdown = (tensor*)calloc(L, sizeof(tensor));
  m->attn_norm = (double*)malloc(sizeof(double) * L * d);
  m->ffn_norm = (double*)malloc(sizeof(double) * L * d);
  m->final_norm = (double*)malloc(sizeof(double) * d);
  if (!m->wqkv || !m->wo || !m->wgu || !m->wdown || !m->attn_norm || !m->ffn_norm || !m->final_norm) {
    orc_model_free(m);
    return NULL;
  }
  err |= talloc(&m->embed, (int64_t)c->vocab * d, bf);
  err |= talloc(&m->lm_head, (int64_t)c->vocab * d, bf);
  for (int l = 0; l < L; ++l) {
    err |= talloc(&m->wqkv[l], qkv_rows(c) * d, bf);
    err |= talloc(&m->wo[l], (int64_t)d * qd, bf);
    err |= talloc(&m->wgu[l], 2 * (int64_t)c->ffn_dim * d, bf);
    err |= talloc(&m->wdown[l], (int64_t)d * c->ffn_dim, bf);
  }
  if (err) {
    orc_model_free(m);
    return NULL;
  }
  for (int64_t i = 0; i < (int64_t)L * d; ++i) m->attn_norm[i] = m->ffn_norm[i] = 1.0;
  for (int i = 0; i < d; ++i) m->final_norm[i] = 1.0;
  if (c->synth) {
    tfill(&m->embed, c->seed, SYNTH_TID_EMBED, c->sigma);
    tfill(&m->lm_head, c->seed, SYNTH_TID_LMHEAD, c->sigma);
    for (int l = 0; l < L; ++l) {
      double late = (l >= L / 2) ? c->late_scale : 1.0;
      tfill(&m->wqkv[l], c->seed, synth_layer_tid(l, SYNTH_LT_WQKV), c->sigma);
      tfill(&m->wo[l], c->seed, synth_layer_tid(l, SYNTH_LT_WO), c->sigma * late);
      tfill(&m->wgu[l], c->seed, synth_layer_tid(l, SYNTH_LT_WGU), c->sigma);
      tfill(&m->wdown[l], c->seed, synth_layer_tid(l, SYNTH_LT_WDOWN), c->sigma * late);
    }
  }
  return m;
}

void orc_model_free(orc_model* m) {
  if (!m) return;
  tfree(&m->embed);
  tfree(&m->lm_head);
  for (int l = 0; l < m->c.n_layers; ++l) {
    if (m->wqkv) tfree(&m->wqkv[l]);
    if (m->wo) tfree(&m->wo[l]);
    if (m->wgu) tfree(&m->wgu[l]);
    if (m->wdown) tfree(&m->wdown[l]);
  }
  free(m->wqkv);
  free(m->wo);
  free(m->wgu);
  free(m->wdown);
  free(m->attn_norm);
  free(m->ffn_norm);
  free(m->final_norm);
  free(m);
}

static tensor* pick(const orc_model* m, int which, int layer) {
  int L = m->c.n_layers;
  if ((which >= ORC_T_WQKV) && (layer < 0 || layer >= L)) return NULL;
  switch (which) {
    case ORC_T_EMBED: return (tensor*)&m->embed;
    case ORC_T_LMHEAD: return (tensor*)&m->lm_head;
    case ORC_T_WQKV: return &m->wqkv[layer];
    case ORC_T_WO: return &m->wo[layer];
    case ORC_T_WGU: return &m->wgu[layer];
    case ORC_T_WDOWN: return &m->wdown[layer];
    default: return NULL;
  }
}

static double* pick_norm(const orc_model* m, int which, int layer) {
  int L = m->c.n_layers, d = m->c.d_model;
  if (which == ORC_T_FINAL_NORM) return m->final_norm;
  if (layer < 0 || layer >= L) return NULL;
  if (which == ORC_T_ATTN_NORM) return m->attn_norm + (int64_t)layer * d;
  if (which == ORC_T_FFN_NORM) return m->ffn_norm + (int64_t)layer * d;
  return NULL;
}

/* Overwrite one tensor (values are stored in the model's storage type; bf16
 * storage rounds to nearest even). */
int orc_model_set(orc_model* m, int which, int layer, const double* data, int64_t n) {
  double* nv = (which >= ORC_T_FINAL_NORM && which <= ORC_T_FFN_NORM) ? pick_norm(m, which, layer) : NULL;
  if (nv) {
    if (n != m->c.d_model) return ORC_ERR_ARG;
    memcpy(nv, data, sizeof(double) * n);
    return ORC_OK;
  }
  tensor* t = pick(m, which, layer);
  if (!t || n != t->n) return ORC_ERR_ARG;
  for (int64_t i = 0; i < n; ++i) {
    if (t->b)
      t->b[i] = synth_f32_to_bf16((float)data[i]);
    else
      t->f[i] = (float)data[i];
  }
  return ORC_OK;
}

double orc_model_get(const orc_model* m, int which, int layer, int64_t idx) {
  double* nv = (which >= ORC_T_FINAL_NORM && which <= ORC_T_FFN_NORM) ? pick_norm(m, which, layer) : NULL;
  if (nv) return (idx >= 0 && idx < m->c.d_model) ? nv[idx] : NAN;
  tensor* t = pick(m, which, layer);
  if (!t || idx < 0 || idx >= t->n) return NAN;
  return tget(t, idx);
}

/* ------------------------------------------------------------ session / KV */

orc_sess* orc_sess_create(const orc_model* m, int max_seq) {
  if (!m || max_seq < 1) return NULL;
  orc_sess* s = (orc_sess*)calloc(1, sizeof(orc_sess));
  if (!s) return NULL;
  const orc_cfg* c = &m->c;
  s->m = m;
  s->max_seq = max_seq;
  size_t n = (size_t)c->n_layers * 2 * c->n_kv_heads * (size_t)max_seq * c->head_dim;
  s->kv = (double*)calloc(n, sizeof(double));
  s->trace_cap = 4096;
  s->trace = (double*)calloc((size_t)s->trace_cap, sizeof(double));
  if (!s->kv || !s->trace) {
    orc_sess_free(s);
    return NULL;
  }
  return s;
}

void orc_sess_free(orc_sess* s) {
  if (!s) return;
  free(s->kv);
  free(s->trace);
  free(s);
}

int orc_sess_kv_len(const orc_sess* s) { return s->kv_len; }
int orc_sess_x(const orc_sess* s) { return s->have_x ? s->x : -1; }

static inline double* kv_row(const orc_sess* s, int layer, int kv, int head, int pos) {
  const orc_cfg* c = &s->m->c;
  size_t idx = ((((size_t)layer * 2 + kv) * c->n_kv_heads + head) * (size_t)s->max_seq + pos) *
               (size_t)c->head_dim;
  return s->kv + idx;
}

double orc_sess_kv(const orc_sess* s, int layer, int kv, int head, int pos, int i) {
  return kv_row(s, layer, kv, head, pos)[i];
}

/* ----------------------------------------------------------- decoder blocks */

/* y[r] = sum_k W[row0 + r][k] * x[k], r < nrows; k ascending. */
static void matvec(const tensor* W, int64_t row0, int64_t nrows, int64_t K, const double* x,
                   double* y) {
#pragma omp parallel for schedule(static) if (nrows * K > 65536)
  for (int64_t r = 0; r < nrows; ++r) {
    int64_t base = (row0 + r) * K;
    double acc = 0.0;
    for (int64_t k = 0; k < K; ++k) acc += tget(W, base + k) * x[k];
    y[r] = acc;
  }
}

/* y = W x for one of the model's matrices (which = ORC_T_*, layer for the
 * per-layer ones); x has the matrix's column count. */
int orc_matvec(const orc_model* m, int which, int layer, const double* x, double* y) {
  const orc_cfg* c = &m->c;
  tensor* t = pick(m, which, layer);
  if (!t) return ORC_ERR_ARG;
  int64_t qd = (int64_t)c->n_heads * c->head_dim;
  int64_t rows, cols;
  switch (which) {
    case ORC_T_EMBED:
    case ORC_T_LMHEAD: rows = c->vocab; cols = c->d_model; break;
    case ORC_T_WQKV: rows = qkv_rows(c); cols = c->d_model; break;
    case ORC_T_WO: rows = c->d_model; cols = qd; break;
    case ORC_T_WGU: rows = 2 * (int64_t)c->ffn_dim; cols = c->d_model; break;
    default: rows = c->d_model; cols = c->ffn_dim; break;
  }
  matvec(t, 0, rows, cols, x, y);
  return ORC_OK;
}

/* y[r] = sum_k W[row0 + r][k] x[k] for rows of a synthetic matrix whose
 * element (i, k) is the generator's value for flat index i*K + k (bf16-rounded
 * when bf16); lets full-size matrices be checked on sampled rows without
 * materialising them. */
int orc_matvec_synth(uint32_t seed, uint32_t tid, double sigma, int bf16, int64_t row0,
                     int64_t nrows, int64_t K, const double* x, double* y) {
#pragma omp parallel for schedule(static)
  for (int64_t r = 0; r < nrows; ++r) {
    double acc = 0.0;
    for (int64_t k = 0; k < K; ++k) {
      float w = synth_weight_f32(seed, tid, (uint64_t)((row0 + r) * K + k), sigma);
      if (bf16) w = synth_bf16_to_f32(synth_f32_to_bf16(w));
      acc += (double)w * x[k];
    }
    y[r] = acc;
  }
  return ORC_OK;
}

/* RMSNorm: out = x / sqrt(mean(x^2) + eps) * g. */
static void rmsnorm(const double* x, const double* g, int d, double eps, double* out) {
  double ss = 0.0;
  for (int i = 0; i < d; ++i) ss += x[i] * x[i];
  double r = 1.0 / sqrt(ss / d + eps);
  for (int i = 0; i < d; ++i) out[i] = x[i] * r * g[i];
}

/* Rotary embedding of one head vector at position pos, pairing element i with
 * element i + hd/2 (the "rotate half" layout of Llama checkpoints):
 * (a, b) -> (a cos t - b sin t, b cos t + a sin t), t = pos * theta^(-2i/hd). */
static void rope(double* v, int hd, int pos, double theta) {
  int half = hd / 2;
  for (int i = 0; i < half; ++i) {
    double inv_freq = 1.0 / pow(theta, (2.0 * i) / hd);
    double t = (double)pos * inv_freq;
    double cs = cos(t), sn = sin(t);
    double a = v[i], b = v[i + half];
    v[i] = a * cs - b * sn;
    v[i + half] = b * cs + a * sn;
  }
}

static double silu(double g) { return g / (1.0 + exp(-g)); }

/* One decoder block for one row at position pos: pre-norm attention with GQA
 * (query head h reads KV head h / (n_heads / n_kv_heads)), causal over
 * positions [0, pos], then pre-norm SwiGLU FFN; both with residual adds. */
static void block_row(orc_sess* s, int l, int pos, double* h, double* buf) {
  const orc_model* m = s->m;
  const orc_cfg* c = &m->c;
  int d = c->d_model, hd = c->head_dim, Hq = c->n_heads, Hkv = c->n_kv_heads, F = c->ffn_dim;
  int64_t qd = (int64_t)Hq * hd, kvd = (int64_t)Hkv * hd;
  double* xn = buf;               /* d */
  double* qkv = xn + d;           /* qd + 2 kvd */
  double* att = qkv + qd + 2 * kvd; /* qd */
  double* y = att + qd;           /* max(d, 2F) */
  double* act = y + (d > 2 * F ? d : 2 * F); /* F */
  double* sc = act + F;           /* pos + 1 */

  rmsnorm(h, m->attn_norm + (int64_t)l * d, d, c->rms_eps, xn);
  matvec(&m->wqkv[l], 0, qd + 2 * kvd, d, xn, qkv);
  double* q = qkv;
  double* k = qkv + qd;
  double* v = k + kvd;
  for (int hh = 0; hh < Hq; ++hh) rope(q + (int64_t)hh * hd, hd, pos, c->rope_theta);
  for (int hh = 0; hh < Hkv; ++hh) rope(k + (int64_t)hh * hd, hd, pos, c->rope_theta);
  for (int hh = 0; hh < Hkv; ++hh) {
    memcpy(kv_row(s, l, 0, hh, pos), k + (int64_t)hh * hd, sizeof(double) * hd);
    memcpy(kv_row(s, l, 1, hh, pos), v + (int64_t)hh * hd, sizeof(double) * hd);
  }
  int group = Hq / Hkv;
  double scale = 1.0 / sqrt((double)hd);
  /* heads are independent: long contexts spread them over threads, each
   * with its own score row (the per-head arithmetic is the same either way) */
  int par = (int64_t)Hq * (pos + 1) * hd > (1 << 20);
#pragma omp parallel if (par)
  {
    double* scr = par ? (double*)malloc(sizeof(double) * (size_t)(pos + 1)) : sc;
#pragma omp for schedule(static)
    for (int hh = 0; hh < Hq; ++hh) {
      if (!scr) continue; /* out of memory: the caller sees NaN outputs */
      int g = hh / group;
      const double* qh = q + (int64_t)hh * hd;
      double mx = -INFINITY;
      for (int t = 0; t <= pos; ++t) {
        const double* kt = kv_row(s, l, 0, g, t);
        double dot = 0.0;
        for (int i = 0; i < hd; ++i) dot += qh[i] * kt[i];
        scr[t] = dot * scale;
        if (scr[t] > mx) mx = scr[t];
      }
      double sum = 0.0;
      for (int t = 0; t <= pos; ++t) {
        scr[t] = exp(scr[t] - mx);
        sum += scr[t];
      }
      double* o = att + (int64_t)hh * hd;
      for (int i = 0; i < hd; ++i) o[i] = 0.0;
      for (int t = 0; t <= pos; ++t) {
        const double* vt = kv_row(s, l, 1, g, t);
        double p = scr[t] / sum;
        for (int i = 0; i < hd; ++i) o[i] += p * vt[i];
      }
    }
    if (par) free(scr);
  }
  matvec(&m->wo[l], 0, d, qd, att, y);
  for (int i = 0; i < d; ++i) h[i] += y[i];

  rmsnorm(h, m->ffn_norm + (int64_t)l * d, d, c->rms_eps, xn);
  matvec(&m->wgu[l], 0, 2 * (int64_t)F, d, xn, y); /* rows [0,F) gate, [F,2F) up */
  for (int i = 0; i < F; ++i) act[i] = silu(y[i]) * y[F + i];
  matvec(&m->wdown[l], 0, d, F, act, y);
  for (int i = 0; i < d; ++i) h[i] += y[i];
}

static size_t block_buf_len(const orc_cfg* c, int max_seq) {
  int64_t qd = (int64_t)c->n_heads * c->head_dim, kvd = (int64_t)c->n_kv_heads * c->head_dim;
  int64_t ymax = c->d_model > 2 * c->ffn_dim ? c->d_model : 2 * c->ffn_dim;
  return (size_t)(c->d_model + qd + 2 * kvd + qd + ymax + c->ffn_dim + max_seq + 1);
}

/* Runs layers [l_from, l_to) (0-indexed) on M rows at positions pos0 + m,
 * writing their KV.  h is [M][d]: with l_from == 0 it is set to the token
 * embeddings, otherwise it holds the hidden states after layer l_from. */
int orc_forward(orc_sess* s, const int32_t* tok, int M, int pos0, int l_from, int l_to, double* h) {
  const orc_cfg* c = &s->m->c;
  int d = c->d_model;
  if (M < 1 || pos0 < 0 || l_from < 0 || l_to > c->n_layers || l_from > l_to) return ORC_ERR_ARG;
  if (pos0 + M > s->max_seq) return ORC_ERR_CAPACITY;
  if (l_from == 0) {
    for (int mm = 0; mm < M; ++mm) {
      if (tok[mm] < 0 || tok[mm] >= c->vocab) return ORC_ERR_ARG;
      for (int i = 0; i < d; ++i) h[(int64_t)mm * d + i] = tget(&s->m->embed, (int64_t)tok[mm] * d + i);
    }
  }
  double* buf = (double*)malloc(sizeof(double) * block_buf_len(c, s->max_seq));
  if (!buf) return ORC_ERR_NOMEM;
  for (int l = l_from; l < l_to; ++l)
    for (int mm = 0; mm < M; ++mm) block_row(s, l, pos0 + mm, h + (int64_t)mm * d, buf);
  free(buf);
  return ORC_OK;
}

/* ------------------------------------------------------------- exit head */

/* Early-exit prediction: z = W_lm * RMSNorm_final(h) (shared head). */
int orc_logits(const orc_model* m, const double* h, double* z) {
  const orc_cfg* c = &m->c;
  double* xn = (double*)malloc(sizeof(double) * c->d_model);
  if (!xn) return ORC_ERR_NOMEM;
  rmsnorm(h, m->final_norm, c->d_model, c->rms_eps, xn);
  matvec(&m->lm_head, 0, c->vocab, c->d_model, xn, z);
  free(xn);
  return ORC_OK;
}

/* Statistics of P = softmax(z) (§3.1.1):
 *   C_k = -(1/k) sum_{j<=k} log P(j) over the k most probable tokens,
 *   H   = -sum_v P(v) log P(v),
 *   pmax = max_v P(v) (the per-step term of C_trace),
 * plus the greedy token (argmax, lowest id on ties) and the top-1/top-2 logit
 * margin that decides whether two implementations must agree on it. */
void orc_stats_from_logits(const double* z, int V, int topk, orc_stats* st) {
  memset(st, 0, sizeof(*st));
  if (topk < 1) topk = 1;
  if (topk > ORC_TOPK_MAX) topk = ORC_TOPK_MAX;
  if (topk > V) topk = V;
  st->topk = topk;
  /* top-k by repeated selection: largest value, then lowest index */
  for (int j = 0; j < topk; ++j) {
    int best = -1;
    for (int v = 0; v < V; ++v) {
      int taken = 0;
      for (int q = 0; q < j; ++q) taken |= (st->top_idx[q] == v);
      if (taken) continue;
      if (best < 0 || z[v] > z[best]) best = v;
    }
    st->top_idx[j] = best;
    st->top_logit[j] = z[best];
  }
  st->argmax = st->top_idx[0];
  st->zmax = st->top_logit[0];
  double sum = 0.0;
  for (int v = 0; v < V; ++v) sum += exp(z[v] - st->zmax);
  st->lse = st->zmax + log(sum);
  double H = 0.0;
  for (int v = 0; v < V; ++v) {
    double lp = z[v] - st->lse;
    H -= exp(lp) * lp;
  }
  st->entropy = H;
  double ck = 0.0;
  for (int j = 0; j < topk; ++j) ck += st->top_logit[j] - st->lse;
  st->conf_k = -ck / topk;
  st->pmax = exp(st->zmax - st->lse);
  if (V >= 2) {
    int second = -1;
    for (int v = 0; v < V; ++v) {
      if (v == st->argmax) continue;
      if (second < 0 || z[v] > z[second]) second = v;
    }
    st->margin = st->zmax - z[second];
  }
}

int orc_exit_head(const orc_model* m, const double* h, double* z_opt, int topk, orc_stats* st) {
  int V = m->c.vocab;
  double* z = z_opt ? z_opt : (double*)malloc(sizeof(double) * V);
  if (!z) return ORC_ERR_NOMEM;
  int rc = orc_logits(m, h, z);
  if (rc == ORC_OK) orc_stats_from_logits(z, V, topk, st);
  if (!z_opt) free(z);
  return rc;
}

/* ------------------------------------------------------------ policy / Q */

/* Q-network (§3.2 "Target Q network"): a small MLP,
 * Q = W2 relu(W1 s + b1) + b2, outputs (Q_continue, Q_exit). */
void orc_qnet(const float* P, int in, int hidden, const double* s, double q[2]) {
  const float* W1 = P;
  const float* b1 = W1 + (int64_t)hidden * in;
  const float* W2 = b1 + hidden;
  const float* b2 = W2 + 2 * (int64_t)hidden;
  double a[2] = {b2[0], b2[1]};
  for (int j = 0; j < hidden; ++j) {
    double z = b1[j];
    for (int i = 0; i < in; ++i) z += (double)W1[(int64_t)j * in + i] * s[i];
    double r = z > 0.0 ? z : 0.0;
    a[0] += (double)W2[j] * r;
    a[1] += (double)W2[hidden + j] * r;
  }
  q[0] = a[0];
  q[1] = a[1];
}

void orc_trace_push(orc_sess* s, double pmax) {
  if (s->trace_n == s->trace_cap) {
    memmove(s->trace, s->trace + s->trace_cap / 2, sizeof(double) * (s->trace_cap / 2));
    s->trace_n = s->trace_cap / 2;
  }
  s->trace[s->trace_n++] = pmax;
}

/* C_trace (§3.1.1): -(1/T) sum_{k=1..T} log pmax_{t-k}, the full model's
 * max-probability at the T most recent input positions; with fewer than T
 * positions so far, the mean over the ones there are (0 with none). */
double orc_trace_conf(const orc_sess* s, int T) {
  int n = s->trace_n < T ? s->trace_n : T;
  if (n <= 0) return 0.0;
  double acc = 0.0;
  for (int i = s->trace_n - n; i < s->trace_n; ++i) acc += log(s->trace[i]);
  return -acc / n;
}

/* Greedy action of the Q-network; ties choose continue (= 0).  The state is
 * the paper's (C_k, H, C_trace) (§3.1.1) when the network has 3 inputs, or,
 * with d_model + 1 inputs, the pooled state: the mean over this round's rows
 * so far (pool_n of them, summed in pool) of the exit hidden state after the
 * final RMSNorm, followed by the exit distribution's max-probability.
 * Records the decision in the round log (pooled state logged as (pmax,
 * rows pooled, Euclidean norm of the mean)). */
static int q_decide(orc_sess* s, const orc_policy* P, const orc_stats* st, const double* pool,
                    int pool_n, orc_round_log* lg) {
  const int d = s->m->c.d_model;
  double q[2], logged[3];
  if (P->q_in == 3) {
    double sv[3] = {st->conf_k, st->entropy, orc_trace_conf(s, P->trace_T)};
    orc_qnet(P->q_params, 3, P->q_hidden, sv, q);
    for (int j = 0; j < 3; ++j) logged[j] = sv[j];
  } else {
    double* sv = (double*)malloc(sizeof(double) * (size_t)(d + 1));
    if (!sv) return -1;
    double nrm = 0.0;
    for (int i = 0; i < d; ++i) {
      sv[i] = pool[i] / pool_n;
      nrm += sv[i] * sv[i];
    }
    sv[d] = st->pmax;
    orc_qnet(P->q_params, d + 1, P->q_hidden, sv, q);
    free(sv);
    logged[0] = st->pmax;
    logged[1] = pool_n;
    logged[2] = sqrt(nrm);
  }
  int a = q[1] > q[0] ? 1 : 0;
  if (lg->n_q < ORC_MAX_Q) {
    int i = lg->n_q++;
    lg->q_action[i] = a;
    lg->q_val[i][0] = q[0];
    lg->q_val[i][1] = q[1];
    for (int j = 0; j < 3; ++j) lg->q_state[i][j] = logged[j];
  }
  return a;
}

/* Draft & Verify-style rule (a §4.1 baseline): drafting goes on after a
 * draft whose max-probability is at least the threshold.  Logged like a Q
 * decision with values (threshold, pmax), so its margin is |pmax - tau|. */
static int threshold_decide(const orc_policy* P, const orc_stats* st, orc_round_log* lg) {
  int a = st->pmax >= P->conf_threshold ? 1 : 0;
  if (lg->n_q < ORC_MAX_Q) {
    int i = lg->n_q++;
    lg->q_action[i] = a;
    lg->q_val[i][0] = P->conf_threshold;
    lg->q_val[i][1] = st->pmax;
    lg->q_state[i][0] = st->conf_k;
    lg->q_state[i][1] = st->entropy;
    lg->q_state[i][2] = 0.0;
  }
  return a;
}

/* ------------------------------------------------------ sampled decoding */

/* Tempered distribution of logits z at temperature T > 0:
 * P(v) = exp((z_v - max z) / T) / sum_w exp((z_w - max z) / T). */
void orc_tempered(const double* z, int V, double temperature, double* p) {
  double zmax = z[0];
  for (int v = 1; v < V; ++v)
    if (z[v] > zmax) zmax = z[v];
  double S = 0.0;
  for (int v = 0; v < V; ++v) {
    p[v] = exp((z[v] - zmax) / temperature);
    S += p[v];
  }
  for (int v = 0; v < V; ++v) p[v] /= S;
}

/* Inverse-CDF draw from non-negative weights w (normalised or not): with
 * W = sum_v w_v and C_v = w_0 + ... + w_v in token order, the token is the
 * first v with C_v > u W.  *margin = min(u W - C_{v-1}, C_v - u W) / W, the
 * distance of u W to the nearer end of the token's interval, relative to W.
 * Returns -1 when W is not positive; when rounding leaves u W at or beyond
 * the accumulated sum, the last token of positive weight (margin 0). */
int orc_draw(const double* w, int V, double u, double* margin) {
  double W = 0.0;
  for (int v = 0; v < V; ++v) W += w[v];
  *margin = 0.0;
  if (!(W > 0.0)) return -1;
  const double T = u * W;
  double c = 0.0;
  int last = -1;
  for (int v = 0; v < V; ++v) {
    const double nx = c + w[v];
    if (w[v] > 0.0) last = v;
    if (nx > T) {
      *margin = fmin(T - c, nx - T) / W;
      return v;
    }
    c = nx;
  }
  return last;
}

/* One acceptance test of speculative sampling (the acceptance rule of §4.1):
 * draft d, drawn from the draft distribution q, is kept when r q(d) < p(d),
 * i.e. with probability min(1, p(d) / q(d)); otherwise the emitted token is
 * drawn with u from the residual max(0, p - q), normalised (from p itself
 * should the residual carry no mass).  Either way the emitted token follows
 * p.  res (V doubles) is scratch.  *accept_margin = (p(d) - r q(d)) /
 * max(p(d), r q(d)), positive exactly when d is kept. */
int orc_spec_step(const double* p, const double* q, int V, int d, double r, double u,
                  double* res, int* accepted, double* accept_margin, double* draw_margin) {
  const double pd = p[d], rq = r * q[d];
  const double den = fmax(pd, rq);
  *accept_margin = den > 0.0 ? (pd - rq) / den : 0.0;
  *draw_margin = 0.0;
  if (rq < pd) {
    *accepted = 1;
    return d;
  }
  *accepted = 0;
  for (int v = 0; v < V; ++v) res[v] = fmax(p[v] - q[v], 0.0);
  int t = orc_draw(res, V, u, draw_margin);
  if (t < 0) t = orc_draw(p, V, u, draw_margin);
  return t;
}

static double uniform_of(uint32_t seed, int pos, int purpose, int i) {
  return (double)synth_sample_uniform(seed, (uint32_t)pos, (uint32_t)purpose, (uint32_t)i);
}

/* ------------------------------------------------------------ generation */

static int check_policy(const orc_model* m, const orc_policy* P) {
  int L = m->c.n_layers;
  if (P->kind == ORC_POLICY_AR) return ORC_OK;
  if (P->kmax < 1 || P->kmax > ORC_MAX_K - 1) return ORC_ERR_ARG;
  if (P->kind == ORC_POLICY_STATIC) {
    if (P->static_l < 1 || P->static_l > L || P->static_k < 1) return ORC_ERR_ARG;
    return ORC_OK;
  }
  if (P->kind == ORC_POLICY_THRESHOLD) {
    if (P->static_l < 1 || P->static_l > L) return ORC_ERR_ARG;
    if (!(P->conf_threshold > 0.0 && P->conf_threshold <= 1.0)) return ORC_ERR_ARG;
    return ORC_OK;
  }
  if (P->kind != ORC_POLICY_LEDE) return ORC_ERR_ARG;
  if (P->fixed_k < 0 || P->fixed_k > ORC_MAX_K - 1) return ORC_ERR_ARG;
  if (P->n_cand < 1 || P->n_cand > ORC_MAX_CAND || !P->q_params ||
      (P->q_in != 3 && P->q_in != m->c.d_model + 1) || P->q_hidden < 1 || P->trace_T < 1)
    return ORC_ERR_ARG;
  for (int j = 0; j < P->n_cand; ++j) {
    if (P->cand[j] < 1 || P->cand[j] > L) return ORC_ERR_ARG;
    if (j && P->cand[j] <= P->cand[j - 1]) return ORC_ERR_ARG;
  }
  return ORC_OK;
}

/* Full-model rows [0, n) of ids at positions 0..n-1; the max-probabilities of
 * the last min(T, n) rows seed the trace. */
static int run_prompt(orc_sess* s, const int32_t* ids, int n, int trace_T, int32_t* last_argmax,
                      double* z_last) {
  const orc_cfg* c = &s->m->c;
  int d = c->d_model;
  double* h = (double*)malloc(sizeof(double) * (size_t)n * d);
  if (!h) return ORC_ERR_NOMEM;
  int rc = orc_forward(s, ids, n, 0, 0, c->n_layers, h);
  s->trace_n = 0;
  int first = n - trace_T > 0 ? n - trace_T : 0;
  for (int r = first; rc == ORC_OK && r < n; ++r) {
    orc_stats st;
    rc = orc_exit_head(s->m, h + (int64_t)r * d, r == n - 1 ? z_last : NULL, 1, &st);
    orc_trace_push(s, st.pmax);
    if (r == n - 1 && last_argmax) *last_argmax = st.argmax;
  }
  free(h);
  return rc;
}

/* Prompt prefill: KV for ids[0..n), trace seeded; the first generated token
 * (greedy, full model) becomes the pending token x at position n. */
int orc_prefill(orc_sess* s, const int32_t* ids, int n, int trace_T, int32_t* first) {
  if (n < 1 || trace_T < 1) return ORC_ERR_ARG;
  if (n + 1 > s->max_seq) return ORC_ERR_CAPACITY;
  s->kv_len = 0;
  s->have_x = 0;
  int32_t x = -1;
  int rc = run_prompt(s, ids, n, trace_T, &x, NULL);
  if (rc) return rc;
  s->kv_len = n;
  s->x = x;
  s->have_x = 1;
  if (first) *first = x;
  return ORC_OK;
}

/* Prefill whose first generated token is drawn from the full model's
 * distribution at the given temperature (> 0), with the uniform keyed by the
 * last prompt position n - 1 (purpose 2, index 0); temperature 0 is
 * orc_prefill.  *margin receives the draw's margin (orc_draw). */
int orc_prefill_sampled(orc_sess* s, const int32_t* ids, int n, int trace_T, double temperature,
                        uint32_t seed, int32_t* first, double* margin) {
  if (margin) *margin = 0.0;
  if (!(temperature > 0.0)) return orc_prefill(s, ids, n, trace_T, first);
  if (n < 1 || trace_T < 1) return ORC_ERR_ARG;
  if (n + 1 > s->max_seq) return ORC_ERR_CAPACITY;
  const int V = s->m->c.vocab;
  s->kv_len = 0;
  s->have_x = 0;
  double* z = (double*)malloc(sizeof(double) * 2 * (size_t)V);
  if (!z) return ORC_ERR_NOMEM;
  int32_t x = -1;
  int rc = run_prompt(s, ids, n, trace_T, &x, z);
  if (rc == ORC_OK) {
    double mg;
    orc_tempered(z, V, temperature, z + V);
    x = orc_draw(z + V, V, uniform_of(seed, n - 1, 2, 0), &mg);
    if (margin) *margin = mg;
    s->kv_len = n;
    s->x = x;
    s->have_x = 1;
    if (first) *first = x;
  }
  free(z);
  return rc;
}

/* Resume from a known sequence: KV for ids[0..n-1), pending token ids[n-1]. */
int orc_resume(orc_sess* s, const int32_t* ids, int n, int trace_T) {
  if (n < 2 || trace_T < 1) return ORC_ERR_ARG;
  if (ids[n - 1] < 0 || ids[n - 1] >= s->m->c.vocab) return ORC_ERR_ARG;
  if (n > s->max_seq) return ORC_ERR_CAPACITY;
  s->kv_len = 0;
  s->have_x = 0;
  int rc = run_prompt(s, ids, n - 1, trace_T, NULL, NULL);
  if (rc) return rc;
  s->kv_len = n - 1;
  s->x = ids[n - 1];
  s->have_x = 1;
  return ORC_OK;
}

/* One speculation round emitting 1..cap tokens (§3.3):
 *  1. walk: run the pending token x through the layers up to each candidate
 *     layer in turn; at each, the Q-network sees the state of P^(l) and picks
 *     continue or exit; the last candidate forces an exit.  The exit layer is
 *     l* and the first draft d_1 = argmax P^(l*).  (Static policy: one
 *     candidate, l* = E.)
 *  2. adaptive drafting: after each draft d_i, the Q-network's action on the
 *     state that produced d_i decides: exit -> draft d_{i+1} by running d_i
 *     through layers 1..l*; continue -> stop.  At most kcap = min(kmax,
 *     cap - 1) drafts.  (Static: exactly d drafts, clipped to kcap.)
 *  3. verify: the full model over [x, d_1..d_k] at positions p..p+k gives
 *     g_0..g_k (greedy).
 *  4. accept: a = the longest prefix with d_i = g_{i-1}; emit d_1..d_a, g_a.
 *  5. rollback: KV length p + a + 1, pending token g_a, and the full-model
 *     max-probabilities of rows 0..a join the trace.
 * With temperature T > 0 (speculative sampling, §4.1): d_i is drawn from the
 * exit distribution at temperature T (uniform U(p, 0, i-1)); step 4 tests
 * d_1, d_2, ... in turn with orc_spec_step against the full model's row i-1
 * at temperature T (r = U(p, 1, i-1), u = U(p, 2, 0)) and stops at the first
 * rejection, whose residual draw is the last emitted token; when all k
 * drafts are kept, the last token is drawn from row k with U(p, 2, 0).  The
 * Q-network and the trace still see the exit statistics at temperature 1. */
int orc_round(orc_sess* s, const orc_policy* P, int cap, orc_round_log* lg) {
  const orc_model* m = s->m;
  const orc_cfg* c = &m->c;
  int d = c->d_model, L = c->n_layers, V = c->vocab;
  memset(lg, 0, sizeof(*lg));
  if (!s->have_x) return ORC_ERR_STATE;
  if (cap < 1) return ORC_ERR_ARG;
  int rc = check_policy(m, P);
  if (rc) return rc;
  if (!(P->temperature >= 0.0)) return ORC_ERR_ARG;
  const int sampled = P->temperature > 0.0;
  const double Tmp = P->temperature;
  int topk = P->topk > 0 ? P->topk : 5;
  int p = s->kv_len, x = s->x;
  int kcap = 0;
  if (P->kind != ORC_POLICY_AR) {
    kcap = P->kmax < cap - 1 ? P->kmax : cap - 1;
    if (P->kind == ORC_POLICY_STATIC && P->static_k < kcap) kcap = P->static_k;
    /* the ablation without adaptive drafting drafts a fixed length (Table 3) */
    if (P->kind == ORC_POLICY_LEDE && P->fixed_k > 0 && P->fixed_k < kcap) kcap = P->fixed_k;
  }
  if (p + kcap + 1 > s->max_seq) return ORC_ERR_CAPACITY;
  lg->pos = p;
  lg->x = x;
  lg->kcap = kcap;
  lg->sampled = sampled;

  int32_t drafts[ORC_MAX_K];
  int k = 0;
  double* h = (double*)malloc(sizeof(double) * (size_t)(kcap + 1) * d);
  /* sampled decoding: exit logits, draft distributions q_1..q_kcap, the
   * verify rows' distributions and a residual row */
  double* z = NULL;
  double* q = NULL;
  double* pv = NULL;
  double* res = NULL;
  /* pooled Q-network state: sum of the round's final-normed exit states */
  const int pooled = P->kind == ORC_POLICY_LEDE && P->q_in == d + 1;
  double* pool = NULL;
  double* hn = NULL;
  int pool_n = 0;
  if (pooled) {
    pool = (double*)malloc(sizeof(double) * (size_t)d);
    hn = (double*)malloc(sizeof(double) * (size_t)d);
    if (!pool || !hn) {
      free(pool);
      free(hn);
      free(h);
      return ORC_ERR_NOMEM;
    }
  }
  if (sampled) {
    z = (double*)malloc(sizeof(double) * (size_t)V);
    q = (double*)malloc(sizeof(double) * (size_t)(kcap > 0 ? kcap : 1) * V);
    pv = (double*)malloc(sizeof(double) * (size_t)(kcap + 1) * V);
    res = (double*)malloc(sizeof(double) * (size_t)V);
  }
  if (!h || (sampled && (!z || !q || !pv || !res))) {
    rc = ORC_ERR_NOMEM;
    goto out;
  }
  if (kcap > 0) {
    int n_c = P->kind == ORC_POLICY_LEDE ? P->n_cand : 1;
    int done = 0, lstar = 0, keep = 0;
    orc_stats st;
    for (int j = 0; j < n_c; ++j) {
      int cj = P->kind == ORC_POLICY_LEDE ? P->cand[j] : P->static_l;
      rc = orc_forward(s, &x, 1, p, done, cj, h);
      if (rc) goto out;
      done = cj;
      rc = orc_exit_head(m, h, z, topk, &st);
      if (rc) goto out;
      lg->visited[lg->n_visited++] = cj;
      if (pooled) {  /* this round's rows at layer cj: the pending token only */
        rmsnorm(h, m->final_norm, d, c->rms_eps, pool);
        pool_n = 1;
      }
      int act, aq = 1;
      if (P->kind == ORC_POLICY_LEDE) aq = q_decide(s, P, &st, pool, pool_n, lg);
      if (aq < 0) {
        rc = ORC_ERR_NOMEM;
        goto out;
      }
      act = (j == n_c - 1) ? 1 : aq;
      if (act) {
        lstar = cj;
        /* whether d_1 is followed by more drafts */
        if (P->kind == ORC_POLICY_THRESHOLD)
          keep = threshold_decide(P, &st, lg);
        else if (P->kind == ORC_POLICY_LEDE && P->fixed_k > 0)
          keep = 1;
        else
          keep = aq;
        break;
      }
    }
    lg->lstar = lstar;
    if (sampled) {
      orc_tempered(z, V, Tmp, q);
      drafts[0] = orc_draw(q, V, uniform_of(P->sample_seed, p, 0, 0), &lg->draft_margin[0]);
    } else {
      drafts[0] = st.argmax;
      lg->draft_margin[0] = st.margin;
    }
    k = 1;
    while (k < kcap && keep) {
      rc = orc_forward(s, &drafts[k - 1], 1, p + k, 0, lstar, h);
      if (rc) goto out;
      rc = orc_exit_head(m, h, z, topk, &st);
      if (rc) goto out;
      if (pooled) {  /* add draft row k's final-normed state at l* */
        rmsnorm(h, m->final_norm, d, c->rms_eps, hn);
        for (int i = 0; i < d; ++i) pool[i] += hn[i];
        ++pool_n;
      }
      if (sampled) {
        orc_tempered(z, V, Tmp, q + (int64_t)k * V);
        drafts[k] = orc_draw(q + (int64_t)k * V, V, uniform_of(P->sample_seed, p, 0, k),
                             &lg->draft_margin[k]);
      } else {
        drafts[k] = st.argmax;
        lg->draft_margin[k] = st.margin;
      }
      ++k;
      if (P->kind == ORC_POLICY_THRESHOLD)
        keep = threshold_decide(P, &st, lg);
      else if (P->kind == ORC_POLICY_LEDE && P->fixed_k == 0)
        keep = q_decide(s, P, &st, pool, pool_n, lg);
      else
        keep = 1;
      if (keep < 0) {
        rc = ORC_ERR_NOMEM;
        goto out;
      }
      /* the "discard" reading of adaptive drafting: the continue action
       * is about the draft it was taken on, which is dropped */
      if (!keep && P->kind == ORC_POLICY_LEDE && P->fixed_k == 0 && P->discard_on_continue) --k;
    }
  }
  lg->k = k;
  for (int i = 0; i < k; ++i) lg->drafts[i] = drafts[i];

  {
    int32_t tok[ORC_MAX_K + 1];
    tok[0] = x;
    for (int i = 0; i < k; ++i) tok[i + 1] = drafts[i];
    rc = orc_forward(s, tok, k + 1, p, 0, L, h);
    if (rc) goto out;
    for (int i = 0; i <= k; ++i) {
      orc_stats st;
      rc = orc_exit_head(m, h + (int64_t)i * d, z, 1, &st);
      if (rc) goto out;
      lg->verify_tok[i] = st.argmax;
      lg->verify_margin[i] = st.margin;
      lg->verify_pmax[i] = st.pmax;
      if (sampled) orc_tempered(z, V, Tmp, pv + (int64_t)i * V);
    }
    int a = 0, last;
    if (sampled) {
      last = -1;
      while (a < k) {
        int kept;
        const int t = orc_spec_step(pv + (int64_t)a * V, q + (int64_t)a * V, V, drafts[a],
                                    uniform_of(P->sample_seed, p, 1, a),
                                    uniform_of(P->sample_seed, p, 2, 0), res, &kept,
                                    &lg->accept_margin[a], &lg->fix_margin);
        if (!kept) {
          last = t;
          break;
        }
        ++a;
      }
      if (last < 0)
        last = orc_draw(pv + (int64_t)k * V, V, uniform_of(P->sample_seed, p, 2, 0),
                        &lg->fix_margin);
    } else {
      while (a < k && drafts[a] == lg->verify_tok[a]) ++a;
      last = lg->verify_tok[a];
    }
    lg->a = a;
    for (int i = 0; i < a; ++i) lg->emitted[i] = drafts[i];
    lg->emitted[a] = last;
    lg->n_emit = a + 1;
    s->kv_len = p + a + 1;
    s->x = last;
    for (int i = 0; i <= a; ++i) orc_trace_push(s, lg->verify_pmax[i]);
  }
out:
  free(h);
  free(pool);
  free(hn);
  free(z);
  free(q);
  free(pv);
  free(res);
  return rc;
}

/* Rounds until n_new tokens have been emitted after the pending token. */
int orc_generate(orc_sess* s, const orc_policy* P, int n_new, int32_t* out, orc_round_log* logs,
                 int logs_cap, int* n_rounds) {
  int done = 0, r = 0;
  while (done < n_new) {
    orc_round_log lg;
    int rc = orc_round(s, P, n_new - done, &lg);
    if (rc) return rc;
    for (int i = 0; i < lg.n_emit; ++i) out[done + i] = lg.emitted[i];
    done += lg.n_emit;
    if (logs && r < logs_cap) logs[r] = lg;
    ++r;
  }
  if (n_rounds) *n_rounds = r;
  return ORC_OK;
}

int orc_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
