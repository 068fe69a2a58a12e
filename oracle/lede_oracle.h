/*
 * lede_oracle.h -- TEST INFRASTRUCTURE: the plain CPU reference of LEDE's
 * self-speculative decoding loop.  Only tests/, __graft_entry__.smoke() and
 * bench.py's cpu_baseline / reference leg may load it; the product path never
 * does.  It shares no code with the CUDA path except synth/synth.h (seeded
 * inputs).
 *
 * Arithmetic is fp64 throughout (weights are read exactly from their bf16 or
 * fp32 storage); every row of every matrix-vector product and every query of
 * attention is computed independently in one fixed order, so an M-row pass
 * equals M single-row passes bit for bit.
 */
#ifndef LEDE_ORACLE_H
#define LEDE_ORACLE_H

#include <stdint.h>

#define ORC_MAX_CAND 32
#define ORC_MAX_K 32
#define ORC_MAX_Q 64
#define ORC_TOPK_MAX 8

enum { ORC_OK = 0, ORC_ERR_ARG = 1, ORC_ERR_CAPACITY = 2, ORC_ERR_STATE = 3, ORC_ERR_NOMEM = 4 };
enum { ORC_POLICY_AR = 0, ORC_POLICY_STATIC = 1, ORC_POLICY_LEDE = 2, ORC_POLICY_THRESHOLD = 3 };
/* tensor selectors for orc_model_set / orc_model_get */
enum {
  ORC_T_EMBED = 0, ORC_T_LMHEAD = 1, ORC_T_FINAL_NORM = 2, ORC_T_ATTN_NORM = 3, ORC_T_FFN_NORM = 4,
  ORC_T_WQKV = 5, ORC_T_WO = 6, ORC_T_WGU = 7, ORC_T_WDOWN = 8
};

typedef struct {
  int32_t n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn_dim, vocab;
  int32_t bf16;  /* 1: matrices stored as bf16, 0: fp32 */
  double rms_eps, rope_theta;
  double sigma;      /* weight standard deviation */
  double late_scale; /* extra factor on wo and wdown of layers >= n_layers/2 */
  uint32_t seed;
  int32_t synth;     /* 1: fill weights from synth.h; 0: zero matrices, unit norms */
} orc_cfg;

typedef struct {
  int32_t argmax;                    /* lowest index among the maximal logits */
  int32_t topk;                      /* k of C_k */
  int32_t top_idx[ORC_TOPK_MAX];     /* descending logit, ties by lower index */
  double top_logit[ORC_TOPK_MAX];
  double zmax, lse;                  /* max logit, log-sum-exp */
  double entropy;                    /* H^l */
  double conf_k;                     /* C^l_k */
  double pmax;                       /* max probability */
  double margin;                     /* top-1 minus top-2 logit */
} orc_stats;

typedef struct {
  int32_t kind;                      /* ORC_POLICY_* */
  int32_t n_cand;
  int32_t cand[ORC_MAX_CAND];        /* ascending, 1..n_layers */
  int32_t kmax;
  int32_t static_l, static_k;
  int32_t q_in, q_hidden;            /* 3: state (C_k, H, C_trace); d_model + 1: pooled state */
  int32_t trace_T, topk;
  const float* q_params;             /* W1[h][in], b1[h], W2[2][h], b2[2] */
  int32_t fixed_k;                   /* LEDE: 0 adaptive drafting; > 0 fixed draft length */
  double conf_threshold;             /* THRESHOLD: drafting goes on while pmax >= this */
  double temperature;                /* 0: greedy; > 0: speculative sampling at this temperature */
  uint32_t sample_seed;              /* key of the uniforms (synth_sample_uniform) */
  int32_t discard_on_continue;       /* LEDE adaptive drafting: a continue drops its draft */
} orc_policy;

typedef struct {
  int32_t pos, x, kcap, n_visited, lstar, k, a, n_emit, n_q;
  int32_t visited[ORC_MAX_CAND];
  int32_t drafts[ORC_MAX_K];
  int32_t verify_tok[ORC_MAX_K + 1];
  int32_t emitted[ORC_MAX_K + 1];
  int32_t q_action[ORC_MAX_Q];
  double draft_margin[ORC_MAX_K];
  double verify_margin[ORC_MAX_K + 1];
  double verify_pmax[ORC_MAX_K + 1];
  double q_val[ORC_MAX_Q][2];
  double q_state[ORC_MAX_Q][3];
  int32_t sampled;                   /* 1 when the round sampled (temperature > 0) */
  double accept_margin[ORC_MAX_K];   /* (p(d) - r q(d)) / max(p(d), r q(d)); > 0 accepts */
  double fix_margin;                 /* distance of the last draw to a CDF boundary / mass */
} orc_round_log;

typedef struct orc_model orc_model;
typedef struct orc_sess orc_sess;

orc_model* orc_model_create(const orc_cfg* cfg);
void orc_model_free(orc_model* m);
int orc_model_set(orc_model* m, int which, int layer, const double* data, int64_t n);
double orc_model_get(const orc_model* m, int which, int layer, int64_t idx);

orc_sess* orc_sess_create(const orc_model* m, int max_seq);
void orc_sess_free(orc_sess* s);
int orc_sess_kv_len(const orc_sess* s);
int orc_sess_x(const orc_sess* s);
double orc_sess_kv(const orc_sess* s, int layer, int kv, int head, int pos, int i);

int orc_forward(orc_sess* s, const int32_t* tok, int M, int pos0, int l_from, int l_to, double* h);
int orc_logits(const orc_model* m, const double* h, double* z);
int orc_matvec(const orc_model* m, int which, int layer, const double* x, double* y);
int orc_matvec_synth(uint32_t seed, uint32_t tid, double sigma, int bf16, int64_t row0,
                     int64_t nrows, int64_t K, const double* x, double* y);
void orc_stats_from_logits(const double* z, int V, int topk, orc_stats* st);
int orc_exit_head(const orc_model* m, const double* h, double* z_opt, int topk, orc_stats* st);
void orc_qnet(const float* params, int in, int hidden, const double* s, double q[2]);
double orc_trace_conf(const orc_sess* s, int T);
void orc_trace_push(orc_sess* s, double pmax);
int orc_prefill(orc_sess* s, const int32_t* ids, int n, int trace_T, int32_t* first);
int orc_prefill_sampled(orc_sess* s, const int32_t* ids, int n, int trace_T, double temperature,
                        uint32_t seed, int32_t* first, double* margin);
void orc_tempered(const double* z, int V, double temperature, double* p);
int orc_draw(const double* w, int V, double u, double* margin);
int orc_spec_step(const double* p, const double* q, int V, int d, double r, double u,
                  double* res, int* accepted, double* accept_margin, double* draw_margin);
int orc_resume(orc_sess* s, const int32_t* ids, int n, int trace_T);
int orc_round(orc_sess* s, const orc_policy* P, int cap, orc_round_log* lg);
int orc_generate(orc_sess* s, const orc_policy* P, int n_new, int32_t* out, orc_round_log* logs,
                 int logs_cap, int* n_rounds);
int orc_num_threads(void);

#endif
