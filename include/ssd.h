/*
 * ssd.h -- C ABI of the GB300 self-speculative decoding engine (LEDE policy).
 *
 * One call to ssd_step() runs one speculation round of "Experience-Driven
 * Dynamic Exits for LLMs with Reinforcement Learning" on the GPU:
 *   (1) the Q-network walks the candidate exit layers during the first
 *       token's forward pass and exits at l* (§3.1.2 Action Space, §3.3);
 *   (2) the first l* layers plus the shared final RMSNorm and LM head draft
 *       tokens greedily, the Q-network deciding after each draft whether to
 *       keep drafting (§3.3, adaptive drafting);
 *   (3) the full model verifies the pending token and all k drafts in one
 *       forward pass over k + 1 positions;
 *   (4) greedy prefix-match acceptance (the greedy case of speculative
 *       acceptance, §4.1 Evaluation Setup);
 *   (5) KV-cache rollback to the accepted length.
 * The state the Q-network sees is (C_5, H, C_trace) of the exit layer's
 * next-token distribution (§3.1.1; k = 5, T = 20 by default).
 *
 * Everything between ssd_prefill/ssd_resume and the end of ssd_generate runs
 * on the device: decisions, drafts and acceptance never return to the host
 * between draft tokens (CUDA graphs with device-side conditional nodes).
 *
 * Conventions
 *  - Every call returns an ssd_status; nothing throws or exits.  On failure
 *    ssd_last_error(ctx) holds a message.
 *  - Device memory (weights, workspace) is owned by the caller and borrowed by
 *    the context until ssd_destroy; the library allocates no device memory.
 *  - Host arrays passed in are caller-owned and read during the call only.
 *  - All work is enqueued on the caller's CUDA stream given at ssd_init_model.
 *  - Layouts: row-major matrices [rows][cols] in the model dtype (fp32 or
 *    bf16), 16-byte aligned; d_model, ffn_dim and n_heads*head_dim must be
 *    multiples of 8.  Token ids are int32 in [0, vocab).
 */
#ifndef SSD_H
#define SSD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SSD_OK = 0,
  SSD_ERR_INVALID_ARG = 1, /* bad pointer, shape, policy or size; nothing enqueued */
  SSD_ERR_CUDA = 2,        /* a CUDA runtime call failed; message in ssd_last_error */
  SSD_ERR_CAPACITY = 3,    /* the KV cache (max_seq) or an output buffer is too small */
  SSD_ERR_STATE = 4,       /* call out of order, e.g. ssd_step before ssd_prefill */
  SSD_ERR_DEVICE_FLAG = 5, /* a device-side consistency check failed during the call */
  SSD_ERR_UNSUPPORTED = 6  /* shape or option this build does not handle */
} ssd_status;

typedef enum { SSD_DTYPE_F32 = 0, SSD_DTYPE_BF16 = 1 } ssd_dtype;

/* Llama-style decoder: pre-RMSNorm, rotary embedding pairing element i with
 * i + head_dim/2, grouped-query attention (query head h reads KV head
 * h / (n_heads / n_kv_heads)), SwiGLU FFN, untied embedding and LM head.
 * Early exits after any layer go through the shared final RMSNorm + LM head. */
typedef struct {
  int32_t n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn_dim, vocab;
  int32_t max_seq; /* KV-cache capacity in positions */
  float rms_eps, rope_theta;
  int32_t dtype;   /* ssd_dtype: weights, embeddings, norm weights and KV cache */
} ssd_model_cfg;

/* Device pointers in the model dtype.  Per-layer entries are HOST arrays of
 * n_layers device pointers; they are copied at ssd_init_model. */
typedef struct {
  const void* embed;              /* [vocab][d_model] */
  const void* lm_head;            /* [vocab][d_model] */
  const void* final_norm;         /* [d_model] */
  const void* const* attn_norm;   /* [d_model] */
  const void* const* wqkv;        /* [(n_heads + 2 n_kv_heads) head_dim][d_model], rows q | k | v */
  const void* const* wo;          /* [d_model][n_heads head_dim] */
  const void* const* ffn_norm;    /* [d_model] */
  const void* const* w_gate_up;   /* [2 ffn_dim][d_model], rows gate | up */
  const void* const* w_down;      /* [d_model][ffn_dim] */
} ssd_weights;

typedef enum {
  SSD_POLICY_AR = 0,
  SSD_POLICY_STATIC = 1,
  SSD_POLICY_LEDE = 2,
  SSD_POLICY_THRESHOLD = 3
} ssd_policy_kind;

/* Speculation policy (§3.3 and the baselines and ablations of §4.1, Table 3).
 *  AR:        plain decoding with the full model (one token per round; greedy,
 *             or drawn at the policy's temperature).
 *  STATIC:    fixed exit layer static_l and draft length static_k (LayerSkip).
 *  LEDE:      Q-network over candidate exit layers cand_layers[0..n_cand),
 *             ascending in 1..n_layers; forced exit at the last one; adaptive
 *             drafting.  n_cand = 1 is the ablation without dynamic exit
 *             (exit layer fixed, drafting still decided by the Q-network);
 *             fixed_k > 0 is the ablation without adaptive drafting (the walk
 *             picks l*, then exactly min(fixed_k, cap) tokens are drafted and
 *             the Q-network is not consulted after a draft).
 *  THRESHOLD: fixed exit layer static_l; after each draft, drafting goes on
 *             while that draft's max-probability is >= conf_threshold, up to
 *             kmax (a Draft & Verify-style confidence rule with a fixed
 *             threshold).
 * kmax caps the drafts per round (1..16).  qnet_params (host fp32, copied) packs
 * W1[qnet_hidden][qnet_in], b1[qnet_hidden], W2[2][qnet_hidden], b2[2]; output
 * 0 is Q(continue), output 1 is Q(exit); ties pick continue.  The state is
 * the paper's s = (C_k, H, C_trace) of the exit distribution (§3.1.1) when
 * qnet_in = 3; with qnet_in = d_model + 1 it is the pooled state: the mean,
 * over the round's rows so far at the exit layer (the pending token in the
 * walk; the pending token and the drafts so far while drafting), of the exit
 * hidden state after the final RMSNorm, followed by the exit distribution's
 * max-probability. */
typedef struct {
  int32_t kind;
  int32_t n_cand;
  const int32_t* cand_layers;
  int32_t kmax;
  int32_t static_l, static_k;
  int32_t qnet_in, qnet_hidden; /* qnet_in: 3 or d_model + 1 (state below) */
  const float* qnet_params;
  int32_t trace_T; /* C_trace window, 1..64 (paper: 20) */
  int32_t topk;    /* k of the token confidence, 1..8 (paper: 5) */
  int32_t fixed_k; /* LEDE: 0 = adaptive drafting; 1..16 = fixed draft length */
  float conf_threshold; /* THRESHOLD: (0, 1] */
  /* Sampled decoding (speculative sampling, §4.1): temperature 0 is greedy;
   * > 0 samples drafts from the exit distribution and the emitted tokens
   * from the full model's, both at this temperature, with the acceptance
   * rule that keeps the full model's distribution; uniforms come from the
   * counter-based generator keyed by sample_seed and the round's position. */
  float temperature;
  uint32_t sample_seed;
  /* LEDE adaptive drafting: 0 (default) keeps each draft and lets the
   * decision on its state say whether to draft another; 1 drops a draft
   * whose decision is continue (the action is about the draft it was taken
   * on) and stops drafting.  The walk's exit always keeps d_1. */
  int32_t discard_on_continue;
} ssd_policy;

typedef struct {
  int32_t exit_layer; /* l* (0 for an AR round) */
  int32_t n_drafted;  /* k */
  int32_t n_accepted; /* a: accepted drafts */
  int32_t n_visited;  /* candidate layers evaluated by the walk */
  int32_t n_emitted;  /* a + 1 */
  int32_t pos;        /* position of the pending token at round start */
} ssd_round_info;

#define SSD_TRACE_MAXK 16
#define SSD_TRACE_MAXQ 48
#define SSD_TRACE_MAXC 16
/* Full per-round record (for metrics E, d, acceptance rate, and for parity). */
typedef struct {
  int32_t pos, x, kcap, n_visited, lstar, k, a, n_emit, n_q, pad;
  int32_t visited[SSD_TRACE_MAXC];
  int32_t drafts[SSD_TRACE_MAXK];
  int32_t verify_tok[SSD_TRACE_MAXK + 1];
  int32_t emitted[SSD_TRACE_MAXK + 1];
  int32_t q_action[SSD_TRACE_MAXQ];
  float draft_margin[SSD_TRACE_MAXK];      /* top-1 minus top-2 logit of each draft (greedy);
                                            * sampled: distance of the draw to the nearer end
                                            * of the token's CDF interval, over the mass */
  float verify_margin[SSD_TRACE_MAXK + 1];
  float verify_pmax[SSD_TRACE_MAXK + 1];
  float q_val[SSD_TRACE_MAXQ][2];
  float q_state[SSD_TRACE_MAXQ][3];
  /* sampled decoding only: margin of each acceptance test of d_i,
   * (p(d) - r q(d)) / max(p(d), r q(d)) (> 0 keeps d_i), and the margin of
   * the round's last draw (as draft_margin) */
  int32_t sampled, pad2;
  float accept_margin[SSD_TRACE_MAXK];
  float fix_margin;
} ssd_round_trace;

typedef struct ssd_ctx ssd_ctx;

/* Bytes of device workspace (KV cache, activations, control block, traces)
 * the caller must provide to ssd_init_model for this configuration. */
size_t ssd_workspace_bytes(const ssd_model_cfg* cfg);

/* Validates cfg and weights, lays out the workspace (256-byte aligned) and
 * uploads the rotary table.  cuda_stream is a cudaStream_t (NULL = legacy
 * default stream).  The context borrows weights and workspace. */
ssd_status ssd_init_model(const ssd_model_cfg* cfg, const ssd_weights* weights, void* workspace,
                          size_t workspace_bytes, void* cuda_stream, ssd_ctx** out);

/* Sets the policy and (re)builds the round and generation graphs.  Keeps the
 * KV cache and sequence state. */
ssd_status ssd_set_policy(ssd_ctx* ctx, const ssd_policy* policy);

/* Runs ids[0..n) (host) through the full model from position 0, seeds the
 * C_trace window with the full model's max-probabilities of the last trace_T
 * positions, and returns the next token, which becomes the pending token:
 * the greedy one, or with a policy temperature > 0 (set before this call) a
 * draw from the full model's distribution at that temperature, its uniform
 * keyed by (sample_seed, n - 1).  Needs n + 1 <= max_seq.  Synchronises the stream once. */
ssd_status ssd_prefill(ssd_ctx* ctx, const int32_t* ids, int32_t n, int32_t* first_token);

/* Like ssd_prefill over ids[0..n-1) but takes ids[n-1] as the pending token
 * (resumes a sequence whose last token is already chosen).  n >= 2. */
ssd_status ssd_resume(ssd_ctx* ctx, const int32_t* ids, int32_t n);

/* One speculation round, emitting 1..cap tokens into out_ids (host).  The
 * round drafts at most min(kmax, cap - 1) tokens.  Synchronises once. */
ssd_status ssd_step(ssd_ctx* ctx, int32_t* out_ids, int32_t cap, int32_t* n_out,
                    ssd_round_info* info);

/* Rounds until exactly max_new tokens have been emitted after the pending
 * token; out_ids (host) receives them.  rounds (host, optional) receives one
 * record per round up to rounds_cap; *n_rounds is the total.  One graph
 * launch, one synchronisation. */
ssd_status ssd_generate(ssd_ctx* ctx, int32_t max_new, int32_t* out_ids, int32_t* n_out,
                        ssd_round_info* rounds, int32_t rounds_cap, int32_t* n_rounds);

/* Enqueue-only form of ssd_generate: launches the generation graph on the
 * context's stream and returns without synchronising.  out_ids_dev is a
 * device buffer of max_new int32.  Read results later with
 * ssd_generate_result() after the stream has been synchronised. */
ssd_status ssd_generate_async(ssd_ctx* ctx, int32_t max_new, int32_t* out_ids_dev);

/* After ssd_generate_async and a stream synchronisation: number of rounds
 * and emitted tokens, device error flag check, and optional per-round
 * records (host). */
ssd_status ssd_generate_result(ssd_ctx* ctx, int32_t* n_rounds, int32_t* n_emitted,
                               ssd_round_trace* traces, int32_t traces_cap);

/* Full per-round records of the most recent ssd_step / ssd_generate call. */
ssd_status ssd_read_traces(ssd_ctx* ctx, ssd_round_trace* traces, int32_t cap, int32_t* n);

/* Message for the last failing call on ctx (or the last failing
 * ssd_init_model when ctx is NULL). */
const char* ssd_last_error(const ssd_ctx* ctx);

void ssd_destroy(ssd_ctx* ctx);

#ifdef __cplusplus
}
#endif

#endif /* SSD_H */
