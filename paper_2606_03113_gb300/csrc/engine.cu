// engine.cu -- the C ABI (include/ssd.h, include/ssd_ops.h): workspace layout,
// validation, prefill, and the CUDA graphs that run speculation rounds with
// every decision taken on the device.
//
// Round graph (one speculation round, §3.3; greedy or speculative-sampling
// acceptance, §4.1):
//   round_begin ─ IF(kcap > 0) { walk ; draft_begin ; WHILE(keep) { draft } } ─ verify ─ accept
//   walk  = embed(x) · layers(1..c_1) · head · decide_1 ·
//           IF(continue) { layers(c_1+1..c_2) · head · decide_2 · IF(continue) { ... } }
//   draft = embed(d_k) · SWITCH(l* index) { layers(1..c_j) } · head · decide
//   verify = embed(x, d_1..d_k) · layers(1..L) · head over k + 1 rows
// Generation graph: WHILE(emitted < max_new) { round }.
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <cmath>
#include <string>
#include <vector>

#include "kernels.h"
#include "pipe.cuh"

using namespace ssd;

namespace {

thread_local std::string g_init_error;

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

struct Carve {
  char* base;
  size_t off = 0;
  template <typename P>
  P* take(size_t bytes) {
    P* p = base ? reinterpret_cast<P*>(base + off) : nullptr;
    off = align256(off + bytes);
    return p;
  }
};

constexpr int kMaxQHidden = 1024;
constexpr int kPrefillChunk = 16;

// Lays out every device buffer in the workspace; returns the total size.
size_t layout(const ssd_model_cfg& c, char* base, Dims* D, Bufs* B) {
  Dims d{};
  d.L = c.n_layers;
  d.d = c.d_model;
  d.Hq = c.n_heads;
  d.Hkv = c.n_kv_heads;
  d.hd = c.head_dim;
  d.F = c.ffn_dim;
  d.V = c.vocab;
  d.max_seq = c.max_seq;
  d.qd = c.n_heads * c.head_dim;
  d.kvd = c.n_kv_heads * c.head_dim;
  d.nsplit = (c.max_seq + kAttnKeys - 1) / kAttnKeys;
  d.eps = c.rms_eps;
  d.num_sms = kMaxBlocks;  // set to the device's SM count at init
  d.ss_tiles = (c.d_model + 15) / 16;
  d.ss_nt = (c.d_model + 255) / 256;
  d.max_tiles = std::max(
      std::max(head_tiles(c.vocab), c.ffn_dim / 16 + 1),
      std::max((c.n_heads + 2 * c.n_kv_heads) * c.head_dim / 16 + 2, c.d_model / 16 + 1));
  const size_t elt = c.dtype == SSD_DTYPE_BF16 ? 2 : 4;
  Carve cv{base};
  Bufs b{};
  b.ctl = cv.take<Ctl>(sizeof(Ctl));
  b.h = cv.take<float>(sizeof(float) * kMaxM * d.d);
  b.ss = cv.take<float>(sizeof(float) * 2 * kMaxM);
  b.ss_tile = cv.take<float>(sizeof(float) * 2 * 2 * kMaxM * (size_t)kMaxBlocks);
  b.ss_counter = cv.take<uint32_t>(sizeof(uint32_t) * 2);
  b.ss_part = cv.take<float>(sizeof(float) * 2 * (size_t)d.ss_nt * kMaxM);
  b.gpart = cv.take<float>(sizeof(float) * std::max((size_t)kMaxBlocks * 2 * 32 * kMaxM,
                                                      tile_part_floats(kMaxBlocks)));
  b.tile_counter = cv.take<uint32_t>(sizeof(uint32_t) * (size_t)d.max_tiles);

  b.xq = cv.take<float>(sizeof(float) * kMaxM * d.qd);
  b.attn_part = cv.take<float>(sizeof(float) * kMaxM * d.Hq * (size_t)d.nsplit * d.hd);
  b.attn_ml = cv.take<float>(sizeof(float) * kMaxM * d.Hq * (size_t)d.nsplit * 2);
  b.attn_counter = cv.take<uint32_t>(sizeof(uint32_t) * (size_t)d.Hkv * kMaxM);
  b.chain_bar = cv.take<uint32_t>(sizeof(uint32_t) * 2);
  b.attn_out = cv.take<float>(sizeof(float) * kMaxM * d.qd);
  b.act = cv.take<float>(sizeof(float) * kMaxM * d.F);
  b.logits = cv.take<float>(sizeof(float) * kMaxM * (size_t)d.V);
  b.draft_logits = cv.take<float>(sizeof(float) * kMaxDraft * (size_t)d.V);
  b.head_part = cv.take<void>(sizeof(HeadPart) * kMaxM * 2 * (size_t)kMaxBlocks);
  b.head_counter = cv.take<uint32_t>(sizeof(uint32_t));
  b.stats = cv.take<RowStats>(sizeof(RowStats) * kMaxM);
  b.rope = cv.take<float2>(sizeof(float2) * (size_t)d.max_seq * (d.hd / 2));
  b.kv = cv.take<void>(elt * (size_t)d.L * 2 * d.Hkv * (size_t)d.max_seq * d.hd);
  // largest network: d + 1 inputs (pooled state), kMaxQHidden hidden units
  b.qparams = cv.take<float>(sizeof(float) * ((size_t)kMaxQHidden * (d.d + 4) + 2));
  b.pool = cv.take<float>(sizeof(float) * (size_t)d.d);
  b.out_tok = cv.take<int32_t>(sizeof(int32_t) * (size_t)d.max_seq);
  b.traces = cv.take<ssd_round_trace>(sizeof(ssd_round_trace) * (size_t)d.max_seq);
  b.pre_tok = cv.take<int32_t>(sizeof(int32_t) * (size_t)d.max_seq);
  if (D) *D = d;
  if (B) *B = b;
  return cv.off;
}

const char* check_cfg(const ssd_model_cfg* c) {
  if (!c) return "cfg is NULL";
  if (c->dtype != SSD_DTYPE_F32 && c->dtype != SSD_DTYPE_BF16) return "dtype must be F32 or BF16";
  if (c->n_layers < 1 || c->n_layers > 1024) return "n_layers out of range";
  if (c->d_model < 8 || c->d_model % 8) return "d_model must be a positive multiple of 8";
  if (c->n_heads < 1 || c->n_kv_heads < 1 || c->n_heads % c->n_kv_heads)
    return "n_heads must be a positive multiple of n_kv_heads";
  if (c->head_dim < 8 || c->head_dim % 8 || c->head_dim > 256)
    return "head_dim must be a multiple of 8 in [8, 256]";
  if (c->ffn_dim < 8 || c->ffn_dim % 8) return "ffn_dim must be a positive multiple of 8";
  if ((c->n_heads * c->head_dim) % 8) return "n_heads*head_dim must be a multiple of 8";
  if (c->vocab < 2 || c->vocab % 2) return "vocab must be even and >= 2";
  if (c->max_seq < 2) return "max_seq must be >= 2";
  if (!(c->rms_eps >= 0.f) || !(c->rope_theta > 0.f)) return "rms_eps >= 0 and rope_theta > 0";
  return nullptr;
}

bool aligned16(const void* p) { return p && ((uintptr_t)p & 15u) == 0; }

}  // namespace

struct ssd_ctx {
  ssd_model_cfg cfg{};
  Dims D{};
  Bufs B{};
  const void* embed = nullptr;
  const void* lm_head = nullptr;
  const void* final_norm = nullptr;
  std::vector<LayerW> layers;
  std::vector<CUtensorMap> wmaps;  // bf16: [L][4] layer matrices, then the LM head
  TileMaps tmaps{};                // bf16: the input buffers
  cudaStream_t stream = nullptr;
  cudaStream_t cap = nullptr;
  std::string err;
  // policy
  bool have_policy = false;
  int kind = SSD_POLICY_AR;
  std::vector<int> cand;
  int kmax = 0, static_l = 0, static_k = 0, q_hidden = 0, trace_T = 20, topk = 5, fixed_k = 0;
  int q_in = 3;
  bool sampled = false;  // temperature > 0: the exit heads write their logits
  // graphs
  cudaGraph_t round_g = nullptr, gen_g = nullptr;
  cudaGraphExec_t round_x = nullptr, gen_x = nullptr;
  // sequence state mirrored on the host after each synchronising call
  bool have_x = false;
  bool async_pending = false;
  int pos_host = 0;
  int last_rounds = 0;
};

namespace {

ssd_status fail(ssd_ctx* x, ssd_status s, const std::string& msg) {
  if (x)
    x->err = msg;
  else
    g_init_error = msg;
  return s;
}

ssd_status cuda_fail(ssd_ctx* x, const char* what, cudaError_t e) {
  std::string m = std::string(what) + ": " + cudaGetErrorName(e) + " (" + cudaGetErrorString(e) + ")";
  cudaGetLastError();
  return fail(x, SSD_ERR_CUDA, m);
}

#define CK(x, call)                                   \
  do {                                                \
    cudaError_t e_ = (call);                          \
    if (e_ != cudaSuccess) return cuda_fail(x, #call, e_); \
  } while (0)

RowSel rows(int mode) { return RowSel{mode, 0, 0, nullptr}; }
RowSel rows_explicit(int pos0, int M, const int32_t* tok) {
  return RowSel{kRowsExplicit, pos0, M, tok};
}

// ------------------------------------------------------------ graph building

// Appends kernels to graph g by capturing the private stream into it.
struct Seq {
  ssd_ctx* x;
  cudaGraph_t g;
  cudaGraphNode_t last = nullptr;
  cudaError_t begin() {
    g_pdl_ok = false;
    return cudaStreamBeginCaptureToGraph(x->cap, g, last ? &last : nullptr, nullptr, last ? 1 : 0,
                                         cudaStreamCaptureModeThreadLocal);
  }
  cudaError_t end() {
    cudaStreamCaptureStatus st;
    const cudaGraphNode_t* deps = nullptr;
    size_t nd = 0;
    cudaError_t e = cudaStreamGetCaptureInfo(x->cap, &st, nullptr, nullptr, &deps, nullptr, &nd);
    if (e != cudaSuccess) return e;
    if (nd > 1) return cudaErrorStreamCaptureUnjoined;
    if (nd == 1) last = deps[0];
    cudaGraph_t out = nullptr;
    return cudaStreamEndCapture(x->cap, &out);
  }
  cudaError_t cond(cudaGraphConditionalHandle h, cudaGraphConditionalNodeType type, unsigned n,
                   cudaGraph_t* bodies) {
    cudaGraphNodeParams p = {cudaGraphNodeTypeConditional};
    p.conditional.handle = h;
    p.conditional.type = type;
    p.conditional.size = n;
    cudaGraphNode_t node;
    cudaError_t e = cudaGraphAddNode(&node, g, last ? &last : nullptr, nullptr, last ? 1 : 0, &p);
    if (e != cudaSuccess) return e;
    for (unsigned i = 0; i < n; ++i) bodies[i] = p.conditional.phGraph_out[i];
    last = node;
    return cudaSuccess;
  }
};

#define GK(call)                                \
  do {                                          \
    cudaError_t e_ = (call);                    \
    if (e_ != cudaSuccess) return e_;           \
  } while (0)

const TileMaps* tile_maps(const ssd_ctx* x) {
  return x->cfg.dtype == SSD_DTYPE_BF16 ? &x->tmaps : nullptr;
}

const CUtensorMap* lm_map(const ssd_ctx* x) {
  return x->cfg.dtype == SSD_DTYPE_BF16 ? &x->wmaps[4 * (size_t)x->cfg.n_layers] : nullptr;
}

// mrows: the most rows the launches will see (1: the single-row kernels).
cudaError_t enqueue_layers(ssd_ctx* x, int l_from, int l_to, RowSel sel, int mrows,
                           cudaStream_t st) {
  if (x->cfg.dtype == SSD_DTYPE_BF16 && g_chain_enabled && l_to > l_from) {
    // QKV of the first layer, then per layer: attention, and O + gate/up +
    // down + the next layer's QKV as one persistent launch
    GK(launch_layer_part(x->D, x->B, x->cfg.dtype, x->layers[l_from], tile_maps(x), l_from, 0, sel,
                         mrows, st));
    for (int l = l_from; l < l_to; ++l) {
      GK(launch_layer_part(x->D, x->B, x->cfg.dtype, x->layers[l], tile_maps(x), l, 1, sel, mrows,
                           st));
      GK(launch_tile_chain(x->D, x->B, *tile_maps(x), x->layers[l],
                           l + 1 < l_to ? &x->layers[l + 1] : nullptr, l, sel, mrows, st));
    }
    return cudaSuccess;
  }
  for (int l = l_from; l < l_to; ++l)
    GK(launch_layer(x->D, x->B, x->cfg.dtype, x->layers[l], tile_maps(x), l, sel, mrows, st));
  return cudaSuccess;
}

cudaError_t enqueue_head(ssd_ctx* x, RowSel sel, int mrows, int topk, bool logits,
                         cudaStream_t st) {
  return launch_head(x->D, x->B, x->cfg.dtype, x->lm_head, lm_map(x), tile_maps(x), x->final_norm,
                     topk, logits, sel, mrows, st);
}

// Walk segment j: layers (done, c_j], exit head, decision; nested IF for j+1.
cudaError_t build_walk(ssd_ctx* x, Seq& s, const std::vector<int>& cands, int j, int done) {
  const int J = (int)cands.size();
  const bool last = j == J - 1;
  cudaGraphConditionalHandle next = 0;
  if (!last) GK(cudaGraphConditionalHandleCreate(&next, s.g, 0, 0));
  GK(s.begin());
  if (j == 0) GK(launch_embed(x->D, x->B, x->cfg.dtype, x->embed, rows(kRowsWalk), false, 0, x->cap));
  GK(enqueue_layers(x, done, cands[j], rows(kRowsWalk), 1, x->cap));
  GK(enqueue_head(x, rows(kRowsWalk), 1, x->topk, x->sampled, x->cap));
  GK(launch_decide(x->D, x->B, kDecideWalk, j, last ? 1 : 0, cands[j], x->final_norm,
                   x->cfg.dtype, next, 0, x->cap));
  GK(s.end());
  if (last) return cudaSuccess;
  cudaGraph_t body;
  GK(s.cond(next, cudaGraphCondTypeIf, 1, &body));
  Seq sub{x, body};
  return build_walk(x, sub, cands, j + 1, cands[j]);
}

// IF body of a speculative round: walk, then the drafting loop.
cudaError_t build_draft_phase(ssd_ctx* x, cudaGraph_t body) {
  Seq s{x, body};
  std::vector<int> cands = x->kind == SSD_POLICY_LEDE ? x->cand : std::vector<int>{x->static_l};
  const int J = (int)cands.size();
  GK(build_walk(x, s, cands, 0, 0));
  cudaGraphConditionalHandle hw;
  GK(cudaGraphConditionalHandleCreate(&hw, body, 0, 0));
  GK(s.begin());
  GK(launch_draft_begin(x->B, hw, x->cap));
  GK(s.end());
  cudaGraph_t wbody;
  GK(s.cond(hw, cudaGraphCondTypeWhile, 1, &wbody));
  Seq w{x, wbody};
  if (J > 1) {
    cudaGraphConditionalHandle hs;
    GK(cudaGraphConditionalHandleCreate(&hs, wbody, 0, 0));
    GK(w.begin());
    GK(launch_embed(x->D, x->B, x->cfg.dtype, x->embed, rows(kRowsDraft), false, hs, x->cap));
    GK(w.end());
    std::vector<cudaGraph_t> cases(J);
    GK(w.cond(hs, cudaGraphCondTypeSwitch, (unsigned)J, cases.data()));
    for (int j = 0; j < J; ++j) {
      Seq c{x, cases[j]};
      GK(c.begin());
      GK(enqueue_layers(x, 0, cands[j], rows(kRowsDraft), 1, x->cap));
      GK(c.end());
    }
    GK(w.begin());
  } else {
    GK(w.begin());
    GK(launch_embed(x->D, x->B, x->cfg.dtype, x->embed, rows(kRowsDraft), false, 0, x->cap));
    GK(enqueue_layers(x, 0, cands[0], rows(kRowsDraft), 1, x->cap));
  }
  GK(enqueue_head(x, rows(kRowsDraft), 1, x->topk, x->sampled, x->cap));
  GK(launch_decide(x->D, x->B, kDecideDraft, 0, 0, 0, x->final_norm, x->cfg.dtype, 0, hw,
                   x->cap));
  return w.end();
}

// One round appended to graph g; gen != 0 when g is the body of the
// generation loop.
cudaError_t build_round(ssd_ctx* x, cudaGraph_t g, cudaGraphConditionalHandle gen) {
  Seq s{x, g};
  const bool spec = x->kind != SSD_POLICY_AR;
  cudaGraphConditionalHandle hd = 0;
  if (spec) GK(cudaGraphConditionalHandleCreate(&hd, g, 0, 0));
  GK(s.begin());
  GK(launch_round_begin(x->D, x->B, hd, x->cap));
  GK(s.end());
  if (spec) {
    cudaGraph_t body;
    GK(s.cond(hd, cudaGraphCondTypeIf, 1, &body));
    GK(build_draft_phase(x, body));
  }
  GK(s.begin());
  GK(launch_embed(x->D, x->B, x->cfg.dtype, x->embed, rows(kRowsVerify), spec, 0, x->cap));
  const int mrows = spec ? std::min(x->kmax + 1, kMaxM) : 1;
  GK(enqueue_layers(x, 0, x->D.L, rows(kRowsVerify), mrows, x->cap));
  GK(enqueue_head(x, rows(kRowsVerify), mrows, x->topk, x->sampled, x->cap));
  GK(launch_accept(x->D, x->B, gen, x->cap));
  return s.end();
}

void destroy_graphs(ssd_ctx* x) {
  if (x->round_x) cudaGraphExecDestroy(x->round_x);
  if (x->gen_x) cudaGraphExecDestroy(x->gen_x);
  if (x->round_g) cudaGraphDestroy(x->round_g);
  if (x->gen_g) cudaGraphDestroy(x->gen_g);
  x->round_x = x->gen_x = nullptr;
  x->round_g = x->gen_g = nullptr;
}

cudaError_t build_graphs(ssd_ctx* x) {
  destroy_graphs(x);
  GK(cudaGraphCreate(&x->round_g, 0));
  GK(build_round(x, x->round_g, 0));
  GK(cudaGraphInstantiate(&x->round_x, x->round_g, 0));
  GK(cudaGraphCreate(&x->gen_g, 0));
  cudaGraphConditionalHandle hg;
  GK(cudaGraphConditionalHandleCreate(&hg, x->gen_g, 1, cudaGraphCondAssignDefault));
  Seq top{x, x->gen_g};
  cudaGraph_t body;
  GK(top.cond(hg, cudaGraphCondTypeWhile, 1, &body));
  GK(build_round(x, body, hg));
  GK(cudaGraphInstantiate(&x->gen_x, x->gen_g, 0));
  GK(cudaGraphUpload(x->round_x, x->stream));
  GK(cudaGraphUpload(x->gen_x, x->stream));
  return cudaSuccess;
}

ssd_status read_ctl(ssd_ctx* x, Ctl* h) {
  CK(x, cudaMemcpyAsync(h, x->B.ctl, sizeof(Ctl), cudaMemcpyDeviceToHost, x->stream));
  return SSD_OK;
}

ssd_status check_flag(ssd_ctx* x, const Ctl& c) {
  if (c.err) {
    char buf[128];
    snprintf(buf, sizeof buf, "device consistency check failed (flags 0x%x)", c.err);
    return fail(x, SSD_ERR_DEVICE_FLAG, buf);
  }
  return SSD_OK;
}

// Full-model pass over ids[0..n) (already in pre_tok) from position 0 in
// chunks; max-probabilities of the last trace_T rows seed the C_trace window.
ssd_status run_prompt(ssd_ctx* x, int n) {
  const int T = x->trace_T;
  CK(x, launch_reset_sequence(x->B, x->stream));
  for (int c0 = 0; c0 < n; c0 += kPrefillChunk) {
    const int M = std::min(kPrefillChunk, n - c0);
    const RowSel sel = rows_explicit(c0, M, x->B.pre_tok + c0);
    CK(x, launch_embed(x->D, x->B, x->cfg.dtype, x->embed, sel, true, 0, x->stream));
    CK(x, enqueue_layers(x, 0, x->D.L, sel, kPrefillChunk, x->stream));
    if (c0 + M > n - T || c0 + M == n) {
      CK(x, enqueue_head(x, sel, kPrefillChunk, x->topk, x->sampled, x->stream));
      const int first = std::max(c0, n - T) - c0;
      if (first < M) CK(x, launch_trace_push(x->B, first, M - first, x->stream));
    }
  }
  return SSD_OK;
}

bool tokens_ok(const int32_t* ids, int n, int V) {
  for (int i = 0; i < n; ++i)
    if (ids[i] < 0 || ids[i] >= V) return false;
  return true;
}

void summarize(const ssd_round_trace& t, ssd_round_info* r) {
  r->exit_layer = t.lstar;
  r->n_drafted = t.k;
  r->n_accepted = t.a;
  r->n_visited = t.n_visited;
  r->n_emitted = t.n_emit;
  r->pos = t.pos;
}

int kcap_for(const ssd_ctx* x, int budget) {
  if (x->kind == SSD_POLICY_AR) return 0;
  int k = std::min(x->kmax, budget - 1);
  if (x->kind == SSD_POLICY_STATIC) k = std::min(k, x->static_k);
  if (x->kind == SSD_POLICY_LEDE && x->fixed_k > 0) k = std::min(k, x->fixed_k);
  return std::max(k, 0);
}

}  // namespace

// =================================================================== C ABI

extern "C" {

size_t ssd_workspace_bytes(const ssd_model_cfg* cfg) {
  if (check_cfg(cfg)) return 0;
  return layout(*cfg, nullptr, nullptr, nullptr);
}

ssd_status ssd_init_model(const ssd_model_cfg* cfg, const ssd_weights* w, void* workspace,
                          size_t workspace_bytes, void* cuda_stream, ssd_ctx** out) {
  if (!out) return fail(nullptr, SSD_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  if (const char* why = check_cfg(cfg)) return fail(nullptr, SSD_ERR_INVALID_ARG, why);
  if (!w || !aligned16(w->embed) || !aligned16(w->lm_head) || !aligned16(w->final_norm) ||
      !w->attn_norm || !w->wqkv || !w->wo || !w->ffn_norm || !w->w_gate_up || !w->w_down)
    return fail(nullptr, SSD_ERR_INVALID_ARG, "weights: NULL or unaligned pointer");
  for (int l = 0; l < cfg->n_layers; ++l)
    if (!aligned16(w->attn_norm[l]) || !aligned16(w->wqkv[l]) || !aligned16(w->wo[l]) ||
        !aligned16(w->ffn_norm[l]) || !aligned16(w->w_gate_up[l]) || !aligned16(w->w_down[l]))
      return fail(nullptr, SSD_ERR_INVALID_ARG, "layer weights: NULL or unaligned pointer");
  const size_t need = layout(*cfg, nullptr, nullptr, nullptr);
  if (!workspace || ((uintptr_t)workspace & 255u))
    return fail(nullptr, SSD_ERR_INVALID_ARG, "workspace must be non-NULL and 256-byte aligned");
  if (workspace_bytes < need) return fail(nullptr, SSD_ERR_CAPACITY, "workspace too small");
  if (cfg->head_dim % 32 || cfg->ffn_dim % 16)
    return fail(nullptr, SSD_ERR_UNSUPPORTED, "head_dim must be a multiple of 32, ffn_dim of 16");
  if (cfg->dtype == SSD_DTYPE_BF16 && cfg->head_dim != 128)
    return fail(nullptr, SSD_ERR_UNSUPPORTED, "bf16 models need head_dim 128");
  int dev = 0, sms = 0;
  cudaError_t e0 = cudaGetDevice(&dev);
  if (e0 == cudaSuccess) e0 = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e0 == cudaSuccess) e0 = prepare_gemv_kernels();
  if (e0 == cudaSuccess && cfg->dtype == SSD_DTYPE_BF16) e0 = prepare_tile_kernels();
  if (e0 != cudaSuccess) return cuda_fail(nullptr, "ssd_init_model device query", e0);
  if (const char* v = getenv("SSD_NO_PDL")) g_pdl_enabled = !(v[0] == '1');
  if (const char* v = getenv("SSD_NO_CHAIN")) g_chain_enabled = !(v[0] == '1');
  ssd_ctx* x = new ssd_ctx();
  x->cfg = *cfg;
  layout(*cfg, static_cast<char*>(workspace), &x->D, &x->B);
  // persistent grids: one block per SM of this context, all resident at once
  // (their phase barriers and split-tile fix-ups wait on other blocks)
  int per_sm = 1;
  if (cfg->dtype == SSD_DTYPE_BF16) {
    per_sm = tile_blocks_per_sm();
    if (per_sm < 1) {
      delete x;
      return fail(nullptr, SSD_ERR_UNSUPPORTED, "tensor-core kernels cannot be resident on an SM");
    }
  }
  x->D.num_sms = std::min(sms * std::min(per_sm, 1), kMaxBlocks);
  x->embed = w->embed;
  x->lm_head = w->lm_head;
  x->final_norm = w->final_norm;
  x->layers.resize(cfg->n_layers);
  for (int l = 0; l < cfg->n_layers; ++l)
    x->layers[l] = LayerW{w->attn_norm[l], w->wqkv[l], w->wo[l], w->ffn_norm[l], w->w_gate_up[l],
                          w->w_down[l], {nullptr, nullptr, nullptr, nullptr}};
  if (cfg->dtype == SSD_DTYPE_BF16) {
    // tensor maps of every weight matrix and of the input buffers
    const int L = cfg->n_layers, d = cfg->d_model, F = cfg->ffn_dim;
    const int qkv = (cfg->n_heads + 2 * cfg->n_kv_heads) * cfg->head_dim;
    const int qd = cfg->n_heads * cfg->head_dim;
    x->wmaps.resize(4 * (size_t)L + 1);
    bool ok = true;
    for (int l = 0; l < L && ok; ++l) {
      CUtensorMap* m = &x->wmaps[4 * (size_t)l];
      ok = encode_weight_map(m, w->wqkv[l], qkv, d) && encode_weight_map(m + 1, w->wo[l], d, qd) &&
           encode_weight_map(m + 2, w->w_gate_up[l], 2 * F, d) &&
           encode_weight_map(m + 3, w->w_down[l], d, F);
      for (int k = 0; k < 4; ++k) x->layers[l].tm[k] = m + k;
    }
    ok = ok && encode_weight_map(&x->wmaps[4 * (size_t)L], w->lm_head, cfg->vocab, d) &&
         encode_input_maps(x->tmaps.h, x->B.h, d) &&
         encode_input_maps(x->tmaps.attn_out, x->B.attn_out, qd) &&
         encode_input_maps(x->tmaps.act, x->B.act, F);
    if (!ok) {
      delete x;
      return fail(nullptr, SSD_ERR_CUDA, "tensor-map encoding failed");
    }
  }
  x->stream = static_cast<cudaStream_t>(cuda_stream);
  cudaError_t e = cudaStreamCreateWithFlags(&x->cap, cudaStreamNonBlocking);
  if (e != cudaSuccess) {
    ssd_status s = cuda_fail(nullptr, "cudaStreamCreateWithFlags", e);
    delete x;
    return s;
  }
  // rotary table (cos, sin) of pos * theta^(-2i/hd), computed in double
  const int half = cfg->head_dim / 2;
  std::vector<float2> rope((size_t)cfg->max_seq * half);
  for (int p = 0; p < cfg->max_seq; ++p)
    for (int i = 0; i < half; ++i) {
      const double inv = 1.0 / std::pow((double)cfg->rope_theta, (2.0 * i) / cfg->head_dim);
      const double t = (double)p * inv;
      rope[(size_t)p * half + i] = make_float2((float)std::cos(t), (float)std::sin(t));
    }
  e = cudaMemcpyAsync(x->B.rope, rope.data(), sizeof(float2) * rope.size(), cudaMemcpyHostToDevice,
                      x->stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(x->B.ctl, 0, sizeof(Ctl), x->stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(x->B.head_counter, 0, sizeof(uint32_t), x->stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(x->B.ss, 0, sizeof(float) * 2 * kMaxM, x->stream);
  if (e == cudaSuccess)
    e = cudaMemsetAsync(x->B.ss_part, 0, sizeof(float) * 2 * (size_t)x->D.ss_nt * kMaxM, x->stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(x->B.ss_counter, 0, sizeof(uint32_t) * 2, x->stream);
  if (e == cudaSuccess)
    e = cudaMemsetAsync(x->B.attn_counter, 0, sizeof(uint32_t) * (size_t)x->D.Hkv * kMaxM, x->stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(x->B.chain_bar, 0, sizeof(uint32_t) * 2, x->stream);
  if (e == cudaSuccess)
    e = cudaMemsetAsync(x->B.tile_counter, 0, sizeof(uint32_t) * (size_t)x->D.max_tiles, x->stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(x->stream);
  if (e != cudaSuccess) {
    ssd_status s = cuda_fail(nullptr, "ssd_init_model upload", e);
    cudaStreamDestroy(x->cap);
    delete x;
    return s;
  }
  *out = x;
  return SSD_OK;
}

ssd_status ssd_set_policy(ssd_ctx* x, const ssd_policy* p) {
  if (!x) return fail(nullptr, SSD_ERR_INVALID_ARG, "ctx is NULL");
  if (!p) return fail(x, SSD_ERR_INVALID_ARG, "policy is NULL");
  const int L = x->cfg.n_layers;
  DevPolicy dp{};
  dp.kind = p->kind;
  dp.trace_T = p->trace_T > 0 ? p->trace_T : 20;
  dp.topk = p->topk > 0 ? p->topk : 5;
  if (dp.trace_T > kTraceCap) return fail(x, SSD_ERR_INVALID_ARG, "trace_T must be in 1..64");
  if (dp.topk > kTopK) return fail(x, SSD_ERR_INVALID_ARG, "topk must be in 1..8");
  if (p->kind != SSD_POLICY_AR && p->kind != SSD_POLICY_STATIC && p->kind != SSD_POLICY_LEDE &&
      p->kind != SSD_POLICY_THRESHOLD)
    return fail(x, SSD_ERR_INVALID_ARG, "unknown policy kind");
  if (p->kind != SSD_POLICY_AR && (p->kmax < 1 || p->kmax > kMaxDraft))
    return fail(x, SSD_ERR_INVALID_ARG, "kmax must be in 1..16");
  std::vector<int> cand;
  if (p->kind == SSD_POLICY_STATIC) {
    if (p->static_l < 1 || p->static_l > L || p->static_k < 1)
      return fail(x, SSD_ERR_INVALID_ARG, "static_l must be in 1..n_layers and static_k >= 1");
  }
  if (!(p->temperature >= 0.f && p->temperature <= 100.f))
    return fail(x, SSD_ERR_INVALID_ARG, "temperature must be in [0, 100]");
  if (p->kind == SSD_POLICY_THRESHOLD) {
    if (p->static_l < 1 || p->static_l > L)
      return fail(x, SSD_ERR_INVALID_ARG, "static_l must be in 1..n_layers");
    if (!(p->conf_threshold > 0.f && p->conf_threshold <= 1.f))
      return fail(x, SSD_ERR_INVALID_ARG, "conf_threshold must be in (0, 1]");
  }
  if (p->kind == SSD_POLICY_LEDE && (p->fixed_k < 0 || p->fixed_k > kMaxDraft))
    return fail(x, SSD_ERR_INVALID_ARG, "fixed_k must be in 0..16");
  if (p->kind == SSD_POLICY_LEDE) {
    if (p->n_cand < 1 || p->n_cand > kMaxCand || !p->cand_layers)
      return fail(x, SSD_ERR_INVALID_ARG, "n_cand must be in 1..16");
    for (int j = 0; j < p->n_cand; ++j) {
      const int c = p->cand_layers[j];
      if (c < 1 || c > L || (j && c <= p->cand_layers[j - 1]))
        return fail(x, SSD_ERR_INVALID_ARG, "cand_layers must ascend within 1..n_layers");
      cand.push_back(c);
      dp.cand[j] = c;
    }
    if (p->qnet_in != 3 && p->qnet_in != x->cfg.d_model + 1)
      return fail(x, SSD_ERR_INVALID_ARG, "qnet_in must be 3 or d_model + 1");
    if (p->qnet_hidden < 1 || p->qnet_hidden > kMaxQHidden || !p->qnet_params)
      return fail(x, SSD_ERR_INVALID_ARG, "qnet_hidden must be in 1..1024 with parameters");
  }
  dp.kmax = p->kmax;
  dp.static_l = p->static_l;
  dp.static_k = p->static_k;
  dp.n_cand = (int)cand.size();
  dp.q_hidden = p->kind == SSD_POLICY_LEDE ? p->qnet_hidden : 0;
  dp.q_in = p->kind == SSD_POLICY_LEDE ? p->qnet_in : 3;
  dp.fixed_k = p->kind == SSD_POLICY_LEDE ? p->fixed_k : 0;
  dp.tau = p->kind == SSD_POLICY_THRESHOLD ? p->conf_threshold : 0.f;
  dp.temp = p->temperature;
  dp.discard = p->kind == SSD_POLICY_LEDE && p->discard_on_continue ? 1 : 0;
  dp.seed = p->sample_seed;
  CK(x, cudaMemcpyAsync(&x->B.ctl->pol, &dp, sizeof(dp), cudaMemcpyHostToDevice, x->stream));
  if (p->kind == SSD_POLICY_LEDE)
    CK(x, cudaMemcpyAsync(x->B.qparams, p->qnet_params,
                          sizeof(float) * ((size_t)p->qnet_hidden * (p->qnet_in + 3) + 2),
                          cudaMemcpyHostToDevice, x->stream));
  CK(x, cudaStreamSynchronize(x->stream));
  // The graphs depend on the policy kind, the candidate (or static) exit
  // layers, kmax, topk and whether the heads write logits; everything else
  // is read on the device from the policy just copied.
  const int kmax_new = p->kind == SSD_POLICY_AR ? 0 : p->kmax;
  const bool sampled = p->temperature > 0.f;
  const bool same_graphs = x->have_policy && x->kind == p->kind && x->cand == cand &&
                           x->kmax == kmax_new && x->static_l == p->static_l &&
                           x->topk == dp.topk && x->sampled == sampled;
  x->kind = p->kind;
  x->cand = cand;
  x->kmax = kmax_new;
  x->static_l = p->static_l;
  x->static_k = p->static_k;
  x->fixed_k = dp.fixed_k;
  x->q_hidden = dp.q_hidden;
  x->q_in = dp.q_in;
  x->trace_T = dp.trace_T;
  x->topk = dp.topk;
  x->sampled = sampled;
  if (same_graphs) return SSD_OK;
  cudaError_t e = build_graphs(x);
  if (e != cudaSuccess) {
    destroy_graphs(x);
    x->have_policy = false;
    return cuda_fail(x, "building the round graphs", e);
  }
  x->have_policy = true;
  return SSD_OK;
}

ssd_status ssd_prefill(ssd_ctx* x, const int32_t* ids, int32_t n, int32_t* first_token) {
  if (!x) return fail(nullptr, SSD_ERR_INVALID_ARG, "ctx is NULL");
  if (!ids || n < 1) return fail(x, SSD_ERR_INVALID_ARG, "ids must hold n >= 1 tokens");
  if (!tokens_ok(ids, n, x->cfg.vocab)) return fail(x, SSD_ERR_INVALID_ARG, "token id out of range");
  if (n + 1 > x->cfg.max_seq) return fail(x, SSD_ERR_CAPACITY, "prompt does not fit max_seq");
  x->have_x = false;
  x->async_pending = false;
  CK(x, cudaMemcpyAsync(x->B.pre_tok, ids, sizeof(int32_t) * n, cudaMemcpyHostToDevice, x->stream));
  ssd_status s = run_prompt(x, n);
  if (s) return s;
  const int last_M = (n - 1) % kPrefillChunk + 1;
  CK(x, launch_set_pending(x->D, x->B, last_M - 1, -1, n, x->stream));
  Ctl c;
  if ((s = read_ctl(x, &c))) return s;
  CK(x, cudaStreamSynchronize(x->stream));
  if ((s = check_flag(x, c))) return s;
  x->have_x = true;
  x->pos_host = c.pos;
  if (first_token) *first_token = c.x;
  return SSD_OK;
}

ssd_status ssd_resume(ssd_ctx* x, const int32_t* ids, int32_t n) {
  if (!x) return fail(nullptr, SSD_ERR_INVALID_ARG, "ctx is NULL");
  if (!ids || n < 2) return fail(x, SSD_ERR_INVALID_ARG, "ids must hold n >= 2 tokens");
  if (!tokens_ok(ids, n, x->cfg.vocab)) return fail(x, SSD_ERR_INVALID_ARG, "token id out of range");
  if (n > x->cfg.max_seq) return fail(x, SSD_ERR_CAPACITY, "sequence does not fit max_seq");
  x->have_x = false;
  x->async_pending = false;
  CK(x, cudaMemcpyAsync(x->B.pre_tok, ids, sizeof(int32_t) * (n - 1), cudaMemcpyHostToDevice,
                        x->stream));
  ssd_status s = run_prompt(x, n - 1);
  if (s) return s;
  CK(x, launch_set_pending(x->D, x->B, 0, ids[n - 1], n - 1, x->stream));
  Ctl c;
  if ((s = read_ctl(x, &c))) return s;
  CK(x, cudaStreamSynchronize(x->stream));
  if ((s = check_flag(x, c))) return s;
  x->have_x = true;
  x->pos_host = c.pos;
  return SSD_OK;
}

ssd_status ssd_step(ssd_ctx* x, int32_t* out_ids, int32_t cap, int32_t* n_out,
                    ssd_round_info* info) {
  if (!x) return fail(nullptr, SSD_ERR_INVALID_ARG, "ctx is NULL");
  if (!x->have_policy) return fail(x, SSD_ERR_STATE, "no policy set");
  if (!x->have_x || x->async_pending) return fail(x, SSD_ERR_STATE, "no prefilled sequence");
  if (!out_ids || cap < 1) return fail(x, SSD_ERR_INVALID_ARG, "out_ids must hold cap >= 1");
  if (x->pos_host + kcap_for(x, cap) + 1 > x->cfg.max_seq)
    return fail(x, SSD_ERR_CAPACITY, "KV cache full");
  CK(x, launch_begin_call(x->B, cap, x->stream));
  CK(x, cudaGraphLaunch(x->round_x, x->stream));
  Ctl c;
  ssd_status s = read_ctl(x, &c);
  if (s) return s;
  std::vector<int32_t> tok(cap);
  ssd_round_trace tr;
  CK(x, cudaMemcpyAsync(tok.data(), x->B.out_tok, sizeof(int32_t) * cap, cudaMemcpyDeviceToHost,
                        x->stream));
  CK(x, cudaMemcpyAsync(&tr, x->B.traces, sizeof(tr), cudaMemcpyDeviceToHost, x->stream));
  CK(x, cudaStreamSynchronize(x->stream));
  x->pos_host = c.pos;
  x->last_rounds = c.round_idx;
  if ((s = check_flag(x, c))) return s;
  if (c.n_out < 1 || c.n_out > cap) return fail(x, SSD_ERR_DEVICE_FLAG, "round emitted no tokens");
  memcpy(out_ids, tok.data(), sizeof(int32_t) * c.n_out);
  if (n_out) *n_out = c.n_out;
  if (info) summarize(tr, info);
  return SSD_OK;
}

ssd_status ssd_generate_async(ssd_ctx* x, int32_t max_new, int32_t* out_ids_dev) {
  if (!x) return fail(nullptr, SSD_ERR_INVALID_ARG, "ctx is NULL");
  if (!x->have_policy) return fail(x, SSD_ERR_STATE, "no policy set");
  if (!x->have_x || x->async_pending) return fail(x, SSD_ERR_STATE, "no prefilled sequence");
  if (max_new < 1) return fail(x, SSD_ERR_INVALID_ARG, "max_new must be >= 1");
  if (x->pos_host + max_new + x->kmax + 1 > x->cfg.max_seq)
    return fail(x, SSD_ERR_CAPACITY, "KV cache too small for max_new tokens");
  CK(x, launch_begin_call(x->B, max_new, x->stream));
  CK(x, cudaGraphLaunch(x->gen_x, x->stream));
  if (out_ids_dev)
    CK(x, cudaMemcpyAsync(out_ids_dev, x->B.out_tok, sizeof(int32_t) * max_new,
                          cudaMemcpyDeviceToDevice, x->stream));
  x->async_pending = true;
  return SSD_OK;
}

ssd_status ssd_generate_result(ssd_ctx* x, int32_t* n_rounds, int32_t* n_emitted,
                               ssd_round_trace* traces, int32_t traces_cap) {
  if (!x) return fail(nullptr, SSD_ERR_INVALID_ARG, "ctx is NULL");
  if (!x->async_pending) return fail(x, SSD_ERR_STATE, "no generation in flight");
  Ctl c;
  ssd_status s = read_ctl(x, &c);
  if (s) return s;
  CK(x, cudaStreamSynchronize(x->stream));
  x->async_pending = false;
  x->pos_host = c.pos;
  x->last_rounds = c.round_idx;
  if ((s = check_flag(x, c))) return s;
  if (n_rounds) *n_rounds = c.round_idx;
  if (n_emitted) *n_emitted = c.n_out;
  if (traces && traces_cap > 0) {
    const int n = std::min(traces_cap, c.round_idx);
    CK(x, cudaMemcpy(traces, x->B.traces, sizeof(ssd_round_trace) * n, cudaMemcpyDeviceToHost));
  }
  return SSD_OK;
}

ssd_status ssd_generate(ssd_ctx* x, int32_t max_new, int32_t* out_ids, int32_t* n_out,
                        ssd_round_info* rounds, int32_t rounds_cap, int32_t* n_rounds) {
  if (!x) return fail(nullptr, SSD_ERR_INVALID_ARG, "ctx is NULL");
  if (!out_ids) return fail(x, SSD_ERR_INVALID_ARG, "out_ids is NULL");
  ssd_status s = ssd_generate_async(x, max_new, nullptr);
  if (s) return s;
  CK(x, cudaMemcpyAsync(out_ids, x->B.out_tok, sizeof(int32_t) * max_new, cudaMemcpyDeviceToHost,
                        x->stream));
  std::vector<ssd_round_trace> tr;
  int32_t nr = 0, ne = 0;
  if ((s = ssd_generate_result(x, &nr, &ne, nullptr, 0))) return s;
  if (ne != max_new) return fail(x, SSD_ERR_DEVICE_FLAG, "generation emitted a wrong count");
  if (n_out) *n_out = ne;
  if (n_rounds) *n_rounds = nr;
  if (rounds && rounds_cap > 0) {
    const int n = std::min(rounds_cap, nr);
    tr.resize(n);
    CK(x, cudaMemcpy(tr.data(), x->B.traces, sizeof(ssd_round_trace) * n, cudaMemcpyDeviceToHost));
    for (int i = 0; i < n; ++i) summarize(tr[i], &rounds[i]);
  }
  return SSD_OK;
}

ssd_status ssd_read_traces(ssd_ctx* x, ssd_round_trace* traces, int32_t cap, int32_t* n) {
  if (!x) return fail(nullptr, SSD_ERR_INVALID_ARG, "ctx is NULL");
  if (x->async_pending) return fail(x, SSD_ERR_STATE, "generation in flight");
  const int m = std::min(cap, x->last_rounds);
  if (traces && m > 0)
    CK(x, cudaMemcpy(traces, x->B.traces, sizeof(ssd_round_trace) * m, cudaMemcpyDeviceToHost));
  if (n) *n = x->last_rounds;
  return SSD_OK;
}

const char* ssd_last_error(const ssd_ctx* x) {
  return x ? x->err.c_str() : g_init_error.c_str();
}

void ssd_destroy(ssd_ctx* x) {
  if (!x) return;
  if (x->stream) cudaStreamSynchronize(x->stream);
  destroy_graphs(x);
  if (x->cap) cudaStreamDestroy(x->cap);
  delete x;
}

// ------------------------------------------------------------- ssd_ops.h

ssd_status ssd_forward_exit(ssd_ctx* x, const int32_t* ids, int32_t M, int32_t pos0,
                            int32_t l_exit, int32_t topk, float* logits, ssd_exit_stats* stats) {
  if (!x) return fail(nullptr, SSD_ERR_INVALID_ARG, "ctx is NULL");
  if (!ids || M < 1 || M > kMaxM) return fail(x, SSD_ERR_INVALID_ARG, "M must be in 1..17");
  if (l_exit < 1 || l_exit > x->cfg.n_layers || topk < 1 || topk > kTopK)
    return fail(x, SSD_ERR_INVALID_ARG, "l_exit or topk out of range");
  if (pos0 < 0 || pos0 + M > x->cfg.max_seq) return fail(x, SSD_ERR_CAPACITY, "positions beyond max_seq");
  if (!tokens_ok(ids, M, x->cfg.vocab)) return fail(x, SSD_ERR_INVALID_ARG, "token id out of range");
  if (x->async_pending) return fail(x, SSD_ERR_STATE, "generation in flight");
  CK(x, cudaMemcpyAsync(x->B.pre_tok, ids, sizeof(int32_t) * M, cudaMemcpyHostToDevice, x->stream));
  const RowSel sel = rows_explicit(pos0, M, x->B.pre_tok);
  CK(x, launch_embed(x->D, x->B, x->cfg.dtype, x->embed, sel, true, 0, x->stream));
  CK(x, enqueue_layers(x, 0, l_exit, sel, M, x->stream));
  CK(x, enqueue_head(x, sel, M, topk, logits != nullptr, x->stream));
  std::vector<RowStats> st(M);
  CK(x, cudaMemcpyAsync(st.data(), x->B.stats, sizeof(RowStats) * M, cudaMemcpyDeviceToHost,
                        x->stream));
  if (logits)
    CK(x, cudaMemcpyAsync(logits, x->B.logits, sizeof(float) * (size_t)M * x->cfg.vocab,
                          cudaMemcpyDeviceToHost, x->stream));
  CK(x, cudaStreamSynchronize(x->stream));
  if (stats)
    for (int m = 0; m < M; ++m) {
      ssd_exit_stats& o = stats[m];
      o.argmax = st[m].argmax;
      for (int q = 0; q < kTopK; ++q) {
        o.top_idx[q] = st[m].top_idx[q];
        o.top_logit[q] = st[m].top_logit[q];
      }
      o.zmax = st[m].zmax;
      o.lse = st[m].lse;
      o.entropy = st[m].entropy;
      o.conf_k = st[m].conf_k;
      o.pmax = st[m].pmax;
      o.margin = st[m].margin;
    }
  return SSD_OK;
}

ssd_status ssd_qnet_eval(ssd_ctx* x, const float* states, int32_t n, float* q) {
  if (!x) return fail(nullptr, SSD_ERR_INVALID_ARG, "ctx is NULL");
  if (x->kind != SSD_POLICY_LEDE || !x->have_policy)
    return fail(x, SSD_ERR_STATE, "no LEDE policy set");
  if (x->q_in != 3) return fail(x, SSD_ERR_STATE, "the policy's Q-network does not take 3 inputs");
  const int cap = (int)std::min<size_t>(4096, (size_t)kMaxM * x->cfg.vocab / 5);
  if (!states || !q || n < 1 || n > cap) return fail(x, SSD_ERR_INVALID_ARG, "bad state batch");
  float* ds = x->B.logits;  // scratch: the logits buffer
  float* dq = ds + 3 * (size_t)n;
  CK(x, cudaMemcpyAsync(ds, states, sizeof(float) * 3 * n, cudaMemcpyHostToDevice, x->stream));
  CK(x, launch_qnet_eval(x->B, x->q_hidden, ds, n, dq, x->stream));
  CK(x, cudaMemcpyAsync(q, dq, sizeof(float) * 2 * n, cudaMemcpyDeviceToHost, x->stream));
  CK(x, cudaStreamSynchronize(x->stream));
  return SSD_OK;
}

ssd_status ssd_read_kv(ssd_ctx* x, int32_t layer, int32_t kind, int32_t head, int32_t p0, int32_t n,
                       float* out) {
  if (!x) return fail(nullptr, SSD_ERR_INVALID_ARG, "ctx is NULL");
  if (layer < 0 || layer >= x->cfg.n_layers || kind < 0 || kind > 1 || head < 0 ||
      head >= x->cfg.n_kv_heads || p0 < 0 || n < 1 || p0 + n > x->cfg.max_seq || !out)
    return fail(x, SSD_ERR_INVALID_ARG, "KV slice out of range");
  const int hd = x->cfg.head_dim;
  const int per = (int)std::max<size_t>(1, (size_t)kMaxM * x->cfg.vocab / hd);
  for (int s = 0; s < n; s += per) {
    const int c = std::min(per, n - s);
    CK(x, launch_kv_to_f32(x->D, x->B, x->cfg.dtype, layer, kind, head, p0 + s, c, x->B.logits,
                           x->stream));
    CK(x, cudaMemcpyAsync(out + (size_t)s * hd, x->B.logits, sizeof(float) * c * hd,
                          cudaMemcpyDeviceToHost, x->stream));
    CK(x, cudaStreamSynchronize(x->stream));
  }
  return SSD_OK;
}

ssd_status ssd_read_state(ssd_ctx* x, int32_t* tok, int32_t* pos, float* trace, int32_t cap,
                          int32_t* n_trace) {
  if (!x) return fail(nullptr, SSD_ERR_INVALID_ARG, "ctx is NULL");
  Ctl c;
  ssd_status s = read_ctl(x, &c);
  if (s) return s;
  CK(x, cudaStreamSynchronize(x->stream));
  if (tok) *tok = c.x;
  if (pos) *pos = c.pos;
  const int n = c.trace_n;
  if (n_trace) *n_trace = n;
  if (trace)
    for (int i = 0; i < std::min(cap, n); ++i)
      trace[i] = c.trace[(c.trace_head - n + i + kTraceCap) % kTraceCap];
  return SSD_OK;
}

ssd_status ssd_op_gemv(ssd_ctx* x, int32_t which, int32_t layer, int32_t M, const float* x_dev,
                       float* y_dev, void* stream) {
  if (!x) return fail(nullptr, SSD_ERR_INVALID_ARG, "ctx is NULL");
  if (M < 1 || M > kMaxM || !x_dev || !y_dev) return fail(x, SSD_ERR_INVALID_ARG, "bad M or buffer");
  if (which != 4 && (layer < 0 || layer >= x->cfg.n_layers))
    return fail(x, SSD_ERR_INVALID_ARG, "layer out of range");
  const ssd_model_cfg& c = x->cfg;
  const void* W = nullptr;
  int rows = 0, cols = 0;
  switch (which) {
    case 0: W = x->layers[layer].wqkv; rows = (c.n_heads + 2 * c.n_kv_heads) * c.head_dim; cols = c.d_model; break;
    case 1: W = x->layers[layer].wo; rows = c.d_model; cols = c.n_heads * c.head_dim; break;
    case 2: W = x->layers[layer].wgu; rows = 2 * c.ffn_dim; cols = c.d_model; break;
    case 3: W = x->layers[layer].wdown; rows = c.d_model; cols = c.ffn_dim; break;
    case 4: W = x->lm_head; rows = c.vocab; cols = c.d_model; break;
    default: return fail(x, SSD_ERR_INVALID_ARG, "which must be 0..4");
  }
  cudaStream_t st = stream ? static_cast<cudaStream_t>(stream) : x->stream;
  if (c.dtype == SSD_DTYPE_BF16) {
    const CUtensorMap& wm = which == 4 ? x->wmaps[4 * (size_t)c.n_layers]
                                       : x->wmaps[4 * (size_t)layer + which];
    if (((uintptr_t)x_dev & 15u) || ((size_t)cols * 4) % 16)
      return fail(x, SSD_ERR_INVALID_ARG, "x_dev must be 16-byte aligned");
    CK(x, launch_tile_plain(x->D, x->B, wm, rows, cols, x_dev, M, y_dev, st));
  } else {
    CK(x, launch_gemv_plain(x->D, x->B, c.dtype, W, rows, cols, x_dev, M, y_dev, st));
  }
  return SSD_OK;
}

ssd_status ssd_op_layer(ssd_ctx* x, int32_t kernel, int32_t layer, int32_t M, int32_t pos0,
                        void* stream) {
  if (!x) return fail(nullptr, SSD_ERR_INVALID_ARG, "ctx is NULL");
  if (M < 1 || M > kMaxM || pos0 < 0 || pos0 + M > x->cfg.max_seq)
    return fail(x, SSD_ERR_INVALID_ARG, "M must be in 1..17 with pos0 + M <= max_seq");
  if (kernel < 0 || kernel > 6 || (kernel != 5 && (layer < 0 || layer >= x->cfg.n_layers)))
    return fail(x, SSD_ERR_INVALID_ARG, "kernel must be 0..6 and layer in range");
  if (kernel == 6 && x->cfg.dtype != SSD_DTYPE_BF16)
    return fail(x, SSD_ERR_INVALID_ARG, "the chained kernel is a bf16 kernel");
  cudaStream_t st = stream ? static_cast<cudaStream_t>(stream) : x->stream;
  const RowSel sel = rows_explicit(pos0, M, x->B.pre_tok);
  if (kernel == 5)
    CK(x, enqueue_head(x, sel, M, x->topk, false, st));
  else if (kernel == 6)
    CK(x, launch_tile_chain(x->D, x->B, *tile_maps(x), x->layers[layer],
                            layer + 1 < x->cfg.n_layers ? &x->layers[layer + 1] : nullptr, layer,
                            sel, M, st));
  else
    CK(x, launch_layer_part(x->D, x->B, x->cfg.dtype, x->layers[layer], tile_maps(x), layer,
                            kernel, sel, M, st));
  return SSD_OK;
}

ssd_status ssd_synth_fill(void* dst, int32_t dtype, uint64_t n, uint32_t seed, uint32_t tid,
                          double sigma, void* stream) {
  if (!dst || (dtype != SSD_DTYPE_F32 && dtype != SSD_DTYPE_BF16))
    return fail(nullptr, SSD_ERR_INVALID_ARG, "bad destination or dtype");
  if (n == 0) return SSD_OK;
  cudaError_t e = launch_synth_fill(dst, dtype, n, seed, tid, sigma, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? SSD_OK : cuda_fail(nullptr, "ssd_synth_fill", e);
}

ssd_status ssd_read_probe(const void* src, uint64_t bytes, uint32_t* sink, void* stream) {
  if (!src || !sink || bytes % 16 || ((uintptr_t)src & 15u))
    return fail(nullptr, SSD_ERR_INVALID_ARG, "src/sink NULL, or bytes/src not 16-byte multiples");
  cudaError_t e = launch_read_probe(src, bytes, sink, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? SSD_OK : cuda_fail(nullptr, "ssd_read_probe", e);
}

}  // extern "C"
