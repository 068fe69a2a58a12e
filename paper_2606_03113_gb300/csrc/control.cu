// control.cu -- the device-side control flow of a speculation round: token
// embedding, round set-up, the Q-network decision at a candidate exit layer or
// after a draft, greedy acceptance with KV rollback and the C_trace window.
// Decisions set CUDA-graph conditional handles, so the walk, the drafting loop
// and the generation loop run without returning to the host.
#include <math.h>

#include "../../synth/synth.h"
#include "kernels.h"
#include "pipe.cuh"

namespace ssd {

__device__ __forceinline__ void set_cond(cudaGraphConditionalHandle h, unsigned v) {
  if (h) cudaGraphSetConditional(h, v);
}

__device__ __forceinline__ void trace_push(Ctl* c, float p) {
  c->trace[c->trace_head] = p;
  c->trace_head = (c->trace_head + 1) % kTraceCap;
  if (c->trace_n < kTraceCap) ++c->trace_n;
}

// C_trace = -(1/n) sum log pmax over the n = min(T, count) most recent entries
// (§3.1.1, average trace of token confidence).
__device__ float trace_conf(const Ctl* c, int T) {
  const int n = min(T, c->trace_n);
  if (n <= 0) return 0.f;
  float acc = 0.f;
  for (int i = n; i >= 1; --i) acc += logf(c->trace[(c->trace_head - i + kTraceCap) % kTraceCap]);
  return -acc / (float)n;
}

// ------------------------------------------------- sampled decoding (§4.1)
// Speculative sampling draws drafts from the exit distribution and emitted
// tokens from the full model's, both at temperature T:
// P(v) = exp((z_v - max z) / T) / sum_w exp((z_w - max z) / T).
// Every reduction below runs in a fixed order (contiguous per-thread chunks
// of the vocabulary, chunk sums added in chunk order by one thread), so a
// draw depends only on the logits and the uniform, never on scheduling.
// The uniforms come from synth_sample_uniform keyed by the round's pending
// position: purpose 0 the draw of draft i, 1 the acceptance test of draft i,
// 2 the round's last draw.

constexpr int kSampleThreads = 256;  // block size of k_decide and k_accept

struct SampleSmem {
  float part[kSampleThreads];  // chunk sums, then their exclusive prefix
  float red[kSampleThreads / 32];
  float total, zmax;
  int tok;
  float margin;
};

__device__ __forceinline__ void chunk_of(int V, int& v0, int& v1) {
  const int C = (V + (int)blockDim.x - 1) / (int)blockDim.x;
  v0 = min(V, (int)threadIdx.x * C);
  v1 = min(V, v0 + C);
}

// Maximum of z[0..V) broadcast to the block (exact in any order).
__device__ float block_zmax(const float* __restrict__ z, int V, SampleSmem& sm) {
  int v0, v1;
  chunk_of(V, v0, v1);
  float m = -INFINITY;
  for (int v = v0; v < v1; ++v) m = fmaxf(m, z[v]);
  m = warp_max(m);
  if ((threadIdx.x & 31) == 0) sm.red[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    float r = sm.red[0];
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) r = fmaxf(r, sm.red[w]);
    sm.zmax = r;
  }
  __syncthreads();
  const float r = sm.zmax;
  __syncthreads();
  return r;
}

// Sum of w(v) over [0, V) in the fixed chunk order; leaves the exclusive
// prefix of the chunk sums in sm.part and returns the total to every thread.
template <typename W>
__device__ float block_chunk_sums(int V, W w, SampleSmem& sm) {
  int v0, v1;
  chunk_of(V, v0, v1);
  float acc = 0.f;
  for (int v = v0; v < v1; ++v) acc += w(v);
  sm.part[threadIdx.x] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    float c = 0.f;
    for (int i = 0; i < (int)blockDim.x; ++i) {
      const float x = sm.part[i];
      sm.part[i] = c;
      c += x;
    }
    sm.total = c;
  }
  __syncthreads();
  return sm.total;
}

// Inverse-CDF draw from non-negative weights w(v): with W the total and
// C_v = w(0) + ... + w(v) in token order, the token is the first v with
// C_v > u W; *margin = min(u W - C_{v-1}, C_v - u W) / W.  Returns -1 when W
// is not positive; when rounding leaves u W at or beyond the total, the last
// token of positive weight (margin 0).  Every thread of the block calls it.
template <typename W>
__device__ int block_draw(int V, W w, float u, float* margin, SampleSmem& sm) {
  const float S = block_chunk_sums(V, w, sm);
  int v0, v1;
  chunk_of(V, v0, v1);
  if (threadIdx.x == 0) {
    sm.tok = -1;
    sm.margin = 0.f;
  }
  __syncthreads();
  if (S > 0.f) {
    const float T = u * S;
    const float lo = sm.part[threadIdx.x];
    const float hi = threadIdx.x + 1 < blockDim.x ? sm.part[threadIdx.x + 1] : S;
    // chunk intervals [lo, hi) are disjoint: at most one thread holds T
    if (v1 > v0 && T >= lo && T < hi) {
      float c = lo, mg = 0.f;
      int found = -1, last = -1;
      for (int v = v0; v < v1; ++v) {
        const float wv = w(v);
        const float nx = c + wv;
        if (wv > 0.f) last = v;
        if (nx > T) {
          found = v;
          mg = fminf(T - c, nx - T) / S;
          break;
        }
        c = nx;
      }
      sm.tok = found >= 0 ? found : last;
      sm.margin = found >= 0 ? mg : 0.f;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0 && S > 0.f && sm.tok < 0) {
    int v = V - 1;
    while (v > 0 && !(w(v) > 0.f)) --v;
    sm.tok = v;
    sm.margin = 0.f;
  }
  __syncthreads();
  const int tok = sm.tok;
  if (margin) *margin = sm.margin;
  __syncthreads();
  return tok;
}

struct Tempered {
  const float* z;
  float zmax, temp;
  __device__ float operator()(int v) const { return expf((z[v] - zmax) / temp); }
};

// Weights of the residual max(0, p - q) of one acceptance test.
struct Residual {
  Tempered p, q;
  float sp, sq;  // normalisers of p and q
  __device__ float operator()(int v) const { return fmaxf(p(v) / sp - q(v) / sq, 0.f); }
};

// h[m] = embed[token_m] (fp32) and the row's sum of squares for the first
// RMSNorm.  One block per row.  Optionally sets the drafting switch handle to
// the chosen exit-layer index.
template <typename T>
__global__ void k_embed(Dims D, Bufs B, const T* __restrict__ emb, RowSel sel,
                        cudaGraphConditionalHandle sw) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ float red[32];
  Ctl* c = B.ctl;
  int pos0, M;
  resolve_rows(c, sel, pos0, M);
  const int m = blockIdx.x;
  if (blockIdx.x == 0 && threadIdx.x == 0) set_cond(sw, (unsigned)c->lstar_idx);
  if (m >= M) return;
  int tok;
  switch (sel.mode) {
    case kRowsWalk: tok = c->tok[0]; break;
    case kRowsDraft: tok = c->tok[c->k]; break;
    case kRowsVerify: tok = c->tok[m]; break;
    default: tok = sel.tok[m]; break;
  }
  if (tok < 0 || tok >= D.V) {
    if (threadIdx.x == 0) atomicOr(&c->err, (int)kErrToken);
    tok = 0;
  }
  const T* row = emb + (size_t)tok * D.d;
  float* hr = B.h + (size_t)m * D.d;
  // sums of squares per 256-element part (one warp per part), as the
  // tensor-core kernels' residual epilogues write them
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int c = warp; c < D.ss_nt; c += (int)(blockDim.x >> 5)) {
    float sp = 0.f;
    for (int i = c * 256 + lane; i < min(D.d, c * 256 + 256); i += 32) {
      const float v = Elem<T>::to_f(row[i]);
      sp = fmaf(v, v, sp);
    }
    sp = warp_sum(sp);
    if (lane == 0) B.ss_part[(size_t)c * kMaxM + m] = sp;
  }
  float ss = 0.f;
  for (int i = threadIdx.x; i < D.d; i += blockDim.x) {
    const float v = Elem<T>::to_f(row[i]);
    hr[i] = v;
    ss = fmaf(v, v, ss);
  }
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s += red[w];
    B.ss[m] = s;
  }
}

// Draft cap of the round: min(kmax, tokens still to emit - 1), the static
// length for a static policy, and the KV capacity.
__global__ void k_round_begin(Dims D, Bufs B, cudaGraphConditionalHandle draft_if) {
  pdl_wait();
  pdl_launch_dependents();
  Ctl* c = B.ctl;
  const DevPolicy& P = c->pol;
  const int remaining = c->max_new - c->n_out;
  int kcap = 0;
  if (P.kind != SSD_POLICY_AR) {
    kcap = min(P.kmax, remaining - 1);
    if (P.kind == SSD_POLICY_STATIC) kcap = min(kcap, P.static_k);
    if (P.kind == SSD_POLICY_LEDE && P.fixed_k > 0) kcap = min(kcap, P.fixed_k);
  }
  if (c->pos + kcap + 1 > D.max_seq) {
    atomicOr(&c->err, (int)kErrCapacity);
    kcap = max(0, D.max_seq - c->pos - 1);
  }
  kcap = max(kcap, 0);
  c->kcap = kcap;
  c->k = 0;
  c->lstar = 0;
  c->lstar_idx = 0;
  c->keep = 0;
  c->tok[0] = c->x;
  ssd_round_trace& r = c->cur;
  r.pos = c->pos;
  r.x = c->x;
  r.kcap = kcap;
  r.n_visited = 0;
  r.lstar = 0;
  r.k = 0;
  r.a = 0;
  r.n_emit = 0;
  r.n_q = 0;
  r.sampled = P.temp > 0.f ? 1 : 0;
  for (int i = 0; i < SSD_TRACE_MAXK; ++i) r.accept_margin[i] = 0.f;
  r.fix_margin = 0.f;
  set_cond(draft_if, kcap > 0 ? 1u : 0u);
}

// Final RMSNorm of residual row 0 (the exit hidden state of this decision's
// row), added to the round's pool: the walk restarts the pool at each
// candidate layer (its rows: the pending token only), a draft adds its row
// at l*.  Every thread calls it; returns the pool's row count and leaves the
// Euclidean norm of the pooled mean in *norm.
template <typename T>
__device__ int pool_exit_state(const Dims& D, const Bufs& B, const T* __restrict__ g, bool restart,
                               int n_before, float* red, float* norm) {
  const int tid = threadIdx.x, nw = (int)(blockDim.x >> 5);
  const float* h = B.h;
  float acc = 0.f;
  for (int i = tid; i < D.d; i += blockDim.x) acc = fmaf(h[i], h[i], acc);
  acc = warp_sum(acc);
  if ((tid & 31) == 0) red[tid >> 5] = acc;
  __syncthreads();
  float ss = 0.f;
  for (int w = 0; w < nw; ++w) ss += red[w];
  __syncthreads();
  const float rstd = rsqrtf(ss / (float)D.d + D.eps);
  const int n = restart ? 1 : n_before + 1;
  float nrm = 0.f;
  for (int i = tid; i < D.d; i += blockDim.x) {
    const float hn = h[i] * rstd * Elem<T>::to_f(g[i]);
    const float v = restart ? hn : B.pool[i] + hn;
    B.pool[i] = v;
    const float m = v / (float)n;
    nrm = fmaf(m, m, nrm);
  }
  nrm = warp_sum(nrm);
  if ((tid & 31) == 0) red[tid >> 5] = nrm;
  __syncthreads();
  float t = 0.f;
  for (int w = 0; w < nw; ++w) t += red[w];
  __syncthreads();
  *norm = sqrtf(t);
  return n;
}

// Decision at a candidate exit layer (walk) or after a draft (§3.1.2, §3.3).
// LEDE: Q = W2 relu(W1 s + b1) + b2 with s = (C_k, H, C_trace) of the exit
// distribution in stats[0] (3 inputs), or with d_model + 1 inputs the pooled
// state: the mean over this round's rows so far of the exit hidden state
// after the final RMSNorm, then the exit distribution's max-probability;
// greedy action, ties -> continue (0).
//  walk:  exit (or the last candidate, forced) fixes l* and d_1 = argmax; the
//         action itself says whether to keep drafting; continue opens the
//         next walk segment (next_if).
//  draft: record d_{k+1}; keep drafting while the action is exit and k < kcap.
// Static policies exit at their only candidate and draft to their length.
// Variants (Table 3, §4.1 baselines): LEDE with a fixed draft length uses the
// Q-network only in the walk and drafts to the cap; THRESHOLD keeps drafting
// while the draft's max-probability is >= tau (decision logged as (tau, pmax)).
// A pooled decision is logged with state (pmax, rows pooled, |mean|).
__global__ void k_decide(Dims D, Bufs B, int mode, int cand_idx, int is_last, int layer,
                         const void* final_norm, int dtype,
                         cudaGraphConditionalHandle next_if,
                         cudaGraphConditionalHandle draft_while) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ float s_state[3];
  __shared__ float red0[32], red1[32];
  Ctl* c = B.ctl;
  const DevPolicy& P = c->pol;
  const RowStats& st = B.stats[0];
  const bool lede = P.kind == SSD_POLICY_LEDE;
  const bool thr = P.kind == SSD_POLICY_THRESHOLD;
  const bool use_q = lede && (mode == kDecideWalk || P.fixed_k == 0);
  const bool pooled = lede && P.q_in == D.d + 1;
  const int tid = threadIdx.x;
  float q0 = 0.f, q1 = 0.f;
  int n_pool = 0;
  if (pooled) {
    const int n_before = c->pool_n;
    float nrm = 0.f;
    n_pool = dtype == SSD_DTYPE_BF16
                 ? pool_exit_state(D, B, static_cast<const __nv_bfloat16*>(final_norm),
                                   mode == kDecideWalk, n_before, red0, &nrm)
                 : pool_exit_state(D, B, static_cast<const float*>(final_norm),
                                   mode == kDecideWalk, n_before, red0, &nrm);
    if (tid == 0) {
      c->pool_n = n_pool;
      s_state[0] = st.pmax;
      s_state[1] = (float)n_pool;
      s_state[2] = nrm;
    }
  }
  if (use_q && pooled) {
    // one warp per hidden unit at a time; lanes stride over the inputs
    __syncthreads();
    const int H = P.q_hidden, in = D.d + 1, nw = (int)(blockDim.x >> 5);
    const int warp = tid >> 5, lane = tid & 31;
    const float* W1 = B.qparams;
    const float* b1 = W1 + (size_t)H * in;
    const float* W2 = b1 + H;
    const float* b2 = W2 + 2 * H;
    const float pm = st.pmax, fn = (float)n_pool;
    float a0 = 0.f, a1 = 0.f;
    for (int j = warp; j < H; j += nw) {
      const float* w = W1 + (size_t)j * in;
      float z = 0.f;
      for (int i = lane; i < D.d; i += 32) z = fmaf(w[i], B.pool[i] / fn, z);
      z = warp_sum(z);
      z = fmaf(w[D.d], pm, z) + b1[j];
      const float r = fmaxf(z, 0.f);
      a0 = fmaf(W2[j], r, a0);
      a1 = fmaf(W2[H + j], r, a1);
    }
    if (lane == 0) {
      red0[warp] = a0;
      red1[warp] = a1;
    }
    __syncthreads();
    if (tid == 0) {
      for (int w = 0; w < nw; ++w) {
        q0 += red0[w];
        q1 += red1[w];
      }
      q0 += b2[0];
      q1 += b2[1];
    }
  } else if (use_q) {
    if (tid == 0) {
      s_state[0] = st.conf_k;
      s_state[1] = st.entropy;
      s_state[2] = trace_conf(c, P.trace_T);
    }
    __syncthreads();
    const int H = P.q_hidden;
    const float* W1 = B.qparams;
    const float* b1 = W1 + 3 * H;
    const float* W2 = b1 + H;
    const float* b2 = W2 + 2 * H;
    float a0 = 0.f, a1 = 0.f;
    for (int j = tid; j < H; j += blockDim.x) {
      float z = b1[j];
      z = fmaf(W1[3 * j], s_state[0], z);
      z = fmaf(W1[3 * j + 1], s_state[1], z);
      z = fmaf(W1[3 * j + 2], s_state[2], z);
      const float r = fmaxf(z, 0.f);
      a0 = fmaf(W2[j], r, a0);
      a1 = fmaf(W2[H + j], r, a1);
    }
    a0 = warp_sum(a0);
    a1 = warp_sum(a1);
    if ((tid & 31) == 0) {
      red0[tid >> 5] = a0;
      red1[tid >> 5] = a1;
    }
    __syncthreads();
    if (tid == 0) {
      for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
        q0 += red0[w];
        q1 += red1[w];
      }
      q0 += b2[0];
      q1 += b2[1];
    }
  }
  // Draft token of this decision: argmax of the exit distribution (greedy)
  // or a draw from it at the policy's temperature (sampled decoding).
  __shared__ int s_slot, s_tok;
  __shared__ float s_margin;
  __shared__ SampleSmem sm;
  const bool sampled = P.temp > 0.f;
  if (tid == 0) {
    const int aq = use_q ? (q1 > q0 ? 1 : 0) : 1;
    int slot = -1;
    if (mode == kDecideWalk) {
      if (is_last || aq) slot = 0;
    } else {
      const int k = c->k;
      if (k >= 1 && k < c->kcap && k < kMaxDraft) slot = k;
    }
    s_slot = slot;
    s_tok = st.argmax;
    s_margin = st.margin;
  }
  if (sampled) {
    __syncthreads();
    const int slot = s_slot;
    if (slot >= 0) {
      const float* z = B.logits;  // row 0: this exit's logits
      float* keep = B.draft_logits + (size_t)slot * D.V;
      for (int v = tid; v < D.V; v += blockDim.x) keep[v] = z[v];
      const float zmax = block_zmax(z, D.V, sm);
      const Tempered q{z, zmax, P.temp};
      float mg = 0.f;
      const int d = block_draw(D.V, q, synth_sample_uniform(P.seed, (uint32_t)c->pos, 0u,
                                                            (uint32_t)slot), &mg, sm);
      if (tid == 0) {
        c->dq_zmax[slot] = zmax;
        c->dq_sum[slot] = sm.total;
        s_tok = d;
        s_margin = mg;
      }
    }
  }
  if (tid != 0) return;
  ssd_round_trace& r = c->cur;
  const int aq = use_q ? (q1 > q0 ? 1 : 0) : 1;
  // keep drafting after this decision?
  const int go = thr ? (st.pmax >= P.tau ? 1 : 0) : ((lede && P.fixed_k > 0) ? 1 : aq);
  if ((use_q || thr) && r.n_q < SSD_TRACE_MAXQ) {
    const int i = r.n_q++;
    r.q_action[i] = use_q ? aq : go;
    r.q_val[i][0] = use_q ? q0 : P.tau;
    r.q_val[i][1] = use_q ? q1 : st.pmax;
    r.q_state[i][0] = use_q ? s_state[0] : st.conf_k;
    r.q_state[i][1] = use_q ? s_state[1] : st.entropy;
    r.q_state[i][2] = use_q ? s_state[2] : 0.f;
  }
  const int dtok = s_tok;
  if (st.argmax < 0 || st.argmax >= D.V || dtok < 0 || dtok >= D.V) {
    atomicOr(&c->err, (int)kErrToken);
  }
  if (mode == kDecideWalk) {
    if (r.n_visited < SSD_TRACE_MAXC) r.visited[r.n_visited++] = layer;
    const int act = is_last ? 1 : aq;
    if (act) {
      c->lstar = layer;
      c->lstar_idx = cand_idx;
      c->k = 1;
      c->tok[1] = dtok;
      r.drafts[0] = dtok;
      r.draft_margin[0] = s_margin;
      c->keep = (go && 1 < c->kcap) ? 1 : 0;
      set_cond(next_if, 0u);
    } else {
      set_cond(next_if, 1u);
    }
  } else {
    const int k = c->k;
    if (k < 1 || k >= c->kcap || k >= kMaxDraft) {
      atomicOr(&c->err, (int)kErrControl);
      c->keep = 0;
      set_cond(draft_while, 0u);
      return;
    }
    if (!go && use_q && P.discard) {
      // discard reading: the continue action drops the draft it was taken on
      c->keep = 0;
      set_cond(draft_while, 0u);
      return;
    }
    c->tok[k + 1] = dtok;
    r.drafts[k] = dtok;
    r.draft_margin[k] = s_margin;
    c->k = k + 1;
    c->keep = (go && k + 1 < c->kcap) ? 1 : 0;
    set_cond(draft_while, (unsigned)c->keep);
  }
}

__global__ void k_draft_begin(Bufs B, cudaGraphConditionalHandle draft_while) {
  pdl_wait();
  pdl_launch_dependents();
  set_cond(draft_while, (unsigned)B.ctl->keep);
}

// Verification and acceptance (§4.1: speculative acceptance), one round.
// Greedy (temperature 0): g_i = argmax of verify row i; a = the longest
// prefix with d_i = g_{i-1}; emit d_1..d_a and g_a.
// Sampled (temperature T > 0): p_i = the full model's row i at T, q_i = the
// exit distribution d_i was drawn from; d_1, d_2, ... are tested in turn and
// d_i is kept when r_i q_i(d_i) < p_{i-1}(d_i) (probability min(1, p/q));
// the first rejected test ends the round with a draw from the residual
// max(0, p_{i-1} - q_i) (from p_{i-1} should it carry no mass); when all k
// are kept, the last token is drawn from p_k.  The emitted tokens then
// follow the full model's distribution at T whatever the drafts were.
// Either way the KV length becomes pos + a + 1 (rows beyond it are stale and
// rewritten before any read), the full model's max-probabilities of rows
// 0..a join the C_trace window and the last emitted token is the next
// pending token.
__global__ void k_accept(Dims D, Bufs B, cudaGraphConditionalHandle gen_while) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ SampleSmem sm;
  __shared__ int s_a, s_last;
  Ctl* c = B.ctl;
  ssd_round_trace& r = c->cur;
  const DevPolicy& P = c->pol;
  const bool sampled = P.temp > 0.f;
  const int k = c->k;
  if (sampled) {
    const uint32_t pos = (uint32_t)c->pos;
    const float u_last = synth_sample_uniform(P.seed, pos, 2u, 0u);
    int a = 0, last = -1;
    float fix = 0.f;
    while (a < k && a < kMaxDraft) {
      const float* zp = B.logits + (size_t)a * D.V;
      const float* zq = B.draft_logits + (size_t)a * D.V;
      const float zmp = block_zmax(zp, D.V, sm);
      const Tempered pt{zp, zmp, P.temp};
      const float sp = block_chunk_sums(D.V, pt, sm);
      const Tempered qt{zq, c->dq_zmax[a], P.temp};
      const float sq = c->dq_sum[a];
      const int d = c->tok[a + 1];
      const bool ok_d = d >= 0 && d < D.V && sp > 0.f && sq > 0.f;
      const float pd = ok_d ? pt(d) / sp : 0.f;
      const float qd = ok_d ? qt(d) / sq : 0.f;
      const float rq = synth_sample_uniform(P.seed, pos, 1u, (uint32_t)a) * qd;
      const float den = fmaxf(pd, rq);
      if (threadIdx.x == 0) r.accept_margin[a] = den > 0.f ? (pd - rq) / den : 0.f;
      if (ok_d && rq < pd) {
        ++a;
        continue;
      }
      const Residual res{pt, qt, sp, sq};
      last = block_draw(D.V, res, u_last, &fix, sm);
      if (last < 0) last = block_draw(D.V, pt, u_last, &fix, sm);
      break;
    }
    if (last < 0) {
      const float* zp = B.logits + (size_t)a * D.V;
      const float zmp = block_zmax(zp, D.V, sm);
      last = block_draw(D.V, Tempered{zp, zmp, P.temp}, u_last, &fix, sm);
    }
    if (threadIdx.x == 0) {
      s_a = a;
      s_last = last;
      r.fix_margin = fix;
    }
  }
  if (threadIdx.x != 0) return;
  int a = 0, g;
  if (sampled) {
    a = s_a;
    g = s_last;
    if (g < 0 || g >= D.V) {
      atomicOr(&c->err, (int)kErrToken);
      g = 0;
    }
  } else {
    while (a < k && c->tok[a + 1] == B.stats[a].argmax) ++a;
    g = B.stats[a].argmax;
  }
  for (int i = 0; i <= k; ++i) {
    r.verify_tok[i] = B.stats[i].argmax;
    r.verify_margin[i] = B.stats[i].margin;
    r.verify_pmax[i] = B.stats[i].pmax;
  }
  for (int i = 0; i < a; ++i) r.emitted[i] = c->tok[i + 1];
  r.emitted[a] = g;
  for (int i = 0; i <= a; ++i) {
    if (c->n_out + i < D.max_seq) B.out_tok[c->n_out + i] = r.emitted[i];
    trace_push(c, B.stats[i].pmax);
  }
  r.sampled = sampled ? 1 : 0;
  r.lstar = c->lstar;
  r.k = k;
  r.a = a;
  r.n_emit = a + 1;
  if (c->round_idx < D.max_seq) B.traces[c->round_idx] = r;
  else atomicOr(&c->err, (int)kErrTraceFull);
  c->n_out += a + 1;
  c->pos += a + 1;
  c->x = g;
  c->round_idx += 1;
  set_cond(gen_while, c->n_out < c->max_new ? 1u : 0u);
}

__global__ void k_begin_call(Bufs B, int max_new) {
  pdl_wait();
  pdl_launch_dependents();
  Ctl* c = B.ctl;
  c->max_new = max_new;
  c->n_out = 0;
  c->round_idx = 0;
  c->err = 0;
}

__global__ void k_reset_sequence(Bufs B) {
  pdl_wait();
  pdl_launch_dependents();
  Ctl* c = B.ctl;
  c->pos = 0;
  c->x = 0;
  c->n_out = 0;
  c->round_idx = 0;
  c->trace_n = 0;
  c->trace_head = 0;
  c->err = 0;
}

__global__ void k_trace_push(Bufs B, int first_row, int n_rows) {
  pdl_wait();
  pdl_launch_dependents();
  for (int i = 0; i < n_rows; ++i) trace_push(B.ctl, B.stats[first_row + i].pmax);
}

// Pending token after a prompt: the given token, or (token < 0) the argmax
// of stats[row], or with a sampling temperature a draw from logits row `row`
// keyed by the last prompt position pos - 1 (purpose 2, index 0).
__global__ void k_set_pending(Dims D, Bufs B, int row, int token, int pos) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ SampleSmem sm;
  Ctl* c = B.ctl;
  const DevPolicy& P = c->pol;
  int x = token;
  if (token < 0 && P.temp > 0.f) {
    const float* z = B.logits + (size_t)row * D.V;
    const float zmax = block_zmax(z, D.V, sm);
    x = block_draw(D.V, Tempered{z, zmax, P.temp},
                   synth_sample_uniform(P.seed, (uint32_t)(pos - 1), 2u, 0u), nullptr, sm);
  }
  if (threadIdx.x != 0) return;
  if (token < 0 && !(P.temp > 0.f)) x = B.stats[row].argmax;
  if (x < 0 || x >= D.V) {
    atomicOr(&c->err, (int)kErrToken);
    x = 0;
  }
  c->x = x;
  c->pos = pos;
}

__global__ void k_qnet_eval(Bufs B, int H, const float* __restrict__ states, int n,
                            float* __restrict__ q) {
  pdl_wait();
  pdl_launch_dependents();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const float* W1 = B.qparams;
  const float* b1 = W1 + 3 * H;
  const float* W2 = b1 + H;
  const float* b2 = W2 + 2 * H;
  const float s0 = states[3 * i], s1 = states[3 * i + 1], s2 = states[3 * i + 2];
  float a0 = 0.f, a1 = 0.f;
  for (int j = 0; j < H; ++j) {
    float z = b1[j];
    z = fmaf(W1[3 * j], s0, z);
    z = fmaf(W1[3 * j + 1], s1, z);
    z = fmaf(W1[3 * j + 2], s2, z);
    const float r = fmaxf(z, 0.f);
    a0 = fmaf(W2[j], r, a0);
    a1 = fmaf(W2[H + j], r, a1);
  }
  q[2 * i] = a0 + b2[0];
  q[2 * i + 1] = a1 + b2[1];
}

// Test fixture: seeded synthetic weights (synth.h), grid-stride.
__global__ void k_synth_fill(void* dst, int dtype, uint64_t n, uint32_t seed, uint32_t tid,
                             double sigma) {
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    const float v = synth_weight_f32(seed, tid, i, sigma);
    if (dtype == SSD_DTYPE_BF16)
      static_cast<uint16_t*>(dst)[i] = synth_f32_to_bf16(v);
    else
      static_cast<float*>(dst)[i] = v;
  }
}

template <typename T>
__global__ void k_kv_to_f32(Dims D, Bufs B, int layer, int kind, int head, int p0, int n,
                            float* out) {
  pdl_wait();
  pdl_launch_dependents();
  const T* kv = static_cast<const T*>(B.kv) + (size_t)layer * 2 * D.Hkv * D.max_seq * D.hd +
                ((size_t)(kind * D.Hkv + head) * D.max_seq + p0) * D.hd;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n * D.hd; i += gridDim.x * blockDim.x)
    out[i] = Elem<T>::to_f(kv[i]);
}

// ---------------------------------------------------------------- launchers

cudaError_t launch_embed(const Dims& D, const Bufs& B, int dtype, const void* embed, RowSel sel,
                         bool big, cudaGraphConditionalHandle sw, cudaStream_t st) {
  const int grid = big ? kMaxM : 1;
  if (dtype == SSD_DTYPE_BF16)
      return launch_ex(k_embed<__nv_bfloat16>, dim3(grid), dim3(256), 0, st, D, B,
                     static_cast<const __nv_bfloat16*>(embed), sel, sw);
  return launch_ex(k_embed<float>, dim3(grid), dim3(256), 0, st, D, B,
                   static_cast<const float*>(embed), sel, sw);
}

cudaError_t launch_round_begin(const Dims& D, const Bufs& B, cudaGraphConditionalHandle draft_if,
                               cudaStream_t st) {
  return launch_ex(k_round_begin, dim3(1), dim3(1), 0, st, D, B, draft_if);
}

cudaError_t launch_decide(const Dims& D, const Bufs& B, int mode, int cand_idx, int is_last,
                          int layer, const void* final_norm, int dtype,
                          cudaGraphConditionalHandle next_if,
                          cudaGraphConditionalHandle draft_while, cudaStream_t st) {
  return launch_ex(k_decide, dim3(1), dim3(kSampleThreads), 0, st, D, B, mode, cand_idx, is_last,
                   layer, final_norm, dtype, next_if, draft_while);
}

cudaError_t launch_draft_begin(const Bufs& B, cudaGraphConditionalHandle draft_while,
                               cudaStream_t st) {
  return launch_ex(k_draft_begin, dim3(1), dim3(1), 0, st, B, draft_while);
}

cudaError_t launch_accept(const Dims& D, const Bufs& B, cudaGraphConditionalHandle gen_while,
                          cudaStream_t st) {
  return launch_ex(k_accept, dim3(1), dim3(kSampleThreads), 0, st, D, B, gen_while);
}

cudaError_t launch_begin_call(const Bufs& B, int max_new, cudaStream_t st) {
  return launch_ex(k_begin_call, dim3(1), dim3(1), 0, st, B, max_new);
}

cudaError_t launch_reset_sequence(const Bufs& B, cudaStream_t st) {
  return launch_ex(k_reset_sequence, dim3(1), dim3(1), 0, st, B);
}

cudaError_t launch_trace_push(const Bufs& B, int first_row, int n_rows, cudaStream_t st) {
  return launch_ex(k_trace_push, dim3(1), dim3(1), 0, st, B, first_row, n_rows);
}

cudaError_t launch_set_pending(const Dims& D, const Bufs& B, int stats_row, int token, int pos,
                               cudaStream_t st) {
  return launch_ex(k_set_pending, dim3(1), dim3(kSampleThreads), 0, st, D, B, stats_row, token,
                   pos);
}

cudaError_t launch_qnet_eval(const Bufs& B, int hidden, const float* states, int n, float* q,
                             cudaStream_t st) {
  return launch_ex(k_qnet_eval, dim3((n + 127) / 128), dim3(128), 0, st, B, hidden, states, n, q);
}

cudaError_t launch_synth_fill(void* dst, int dtype, uint64_t n, uint32_t seed, uint32_t tid,
                              double sigma, cudaStream_t st) {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  k_synth_fill<<<sms * 8, 256, 0, st>>>(dst, dtype, n, seed, tid, sigma);
  return cudaGetLastError();
}

cudaError_t launch_kv_to_f32(const Dims& D, const Bufs& B, int dtype, int layer, int kind,
                             int head, int p0, int n, float* out, cudaStream_t st) {
  const int blocks = (n * D.hd + 255) / 256;
  if (dtype == SSD_DTYPE_BF16)
    return launch_ex(k_kv_to_f32<__nv_bfloat16>, dim3(blocks), dim3(256), 0, st, D, B, layer, kind,
                     head, p0, n, out);
  return launch_ex(k_kv_to_f32<float>, dim3(blocks), dim3(256), 0, st, D, B, layer, kind, head, p0,
                   n, out);
}

}  // namespace ssd
