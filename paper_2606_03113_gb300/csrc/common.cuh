// common.cuh -- device-side state and helpers shared by the kernels of the
// self-speculative decoding engine (sm_103a).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/ssd.h"
#include "../../include/ssd_ops.h"

namespace ssd {

constexpr int kMaxM = 17;          // rows of one verify pass: pending token + up to 16 drafts
constexpr int kMaxDraft = 16;
constexpr int kMaxCand = SSD_TRACE_MAXC;
constexpr int kTraceCap = 64;      // C_trace window capacity
constexpr int kTopK = 8;           // max k of the token confidence
constexpr int kWarps = 8;          // warps per block of the matrix-vector kernels
constexpr int kAttnKeys = 64;      // keys per attention split (two per lane)
constexpr int kLayerKernels = 5;   // launches per layer: qkv, attention, o, gate/up, down

// Which rows a kernel works on.  Inside the round graphs they follow the
// device control block; prefill and the op entry points pass them directly.
enum RowMode : int32_t { kRowsExplicit = 0, kRowsWalk = 1, kRowsDraft = 2, kRowsVerify = 3 };
struct RowSel {
  int32_t mode;
  int32_t pos0;  // explicit mode
  int32_t M;     // explicit mode
  const int32_t* tok;  // explicit mode: token ids (device)
};

struct DevPolicy {
  int32_t kind, kmax, static_l, static_k, n_cand, q_hidden, trace_T, topk;
  int32_t cand[kMaxCand];
  int32_t fixed_k;  // LEDE: fixed draft length (0: adaptive)
  int32_t discard;  // LEDE adaptive drafting: drop a draft whose decision is continue
  float tau;        // THRESHOLD: confidence threshold on a draft's max-probability
  int32_t q_in;     // Q-network inputs: 3 (C_k, H, C_trace) or d + 1 (pooled state)
  float temp;       // sampled decoding temperature (0: greedy)
  uint32_t seed;    // sampled decoding seed
};

// Per-row statistics of an exit distribution (mirrors ssd_exit_stats).
struct RowStats {
  int32_t argmax;
  int32_t top_idx[kTopK];
  float top_logit[kTopK];
  float zmax, lse, entropy, conf_k, pmax, margin;
};

// Device control block: the whole sequence / round state lives here so the
// round graphs make every decision on the device.
struct Ctl {
  int32_t x;          // pending token
  int32_t pos;        // its position == KV length
  int32_t max_new;    // tokens to emit in this call
  int32_t n_out;      // tokens emitted so far in this call
  int32_t round_idx;  // rounds completed in this call
  int32_t kcap, k, lstar, lstar_idx, keep, err, pad;
  int32_t tok[kMaxM];  // verify rows: x, d_1..d_k
  int32_t trace_n, trace_head;
  float trace[kTraceCap];  // ring of full-model max-probabilities
  DevPolicy pol;
  float dq_zmax[kMaxDraft], dq_sum[kMaxDraft];  // sampled drafts: max logit, normaliser
  int32_t pool_n;                                // rows in the pooled Q-network state
  ssd_round_trace cur;     // record of the round in flight
};

enum ErrBits : int32_t {
  kErrToken = 1,      // a token id outside [0, vocab)
  kErrCapacity = 2,   // KV capacity would be exceeded
  kErrControl = 4,    // inconsistent round state (l*, k)
  kErrTraceFull = 8,  // more rounds than trace records
  kErrTimeout = 16    // a pipeline wait gave up (see the streamed kernels)
};

__device__ __forceinline__ void resolve_rows(const Ctl* c, const RowSel& s, int& pos0, int& M) {
  switch (s.mode) {
    case kRowsWalk: pos0 = c->pos; M = 1; break;
    case kRowsDraft: pos0 = c->pos + c->k; M = 1; break;
    case kRowsVerify: pos0 = c->pos; M = c->k + 1; break;
    default: pos0 = s.pos0; M = s.M; break;
  }
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// 16-byte streaming load for weights read once per pass: no L1 allocation,
// 256-byte L2 prefetch granule.
__device__ __forceinline__ uint4 ld_stream16(const void* p) {
  uint4 r;
  asm("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4];"
      : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
      : "l"(p));
  return r;
}

template <typename T>
struct Elem;
template <>
struct Elem<float> {
  static constexpr int kPerChunk = 4;
  __device__ static __forceinline__ void unpack(const uint4& u, float* f) {
    f[0] = __uint_as_float(u.x);
    f[1] = __uint_as_float(u.y);
    f[2] = __uint_as_float(u.z);
    f[3] = __uint_as_float(u.w);
  }
  __device__ static __forceinline__ float to_f(float v) { return v; }
  __device__ static __forceinline__ float from_f(float v) { return v; }
};
template <>
struct Elem<__nv_bfloat16> {
  static constexpr int kPerChunk = 8;
  __device__ static __forceinline__ void unpack(const uint4& u, float* f) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      f[2 * i] = __uint_as_float(w[i] << 16);
      f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
  }
  __device__ static __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }
  __device__ static __forceinline__ __nv_bfloat16 from_f(float v) { return __float2bfloat16_rn(v); }
};

// Per-layer weights (device pointers, model dtype).
struct LayerW {
  const void* attn_norm;
  const void* wqkv;
  const void* wo;
  const void* ffn_norm;
  const void* wgu;
  const void* wdown;
  const CUtensorMap* tm[4];  // bf16: tensor maps of wqkv, wo, wgu, wdown (host memory)
};

// Shapes and buffers every kernel may need.
struct Dims {
  int32_t L, d, Hq, Hkv, hd, F, V, max_seq, qd, kvd, nsplit, num_sms, ss_tiles, max_tiles;
  int32_t ss_nt;  // 256-row tiles of a residual row (tensor-core kernels' sum-of-squares parts)
  float eps;
};

struct Bufs {
  Ctl* ctl;
  float* h;          // [kMaxM][d] residual stream
  float* ss;         // [2][kMaxM] sum of squares of h rows: [0] after down/embed, [1] after O
  float* ss_tile;    // [2][2][max blocks][kMaxM] per-block (running, split) partials of ss
  uint32_t* ss_counter;  // [2] block tickets of the residual kernels
  float* ss_part;    // [2][ss_nt][kMaxM] sum of squares of h rows per 256-row tile (bf16
                     // kernels): written by the tile that finishes those rows, summed in
                     // tile order by the RMSNorm that reads them
  float* gpart;      // partial tile sums of blocks sharing a tile: [num_sms][2][32][kMaxM]
                     // (fp32 kernels) or [num_sms][2][2][kMaxM][128] (bf16 tensor-core kernels)
  uint32_t* tile_counter;      // [max tiles] tickets of shared tiles
  float* xq;         // [kMaxM][qd] rotated queries
  float* attn_part;  // [kMaxM][Hq][nsplit][hd] unnormalised partial outputs
  float* attn_ml;    // [kMaxM][Hq][nsplit][2] partial (max, sum)
  uint32_t* attn_counter;  // [Hkv][kMaxM] split tickets of the attention merge
  uint32_t* chain_bar;     // [2] grid-wide phase arrivals / blocks done of the chain kernel
  float* draft_logits;     // [kMaxDraft][V] exit logits of each draft (sampled decoding)
  float* attn_out;   // [kMaxM][qd]
  float* act;        // [kMaxM][F]
  float* logits;     // [kMaxM][V] (written only when requested)
  void* head_part;   // [2][max blocks][kMaxM] per-block (running, split) statistics
  uint32_t* head_counter;  // block ticket of the exit head
  RowStats* stats;   // [kMaxM]
  float2* rope;      // [max_seq][hd/2] (cos, sin)
  void* kv;          // [L][2][Hkv][max_seq][hd]
  float* qparams;    // Q-network parameters
  float* pool;       // [d] pooled Q-network state: sum of the round's final-normed exit rows
  int32_t* out_tok;  // [max_seq] tokens emitted in the current call
  ssd_round_trace* traces;  // [max_seq]
  int32_t* pre_tok;  // [max_seq] prefill / teacher-forced token ids
};

}  // namespace ssd
