/*
 * ssd_ops.h -- finer-grained entry points of the same library (libssd.so),
 * for parity checks against the CPU oracle, kernel timing and test fixtures.
 * Conventions as in ssd.h (status codes, caller-owned memory, the context's
 * stream unless a stream is given).
 */
#ifndef SSD_OPS_H
#define SSD_OPS_H

#include "ssd.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Statistics of one early-exit distribution P^(l) = softmax(z) (§3.1.1):
 * conf_k = C_k = -(1/k) sum of the log-probabilities of the k most probable
 * tokens; entropy = H^l; pmax = max probability (the per-step term of
 * C_trace); argmax = greedy token (lowest id on ties); margin = top-1 minus
 * top-2 logit. */
typedef struct {
  int32_t argmax;
  int32_t top_idx[8];
  float top_logit[8];
  float zmax, lse, entropy, conf_k, pmax, margin;
} ssd_exit_stats;

/* Teacher-forced partial forward (§3.1.1: P_t^(l) from the hidden state at
 * layer l): ids[0..M) (host) at positions pos0..pos0+M-1 run through layers
 * 1..l_exit, writing their KV (positions below pos0 must already hold KV for
 * all l_exit layers), then the shared final RMSNorm and LM head over all M
 * rows.  logits (host, optional) receives [M][vocab] fp32; stats (host,
 * optional) receives M records computed with top-k = topk (1..8).  1 <= M <= 17.
 * Does not change the pending token or the trace.  Synchronises. */
ssd_status ssd_forward_exit(ssd_ctx* ctx, const int32_t* ids, int32_t M, int32_t pos0,
                            int32_t l_exit, int32_t topk, float* logits, ssd_exit_stats* stats);

/* The Q-network of the current LEDE policy on n states (host [n][3] fp32:
 * C_k, H, C_trace) -> q (host [n][2]: Q(continue), Q(exit)).  SSD_ERR_STATE
 * when the policy's network takes the pooled state (qnet_in = d_model + 1).
 * Synchronises. */
ssd_status ssd_qnet_eval(ssd_ctx* ctx, const float* states, int32_t n, float* q);

/* KV-cache rows as fp32: layer (0-based), kind 0 = K (after RoPE) or 1 = V,
 * KV head, positions [p0, p0 + n) -> out (host) [n][head_dim]. */
ssd_status ssd_read_kv(ssd_ctx* ctx, int32_t layer, int32_t kind, int32_t head, int32_t p0,
                       int32_t n, float* out);

/* Sequence state: pending token, its position (= KV length) and the C_trace
 * window (host out[cap], oldest first; *n_trace entries). */
ssd_status ssd_read_state(ssd_ctx* ctx, int32_t* x, int32_t* pos, float* trace, int32_t cap,
                          int32_t* n_trace);

/* One launch of the weight-streaming matrix-vector kernel on the weights of
 * layer `layer`: which = 0 wqkv, 1 wo, 2 w_gate_up, 3 w_down, 4 lm_head
 * (layer ignored).  y[m][r] = sum_c W[r][c] x[m][c] for m < M (1 <= M <= 17),
 * x_dev [M][cols] and y_dev [M][rows] fp32 device buffers.  Enqueued on
 * `stream` (NULL = the context's stream); no synchronisation. */
ssd_status ssd_op_gemv(ssd_ctx* ctx, int32_t which, int32_t layer, int32_t M, const float* x_dev,
                       float* y_dev, void* stream);

/* One launch of one hot-path kernel of layer `layer` exactly as the round
 * graphs launch it, on M rows at positions pos0..pos0+M-1 of the context's
 * own buffers: kernel = 0 QKV (+RoPE, KV append), 1 attention (split-K with
 * the split merge in the same kernel), 2 O projection (+residual), 3 gate/up (+RMSNorm, SwiGLU),
 * 4 down projection (+residual), 5 exit head (final RMSNorm, LM head,
 * statistics; layer ignored), 6 (bf16) the chained launch the layer passes
 * use: O projection, gate/up and down of `layer` and the QKV of layer + 1
 * (when there is one) as the phases of one persistent kernel.  It overwrites the activations and the KV rows
 * at those positions: for timing and profiling, not inside a generation.
 * Needs pos0 + M <= max_seq.  Enqueued on `stream` (NULL = the context's). */
ssd_status ssd_op_layer(ssd_ctx* ctx, int32_t kernel, int32_t layer, int32_t M, int32_t pos0,
                        void* stream);

/* Allocation-free form of ssd_op_gemv (the paper has no counterpart: this is
 * an interface for callers that cannot allocate device memory, e.g. code that
 * runs while a CUDA graph is being captured, where cudaMalloc is not a
 * capturable operation, or a host framework that owns the device's memory
 * pool and allows no other allocations).  Computes y[m][r] = sum_c W[r][c]
 * x[m][c] for m < M exactly as ssd_op_gemv, without a context: W (device,
 * rows x cols, dtype, 16-byte aligned rows), x_dev [M][cols] and y_dev
 * [M][rows] fp32 (device) are the caller's; the kernel's scratch is a fixed
 * static device array inside libssd.so (about 1.1 MB, held on every device
 * that uses it until the process exits).
 * Limits: 1 <= M <= 17 and rows <= 131072 (SSD_ERR_CAPACITY beyond), cols *
 * element size a multiple of 16 (SSD_ERR_INVALID_ARG otherwise).
 * Device-side failure: the kernel's pipeline waits are bounded; one that gives
 * up sets an error word (SSD error bits, 16 = a wait timed out) in the static
 * array and leaves y_dev undefined.  With err_dev (device, one int32, may be
 * NULL) the call enqueues, after the kernel, a copy of that word into
 * *err_dev: 0 once the stream has reached it means y_dev holds the product.
 * The returned status covers only the host-side checks and the launch.
 * The first call on a device looks up the array's device address and sets
 * kernel attributes; make that first call before any stream capture.  Every
 * call clears the scratch's tickets and error word on `stream` and shares the
 * one array, so calls that overlap on the GPU (other streams, other threads)
 * race.  Enqueued on `stream`; no synchronisation; allocates nothing. */
ssd_status ssd_gemv_noalloc(const void* W, int32_t dtype, int32_t rows, int32_t cols,
                            const float* x_dev, int32_t M, float* y_dev, int32_t* err_dev,
                            void* stream);

/* Test fixture: fills dst (device, n elements of dtype) with the seeded
 * synthetic weights of tensor `tid` (see synth/synth.h): element i is
 * synth_weight_f32(seed, tid, i, sigma), rounded to bf16 for SSD_DTYPE_BF16.
 * Enqueued on `stream`; no synchronisation. */
ssd_status ssd_synth_fill(void* dst, int32_t dtype, uint64_t n, uint32_t seed, uint32_t tid,
                          double sigma, void* stream);

/* Measurement fixture: reads `bytes` (multiple of 16) from src (device) with
 * the same streaming loads as the weight kernels and writes one checksum
 * word to sink (device).  Enqueued on `stream`. */
ssd_status ssd_read_probe(const void* src, uint64_t bytes, uint32_t* sink, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SSD_OPS_H */
