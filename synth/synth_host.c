/*
 * synth_host.c -- host entry points over synth.h for Python callers (prompt
 * ids, Q-network parameters, host-side weight fills and the raw Philox block
 * used by the generator's known-answer tests).  No method arithmetic here.
 */
#include "synth.h"

void synth_philox(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  synth_philox4x32_10(ctr, key, out);
}

void synth_fill_f32(uint32_t seed, uint32_t tid, uint64_t start, uint64_t n, double sigma_scaled,
                    float* out) {
  for (uint64_t i = 0; i < n; ++i) out[i] = synth_weight_f32(seed, tid, start + i, sigma_scaled);
}

void synth_fill_bf16(uint32_t seed, uint32_t tid, uint64_t start, uint64_t n, double sigma_scaled,
                     uint16_t* out) {
  for (uint64_t i = 0; i < n; ++i)
    out[i] = synth_f32_to_bf16(synth_weight_f32(seed, tid, start + i, sigma_scaled));
}

void synth_sample_uniforms(uint32_t seed, uint32_t pos, uint32_t purpose, uint32_t n, float* out) {
  for (uint32_t i = 0; i < n; ++i) out[i] = synth_sample_uniform(seed, pos, purpose, i);
}

void synth_prompt(uint32_t seed, uint64_t n, uint32_t vocab, int32_t* out) {
  for (uint64_t i = 0; i < n; ++i) out[i] = synth_token(seed, i, vocab);
}

/* Q-network parameters, packed W1[hidden][in], b1[hidden], W2[out][hidden],
 * b2[out] (fp32).  Each Linear layer draws weights and biases uniformly in
 * (-1/sqrt(fan_in), 1/sqrt(fan_in)), the usual default initialisation. */
void synth_qnet_params(uint32_t seed, int in_dim, int hidden, int out_dim, float* out) {
  uint64_t o = 0;
  double b1 = 1.0 / __builtin_sqrt((double)in_dim);
  double b2 = 1.0 / __builtin_sqrt((double)hidden);
  for (int i = 0; i < hidden * in_dim; ++i, ++o) out[o] = synth_uniform_sym(seed, SYNTH_TID_QNET, o, b1);
  for (int i = 0; i < hidden; ++i, ++o) out[o] = synth_uniform_sym(seed, SYNTH_TID_QNET, o, b1);
  for (int i = 0; i < out_dim * hidden; ++i, ++o) out[o] = synth_uniform_sym(seed, SYNTH_TID_QNET, o, b2);
  for (int i = 0; i < out_dim; ++i, ++o) out[o] = synth_uniform_sym(seed, SYNTH_TID_QNET, o, b2);
}
