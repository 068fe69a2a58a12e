/*
 * synth.h -- seeded synthetic inputs for the LEDE self-speculative decoding
 * workloads: model weights, prompt token ids and Q-network parameters.
 *
 * This header is the ONLY code shared by the CPU oracle (oracle/) and the CUDA
 * path (paper_2606_03113_gb300/csrc/).  It holds none of the method's
 * arithmetic: it only maps (seed, tensor id, element index) to a number.
 *
 * Generator: Philox-4x32-10, the counter-based generator of Salmon, Moraes,
 * Dror and Shaw, "Parallel random numbers: as easy as 1, 2, 3" (SC'11),
 * written here from its published definition (two 32x32->64 multiplies per
 * round, Weyl-sequence key schedule, 10 rounds).
 *
 * Weights: the paper's experiments use trained checkpoints; the synthetic
 * stand-in draws each element from N(0, sigma^2) approximately, as an
 * Irwin-Hall sum of four independent 24-bit uniforms, centred and scaled so
 * that its variance is sigma^2 (tails bounded at +-2*sqrt(3)*sigma).  The sum
 * is an exact integer and the scale is one double multiply, so the value is
 * bitwise identical on any IEEE-754 host or device (no transcendental
 * functions, no fused multiply-add opportunity).  bf16 configurations round
 * the fp32 value to bf16 with round-to-nearest-even.
 *
 * Usable from C (gcc), C++ and CUDA (host and device).
 */
#ifndef SYNTH_H
#define SYNTH_H

#include <stdint.h>

#if defined(__CUDACC__)
#define SYNTH_FN static inline __host__ __device__
#else
#define SYNTH_FN static inline
#endif

/* Philox-4x32 round multipliers and key increments (golden ratio and
 * sqrt(3)-1 in 32-bit fixed point), from the SC'11 paper. */
#define SYNTH_PHILOX_M0 0xD2511F53u
#define SYNTH_PHILOX_M1 0xCD9E8D57u
#define SYNTH_PHILOX_W0 0x9E3779B9u
#define SYNTH_PHILOX_W1 0xBB67AE85u

/* Tensor ids: the third counter word, so every tensor has its own stream. */
#define SYNTH_TID_PROMPT 0u
#define SYNTH_TID_EMBED 1u
#define SYNTH_TID_LMHEAD 2u
#define SYNTH_TID_QNET 3u
/* uniforms of sampled decoding: SYNTH_TID_SAMPLE + purpose */
#define SYNTH_TID_SAMPLE 8u
#define SYNTH_TID_LAYER_BASE 16u
/* per layer i: SYNTH_TID_LAYER_BASE + 4*i + one of: */
#define SYNTH_LT_WQKV 0u
#define SYNTH_LT_WO 1u
#define SYNTH_LT_WGU 2u
#define SYNTH_LT_WDOWN 3u

SYNTH_FN uint32_t synth_layer_tid(uint32_t layer, uint32_t which) {
  return SYNTH_TID_LAYER_BASE + 4u * layer + which;
}

/* One Philox-4x32-10 block: out = philox(ctr, key). */
SYNTH_FN void synth_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2],
                                  uint32_t out[4]) {
  uint32_t c0 = ctr_in[0], c1 = ctr_in[1], c2 = ctr_in[2], c3 = ctr_in[3];
  uint32_t k0 = key_in[0], k1 = key_in[1];
  for (int r = 0; r < 10; ++r) {
    if (r > 0) { /* key schedule: bump before every round but the first */
      k0 += SYNTH_PHILOX_W0;
      k1 += SYNTH_PHILOX_W1;
    }
    uint64_t p0 = (uint64_t)SYNTH_PHILOX_M0 * (uint64_t)c0;
    uint64_t p1 = (uint64_t)SYNTH_PHILOX_M1 * (uint64_t)c2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t n0 = hi1 ^ c1 ^ k0;
    uint32_t n1 = lo1;
    uint32_t n2 = hi0 ^ c3 ^ k1;
    uint32_t n3 = lo0;
    c0 = n0; c1 = n1; c2 = n2; c3 = n3;
  }
  out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* The four 32-bit words for element `idx` of tensor `tid` under `seed`. */
SYNTH_FN void synth_block(uint32_t seed, uint32_t tid, uint64_t idx, uint32_t out[4]) {
  uint32_t ctr[4];
  uint32_t key[2];
  ctr[0] = (uint32_t)idx;
  ctr[1] = (uint32_t)(idx >> 32);
  ctr[2] = tid;
  ctr[3] = 0u;
  key[0] = seed;
  key[1] = 0u;
  synth_philox4x32_10(ctr, key, out);
}

/* Approximately N(0, sigma_scaled^2): Irwin-Hall sum of four 24-bit
 * uniforms a_i in [0, 2^24).  n = 2*sum(a_i) - 4*(2^24 - 1) is an exact
 * integer in [-2^26+4, 2^26-4], symmetric about 0, with variance
 * (4/3)(2^48 - 1); so n * sqrt(3) / 2^25 has variance 1 - 2^-48. */
SYNTH_FN float synth_weight_f32(uint32_t seed, uint32_t tid, uint64_t idx, double sigma_scaled) {
  uint32_t w[4];
  synth_block(seed, tid, idx, w);
  int64_t s = (int64_t)(w[0] >> 8) + (int64_t)(w[1] >> 8) + (int64_t)(w[2] >> 8) +
              (int64_t)(w[3] >> 8);
  int64_t n = 2 * s - 4 * (int64_t)0xFFFFFF;
  double c = sigma_scaled * 1.7320508075688772 / 33554432.0; /* sigma*sqrt(3)/2^25 */
  return (float)((double)n * c);
}

/* fp32 -> bf16 bits, round to nearest even (inputs here are finite). */
SYNTH_FN uint16_t synth_f32_to_bf16(float f) {
  union {
    float f;
    uint32_t u;
  } v;
  v.f = f;
  uint32_t lsb = (v.u >> 16) & 1u;
  return (uint16_t)((v.u + 0x7FFFu + lsb) >> 16);
}

SYNTH_FN float synth_bf16_to_f32(uint16_t b) {
  union {
    float f;
    uint32_t u;
  } v;
  v.u = ((uint32_t)b) << 16;
  return v.f;
}

/* Uniform token id in [0, vocab) for prompt position `idx` (multiply-shift
 * of one 32-bit word; the bias is below 2^-32 * vocab). */
SYNTH_FN int32_t synth_token(uint32_t seed, uint64_t idx, uint32_t vocab) {
  uint32_t w[4];
  synth_block(seed, SYNTH_TID_PROMPT, idx, w);
  return (int32_t)(((uint64_t)w[0] * (uint64_t)vocab) >> 32);
}

/* Uniform in (-bound, bound) for Q-network parameter `idx`: a 24-bit uniform
 * a in [0, 2^24) maps to (2a + 1 - 2^24) / 2^24 * bound. */
SYNTH_FN float synth_uniform_sym(uint32_t seed, uint32_t tid, uint64_t idx, double bound) {
  uint32_t w[4];
  synth_block(seed, tid, idx, w);
  int64_t a = (int64_t)(w[0] >> 8);
  double u = (double)(2 * a + 1 - 16777216) / 16777216.0;
  return (float)(u * bound);
}

/* Uniform in (0, 1) for sampled decoding: purpose (0 draw of draft i, 1
 * acceptance test of draft i, 2 draw of the round's last token) of the round
 * whose pending token sits at position `pos`; i < 64.  A 23-bit uniform a
 * maps to (a + 1/2) / 2^23, exact in fp32 (24 significant bits) and fp64. */
SYNTH_FN float synth_sample_uniform(uint32_t seed, uint32_t pos, uint32_t purpose, uint32_t i) {
  uint32_t w[4];
  synth_block(seed, SYNTH_TID_SAMPLE + purpose, (uint64_t)pos * 64u + i, w);
  return ((float)(w[0] >> 9) + 0.5f) * (1.0f / 8388608.0f);
}

#endif /* SYNTH_H */
