// headpart.cuh -- running statistics of exit-head logits (max, sum of
// exponentials, entropy sum, top-k list) and their deterministic merge, used
// by the streamed kernels' exit-head epilogues.
#pragma once

#include <math.h>

#include "kernels.h"

namespace ssd {

__device__ __forceinline__ bool better(float v1, int i1, float v2, int i2) {
  return v1 > v2 || (v1 == v2 && i1 < i2);
}

__device__ inline void part_empty(HeadPart& p) {
  p.mx = -INFINITY;
  p.S = 0.f;
  p.T = 0.f;
#pragma unroll
  for (int q = 0; q < kTopK; ++q) {
    p.tv[q] = -INFINITY;
    p.ti[q] = 0x7fffffff;
  }
}

// Inserts (v, idx) into the descending top-k list with compare-swaps at fixed
// positions (no runtime indexing, so the list stays in registers).
__device__ __forceinline__ void topk_insert(float (&tv)[kTopK], int (&ti)[kTopK], float v, int idx) {
#pragma unroll
  for (int q = 0; q < kTopK; ++q) {
    const bool b = better(v, idx, tv[q], ti[q]);
    const float tvq = tv[q];
    const int tiq = ti[q];
    tv[q] = b ? v : tvq;
    ti[q] = b ? idx : tiq;
    v = b ? tvq : v;
    idx = b ? tiq : idx;
  }
}

__device__ __forceinline__ void cswap(float (&tv)[kTopK], int (&ti)[kTopK], int i, int j) {
  const bool keep = better(tv[i], ti[i], tv[j], ti[j]);
  const float a = tv[i], b = tv[j];
  const int ia = ti[i], ib = ti[j];
  tv[i] = keep ? a : b;
  ti[i] = keep ? ia : ib;
  tv[j] = keep ? b : a;
  ti[j] = keep ? ib : ia;
}

// a <- merge(a, b); symmetric in a and b (max, commutative sums, a total
// order on (value, index)), so both lanes of a shuffle exchange compute the
// same result.  Top-k: bitonic merge of the two sorted lists (elementwise
// best of a[i] and b[k-1-i], then a sorting network of 12 compare-swaps).
__device__ inline void part_merge(HeadPart& a, const HeadPart& b) {
  static_assert(kTopK == 8, "bitonic network written for 8");
  if (b.S > 0.f) {
    if (a.S > 0.f) {
      const float mx = fmaxf(a.mx, b.mx);
      const float ea = expf(a.mx - mx), eb = expf(b.mx - mx);
      const float S = a.S * ea + b.S * eb;
      const float Tt = ea * (a.T + (a.mx - mx) * a.S) + eb * (b.T + (b.mx - mx) * b.S);
      a.mx = mx;
      a.S = S;
      a.T = Tt;
    } else {
      a.mx = b.mx;
      a.S = b.S;
      a.T = b.T;
    }
  }
#pragma unroll
  for (int i = 0; i < kTopK; ++i) {
    const bool keep = better(a.tv[i], a.ti[i], b.tv[kTopK - 1 - i], b.ti[kTopK - 1 - i]);
    a.tv[i] = keep ? a.tv[i] : b.tv[kTopK - 1 - i];
    a.ti[i] = keep ? a.ti[i] : b.ti[kTopK - 1 - i];
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) cswap(a.tv, a.ti, i, i + 4);
  cswap(a.tv, a.ti, 0, 2);
  cswap(a.tv, a.ti, 1, 3);
  cswap(a.tv, a.ti, 4, 6);
  cswap(a.tv, a.ti, 5, 7);
#pragma unroll
  for (int i = 0; i < 8; i += 2) cswap(a.tv, a.ti, i, i + 1);
}

// Adds one logit z of vocabulary row idx.
__device__ inline void part_add(HeadPart& p, float z, int idx) {
  if (!(z > -INFINITY)) return;
  if (p.S > 0.f) {
    const float mx = fmaxf(p.mx, z);
    const float e_old = expf(p.mx - mx), e_new = expf(z - mx);
    p.T = e_old * (p.T + (p.mx - mx) * p.S) + e_new * (z - mx);
    p.S = p.S * e_old + e_new;
    p.mx = mx;
  } else {
    p.mx = z;
    p.S = 1.f;
    p.T = 0.f;
  }
  topk_insert(p.tv, p.ti, z, idx);
}

__device__ inline HeadPart part_shfl(const HeadPart& p, int off) {
  HeadPart q;
  q.mx = __shfl_xor_sync(0xffffffffu, p.mx, off);
  q.S = __shfl_xor_sync(0xffffffffu, p.S, off);
  q.T = __shfl_xor_sync(0xffffffffu, p.T, off);
#pragma unroll
  for (int t = 0; t < kTopK; ++t) {
    q.tv[t] = __shfl_xor_sync(0xffffffffu, p.tv[t], off);
    q.ti[t] = __shfl_xor_sync(0xffffffffu, p.ti[t], off);
  }
  return q;
}

__device__ inline HeadPart part_load_cg(const HeadPart* src) {
  HeadPart q;
  q.mx = __ldcg(&src->mx);
  q.S = __ldcg(&src->S);
  q.T = __ldcg(&src->T);
#pragma unroll
  for (int t = 0; t < kTopK; ++t) {
    q.tv[t] = __ldcg(&src->tv[t]);
    q.ti[t] = __ldcg(&src->ti[t]);
  }
  return q;
}

// Final statistics of one row from its merged partial: argmax (lowest id on
// ties), log-sum-exp, entropy H = log S - T/S, C_k = lse - mean(top-k
// logits), pmax = 1/S.
__device__ inline void write_row_stats(RowStats& o, const HeadPart& f, int topk) {
  const float logS = logf(f.S);
  o.argmax = f.ti[0];
  o.zmax = f.mx;
  o.lse = f.mx + logS;
  o.entropy = logS - f.T / f.S;
  float tsum = 0.f;
#pragma unroll
  for (int q = 0; q < kTopK; ++q) {
    o.top_idx[q] = f.ti[q];
    o.top_logit[q] = f.tv[q];
    if (q < topk) tsum += f.tv[q];
  }
  o.conf_k = o.lse - tsum / (float)topk;
  o.pmax = 1.0f / f.S;
  o.margin = f.tv[0] - f.tv[1];
}

}  // namespace ssd
