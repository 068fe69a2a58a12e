// attention.cu -- split-K decode attention over the contiguous KV cache for
// 1 (drafting, AR) or k + 1 (verification) query rows, with GQA.
//
// Grid = (key splits of 32, KV heads).  A block stages its 32 keys and values
// once (converted to fp32 in shared memory) and serves every query head of
// the KV group and every query row with them, so a GQA group of G heads and M
// rows share one KV read.  Row m sits at position pos0 + m and attends
// causally to keys [0, pos0 + m] (the new rows' own keys were appended by the
// QKV kernel).  Each (row, head, split) writes an unnormalised partial
// (max, sum, output); the combine kernel merges splits with the log-sum-exp
// rule.
#include <math.h>

#include "kernels.h"
#include "pipe.cuh"

namespace ssd {

template <typename T, int MM>
__global__ void __launch_bounds__(kWarps * 32) k_attn(Dims D, Bufs B, int layer, RowSel sel) {
  extern __shared__ float sm[];
  const int split = blockIdx.x, g = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_wait();
  pdl_launch_dependents();
  int pos0, M;
  resolve_rows(B.ctl, sel, pos0, M);
  const int s0 = split * kAttnChunk;
  if (s0 > pos0 + M - 1) return;  // beyond every row's causal window
  const int hd = D.hd;
  float* Ks = sm;                         // [32][hd + 1] (padded: lane-per-key reads)
  float* Vs = Ks + kAttnChunk * (hd + 1); // [32][hd]
  float* Ps = Vs + kAttnChunk * hd;       // [kWarps][32]
  using E = Elem<T>;
  constexpr int EPC = E::kPerChunk;
  const T* kv = static_cast<const T*>(B.kv) + (size_t)layer * 2 * D.Hkv * D.max_seq * hd;
  const T* kb = kv + ((size_t)g * D.max_seq + s0) * hd;
  const T* vb = kv + ((size_t)(D.Hkv + g) * D.max_seq + s0) * hd;
  const int cpr = hd / EPC;  // chunks per key row
  const int nkeys = min(kAttnChunk, pos0 + M - s0);
  for (int c = threadIdx.x; c < kAttnChunk * cpr; c += blockDim.x) {
    const int key = c / cpr, off = (c - key * cpr) * EPC;
    float kf[EPC], vf[EPC];
    if (key < nkeys) {
      E::unpack(__ldg(reinterpret_cast<const uint4*>(kb + (size_t)key * hd + off)), kf);
      E::unpack(__ldg(reinterpret_cast<const uint4*>(vb + (size_t)key * hd + off)), vf);
    } else {
#pragma unroll
      for (int e = 0; e < EPC; ++e) kf[e] = vf[e] = 0.f;
    }
#pragma unroll
    for (int e = 0; e < EPC; ++e) {
      Ks[key * (hd + 1) + off + e] = kf[e];
      Vs[key * hd + off + e] = vf[e];
    }
  }
  __syncthreads();
  const int G = D.Hq / D.Hkv;
  const float scale = 1.0f / sqrtf((float)hd);
  float* pw = Ps + warp * kAttnChunk;
  for (int gm = warp; gm < G * M; gm += kWarps) {
    const int m = gm / G, qh = g * G + (gm - m * G);
    const int pos = pos0 + m;
    const float* q = B.xq + (size_t)m * D.qd + (size_t)qh * hd;
    const int key = s0 + lane;
    const bool valid = key <= pos;
    float sc = -INFINITY;
    if (valid) {
      float dot = 0.f;
      const float* kr = Ks + lane * (hd + 1);
      for (int i = 0; i < hd; i += 4) {
        const float4 qv = __ldg(reinterpret_cast<const float4*>(q + i));
        dot = fmaf(qv.x, kr[i], dot);
        dot = fmaf(qv.y, kr[i + 1], dot);
        dot = fmaf(qv.z, kr[i + 2], dot);
        dot = fmaf(qv.w, kr[i + 3], dot);
      }
      sc = dot * scale;
    }
    const float mx = warp_max(sc);
    const float p = valid ? expf(sc - mx) : 0.f;
    const float l = warp_sum(p);
    pw[lane] = p;
    __syncwarp();
    const size_t pidx = ((size_t)m * D.Hq + qh) * D.nsplit + split;
    float* part = B.attn_part + pidx * hd;
    for (int dd = lane; dd < hd; dd += 32) {
      float o = 0.f;
#pragma unroll 8
      for (int s = 0; s < kAttnChunk; ++s) o = fmaf(pw[s], Vs[s * hd + dd], o);
      part[dd] = o;
    }
    if (lane == 0) {
      B.attn_ml[2 * pidx] = mx;
      B.attn_ml[2 * pidx + 1] = l;
    }
    __syncwarp();
  }
}

// out[m][qh*hd + d] = sum_s e^{m_s - M} o_s[d] / sum_s e^{m_s - M} l_s over the
// splits that hold keys of row m.
template <int MM>
__global__ void k_attn_combine(Dims D, Bufs B, RowSel sel) {
  const int qh = blockIdx.x, m = blockIdx.y;
  pdl_wait();
  pdl_launch_dependents();
  int pos0, M;
  resolve_rows(B.ctl, sel, pos0, M);
  if (m >= M) return;
  const int nsp = (pos0 + m) / kAttnChunk + 1;
  const size_t base = ((size_t)m * D.Hq + qh) * D.nsplit;
  float gmax = -INFINITY;
  for (int s = 0; s < nsp; ++s) gmax = fmaxf(gmax, B.attn_ml[2 * (base + s)]);
  for (int dd = threadIdx.x; dd < D.hd; dd += blockDim.x) {
    float L = 0.f, O = 0.f;
    for (int s = 0; s < nsp; ++s) {
      const float l = B.attn_ml[2 * (base + s) + 1];
      if (l > 0.f) {
        const float w = expf(B.attn_ml[2 * (base + s)] - gmax);
        L = fmaf(w, l, L);
        O = fmaf(w, B.attn_part[(base + s) * D.hd + dd], O);
      }
    }
    B.attn_out[(size_t)m * D.qd + (size_t)qh * D.hd + dd] = O / L;
  }
}

static size_t attn_smem(int hd) {
  return sizeof(float) * ((size_t)kAttnChunk * (hd + 1) + (size_t)kAttnChunk * hd +
                          (size_t)kWarps * kAttnChunk);
}

template <typename T, int MM>
static cudaError_t attn_t(const Dims& D, const Bufs& B, int layer, RowSel sel, cudaStream_t st) {
  dim3 grid(D.nsplit, D.Hkv);
  const size_t smem = attn_smem(D.hd);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(k_attn<T, MM>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
  }
  cudaError_t e = launch_ex(k_attn<T, MM>, grid, dim3(kWarps * 32), smem, st, D, B, layer, sel);
  if (e != cudaSuccess) return e;
  return launch_ex(k_attn_combine<MM>, dim3(D.Hq, MM), dim3(D.hd < 128 ? D.hd : 128), 0, st, D, B,
                   sel);
}

cudaError_t launch_attention(const Dims& D, const Bufs& B, int dtype, int layer, RowSel sel,
                             bool big, cudaStream_t st) {
  if (dtype == SSD_DTYPE_BF16)
    return big ? attn_t<__nv_bfloat16, kMaxM>(D, B, layer, sel, st)
               : attn_t<__nv_bfloat16, 1>(D, B, layer, sel, st);
  return big ? attn_t<float, kMaxM>(D, B, layer, sel, st) : attn_t<float, 1>(D, B, layer, sel, st);
}

}  // namespace ssd
