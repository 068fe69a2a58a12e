// gemv.cu -- weight-streaming matrix-vector kernels for batch-1 decoding.
//
// Every projection of the decoder (QKV, O, gate/up, down) and the exit LM head
// reads its weight matrix once per pass and multiplies it with M <= 17 input
// rows (1 while drafting, k + 1 while verifying).  At these M the work is
// bound by HBM bandwidth: each warp streams whole rows with 16-byte
// non-allocating loads (several in flight per lane), the input rows come from
// L1/L2, and the row sums are reduced with warp shuffles.  The epilogues are
// fused: RMSNorm of the input (scale applied after the dot product), rotary
// embedding plus KV-cache append, residual add with the sum of squares the next
// RMSNorm needs, SwiGLU, and the first stage of the exit-head statistics.
#include <math.h>

#include <type_traits>

#include "kernels.h"

namespace ssd {

// acc[r][m] = sum_c W_r[c] * x_m[c] * (g[c] if NORM), fully reduced across
// the warp (every lane holds every sum).  K must be a multiple of the chunk.
template <typename T, int MM, int RW, int U, bool NORM>
__device__ __forceinline__ void gemv_rows(const T* const (&wrow)[RW], int K,
                                          const float* __restrict__ x, int xs,
                                          const T* __restrict__ g, int M, float (&acc)[RW][MM]) {
  using E = Elem<T>;
  constexpr int EPC = E::kPerChunk;
  const int nch = K / EPC;
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int r = 0; r < RW; ++r)
#pragma unroll
    for (int m = 0; m < MM; ++m) acc[r][m] = 0.f;

  auto consume = [&](const uint4 (&w)[RW], int c) {
    float wf[RW][EPC];
#pragma unroll
    for (int r = 0; r < RW; ++r) E::unpack(w[r], wf[r]);
    float gv[EPC];
    if (NORM) {
      uint4 gu = __ldg(reinterpret_cast<const uint4*>(g + (size_t)c * EPC));
      E::unpack(gu, gv);
    }
#pragma unroll
    for (int m = 0; m < MM; ++m) {
      if (m < M) {
        float xv[EPC];
        const float4* xp = reinterpret_cast<const float4*>(x + (size_t)m * xs + (size_t)c * EPC);
#pragma unroll
        for (int q = 0; q < EPC / 4; ++q) {
          float4 t = __ldg(xp + q);
          xv[4 * q] = t.x;
          xv[4 * q + 1] = t.y;
          xv[4 * q + 2] = t.z;
          xv[4 * q + 3] = t.w;
        }
        if (NORM) {
#pragma unroll
          for (int e = 0; e < EPC; ++e) xv[e] *= gv[e];
        }
#pragma unroll
        for (int r = 0; r < RW; ++r)
#pragma unroll
          for (int e = 0; e < EPC; ++e) acc[r][m] = fmaf(wf[r][e], xv[e], acc[r][m]);
      }
    }
  };

  int c = lane;
  for (; c + 32 * (U - 1) < nch; c += 32 * U) {
    uint4 w[U][RW];
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int r = 0; r < RW; ++r) w[u][r] = ld_stream16(wrow[r] + (size_t)(c + 32 * u) * EPC);
#pragma unroll
    for (int u = 0; u < U; ++u) consume(w[u], c + 32 * u);
  }
  for (; c < nch; c += 32) {
    uint4 w[RW];
#pragma unroll
    for (int r = 0; r < RW; ++r) w[r] = ld_stream16(wrow[r] + (size_t)c * EPC);
    consume(w, c);
  }
#pragma unroll
  for (int r = 0; r < RW; ++r)
#pragma unroll
    for (int m = 0; m < MM; ++m)
      if (m < M) acc[r][m] = warp_sum(acc[r][m]);
}

// RMSNorm scale 1/sqrt(mean(x^2) + eps) from the stored sum of squares.
__device__ __forceinline__ float norm_scale(float ss, int d, float eps) {
  return 1.0f / sqrtf(ss / (float)d + eps);
}

constexpr int kUnroll = 4;

// ---------------------------------------------------------------- QKV
// Unit = two rows.  Query/key units pair element i with i + hd/2 of one head
// so the rotary embedding is applied in registers; value units are two
// consecutive rows.  Rotated queries go to xq, keys and values to the cache.
template <typename T, int MM>
__global__ void __launch_bounds__(kWarps * 32) k_qkv(Dims D, Bufs B, LayerW W, int layer,
                                                      RowSel sel) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int pos0, M;
  resolve_rows(B.ctl, sel, pos0, M);
  const int half = D.hd / 2;
  const int n_rope = (D.Hq + D.Hkv) * half;
  const int n_units = n_rope + D.Hkv * half;
  const int unit = blockIdx.x * kWarps + warp;
  if (unit >= n_units) return;
  const bool is_v = unit >= n_rope;
  int head = 0, i = 0, r0, r1;
  if (!is_v) {
    head = unit / half;
    i = unit - head * half;
    r0 = head * D.hd + i;
    r1 = r0 + half;
  } else {
    r0 = (D.Hq + D.Hkv) * D.hd + 2 * (unit - n_rope);
    r1 = r0 + 1;
  }
  const T* Wm = static_cast<const T*>(W.wqkv);
  const T* const wr[2] = {Wm + (size_t)r0 * D.d, Wm + (size_t)r1 * D.d};
  float acc[2][MM];
  gemv_rows<T, MM, 2, kUnroll, true>(wr, D.d, B.h, D.d, static_cast<const T*>(W.attn_norm), M,
                                     acc);
  T* kv = static_cast<T*>(B.kv) + (size_t)layer * 2 * D.Hkv * D.max_seq * D.hd;
#pragma unroll
  for (int m = 0; m < MM; ++m) {
    if (m < M && lane == (m & 31)) {
      const float rs = norm_scale(B.ss[m], D.d, D.eps);
      const float y0 = acc[0][m] * rs, y1 = acc[1][m] * rs;
      const int pos = pos0 + m;
      if (!is_v) {
        const float2 cs = B.rope[(size_t)pos * half + i];
        const float o0 = y0 * cs.x - y1 * cs.y;
        const float o1 = y1 * cs.x + y0 * cs.y;
        if (head < D.Hq) {
          float* q = B.xq + (size_t)m * D.qd + (size_t)head * D.hd;
          q[i] = o0;
          q[i + half] = o1;
        } else {
          T* kr = kv + ((size_t)(head - D.Hq) * D.max_seq + pos) * D.hd;
          kr[i] = Elem<T>::from_f(o0);
          kr[i + half] = Elem<T>::from_f(o1);
        }
      } else {
        const int rv = r0 - (D.Hq + D.Hkv) * D.hd;
        const int g = rv / D.hd, j = rv - g * D.hd;
        T* vr = kv + ((size_t)(D.Hkv + g) * D.max_seq + pos) * D.hd;
        vr[j] = Elem<T>::from_f(y0);
        vr[j + 1] = Elem<T>::from_f(y1);
      }
    }
  }
}

// ------------------------------------------------------- residual (O, down)
// h[m][row] += (W x_m)[row].  The next RMSNorm needs sum(h_m^2): each block
// writes the partial of its rows, and the last block to finish adds the
// partials in block order, so the result does not depend on scheduling.
template <typename T, int MM>
__global__ void __launch_bounds__(kWarps * 32) k_resid(Dims D, Bufs B, const T* __restrict__ W,
                                                        int K, const float* __restrict__ x,
                                                        int which, RowSel sel) {
  __shared__ float red[kWarps][kMaxM];
  __shared__ int is_last;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int pos0, M;
  resolve_rows(B.ctl, sel, pos0, M);
  const int unit = blockIdx.x * kWarps + warp;
  const bool valid = unit < D.d / 2;
  if (lane < kMaxM) red[warp][lane] = 0.f;
  if (valid) {
    const int r0 = 2 * unit;
    const T* const wr[2] = {W + (size_t)r0 * K, W + (size_t)(r0 + 1) * K};
    float acc[2][MM];
    gemv_rows<T, MM, 2, kUnroll, false>(wr, K, x, K, nullptr, M, acc);
#pragma unroll
    for (int m = 0; m < MM; ++m) {
      if (m < M && lane == (m & 31)) {
        float* hr = B.h + (size_t)m * D.d + r0;
        const float a = hr[0] + acc[0][m];
        const float b = hr[1] + acc[1][m];
        hr[0] = a;
        hr[1] = b;
        red[warp][m] = a * a + b * b;
      }
    }
  }
  __syncthreads();
  const int nblk = gridDim.x;
  float* part = B.ss_part + (size_t)which * kMaxM * D.res_blocks;
  if (threadIdx.x < M) {
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) s += red[w][threadIdx.x];
    part[(size_t)threadIdx.x * D.res_blocks + blockIdx.x] = s;
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) is_last = atomicAdd(&B.ss_counter[which], 1u) == (unsigned)(nblk - 1);
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  if (threadIdx.x < M) {
    float s = 0.f;
    for (int b = 0; b < nblk; ++b) s += __ldcg(&part[(size_t)threadIdx.x * D.res_blocks + b]);
    B.ss[which * kMaxM + threadIdx.x] = s;
  }
  if (threadIdx.x == 0) B.ss_counter[which] = 0u;
}

// ------------------------------------------------------------- gate / up
// Unit j = rows j (gate) and F + j (up): act = silu(gate) * up.
template <typename T, int MM>
__global__ void __launch_bounds__(kWarps * 32) k_gate_up(Dims D, Bufs B, LayerW W, RowSel sel) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  int pos0, M;
  resolve_rows(B.ctl, sel, pos0, M);
  const int j = blockIdx.x * kWarps + warp;
  if (j >= D.F) return;
  const T* Wm = static_cast<const T*>(W.wgu);
  const T* const wr[2] = {Wm + (size_t)j * D.d, Wm + (size_t)(D.F + j) * D.d};
  float acc[2][MM];
  gemv_rows<T, MM, 2, kUnroll, true>(wr, D.d, B.h, D.d, static_cast<const T*>(W.ffn_norm), M, acc);
#pragma unroll
  for (int m = 0; m < MM; ++m) {
    if (m < M && lane == (m & 31)) {
      const float rs = norm_scale(B.ss[kMaxM + m], D.d, D.eps);
      const float gt = acc[0][m] * rs, up = acc[1][m] * rs;
      B.act[(size_t)m * D.F + j] = gt / (1.0f + expf(-gt)) * up;
    }
  }
}

// ---------------------------------------------------------------- exit head
__device__ __forceinline__ bool better(float v1, int i1, float v2, int i2) {
  return v1 > v2 || (v1 == v2 && i1 < i2);
}

__device__ void part_empty(HeadPart& p) {
  p.mx = -INFINITY;
  p.S = 0.f;
  p.T = 0.f;
#pragma unroll
  for (int q = 0; q < kTopK; ++q) {
    p.tv[q] = -INFINITY;
    p.ti[q] = 0x7fffffff;
  }
}

__device__ void part_insert_topk(HeadPart& p, float v, int idx) {
  if (!better(v, idx, p.tv[kTopK - 1], p.ti[kTopK - 1])) return;
  int q = kTopK - 1;
  while (q > 0 && better(v, idx, p.tv[q - 1], p.ti[q - 1])) {
    p.tv[q] = p.tv[q - 1];
    p.ti[q] = p.ti[q - 1];
    --q;
  }
  p.tv[q] = v;
  p.ti[q] = idx;
}

// a <- merge(a, b): max, rescaled sums and the top-k lists.
__device__ void part_merge(HeadPart& a, const HeadPart& b) {
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
  HeadPart out;
  int ia = 0, ib = 0;
#pragma unroll
  for (int q = 0; q < kTopK; ++q) {
    if (better(a.tv[ia], a.ti[ia], b.tv[ib], b.ti[ib])) {
      out.tv[q] = a.tv[ia];
      out.ti[q] = a.ti[ia];
      ++ia;
    } else {
      out.tv[q] = b.tv[ib];
      out.ti[q] = b.ti[ib];
      ++ib;
    }
  }
#pragma unroll
  for (int q = 0; q < kTopK; ++q) {
    a.tv[q] = out.tv[q];
    a.ti[q] = out.ti[q];
  }
}

// Logits z = W_lm RMSNorm_final(h) for 16 vocabulary rows per block; each
// block writes the statistics partial of its rows for every input row, and
// the last block to finish merges all partials into RowStats.
template <typename T, int MM>
__global__ void __launch_bounds__(kWarps * 32) k_head(Dims D, Bufs B, const T* __restrict__ Wlm,
                                                       const T* __restrict__ gnorm, int topk,
                                                       int write_logits, RowSel sel) {
  __shared__ float zs[kMaxM][kHeadRowsPerBlock];
  __shared__ HeadPart red[kWarps * 32];
  __shared__ int is_last;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, tid = threadIdx.x;
  int pos0, M;
  resolve_rows(B.ctl, sel, pos0, M);
  const int r0 = blockIdx.x * kHeadRowsPerBlock + 2 * warp;
  if (r0 < D.V) {  // V is even, so r0 + 1 < V as well
    const T* const wr[2] = {Wlm + (size_t)r0 * D.d, Wlm + (size_t)(r0 + 1) * D.d};
    float acc[2][MM];
    gemv_rows<T, MM, 2, kUnroll, true>(wr, D.d, B.h, D.d, gnorm, M, acc);
#pragma unroll
    for (int m = 0; m < MM; ++m) {
      if (m < M && lane == (m & 31)) {
        const float rs = norm_scale(B.ss[m], D.d, D.eps);
        const float z0 = acc[0][m] * rs, z1 = acc[1][m] * rs;
        zs[m][2 * warp] = z0;
        zs[m][2 * warp + 1] = z1;
        if (write_logits) {
          B.logits[(size_t)m * D.V + r0] = z0;
          B.logits[(size_t)m * D.V + r0 + 1] = z1;
        }
      }
    }
  } else {
    if (lane < kMaxM) {
      zs[lane][2 * warp] = -INFINITY;
      zs[lane][2 * warp + 1] = -INFINITY;
    }
  }
  __syncthreads();
  HeadPart* parts = static_cast<HeadPart*>(B.head_part);
  const int nblk = gridDim.x;
  if (tid < M) {
    HeadPart p;
    part_empty(p);
    const int base = blockIdx.x * kHeadRowsPerBlock;
    float mx = -INFINITY;
    for (int q = 0; q < kHeadRowsPerBlock; ++q) mx = fmaxf(mx, zs[tid][q]);
    if (mx > -INFINITY) {
      float S = 0.f, Tt = 0.f;
      for (int q = 0; q < kHeadRowsPerBlock; ++q) {
        const float z = zs[tid][q];
        if (z > -INFINITY) {
          const float e = expf(z - mx);
          S += e;
          Tt += e * (z - mx);
          part_insert_topk(p, z, base + q);
        }
      }
      p.mx = mx;
      p.S = S;
      p.T = Tt;
    }
    parts[(size_t)tid * nblk + blockIdx.x] = p;
  }
  __threadfence();
  __syncthreads();
  if (tid == 0) is_last = (atomicAdd(B.head_counter, 1u) == (unsigned)(nblk - 1));
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  for (int m = 0; m < M; ++m) {
    HeadPart acc;
    part_empty(acc);
    for (int b = tid; b < nblk; b += blockDim.x) {
      HeadPart q;
      const HeadPart* src = parts + (size_t)m * nblk + b;
      q.mx = __ldcg(&src->mx);
      q.S = __ldcg(&src->S);
      q.T = __ldcg(&src->T);
#pragma unroll
      for (int t = 0; t < kTopK; ++t) {
        q.tv[t] = __ldcg(&src->tv[t]);
        q.ti[t] = __ldcg(&src->ti[t]);
      }
      part_merge(acc, q);
    }
    red[tid] = acc;
    __syncthreads();
    for (int s = blockDim.x / 2; s > 0; s >>= 1) {
      if (tid < s) part_merge(red[tid], red[tid + s]);
      __syncthreads();
    }
    if (tid == 0) {
      const HeadPart& f = red[0];
      RowStats& o = B.stats[m];
      const float logS = logf(f.S);
      o.argmax = f.ti[0];
      o.zmax = f.mx;
      o.lse = f.mx + logS;
      o.entropy = logS - f.T / f.S;
      float tsum = 0.f;
      for (int q = 0; q < kTopK; ++q) {
        o.top_idx[q] = f.ti[q];
        o.top_logit[q] = f.tv[q];
        if (q < topk) tsum += f.tv[q];
      }
      o.conf_k = o.lse - tsum / (float)topk;
      o.pmax = 1.0f / f.S;
      o.margin = f.tv[0] - f.tv[1];
    }
    __syncthreads();
  }
  if (tid == 0) *B.head_counter = 0u;
}

// --------------------------------------------------------------- plain GEMV
template <typename T, int MM>
__global__ void __launch_bounds__(kWarps * 32) k_gemv_plain(const T* __restrict__ W, int rows,
                                                             int cols, const float* __restrict__ x,
                                                             int M, float* __restrict__ y) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int unit = blockIdx.x * kWarps + warp;
  if (2 * unit >= rows) return;
  const int r0 = 2 * unit;
  const T* const wr[2] = {W + (size_t)r0 * cols, W + (size_t)(r0 + 1) * cols};
  float acc[2][MM];
  gemv_rows<T, MM, 2, kUnroll, false>(wr, cols, x, cols, nullptr, M, acc);
#pragma unroll
  for (int m = 0; m < MM; ++m) {
    if (m < M && lane == (m & 31)) {
      y[(size_t)m * rows + r0] = acc[0][m];
      y[(size_t)m * rows + r0 + 1] = acc[1][m];
    }
  }
}

// ----------------------------------------------------------------- probe
__global__ void k_read_probe(const uint4* __restrict__ src, uint64_t n16, uint32_t* sink) {
  uint32_t acc = 0;
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  for (; i + 3 * stride < n16; i += 4 * stride) {
    const uint4 a = ld_stream16(src + i), b = ld_stream16(src + i + stride);
    const uint4 c = ld_stream16(src + i + 2 * stride), d = ld_stream16(src + i + 3 * stride);
    acc ^= a.x ^ a.y ^ a.z ^ a.w ^ b.x ^ b.y ^ b.z ^ b.w ^ c.x ^ c.y ^ c.z ^ c.w ^ d.x ^ d.y ^ d.z ^ d.w;
  }
  for (; i < n16; i += stride) {
    const uint4 a = ld_stream16(src + i);
    acc ^= a.x ^ a.y ^ a.z ^ a.w;
  }
  if (acc == 0x9E3779B9u) atomicXor(sink, acc);  // keeps the loads live
}

// -------------------------------------------------------------- launchers

// Attention launchers live in attention.cu.
cudaError_t launch_attention(const Dims& D, const Bufs& B, int dtype, int layer, RowSel sel,
                             bool big, cudaStream_t st);

template <typename T, int MM>
static cudaError_t layer_t(const Dims& D, const Bufs& B, const LayerW& w, int layer, RowSel sel,
                           cudaStream_t st);

template <typename T, int MM>
static cudaError_t head_t(const Dims& D, const Bufs& B, const void* lm, const void* fn, int topk,
                          bool logits, RowSel sel, cudaStream_t st) {
  k_head<T, MM><<<head_blocks(D.V), kWarps * 32, 0, st>>>(
      D, B, static_cast<const T*>(lm), static_cast<const T*>(fn), topk, logits ? 1 : 0, sel);
  return cudaGetLastError();
}

cudaError_t launch_head(const Dims& D, const Bufs& B, int dtype, const void* lm_head,
                        const void* final_norm, int topk, bool write_logits, RowSel sel, bool big,
                        cudaStream_t st) {
  if (dtype == SSD_DTYPE_BF16)
    return big ? head_t<__nv_bfloat16, kMaxM>(D, B, lm_head, final_norm, topk, write_logits, sel, st)
               : head_t<__nv_bfloat16, 1>(D, B, lm_head, final_norm, topk, write_logits, sel, st);
  return big ? head_t<float, kMaxM>(D, B, lm_head, final_norm, topk, write_logits, sel, st)
             : head_t<float, 1>(D, B, lm_head, final_norm, topk, write_logits, sel, st);
}

template <typename T, int MM>
static cudaError_t part_t(const Dims& D, const Bufs& B, const LayerW& w, int layer, int part,
                          RowSel sel, cudaStream_t st) {
  const int threads = kWarps * 32;
  switch (part) {
    case 0: {
      const int qkv_units = (D.Hq + 2 * D.Hkv) * D.hd / 2;
      k_qkv<T, MM><<<(qkv_units + kWarps - 1) / kWarps, threads, 0, st>>>(D, B, w, layer, sel);
      break;
    }
    case 1:
      return launch_attention(D, B, std::is_same<T, float>::value ? SSD_DTYPE_F32 : SSD_DTYPE_BF16,
                              layer, sel, MM > 1, st);
    case 2:
      k_resid<T, MM><<<D.res_blocks, threads, 0, st>>>(D, B, static_cast<const T*>(w.wo), D.qd,
                                                       B.attn_out, 1, sel);
      break;
    case 3:
      k_gate_up<T, MM><<<(D.F + kWarps - 1) / kWarps, threads, 0, st>>>(D, B, w, sel);
      break;
    case 4:
      k_resid<T, MM><<<D.res_blocks, threads, 0, st>>>(D, B, static_cast<const T*>(w.wdown), D.F,
                                                       B.act, 0, sel);
      break;
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

template <typename T, int MM>
static cudaError_t layer_t(const Dims& D, const Bufs& B, const LayerW& w, int layer, RowSel sel,
                           cudaStream_t st) {
  for (int part = 0; part < kLayerKernels - 1; ++part) {
    cudaError_t e = part_t<T, MM>(D, B, w, layer, part, sel, st);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_layer_part(const Dims& D, const Bufs& B, int dtype, const LayerW& w, int layer,
                              int part, RowSel sel, bool big, cudaStream_t st) {
  if (dtype == SSD_DTYPE_BF16)
    return big ? part_t<__nv_bfloat16, kMaxM>(D, B, w, layer, part, sel, st)
               : part_t<__nv_bfloat16, 1>(D, B, w, layer, part, sel, st);
  return big ? part_t<float, kMaxM>(D, B, w, layer, part, sel, st)
             : part_t<float, 1>(D, B, w, layer, part, sel, st);
}

cudaError_t launch_layer(const Dims& D, const Bufs& B, int dtype, const LayerW& w, int layer,
                         RowSel sel, bool big, cudaStream_t st) {
  if (dtype == SSD_DTYPE_BF16)
    return big ? layer_t<__nv_bfloat16, kMaxM>(D, B, w, layer, sel, st)
               : layer_t<__nv_bfloat16, 1>(D, B, w, layer, sel, st);
  return big ? layer_t<float, kMaxM>(D, B, w, layer, sel, st)
             : layer_t<float, 1>(D, B, w, layer, sel, st);
}

template <typename T, int MM>
static void plain_t(const void* W, int rows, int cols, const float* x, int M, float* y,
                    cudaStream_t st) {
  const int units = rows / 2;
  k_gemv_plain<T, MM><<<(units + kWarps - 1) / kWarps, kWarps * 32, 0, st>>>(
      static_cast<const T*>(W), rows, cols, x, M, y);
}

cudaError_t launch_gemv_plain(int dtype, const void* W, int rows, int cols, const float* x, int M,
                              float* y, cudaStream_t st) {
  if (dtype == SSD_DTYPE_BF16) {
    if (M == 1) plain_t<__nv_bfloat16, 1>(W, rows, cols, x, M, y, st);
    else plain_t<__nv_bfloat16, kMaxM>(W, rows, cols, x, M, y, st);
  } else {
    if (M == 1) plain_t<float, 1>(W, rows, cols, x, M, y, st);
    else plain_t<float, kMaxM>(W, rows, cols, x, M, y, st);
  }
  return cudaGetLastError();
}

cudaError_t launch_read_probe(const void* src, uint64_t bytes, uint32_t* sink, cudaStream_t st) {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  k_read_probe<<<sms * 4, 512, 0, st>>>(static_cast<const uint4*>(src), bytes / 16, sink);
  return cudaGetLastError();
}

}  // namespace ssd
