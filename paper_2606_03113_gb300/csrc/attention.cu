// attention.cu -- split-K decode attention over the contiguous KV cache for
// 1 (drafting, autoregressive) or k + 1 (verification) query rows, with GQA,
// in one kernel.
//
// Grid = (key splits of kAttnKeys, KV heads).  A block stages its keys and
// values once (fp32 in shared memory) and serves every query head of the KV
// group and every query row with them, so a GQA group of G heads and M rows
// share one KV read.  Row m sits at position pos0 + m and attends causally to
// keys [0, pos0 + m] (the new rows' own keys were appended by the QKV kernel).
//
// Keys before pos0 were written by earlier passes, so a block loads them
// before waiting for the QKV kernel that precedes it (programmatic dependent
// launch) and loads only the M new keys after the wait.  The row window
// (pos0, M) is read before the wait too: every writer of the control block
// runs at least one full dependency before this kernel is launched; it is
// read again after the wait and a mismatch is flagged and handled by
// reloading every key.
//
// Each (row, head, split) writes an unnormalised partial (max, sum, output);
// the last split block to finish a (KV head, row) pair -- a ticket per pair --
// merges its G heads' partials in split order with the log-sum-exp rule, so
// the result does not depend on which block finishes last.  A block that
// finishes several rows merges them all at once (verification passes).
#include <math.h>

#include "kernels.h"
#include "pipe.cuh"

namespace ssd {

namespace {

constexpr int kAK = kAttnKeys;   // keys per split (two per lane)
constexpr int kAThreads = 256;
constexpr int kMergeBatch = 40;  // split partials loaded per round of the merge
constexpr int kMergeBatch4 = 8;  // ... four dimensions each, when merging many rows
constexpr int kAWarps = kAThreads / 32;

// Stages keys [k0, k1) of the split (relative to s0) into shared memory:
// all global loads are issued before any is converted.
template <typename T>
__device__ __forceinline__ void stage_keys(const T* kb, const T* vb, int hd, int k0, int k1,
                                           float* Ks, float* Vs) {
  using E = Elem<T>;
  constexpr int EPC = E::kPerChunk;
  const int cpr = hd / EPC;  // 16-byte chunks per key row
  const int n = (k1 - k0) * cpr;
  constexpr int kUnroll = 4;
  for (int c0 = threadIdx.x; c0 < n; c0 += kAThreads * kUnroll) {
    uint4 ku[kUnroll], vu[kUnroll];
#pragma unroll
    for (int j = 0; j < kUnroll; ++j) {
      const int c = c0 + j * kAThreads;
      if (c < n) {
        const int key = k0 + c / cpr, off = (c % cpr) * EPC;
        ku[j] = __ldg(reinterpret_cast<const uint4*>(kb + (size_t)key * hd + off));
        vu[j] = __ldg(reinterpret_cast<const uint4*>(vb + (size_t)key * hd + off));
      }
    }
#pragma unroll
    for (int j = 0; j < kUnroll; ++j) {
      const int c = c0 + j * kAThreads;
      if (c < n) {
        const int key = k0 + c / cpr, off = (c % cpr) * EPC;
        float kf[EPC], vf[EPC];
        E::unpack(ku[j], kf);
        E::unpack(vu[j], vf);
#pragma unroll
        for (int e = 0; e < EPC; ++e) {
          Ks[key * (hd + 1) + off + e] = kf[e];
          Vs[key * hd + off + e] = vf[e];
        }
      }
    }
  }
}

}  // namespace

template <typename T>
// Three blocks per SM (the shared memory of a split allows three).
__global__ void __launch_bounds__(kAThreads, 3) k_attn(Dims D, Bufs B, int layer, RowSel sel) {
  extern __shared__ float sm[];
  const int split = blockIdx.x, g = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int hd = D.hd;
  const int G = D.Hq / D.Hkv;
  float* Ks = sm;                           // [kAK][hd + 1] (padded: lane-per-key reads)
  float* Vs = Ks + kAK * (hd + 1);          // [kAK][hd]
  float* Ps = Vs + kAK * hd;                // [warps][kAK] probabilities
  int* last_rows = reinterpret_cast<int*>(Ps + kAWarps * kAK);  // [kMaxM] rows this block merges
  __shared__ int s_nlast;

  const T* kv = static_cast<const T*>(B.kv) + (size_t)layer * 2 * D.Hkv * D.max_seq * hd;
  const int s0 = split * kAK;
  const T* kb = kv + ((size_t)g * D.max_seq + s0) * hd;
  const T* vb = kv + ((size_t)(D.Hkv + g) * D.max_seq + s0) * hd;

  // keys written by earlier passes: loaded before the wait
  int pos0, M;
  resolve_rows(B.ctl, sel, pos0, M);
  int nold = min(max(min(pos0, D.max_seq) - s0, 0), kAK);  // clamped: never past the cache
  if (pos0 + M > s0 && nold > 0) stage_keys<T>(kb, vb, hd, 0, nold, Ks, Vs);
  pdl_wait();
  pdl_launch_dependents();
  {
    int p2, m2;
    resolve_rows(B.ctl, sel, p2, m2);
    if (p2 != pos0 || m2 != M) {  // the window moved: reload every key
      if (threadIdx.x == 0) atomicOr(&B.ctl->err, (int)kErrControl);
      pos0 = p2;
      M = m2;
      nold = 0;
    }
  }
  if (s0 > pos0 + M - 1) return;  // beyond every row's causal window
  const int nkeys = min(kAK, pos0 + M - s0);
  if (nkeys > nold) stage_keys<T>(kb, vb, hd, nold, nkeys, Ks, Vs);
  __syncthreads();

  // partial attention of every (row, head) pair of the group over this split
  const float scale = 1.0f / sqrtf((float)hd);
  float* pw = Ps + warp * kAK;
  const int m_first = max(0, s0 - pos0);  // rows that see at least one key here
  const int npairs = G * (M - m_first);
  for (int pi = warp; pi < npairs; pi += kAWarps) {
    const int m = m_first + pi / G, qh = g * G + pi % G;
    const int pos = pos0 + m;
    const float* q = B.xq + (size_t)m * D.qd + (size_t)qh * hd;
    const int ka = lane, kb2 = lane + 32;
    const bool va = s0 + ka <= pos && ka < nkeys, vb2 = s0 + kb2 <= pos && kb2 < nkeys;
    float da = 0.f, db = 0.f;
    const float* kra = Ks + ka * (hd + 1);
    const float* krb = Ks + kb2 * (hd + 1);
    for (int i = 0; i < hd; i += 4) {
      const float4 qv = __ldg(reinterpret_cast<const float4*>(q + i));
      da = fmaf(qv.x, kra[i], da);
      da = fmaf(qv.y, kra[i + 1], da);
      da = fmaf(qv.z, kra[i + 2], da);
      da = fmaf(qv.w, kra[i + 3], da);
      db = fmaf(qv.x, krb[i], db);
      db = fmaf(qv.y, krb[i + 1], db);
      db = fmaf(qv.z, krb[i + 2], db);
      db = fmaf(qv.w, krb[i + 3], db);
    }
    const float sa = va ? da * scale : -INFINITY, sb = vb2 ? db * scale : -INFINITY;
    const float mx = warp_max(fmaxf(sa, sb));
    const float pa = va ? expf(sa - mx) : 0.f, pb = vb2 ? expf(sb - mx) : 0.f;
    const float l = warp_sum(pa + pb);
    pw[ka] = pa;
    pw[kb2] = pb;
    __syncwarp();
    const size_t pidx = ((size_t)m * D.Hq + qh) * D.nsplit + split;
    float* part = B.attn_part + pidx * hd;
    for (int dd = lane; dd < hd; dd += 32) {
      float o = 0.f;
#pragma unroll 8
      for (int s = 0; s < nkeys; ++s) o = fmaf(pw[s], Vs[s * hd + dd], o);
      part[dd] = o;
    }
    if (lane == 0) {
      B.attn_ml[2 * pidx] = mx;
      B.attn_ml[2 * pidx + 1] = l;
    }
    __syncwarp();
  }

  // tickets: the last split of (g, m) merges the group's heads for row m.
  // One thread per row takes the ticket with an acquire-release add after
  // the block barrier, which publishes the block's partials and, for the
  // last split, makes every other split's visible to the whole block.
  if (threadIdx.x == 0) s_nlast = 0;
  __syncthreads();
  if (threadIdx.x < M && threadIdx.x >= m_first) {
    const int m = threadIdx.x;
    const int nsp = (pos0 + m) / kAK + 1;
    uint32_t* cnt = B.attn_counter + (size_t)g * kMaxM + m;
    if (atom_add_acq_rel_gpu(cnt, 1u) == (uint32_t)(nsp - 1)) {
      *cnt = 0u;
      last_rows[atomicAdd(&s_nlast, 1)] = m;
    }
  }
  __syncthreads();
  const int nlast = s_nlast;
  if (nlast == 0) return;
  // merge of every row this block finishes, all rows at once (the key and
  // value buffers are free now): (max, sum) of every (row, head, split) in
  // one round of loads, then the weights e^{m_s - max} and denominators (a
  // warp per (row, head), fixed lane order), then the outputs, each the
  // splits' partials added in split order)
  const int NS = D.nsplit;
  float* Cm = Ks;                                  // [nlast][G][NS] maxima
  float* Cw = Cm + (size_t)nlast * G * NS;         // [nlast][G][NS] sums, then weights
  float* CL = Cw + (size_t)nlast * G * NS;         // [nlast][G] denominators
  const int npr = nlast * G;
  for (int i = threadIdx.x; i < npr * NS; i += kAThreads) {
    const int pr = i / NS, sp = i - pr * NS;
    const int m = last_rows[pr / G], h = pr - (pr / G) * G;
    if (sp > (pos0 + m) / kAK) continue;
    const size_t pidx = ((size_t)m * D.Hq + (size_t)g * G + h) * NS + sp;
    Cm[i] = __ldcg(&B.attn_ml[2 * pidx]);
    Cw[i] = __ldcg(&B.attn_ml[2 * pidx + 1]);
  }
  __syncthreads();
  for (int pr = warp; pr < npr; pr += kAWarps) {
    const int m = last_rows[pr / G];
    const int nsp = (pos0 + m) / kAK + 1;
    const float* cm = Cm + (size_t)pr * NS;
    float* cw = Cw + (size_t)pr * NS;
    float gmax = -INFINITY;
    for (int sp = lane; sp < nsp; sp += 32) gmax = fmaxf(gmax, cm[sp]);
    gmax = warp_max(gmax);
    float L = 0.f;
    for (int sp = lane; sp < nsp; sp += 32) {
      const float l = cw[sp];
      const float w = l > 0.f ? expf(cm[sp] - gmax) : 0.f;
      cw[sp] = w;
      L = fmaf(w, l, L);
    }
    L = warp_sum(L);
    if (lane == 0) CL[pr] = L;
  }
  __syncthreads();
  if (npr * hd <= kAThreads) {
    // few rows: a thread per output, all splits in one round
    for (int o = threadIdx.x; o < npr * hd; o += kAThreads) {
      const int pr = o / hd, dd = o - pr * hd;
      const int m = last_rows[pr / G], h = pr - (pr / G) * G;
      const int nsp = (pos0 + m) / kAK + 1;
      const float* w = Cw + (size_t)pr * NS;
      const float* part = B.attn_part + (((size_t)m * D.Hq + (size_t)g * G + h) * NS) * hd + dd;
      float O = 0.f;
      for (int sc = 0; sc < nsp; sc += kMergeBatch) {
        float pv[kMergeBatch];
#pragma unroll
        for (int j = 0; j < kMergeBatch; ++j)
          pv[j] = sc + j < nsp ? __ldcg(part + (size_t)(sc + j) * hd) : 0.f;
#pragma unroll
        for (int j = 0; j < kMergeBatch; ++j)
          if (sc + j < nsp) O = fmaf(w[sc + j], pv[j], O);
      }
      B.attn_out[(size_t)m * D.qd + (size_t)(g * G + h) * hd + dd] = O / CL[pr];
    }
  } else {
    // many rows (verification): a warp per (row, head), four dimensions per
    // lane; the same sum per output, fewer rounds of loads
    for (int pr = warp; pr < npr; pr += kAWarps) {
      const int m = last_rows[pr / G], h = pr - (pr / G) * G;
      const int nsp = (pos0 + m) / kAK + 1;
      const float* w = Cw + (size_t)pr * NS;
      const float* part = B.attn_part + (((size_t)m * D.Hq + (size_t)g * G + h) * NS) * hd;
      float* out = B.attn_out + (size_t)m * D.qd + (size_t)(g * G + h) * hd;
      for (int d0 = 4 * lane; d0 < hd; d0 += 128) {
        float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int sc = 0; sc < nsp; sc += kMergeBatch4) {
          float4 pv[kMergeBatch4];
#pragma unroll
          for (int j = 0; j < kMergeBatch4; ++j)
            pv[j] = sc + j < nsp
                        ? __ldcg(reinterpret_cast<const float4*>(part + (size_t)(sc + j) * hd + d0))
                        : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
          for (int j = 0; j < kMergeBatch4; ++j)
            if (sc + j < nsp) {
              const float wj = w[sc + j];
              O.x = fmaf(wj, pv[j].x, O.x);
              O.y = fmaf(wj, pv[j].y, O.y);
              O.z = fmaf(wj, pv[j].z, O.z);
              O.w = fmaf(wj, pv[j].w, O.w);
            }
        }
        const float L = CL[pr];
        *reinterpret_cast<float4*>(out + d0) = make_float4(O.x / L, O.y / L, O.z / L, O.w / L);
      }
    }
  }
}

size_t attn_smem(const Dims& D) {
  // keys and values of one split (reused by the merge: maxima, weights and
  // denominators of up to kMaxM rows x G heads x nsplit splits), the warps'
  // probabilities, the rows this block merges
  const int G = D.Hq / D.Hkv;
  const size_t kv = (size_t)kAK * (D.hd + 1) + (size_t)kAK * D.hd;
  const size_t merge = (2 * (size_t)D.nsplit + 1) * kMaxM * G;
  return sizeof(float) * ((kv > merge ? kv : merge) + (size_t)kAWarps * kAK) + sizeof(int) * kMaxM;
}

template <typename T>
static cudaError_t attn_t(const Dims& D, const Bufs& B, int layer, RowSel sel, cudaStream_t st) {
  dim3 grid(D.nsplit, D.Hkv);
  const size_t smem = attn_smem(D);
  if (smem > 48 * 1024) {
    cudaError_t e =
        cudaFuncSetAttribute(k_attn<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
  }
  return launch_ex(k_attn<T>, grid, dim3(kAThreads), smem, st, D, B, layer, sel);
}

cudaError_t launch_attention(const Dims& D, const Bufs& B, int dtype, int layer, RowSel sel,
                             bool /*big*/, cudaStream_t st) {
  if (dtype == SSD_DTYPE_BF16) return attn_t<__nv_bfloat16>(D, B, layer, sel, st);
  return attn_t<float>(D, B, layer, sel, st);
}

}  // namespace ssd
