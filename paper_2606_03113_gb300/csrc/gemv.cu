// gemv.cu -- weight-streaming matrix-vector kernels for batch-1 decoding.
//
// Every projection of the decoder (QKV, O, gate/up, down) and the exit LM head
// reads its weight matrix once per pass and multiplies it with M <= 17 input
// rows (1 while drafting, k + 1 while verifying): at these M the work is bound
// by HBM bandwidth.  Design (one kernel per matrix, persistent grid of one
// block per SM):
//  - the matrix is cut into units of 32 rows x 512 bytes; the units, in
//    (row tile, K) order, are split evenly over the blocks ("stream-K"), so
//    every SM streams the same number of bytes whatever the matrix shape, and
//    a block copies up to four consecutive units of a tile as one stage;
//  - a producer warp copies each stage into a 3-deep shared-memory ring with
//    1-D bulk async copies (one copy of up to 2 KB per row: smaller copies
//    starve the copy engine; evict-first in L2), synchronised by
//    mbarriers; its copies do not wait for the previous kernel (programmatic
//    dependent launch), so the weight stream of one kernel overlaps the tail
//    of the previous one;
//  - eight consumer warps read the stage from shared memory (four rows per
//    warp, so each input load serves four rows; 16 bytes per lane per
//    512-byte step), multiply with the fp32 input rows (from L1/L2) and
//    accumulate; a 32-row tile is reduced with warp shuffles;
//  - a tile split between two blocks is finished by whichever block completes
//    its share last (per-tile ticket), which adds the partial sums in block
//    order, so results do not depend on scheduling;
//  - fused epilogues: RMSNorm of the input (scale applied after the dot
//    product), rotary embedding + KV-cache append, residual add with the sum
//    of squares the next RMSNorm needs, SwiGLU, and the exit-head statistics
//    (max, argmax, top-k, log-sum-exp, entropy) merged in a fixed tree.
#include <math.h>

#include <mutex>
#include <type_traits>

#include "headpart.cuh"
#include "kernels.h"
#include "pipe.cuh"

namespace ssd {

constexpr int kRT = 32;             // rows per tile
constexpr int kRowBytes = 2048;     // bytes of one row per stage (4 units)
constexpr int kUnit = 512;          // bytes of one row per assignment unit
constexpr int kNS = 3;              // ring depth
constexpr int kCWarps = 8;          // consumer warps
constexpr int kCThreads = kCWarps * 32;
constexpr int kThreads = kCThreads + 32;  // + producer warp
constexpr int kRowStride = kRowBytes + 16;  // padded row pitch in shared memory:
                                            // rows of an 8x8 ldmatrix land on distinct banks
constexpr int kStageBytes = kRT * kRowStride;
constexpr int kNB = (kMaxM + 7) / 8;        // 8-token column blocks of the tensor-core path
constexpr int kMaxBlocksDev = 512;  // upper bound on the grid (partial slots per block)

enum RowMap : int { kMapLinear = 0, kMapQKV = 1, kMapGateUp = 2 };

struct Geom {
  int N, K;          // rows, columns (elements)
  int nks;           // 512-byte units per row (per tile)
  int ntiles;
  long long T;       // units (tiles x nks)
  int P;             // blocks
  int row_bytes;     // K * elt
  int map;           // RowMap
  int elt;           // element size in bytes
};

struct StreamArgs {
  Geom g;
  Dims D;
  Bufs B;
  const void* W;
  const void* gnorm;     // RMSNorm weights of the input, or null
  const float* x;        // [M][K] fp32 input rows
  int ss_in;             // which sum-of-squares buffer scales the input (0, 1; -1: none)
  RowSel sel;
};

__host__ __device__ inline long long stage_start(const Geom& g, int b) {
  return g.T * (long long)b / g.P;
}

__device__ inline int block_of_stage(const Geom& g, long long s) {
  int b = (int)(s * g.P / g.T);
  if (b >= g.P) b = g.P - 1;
  while (b + 1 < g.P && stage_start(g, b + 1) <= s) ++b;
  while (b > 0 && stage_start(g, b) > s) --b;
  return b;
}

// Global row of local row r (0..31) of a tile, or -1 past the end.  QKV
// tiles of a query/key head hold rows i..i+15 and their rotary partners
// i+hd/2..i+hd/2+15; gate/up tiles hold gate rows j..j+15 and up rows
// F+j..F+j+15.
__device__ inline int map_row(const Geom& g, const Dims& D, int tile, int r) {
  if (g.map == kMapQKV) {
    const int tpp = D.hd / 32;             // tiles per query/key head
    const int tqk = (D.Hq + D.Hkv) * tpp;
    if (tile < tqk) {
      const int h = tile / tpp, sub = tile - h * tpp;
      return h * D.hd + (r < 16 ? sub * 16 + r : D.hd / 2 + sub * 16 + (r - 16));
    }
    const int row = (D.Hq + D.Hkv) * D.hd + (tile - tqk) * kRT + r;
    return row < g.N ? row : -1;
  }
  if (g.map == kMapGateUp) {
    const int F = g.N / 2;
    const int j = tile * 16 + (r & 15);
    if (j >= F) return -1;
    return r < 16 ? j : F + j;
  }
  const int row = tile * kRT + r;
  return row < g.N ? row : -1;
}

// Local rows handled by consumer warp w: w, w+8, w+16, w+24; (w, w+16) and
// (w+8, w+24) are the pairs the QKV and gate/up epilogues combine.

struct SmemLayout {
  static constexpr size_t ring = 0;
  static constexpr size_t bars = ring + (size_t)kNS * kStageBytes;
  static constexpr size_t rs = bars + 2 * kNS * sizeof(uint64_t);
  static constexpr size_t flag = rs + sizeof(float) * 32;
  static constexpr size_t scratch = flag + 64;  // cross-warp combine buffer
  static constexpr size_t red = scratch + (size_t)(kCWarps + 1) * kMaxM * sizeof(HeadPart);
  template <int MM>
  static constexpr size_t total() {  // + tensor-core partial sums [4 K-quarters][32][8 kNB]
    return red + sizeof(float) * 4 * kRT * 8 * kNB;
  }
};

// Block b owns the exit-head / norm partial of the tile it starts and shares
// with the next block(s) ("split slot"), if its last tile is such a tile.
__device__ inline bool has_split_slot(const Geom& g, int b) {
  const long long sb = stage_start(g, b), se = stage_start(g, b + 1);
  if (se <= sb) return false;
  const long long t = (se - 1) / g.nks;
  if ((t + 1) * g.nks <= se) return false;  // the last tile ends inside the block
  return t * g.nks >= sb;                   // and it starts inside the block
}

struct Shared {
  float* rs;       // [MM] input RMSNorm scale
  int* flag;
  void* scratch;   // [kCWarps][MM] floats or HeadParts
};

// ------------------------------------------------------------ epilogues
//
// pair(): rows (w, w+8) of a tile, one input row m per lane (lane < M), with
// the dot products v0, v1.  Kernels with a running result (residual norm sums,
// exit-head statistics) keep per-lane state; finish() combines it once per
// block and the last block reduces the blocks in a fixed order.

struct NoState {};

// y[m][row] = sum (the plain product, for kernel-level parity and timing).
struct EpiPlain {
  using State = NoState;
  float* y;
  __device__ void init(State&) const {}
  __device__ void pair(const StreamArgs& a, int tile, int w, int m, int, float, float v0, float v1,
                       State&) const {
    const int r0 = map_row(a.g, a.D, tile, w), r1 = map_row(a.g, a.D, tile, w + 16);
    if (r0 >= 0) y[(size_t)m * a.g.N + r0] = v0;
    if (r1 >= 0) y[(size_t)m * a.g.N + r1] = v1;
  }
  __device__ void split_done(const StreamArgs&, int, State&, const Shared&, int, int) const {}
  __device__ void finish(const StreamArgs&, State&, const Shared&, int, int) const {}
};

// Rotary embedding of query/key pairs (element i with i + hd/2, angle
// pos * theta^(-2i/hd) from the table); queries to xq, keys and values to
// the KV cache of `layer` at positions pos0 + m.
template <typename T>
struct EpiQKV {
  using State = NoState;
  int layer;
  __device__ void init(State&) const {}
  __device__ void pair(const StreamArgs& a, int tile, int w, int m, int pos0, float rs, float v0,
                       float v1, State&) const {
    const Dims& D = a.D;
    const int tqk = (D.Hq + D.Hkv) * (D.hd / 32);
    T* kv = static_cast<T*>(a.B.kv) + (size_t)layer * 2 * D.Hkv * D.max_seq * D.hd;
    const int pos = pos0 + m;
    const float y0 = v0 * rs, y1 = v1 * rs;
    const int r0 = map_row(a.g, D, tile, w);
    if (tile < tqk) {
      const int half = D.hd / 2;
      const int head = r0 / D.hd, i = r0 - head * D.hd;
      const float2 cs = a.B.rope[(size_t)pos * half + i];
      const float o0 = y0 * cs.x - y1 * cs.y;
      const float o1 = y1 * cs.x + y0 * cs.y;
      if (head < D.Hq) {
        float* q = a.B.xq + (size_t)m * D.qd + (size_t)head * D.hd;
        q[i] = o0;
        q[i + half] = o1;
      } else {
        T* kr = kv + ((size_t)(head - D.Hq) * D.max_seq + pos) * D.hd;
        kr[i] = Elem<T>::from_f(o0);
        kr[i + half] = Elem<T>::from_f(o1);
      }
    } else {
      const int r1 = map_row(a.g, D, tile, w + 16);
      const int vb = (D.Hq + D.Hkv) * D.hd;
      if (r0 >= 0) {
        const int g = (r0 - vb) / D.hd, j = (r0 - vb) - g * D.hd;
        kv[((size_t)(D.Hkv + g) * D.max_seq + pos) * D.hd + j] = Elem<T>::from_f(y0);
      }
      if (r1 >= 0) {
        const int g = (r1 - vb) / D.hd, j = (r1 - vb) - g * D.hd;
        kv[((size_t)(D.Hkv + g) * D.max_seq + pos) * D.hd + j] = Elem<T>::from_f(y1);
      }
    }
  }
  __device__ void split_done(const StreamArgs&, int, State&, const Shared&, int, int) const {}
  __device__ void finish(const StreamArgs&, State&, const Shared&, int, int) const {}
};

// act[m][j] = silu(gate_j) * up_j.
struct EpiGateUp {
  using State = NoState;
  __device__ void init(State&) const {}
  __device__ void pair(const StreamArgs& a, int tile, int w, int m, int, float rs, float v0,
                       float v1, State&) const {
    const int j = map_row(a.g, a.D, tile, w);
    if (j < 0) return;
    const float gt = v0 * rs, up = v1 * rs;
    a.B.act[(size_t)m * a.D.F + j] = gt / (1.0f + expf(-gt)) * up;
  }
  __device__ void split_done(const StreamArgs&, int, State&, const Shared&, int, int) const {}
  __device__ void finish(const StreamArgs&, State&, const Shared&, int, int) const {}
};

// Combines the per-lane float state of the 8 warps (lane m of each) in warp
// order; every consumer thread calls it; returns the sum in thread m < M.
__device__ inline float combine_warps(float v, const Shared& sh, int tid, int M) {
  float* buf = static_cast<float*>(sh.scratch);
  const int warp = tid >> 5, lane = tid & 31;
  if (lane < M) buf[warp * kMaxM + lane] = v;
  named_sync(1, kCThreads);
  float s = 0.f;
  if (tid < M)
    for (int w = 0; w < kCWarps; ++w) s += buf[w * kMaxM + tid];
  named_sync(1, kCThreads);
  return s;
}

// h[m][row] += y, and sum(h_m^2) over the rows for the next RMSNorm.  Per
// block: one running sum (complete tiles) and one split-slot sum (the tile it
// starts and shares); the last block adds them in block order.
struct EpiResid {
  struct State {
    float ss;
  };
  int which;  // sum-of-squares buffer written (0 after down, 1 after O)
  __device__ void init(State& s) const { s.ss = 0.f; }
  __device__ void pair(const StreamArgs& a, int tile, int w, int m, int, float, float v0, float v1,
                       State& st) const {
    const int r0 = map_row(a.g, a.D, tile, w), r1 = map_row(a.g, a.D, tile, w + 16);
    float* hm = a.B.h + (size_t)m * a.D.d;
    if (r0 >= 0) {
      const float h = hm[r0] + v0;
      hm[r0] = h;
      st.ss = fmaf(h, h, st.ss);
    }
    if (r1 >= 0) {
      const float h = hm[r1] + v1;
      hm[r1] = h;
      st.ss = fmaf(h, h, st.ss);
    }
  }
  __device__ float* slots(const StreamArgs& a) const {
    return a.B.ss_tile + (size_t)which * 2 * kMaxBlocksDev * kMaxM;
  }
  __device__ void split_done(const StreamArgs& a, int b0, State& st, const Shared& sh, int tid,
                             int M) const {
    const float s = combine_warps(st.ss, sh, tid, M);
    if (tid < M) slots(a)[((size_t)kMaxBlocksDev + b0) * kMaxM + tid] = s;
  }
  __device__ void finish(const StreamArgs& a, State& st, const Shared& sh, int tid, int M) const {
    const float s = combine_warps(st.ss, sh, tid, M);
    float* sl = slots(a);
    if (tid < M) sl[(size_t)blockIdx.x * kMaxM + tid] = s;
    __threadfence();
    named_sync(1, kCThreads);
    if (tid == 0) *sh.flag = atomicAdd(&a.B.ss_counter[which], 1u) == (unsigned)(a.g.P - 1);
    named_sync(1, kCThreads);
    if (!*sh.flag) return;
    __threadfence();
    // every thread loads its slots first, then a fixed reduction tree
    float* buf = static_cast<float*>(sh.scratch);
    const int warp = tid >> 5, lane = tid & 31;
    for (int m = 0; m < M; ++m) {
      float v = 0.f;
      for (int b = tid; b < a.g.P; b += kCThreads) {
        v += __ldcg(&sl[(size_t)b * kMaxM + m]);
        if (has_split_slot(a.g, b)) v += __ldcg(&sl[((size_t)kMaxBlocksDev + b) * kMaxM + m]);
      }
      v = warp_sum(v);
      if (lane == 0) buf[warp] = v;
      named_sync(1, kCThreads);
      if (tid == 0) {
        float t = 0.f;
        for (int w = 0; w < kCWarps; ++w) t += buf[w];
        a.B.ss[which * kMaxM + m] = t;
      }
      named_sync(1, kCThreads);
    }
    if (tid == 0) a.B.ss_counter[which] = 0u;
  }
};

// Merges the per-lane statistics of the 8 warps (lane m of each) with a
// fixed shuffle tree and leaves row m's result in out[m] (shared memory).
__device__ inline void combine_parts(const HeadPart& p, const Shared& sh, int tid, int M,
                                     HeadPart* out) {
  HeadPart* buf = static_cast<HeadPart*>(sh.scratch);
  const int warp = tid >> 5, lane = tid & 31;
  if (lane < M) buf[warp * kMaxM + lane] = p;
  named_sync(1, kCThreads);
  for (int m = warp; m < M; m += kCWarps) {
    HeadPart q;
    if (lane < kCWarps)
      q = buf[lane * kMaxM + m];
    else
      part_empty(q);
    for (int off = 4; off > 0; off >>= 1) part_merge(q, part_shfl(q, off));
    if (lane == 0) out[m] = q;
  }
  named_sync(1, kCThreads);
}

// Exit head: z = W_lm RMSNorm_final(h).  Lane m keeps running statistics of
// the logits it produced (max, sum exp, sum exp*(z-max), top-k); per block
// they are merged in warp order, and the last block merges the blocks (and
// the split slots) in a fixed shuffle tree, giving argmax (lowest id on
// ties), log-sum-exp, entropy H = log S - T/S, C_k = lse - mean(top-k
// logits) and pmax = 1/S.
struct EpiHead {
  struct State {
    HeadPart p;
  };
  int topk, write_logits;
  __device__ void init(State& s) const { part_empty(s.p); }
  __device__ void pair(const StreamArgs& a, int tile, int w, int m, int, float rs, float v0,
                       float v1, State& st) const {
    const int r0 = map_row(a.g, a.D, tile, w), r1 = map_row(a.g, a.D, tile, w + 16);
    if (r0 >= 0) {
      const float z = v0 * rs;
      part_add(st.p, z, r0);
      if (write_logits) a.B.logits[(size_t)m * a.D.V + r0] = z;
    }
    if (r1 >= 0) {
      const float z = v1 * rs;
      part_add(st.p, z, r1);
      if (write_logits) a.B.logits[(size_t)m * a.D.V + r1] = z;
    }
  }
  __device__ HeadPart* slots(const StreamArgs& a) const {
    return static_cast<HeadPart*>(a.B.head_part);
  }
  __device__ void split_done(const StreamArgs& a, int b0, State& st, const Shared& sh, int tid,
                             int M) const {
    HeadPart* out = static_cast<HeadPart*>(sh.scratch) + kCWarps * kMaxM;
    combine_parts(st.p, sh, tid, M, out);
    if (tid < M) slots(a)[((size_t)kMaxBlocksDev + b0) * kMaxM + tid] = out[tid];
  }
  __device__ void finish(const StreamArgs& a, State& st, const Shared& sh, int tid, int M) const {
    HeadPart* out = static_cast<HeadPart*>(sh.scratch) + kCWarps * kMaxM;
    combine_parts(st.p, sh, tid, M, out);
    HeadPart* sl = slots(a);
    if (tid < M) sl[(size_t)blockIdx.x * kMaxM + tid] = out[tid];
    __threadfence();
    named_sync(1, kCThreads);
    if (tid == 0) *sh.flag = atomicAdd(a.B.head_counter, 1u) == (unsigned)(a.g.P - 1);
    named_sync(1, kCThreads);
    if (!*sh.flag) return;
    __threadfence();
    // every thread merges its slots, then a fixed shuffle tree per warp and
    // one over the eight warp results
    HeadPart* buf = static_cast<HeadPart*>(sh.scratch);
    const int warp = tid >> 5, lane = tid & 31;
    for (int m = 0; m < M; ++m) {
      HeadPart p;
      part_empty(p);
      for (int b = tid; b < a.g.P; b += kCThreads) {
        part_merge(p, part_load_cg(&sl[(size_t)b * kMaxM + m]));
        if (has_split_slot(a.g, b)) part_merge(p, part_load_cg(&sl[((size_t)kMaxBlocksDev + b) * kMaxM + m]));
      }
      for (int off = 16; off > 0; off >>= 1) part_merge(p, part_shfl(p, off));
      if (lane == 0) buf[warp] = p;
      named_sync(1, kCThreads);
      if (warp == 0) {
        HeadPart f;
        if (lane < kCWarps)
          f = buf[lane];
        else
          part_empty(f);
        for (int off = 4; off > 0; off >>= 1) part_merge(f, part_shfl(f, off));
        if (lane == 0) {
          write_row_stats(a.B.stats[m], f, topk);
        }
      }
      named_sync(1, kCThreads);
    }
    if (tid == 0) *a.B.head_counter = 0u;
  }
};

// ------------------------------------------------------------ the kernel

template <int MM>
__device__ __forceinline__ float pick(const float (&v)[MM], int lane) {
  float r = 0.f;
#pragma unroll
  for (int m = 0; m < MM; ++m)
    if (m == lane) r = v[m];
  return r;
}

// ---- tensor-core helpers (verification rows: M > 1)
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& a0, uint32_t& a1, uint32_t& a2,
                                        uint32_t& a3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(a0), "=r"(a1), "=r"(a2), "=r"(a3)
               : "r"(addr));
}

// d += A(16x16, bf16, row) * B(16x8, bf16, col), fp32 accumulate.
__device__ __forceinline__ void mma_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                          uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Splits (x0, x1) into bf16 high parts and bf16 residuals, packed low-k first:
// x = hi + lo to about 16 significant bits, so two bf16 products keep the
// activations' fp32 precision.
__device__ __forceinline__ void split_bf16x2(float x0, float x1, uint32_t& hi, uint32_t& lo) {
  const __nv_bfloat16 h0 = __float2bfloat16_rn(x0), h1 = __float2bfloat16_rn(x1);
  const __nv_bfloat16 l0 = __float2bfloat16_rn(x0 - __bfloat162float(h0));
  const __nv_bfloat16 l1 = __float2bfloat16_rn(x1 - __bfloat162float(h1));
  hi = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
  lo = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
}

// Stage sequence of a block: from unit u, the run of up to 4 units that stays
// inside the tile and the block's range.  Producer and consumers walk it
// identically.
__device__ __forceinline__ int stage_units(const Geom& g, long long u, long long u_end) {
  const long long j = u % g.nks;
  long long n = g.nks - j;
  if (n > kRowBytes / kUnit) n = kRowBytes / kUnit;
  if (n > u_end - u) n = u_end - u;
  return (int)n;
}

template <typename T, int MM, bool NORM, bool MMA, class Epi>
__global__ void __launch_bounds__(kThreads, 1) k_stream(const StreamArgs a, const Epi epi) {
  static_assert(!MMA || (std::is_same<T, __nv_bfloat16>::value && MM > 1), "tensor path: bf16 rows");
  extern __shared__ __align__(128) unsigned char smem[];
  using E = Elem<T>;
  constexpr int EPC = E::kPerChunk;
  constexpr int CU = kUnit / (int)sizeof(T);  // columns per unit
  unsigned char* ring = smem + SmemLayout::ring;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + SmemLayout::bars);
  uint64_t* empty = full + kNS;
  const Shared sh{reinterpret_cast<float*>(smem + SmemLayout::rs),
                  reinterpret_cast<int*>(smem + SmemLayout::flag), smem + SmemLayout::scratch};

  const Geom& g = a.g;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long u_begin = stage_start(g, blockIdx.x), u_end = stage_start(g, blockIdx.x + 1);
  if (threadIdx.x == 0) {
    for (int i = 0; i < kNS; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kCWarps);
    }
    mbar_init_fence();
  }
  __syncthreads();
  pdl_launch_dependents();

  if (warp == kCWarps) {
    // ---------------- producer: weights do not depend on earlier kernels
    const unsigned char* W = static_cast<const unsigned char*>(a.W);
    const uint64_t pol = evict_first_policy();
    int i = 0;
    for (long long u = u_begin; u < u_end; ++i) {
      const int n = stage_units(g, u, u_end);
      const int slot = i % kNS;
      const uint32_t ph = (uint32_t)(i / kNS) & 1u;
      if (!mbar_wait(&empty[slot], ph ^ 1u)) {
        if (lane == 0) atomicOr(&a.B.ctl->err, (int)kErrTimeout);
        break;
      }
      const int tile = (int)(u / g.nks), j = (int)(u - (long long)tile * g.nks);
      const int off = j * kUnit;
      const int bytes = min(n * kUnit, g.row_bytes - off);
      const int row = map_row(g, a.D, tile, lane);
      const int nvalid = __popc(__ballot_sync(0xffffffffu, row >= 0));
      if (lane == 0) mbar_arrive_expect_tx(&full[slot], (uint32_t)(nvalid * bytes));
      __syncwarp();
      if (row >= 0)
        bulk_g2s(ring + (size_t)slot * kStageBytes + lane * kRowStride,
                 W + (size_t)row * g.row_bytes + off, (uint32_t)bytes, &full[slot], pol);
      u += n;
    }
    // drain: the copies of the last stages have landed before the block exits
    if (lane == 0)
      for (int k = i > kNS ? i - kNS : 0; k < i; ++k) mbar_wait(&full[k % kNS], (uint32_t)(k / kNS) & 1u);
    return;
  }

  // ---------------- consumers
  pdl_wait();
  int pos0, M;
  resolve_rows(a.B.ctl, a.sel, pos0, M);
  const int tid = threadIdx.x;
  if (tid < 32) {
    float r = 1.f;
    if (a.ss_in >= 0 && tid < M) r = 1.0f / sqrtf(a.B.ss[a.ss_in * kMaxM + tid] / (float)g.K + a.D.eps);
    sh.rs[tid] = r;
  }
  named_sync(1, kCThreads);
  const float my_rs = sh.rs[lane];
  const float* x = a.x;
  const T* gn = static_cast<const T*>(a.gnorm);  // used when NORM
  typename Epi::State run;
  epi.init(run);
  float acc[MMA ? 1 : 4][MMA ? 1 : MM];
  float dmm[kNB][4];  // tensor-core accumulators: rows rb*16 + (g, g+8), tokens nb*8 + 2c + (0, 1)
  float* red = reinterpret_cast<float*>(smem + SmemLayout::red);
  const int rloc[4] = {warp, warp + 8, warp + 16, warp + 24};
  int cur = -1;
  bool ok = true;
  int i = 0;
  for (long long u = u_begin; u < u_end; ++i) {
    const int n = stage_units(g, u, u_end);
    const int slot = i % kNS;
    const uint32_t ph = (uint32_t)(i / kNS) & 1u;
    const int tile = (int)(u / g.nks), j = (int)(u - (long long)tile * g.nks);
    u += n;
    if (tile != cur) {
      if (MMA) {
#pragma unroll
        for (int nb = 0; nb < kNB; ++nb)
#pragma unroll
          for (int q = 0; q < 4; ++q) dmm[nb][q] = 0.f;
      } else {
#pragma unroll
        for (int r = 0; r < (MMA ? 1 : 4); ++r)
#pragma unroll
          for (int m = 0; m < (MMA ? 1 : MM); ++m) acc[r][m] = 0.f;
      }
      cur = tile;
    }
    if (ok && !mbar_wait(&full[slot], ph)) {
      if (lane == 0) atomicOr(&a.B.ctl->err, (int)kErrTimeout);
      ok = false;
    }
    const int bytes = min(n * kUnit, g.row_bytes - j * kUnit);
    const unsigned char* stg = ring + (size_t)slot * kStageBytes + lane * 16;
    const int col0 = j * CU + lane * 16 / (int)sizeof(T);
    if constexpr (MMA) {
      // warp = (16-row block rb, 512-byte unit kq of the stage)
      const int rb = warp & 1, kq = warp >> 1;
      if (ok && kq < n) {
        const int ub = min(kUnit, bytes - kq * kUnit);
        const uint32_t abase =
            smem_u32(ring + (size_t)slot * kStageBytes + (rb * 16 + (lane & 15)) * kRowStride +
                     kq * kUnit + (lane >> 4) * 16);
        const int kc0 = (j + kq) * CU + 2 * (lane & 3);
        const int tok0 = lane >> 2;
        for (int kk = 0; kk < ub / 32; ++kk) {
          uint32_t a0, a1, a2, a3;
          ldsm_x4(abase + kk * 32, a0, a1, a2, a3);
          const int kc = kc0 + kk * 16;
          float g0 = 1.f, g1 = 1.f, g8 = 1.f, g9 = 1.f;
          if (NORM) {
            const __nv_bfloat162 ga = *reinterpret_cast<const __nv_bfloat162*>(gn + kc);
            const __nv_bfloat162 gb = *reinterpret_cast<const __nv_bfloat162*>(gn + kc + 8);
            g0 = __low2float(ga);
            g1 = __high2float(ga);
            g8 = __low2float(gb);
            g9 = __high2float(gb);
          }
#pragma unroll
          for (int nb = 0; nb < kNB; ++nb) {
            if (nb * 8 < M) {
              const int tok = nb * 8 + tok0;
              float2 xa = make_float2(0.f, 0.f), xb = make_float2(0.f, 0.f);
              if (tok < M) {
                xa = __ldg(reinterpret_cast<const float2*>(x + (size_t)tok * g.K + kc));
                xb = __ldg(reinterpret_cast<const float2*>(x + (size_t)tok * g.K + kc + 8));
              }
              uint32_t h0, l0, h1, l1;
              split_bf16x2(xa.x * g0, xa.y * g1, h0, l0);
              split_bf16x2(xb.x * g8, xb.y * g9, h1, l1);
              mma_16816(dmm[nb], a0, a1, a2, a3, h0, h1);
              mma_16816(dmm[nb], a0, a1, a2, a3, l0, l1);
            }
          }
        }
      }
    } else if (ok && bytes == kRowBytes) {
      // full stage; the single-row kernel issues every load of the stage
      // before the math, the multi-row one goes one 512-byte step at a time
      constexpr int NSUB = kRowBytes / kUnit;
      constexpr int HOIST = MM <= 2 ? NSUB : 1;
#pragma unroll
      for (int sg = 0; sg < NSUB; sg += HOIST) {
        uint4 wq[HOIST][4];
#pragma unroll
        for (int h = 0; h < HOIST; ++h)
#pragma unroll
          for (int r = 0; r < 4; ++r)
            wq[h][r] = *reinterpret_cast<const uint4*>(stg + rloc[r] * kRowStride + (sg + h) * kUnit);
        float gv[HOIST][EPC];
        if (NORM) {
          uint4 gq[HOIST];
#pragma unroll
          for (int h = 0; h < HOIST; ++h)
            gq[h] = __ldg(reinterpret_cast<const uint4*>(gn + col0 + (sg + h) * CU));
#pragma unroll
          for (int h = 0; h < HOIST; ++h) E::unpack(gq[h], gv[h]);
        }
#pragma unroll
        for (int m = 0; m < MM; ++m) {
          if (m < M) {
            float4 xq[HOIST][EPC / 4];
#pragma unroll
            for (int h = 0; h < HOIST; ++h)
#pragma unroll
              for (int q = 0; q < EPC / 4; ++q)
                xq[h][q] = __ldg(reinterpret_cast<const float4*>(x + (size_t)m * g.K + col0 +
                                                                 (sg + h) * CU) + q);
#pragma unroll
            for (int h = 0; h < HOIST; ++h) {
              float xv[EPC];
#pragma unroll
              for (int q = 0; q < EPC / 4; ++q) {
                xv[4 * q] = xq[h][q].x;
                xv[4 * q + 1] = xq[h][q].y;
                xv[4 * q + 2] = xq[h][q].z;
                xv[4 * q + 3] = xq[h][q].w;
              }
              if (NORM) {
#pragma unroll
                for (int e = 0; e < EPC; ++e) xv[e] *= gv[h][e];
              }
#pragma unroll
              for (int r = 0; r < 4; ++r) {
                float wf[EPC];
                E::unpack(wq[h][r], wf);
#pragma unroll
                for (int e = 0; e < EPC; ++e) acc[r][m] = fmaf(wf[e], xv[e], acc[r][m]);
              }
            }
          }
        }
      }
    } else if (ok) {
      // partial stage (block range edge or ragged end of the row)
      for (int off = lane * 16; off < bytes; off += kUnit) {
        const int col = j * CU + off / (int)sizeof(T);
        float gv[EPC];
        if (NORM) E::unpack(__ldg(reinterpret_cast<const uint4*>(gn + col)), gv);
        float wf[4][EPC];
#pragma unroll
        for (int r = 0; r < 4; ++r)
          E::unpack(*reinterpret_cast<const uint4*>(ring + (size_t)slot * kStageBytes +
                                                    rloc[r] * kRowStride + off), wf[r]);
#pragma unroll
        for (int m = 0; m < MM; ++m) {
          if (m < M) {
            float xv[EPC];
            const float4* xp = reinterpret_cast<const float4*>(x + (size_t)m * g.K + col);
#pragma unroll
            for (int q = 0; q < EPC / 4; ++q) {
              const float4 t4 = __ldg(xp + q);
              xv[4 * q] = t4.x;
              xv[4 * q + 1] = t4.y;
              xv[4 * q + 2] = t4.z;
              xv[4 * q + 3] = t4.w;
            }
            if (NORM) {
#pragma unroll
              for (int e = 0; e < EPC; ++e) xv[e] *= gv[e];
            }
#pragma unroll
            for (int r = 0; r < 4; ++r)
#pragma unroll
              for (int e = 0; e < EPC; ++e) acc[r][m] = fmaf(wf[r][e], xv[e], acc[r][m]);
          }
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[slot]);
    if (j + n != g.nks && u != u_end) continue;

    // ---- tile flush: warp-local unless the tile is shared with other blocks
    float val[4];  // lane m: the four rows' sums for input row m
    if constexpr (MMA) {
      // four K-quarter partials per row, added in quarter order
      named_sync(1, kCThreads);
      const int rb = warp & 1, kq = warp >> 1, gq = lane >> 2, cq = lane & 3;
#pragma unroll
      for (int nb = 0; nb < kNB; ++nb)
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int row = rb * 16 + gq + (q >> 1) * 8, tok = nb * 8 + 2 * cq + (q & 1);
          red[((kq * kRT) + row) * 8 * kNB + tok] = dmm[nb][q];
        }
      named_sync(1, kCThreads);
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        float t = 0.f;
        if (lane < M)
          for (int q = 0; q < 4; ++q) t += red[((q * kRT) + rloc[r]) * 8 * kNB + lane];
        val[r] = t;
      }
    } else {
#pragma unroll
      for (int r = 0; r < (MMA ? 1 : 4); ++r)
#pragma unroll
        for (int m = 0; m < (MMA ? 1 : MM); ++m)
          if (m < M) acc[r][m] = warp_sum(acc[r][m]);
#pragma unroll
      for (int r = 0; r < (MMA ? 1 : 4); ++r) val[r] = pick(acc[r], lane);
    }
    const long long t0 = (long long)tile * g.nks, t1 = t0 + g.nks;
    if (t0 >= u_begin && t1 <= u_end) {
      if (lane < M) {
        epi.pair(a, tile, warp, lane, pos0, my_rs, val[0], val[2], run);
        epi.pair(a, tile, warp + 8, lane, pos0, my_rs, val[1], val[3], run);
      }
      continue;
    }
    // shared with neighbouring blocks: publish this block's partial sums
    const int first_tile = (int)(u_begin / g.nks);
    const int slot2 = tile == first_tile ? 0 : 1;
    float* mine = a.B.gpart + ((size_t)blockIdx.x * 2 + slot2) * kRT * kMaxM;
    if (lane < M)
#pragma unroll
      for (int r = 0; r < 4; ++r) mine[rloc[r] * kMaxM + lane] = val[r];
    __threadfence();
    named_sync(1, kCThreads);
    const int b0 = block_of_stage(g, t0), b1 = block_of_stage(g, t1 - 1);
    if (tid == 0) {
      int contrib = 0;
      for (int b = b0; b <= b1; ++b) contrib += stage_start(g, b) < stage_start(g, b + 1);
      *sh.flag = atomicAdd(&a.B.tile_counter[tile], 1u) == (unsigned)(contrib - 1);
    }
    named_sync(1, kCThreads);
    if (!*sh.flag) continue;
    __threadfence();
    float uu[4] = {0.f, 0.f, 0.f, 0.f};
    if (lane < M)
      for (int b = b0; b <= b1; ++b) {  // block order: independent of who finishes
        const long long sb = stage_start(g, b);
        if (sb == stage_start(g, b + 1)) continue;
        const int sl = tile == (int)(sb / g.nks) ? 0 : 1;
        const float* p = a.B.gpart + ((size_t)b * 2 + sl) * kRT * kMaxM;
#pragma unroll
        for (int r = 0; r < 4; ++r) uu[r] += __ldcg(&p[rloc[r] * kMaxM + lane]);
      }
    if (tid == 0) a.B.tile_counter[tile] = 0u;
    typename Epi::State sp;
    epi.init(sp);
    if (lane < M) {
      epi.pair(a, tile, warp, lane, pos0, my_rs, uu[0], uu[2], sp);
      epi.pair(a, tile, warp + 8, lane, pos0, my_rs, uu[1], uu[3], sp);
    }
    epi.split_done(a, b0, sp, sh, tid, M);
  }
  epi.finish(a, run, sh, tid, M);
}

// ------------------------------------------------------------- launchers

bool g_pdl_enabled = true;
bool g_chain_enabled = true;
thread_local bool g_pdl_ok = true;

static Geom make_geom(const Dims& D, int N, int K, int elt, int map) {
  Geom g{};
  g.N = N;
  g.K = K;
  g.elt = elt;
  g.map = map;
  g.row_bytes = K * elt;
  g.nks = (g.row_bytes + kUnit - 1) / kUnit;
  if (map == kMapGateUp)
    g.ntiles = (N / 2 + 15) / 16;
  else if (map == kMapQKV)
    g.ntiles = (D.Hq + D.Hkv) * (D.hd / 32) + (D.Hkv * D.hd + kRT - 1) / kRT;
  else
    g.ntiles = (N + kRT - 1) / kRT;
  g.T = (long long)g.ntiles * g.nks;
  g.P = D.num_sms;
  return g;
}

// Multi-row bf16 matrices whose rows are whole 512-byte units go through the
// tensor cores; single rows, fp32 and ragged rows through CUDA cores.
template <typename T, int MM>
static bool use_mma(const Geom& g) {
  return std::is_same<T, __nv_bfloat16>::value && MM > 1 && g.row_bytes % kUnit == 0;
}

template <typename T, int MM, bool NORM, class Epi>
static cudaError_t stream_launch(const StreamArgs& a, const Epi& epi, cudaStream_t st) {
  constexpr bool kCan = std::is_same<T, __nv_bfloat16>::value && MM > 1;
  if (kCan && use_mma<T, MM>(a.g))
    return launch_ex(k_stream<T, MM, NORM, kCan, Epi>, dim3(a.g.P), dim3(kThreads),
                     SmemLayout::total<MM>(), st, a, epi);
  return launch_ex(k_stream<T, MM, NORM, false, Epi>, dim3(a.g.P), dim3(kThreads),
                   SmemLayout::total<MM>(), st, a, epi);
}

template <typename T, int MM, bool NORM, class Epi>
static cudaError_t prepare_one() {
  static_assert(SmemLayout::total<MM>() <= 227 * 1024, "shared memory budget");
  constexpr bool kCan = std::is_same<T, __nv_bfloat16>::value && MM > 1;
  cudaError_t e = cudaFuncSetAttribute(k_stream<T, MM, NORM, false, Epi>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)SmemLayout::total<MM>());
  if (e != cudaSuccess || !kCan) return e;
  return cudaFuncSetAttribute(k_stream<T, MM, NORM, kCan, Epi>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)SmemLayout::total<MM>());
}

template <typename T, int MM>
static cudaError_t prepare_t() {
  cudaError_t e;
  if ((e = prepare_one<T, MM, false, EpiPlain>()) != cudaSuccess) return e;
  if ((e = prepare_one<T, MM, true, EpiQKV<T>>()) != cudaSuccess) return e;
  if ((e = prepare_one<T, MM, true, EpiGateUp>()) != cudaSuccess) return e;
  if ((e = prepare_one<T, MM, false, EpiResid>()) != cudaSuccess) return e;
  return prepare_one<T, MM, true, EpiHead>();
}

cudaError_t prepare_gemv_kernels() {
  cudaError_t e;
  if ((e = prepare_t<float, 1>()) != cudaSuccess) return e;
  if ((e = prepare_t<float, kMaxM>()) != cudaSuccess) return e;
  // bf16 models run on the tensor-core kernels (tile.cu); the plain bf16
  // product stays here for the allocation-free entry point
  if ((e = prepare_one<__nv_bfloat16, 1, false, EpiPlain>()) != cudaSuccess) return e;
  return prepare_one<__nv_bfloat16, kMaxM, false, EpiPlain>();
}

// Attention launchers live in attention.cu.
cudaError_t launch_attention(const Dims& D, const Bufs& B, int dtype, int layer, RowSel sel,
                             bool big, cudaStream_t st);

template <typename T, int MM>
static cudaError_t part_t(const Dims& D, const Bufs& B, const LayerW& w, int layer, int part,
                          RowSel sel, cudaStream_t st) {
  const int elt = (int)sizeof(T);
  StreamArgs a{};
  a.D = D;
  a.B = B;
  a.sel = sel;
  switch (part) {
    case 0:
      a.g = make_geom(D, (D.Hq + 2 * D.Hkv) * D.hd, D.d, elt, kMapQKV);
      a.W = w.wqkv;
      a.gnorm = w.attn_norm;
      a.x = B.h;
      a.ss_in = 0;
      return stream_launch<T, MM, true>(a, EpiQKV<T>{layer}, st);
    case 1:
      return launch_attention(D, B, std::is_same<T, float>::value ? SSD_DTYPE_F32 : SSD_DTYPE_BF16,
                              layer, sel, MM > 1, st);
    case 2:
      a.g = make_geom(D, D.d, D.qd, elt, kMapLinear);
      a.W = w.wo;
      a.gnorm = nullptr;
      a.x = B.attn_out;
      a.ss_in = -1;
      return stream_launch<T, MM, false>(a, EpiResid{1}, st);
    case 3:
      a.g = make_geom(D, 2 * D.F, D.d, elt, kMapGateUp);
      a.W = w.wgu;
      a.gnorm = w.ffn_norm;
      a.x = B.h;
      a.ss_in = 1;
      return stream_launch<T, MM, true>(a, EpiGateUp{}, st);
    case 4:
      a.g = make_geom(D, D.d, D.F, elt, kMapLinear);
      a.W = w.wdown;
      a.gnorm = nullptr;
      a.x = B.act;
      a.ss_in = -1;
      return stream_launch<T, MM, false>(a, EpiResid{0}, st);
    default:
      return cudaErrorInvalidValue;
  }
}

cudaError_t launch_layer_part(const Dims& D, const Bufs& B, int dtype, const LayerW& w,
                              const TileMaps* tm, int layer, int part, RowSel sel, int mrows,
                              cudaStream_t st) {
  const bool big = mrows > 1;
  if (dtype == SSD_DTYPE_BF16) {
    if (part == 1) return launch_attention(D, B, dtype, layer, sel, big, st);
    if (!tm) return cudaErrorInvalidValue;
    return launch_tile_part(D, B, *tm, w, layer, part, sel, mrows, st);
  }
  return big ? part_t<float, kMaxM>(D, B, w, layer, part, sel, st)
             : part_t<float, 1>(D, B, w, layer, part, sel, st);
}

cudaError_t launch_layer(const Dims& D, const Bufs& B, int dtype, const LayerW& w,
                         const TileMaps* tm, int layer, RowSel sel, int mrows, cudaStream_t st) {
  for (int part = 0; part < 5; ++part) {  // qkv, attention, o, gate/up, down
    cudaError_t e = launch_layer_part(D, B, dtype, w, tm, layer, part, sel, mrows, st);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

template <typename T, int MM>
static cudaError_t head_t(const Dims& D, const Bufs& B, const void* lm, const void* fn, int topk,
                          bool logits, RowSel sel, cudaStream_t st) {
  StreamArgs a{};
  a.D = D;
  a.B = B;
  a.sel = sel;
  a.g = make_geom(D, D.V, D.d, (int)sizeof(T), kMapLinear);
  a.W = lm;
  a.gnorm = fn;
  a.x = B.h;
  a.ss_in = 0;
  return stream_launch<T, MM, true>(a, EpiHead{topk, logits ? 1 : 0}, st);
}

cudaError_t launch_head(const Dims& D, const Bufs& B, int dtype, const void* lm_head,
                        const CUtensorMap* lm_map, const TileMaps* tm, const void* final_norm,
                        int topk, bool write_logits, RowSel sel, int mrows, cudaStream_t st) {
  if (dtype == SSD_DTYPE_BF16) {
    if (!tm || !lm_map) return cudaErrorInvalidValue;
    return launch_tile_head(D, B, *tm, *lm_map, final_norm, topk, write_logits, sel, mrows, st);
  }
  return mrows > 1 ? head_t<float, kMaxM>(D, B, lm_head, final_norm, topk, write_logits, sel, st)
                   : head_t<float, 1>(D, B, lm_head, final_norm, topk, write_logits, sel, st);
}

template <typename T, int MM>
static cudaError_t plain_t(const Dims& D, const Bufs& B, const void* W, int rows, int cols,
                           const float* x, int M, float* y, cudaStream_t st) {
  StreamArgs a{};
  a.D = D;
  a.B = B;
  a.sel = RowSel{kRowsExplicit, 0, M, nullptr};
  a.g = make_geom(D, rows, cols, (int)sizeof(T), kMapLinear);
  a.W = W;
  a.gnorm = nullptr;
  a.x = x;
  a.ss_in = -1;
  return stream_launch<T, MM, false>(a, EpiPlain{y}, st);
}

cudaError_t launch_gemv_plain(const Dims& D, const Bufs& B, int dtype, const void* W, int rows,
                              int cols, const float* x, int M, float* y, cudaStream_t st) {
  if (dtype == SSD_DTYPE_BF16)
    return M == 1 ? plain_t<__nv_bfloat16, 1>(D, B, W, rows, cols, x, M, y, st)
                  : plain_t<__nv_bfloat16, kMaxM>(D, B, W, rows, cols, x, M, y, st);
  return M == 1 ? plain_t<float, 1>(D, B, W, rows, cols, x, M, y, st)
                : plain_t<float, kMaxM>(D, B, W, rows, cols, x, M, y, st);
}


// ----------------------------------------------- allocation-free variant
//
// ssd_gemv_noalloc: the plain weight-streaming product for callers that can
// not allocate device memory.  Its scratch -- the partial sums of row tiles
// shared by two blocks, their tickets and an error word -- lives in one
// file-scope device array instead of a caller-provided workspace.

constexpr int kNoAllocBlocks = 256;   // grid cap (one block per SM)
constexpr int kNoAllocTiles = 4096;   // row tiles of 32: rows <= 131072
constexpr size_t kNoAllocPart = sizeof(float) * (size_t)kNoAllocBlocks * 2 * kRT * kMaxM;
constexpr size_t kNoAllocCount = sizeof(uint32_t) * kNoAllocTiles;
constexpr size_t kNoAllocCtl = (sizeof(Ctl) + 255) / 256 * 256;
constexpr size_t kNoAllocBytes = kNoAllocPart + kNoAllocCount + kNoAllocCtl;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

namespace {
struct NoAllocDevice {
  bool ready = false;
  unsigned char* scratch = nullptr;  // device address of g_noalloc_scratch
  int sms = 0;
};
std::mutex g_noalloc_mu;
NoAllocDevice g_noalloc_dev[64];
}  // namespace

}  // namespace ssd

extern "C" ssd_status ssd_gemv_noalloc(const void* W, int32_t dtype, int32_t rows, int32_t cols,
                                       const float* x_dev, int32_t M, float* y_dev,
                                       int32_t* err_dev, void* stream) {
  using namespace ssd;
  if (!W || !x_dev || !y_dev || ((uintptr_t)W & 15u) || ((uintptr_t)x_dev & 15u))
    return SSD_ERR_INVALID_ARG;
  if (dtype != SSD_DTYPE_F32 && dtype != SSD_DTYPE_BF16) return SSD_ERR_INVALID_ARG;
  const int elt = dtype == SSD_DTYPE_BF16 ? 2 : 4;
  if (rows < 1 || cols < 1 || M < 1 || ((size_t)cols * elt) % 16) return SSD_ERR_INVALID_ARG;
  if (M > kMaxM || (rows + kRT - 1) / kRT > kNoAllocTiles) return SSD_ERR_CAPACITY;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return SSD_ERR_CUDA;
  NoAllocDevice nd;
  {
    // once per device, with that device current: the array's device address
    // (the symbol's host-side name is not one), kernel attributes, SM count
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    NoAllocDevice& d = g_noalloc_dev[dev];
    if (!d.ready) {
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return SSD_ERR_CUDA;
      if (prepare_gemv_kernels() != cudaSuccess) return SSD_ERR_CUDA;
      int sms = 0;
      if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return SSD_ERR_CUDA;
      d.scratch = static_cast<unsigned char*>(p);
      d.sms = sms < kNoAllocBlocks ? sms : kNoAllocBlocks;
      d.ready = true;
    }
    nd = d;
  }
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  Bufs B{};
  B.gpart = reinterpret_cast<float*>(nd.scratch);
  B.tile_counter = reinterpret_cast<uint32_t*>(nd.scratch + kNoAllocPart);
  B.ctl = reinterpret_cast<Ctl*>(nd.scratch + kNoAllocPart + kNoAllocCount);
  Dims D{};
  D.num_sms = nd.sms;
  // tickets and the error word start at zero on every call
  if (cudaMemsetAsync(B.tile_counter, 0, kNoAllocCount + kNoAllocCtl, st) != cudaSuccess)
    return SSD_ERR_CUDA;
  if (launch_gemv_plain(D, B, dtype, W, rows, cols, x_dev, M, y_dev, st) != cudaSuccess)
    return SSD_ERR_CUDA;
  // the error word a bounded wait sets when it gives up, for the caller to read
  if (err_dev && cudaMemcpyAsync(err_dev, &B.ctl->err, sizeof(int32_t), cudaMemcpyDeviceToDevice,
                                 st) != cudaSuccess)
    return SSD_ERR_CUDA;
  return SSD_OK;
}

namespace ssd {
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

cudaError_t launch_read_probe(const void* src, uint64_t bytes, uint32_t* sink, cudaStream_t st) {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  k_read_probe<<<sms * 4, 512, 0, st>>>(static_cast<const uint4*>(src), bytes / 16, sink);
  return cudaGetLastError();
}

}  // namespace ssd
