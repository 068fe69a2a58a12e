// tile.cu -- tensor-core weight streaming for the bf16 decoder (sm_103a).
//
// Every projection of a bf16 model (QKV, O, gate/up, down) and the exit LM
// head multiplies its weight matrix with M <= 17 input rows (1 while
// drafting, k + 1 while verifying; §3.3) and reads each weight once, so the
// pass is bound by HBM bandwidth.  This kernel streams the matrix through
// shared memory with tensor-TMA and multiplies it on the 5th-generation
// tensor cores:
//  - tiles of 256 output rows; a unit is 256 rows x 64 columns (32 KB, four
//    64 x 64 boxes with the 128-byte swizzle); the units, in (tile, K) order,
//    are split evenly over a persistent grid of one block per SM
//    ("stream-K"), so every SM streams the same bytes whatever the shape;
//  - warp roles (320 threads): a TMA warp fills a 5-deep ring with the
//    unit's weight boxes and its slice of the fp32 input rows (plus the
//    RMSNorm weights); eight worker warps turn the slice into bf16 high and
//    low operand tiles (x = hi + lo to ~16 significant bits); one MMA warp
//    issues tcgen05.mma (M = 128 rows per half, N = 16 or 32 token columns,
//    K = 16) for both halves and both parts into a double-buffered TMEM
//    accumulator, and releases ring slots and operand tiles with
//    tcgen05.commit;
//  - at the end of a tile the workers read the accumulator from TMEM (each
//    thread one row of each half: the rows a fused epilogue pairs, i and
//    i + 128) and run the epilogue; a tile split between blocks is finished
//    by its last contributor, adding the partial sums in block order;
//  - every output element is computed the same way whatever M is (the
//    token columns are independent), so a verification row equals the
//    single-row drafting pass bit for bit.
// The tiles' row order is chosen so that an epilogue's pair of rows sits at
// i and i + 128: rotary pairs (i, i + hd/2) of a head for QKV (hd = 128),
// gate row j and up row F + j for the SwiGLU.
#include <math.h>

#include <cudaTypedefs.h>

#include <mutex>
#include <type_traits>

#include "headpart.cuh"
#include "kernels.h"
#include "pipe.cuh"
#include "tc.cuh"

namespace ssd {

namespace {

constexpr int kTR = 256;                  // output rows per tile (two halves of 128)
constexpr int kKC = 64;                   // columns per unit
constexpr int kWBytes = kTR * kKC * 2;    // weights of one unit (32 KB)
constexpr int kBoxBytes = 64 * kKC * 2;   // one 64 x 64 weight box
constexpr int kWorkers = 8;
constexpr int kWThreads = kWorkers * 32;
constexpr int kTmaWarp = kWorkers, kMmaWarp = kWorkers + 1;
constexpr int kTThreads = (kWorkers + 2) * 32;
constexpr int kLT = (kMaxM + 1) / 2;      // tokens of one parity group
constexpr int kMaxBlocksDev = kMaxBlocks;

enum TMap : int { kTMapLinear = 0, kTMapQKV = 1, kTMapGateUp = 2 };
enum TKind : int { kKPlain = 0, kKQKV = 1, kKGateUp = 2, kKResid = 3, kKHead = 4 };

constexpr size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Shared-memory layout of the instance with TP token rows (8, 16 or 24): the
// MMA's N is 2 TP (bf16 high parts of the tokens in rows 0..TP-1, low parts
// in rows TP..2TP-1).  Every ring slot holds a unit's weights, its operand
// tile and its input slice, all released by the one commit of the unit's
// MMAs.
template <int TP, bool HEAD>
struct TL {
  static constexpr int N = 2 * TP;
  static constexpr int NS = TP == 24 ? 4 : (TP == 8 && !HEAD ? 6 : 5);  // ring depth
  static constexpr int XB = TP * kKC * 4;                   // input box: TP rows x 64 fp32
  static constexpr int XS = (int)align_up(XB + kKC * 2, 128);  // + RMSNorm weight slice
  static constexpr int BB = N * 128;                        // operand tile (multiple of 1024)
  static constexpr uint32_t kCols = 4 * N <= 64 ? 64 : (4 * N <= 128 ? 128 : 256);
  static constexpr size_t ring = 0;
  static constexpr size_t bt = ring + (size_t)NS * kWBytes;
  static constexpr size_t xs = bt + (size_t)NS * BB;
  static constexpr size_t bars = align_up(xs + (size_t)NS * XS, 16);
  // wfull[NS], xfull[NS], empty[NS], bfull[NS], accfull[2], accempty[2], drain
  static constexpr int kNBars = 4 * NS + 5;
  static constexpr size_t tslot = bars + 8 * (size_t)kNBars;
  static constexpr size_t flag = tslot + 8;
  static constexpr size_t rs = flag + 8;
  static constexpr size_t red = rs + 4 * 32;
  // exit-head statistics (running, split tile, merge), only in the head's instances
  static constexpr size_t run = align_up(red + 4 * (size_t)kWorkers * kLT, 16);
  static constexpr size_t spl = run + (HEAD ? sizeof(HeadPart) * kWorkers * kLT : 0);
  static constexpr size_t comb = spl + (HEAD ? sizeof(HeadPart) * kWorkers * kLT : 0);
  static constexpr size_t used = comb + (HEAD ? sizeof(HeadPart) * kMaxM : 0);
  static constexpr size_t total = used + 1024;  // the base is aligned up to 1024 in the kernel
  static_assert(total <= 227 * 1024, "shared memory budget");
  static_assert(BB % 1024 == 0 && XS % 128 == 0, "operand / slice alignment");
};

struct TGeom {
  int N, K;          // rows, columns
  int nks;           // units per tile (64-column chunks)
  int ntiles;
  int T;            // units (T * kMaxBlocks < 2^31, checked by the launcher)
  int P;             // blocks
  int map;
};

struct TArgs {
  TGeom g;
  Dims D;
  Bufs B;
  const __nv_bfloat16* gnorm;  // RMSNorm weights of the input, or null
  int ss_in;                   // sum-of-squares buffer of the input scale (-1: none)
  RowSel sel;
  int layer;                   // QKV: KV-cache layer
  int which;                   // residual: sum-of-squares buffer written
  int topk, write_logits;      // exit head
  float* y;                    // plain product output [M][N]
};

// First unit of block b.  32-bit arithmetic: the split-tile fix-ups evaluate
// this for every contributor, and 64-bit division would dominate them.
__host__ __device__ inline int t_start(const TGeom& g, int b) {
  return (int)((unsigned)g.T * (unsigned)b / (unsigned)g.P);
}

__device__ inline int t_block_of(const TGeom& g, int s) {
  int b = (int)((unsigned)s * (unsigned)g.P / (unsigned)g.T);
  if (b >= g.P) b = g.P - 1;
  while (b + 1 < g.P && t_start(g, b + 1) <= s) ++b;
  while (b > 0 && t_start(g, b) > s) --b;
  return b;
}

// Block b owns the split slot of the tile it starts and shares with the next
// block(s), if its last tile is such a tile.
__device__ inline bool t_has_split_slot(const TGeom& g, int b) {
  const int sb = t_start(g, b), se = t_start(g, b + 1);
  if (se <= sb) return false;
  const int t = (se - 1) / g.nks;
  if ((t + 1) * g.nks <= se) return false;
  return t * g.nks >= sb;
}

// Global row of stage row s (0..255) of a tile, or -1 past the end.
__device__ inline int trow(const TGeom& g, int tile, int s) {
  if (g.map == kTMapGateUp) {
    const int F = g.N / 2;
    const int j = tile * 128 + (s & 127);
    if (j >= F) return -1;
    return s < 128 ? j : F + j;
  }
  int r;
  if (g.map == kTMapQKV) {
    const int b = s >> 6;
    r = tile * 256 + ((b & 1) << 7) + ((b >> 1) << 6) + (s & 63);
  } else {
    r = tile * 256 + s;
  }
  return r < g.N ? r : -1;
}

// First row of weight box b (0..3) of a tile: stage rows 64b..64b+63.
__device__ inline int box_row(const TGeom& g, int tile, int b) {
  if (g.map == kTMapGateUp) return (b < 2 ? 0 : g.N / 2) + tile * 128 + 64 * (b & 1);
  if (g.map == kTMapQKV) return tile * 256 + ((b & 1) << 7) + ((b >> 1) << 6);
  return tile * 256 + 64 * b;
}

__device__ __forceinline__ uint32_t swz(int m, int j) {
  return (uint32_t)((m >> 3) * 1024 + (m & 7) * 128 + ((j ^ (m & 7)) << 4));
}

__device__ __forceinline__ uint32_t pack_bf16(__nv_bfloat16 a, __nv_bfloat16 b) {
  return (uint32_t)__bfloat16_as_ushort(a) | ((uint32_t)__bfloat16_as_ushort(b) << 16);
}

struct Ring {
  uint64_t* full;
  uint64_t* empty;
  uint64_t* bfull;
  uint64_t* bempty;
  uint64_t* accfull;
  uint64_t* accempty;
  uint64_t* drain;
};

__device__ __forceinline__ void flag_timeout(const Bufs& B) {
  atomicOr(&B.ctl->err, (int)kErrTimeout);
}

// ------------------------------------------------------------ epilogues

// Adds the values of one (row pair, token) to the outputs.
template <int KIND>
__device__ __forceinline__ void t_pair(const TArgs& a, int tile, int s, int t, int pos0, float rs,
                                       float v0, float v1, float& ss) {
  const Dims& D = a.D;
  if constexpr (KIND == kKPlain) {
    const int r0 = trow(a.g, tile, s), r1 = trow(a.g, tile, s + 128);
    if (r0 >= 0) a.y[(size_t)t * a.g.N + r0] = v0;
    if (r1 >= 0) a.y[(size_t)t * a.g.N + r1] = v1;
  } else if constexpr (KIND == kKQKV) {
    // rotary embedding of the pair (i, i + hd/2) of a query / key head
    // (angle pos * theta^(-2i/hd) from the table), or two value rows
    const int r0 = trow(a.g, tile, s);
    if (r0 < 0) return;
    const int head = r0 / D.hd, i = r0 - head * D.hd;  // i < hd/2
    const int pos = pos0 + t;
    const float y0 = v0 * rs, y1 = v1 * rs;
    __nv_bfloat16* kv =
        static_cast<__nv_bfloat16*>(a.B.kv) + (size_t)a.layer * 2 * D.Hkv * D.max_seq * D.hd;
    if (head < D.Hq + D.Hkv) {
      const int half = D.hd / 2;
      const float2 cs = a.B.rope[(size_t)pos * half + i];
      const float o0 = y0 * cs.x - y1 * cs.y;
      const float o1 = y1 * cs.x + y0 * cs.y;
      if (head < D.Hq) {
        float* q = a.B.xq + (size_t)t * D.qd + (size_t)head * D.hd;
        q[i] = o0;
        q[i + half] = o1;
      } else {
        __nv_bfloat16* kr = kv + ((size_t)(head - D.Hq) * D.max_seq + pos) * D.hd;
        kr[i] = __float2bfloat16_rn(o0);
        kr[i + half] = __float2bfloat16_rn(o1);
      }
    } else {
      const int g = head - D.Hq - D.Hkv;
      __nv_bfloat16* vr = kv + ((size_t)(D.Hkv + g) * D.max_seq + pos) * D.hd;
      vr[i] = __float2bfloat16_rn(y0);
      const int r1 = trow(a.g, tile, s + 128);
      if (r1 >= 0) vr[i + D.hd / 2] = __float2bfloat16_rn(y1);
    }
  } else if constexpr (KIND == kKGateUp) {
    // act[t][j] = silu(gate_j) * up_j
    const int j = trow(a.g, tile, s);
    if (j < 0) return;
    const float gt = v0 * rs, up = v1 * rs;
    a.B.act[(size_t)t * D.F + j] = gt / (1.0f + expf(-gt)) * up;
  } else if constexpr (KIND == kKResid) {
    // h[t][row] += y, and the sum of squares the next RMSNorm needs
    const int r0 = trow(a.g, tile, s), r1 = trow(a.g, tile, s + 128);
    float* hm = a.B.h + (size_t)t * D.d;
    if (r0 >= 0) {
      const float h = __ldcg(hm + r0) + v0;  // L2: rows a previous phase wrote
      hm[r0] = h;
      ss = fmaf(h, h, ss);
    }
    if (r1 >= 0) {
      const float h = __ldcg(hm + r1) + v1;
      hm[r1] = h;
      ss = fmaf(h, h, ss);
    }
  }
}

// Residual add with the rows' previous values already loaded (split-tile
// fix-ups load them together with the contributors' partial sums).
__device__ __forceinline__ void t_resid_pre(const TArgs& a, int tile, int s, int t, float v0,
                                            float v1, float h0, float h1, float& ss) {
  const int r0 = trow(a.g, tile, s), r1 = trow(a.g, tile, s + 128);
  float* hm = a.B.h + (size_t)t * a.D.d;
  if (r0 >= 0) {
    const float h = h0 + v0;
    hm[r0] = h;
    ss = fmaf(h, h, ss);
  }
  if (r1 >= 0) {
    const float h = h1 + v1;
    hm[r1] = h;
    ss = fmaf(h, h, ss);
  }
}

// Exit head, one token, whole warp: the logits of the lane's two rows enter
// a per-lane partial, merged over the warp by a fixed shuffle tree; lane 0
// merges the result into `acc` (shared memory, one slot per warp and token).
__device__ __forceinline__ void t_head_token(const TArgs& a, int tile, int s, int t, float rs,
                                             float v0, float v1, HeadPart* acc, int lane) {
  const int r0 = trow(a.g, tile, s), r1 = trow(a.g, tile, s + 128);
  HeadPart p;
  part_empty(p);
  if (r0 >= 0) {
    const float z = v0 * rs;
    part_add(p, z, r0);
    if (a.write_logits) a.B.logits[(size_t)t * a.D.V + r0] = z;
  }
  if (r1 >= 0) {
    const float z = v1 * rs;
    part_add(p, z, r1);
    if (a.write_logits) a.B.logits[(size_t)t * a.D.V + r1] = z;
  }
  for (int off = 16; off > 0; off >>= 1) part_merge(p, part_shfl(p, off));
  if (lane == 0) part_merge(*acc, p);
}

}  // namespace

// ------------------------------------------------------------ the kernels

// Waits until *bar >= target (acquire load); false after ~2^24 polls.
__device__ __forceinline__ bool counter_wait(const uint32_t* bar, uint32_t target) {
  for (uint32_t i = 0; i < kSpinLimit; ++i) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(bar) : "memory");
    if (v >= target) return true;
    __nanosleep(32);
  }
  return false;
}


// Shared-memory views of one block (layout TL<TP, HEAD>).
template <int TP, bool HEAD>
struct Blk {
  using S = TL<TP, HEAD>;
  unsigned char* smem;
  uint64_t *full, *xfull, *empty, *bfull, *accfull, *accempty, *drain;
  uint32_t* tslot;
  int* sflag;
  float *srs, *red;
  HeadPart *run, *spl, *comb;

  __device__ explicit Blk(unsigned char* raw) {
    smem = reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(raw) + 1023) &
                                            ~static_cast<uintptr_t>(1023));
    full = reinterpret_cast<uint64_t*>(smem + S::bars);  // weights landed
    xfull = full + S::NS;                                // input slice landed
    empty = xfull + S::NS;                               // slot released by the MMAs
    bfull = empty + S::NS;                               // operand tile written
    accfull = bfull + S::NS;
    accempty = accfull + 2;
    drain = accempty + 2;
    tslot = reinterpret_cast<uint32_t*>(smem + S::tslot);
    sflag = reinterpret_cast<int*>(smem + S::flag);
    srs = reinterpret_cast<float*>(smem + S::rs);
    red = reinterpret_cast<float*>(smem + S::red);
    run = reinterpret_cast<HeadPart*>(smem + S::run);
    spl = reinterpret_cast<HeadPart*>(smem + S::spl);
    comb = reinterpret_cast<HeadPart*>(smem + S::comb);
  }

  // barriers (thread 0), TMEM allocation (the MMA warp); every thread waits
  __device__ uint32_t setup(int warp, int mma_warp) {
    if (threadIdx.x == 0) {
      for (int i = 0; i < S::NS; ++i) {
        mbar_init(&full[i], 1);
        mbar_init(&xfull[i], 1);
        mbar_init(&empty[i], 1);         // MMA commit
        mbar_init(&bfull[i], kWorkers);  // operand tile written
      }
      for (int i = 0; i < 2; ++i) {
        mbar_init(&accfull[i], 1);
        mbar_init(&accempty[i], kWorkers);
      }
      mbar_init(drain, 1);
      mbar_init_fence();
    }
    if (warp == mma_warp) tc_alloc(tslot, S::kCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    return *tslot;
  }

  // workers: zeroed operand tiles (rows past M stay zero), empty statistics
  __device__ void clear_operands(int tid) {
    uint4* z = reinterpret_cast<uint4*>(smem + S::bt);
    for (int i = tid; i < S::NS * S::BB / 16; i += kWThreads) z[i] = make_uint4(0, 0, 0, 0);
    if constexpr (HEAD)
      for (int i = tid; i < kWorkers * kLT; i += kWThreads) part_empty(run[i]);
    fence_proxy_async_smem();
    named_sync(1, kWThreads);
  }
};

// MMA issue (one thread) for the block's units [u_begin, u_begin + n) of one
// matrix: per unit both 128-row halves times four K-steps of 16, high and low
// parts as one N = 2 TP operand.  gi0 is the block's count of units before
// this matrix (ring slot and phase parity continue across the matrices of a
// chain), tc the running tile count (double-buffered TMEM accumulator).
template <int TP, bool HEAD>
__device__ bool mma_units(const Blk<TP, HEAD>& k, const TGeom& g, int u_begin, int n, int gi0,
                          int& tc, uint32_t tmem) {
  using S = TL<TP, HEAD>;
  constexpr int NS = S::NS, N = S::N;
  constexpr uint32_t idesc = idesc_bf16_f32(128, N);
  for (int i = 0; i < n; ++i) {
    const int gi = gi0 + i;
    const int u = u_begin + i;
    const int slot = gi % NS;
    const uint32_t ph = (uint32_t)(gi / NS) & 1u;
    const bool first = (i == 0) || (u % g.nks == 0);
    const bool last = (i == n - 1) || ((u + 1) % g.nks == 0);
    if (first) {
      ++tc;
      if (!mbar_wait(&k.accempty[tc & 1], ((uint32_t)(tc >> 1) & 1u) ^ 1u)) return false;
    }
    if (!mbar_wait(&k.full[slot], ph) || !mbar_wait(&k.bfull[slot], ph)) return false;
    tc_fence_after();
    const uint32_t abase = smem_u32(k.smem + S::ring + (size_t)slot * kWBytes);
    const uint32_t bbase = smem_u32(k.smem + S::bt + (size_t)slot * S::BB);
    const uint32_t dbase = tmem + (uint32_t)((tc & 1) * 2 * N);
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
      for (int kk = 0; kk < kKC / 16; ++kk)
        tc_mma_bf16(dbase + h * N, sdesc_k128(abase + h * (kWBytes / 2) + kk * 32),
                    sdesc_k128(bbase + kk * 32), idesc, !first || kk > 0);
    tc_commit(&k.empty[slot]);
    if (last) tc_commit(&k.accfull[tc & 1]);
  }
  return true;
}

// Workers (eight warps) for the block's units of one matrix: operand tiles
// from the input slices, then the fused epilogue of every tile.  The RMSNorm
// scale of the input rows is read first (from the sum-of-squares parts).
template <int TP, int KIND, bool NORM>
__device__ void worker_units(const TArgs& a, const Blk<TP, KIND == kKHead>& k, uint32_t tmem,
                             int u_begin, int n, int gi0, int& tc, bool& ok, int pos0, int M) {
  using S = TL<TP, KIND == kKHead>;
  constexpr int NS = S::NS, N = S::N;
  constexpr int LTN = TP / 2;                 // tokens per parity group read back
  constexpr int LTR = LTN < kLT ? LTN : kLT;  // ... of which can be rows (t < kMaxM)
  const TGeom& g = a.g;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, tid = threadIdx.x;
  float* srs = k.srs;
  float* red = k.red;
  int* sflag = k.sflag;
  HeadPart* run = k.run;
  HeadPart* spl = k.spl;
  if (tid < 32) {
    // RMSNorm scale of row tid: the input's sum of squares is kept as parts
    // of 256 elements, added here in part order
    float r = 1.f;
    if (a.ss_in >= 0 && tid < M) {
      const float* sp = a.B.ss_part + (size_t)a.ss_in * a.D.ss_nt * kMaxM + tid;
      float sum = 0.f;
#pragma unroll 8
      for (int c = 0; c < a.D.ss_nt; ++c) sum += __ldcg(&sp[(size_t)c * kMaxM]);
      r = 1.0f / sqrtf(sum / (float)g.K + a.D.eps);
    }
    srs[tid] = r;
  }
  named_sync(1, kWThreads);
  const int q = warp & 3, grp = warp >> 2;
  const int srow = 32 * q + lane;  // stage row of half 0 (half 1: + 128)
  float rs_t[LTN];
#pragma unroll
  for (int lt = 0; lt < LTN; ++lt) rs_t[lt] = srs[2 * lt + grp];
  const int u_end = u_begin + n;
  const int first_tile = u_begin / g.nks;

  // Residual kernels: sum of squares of the tile's 256 updated rows per
  // token (fixed order: lanes, then the four row quarters), one part of the
  // next RMSNorm's input
  auto tile_ss = [&](const float (&ssv)[LTN], int tile) {
#pragma unroll
    for (int lt = 0; lt < LTR; ++lt) {
      const float sw = warp_sum(ssv[lt]);
      if (lane == 0) red[warp * kLT + lt] = sw;
    }
    named_sync(1, kWThreads);
    if (tid < M) {
      float sum = 0.f;
      for (int qq = 0; qq < 4; ++qq) sum += red[((tid & 1) * 4 + qq) * kLT + (tid >> 1)];
      a.B.ss_part[((size_t)a.which * a.D.ss_nt + tile) * kMaxM + tid] = sum;
    }
    named_sync(1, kWThreads);
  };

  // per-tile epilogue: TMEM -> registers (high + low parts) -> fused epilogue
  auto epilogue = [&](int tile, int tcv) {
    const int buf = tcv & 1;
    if (ok) {
      const bool w = __all_sync(0xffffffffu, mbar_wait(&k.accfull[buf], (uint32_t)(tcv >> 1) & 1u));
      if (!w) {
        if (lane == 0) flag_timeout(a.B);
        ok = false;
      }
    }
    tc_fence_after();
    float v[2][TP];
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
      for (int c = 0; c < TP / 8; ++c) {
        float hi8[8], lo8[8];
        if (ok) {
          const uint32_t col =
              tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * 2 * N + h * N + c * 8);
          tc_ld8(col, hi8);
          tc_ld8(col + TP, lo8);
        } else {
#pragma unroll
          for (int e = 0; e < 8; ++e) hi8[e] = lo8[e] = 0.f;
        }
#pragma unroll
        for (int e = 0; e < 8; ++e) v[h][c * 8 + e] = hi8[e] + lo8[e];
      }
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(&k.accempty[buf]);
    const int t0 = tile * g.nks, t1 = t0 + g.nks;
    if (t0 >= u_begin && t1 <= u_end) {
      float ssv[LTN];
#pragma unroll
      for (int lt = 0; lt < LTN; ++lt) ssv[lt] = 0.f;
#pragma unroll
      for (int lt = 0; lt < LTN; ++lt) {
        const int t = 2 * lt + grp;
        if (t >= M) break;
        const float v0 = grp ? v[0][2 * lt + 1] : v[0][2 * lt];
        const float v1 = grp ? v[1][2 * lt + 1] : v[1][2 * lt];
        if constexpr (KIND == kKHead)
          t_head_token(a, tile, srow, t, rs_t[lt], v0, v1, &run[warp * kLT + lt], lane);
        else
          t_pair<KIND>(a, tile, srow, t, pos0, rs_t[lt], v0, v1, ssv[lt]);
      }
      if constexpr (KIND == kKResid) tile_ss(ssv, tile);
      return;
    }
    // Shared with neighbouring blocks.  The tile's first contributor b0 (for
    // which it is always the last tile of its range) finishes it: the others
    // publish their partial sums and count themselves in without waiting;
    // b0 waits for that count, keeps its own partial in registers and adds
    // the others' in block order.
    const int b0 = t_block_of(g, t0), b1 = t_block_of(g, t1 - 1);
    if ((int)blockIdx.x != b0) {
      const int slot2 = tile == first_tile ? 0 : 1;
      float* mine = a.B.gpart + ((size_t)blockIdx.x * 2 + slot2) * 2 * kMaxM * 128;
#pragma unroll
      for (int lt = 0; lt < LTN; ++lt) {
        const int t = 2 * lt + grp;
        if (t >= M) break;
        mine[(size_t)t * 128 + srow] = grp ? v[0][2 * lt + 1] : v[0][2 * lt];
        mine[(size_t)(kMaxM + t) * 128 + srow] = grp ? v[1][2 * lt + 1] : v[1][2 * lt];
      }
      named_sync(1, kWThreads);
      if (tid == 0) red_release_gpu(&a.B.tile_counter[tile], 1u);
      return;
    }
    // residual kernels: the rows' previous values (written by an earlier
    // phase or kernel), loaded while the contributors are counted in
    float hp0[LTN], hp1[LTN];
    if constexpr (KIND == kKResid) {
      const int r0 = trow(g, tile, srow), r1 = trow(g, tile, srow + 128);
#pragma unroll
      for (int lt = 0; lt < LTN; ++lt) {
        const int t = 2 * lt + grp;
        const float* hm = a.B.h + (size_t)(t < M ? t : 0) * a.D.d;
        hp0[lt] = (t < M && r0 >= 0) ? __ldcg(hm + r0) : 0.f;
        hp1[lt] = (t < M && r1 >= 0) ? __ldcg(hm + r1) : 0.f;
      }
    }
    if (tid == 0) {
      int contrib = 0;
      for (int b = b0; b <= b1; ++b) contrib += t_start(g, b) < t_start(g, b + 1);
      *sflag = counter_wait(&a.B.tile_counter[tile], (uint32_t)(contrib - 1)) ? 1 : 0;
      a.B.tile_counter[tile] = 0u;
    }
    named_sync(1, kWThreads);
    if (!*sflag && tid == 0) flag_timeout(a.B);
    float ss_sp[LTN];
#pragma unroll
    for (int lt = 0; lt < LTN; ++lt) ss_sp[lt] = 0.f;
    if constexpr (KIND == kKHead) {
      if (lane == 0)
        for (int lt = 0; lt < kLT; ++lt) part_empty(spl[warp * kLT + lt]);
      __syncwarp();
    }
    // Partial sums of the contributors, added in block order (independent of
    // who finishes last).  The loads of several contributors (and all
    // tokens) are issued before any is used, so the fix-up costs a few L2
    // round trips rather than one per contributor and token.  Unused slots
    // read block 0's partials (valid memory) and add zero.
    constexpr int GB = LTN <= 4 ? 4 : (LTN <= 8 ? 2 : 1);
    float u0[LTN], u1[LTN];
#pragma unroll
    for (int lt = 0; lt < LTN; ++lt) {  // b0's own partial first (0 + x: exactly x)
      const int t = 2 * lt + grp;
      u0[lt] = t < M ? (grp ? v[0][2 * lt + 1] : v[0][2 * lt]) : 0.f;
      u1[lt] = t < M ? (grp ? v[1][2 * lt + 1] : v[1][2 * lt]) : 0.f;
    }
    if (M == 1) {
      // one token (drafting, autoregressive steps): sixteen contributors per round
      for (int b = grp == 0 ? b0 + 1 : b1 + 1; b <= b1; b += 16) {
        float c0[16], c1[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const int bb = b + j;
          bool use = false;
          int sl = 0;
          if (bb <= b1) {
            const int sb = t_start(g, bb);
            use = sb != t_start(g, bb + 1);
            sl = tile == (int)(sb / g.nks) ? 0 : 1;
          }
          const float* p = a.B.gpart + ((size_t)(use ? bb : 0) * 2 + sl) * 2 * kMaxM * 128;
          const float x0 = __ldcg(&p[srow]);
          const float x1 = __ldcg(&p[(size_t)kMaxM * 128 + srow]);
          c0[j] = use ? x0 : 0.f;
          c1[j] = use ? x1 : 0.f;
        }
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          u0[0] += c0[j];
          u1[0] += c1[j];
        }
      }
    } else
      for (int b = b0 + 1; b <= b1; b += GB) {
        float c0[GB][LTN], c1[GB][LTN];
#pragma unroll
        for (int j = 0; j < GB; ++j) {
          const int bb = b + j;
          bool use = false;
          int sl = 0;
          if (bb <= b1) {
            const int sb = t_start(g, bb);
            use = sb != t_start(g, bb + 1);
            sl = tile == (int)(sb / g.nks) ? 0 : 1;
          }
          const float* p = a.B.gpart + ((size_t)(use ? bb : 0) * 2 + sl) * 2 * kMaxM * 128;
#pragma unroll
          for (int lt = 0; lt < LTN; ++lt) {
            const int t = 2 * lt + grp;
            const int tt = t < M ? t : 0;
            const float x0 = __ldcg(&p[(size_t)tt * 128 + srow]);
            const float x1 = __ldcg(&p[(size_t)(kMaxM + tt) * 128 + srow]);
            c0[j][lt] = use ? x0 : 0.f;
            c1[j][lt] = use ? x1 : 0.f;
          }
        }
#pragma unroll
        for (int j = 0; j < GB; ++j)
#pragma unroll
          for (int lt = 0; lt < LTN; ++lt) {
            u0[lt] += c0[j][lt];
            u1[lt] += c1[j][lt];
          }
      }
#pragma unroll
    for (int lt = 0; lt < LTN; ++lt) {
      const int t = 2 * lt + grp;
      if (t >= M) break;
      if constexpr (KIND == kKHead)
        t_head_token(a, tile, srow, t, rs_t[lt], u0[lt], u1[lt], &spl[warp * kLT + lt], lane);
      else if constexpr (KIND == kKResid)
        t_resid_pre(a, tile, srow, t, u0[lt], u1[lt], hp0[lt], hp1[lt], ss_sp[lt]);
      else
        t_pair<KIND>(a, tile, srow, t, pos0, rs_t[lt], u0[lt], u1[lt], ss_sp[lt]);
    }
    // the split tile's statistics: residual sums of squares as the tile's
    // part; exit-head statistics to the split slot of its first block
    if constexpr (KIND == kKResid) {
      tile_ss(ss_sp, tile);
    } else if constexpr (KIND == kKHead) {
      named_sync(1, kWThreads);
      if (tid < M) {
        HeadPart p;
        part_empty(p);
        for (int qq = 0; qq < 4; ++qq) part_merge(p, spl[((tid & 1) * 4 + qq) * kLT + (tid >> 1)]);
        static_cast<HeadPart*>(a.B.head_part)[((size_t)kMaxBlocksDev + b0) * kMaxM + tid] = p;
      }
      named_sync(1, kWThreads);
    }
  };

  int prev_tile = -1;
  for (int i = 0; i < n; ++i) {
    const int gi = gi0 + i;
    const int u = u_begin + i;
    const int slot = gi % NS;
    const int tile = u / g.nks, kc = u - tile * g.nks;
    if (i == 0 || kc == 0) ++tc;
    // operand tile of unit i, built while its weights are still in flight:
    // the slot's previous use was released before its copies were issued,
    // so only the input slice's arrival is waited for
    if (ok) {
      const bool w = __all_sync(0xffffffffu, mbar_wait(&k.xfull[slot], (uint32_t)(gi / NS) & 1u));
      if (!w) {
        if (lane == 0) flag_timeout(a.B);
        ok = false;
      }
    }
    if (ok) {
      const unsigned char* xs = k.smem + S::xs + (size_t)slot * S::XS;
      unsigned char* bt = k.smem + S::bt + (size_t)slot * S::BB;
      const int kvalid = g.K - kc * kKC;
      for (int task = tid; task < M * 8; task += kWThreads) {
        const int m = task >> 3, j = task & 7;
        const float4 x0 = *reinterpret_cast<const float4*>(xs + m * (kKC * 4) + j * 32);
        const float4 x1 = *reinterpret_cast<const float4*>(xs + m * (kKC * 4) + j * 32 + 16);
        float xv[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
        if (NORM) {
          const uint4 gq = *reinterpret_cast<const uint4*>(xs + S::XB + j * 16);
          float gv[8];
          Elem<__nv_bfloat16>::unpack(gq, gv);
#pragma unroll
          for (int e = 0; e < 8; ++e) xv[e] *= gv[e];
        }
#pragma unroll
        for (int e = 0; e < 8; ++e)
          if (j * 8 + e >= kvalid) xv[e] = 0.f;
        uint32_t hi[4], lo[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const __nv_bfloat16 h0 = __float2bfloat16_rn(xv[2 * e]);
          const __nv_bfloat16 h1 = __float2bfloat16_rn(xv[2 * e + 1]);
          hi[e] = pack_bf16(h0, h1);
          lo[e] = pack_bf16(__float2bfloat16_rn(xv[2 * e] - __bfloat162float(h0)),
                            __float2bfloat16_rn(xv[2 * e + 1] - __bfloat162float(h1)));
        }
        *reinterpret_cast<uint4*>(bt + swz(m, j)) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
        *reinterpret_cast<uint4*>(bt + swz(TP + m, j)) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
      }
      fence_proxy_async_smem();
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&k.bfull[slot]);
    // epilogue of the tile the previous unit completed
    if (i > 0 && kc == 0) epilogue(prev_tile, tc - 1);
    prev_tile = tile;
  }
  if (n > 0) epilogue(prev_tile, tc);
}

template <int TP, int KIND, bool NORM>
__global__ void __launch_bounds__(kTThreads, 1)
    k_tile(const __grid_constant__ CUtensorMap wmap, const __grid_constant__ CUtensorMap xmap,
           const TArgs a) {
  using S = TL<TP, KIND == kKHead>;
  constexpr int NS = S::NS;
  extern __shared__ unsigned char smem_raw[];
  Blk<TP, KIND == kKHead> k(smem_raw);
  unsigned char* smem = k.smem;
  const TGeom& g = a.g;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, tid = threadIdx.x;
  const int u_begin = t_start(g, blockIdx.x), u_end = t_start(g, blockIdx.x + 1);
  const int n = u_end - u_begin;
  const uint32_t tmem = k.setup(warp, kMmaWarp);
  pdl_launch_dependents();

  if (warp == kTmaWarp) {
    // ---------------- TMA: weights need nothing from earlier kernels, the
    // input slices wait for them
    if (lane == 0 && n > 0) {
      const uint64_t pol = evict_first_policy();
      tma_prefetch_desc(&wmap);
      tma_prefetch_desc(&xmap);
      auto issue_w = [&](int i) -> bool {
        const int slot = i % NS;
        if (!mbar_wait(&k.empty[slot], ((uint32_t)(i / NS) & 1u) ^ 1u)) return false;
        const int u = u_begin + i;
        const int tile = u / g.nks, kc = u - tile * g.nks;
        mbar_arrive_expect_tx(&k.full[slot], (uint32_t)kWBytes);
        unsigned char* dst = smem + S::ring + (size_t)slot * kWBytes;
#pragma unroll
        for (int b = 0; b < 4; ++b)
          tma_load_2d(dst + b * kBoxBytes, &wmap, kc * kKC, box_row(g, tile, b), &k.full[slot], pol);
        return true;
      };
      const int npre = n < NS ? n : NS;
      bool ok = true;
      for (int i = 0; i < npre && ok; ++i) ok = issue_w(i);
      pdl_wait();
      const int K = g.K;
      for (int i = 0; i < n && ok; ++i) {
        if (i >= npre) ok = issue_w(i);
        if (!ok) break;
        const int slot = i % NS;
        const int kc = (u_begin + i) % g.nks;
        unsigned char* xdst = smem + S::xs + (size_t)slot * S::XS;
        const int cols = min(kKC, K - kc * kKC);
        const uint32_t gbytes = NORM ? (uint32_t)cols * 2u : 0u;
        mbar_arrive_expect_tx(&k.xfull[slot], (uint32_t)S::XB + gbytes);
        tma_load_2d(xdst, &xmap, kc * kKC, 0, &k.xfull[slot], pol);
        if (NORM) bulk_g2s(xdst + S::XB, a.gnorm + (size_t)kc * kKC, gbytes, &k.xfull[slot], pol);
      }
      if (!ok) flag_timeout(a.B);
      // every copy has landed before the block exits
      for (int j = n > NS ? n - NS : 0; j < n; ++j) {
        mbar_wait(&k.full[j % NS], (uint32_t)(j / NS) & 1u);
        mbar_wait(&k.xfull[j % NS], (uint32_t)(j / NS) & 1u);
      }
    }
  } else if (warp == kMmaWarp) {
    // ---------------- MMA issue (one thread)
    if (lane == 0 && n > 0) {
      int tc = -1;
      if (!mma_units(k, g, u_begin, n, 0, tc, tmem)) flag_timeout(a.B);
      // every MMA has completed before TMEM is released
      tc_commit(k.drain);
      if (!mbar_wait(k.drain, 0)) flag_timeout(a.B);
    }
  } else {
    // ---------------- workers: operand tiles and epilogues
    pdl_wait();
    int pos0, M;
    resolve_rows(a.B.ctl, a.sel, pos0, M);
    if (M > TP) M = TP;  // the launcher picks TP >= M
    k.clear_operands(tid);
    int tc = -1;
    bool ok = true;
    worker_units<TP, KIND, NORM>(a, k, tmem, u_begin, n, 0, tc, ok, pos0, M);

    // ---- exit head: per-block statistics, and the last block's fixed-order merge
    if constexpr (KIND == kKHead) {
      HeadPart* run = k.run;
      HeadPart* comb = k.comb;
      int* sflag = k.sflag;
      HeadPart* sl = static_cast<HeadPart*>(a.B.head_part);
      named_sync(1, kWThreads);
      if (tid < M) {
        HeadPart p;
        part_empty(p);
        for (int qq = 0; qq < 4; ++qq) part_merge(p, run[((tid & 1) * 4 + qq) * kLT + (tid >> 1)]);
        sl[(size_t)blockIdx.x * kMaxM + tid] = p;
      }
      named_sync(1, kWThreads);
      if (tid == 0) *sflag = atom_add_acq_rel_gpu(a.B.head_counter, 1u) == (unsigned)(g.P - 1);
      named_sync(1, kWThreads);
      if (*sflag) {
        // per row: every worker thread takes blocks tid, tid + 256, ... (the
        // running and split slots loaded together), then a shuffle tree per
        // warp and a tree over the eight warps; the order does not depend on M
        for (int m = 0; m < M; ++m) {
          HeadPart p;
          part_empty(p);
          for (int b = tid; b < g.P; b += kWThreads) {
            const bool sp = t_has_split_slot(g, b);
            const HeadPart x = part_load_cg(&sl[(size_t)b * kMaxM + m]);
            const HeadPart y = part_load_cg(&sl[((size_t)kMaxBlocksDev + (sp ? b : 0)) * kMaxM + m]);
            part_merge(p, x);
            if (sp) part_merge(p, y);
          }
          for (int off = 16; off > 0; off >>= 1) part_merge(p, part_shfl(p, off));
          if (lane == 0) comb[warp] = p;
          named_sync(1, kWThreads);
          if (warp == 0) {
            HeadPart f;
            if (lane < kWorkers)
              f = comb[lane];
            else
              part_empty(f);
            for (int off = 4; off > 0; off >>= 1) part_merge(f, part_shfl(f, off));
            if (lane == 0) write_row_stats(a.B.stats[m], f, a.topk);
          }
          named_sync(1, kWThreads);
        }
        if (tid == 0) *a.B.head_counter = 0u;
      }
    }
  }

  // TMEM is released once every MMA has completed and every read is done
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kMmaWarp) tc_dealloc(tmem, S::kCols);
}

// ---------------------------------------------------------- the chain kernel
//
// One layer's MLP half and the next layer's QKV in one persistent launch:
// phase 0 O projection + residual, 1 RMSNorm + gate/up + SwiGLU, 2 down
// projection + residual, 3 (optional) RMSNorm + QKV + RoPE + KV append of the
// next layer.  Each phase is exactly the matrix pass of k_tile (same units,
// same stream-K split, same arithmetic and fix-up order, so results are bit
// for bit those of four k_tile launches).  What changes is the pipeline: a
// weight thread streams every phase's units through the ring without
// waiting for anything but free slots, so the next phase's weights arrive
// while the current phase finishes its split tiles; an input thread issues a
// phase's input slices once every block has finished the previous phase (a
// grid-wide arrival counter; the grid is one block per SM, all resident).

constexpr int kXWarp = kWorkers + 2;
constexpr int kCThreads = (kWorkers + 3) * 32;

struct ChainArgs {
  TArgs ph[4];
  int nph;
  uint32_t* bar;  // [0] arrivals of finished phases, [1] blocks done (self-resetting)
};

struct ChainMaps {
  CUtensorMap w[4];  // weights of each phase
  CUtensorMap x[4];  // input rows of each phase
};

template <int TP, bool QKV4>
__global__ void __launch_bounds__(kCThreads, 1)
    k_chain(const __grid_constant__ ChainMaps maps, const __grid_constant__ ChainArgs ca) {
  using S = TL<TP, false>;
  constexpr int NS = S::NS;
  constexpr int NPH = QKV4 ? 4 : 3;
  extern __shared__ unsigned char smem_raw[];
  Blk<TP, false> k(smem_raw);
  unsigned char* smem = k.smem;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, tid = threadIdx.x;
  const int P = ca.ph[0].g.P;
  const uint32_t tmem = k.setup(warp, kMmaWarp);
  pdl_launch_dependents();

  if (warp == kTmaWarp) {
    // ---------------- weights: every phase, back to back
    if (lane == 0) {
      const uint64_t pol = evict_first_policy();
      for (int p = 0; p < NPH; ++p) tma_prefetch_desc(&maps.w[p]);
      bool ok = true;
      int gi = 0;
      for (int p = 0; p < NPH && ok; ++p) {
        const TGeom& g = ca.ph[p].g;
        const int u_begin = t_start(g, blockIdx.x), n = t_start(g, blockIdx.x + 1) - u_begin;
        for (int i = 0; i < n; ++i, ++gi) {
          const int slot = gi % NS;
          if (!mbar_wait(&k.empty[slot], ((uint32_t)(gi / NS) & 1u) ^ 1u)) {
            ok = false;
            break;
          }
          const int u = u_begin + i;
          const int tile = u / g.nks, kc = u - tile * g.nks;
          mbar_arrive_expect_tx(&k.full[slot], (uint32_t)kWBytes);
          unsigned char* dst = smem + S::ring + (size_t)slot * kWBytes;
#pragma unroll
          for (int b = 0; b < 4; ++b)
            tma_load_2d(dst + b * kBoxBytes, &maps.w[p], kc * kKC, box_row(g, tile, b), &k.full[slot],
                        pol);
        }
      }
      if (!ok) flag_timeout(ca.ph[0].B);
      for (int j = gi > NS ? gi - NS : 0; j < gi; ++j) mbar_wait(&k.full[j % NS], (uint32_t)(j / NS) & 1u);
    }
  } else if (warp == kXWarp) {
    // ---------------- input slices: phase p after every block finished p - 1
    if (lane == 0) {
      const uint64_t pol = evict_first_policy();
      for (int p = 0; p < NPH; ++p) tma_prefetch_desc(&maps.x[p]);
      pdl_wait();
      bool ok = true;
      int gi = 0;
      for (int p = 0; p < NPH; ++p) {
        const TArgs& a = ca.ph[p];
        const TGeom& g = a.g;
        if (p > 0) {
          if (!counter_wait(ca.bar, (uint32_t)(p * P))) ok = false;
          // inputs written by other blocks' generic stores, read by TMA
          asm volatile("fence.proxy.async.global;" ::: "memory");
        }
        const int u_begin = t_start(g, blockIdx.x), n = t_start(g, blockIdx.x + 1) - u_begin;
        const bool norm = a.gnorm != nullptr;
        for (int i = 0; i < n && ok; ++i, ++gi) {
          const int slot = gi % NS;
          if (!mbar_wait(&k.empty[slot], ((uint32_t)(gi / NS) & 1u) ^ 1u)) {
            ok = false;
            break;
          }
          const int kc = (u_begin + i) % g.nks;
          unsigned char* xdst = smem + S::xs + (size_t)slot * S::XS;
          const int cols = min(kKC, g.K - kc * kKC);
          const uint32_t gbytes = norm ? (uint32_t)cols * 2u : 0u;
          mbar_arrive_expect_tx(&k.xfull[slot], (uint32_t)S::XB + gbytes);
          tma_load_2d(xdst, &maps.x[p], kc * kKC, 0, &k.xfull[slot], pol);
          if (norm) bulk_g2s(xdst + S::XB, a.gnorm + (size_t)kc * kKC, gbytes, &k.xfull[slot], pol);
        }
        if (!ok) break;
      }
      if (!ok) flag_timeout(ca.ph[0].B);
      for (int j = gi > NS ? gi - NS : 0; j < gi; ++j) mbar_wait(&k.xfull[j % NS], (uint32_t)(j / NS) & 1u);
    }
  } else if (warp == kMmaWarp) {
    // ---------------- MMA issue (one thread), every phase
    if (lane == 0) {
      int tc = -1, gi = 0;
      bool ok = true;
      for (int p = 0; p < NPH && ok; ++p) {
        const TGeom& g = ca.ph[p].g;
        const int u_begin = t_start(g, blockIdx.x), n = t_start(g, blockIdx.x + 1) - u_begin;
        ok = mma_units(k, g, u_begin, n, gi, tc, tmem);
        gi += n;
      }
      if (!ok) flag_timeout(ca.ph[0].B);
      tc_commit(k.drain);
      if (!mbar_wait(k.drain, 0)) flag_timeout(ca.ph[0].B);
    }
  } else if (warp < kWorkers) {
    // ---------------- workers, phase by phase
    pdl_wait();
    int pos0, M;
    resolve_rows(ca.ph[0].B.ctl, ca.ph[0].sel, pos0, M);
    if (M > TP) M = TP;
    k.clear_operands(tid);
    int tc = -1, gi = 0;
    bool ok = true;
    auto phase = [&](auto kind, auto norm, int p) {
      constexpr int KIND = decltype(kind)::value;
      constexpr bool NORM = decltype(norm)::value;
      const TArgs& a = ca.ph[p];
      if (p > 0) {
        // every block finished phase p - 1: one thread acquires, the CTA
        // barrier orders the other workers' reads after it (all reads of
        // other blocks' outputs go to L2)
        if (tid == 0) *k.sflag = counter_wait(ca.bar, (uint32_t)(p * P)) ? 1 : 0;
        named_sync(1, kWThreads);
        if (!*k.sflag) ok = false;
        named_sync(1, kWThreads);
      }
      const int u_begin = t_start(a.g, blockIdx.x), n = t_start(a.g, blockIdx.x + 1) - u_begin;
      worker_units<TP, KIND, NORM>(a, k, tmem, u_begin, n, gi, tc, ok, pos0, M);
      gi += n;
      // this block's outputs of phase p are written: arrive
      named_sync(1, kWThreads);
      if (tid == 0) red_release_gpu(ca.bar, 1u);
    };
    phase(std::integral_constant<int, kKResid>{}, std::false_type{}, 0);
    phase(std::integral_constant<int, kKGateUp>{}, std::true_type{}, 1);
    phase(std::integral_constant<int, kKResid>{}, std::false_type{}, 2);
    if constexpr (QKV4) phase(std::integral_constant<int, kKQKV>{}, std::true_type{}, 3);
    // the last block out resets the counters for the next launch (every
    // block has passed all of its waits by now)
    if (tid == 0 && atomicAdd(ca.bar + 1, 1u) == (uint32_t)(P - 1)) {
      ca.bar[0] = 0u;
      ca.bar[1] = 0u;
      __threadfence();
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kMmaWarp) tc_dealloc(tmem, S::kCols);
}

// ------------------------------------------------------------- host side

namespace {

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

bool get_encoder() {
  std::call_once(g_encode_once, [] {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  return g_encode != nullptr;
}

TGeom make_tgeom(const Dims& D, int N, int K, int map) {
  TGeom g{};
  g.N = N;
  g.K = K;
  g.map = map;
  g.nks = (K + kKC - 1) / kKC;
  if (map == kTMapGateUp)
    g.ntiles = (N / 2 + 127) / 128;
  else
    g.ntiles = (N + kTR - 1) / kTR;
  g.T = g.ntiles * g.nks;
  g.P = D.num_sms;
  return g;
}

template <int TP, int KIND, bool NORM>
cudaError_t tile_launch(const CUtensorMap& wm, const CUtensorMap& xm, const TArgs& a,
                        cudaStream_t st) {
  // unit indices are 32-bit: T * blocks must stay below 2^31
  if (a.g.T < 1 || a.g.T > (1 << 22) || a.g.P < 1 || a.g.P > kMaxBlocksDev)
    return cudaErrorInvalidValue;
  return launch_ex(k_tile<TP, KIND, NORM>, dim3(a.g.P), dim3(kTThreads),
                   TL<TP, KIND == kKHead>::total, st, wm, xm, a);
}

// Token rows of the instance for launches of up to mrows rows.
int tp_index(int mrows) { return mrows <= 8 ? 0 : (mrows <= 16 ? 1 : 2); }

template <int KIND, bool NORM>
cudaError_t tile_dispatch(const CUtensorMap& wm, const CUtensorMap* xm3, const TArgs& a, int mrows,
                          cudaStream_t st) {
  switch (tp_index(mrows)) {
    case 0: return tile_launch<8, KIND, NORM>(wm, xm3[0], a, st);
    case 1: return tile_launch<16, KIND, NORM>(wm, xm3[1], a, st);
    default: return tile_launch<24, KIND, NORM>(wm, xm3[2], a, st);
  }
}

template <int TP, int KIND, bool NORM>
cudaError_t prep_one() {
  return cudaFuncSetAttribute(k_tile<TP, KIND, NORM>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)TL<TP, KIND == kKHead>::total);
}

template <int TP, bool QKV4>
cudaError_t chain_launch(const ChainMaps& m, const ChainArgs& a, cudaStream_t st) {
  return launch_ex(k_chain<TP, QKV4>, dim3(a.ph[0].g.P), dim3(kCThreads), TL<TP, false>::total, st,
                   m, a);
}

template <int TP>
cudaError_t prep_chain() {
  cudaError_t e = cudaFuncSetAttribute(k_chain<TP, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)TL<TP, false>::total);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_chain<TP, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)TL<TP, false>::total);
}

template <int KIND, bool NORM>
cudaError_t prep_kind() {
  cudaError_t e = prep_one<8, KIND, NORM>();
  if (e == cudaSuccess) e = prep_one<16, KIND, NORM>();
  return e != cudaSuccess ? e : prep_one<24, KIND, NORM>();
}

}  // namespace

bool encode_weight_map(CUtensorMap* m, const void* W, int rows, int cols) {
  if (!get_encoder() || !W || ((uintptr_t)W & 15u) || ((size_t)cols * 2) % 16) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {64, 64};
  cuuint32_t es[2] = {1, 1};
  return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(W), dims, strides, box,
                  es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool encode_input_map(CUtensorMap* m, const float* x, int cols, int rows, int box_rows) {
  if (!get_encoder() || !x || ((uintptr_t)x & 15u) || ((size_t)cols * 4) % 16 || rows < 1 ||
      rows > kMaxM || box_rows < 1 || box_rows > 256)
    return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 4};
  cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
  cuuint32_t es[2] = {1, 1};
  return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(x), dims, strides, box,
                  es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                  CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

cudaError_t prepare_tile_kernels() {
  cudaError_t e;
  if ((e = prep_kind<kKPlain, false>()) != cudaSuccess) return e;
  if ((e = prep_kind<kKQKV, true>()) != cudaSuccess) return e;
  if ((e = prep_kind<kKGateUp, true>()) != cudaSuccess) return e;
  if ((e = prep_kind<kKResid, false>()) != cudaSuccess) return e;
  if ((e = prep_chain<8>()) != cudaSuccess) return e;
  if ((e = prep_chain<16>()) != cudaSuccess) return e;
  if ((e = prep_chain<24>()) != cudaSuccess) return e;
  return prep_kind<kKHead, true>();
}

// Blocks of the tensor-core kernels that can be resident on one SM at once
// (the smallest over the instances; 1 with their 200+ KB of shared memory),
// or 0 when one cannot be: the persistent grids wait on each other's blocks
// (phase barriers, split-tile fix-ups), so every block must be resident.
int tile_blocks_per_sm() {
  int lo = 1 << 30;
  auto occ = [&](const void* fn, int threads, size_t smem) {
    int nb = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, fn, threads, smem) != cudaSuccess) nb = 0;
    lo = nb < lo ? nb : lo;
  };
  occ((const void*)k_chain<8, true>, kCThreads, TL<8, false>::total);
  occ((const void*)k_chain<16, true>, kCThreads, TL<16, false>::total);
  occ((const void*)k_chain<24, true>, kCThreads, TL<24, false>::total);
  occ((const void*)k_tile<8, kKHead, true>, kTThreads, TL<8, true>::total);
  occ((const void*)k_tile<24, kKQKV, true>, kTThreads, TL<24, false>::total);
  return lo;
}

size_t tile_part_floats(int num_sms) { return (size_t)num_sms * 2 * 2 * kMaxM * 128; }

bool encode_input_maps(CUtensorMap (&m)[3], const float* x, int cols) {
  return encode_input_map(&m[0], x, cols, kMaxM, 8) && encode_input_map(&m[1], x, cols, kMaxM, 16) &&
         encode_input_map(&m[2], x, cols, kMaxM, 24);
}

cudaError_t launch_tile_part(const Dims& D, const Bufs& B, const TileMaps& tm, const LayerW& w,
                             int layer, int part, RowSel sel, int mrows, cudaStream_t st) {
  TArgs a{};
  a.D = D;
  a.B = B;
  a.sel = sel;
  a.layer = layer;
  switch (part) {
    case 0:
      a.g = make_tgeom(D, (D.Hq + 2 * D.Hkv) * D.hd, D.d, kTMapQKV);
      a.gnorm = static_cast<const __nv_bfloat16*>(w.attn_norm);
      a.ss_in = 0;
      return tile_dispatch<kKQKV, true>(*w.tm[0], tm.h, a, mrows, st);
    case 2:
      a.g = make_tgeom(D, D.d, D.qd, kTMapLinear);
      a.ss_in = -1;
      a.which = 1;
      return tile_dispatch<kKResid, false>(*w.tm[1], tm.attn_out, a, mrows, st);
    case 3:
      a.g = make_tgeom(D, 2 * D.F, D.d, kTMapGateUp);
      a.gnorm = static_cast<const __nv_bfloat16*>(w.ffn_norm);
      a.ss_in = 1;
      return tile_dispatch<kKGateUp, true>(*w.tm[2], tm.h, a, mrows, st);
    case 4:
      a.g = make_tgeom(D, D.d, D.F, kTMapLinear);
      a.ss_in = -1;
      a.which = 0;
      return tile_dispatch<kKResid, false>(*w.tm[3], tm.act, a, mrows, st);
    default:
      return cudaErrorInvalidValue;
  }
}

cudaError_t launch_tile_chain(const Dims& D, const Bufs& B, const TileMaps& tm, const LayerW& w,
                              const LayerW* next, int layer, RowSel sel, int mrows,
                              cudaStream_t st) {
  const int tp = tp_index(mrows);
  ChainArgs ca{};
  ChainMaps cm{};
  for (int p = 0; p < 4; ++p) {
    ca.ph[p].D = D;
    ca.ph[p].B = B;
    ca.ph[p].sel = sel;
    ca.ph[p].layer = layer;
    ca.ph[p].ss_in = -1;
  }
  // O projection + residual
  ca.ph[0].g = make_tgeom(D, D.d, D.qd, kTMapLinear);
  ca.ph[0].which = 1;
  cm.w[0] = *w.tm[1];
  cm.x[0] = tm.attn_out[tp];
  // RMSNorm + gate/up + SwiGLU
  ca.ph[1].g = make_tgeom(D, 2 * D.F, D.d, kTMapGateUp);
  ca.ph[1].gnorm = static_cast<const __nv_bfloat16*>(w.ffn_norm);
  ca.ph[1].ss_in = 1;
  cm.w[1] = *w.tm[2];
  cm.x[1] = tm.h[tp];
  // down projection + residual
  ca.ph[2].g = make_tgeom(D, D.d, D.F, kTMapLinear);
  ca.ph[2].which = 0;
  cm.w[2] = *w.tm[3];
  cm.x[2] = tm.act[tp];
  ca.nph = 3;
  if (next) {  // the next layer's RMSNorm + QKV + RoPE + KV append
    ca.ph[3].g = make_tgeom(D, (D.Hq + 2 * D.Hkv) * D.hd, D.d, kTMapQKV);
    ca.ph[3].gnorm = static_cast<const __nv_bfloat16*>(next->attn_norm);
    ca.ph[3].ss_in = 0;
    ca.ph[3].layer = layer + 1;
    cm.w[3] = *next->tm[0];
    cm.x[3] = tm.h[tp];
    ca.nph = 4;
  }
  for (int p = 0; p < ca.nph; ++p)
    if (ca.ph[p].g.T < 1 || ca.ph[p].g.T > (1 << 22) || ca.ph[p].g.P < 1 ||
        ca.ph[p].g.P > kMaxBlocksDev)
      return cudaErrorInvalidValue;
  ca.bar = B.chain_bar;
  switch (tp) {
    case 0: return next ? chain_launch<8, true>(cm, ca, st) : chain_launch<8, false>(cm, ca, st);
    case 1: return next ? chain_launch<16, true>(cm, ca, st) : chain_launch<16, false>(cm, ca, st);
    default: return next ? chain_launch<24, true>(cm, ca, st) : chain_launch<24, false>(cm, ca, st);
  }
}

cudaError_t launch_tile_head(const Dims& D, const Bufs& B, const TileMaps& tm,
                             const CUtensorMap& lm, const void* final_norm, int topk,
                             bool write_logits, RowSel sel, int mrows, cudaStream_t st) {
  TArgs a{};
  a.D = D;
  a.B = B;
  a.sel = sel;
  a.g = make_tgeom(D, D.V, D.d, kTMapLinear);
  a.gnorm = static_cast<const __nv_bfloat16*>(final_norm);
  a.ss_in = 0;
  a.topk = topk;
  a.write_logits = write_logits ? 1 : 0;
  return tile_dispatch<kKHead, true>(lm, tm.h, a, mrows, st);
}

cudaError_t launch_tile_plain(const Dims& D, const Bufs& B, const CUtensorMap& wm, int rows,
                              int cols, const float* x, int M, float* y, cudaStream_t st) {
  CUtensorMap xm[3];
  const int tp = tp_index(M);
  if (!encode_input_map(&xm[tp], x, cols, M, tp == 0 ? 8 : (tp == 1 ? 16 : 24)))
    return cudaErrorInvalidValue;
  TArgs a{};
  a.D = D;
  a.B = B;
  a.sel = RowSel{kRowsExplicit, 0, M, nullptr};
  a.g = make_tgeom(D, rows, cols, kTMapLinear);
  a.ss_in = -1;
  a.y = y;
  return tile_dispatch<kKPlain, false>(wm, xm, a, M, st);
}

}  // namespace ssd
