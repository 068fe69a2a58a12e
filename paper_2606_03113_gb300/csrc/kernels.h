// kernels.h -- host-side launchers of the engine's kernels (internal).
#pragma once

#include "common.cuh"

namespace ssd {

// Statistics partial of one block of vocabulary rows (exit head, first stage).
struct HeadPart {
  float mx;  // max logit (== tv[0] when the block has rows)
  float S;   // sum exp(z - mx)
  float T;   // sum exp(z - mx) (z - mx)
  float tv[kTopK];
  int32_t ti[kTopK];
};

// Per-block partial slots of the streamed kernels (running + split), for up
// to kMaxBlocks blocks.
constexpr int kMaxBlocks = 512;
inline int head_tiles(int V) { return (V + 15) / 16; }

// Tensor maps of the engine's fp32 input buffers ([kMaxM][K] each), read by
// the bf16 tensor-core kernels one 64-column slice per unit.
struct TileMaps {
  CUtensorMap h[3], attn_out[3], act[3];  // boxes of 8, 16, 24 rows
};

// Encodes the tensor map of a bf16 weight matrix [rows][cols] (64 x 64 boxes,
// 128-byte swizzle) or of an fp32 input [rows][cols] (64 x kMaxM boxes).
bool encode_weight_map(CUtensorMap* m, const void* W, int rows, int cols);
bool encode_input_map(CUtensorMap* m, const float* x, int cols, int rows, int box_rows);
bool encode_input_maps(CUtensorMap (&m)[3], const float* x, int cols);
cudaError_t prepare_tile_kernels();
// Resident blocks per SM of the tensor-core kernels (0: cannot be resident).
int tile_blocks_per_sm();
// Floats of the tensor-core kernels' split-tile partials for `num_sms` blocks.
size_t tile_part_floats(int num_sms);
cudaError_t launch_tile_part(const Dims& D, const Bufs& B, const TileMaps& tm, const LayerW& w,
                             int layer, int part, RowSel sel, int mrows, cudaStream_t st);
// One launch of a layer's O projection, gate/up and down (and, with next, the
// next layer's QKV) as the phases of one persistent kernel.
cudaError_t launch_tile_chain(const Dims& D, const Bufs& B, const TileMaps& tm, const LayerW& w,
                              const LayerW* next, int layer, RowSel sel, int mrows,
                              cudaStream_t st);
cudaError_t launch_tile_head(const Dims& D, const Bufs& B, const TileMaps& tm,
                             const CUtensorMap& lm, const void* final_norm, int topk,
                             bool write_logits, RowSel sel, int mrows, cudaStream_t st);
cudaError_t launch_tile_plain(const Dims& D, const Bufs& B, const CUtensorMap& wm, int rows,
                              int cols, const float* x, int M, float* y, cudaStream_t st);

// mrows is the largest number of rows a launch may see: 1 selects the
// single-row kernels, more the multi-row ones (bf16: the tensor-core instance
// with 8, 16 or 24 token rows, the smallest that holds mrows).  big
// (embedding, attention) is mrows > 1.
cudaError_t launch_embed(const Dims& D, const Bufs& B, int dtype, const void* embed, RowSel sel,
                         bool big, cudaGraphConditionalHandle set_lstar_switch, cudaStream_t st);
cudaError_t launch_layer(const Dims& D, const Bufs& B, int dtype, const LayerW& w,
                         const TileMaps* tm, int layer, RowSel sel, int mrows, cudaStream_t st);
// One kernel of a layer (0 qkv, 1 attention + combine, 2 o, 3 gate/up, 4 down).
cudaError_t launch_layer_part(const Dims& D, const Bufs& B, int dtype, const LayerW& w,
                              const TileMaps* tm, int layer, int part, RowSel sel, int mrows,
                              cudaStream_t st);
cudaError_t launch_head(const Dims& D, const Bufs& B, int dtype, const void* lm_head,
                        const CUtensorMap* lm_map, const TileMaps* tm, const void* final_norm,
                        int topk, bool write_logits, RowSel sel, int mrows, cudaStream_t st);
cudaError_t launch_round_begin(const Dims& D, const Bufs& B, cudaGraphConditionalHandle draft_if,
                               cudaStream_t st);
cudaError_t launch_decide(const Dims& D, const Bufs& B, int mode, int cand_idx, int is_last,
                          int layer, const void* final_norm, int dtype,
                          cudaGraphConditionalHandle next_if,
                          cudaGraphConditionalHandle draft_while, cudaStream_t st);
cudaError_t launch_draft_begin(const Bufs& B, cudaGraphConditionalHandle draft_while,
                               cudaStream_t st);
cudaError_t launch_accept(const Dims& D, const Bufs& B, cudaGraphConditionalHandle gen_while,
                          cudaStream_t st);
cudaError_t launch_begin_call(const Bufs& B, int max_new, cudaStream_t st);
cudaError_t launch_reset_sequence(const Bufs& B, cudaStream_t st);
cudaError_t launch_trace_push(const Bufs& B, int first_row, int n_rows, cudaStream_t st);
cudaError_t launch_set_pending(const Dims& D, const Bufs& B, int stats_row, int token, int pos,
                               cudaStream_t st);
cudaError_t launch_qnet_eval(const Bufs& B, int hidden, const float* states, int n, float* q,
                             cudaStream_t st);
cudaError_t launch_gemv_plain(const Dims& D, const Bufs& B, int dtype, const void* W, int rows,
                              int cols, const float* x, int M, float* y, cudaStream_t st);
// Raises the dynamic shared-memory limit of every streamed-kernel instance.
cudaError_t prepare_gemv_kernels();
cudaError_t launch_synth_fill(void* dst, int dtype, uint64_t n, uint32_t seed, uint32_t tid,
                              double sigma, cudaStream_t st);
cudaError_t launch_read_probe(const void* src, uint64_t bytes, uint32_t* sink, cudaStream_t st);
cudaError_t launch_kv_to_f32(const Dims& D, const Bufs& B, int dtype, int layer, int kind,
                             int head, int p0, int n, float* out, cudaStream_t st);

enum DecideMode : int { kDecideWalk = 0, kDecideDraft = 1 };

}  // namespace ssd
