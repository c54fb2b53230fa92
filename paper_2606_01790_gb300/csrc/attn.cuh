// Launch interface of the window-attention producer (attn.cu).
#pragma once

#include "common.cuh"

namespace starkv {

constexpr int kAttnThreads = 512;   // 16 warps: TMA, MMA, 2 idle, 8 softmax, 4 V conversion
constexpr int kAttnUnitKeys = 64;   // keys per pipeline unit

struct AttnSeq {
  int Lp;              // past keys
  int nu;              // ceil(Lp / 64) units per (layer, group) row
  int64_t unit_base;   // flat index of this sequence's first unit in the launch
  float* o;            // [n_layers][H][w][d] attention output, or NULL
  float* lse;          // [n_layers][H][w] natural-log normaliser
};

struct AttnParams {
  CUtensorMap tmk[kMaxBatch];    // K: dims (d, L, n_layers*G), box (64, 64, 1), 128B swizzle
  CUtensorMap tmv[kMaxBatch];    // V: the same
  CUtensorMap tmqa[kMaxBatch];   // Q: dims (d, H*w, n_layers), box (64, min(rows, 128), 1)
  CUtensorMap tmqb[kMaxBatch];   // Q: box (64, rows - 128, 1) when rows > 128
  AttnSeq seq[kMaxBatch];
  int nseq, layer0, nlayers, G;
  int rows;            // (H / G) * w window rows per group
  int n_mtiles;        // ceil(rows / 128)
  int q_rows;          // rows rounded up to 16 (shared-memory Q rows per half)
  int kv_stages;       // depth of the K and V rings (attn_kv_stages)
  int grid;            // CTAs of the main kernel (defines the piece partition)
  int64_t total_units;
  float scale2;        // log2(e) / sqrt(d)
  float2* part_ml;     // [nrows + grid][256] (reference m, sum l) of each piece
  float* part_o;       // [nrows + grid][256][128] unnormalised output of each piece
  uint32_t* err;
  uint64_t wait_ns;
};

size_t attn_smem_bytes(int q_rows, int kv_stages);
// deepest K / V ring (at most 4) that fits the shared memory
int attn_kv_stages(int q_rows);
cudaError_t attn_configure();
// Slots of piece partials a launch needs: one per (seq, layer, group) row plus
// one per CTA of the main kernel.
inline int64_t attn_slots(int nrows, int grid) { return static_cast<int64_t>(nrows) + grid; }
// Main kernel over the flat (seq, layer, group, 64-key unit) space (nothing
// when it is empty), then the per-row combine of the pieces into o and lse.
cudaError_t attn_main_launch(const AttnParams& p, cudaStream_t stream);
cudaError_t attn_combine_launch(const AttnParams& p, cudaStream_t stream);

}  // namespace starkv
