// Launch interface of the scoring kernels (score.cu).
#pragma once

#include "common.cuh"

namespace starkv {

constexpr int kScoreThreads = 640;   // 20 warps: TMA, MMA, 2 idle, 16 epilogue

struct ScoreSeq {
  int Lp;              // scored (historical) keys
  int nt;              // ceil(Lp / 128) key tiles per (layer, group) row
  int64_t tile_base;   // flat index of this sequence's first tile in the launch
  float* s_raw;        // [nlayers][G][kRawCopies][raw_stride(Lp)] unpooled group sums, one copy per column quarter
  const float* lse;    // [n_layers][H][w] supplied row normalisers (natural log) or NULL
};

struct ScoreParams {
  CUtensorMap tmk[kMaxBatch];    // K: dims (d, L, n_layers*G), box (64, 128, 1), 128B swizzle
  CUtensorMap tmqa[kMaxBatch];   // Q: dims (d, H*w, n_layers), box (64, min(rows, 128), 1)
  CUtensorMap tmqb[kMaxBatch];   // Q: same, box (64, rows - 128, 1) when rows > 128
  CUtensorMap tmq2[kMaxBatch];   // Q: same, box (64, n2, 1)
  ScoreSeq seq[kMaxBatch];
  int nseq, layer0, nlayers, G;
  int rows;            // (H / G) * w window rows per group
  int n2;              // rows rounded up to 16 (pass-2 MMA N)
  int n_mtiles;        // ceil(rows / 128) (pass-1 M tiles)
  int q_rows;          // shared-memory Q rows per 64-column half (= n2)
  int kstages;         // K-tile pipeline depth (from the shared-memory budget)
  int grid1;           // pass-1 grid size (defines the partial-slot partition)
  int64_t total_tiles;
  float scale2;        // log2(e) / sqrt(d)
  float2* partials;    // [total_tiles][kMaxRows] (max2, sum) at each piece's first tile
  uint32_t* err;
  uint64_t wait_ns;
};

size_t score_smem_bytes(int q_rows, int kstages);
int score_kstages(int q_rows);
cudaError_t score_configure();
cudaError_t score_lse_launch(const ScoreParams& p, int grid, cudaStream_t stream);
cudaError_t score_accum_launch(const ScoreParams& p, int grid, cudaStream_t stream);
cudaError_t pool_launch(const SeqBatch& b, int G, int H, int pool, int lp_max, cudaStream_t stream);
cudaError_t wait_probe_launch(uint32_t* err, uint64_t limit_ns, cudaStream_t stream);

}  // namespace starkv
