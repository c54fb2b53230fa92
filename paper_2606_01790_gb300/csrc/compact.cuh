// Launch interface of the KV compaction kernel (compact.cu).
#pragma once

#include "common.cuh"

namespace starkv {

// per_head: idx and meta_out hold one row per KV group ([G][B], [G][B + w]).
cudaError_t compact_launch(const SeqBatch& b, int G, int w, int per_head, int rows_out_max, uint32_t* err,
                           cudaStream_t stream);

}  // namespace starkv
