// Launch interface of the KV compaction kernel (compact.cu).
#pragma once

#include "common.cuh"

namespace starkv {

cudaError_t compact_launch(const SeqBatch& b, int G, int w, int rows_out_max, int num_sms, uint32_t* err,
                           cudaStream_t stream);

}  // namespace starkv
