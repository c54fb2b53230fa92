// Launch interface of the calibration / selection kernels (select.cu).
#pragma once

#include "common.cuh"

namespace starkv {

size_t group_stats_smem_bytes(int R, int C);
cudaError_t select_configure();
// MI_g, phi_g and the m_g update per (seq, layer, group); with from_raw the
// kernel first pools the unpooled sums into S.
cudaError_t group_stats_launch(const SeqBatch& b, const KParams& kp, const DevState& st, bool from_raw,
                               cudaStream_t stream);
// Prior, temperature, fused score and top-B per (seq, layer).
cudaError_t select_launch(const SeqBatch& b, const KParams& kp, const DevState& st, cudaStream_t stream);

}  // namespace starkv
