// Launch interface of the calibration / selection kernel (select.cu).
#pragma once

#include "common.cuh"

namespace starkv {

// Tokens per (layer, group) row whose keys and cells the kernel keeps in
// shared memory; longer rows use the workspace region SeqView::vis.
int calibrate_capacity(int K, int M, int R, int C);
cudaError_t select_configure();
// MI, temporal factor, prior, temperature, fused score and top-B of every
// (seq, layer) of the batch: one cluster of min(G, 8) CTAs each.  With from_raw the
// kernel first pools the unpooled group sums into S.
cudaError_t calibrate_launch(const SeqBatch& b, const KParams& kp, const DevState& st, bool from_raw, int lp_max,
                             cudaStream_t stream);

}  // namespace starkv
