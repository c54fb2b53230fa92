// Internal definitions shared by the kernels and the C ABI layer.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "../../include/starkv.h"

namespace starkv {

constexpr int kHeadDim = 128;       // d
constexpr int kTileKeys = 128;      // keys per MMA tile (M of pass 2, N of pass 1)
constexpr int kMaxRows = 256;       // (H / G) * w window rows per group
constexpr int kMaxGroups = 32;      // G (KV heads; the global mode up to one per query head)
constexpr int kMaxCluster = 8;      // CTAs of a calibration cluster (portable cluster size)
constexpr int kMaxBatch = 32;       // sequences per launch (kernel-parameter arrays)
constexpr int kMaxBins = 64;        // K rank bins
constexpr int kMaxHist = 4096;      // K * M^2
constexpr int kMaxGrid = 16384;     // R * C
constexpr int kRawCopies = 4;       // unpooled group sums: one copy per pass-2 column quarter

// device error word bits
constexpr uint32_t kErrTimeout = 1u;
constexpr uint32_t kErrMeta = 2u;
constexpr uint32_t kErrIndex = 4u;

// Token metadata word (Sec. 3.1): bit 31 visual, 20..30 frame, 10..19 row, 0..9 col.
__host__ __device__ __forceinline__ bool meta_visual(uint32_t m) { return (m >> 31) != 0; }
__host__ __device__ __forceinline__ int meta_frame(uint32_t m) { return (m >> 20) & 0x7FF; }
__host__ __device__ __forceinline__ int meta_row(uint32_t m) { return (m >> 10) & 0x3FF; }
__host__ __device__ __forceinline__ int meta_col(uint32_t m) { return m & 0x3FF; }

// Device-resident per-(slot, layer) state, structure-of-arrays.
struct DevState {
  int32_t* n;          // [slots][layers] steps seen
  double* mi_bar;      // [slots][layers][G] MI EMA (Eq. 6)
  float* m;            // [slots][layers][G][R*C] temporal EMA m_g (Eq. 8)
  double* mi_cur;      // [slots][layers][G] MI of the current step (group_stats -> select)
  float* phi_cur;      // [slots][layers][G] phi_g of the current step
  uint32_t* err;       // device error word
};

// Hyper-parameters as the kernels use them.
struct KParams {
  int n_layers, H, G, w, R, C, pool, K, M, n_warmup, n_ramp;
  float lambda, tau, rho_mi, rho_t, delta, d_min, t_min, t_max, eps, eps_h;
  int per_head;        // selection mode: 0 = one global top-B per layer, 1 = one per KV group
  int decay_mode;      // 0 exponential (Eq. 9), 1 linear, 2 power law
  int aeb_mode;        // 0 entropy (Sec. 3.6), 1 peak confidence
  int mi_span;         // 0 every historical visual token, 1 the newest frame's
  uint64_t wait_ns;    // bounded-wait limit
};

// One sequence of a launch, as the select / group-stats / compact kernels see it.
struct SeqView {
  const __nv_bfloat16* k;
  const __nv_bfloat16* v;
  const uint32_t* meta;
  int64_t meta_layer_stride;
  int64_t meta_group_stride;   // 0: one row shared by the groups
  int L, Lp, cur_frame, budget, slot, pad_;
  __nv_bfloat16* k_out;
  __nv_bfloat16* v_out;
  uint32_t* meta_out;
  int32_t* idx;    // [n_layers][P][B]
  float* S;        // [n_layers][G][Lp] (a workspace region when the caller passed NULL)
  float* s_raw;    // [n_layers_in_launch][G][kRawCopies][raw_stride(Lp)] unpooled sums (workspace) or NULL
  float* score;    // [n_layers][P][Lp] fused score, P = 1 or G (a workspace region when NULL)
  float* stats;    // optional
  uint32_t* vis;   // [n_layers_in_launch][G][3 Lp] keys, candidate list and cells of
                   // rows too long for shared memory (workspace), else NULL
};

struct SeqBatch {
  SeqView s[kMaxBatch];
  int nseq;
  int layer0;      // first layer of the launch
  int nlayers;     // layers in the launch
};

__host__ __device__ __forceinline__ int ceil_div(int a, int b) { return (a + b - 1) / b; }

// Row stride (floats) of the unpooled group sums: L_p rounded up to 4, so that
// every row starts on a 16-byte boundary.
__host__ __device__ __forceinline__ int raw_stride(int lp) { return (lp + 3) & ~3; }

}  // namespace starkv
