// Compressed cache of Sec. 3.7, Eq. (11):
//   K' = [K_past[I]; K_rec],  V' = [V_past[I]; V_rec],  meta' likewise.
// A bit copy bound by HBM bandwidth.  A warp task is 32 consecutive output
// rows of one (tensor, group): lane i resolves the source row of output row
// i, the source rows are broadcast by shuffle, and every instruction moves
// two 256-byte rows (d = 128 bf16) as one 16-byte access per lane, with eight
// such accesses per lane in flight.  In the per-KV-head selection mode group g
// gathers its own index row I_g and writes its own metadata row.
#include "common.cuh"
#include "ptx.cuh"
#include "compact.cuh"

namespace starkv {

namespace {

constexpr int kCompactThreads = 256;
constexpr int kWarps = kCompactThreads / 32;
constexpr int kTaskRows = 32;   // output rows per warp task
constexpr int kInFlight = 8;    // 16-byte accesses per lane in flight (16 rows per warp)

__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ void st_stream(uint4* p, const uint4& v) {
  asm volatile("st.global.cs.v4.u32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w)
               : "memory");
}

}  // namespace

// grid: (blocks, nlayers, nseq).  Tasks of one (seq, layer): 2 tensors x G x
// ceil((B + w) / 32) row blocks, one per warp, strided over the grid.
__global__ void __launch_bounds__(kCompactThreads) k_compact(const __grid_constant__ SeqBatch b, int G, int w,
                                                              int per_head, uint32_t* err) {
  griddep_launch_dependents();
  griddep_wait();   // idx comes from the previous kernel
  const SeqView& sv = b.s[blockIdx.z];
  const int layer = b.layer0 + blockIdx.y;
  const int B = sv.budget, Lp = sv.Lp, L = sv.L;
  const int rows_out = B + w;
  const int lane = threadIdx.x & 31, half = lane >> 4, hl = lane & 15;
  const int P = per_head ? G : 1;   // index / metadata rows per layer
  const int32_t* idx_l = sv.idx + static_cast<int64_t>(layer) * P * B;
  const uint32_t* meta_l = sv.meta + static_cast<int64_t>(layer) * sv.meta_layer_stride;
  uint32_t* meta_out_l = sv.meta_out + static_cast<int64_t>(layer) * P * rows_out;
  const int nblk = ceil_div(rows_out, kTaskRows);
  const int ntask = 2 * G * nblk;
  for (int task = blockIdx.x * kWarps + (threadIdx.x >> 5); task < ntask; task += gridDim.x * kWarps) {
    const int tensor = task / (G * nblk);
    const int rem = task - tensor * G * nblk;
    const int g = rem / nblk, r0 = (rem - g * nblk) * kTaskRows;
    const int p = per_head ? g : 0;
    // source row of output row r0 + lane
    const int r = r0 + lane;
    int src = 0;
    if (r < rows_out) {
      src = r < B ? idx_l[static_cast<int64_t>(p) * B + r] : Lp + (r - B);
      // a kept index must name a past token (< L_p): the window rows follow it
      if (src < 0 || src >= (r < B ? Lp : L)) {   // report, copy row 0
        atomicOr(err, kErrIndex);
        src = 0;
      }
      if (tensor == 0 && g == p) meta_out_l[static_cast<int64_t>(p) * rows_out + r] = meta_l[p * sv.meta_group_stride + src];
    }
    const __nv_bfloat16* in = (tensor == 0 ? sv.k : sv.v) + (static_cast<int64_t>(layer) * G + g) * L * kHeadDim;
    __nv_bfloat16* out = (tensor == 0 ? sv.k_out : sv.v_out) + (static_cast<int64_t>(layer) * G + g) * rows_out * kHeadDim;
    const uint4* in4 = reinterpret_cast<const uint4*>(in) + hl;
    uint4* out4 = reinterpret_cast<uint4*>(out) + static_cast<int64_t>(r0) * (kHeadDim / 8) + hl;
    const int nrows = min(kTaskRows, rows_out - r0);
#pragma unroll
    for (int j0 = 0; j0 < kTaskRows; j0 += 2 * kInFlight) {
      uint4 v[kInFlight];
#pragma unroll
      for (int k = 0; k < kInFlight; ++k) {
        const int row = j0 + 2 * k + half;
        const int s_row = __shfl_sync(0xffffffffu, src, row);
        if (row < nrows) v[k] = ld_stream(in4 + static_cast<int64_t>(s_row) * (kHeadDim / 8));
      }
#pragma unroll
      for (int k = 0; k < kInFlight; ++k) {
        const int row = j0 + 2 * k + half;
        if (row < nrows) st_stream(out4 + row * (kHeadDim / 8), v[k]);
      }
    }
  }
}

cudaError_t compact_launch(const SeqBatch& b, int G, int w, int per_head, int rows_out_max, uint32_t* err,
                           cudaStream_t stream) {
  if (rows_out_max <= 0) return cudaSuccess;
  const int ntask = 2 * G * ceil_div(rows_out_max, kTaskRows);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(ceil_div(ntask, kWarps)), b.nlayers, b.nseq);
  cfg.blockDim = dim3(kCompactThreads);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // starts under the previous kernel's tail
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_compact, b, G, w, per_head, err);
}

}  // namespace starkv
