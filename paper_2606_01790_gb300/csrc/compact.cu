// Compressed cache of Sec. 3.7, Eq. (11) (Algorithm 1 last step):
//   K' = [K_past[I]; K_rec],  V' = [V_past[I]; V_rec],  meta' likewise.
// A bit copy bound by HBM bandwidth: every 256-byte row (d = 128 bf16) moves
// as one 16-lane x 16-byte vector access, four rows per half-warp in flight.
#include "common.cuh"
#include "compact.cuh"

namespace starkv {

namespace {

constexpr int kCompactThreads = 256;
constexpr int kRowsInFlight = 4;

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

// grid: (blocks, nlayers, nseq).  Rows of one (seq, layer): 2 tensors x G x (B + w).
__global__ void __launch_bounds__(kCompactThreads) k_compact(const __grid_constant__ SeqBatch b, int G, int w,
                                                              uint32_t* err) {
  const SeqView& sv = b.s[blockIdx.z];
  const int layer = b.layer0 + blockIdx.y;
  const int B = sv.budget, Lp = sv.Lp, L = sv.L;
  const int rows_out = B + w;
  const int32_t* idx = sv.idx + static_cast<int64_t>(layer) * B;
  const int64_t in_layer = static_cast<int64_t>(layer) * G * L;          // rows
  const int64_t out_layer = static_cast<int64_t>(layer) * G * rows_out;  // rows

  // metadata: one thread per output row
  const uint32_t* meta = sv.meta + static_cast<int64_t>(layer) * sv.meta_layer_stride;
  uint32_t* meta_out = sv.meta_out + static_cast<int64_t>(layer) * rows_out;
  for (int r = blockIdx.x * blockDim.x + threadIdx.x; r < rows_out; r += gridDim.x * blockDim.x) {
    int src = r < B ? idx[r] : Lp + (r - B);
    if (src < 0 || src >= L) {   // an index outside the cache: report, copy row 0
      atomicOr(err, kErrIndex);
      src = 0;
    }
    meta_out[r] = meta[src];
  }

  // K and V rows: a half-warp per row, 16 lanes x 16 bytes
  const int hl = threadIdx.x & 15;
  const int64_t n_items = 2LL * G * rows_out;
  const int64_t hw0 = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 4;
  const int64_t hstride = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 4;
  for (int64_t base = hw0; base < n_items; base += hstride * kRowsInFlight) {
    uint4 v[kRowsInFlight];
    uint4* dst[kRowsInFlight];
#pragma unroll
    for (int i = 0; i < kRowsInFlight; ++i) {
      const int64_t item = base + i * hstride;
      dst[i] = nullptr;
      if (item < n_items) {
        const int tensor = static_cast<int>(item / (static_cast<int64_t>(G) * rows_out));
        const int rem = static_cast<int>(item - static_cast<int64_t>(tensor) * G * rows_out);
        const int g = rem / rows_out, r = rem - g * rows_out;
        int src = r < B ? idx[r] : Lp + (r - B);
        if (src < 0 || src >= L) src = 0;   // reported by the metadata loop above
        const __nv_bfloat16* in = tensor == 0 ? sv.k : sv.v;
        __nv_bfloat16* out = tensor == 0 ? sv.k_out : sv.v_out;
        const uint4* s = reinterpret_cast<const uint4*>(in + (in_layer + static_cast<int64_t>(g) * L + src) * kHeadDim);
        dst[i] = reinterpret_cast<uint4*>(out + (out_layer + static_cast<int64_t>(g) * rows_out + r) * kHeadDim) + hl;
        v[i] = ld_stream(s + hl);
      }
    }
#pragma unroll
    for (int i = 0; i < kRowsInFlight; ++i)
      if (dst[i]) st_stream(dst[i], v[i]);
  }
}

cudaError_t compact_launch(const SeqBatch& b, int G, int w, int rows_out_max, int num_sms, uint32_t* err,
                           cudaStream_t stream) {
  if (rows_out_max <= 0) return cudaSuccess;
  // enough half-warps for every row of a (seq, layer) with kRowsInFlight rows each,
  // capped so the whole launch stays a few waves of the GPU
  const int64_t rows = 2LL * G * rows_out_max;
  int64_t blocks = (rows * 16 / kRowsInFlight + kCompactThreads - 1) / kCompactThreads;
  const int64_t cap = (8LL * num_sms + b.nlayers * b.nseq - 1) / (b.nlayers * b.nseq);
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  dim3 grid(static_cast<unsigned>(blocks), b.nlayers, b.nseq);
  k_compact<<<grid, kCompactThreads, 0, stream>>>(b, G, w, err);
  return cudaGetLastError();
}

}  // namespace starkv
