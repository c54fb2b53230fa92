// Calibration and selection of Sec. 3.4 - 3.7 (Algorithm 1 from s_bar to I).
//
// k_group_stats, one CTA per (seq, layer, group g):
//   (optionally) AvgPool1D + group mean of the unpooled sums -> S[g, :]   (Eqs. 3-4)
//   RankBin: K equal-frequency bins of S[g, visual] by an exact multi-target
//            radix select (4 x 8-bit digit passes) on order-preserving keys,
//            ties broken by position with a block-wide ordered count;
//   SpatialBin + joint histogram (shared-memory atomics) -> plug-in MI_g  (Eq. 5)
//   phi_g = cos(current-frame row on the patch grid, m_g); m_g EMA update (Eq. 8)
// k_select, one CTA per (seq, layer):
//   MI EMA -> min-max -> softmax prior w (Eqs. 6-7), lambda schedule;
//   s_bar, g*, entropy H and temperature T (Sec. 3.6);
//   s_t = max(s_bar beta D, 0)^(1/T) (Eq. final_score, Eq. 9);
//   global top-B with ties to the lower index by radix select on
//   order-preserving keys + ordered stream compaction -> ascending indices.
#include "common.cuh"
#include "select.cuh"

namespace starkv {

namespace {

constexpr int kStatsThreads = 512;
constexpr int kSelectThreads = 1024;
constexpr int kMaxTargets = 15;   // K - 1 with K <= 16

// Order-preserving map float -> uint32 (a < b  <=>  key(a) < key(b) for non-NaN).
__device__ __forceinline__ uint32_t order_key(float x) {
  const uint32_t u = __float_as_uint(x);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

template <typename T>
__device__ __forceinline__ T warp_sum(T v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Block-wide sum (all threads get the result).  `red` holds >= 32 T.
template <typename T>
__device__ T block_sum(T v, T* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  T t = lane < nw ? red[lane] : T(0);
  t = warp_sum(t);
  return t;
}

// Warp-cooperative search in a 256-bin histogram: the digit whose bin holds
// rank `rank` (0-based) and the count of keys in lower bins.
__device__ __forceinline__ void find_digit(const int* hist, int rank, int* digit, int* below) {
  const int lane = threadIdx.x & 31;
  int local[8];
  int sum = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    local[i] = hist[lane * 8 + i];
    sum += local[i];
  }
  int incl = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  const int excl = incl - sum;
  const unsigned hit = __ballot_sync(0xffffffffu, rank >= excl && rank < incl);
  const int src = __ffs(hit) - 1;
  if (lane == src) {
    int c = excl;
    for (int i = 0; i < 8; ++i) {
      if (rank < c + local[i]) {
        *digit = lane * 8 + i;
        *below = c;
        break;
      }
      c += local[i];
    }
  }
}

// Exclusive scan of one int per thread over the block; `tmp` holds >= 32 ints.
__device__ int block_exclusive_scan(int v, int* tmp, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  __syncthreads();
  if (lane == 31) tmp[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int w = lane < nw ? tmp[lane] : 0;
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += y;
    }
    if (lane < nw) tmp[lane] = wi - w;
    if (lane == nw - 1) tmp[32] = wi;
  }
  __syncthreads();
  if (total) *total = tmp[32];
  return tmp[warp] + incl - v;
}

struct StatsShared {
  int hist[kMaxTargets][256];
  uint32_t prefix[kMaxTargets];
  int rem[kMaxTargets];
  int less[kMaxTargets];
  int reach[kMaxTargets];
  int eqbase[kMaxTargets];
  int digit[kMaxTargets];
  int below[kMaxTargets];
  int tmp[33];
  double dred[32];
  int joint[kMaxHist];
};

}  // namespace

template <bool FROM_RAW>
__global__ void __launch_bounds__(kStatsThreads) k_group_stats(const __grid_constant__ SeqBatch b,
                                                               const __grid_constant__ KParams kp,
                                                               DevState st) {
  extern __shared__ __align__(16) uint8_t smem_raw[];
  StatsShared& sh = *reinterpret_cast<StatsShared*>(smem_raw);
  float* cur = reinterpret_cast<float*>(smem_raw + sizeof(StatsShared));  // [R*C]

  const SeqView& sv = b.s[blockIdx.z];
  const int g = blockIdx.x, ll = blockIdx.y, layer = b.layer0 + ll;
  const int Lp = sv.Lp, G = kp.G, K = kp.K, M = kp.M, R = kp.R, C = kp.C;
  const int tid = threadIdx.x, nth = blockDim.x;
  const int warp = tid >> 5, lane = tid & 31;
  float* S = sv.S + (static_cast<int64_t>(layer) * G + g) * Lp;
  const uint32_t* meta = sv.meta + static_cast<int64_t>(layer) * sv.meta_layer_stride;
  const int sl = sv.slot * kp.n_layers + layer;

  // ---- Eqs. (3)-(4): pool along tokens and average the group's heads
  if (FROM_RAW) {
    const float* raw = sv.s_raw + static_cast<int64_t>(ll * G + g) * Lp;
    const float scale = static_cast<float>(G) / static_cast<float>(kp.H) / static_cast<float>(kp.pool);
    const int half = kp.pool >> 1;
    for (int t = tid; t < Lp; t += nth) {
      float acc = 0.f;
      for (int j = -half; j <= half; ++j) {
        const int u = t + j;
        if (u >= 0 && u < Lp) acc += raw[u];
      }
      S[t] = acc * scale;
    }
  }
  // ---- count visual tokens, validate their patch coordinates
  int nv = 0;
  for (int t = tid; t < Lp; t += nth) {
    const uint32_t mt = meta[t];
    if (meta_visual(mt)) {
      ++nv;
      if (meta_row(mt) >= R || meta_col(mt) >= C) atomicOr(st.err, kErrMeta);
    }
  }
  for (int i = tid; i < K * M * M; i += nth) sh.joint[i] = 0;
  for (int i = tid; i < R * C; i += nth) cur[i] = 0.f;
  nv = static_cast<int>(block_sum<double>(static_cast<double>(nv), sh.dred) + 0.5);
  const int N = nv;
  const int nt = K - 1;
  if (tid < nt) {
    const int b1 = tid + 1;
    const int Rb = static_cast<int>((static_cast<int64_t>(b1) * N + K - 1) / K);  // ceil(bN/K)
    sh.reach[tid] = Rb < N;
    sh.rem[tid] = Rb;
    sh.prefix[tid] = 0;
    sh.less[tid] = 0;
  }
  __syncthreads();

  double mi = 0.0;
  if (N > 0) {
    // ---- Sec. 3.4 RankBin: the key at each boundary rank, 4 radix passes
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      const int nh = pass == 0 ? 1 : nt;   // pass 0: one histogram serves every target
      for (int i = tid; i < nh * 256; i += nth) (&sh.hist[0][0])[i] = 0;
      __syncthreads();
      for (int t = tid; t < Lp; t += nth) {
        if (!meta_visual(meta[t])) continue;
        const uint32_t u = order_key(S[t]);
        if (pass == 0) {
          atomicAdd(&sh.hist[0][u >> 24], 1);
        } else {
          for (int j = 0; j < nt; ++j)
            if (sh.reach[j] && ((u ^ sh.prefix[j]) >> (shift + 8)) == 0)
              atomicAdd(&sh.hist[j][(u >> shift) & 255], 1);
        }
      }
      __syncthreads();
      if (warp < nt && sh.reach[warp]) {
        find_digit(pass == 0 ? sh.hist[0] : sh.hist[warp], sh.rem[warp], &sh.digit[warp], &sh.below[warp]);
        __syncwarp();
        if (lane == 0) {
          sh.prefix[warp] |= static_cast<uint32_t>(sh.digit[warp]) << shift;
          sh.rem[warp] -= sh.below[warp];
          sh.less[warp] += sh.below[warp];
        }
      }
      __syncthreads();
    }
    // ---- ties: rank among equal keys in index order (contiguous chunks per thread)
    const int cs = ceil_div(Lp, nth);
    const int t0 = min(Lp, tid * cs), t1 = min(Lp, t0 + cs);
    int eq_local[kMaxTargets];
    for (int j = 0; j < nt; ++j) eq_local[j] = 0;
    for (int t = t0; t < t1; ++t) {
      if (!meta_visual(meta[t])) continue;
      const uint32_t u = order_key(S[t]);
      for (int j = 0; j < nt; ++j) eq_local[j] += (sh.reach[j] && u == sh.prefix[j]);
    }
    for (int j = 0; j < nt; ++j) eq_local[j] = block_exclusive_scan(eq_local[j], sh.tmp, nullptr);
    // ---- bins, spatial cells, joint histogram
    const int MM = M * M;
    for (int t = t0; t < t1; ++t) {
      const uint32_t mt = meta[t];
      if (!meta_visual(mt)) continue;
      const uint32_t u = order_key(S[t]);
      int bin = 0;
      for (int j = 0; j < nt; ++j) {
        if (!sh.reach[j]) continue;
        const uint32_t v = sh.prefix[j];
        if (u > v || (u == v && eq_local[j] >= sh.rem[j])) ++bin;
        eq_local[j] += (u == v);
      }
      const int r = meta_row(mt), c = meta_col(mt);
      if (r < R && c < C) atomicAdd(&sh.joint[bin * MM + (r * M / R) * M + (c * M / C)], 1);
    }
    __syncthreads();
    // ---- Eq. (5): plug-in MI from the joint histogram (fp64)
    const double invN = 1.0 / static_cast<double>(N);
    for (int e = tid; e < K * MM; e += nth) {
      const int n = sh.joint[e];
      if (n == 0) continue;
      const int bb = e / MM, cc = e - bb * MM;
      int nb = 0, nc = 0;
      for (int i = 0; i < MM; ++i) nb += sh.joint[bb * MM + i];
      for (int i = 0; i < K; ++i) nc += sh.joint[i * MM + cc];
      mi += n * invN * log(static_cast<double>(n) * N / (static_cast<double>(nb) * nc));
    }
  }
  mi = block_sum<double>(mi, sh.dred);

  // ---- Sec. 3.5: current-frame row on the patch grid, phi_g, m_g update
  for (int t = tid; t < Lp; t += nth) {
    const uint32_t mt = meta[t];
    if (meta_visual(mt) && meta_frame(mt) == sv.cur_frame) {
      const int r = meta_row(mt), c = meta_col(mt);
      if (r < R && c < C) atomicAdd(&cur[r * C + c], S[t]);
    }
  }
  __syncthreads();
  float* m = st.m + static_cast<int64_t>(sl * G + g) * (R * C);
  double dot = 0.0, ncur = 0.0, nm = 0.0;
  for (int i = tid; i < R * C; i += nth) {
    const double a = cur[i], bm = m[i];
    dot += a * bm;
    ncur += a * a;
    nm += bm * bm;
  }
  dot = block_sum<double>(dot, sh.dred);
  ncur = block_sum<double>(ncur, sh.dred);
  nm = block_sum<double>(nm, sh.dred);
  float phi = 0.f;
  if (ncur > 0.0) {
    if (nm > 0.0) {
      phi = static_cast<float>(dot / (sqrt(ncur) * sqrt(nm)));
      const float rt = kp.rho_t;
      for (int i = tid; i < R * C; i += nth) m[i] = rt * m[i] + (1.f - rt) * cur[i];
    } else {
      for (int i = tid; i < R * C; i += nth) m[i] = cur[i];
    }
  }
  if (tid == 0) {
    st.mi_cur[sl * G + g] = mi;
    st.phi_cur[sl * G + g] = phi;
  }
}

__global__ void __launch_bounds__(kSelectThreads) k_select(const __grid_constant__ SeqBatch b,
                                                           const __grid_constant__ KParams kp,
                                                           DevState st) {
  __shared__ int hist[256];
  __shared__ int tmp[33];
  __shared__ double dred[32];
  __shared__ float w_s[kMaxGroups], phi_s[kMaxGroups];
  __shared__ float lam_s;
  __shared__ int digit_s, below_s;

  const SeqView& sv = b.s[blockIdx.y];
  const int ll = blockIdx.x, layer = b.layer0 + ll;
  const int Lp = sv.Lp, G = kp.G;
  const int tid = threadIdx.x, nth = blockDim.x, warp = tid >> 5;
  const float* S = sv.S + static_cast<int64_t>(layer) * G * Lp;
  const uint32_t* meta = sv.meta + static_cast<int64_t>(layer) * sv.meta_layer_stride;
  float* score = sv.score + static_cast<int64_t>(layer) * Lp;
  const int sl = sv.slot * kp.n_layers + layer;
  float* stats = sv.stats ? sv.stats + static_cast<int64_t>(layer) * (8 + 4 * G) : nullptr;

  // ---- Eqs. (6)-(7): MI EMA, min-max, softmax prior; lambda schedule
  if (tid == 0) {
    const int n = st.n[sl];
    double mib[kMaxGroups];
    double lo = 1e300, hi = -1e300;
    for (int g = 0; g < G; ++g) {
      const double cur = st.mi_cur[sl * G + g];
      const double prev = st.mi_bar[sl * G + g];
      mib[g] = n == 0 ? cur : kp.rho_mi * prev + (1.0 - kp.rho_mi) * cur;
      st.mi_bar[sl * G + g] = mib[g];
      lo = fmin(lo, mib[g]);
      hi = fmax(hi, mib[g]);
    }
    double e[kMaxGroups], zmax = -1e300, zs = 0.0;
    for (int g = 0; g < G; ++g) {
      e[g] = ((mib[g] - lo) / ((hi - lo) + kp.eps)) / kp.tau;
      zmax = fmax(zmax, e[g]);
    }
    for (int g = 0; g < G; ++g) {
      e[g] = exp(e[g] - zmax);
      zs += e[g];
    }
    for (int g = 0; g < G; ++g) {
      w_s[g] = static_cast<float>(e[g] / zs);
      phi_s[g] = st.phi_cur[sl * G + g];
    }
    float lam = 0.f;
    if (n >= kp.n_warmup)
      lam = kp.n_ramp <= 0 ? kp.lambda
                           : kp.lambda * fminf(1.f, static_cast<float>(n - kp.n_warmup) / kp.n_ramp);
    lam_s = lam;
    if (stats) {
      stats[2] = lam;
      stats[3] = static_cast<float>(n);
      stats[6] = static_cast<float>(sv.budget);
      stats[7] = 0.f;
      for (int g = 0; g < G; ++g) {
        stats[8 + g] = static_cast<float>(st.mi_cur[sl * G + g]);
        stats[8 + G + g] = static_cast<float>(mib[g]);
        stats[8 + 2 * G + g] = w_s[g];
        stats[8 + 3 * G + g] = phi_s[g];
      }
    }
    st.n[sl] = n + 1;
  }
  __syncthreads();

  // ---- Eq. (4): s_bar; Sec. 3.6: Z = sum s_bar
  const float invG = 1.f / static_cast<float>(G);
  double z = 0.0;
  int nv = 0;
  for (int t = tid; t < Lp; t += nth) {
    float acc = 0.f;
    for (int g = 0; g < G; ++g) acc += S[static_cast<int64_t>(g) * Lp + t];
    const float sbar = acc * invG;
    score[t] = sbar;
    z += sbar;
    nv += meta_visual(meta[t]);
  }
  z = block_sum<double>(z, dred);
  const double nvd = block_sum<double>(static_cast<double>(nv), dred);
  // ---- Sec. 3.6: H = -sum p log(p + eps) / log L_p, T
  const float invz = static_cast<float>(1.0 / (z + kp.eps_h));
  double hs = 0.0;
  for (int t = tid; t < Lp; t += nth) {
    const float p = score[t] * invz;
    hs += static_cast<double>(p * logf(p + kp.eps_h));
  }
  hs = block_sum<double>(hs, dred);
  const double Hn = Lp > 1 ? -hs / log(static_cast<double>(Lp)) : 0.0;
  const float T = static_cast<float>(kp.t_min + (kp.t_max - kp.t_min) * Hn);
  const float invT = 1.f / T;
  if (tid == 0 && stats) {
    stats[0] = static_cast<float>(Hn);
    stats[1] = T;
    stats[4] = static_cast<float>(z);
    stats[5] = static_cast<float>(nvd);
  }
  // ---- Eq. (final_score) with Eq. (9): fused score
  const float lam = lam_s;
  for (int t = tid; t < Lp; t += nth) {
    float best = S[t];
    int gs = 0;
    for (int g = 1; g < G; ++g) {
      const float v = S[static_cast<int64_t>(g) * Lp + t];
      if (v > best) {
        best = v;
        gs = g;
      }
    }
    const float sbar = score[t];
    const float beta = (1.f - lam) + lam * static_cast<float>(G) * w_s[gs];
    float d = 1.f;
    const uint32_t mt = meta[t];
    if (meta_visual(mt)) {
      const float df = static_cast<float>(sv.cur_frame - meta_frame(mt));
      d = kp.d_min + (1.f - kp.d_min) * expf(-kp.delta * df * phi_s[gs]);
    }
    score[t] = powf(fmaxf(sbar * beta * d, 0.f), invT);
  }
  __syncthreads();

  // ---- Sec. 3.7: global top-B, ties to the lower index
  const int B = sv.budget;
  if (B <= 0) return;
  int32_t* idx = sv.idx + static_cast<int64_t>(layer) * B;
  // descending order of s = ascending order of ~key(s)
  uint32_t prefix = 0;
  int rank = B - 1, less = 0;
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    for (int i = tid; i < 256; i += nth) hist[i] = 0;
    __syncthreads();
    for (int t = tid; t < Lp; t += nth) {
      const uint32_t u = ~order_key(score[t]);
      if (pass == 0 || ((u ^ prefix) >> (shift + 8)) == 0) atomicAdd(&hist[(u >> shift) & 255], 1);
    }
    __syncthreads();
    if (warp == 0) find_digit(hist, rank, &digit_s, &below_s);
    __syncthreads();
    prefix |= static_cast<uint32_t>(digit_s) << shift;
    rank -= below_s;
    less += below_s;
    __syncthreads();
  }
  // selected: u < prefix, or u == prefix among the first rank + 1 equal keys
  const int cs = ceil_div(Lp, nth);
  const int t0 = min(Lp, tid * cs), t1 = min(Lp, t0 + cs);
  int nlt = 0, neq = 0;
  for (int t = t0; t < t1; ++t) {
    const uint32_t u = ~order_key(score[t]);
    nlt += u < prefix;
    neq += u == prefix;
  }
  int lt_before = block_exclusive_scan(nlt, tmp, nullptr);
  int eq_before = block_exclusive_scan(neq, tmp, nullptr);
  for (int t = t0; t < t1; ++t) {
    const uint32_t u = ~order_key(score[t]);
    int pos = -1;
    if (u < prefix) {
      pos = lt_before + min(eq_before, rank + 1);
      ++lt_before;
    } else if (u == prefix) {
      if (eq_before <= rank) pos = lt_before + eq_before;
      ++eq_before;
    }
    if (pos >= B) atomicOr(st.err, kErrIndex);   // cannot happen for a correct select
    else if (pos >= 0) idx[pos] = t;
  }
}

size_t group_stats_smem_bytes(int R, int C) { return sizeof(StatsShared) + sizeof(float) * R * C; }

cudaError_t select_configure() {
  const int bytes = static_cast<int>(group_stats_smem_bytes(128, 128));
  cudaError_t e = cudaFuncSetAttribute(k_group_stats<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_group_stats<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

cudaError_t group_stats_launch(const SeqBatch& b, const KParams& kp, const DevState& st, bool from_raw,
                               cudaStream_t stream) {
  dim3 grid(kp.G, b.nlayers, b.nseq);
  const size_t bytes = group_stats_smem_bytes(kp.R, kp.C);
  if (from_raw)
    k_group_stats<true><<<grid, kStatsThreads, bytes, stream>>>(b, kp, st);
  else
    k_group_stats<false><<<grid, kStatsThreads, bytes, stream>>>(b, kp, st);
  return cudaGetLastError();
}

cudaError_t select_launch(const SeqBatch& b, const KParams& kp, const DevState& st, cudaStream_t stream) {
  dim3 grid(b.nlayers, b.nseq);
  k_select<<<grid, kSelectThreads, 0, stream>>>(b, kp, st);
  return cudaGetLastError();
}

}  // namespace starkv
