// Calibration and selection of Sec. 3.4 - 3.7 (from s_bar to the index set I):
// one thread-block cluster of n = min(G, 8) CTAs per (sequence, layer).
//
// Phase 1, CTA r of the cluster works on groups g = r, r + n, ... (group r
// alone when G <= 8), one after the other:
//   (step path) AvgPool1D + group mean of the unpooled sums -> S[g, :] (Eqs. 3-4);
//   RankBin: the K - 1 equal-frequency boundaries of S[g, visual tokens] on
//     order-preserving keys, equal keys ordered by position: a 4096-bucket
//     histogram spread linearly over the row's key range locates each
//     boundary's bucket; tokens of a boundary-free bucket go straight to their
//     bin, and the few tokens of the boundary buckets are ranked pairwise by
//     (key, position).  Only when a boundary bucket holds more than 2048
//     tokens (many equal scores) does an exact radix select over four 8-bit
//     digits take over;
//   SpatialBin + joint histogram -> plug-in MI_g                        (Eq. 5);
//   phi_g = cos(current-frame row on the patch grid, m_g); m_g update    (Eq. 8).
// Phase 2, CTA r of the cluster works on tokens [r Lp / n, (r + 1) Lp / n):
//   MI EMA, min-max and softmax prior, lambda schedule                  (Eqs. 6-7);
//   s_bar, g*, Z = sum s_bar and the entropy H (Sec. 3.6), the per-CTA
//     partial sums exchanged through distributed shared memory;
//   s_t = max(s_bar beta D, 0)^(1/T)                     (Eq. final_score, Eq. 9);
//   global top-B with ties to the lower index (Sec. 3.7): a 4096-bucket
//     histogram over the cluster's key range, summed over the cluster, finds
//     the boundary bucket; its tokens (at most 2048) are gathered from every
//     CTA and ranked pairwise by (key, position); an ordered compaction with
//     offsets from the lower-ranked CTAs writes I.  A boundary bucket with
//     more tokens (many equal scores) falls back to an exact radix select
//     (12 + 10 + 10-bit digits) whose digit histograms are summed over the
//     cluster.
// Per-KV-head selection mode: in phase 2 CTA g works on its own row instead,
//   s_{g,t} = max(S[g,t] beta_g D_{g,t}, 0)^(1/T_g) with phi_g and the entropy of
//   S[g, .], and the same bucket / pairwise select over that row alone.
#include <algorithm>

#include "common.cuh"
#include "ptx.cuh"
#include "select.cuh"

namespace starkv {

namespace {

constexpr int kCalThreads = 1024;
constexpr int kMaxTargets = 15;      // K - 1 with K <= 16
constexpr int kBins0 = 4096;         // first radix digit: key bits 31..20
constexpr int kBins1 = 1024;         // second and third digits: bits 19..10 and 9..0
constexpr uint16_t kNoCell = 0xFFFF; // not a (valid) visual token
constexpr unsigned kFullMask = 0xffffffffu;
constexpr int kBruteMax = 2048;      // largest boundary bucket ranked pairwise
constexpr int kCandMax = 2048;       // largest top-B boundary bucket ranked pairwise
constexpr float kLn2 = 0.6931471805599453f;
constexpr size_t kSmemMax = 227 * 1024;

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

// Sum over the 1024 threads, in a fixed order; every thread gets the result.
template <typename T>
__device__ T block_sum(T v, T* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  return warp_sum(red[lane]);
}

// Exclusive scan of one int per thread over the block; `tmp` holds >= 33 ints.
__device__ int block_excl_scan(int v, int* tmp, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
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
    const int w = tmp[lane];
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += y;
    }
    tmp[lane] = wi - w;
    if (lane == 31) tmp[32] = wi;
  }
  __syncthreads();
  if (total) *total = tmp[32];
  return tmp[warp] + incl - v;
}

// One warp: the bin of a 256-bin histogram that holds rank `rank` (0-based)
// and the count of keys in lower bins; written by the lane that finds it.
__device__ void warp_find_256(const int* hist, int rank, int* digit, int* below) {
  const int lane = threadIdx.x & 31;
  const int4 q0 = reinterpret_cast<const int4*>(hist + lane * 8)[0];
  const int4 q1 = reinterpret_cast<const int4*>(hist + lane * 8)[1];
  const int v[8] = {q0.x, q0.y, q0.z, q0.w, q1.x, q1.y, q1.z, q1.w};
  const int sum = ((v[0] + v[1]) + (v[2] + v[3])) + ((v[4] + v[5]) + (v[6] + v[7]));
  int incl = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(kFullMask, incl, o);
    if (lane >= o) incl += y;
  }
  const int excl = incl - sum;
  if (rank >= excl && rank < incl) {
    int c = excl, d = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i)
      if (d == i && rank >= c + v[i]) {
        c += v[i];
        d = i + 1;
      }
    *digit = lane * 8 + d;
    *below = c;
  }
}

struct CalShared {
  uint32_t prefix[kMaxTargets];   // RankBin boundary keys, built digit by digit
  int rem[kMaxTargets];           // rank of the boundary among the keys sharing its prefix
  int reach[kMaxTargets];         // boundary rank < N
  int dig[kMaxTargets], below[kMaxTargets];
  int eqcnt[kMaxTargets];         // keys equal to the boundary key
  int slot_of[kMaxTargets];       // boundary -> its slot (boundary bucket), in bucket order
  int slot_off[kMaxTargets];      // slot -> first entry of its candidates in the pool
  int slot_n[kMaxTargets];        // slot -> tokens in its bucket
  int slot_j0[kMaxTargets];       // slot -> first boundary in it (= boundaries in lower buckets)
  int slot_cnt[kMaxTargets];      // slot -> candidates placed so far
  int nslot, ncand_all, brute;
  int ncand[32];                  // boundary-bucket tokens of each warp's segment
  int eqw[32][kMaxTargets];       // keys equal to each boundary before each warp's segment
  int nb[16];                     // rank-bin marginals
  int scan[33];
  float fred[32];
  double mib_old[kMaxGroups];     // MI EMA before this step, per group
  float w[kMaxGroups], ph[kMaxGroups];
  float lam;
  int n_old;
  int any_tie;
  float fredn[4][32];             // multi-value block reductions
  uint32_t uredn[3][32];
  float pz[kMaxCluster], pzl[kMaxCluster], pv[kMaxCluster];   // every CTA's phase-2 partials
  uint32_t pkmin[kMaxCluster], pkmax[kMaxCluster], psmax[kMaxCluster];
  int pncand[kMaxCluster], pbelow[kMaxCluster];
  // read by the other CTAs of the cluster
  float mi[kMaxGroups / kMaxCluster], phi[kMaxGroups / kMaxCluster];   // this CTA's groups (phase 1)
  float zpart, hpart, vpart;      // this CTA's token range (phase 2)
  uint32_t kminp, kmaxp, smaxp;
  int tcand, nbelow;              // top-B boundary-bucket candidates, tokens below it
  int lowcnt;                     // kept candidates of the lower-ranked CTAs
  int nlt, neq;
  // top-B select
  int tb, tcnt;                   // boundary bucket and its token count
  uint32_t tprefix, tkey;
  int trank, tpos;
};

// Sums of NF floats, the minimum of `mn` and the maximum of `mx` over the
// 1024 threads with one pair of barriers; every thread gets the results.
template <int NF>
__device__ void block_reduce(float (&v)[NF], uint32_t& mn, uint32_t& mx, CalShared& sh, uint32_t* mx2 = nullptr) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int k = 0; k < NF; ++k) v[k] = warp_sum(v[k]);
  mn = __reduce_min_sync(kFullMask, mn);
  mx = __reduce_max_sync(kFullMask, mx);
  if (mx2) *mx2 = __reduce_max_sync(kFullMask, *mx2);
  __syncthreads();
  if (lane == 0) {
#pragma unroll
    for (int k = 0; k < NF; ++k) sh.fredn[k][warp] = v[k];
    sh.uredn[0][warp] = mn;
    sh.uredn[1][warp] = mx;
    if (mx2) sh.uredn[2][warp] = *mx2;
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < NF; ++k) v[k] = warp_sum(sh.fredn[k][lane]);
  mn = __reduce_min_sync(kFullMask, sh.uredn[0][lane]);
  mx = __reduce_max_sync(kFullMask, sh.uredn[1][lane]);
  if (mx2) *mx2 = __reduce_max_sync(kFullMask, sh.uredn[2][lane]);
}

// Sum of the int4 at `p` over the CTAs [r_lo, r_hi) of the cluster: every
// remote load is issued before the first add.
__device__ __forceinline__ int4 sum_peers_v4(const int* p, int r_lo, int r_hi) {
  int4 q[kMaxCluster];
#pragma unroll
  for (int r = 0; r < kMaxCluster; ++r)
    if (r < r_hi - r_lo) q[r] = dsmem_ld_v4(dsmem_map(p, r_lo + r));
  int4 h = make_int4(0, 0, 0, 0);
#pragma unroll
  for (int r = 0; r < kMaxCluster; ++r)
    if (r < r_hi - r_lo) {
      h.x += q[r].x;
      h.y += q[r].y;
      h.z += q[r].z;
      h.w += q[r].w;
    }
  return h;
}

constexpr size_t align16(size_t x) { return (x + 15) & ~size_t(15); }
constexpr size_t kCalSharedBytes = align16(sizeof(CalShared));
constexpr int kBucketTable = kBins0;   // bytes: rank bin of each digit-1 bucket, or 0x80 | slot

// bucket histogram (4096) / top-B digits (4096 + 1024) / fallback digits (15 x 256)
__host__ __device__ __forceinline__ int hist_ints(int K) {
  (void)K;
  return kBins0 + kBins1;
}

size_t fixed_bytes(int K, int M, int R, int C) {
  return kCalSharedBytes + static_cast<size_t>(hist_ints(K)) * 4 + align16(static_cast<size_t>(K) * M * M * 4) +
         align16(static_cast<size_t>(R) * C * 4) + align16(R) + align16(C) + kBucketTable;
}

// Per token of a row kept on chip: key (4 B), candidate slot (4 B), cell (2 B).
constexpr size_t kBytesPerToken = 10;

}  // namespace

// Exact boundaries inside the boundary buckets by a radix select over their
// tokens (four 8-bit digits), equal keys ordered by position.  For rows whose
// boundary buckets hold too many tokens to rank pairwise (many equal scores).
// Adds the boundary-bucket tokens to the joint histogram.
template <typename BucketF>
__device__ void calibrate_refine_radix(CalShared& sh, int* hist, int* joint, const uint32_t* keys,
                                       const uint16_t* cells, uint32_t* cand, const uint8_t* btab, int MM, int nt,
                                       int s0, int s1, BucketF bucket_of) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const unsigned lanes_below = (1u << lane) - 1u;
  // each warp's segment keeps its candidates in position order
  int nc = 0;
  for (int base = s0; base < s1; base += 32) {
    const int t = base + lane;
    const bool c = t < s1 && cells[t] != kNoCell && (btab[bucket_of(keys[t])] & 0x80);
    const unsigned m = __ballot_sync(kFullMask, c);
    if (c) cand[s0 + nc + __popc(m & lanes_below)] = static_cast<uint32_t>(t);
    nc += __popc(m);
  }
  if (lane == 0) sh.ncand[warp] = nc;
  if (tid < nt) sh.prefix[tid] = 0;
  __syncthreads();
  const int ncw = sh.ncand[warp];
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    const uint32_t hmask = pass == 0 ? 0u : (0xFFFFFFFFu << (shift + 8));
    for (int i = tid; i < nt * 256; i += kCalThreads) hist[i] = 0;
    __syncthreads();
    for (int i = lane; i < ncw; i += 32) {
      const uint32_t u = keys[cand[s0 + i]];
      const int sl2 = btab[bucket_of(u)] & 0x7F;
      for (int j = sh.slot_j0[sl2]; j < nt && sh.reach[j] && sh.slot_of[j] == sl2; ++j)
        if (((u ^ sh.prefix[j]) & hmask) == 0) atomicAdd(&hist[j * 256 + ((u >> shift) & 255)], 1);
    }
    __syncthreads();
    if (warp < nt && sh.reach[warp]) warp_find_256(hist + warp * 256, sh.rem[warp], &sh.dig[warp], &sh.below[warp]);
    __syncthreads();
    if (tid < nt && sh.reach[tid]) {
      sh.prefix[tid] |= static_cast<uint32_t>(sh.dig[tid]) << shift;
      sh.rem[tid] -= sh.below[tid];
    }
    __syncthreads();
  }
  // equal keys before each warp's segment, per boundary
  for (int j = 0; j < nt; ++j) {
    int cnt = 0;
    for (int i = lane; i < ncw; i += 32) cnt += keys[cand[s0 + i]] == sh.prefix[j];
    cnt = warp_sum(cnt);
    if (lane == 0) sh.eqw[warp][j] = cnt;
  }
  __syncthreads();
  if (tid < nt) {
    int run = 0;
    for (int w = 0; w < 32; ++w) {
      const int c = sh.eqw[w][tid];
      sh.eqw[w][tid] = run;
      run += c;
    }
  }
  __syncthreads();
  int eqrun[kMaxTargets];
#pragma unroll
  for (int j = 0; j < kMaxTargets; ++j) eqrun[j] = j < nt ? sh.eqw[warp][j] : 0;
  for (int base = 0; base < ncw; base += 32) {
    const int i = base + lane;
    const bool ok = i < ncw;
    const int t = ok ? static_cast<int>(cand[s0 + i]) : 0;
    const uint32_t u = ok ? keys[t] : 0;
    int bin = 0;
#pragma unroll
    for (int j = 0; j < kMaxTargets; ++j) {
      if (j >= nt) break;
      const uint32_t P = sh.prefix[j];
      const unsigned m = __ballot_sync(kFullMask, ok && u == P);
      if (ok && sh.reach[j]) {
        if (u > P) ++bin;
        else if (u == P && eqrun[j] + __popc(m & lanes_below) >= sh.rem[j]) ++bin;
      }
      eqrun[j] += __popc(m);
    }
    if (ok) atomicAdd(&joint[bin * MM + cells[t]], 1);
  }
}

// MULTI: more groups than CTAs in the cluster (G > kMaxCluster, global mode);
// the GQA shapes (G <= kMaxCluster) compile without the group loop.
template <bool FROM_RAW, bool MULTI>
__global__ void __launch_bounds__(kCalThreads, 1) k_calibrate(const __grid_constant__ SeqBatch b,
                                                              const __grid_constant__ KParams kp, DevState st,
                                                              int capl) {
  extern __shared__ __align__(16) uint8_t smem_raw[];
  CalShared& sh = *reinterpret_cast<CalShared*>(smem_raw);
  const int G = kp.G, K = kp.K, M = kp.M, R = kp.R, C = kp.C, MM = M * M, RC = R * C, nt = K - 1;
  int* hist = reinterpret_cast<int*>(smem_raw + kCalSharedBytes);
  int* joint = hist + hist_ints(K);
  float* cur = reinterpret_cast<float*>(joint + ((K * MM + 3) & ~3));
  uint8_t* rowc = reinterpret_cast<uint8_t*>(cur + ((RC + 3) & ~3));
  uint8_t* colc = rowc + ((R + 15) & ~15);
  uint8_t* btab = colc + ((C + 15) & ~15);
  uint32_t* skeys = reinterpret_cast<uint32_t*>(btab + kBucketTable);
  uint32_t* scand = skeys + capl;
  uint16_t* scells = reinterpret_cast<uint16_t*>(scand + capl);

  const SeqView& sv = b.s[blockIdx.z];
  // the cluster spans grid x: one CTA per group, or kMaxCluster CTAs when G is
  // larger (global mode), CTA `rank` then taking groups rank, rank + ncta, ...
  const int rank = blockIdx.x, ncta = MULTI ? static_cast<int>(gridDim.x) : G;
  const int ll = blockIdx.y, layer = b.layer0 + ll;
  const int Lp = sv.Lp;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int sl = sv.slot * kp.n_layers + layer;
  const bool in_smem = Lp <= capl;
  // metadata row of group gi (the one shared row when meta_group_stride is 0)
  auto meta_of = [&](int gi) {
    return sv.meta + static_cast<int64_t>(layer) * sv.meta_layer_stride + gi * sv.meta_group_stride;
  };
  // the per-token arrays of row r: shared memory, or row r's workspace region
  auto keys_of = [&](int r) { return in_smem ? skeys : sv.vis + static_cast<int64_t>(ll * G + r) * Lp * 3; };
  // row `rank`'s arrays (the only ones without MULTI)
  const uint32_t* const meta0 = meta_of(rank);
  uint32_t* const keys0 = keys_of(rank);
  // phase 1 walks the row in one contiguous segment per warp, so that warp
  // order and lane order are position order
  const int seg = ceil_div(Lp, 32 * 32) * 32;
  const int s0 = min(Lp, warp * seg), s1 = min(Lp, s0 + seg);

  if (tid == 0) sh.any_tie = 0;
  for (int i = tid; i < kBins0; i += kCalThreads) hist[i] = 0;
  for (int i = tid; i < K * MM; i += kCalThreads) joint[i] = 0;
  for (int i = tid; i < RC; i += kCalThreads) cur[i] = 0.f;
  for (int r = tid; r < R; r += kCalThreads) rowc[r] = static_cast<uint8_t>(r * M / R);
  for (int c = tid; c < C; c += kCalThreads) colc[c] = static_cast<uint8_t>(c * M / C);
  // this CTA's groups' temporal EMA rows (state of the previous step, read
  // after phase 1) on their way into L2
  for (int gi = rank; gi < G; gi += ncta) {
    if (tid * 32 < RC) prefetch_l2(st.m + static_cast<int64_t>(sl * G + gi) * RC + tid * 32);
    if (!MULTI) break;
  }
  __syncthreads();
  // the set-up above overlaps the previous kernel's tail; its outputs are read below
  griddep_launch_dependents();
  griddep_wait();
  if (tid < G) sh.mib_old[tid] = st.mi_bar[sl * G + tid];
  if (tid == 0) sh.n_old = st.n[sl];

  // ================= phase 1: groups rank, rank + ncta, ... =================
  float* mrow_last = nullptr;   // the last group's m_g row and its update (0 none, 1 EMA, 2 first row),
  int mupd_last = 0;            // done while the phase-1 cluster barrier settles
  for (int g = rank, gl = 0; MULTI ? g < G : gl == 0; g += ncta, ++gl) {
  const uint32_t* meta = MULTI ? meta_of(g) : meta0;
  float* S = sv.S + (static_cast<int64_t>(layer) * G + g) * Lp;
  uint32_t* keys = MULTI ? keys_of(g) : keys0;
  uint32_t* cand = in_smem ? scand : keys + Lp;
  uint16_t* cells = in_smem ? scells : reinterpret_cast<uint16_t*>(keys + 2 * static_cast<int64_t>(Lp));
  // ---- the row, staged in shared memory by one pass of independent loads:
  // the unpooled sums (the four column-quarter copies added in order) or the
  // given S, into the candidate region; the metadata words into the key region
  const float pscale = static_cast<float>(G) / static_cast<float>(kp.H) / static_cast<float>(kp.pool);
  const int half = kp.pool >> 1;
  const int rs = raw_stride(Lp);
  const float* raw = FROM_RAW ? sv.s_raw + static_cast<int64_t>(ll * G + g) * kRawCopies * rs : nullptr;
  float* stage = reinterpret_cast<float*>(cand);
  // the step's rows held on chip: four consecutive tokens per thread and
  // 16-byte accesses (unpooled rows are 16-byte aligned; the metadata row is
  // read in 16 bytes when its address allows)
  const bool vec = FROM_RAW && in_smem;
  if (vec) {
    const bool meta16 = (reinterpret_cast<uintptr_t>(meta) & 15) == 0;
    for (int t00 = 4 * tid; t00 < Lp; t00 += 8 * kCalThreads) {
      float4 v[2];
      uint4 mw[2];
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const int t0 = t00 + 4 * k * kCalThreads;
        v[k] = make_float4(0.f, 0.f, 0.f, 0.f);
        mw[k] = make_uint4(0u, 0u, 0u, 0u);
        if (t0 < Lp) {
#pragma unroll
          for (int c = 0; c < kRawCopies; ++c) {   // copies added in order, as in the scalar path
            const float4 q = *reinterpret_cast<const float4*>(raw + c * rs + t0);
            v[k].x += q.x;
            v[k].y += q.y;
            v[k].z += q.z;
            v[k].w += q.w;
          }
          if (meta16 && t0 + 3 < Lp) {
            mw[k] = *reinterpret_cast<const uint4*>(meta + t0);
          } else {
            mw[k].x = meta[t0];
            if (t0 + 1 < Lp) mw[k].y = meta[t0 + 1];
            if (t0 + 2 < Lp) mw[k].z = meta[t0 + 2];
            if (t0 + 3 < Lp) mw[k].w = meta[t0 + 3];
          }
        }
      }
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const int t0 = t00 + 4 * k * kCalThreads;
        if (t0 < Lp) {   // the arrays hold capl >= Lp rounded up to 16 entries
          reinterpret_cast<float4*>(stage)[t0 >> 2] = v[k];
          reinterpret_cast<uint4*>(keys)[t0 >> 2] = mw[k];
        }
      }
    }
  } else {
    for (int t0 = 0; t0 < Lp; t0 += 4 * kCalThreads) {
      float v[4];
      uint32_t mw[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int t = t0 + k * kCalThreads + tid;
        v[k] = 0.f;
        mw[k] = 0u;
        if (t < Lp) {
          mw[k] = meta[t];
          if (FROM_RAW) {
            float r = 0.f;
#pragma unroll
            for (int c = 0; c < kRawCopies; ++c) r += raw[c * rs + t];
            v[k] = r;
          } else {
            v[k] = S[t];
          }
        }
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int t = t0 + k * kCalThreads + tid;
        if (t < Lp) {
          stage[t] = v[k];
          keys[t] = mw[k];
        }
      }
    }
  }
  __syncthreads();
  // ---- pooling (Eqs. 3-4), keys and cells of the visual tokens, their key
  // range, the current frame on the patch grid
  int nv = 0;
  uint32_t kmin = 0xFFFFFFFFu, kmax = 0u;
  auto pooled = [&](int t) {   // window sum in tap order, zero outside the row
    float acc = 0.f;
    if (half == 2 && t >= 2 && t + 2 < Lp) {   // the default window, away from the ends
      const float x0 = stage[t - 2], x1 = stage[t - 1], x2 = stage[t], x3 = stage[t + 1], x4 = stage[t + 2];
      acc = (((x0 + x1) + x2) + x3) + x4;
    } else {
      for (int j = -half; j <= half; ++j) {
        const int u = t + j;
        acc += (u >= 0 && u < Lp) ? stage[u] : 0.f;
      }
    }
    return acc * pscale;
  };
  // key and cell of one token; the current frame's tokens go onto the grid
  auto classify = [&](float s, uint32_t mt, uint32_t& key, uint16_t& cell) {
    cell = kNoCell;
    key = 0;
    if (meta_visual(mt)) {
      const int r = meta_row(mt), c = meta_col(mt);
      if (r < R && c < C) {
        const bool newest = meta_frame(mt) == sv.cur_frame;
        if (newest) atomicAdd(&cur[r * C + c], s);
        if (kp.mi_span == 0 || newest) {   // a token of the MI span (Sec. 3.4)
          key = order_key(s);
          cell = static_cast<uint16_t>(rowc[r] * M + colc[c]);
          ++nv;
          kmin = min(kmin, key);
          kmax = max(kmax, key);
        }
      } else {
        atomicOr(st.err, kErrMeta);
      }
    }
  };
  if (vec) {
    const float4* st4 = reinterpret_cast<const float4*>(stage);
    const bool s16 = (reinterpret_cast<uintptr_t>(S) & 15) == 0;   // S row on a 16-byte boundary
    // two vectors of four tokens per thread and pass: both vectors' loads are
    // issued before either's arithmetic and stores
    for (int t00 = 4 * tid; t00 < Lp; t00 += 8 * kCalThreads) {
      float4 a[2], b[2], c[2];
      uint4 m4[2];
      bool in[2], fast[2];
#pragma unroll
      for (int v = 0; v < 2; ++v) {
        const int t0 = t00 + 4 * v * kCalThreads;
        in[v] = t0 < Lp;
        fast[v] = in[v] && half == 2 && t0 >= 4 && t0 + 8 <= Lp;   // x[t0 - 4 .. t0 + 7] in three 16-byte loads
        a[v] = b[v] = c[v] = make_float4(0.f, 0.f, 0.f, 0.f);
        m4[v] = make_uint4(0u, 0u, 0u, 0u);
        if (fast[v]) {
          a[v] = st4[(t0 >> 2) - 1];
          b[v] = st4[t0 >> 2];
          c[v] = st4[(t0 >> 2) + 1];
        }
        if (in[v]) m4[v] = reinterpret_cast<const uint4*>(keys)[t0 >> 2];
      }
#pragma unroll
      for (int v = 0; v < 2; ++v) {
        const int t0 = t00 + 4 * v * kCalThreads;
        if (!in[v]) continue;
        float sv4[4];
        if (fast[v]) {
          const float x[12] = {a[v].x, a[v].y, a[v].z, a[v].w, b[v].x, b[v].y, b[v].z, b[v].w,
                               c[v].x, c[v].y, c[v].z, c[v].w};
#pragma unroll
          for (int k = 0; k < 4; ++k)
            sv4[k] = ((((x[k + 2] + x[k + 3]) + x[k + 4]) + x[k + 5]) + x[k + 6]) * pscale;
        } else {
#pragma unroll
          for (int k = 0; k < 4; ++k) sv4[k] = t0 + k < Lp ? pooled(t0 + k) : 0.f;
        }
        const uint32_t mts[4] = {m4[v].x, m4[v].y, m4[v].z, m4[v].w};
        uint32_t ks[4];
        uint16_t cs[4];
        if (s16 && t0 + 3 < Lp) *reinterpret_cast<float4*>(S + t0) = make_float4(sv4[0], sv4[1], sv4[2], sv4[3]);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          ks[k] = 0u;
          cs[k] = kNoCell;
          if (t0 + k < Lp) {
            if (!s16 || t0 + 3 >= Lp) S[t0 + k] = sv4[k];
            classify(sv4[k], mts[k], ks[k], cs[k]);
          }
        }
        reinterpret_cast<uint4*>(keys)[t0 >> 2] = make_uint4(ks[0], ks[1], ks[2], ks[3]);
        reinterpret_cast<uint2*>(cells)[t0 >> 2] =
            make_uint2(static_cast<uint32_t>(cs[0]) | (static_cast<uint32_t>(cs[1]) << 16),
                       static_cast<uint32_t>(cs[2]) | (static_cast<uint32_t>(cs[3]) << 16));
      }
    }
  } else {
    for (int t = tid; t < Lp; t += kCalThreads) {
      float s;
      if (FROM_RAW) {
        s = pooled(t);
        S[t] = s;
      } else {
        s = stage[t];
      }
      uint32_t key;
      uint16_t cell;
      classify(s, keys[t], key, cell);
      keys[t] = key;
      cells[t] = cell;
    }
  }
  int N;
  {
    float nvf[1] = {static_cast<float>(nv)};   // counts below 2^24: exact in fp32
    block_reduce<1>(nvf, kmin, kmax, sh);
    N = static_cast<int>(nvf[0]);
  }
  // Sec. 3.4 RankBin, first digit: 4096 buckets spread linearly over the
  // row's key range (monotone in the key, so bucket order is key order)
  const float binv = 4096.f / (static_cast<float>(kmax - kmin) + 1.f);
  auto bucket_of = [&](uint32_t u) {
    return min(kBins0 - 1, static_cast<int>(static_cast<float>(u - kmin) * binv));
  };
  if (tid < nt) {
    const int Rb = static_cast<int>((static_cast<int64_t>(tid + 1) * N + K - 1) / K);  // ceil(bN/K)
    sh.reach[tid] = Rb < N;
    sh.rem[tid] = Rb;
    sh.prefix[tid] = 0;
    sh.dig[tid] = 0;
    sh.below[tid] = 0;
    sh.eqcnt[tid] = 0;
  }
  if (tid < kMaxTargets) sh.slot_cnt[tid] = 0;
  __syncthreads();

  float mi = 0.f;
  if (N > 0) {
    // (token order does not matter here: four consecutive tokens per thread
    // when the row is on chip, else the warp segments)
    auto each_visual = [&](auto&& f) {
      if (in_smem) {
        for (int t0 = 4 * tid; t0 < Lp; t0 += 4 * kCalThreads) {
          const uint4 k4 = reinterpret_cast<const uint4*>(keys)[t0 >> 2];
          const uint2 c2 = reinterpret_cast<const uint2*>(cells)[t0 >> 2];
          const uint32_t ku[4] = {k4.x, k4.y, k4.z, k4.w};
          const uint32_t cu[4] = {c2.x & 0xFFFFu, c2.x >> 16, c2.y & 0xFFFFu, c2.y >> 16};
#pragma unroll
          for (int k = 0; k < 4; ++k)
            if (t0 + k < Lp && cu[k] != kNoCell) f(t0 + k, ku[k], static_cast<int>(cu[k]));
        }
      } else {
        for (int base = s0; base < s1; base += 32) {
          const int t = base + lane;
          const int cell = t < s1 ? cells[t] : kNoCell;
          if (cell != kNoCell) f(t, keys[t], cell);
        }
      }
    };
    each_visual([&](int, uint32_t u, int) { atomicAdd(&hist[bucket_of(u)], 1); });
    __syncthreads();
    {
      const int4 h = reinterpret_cast<const int4*>(hist)[tid];
      const int sum = (h.x + h.y) + (h.z + h.w);
      const int excl = block_excl_scan(sum, sh.scan, nullptr);
      for (int j = 0; j < nt; ++j) {
        const int r = sh.rem[j];
        if (sh.reach[j] && r >= excl && r < excl + sum) {
          int c = excl, d = 0;
          if (r >= c + h.x) { c += h.x; d = 1; }
          if (d == 1 && r >= c + h.y) { c += h.y; d = 2; }
          if (d == 2 && r >= c + h.z) { c += h.z; d = 3; }
          sh.dig[j] = tid * 4 + d;
          sh.below[j] = c;
        }
      }
      __syncthreads();
      if (warp == 0) {
        // boundaries are in rank order, so their buckets are non-decreasing;
        // a slot is one boundary bucket with its candidate tokens.  Lane j is
        // boundary j (nt <= 15; the reachable ones are a prefix).
        const bool rj = lane < nt && sh.reach[lane];
        const int dj = lane < nt ? sh.dig[lane] : -1;
        const int dprev = __shfl_up_sync(kFullMask, dj, 1);
        const bool isnew = rj && (lane == 0 || dj != dprev);
        const unsigned newmask = __ballot_sync(kFullMask, isnew);
        const int slot = __popc(newmask & ((2u << lane) - 1u)) - 1;   // slots opened at lanes <= this one
        const int n = isnew ? hist[dj] : 0;
        int incl = n;   // running candidate offset over the slots
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int y = __shfl_up_sync(kFullMask, incl, o);
          if (lane >= o) incl += y;
        }
        if (isnew) {
          sh.slot_off[slot] = incl - n;
          sh.slot_n[slot] = n;
          sh.slot_j0[slot] = lane;
        }
        if (rj) {
          sh.slot_of[lane] = slot;
          sh.rem[lane] -= sh.below[lane];   // rank inside the bucket
        }
        const int total = __shfl_sync(kFullMask, incl, 31);
        const int nmax = __reduce_max_sync(kFullMask, static_cast<unsigned>(n));
        if (lane == 0) {
          sh.nslot = __popc(newmask);
          sh.ncand_all = total;
          sh.brute = total <= Lp / 2 && nmax <= kBruteMax;
        }
      }
      __syncthreads();
    }
    // ---- bucket table: a bucket without a boundary puts all its tokens in
    // one rank bin (the boundaries below it); a boundary bucket is refined
    static_assert(kBins0 == 4 * kCalThreads, "four buckets per thread");
    {
      const int bk0 = 4 * tid;   // this thread's four consecutive buckets, each boundary read once
      int below[4] = {0, 0, 0, 0}, slot[4] = {-1, -1, -1, -1};
      for (int j = 0; j < nt; ++j) {
        if (!sh.reach[j]) break;
        const int d = sh.dig[j], so = sh.slot_of[j];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          below[k] += d < bk0 + k;
          if (d == bk0 + k) slot[k] = so;
        }
      }
      uint32_t packed = 0u;
#pragma unroll
      for (int k = 0; k < 4; ++k)
        packed |= static_cast<uint32_t>(static_cast<uint8_t>(slot[k] >= 0 ? (0x80 | slot[k]) : below[k])) << (8 * k);
      reinterpret_cast<uint32_t*>(btab)[tid] = packed;
    }
    __syncthreads();
    const bool brute = sh.brute;
    // ---- joint histogram of the settled tokens; boundary-bucket tokens go
    // to their slot's (key, position) pool
    uint32_t* pool = cand;   // [2 * candidates]
    each_visual([&](int t, uint32_t u, int cell) {
      const int v = btab[bucket_of(u)];
      if (!(v & 0x80)) {
        atomicAdd(&joint[v * MM + cell], 1);
      } else if (brute) {
        const int sl2 = v & 0x7F;
        const int i = sh.slot_off[sl2] + atomicAdd(&sh.slot_cnt[sl2], 1);
        pool[2 * i] = u;
        pool[2 * i + 1] = static_cast<uint32_t>(t);
      }
    });
    __syncthreads();
    if (brute) {
      // exact rank of each candidate inside its bucket by (key, position),
      // then the boundaries of its bucket at or below that rank
      const int nslot = sh.nslot;
      for (int i = tid; i < sh.ncand_all; i += kCalThreads) {
        int sl2 = 0;
        while (sl2 + 1 < nslot && sh.slot_off[sl2 + 1] <= i) ++sl2;
        const uint32_t ki = pool[2 * i], ti = pool[2 * i + 1];
        const int o = sh.slot_off[sl2], n = sh.slot_n[sl2];
        int rank = 0;
        for (int j = o; j < o + n; ++j) {
          const uint32_t kj = pool[2 * j], tj = pool[2 * j + 1];
          rank += (kj < ki) || (kj == ki && tj < ti);
        }
        int bin = sh.slot_j0[sl2];
        for (int j = sh.slot_j0[sl2]; j < nt && sh.reach[j] && sh.slot_of[j] == sl2; ++j) bin += sh.rem[j] <= rank;
        atomicAdd(&joint[bin * MM + cells[ti]], 1);
      }
    } else {
      calibrate_refine_radix(sh, hist, joint, keys, cells, cand, btab, MM, nt, s0, s1, bucket_of);
    }
    __syncthreads();
    // ---- Eq. (5): plug-in MI (nats) from the joint histogram
    int* ncell = hist;   // cell marginals
    for (int c = tid; c < MM; c += kCalThreads) {
      int s = 0;
      for (int bb = 0; bb < K; ++bb) s += joint[bb * MM + c];
      ncell[c] = s;
    }
    if (warp < K) {
      int s = 0;
      for (int i = lane; i < MM; i += 32) s += joint[warp * MM + i];
      s = warp_sum(s);
      if (lane == 0) sh.nb[warp] = s;
    }
    __syncthreads();
    const float fN = static_cast<float>(N);
    float acc = 0.f;
    for (int i = tid; i < K * MM; i += kCalThreads) {   // one (bin, cell) term per thread
      const int bb = i / MM, c = i - bb * MM;
      const int n = joint[i];
      if (n == 0) continue;
      const float fn = static_cast<float>(n);
      acc += fn * logf(fn * fN / (static_cast<float>(sh.nb[bb]) * static_cast<float>(ncell[c])));
    }
    mi = block_sum<float>(acc, sh.fred) / fN;
  }

  // ---- Sec. 3.5: phi_g = cos(current row, m_g); m_g EMA update (Eq. 8)
  float* mrow = st.m + static_cast<int64_t>(sl * G + g) * RC;
  float dot = 0.f, ncur = 0.f, nm = 0.f;
  for (int i = tid; i < RC; i += kCalThreads) {
    const float a = cur[i], bm = mrow[i];
    dot = fmaf(a, bm, dot);
    ncur = fmaf(a, a, ncur);
    nm = fmaf(bm, bm, nm);
  }
  {
    float r3[3] = {dot, ncur, nm};
    uint32_t u0 = 0u, u1 = 0u;
    block_reduce<3>(r3, u0, u1, sh);
    dot = r3[0];
    ncur = r3[1];
    nm = r3[2];
  }
  float phi = 0.f;
  int mupd = 0;
  if (ncur > 0.f) {
    mupd = nm > 0.f ? 1 : 2;
    if (nm > 0.f) phi = dot / (sqrtf(ncur) * sqrtf(nm));
  }
  if (MULTI && g + ncta < G) {   // an earlier group of this CTA: its current row is cleared next
    const float rt = kp.rho_t;
    if (mupd == 1)
      for (int i = tid; i < RC; i += kCalThreads) mrow[i] = rt * mrow[i] + (1.f - rt) * cur[i];
    else if (mupd == 2)
      for (int i = tid; i < RC; i += kCalThreads) mrow[i] = cur[i];
  } else {
    mrow_last = mrow;
    mupd_last = mupd;
  }
  if (tid == 0) {
    sh.mi[gl] = mi;
    sh.phi[gl] = phi;
    st.mi_cur[sl * G + g] = mi;
    st.phi_cur[sl * G + g] = phi;
  }
  if (MULTI && g + ncta < G) {   // the next group of this CTA starts from clean arrays
    __syncthreads();
    if (tid == 0) sh.any_tie = 0;
    for (int i = tid; i < kBins0; i += kCalThreads) hist[i] = 0;
    for (int i = tid; i < K * MM; i += kCalThreads) joint[i] = 0;
    for (int i = tid; i < RC; i += kCalThreads) cur[i] = 0.f;
    __syncthreads();
  }
  }   // phase-1 group loop
  // every group's S row, MI_g and phi_g are written: the peers may read them
  // once the barrier completes; the last group's m_g (read by no peer) and the
  // top-B histogram's zeroing go in between
  cluster_arrive();
  {
    const float rt = kp.rho_t;
    if (mupd_last == 1)
      for (int i = tid; i < RC; i += kCalThreads) mrow_last[i] = rt * mrow_last[i] + (1.f - rt) * cur[i];
    else if (mupd_last == 2)
      for (int i = tid; i < RC; i += kCalThreads) mrow_last[i] = cur[i];
  }
  for (int i = tid; i < kBins0; i += kCalThreads) hist[i] = 0;   // top-B digit 1 (below)
  cluster_wait();

  // ================= phase 2 =================
  // global mode: CTA r scores and selects tokens [r Lp / ncta, (r + 1) Lp / ncta)
  // of s_bar; per-KV-head mode (one CTA per group): CTA g its own row S[g, .]
  const bool per_head = kp.per_head != 0;
  const int g = rank;   // per-KV-head mode: this CTA's group
  const uint32_t* meta = MULTI ? meta_of(0) : meta0;   // global mode: the shared row
  uint32_t* keys = keys0;
  uint32_t* cand = in_smem ? scand : keys + Lp;
  float* stats = sv.stats ? sv.stats + static_cast<int64_t>(layer) * (8 + 6 * G) : nullptr;
  // ---- Eqs. (6)-(7): MI EMA (double state), min-max, softmax prior; lambda
  // schedule.  The same arithmetic in every CTA; CTA 0 stores the new state.
  // warp 0, lane gg < G: group gg's MI (from CTA gg % ncta), its EMA, then
  // the min-max and the softmax over the groups by warp reductions
  static_assert(kMaxGroups <= 32, "one lane per group");
  if (warp == 0) {
    const int n = sh.n_old;
    const bool on = lane < G;
    double mib = 0.0;
    float mic = 0.f, mf = 0.f;
    if (on) {
      const int owner = MULTI ? lane % ncta : lane, slot = MULTI ? lane / ncta : 0;
      mic = dsmem_ld_f32(dsmem_map(&sh.mi[slot], owner));
      sh.ph[lane] = dsmem_ld_f32(dsmem_map(&sh.phi[slot], owner));
      mib = n == 0 ? static_cast<double>(mic)
                   : kp.rho_mi * sh.mib_old[lane] + (1.0 - kp.rho_mi) * static_cast<double>(mic);
      mf = static_cast<float>(mib);
    }
    float lo = on ? mf : 3.4e38f, hi = on ? mf : -3.4e38f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      lo = fminf(lo, __shfl_xor_sync(kFullMask, lo, o));
      hi = fmaxf(hi, __shfl_xor_sync(kFullMask, hi, o));
    }
    const float inv = 1.f / (((hi - lo) + kp.eps) * kp.tau);
    const float e = on ? (mf - lo) * inv : -3.4e38f;
    float zmax = e;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) zmax = fmaxf(zmax, __shfl_xor_sync(kFullMask, zmax, o));
    const float ex = on ? expf(e - zmax) : 0.f;
    const float zs = warp_sum(ex);
    const float wg = ex / zs;
    if (on) sh.w[lane] = wg;
    float lam = 0.f;
    if (n >= kp.n_warmup)
      lam = kp.n_ramp <= 0 ? kp.lambda
                           : kp.lambda * fminf(1.f, static_cast<float>(n - kp.n_warmup) / kp.n_ramp);
    if (lane == 0) sh.lam = lam;
    if (rank == 0) {
      if (on) st.mi_bar[sl * G + lane] = mib;
      if (lane == 0) st.n[sl] = n + 1;
      if (stats) {
        if (lane == 0) {
          stats[2] = lam;
          stats[3] = static_cast<float>(n);
          stats[6] = static_cast<float>(sv.budget);
          stats[7] = 0.f;
        }
        if (on) {
          stats[8 + lane] = mic;
          stats[8 + G + lane] = mf;
          stats[8 + 2 * G + lane] = wg;
          stats[8 + 3 * G + lane] = sh.ph[lane];
        }
      }
    }
  }
  __syncthreads();   // w and lambda are read by every thread below
  // (range boundaries on multiples of 4 tokens, so that the ranges can be read in 16 bytes)
  auto split = [&](int r) {
    const int64_t t = (static_cast<int64_t>(r) * Lp / ncta + 3) & ~static_cast<int64_t>(3);
    return static_cast<int>(t < Lp ? t : Lp);
  };
  const int ta = per_head ? 0 : split(rank);
  const int tb = per_head ? Lp : split(rank + 1);
  const int nr = tb - ta;
  const float* S0 = sv.S + static_cast<int64_t>(layer) * G * Lp;
  const float invG = 1.f / static_cast<float>(G);
  const float lam = sh.lam;
  // ---- one pass over the range: s_bar and g* (Eq. 4; per-KV-head mode:
  // S[g, t] and g itself); Z = sum s and sum s log2 s (Sec. 3.6, one pass:
  // H = -sum p log p / log L_p with p = s / (Z + eps), where the eps inside
  // the log changes H by less than L_p eps); the untempered fused score
  // x_t = max(s beta D, 0) (Eq. final_score with Eq. 9).  s_t = x_t^(1/T) is
  // increasing in x_t, so the top-B select ranks the keys of x_t.
  float* xs = reinterpret_cast<float*>(cand);   // [nr]
  float z = 0.f, zl = 0.f, nvf = 0.f;
  uint32_t kmn = 0xFFFFFFFFu, kmx = 0u;
  uint32_t smx = 0u;   // the largest s (non-negative: its bits order like the values)
  auto fuse = [&](int i, float sb, int gs, uint32_t mt) {
    z += sb;
    smx = max(smx, __float_as_uint(fmaxf(sb, 0.f)));
    if (sb > 0.f) zl += sb * lg2_approx(sb);
    const float beta = (1.f - lam) + lam * static_cast<float>(G) * sh.w[gs];
    float d = 1.f;
    if (meta_visual(mt)) {
      nvf += 1.f;
      const float df = static_cast<float>(sv.cur_frame - meta_frame(mt));
      float shape;
      if (kp.decay_mode == 1) shape = fmaxf(0.f, 1.f - kp.delta * (df * sh.ph[gs]));
      else if (kp.decay_mode == 2) shape = powf(1.f + df * sh.ph[gs], -kp.delta);
      else shape = expf(-kp.delta * df * sh.ph[gs]);
      d = kp.d_min + (1.f - kp.d_min) * shape;
    }
    const float x = fmaxf(sb * beta * d, 0.f);
    const uint32_t key = ~order_key(x);   // descending score = ascending key
    xs[i] = x;
    keys[i] = key;
    kmn = min(kmn, key);
    kmx = max(kmx, key);
  };
  if (per_head) {
    const float* Sg = S0 + static_cast<int64_t>(g) * Lp;
    for (int i0 = 0; i0 < nr; i0 += 4 * kCalThreads) {
      float v[4];
      uint32_t mw[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int i = i0 + k * kCalThreads + tid;
        v[k] = 0.f;
        mw[k] = 0u;
        if (i < nr) {
          v[k] = Sg[i];
          mw[k] = meta[i];
        }
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int i = i0 + k * kCalThreads + tid;
        if (i < nr) fuse(i, v[k], g, mw[k]);
      }
    }
  } else if ((Lp & 3) == 0 && ((reinterpret_cast<uintptr_t>(S0) | reinterpret_cast<uintptr_t>(meta)) & 15) == 0) {
    // four consecutive tokens per thread, every group's row and the metadata
    // read in 16 bytes (ta and Lp are multiples of 4)
    for (int i0 = 4 * tid; i0 < nr; i0 += 4 * kCalThreads) {
      const int t = ta + i0;
      const uint4 m4 = *reinterpret_cast<const uint4*>(meta + t);
      float4 acc = *reinterpret_cast<const float4*>(S0 + t), best = acc;
      int gs[4] = {0, 0, 0, 0};
      auto take = [&](int gg) {
        const float4 q = *reinterpret_cast<const float4*>(S0 + static_cast<int64_t>(gg) * Lp + t);
        acc.x += q.x;
        acc.y += q.y;
        acc.z += q.z;
        acc.w += q.w;
        if (q.x > best.x) { best.x = q.x; gs[0] = gg; }
        if (q.y > best.y) { best.y = q.y; gs[1] = gg; }
        if (q.z > best.z) { best.z = q.z; gs[2] = gg; }
        if (q.w > best.w) { best.w = q.w; gs[3] = gg; }
      };
      if (!MULTI) {   // GQA: unrolled, every row's load issued up front
#pragma unroll
        for (int gg = 1; gg < kMaxCluster; ++gg) {
          if (gg >= G) break;
          take(gg);
        }
      } else {
        for (int gg = 1; gg < G; ++gg) take(gg);
      }
      fuse(i0, acc.x * invG, gs[0], m4.x);
      fuse(i0 + 1, acc.y * invG, gs[1], m4.y);
      fuse(i0 + 2, acc.z * invG, gs[2], m4.z);
      fuse(i0 + 3, acc.w * invG, gs[3], m4.w);
    }
  } else {
    for (int i = tid; i < nr; i += kCalThreads) {
      const int t = ta + i;
      // s_bar (Eq. 4) and its governing group g* (lowest on ties)
      float best = S0[t], acc = best;
      int gs = 0;
      for (int gg = 1; gg < G; ++gg) {
        const float v = S0[static_cast<int64_t>(gg) * Lp + t];
        acc += v;
        if (v > best) {
          best = v;
          gs = gg;
        }
      }
      fuse(i, acc * invG, gs, meta[t]);
    }
  }
  {
    float r3[3] = {z, zl, nvf};
    block_reduce<3>(r3, kmn, kmx, sh, &smx);
    z = r3[0];
    zl = r3[1];
    nvf = r3[2];
  }
  if (tid == 0) {
    sh.zpart = z;
    sh.hpart = zl;
    sh.vpart = nvf;
    sh.kminp = kmn;
    sh.kmaxp = kmx;
    sh.smaxp = smx;
  }
  cluster_sync();
  if (tid < ncta) {   // every CTA's partials, one peer per thread
    sh.pz[tid] = dsmem_ld_f32(dsmem_map(&sh.zpart, tid));
    sh.pzl[tid] = dsmem_ld_f32(dsmem_map(&sh.hpart, tid));
    sh.pv[tid] = dsmem_ld_f32(dsmem_map(&sh.vpart, tid));
    sh.pkmin[tid] = static_cast<uint32_t>(dsmem_ld_s32(dsmem_map(&sh.kminp, tid)));
    sh.pkmax[tid] = static_cast<uint32_t>(dsmem_ld_s32(dsmem_map(&sh.kmaxp, tid)));
    sh.psmax[tid] = static_cast<uint32_t>(dsmem_ld_s32(dsmem_map(&sh.smaxp, tid)));
  }
  __syncthreads();
  // the AEB signal of a row from its sums: the normalised entropy (Sec. 3.6)
  // or, with aeb_mode 1, the peak mass p_max = max s / (sum s + eps); T grows
  // with the entropy and falls with the peak mass
  auto entropy = [&](float Zr, float ZL2r, uint32_t smaxr) {   // ZL2r = sum s log2 s
    const float Ze = Zr + kp.eps_h;
    if (kp.aeb_mode == 1) return __uint_as_float(smaxr) / Ze;
    const float plogp = Zr > 0.f ? kLn2 * ZL2r / Ze - (Zr / Ze) * logf(Ze) : 0.f;
    return Lp > 1 ? -plogp / logf(static_cast<float>(Lp)) : 0.f;
  };
  auto temperature = [&](float sig) {
    return kp.t_min + (kp.t_max - kp.t_min) * (kp.aeb_mode == 1 ? 1.f - sig : sig);
  };
  float Hn, T;
  uint32_t kmin2 = kmn, kmax2 = kmx;   // key range of the selection
  if (per_head) {
    Hn = entropy(z, zl, smx);   // this CTA's own row
    T = temperature(Hn);
    if (tid == 0 && rank == 0 && stats) {
      float hs = 0.f, ts = 0.f, zs = 0.f;
      for (int r = 0; r < G; ++r) {
        const float Hr = entropy(sh.pz[r], sh.pzl[r], sh.psmax[r]);
        const float Tr = temperature(Hr);
        stats[8 + 4 * G + r] = Hr;
        stats[8 + 5 * G + r] = Tr;
        hs += Hr;
        ts += Tr;
        zs += sh.pz[r];
      }
      stats[0] = hs * invG;
      stats[1] = ts * invG;
      stats[4] = zs * invG;   // sum_t s_bar_t = mean over g of the row sums
      stats[5] = nvf;
    }
  } else {
    float Z = 0.f, ZL = 0.f, NV = 0.f;
    uint32_t SM = 0u;
    kmin2 = 0xFFFFFFFFu;
    kmax2 = 0u;
    for (int r = 0; r < ncta; ++r) {
      Z += sh.pz[r];
      ZL += sh.pzl[r];
      NV += sh.pv[r];
      SM = max(SM, sh.psmax[r]);
      kmin2 = min(kmin2, sh.pkmin[r]);
      kmax2 = max(kmax2, sh.pkmax[r]);
    }
    Hn = entropy(Z, ZL, SM);
    T = temperature(Hn);
    if (tid == 0 && rank == 0 && stats) {
      stats[0] = Hn;
      stats[1] = T;
      stats[4] = Z;
      stats[5] = NV;
      for (int r = 0; r < G; ++r) {
        stats[8 + 4 * G + r] = Hn;
        stats[8 + 5 * G + r] = T;
      }
    }
  }
  // ---- Sec. 3.6: s_t = x_t^(1/T) = 2^(log2(x_t) / T) (hardware exp2 / log2,
  // relative error a few 1e-7); first level of the top-B select: 4096
  // buckets spread linearly over the selection's key range (monotone in the key)
  const float invT = 1.f / T;
  float* score = per_head ? sv.score + (static_cast<int64_t>(layer) * G + g) * Lp
                          : sv.score + static_cast<int64_t>(layer) * Lp + ta;
  const float sbinv = kmax2 >= kmin2 ? 4096.f / (static_cast<float>(kmax2 - kmin2) + 1.f) : 0.f;
  auto sbucket = [&](uint32_t u) {
    return min(kBins0 - 1, static_cast<int>(static_cast<float>(u - kmin2) * sbinv));
  };
  const int B = sv.budget;   // the same in every CTA of the cluster
  for (int i = tid; i < nr; i += kCalThreads) atomicAdd(&hist[sbucket(keys[i])], 1);
  // global mode: the peers read this CTA's histogram next; the tempered
  // scores, which no peer reads, are written while the cluster barrier settles
  const bool early_arrive = B > 0 && !per_head;
  if (early_arrive) cluster_arrive();
  for (int i = tid; i < nr; i += kCalThreads) score[i] = ex2_approx(invT * lg2_approx(xs[i]));

  // ---- Sec. 3.7: top-B, ties to the lower index (global mode: over the
  // cluster; per-KV-head mode: over this CTA's row, block barriers only)
  bool done_remote = false;   // arrived at the final cluster barrier after the last remote read
  if (B > 0) {
    const int r_lo = per_head ? g : 0, r_hi = per_head ? g + 1 : ncta;
    auto sel_sync = [&]() {
      if (per_head) __syncthreads();
      else cluster_sync();
    };
    if (early_arrive) cluster_wait();   // every bucket histogram of the selection is complete
    else __syncthreads();
    {
      int4 h = sum_peers_v4(hist + 4 * tid, r_lo, r_hi);
      const int sum = (h.x + h.y) + (h.z + h.w);
      const int excl = block_excl_scan(sum, sh.scan, nullptr);
      const int rank = B - 1;
      if (rank >= excl && rank < excl + sum) {
        int c = excl, d = 0, n = h.x;
        if (rank >= c + h.x) { c += h.x; d = 1; n = h.y; }
        if (d == 1 && rank >= c + h.y) { c += h.y; d = 2; n = h.z; }
        if (d == 2 && rank >= c + h.z) { c += h.z; d = 3; n = h.w; }
        sh.tb = tid * 4 + d;
        sh.trank = rank - c;
        sh.tcnt = n;
      }
    }
    __syncthreads();
    const int bstar = sh.tb, rkb = sh.trank, ncb = sh.tcnt;
    int32_t* idx = sv.idx + (static_cast<int64_t>(layer) * (per_head ? G : 1) + (per_head ? g : 0)) * B;
    const int cs = ceil_div(nr, kCalThreads);
    const int i0 = min(nr, tid * cs), i1 = min(nr, i0 + cs);
    // the same decision in every CTA: it depends on the summed histogram only
    if (ncb <= kCandMax && ncb <= capl / 4) {
      // the boundary bucket's tokens as (key, position) pairs in shared memory
      // (the cell array is free in this phase), the tokens below it counted
      uint32_t* clist = reinterpret_cast<uint32_t*>(scells);
      if (tid == 0) sh.tcand = 0;
      __syncthreads();
      float below = 0.f;
      for (int i = tid; i < nr; i += kCalThreads) {
        const uint32_t u = keys[i];
        const int bk = sbucket(u);
        if (bk < bstar) {
          below += 1.f;
        } else if (bk == bstar) {
          const int j = atomicAdd(&sh.tcand, 1);
          clist[2 * j] = u;
          clist[2 * j + 1] = static_cast<uint32_t>(ta + i);
        }
      }
      {
        float b1[1] = {below};
        uint32_t u0 = 0u, u1 = 0u;
        block_reduce<1>(b1, u0, u1, sh);
        if (tid == 0) sh.nbelow = static_cast<int>(b1[0]);
      }
      sel_sync();   // every candidate list is complete
      if (tid >= r_lo && tid < r_hi) {
        sh.pncand[tid] = dsmem_ld_s32(dsmem_map(&sh.tcand, tid));
        sh.pbelow[tid] = dsmem_ld_s32(dsmem_map(&sh.nbelow, tid));
      }
      __syncthreads();
      // gather the candidates of the selection into the histogram area (no
      // peer reads it any more), then rank each by (key, position)
      uint32_t* all = reinterpret_cast<uint32_t*>(hist);
      int nall = 0, nlow = 0;
      if (tid == 0) sh.lowcnt = 0;
      for (int r = r_lo; r < r_hi; ++r) {
        const int n = sh.pncand[r];
        for (int j = tid; j < 2 * n; j += kCalThreads)
          all[2 * nall + j] = static_cast<uint32_t>(dsmem_ld_s32(dsmem_map(clist + j, r)));
        nall += n;
        if (r < rank) nlow += sh.pbelow[r];
      }
      __syncthreads();
      if (!per_head) {   // no peer's shared memory is read after this point
        cluster_arrive();
        done_remote = true;
      }
      for (int i = tid; i < nall; i += kCalThreads) {
        const uint32_t ki = all[2 * i], ti = all[2 * i + 1];
        int rank = 0;
        for (int j = 0; j < nall; ++j) {
          const uint32_t kj = all[2 * j], tj = all[2 * j + 1];
          rank += (kj < ki) || (kj == ki && tj < ti);
        }
        if (rank == rkb) {
          sh.tkey = ki;
          sh.tpos = static_cast<int>(ti);
        }
        // kept (rank <= the B-th's: the order is by key, then position) and
        // before this CTA's range: a kept candidate of a lower-ranked CTA
        if (rank <= rkb && static_cast<int>(ti) < ta) atomicAdd(&sh.lowcnt, 1);
      }
      __syncthreads();
      const uint32_t kT = sh.tkey;
      const uint32_t tT = static_cast<uint32_t>(sh.tpos);
      auto kept = [&](uint32_t u, uint32_t t) { return u < kT || (u == kT && t <= tT); };
      int nk = 0;
      for (int i = i0; i < i1; ++i) nk += kept(keys[i], static_cast<uint32_t>(ta + i));
      // kept tokens of the lower-ranked CTAs: all of their tokens below the
      // boundary bucket and their kept candidates
      int pos = nlow + sh.lowcnt + block_excl_scan(nk, sh.scan, nullptr);
      for (int i = i0; i < i1; ++i) {
        if (!kept(keys[i], static_cast<uint32_t>(ta + i))) continue;
        if (pos >= B) atomicOr(st.err, kErrIndex);   // cannot happen for a correct select
        else idx[pos] = ta + i;
        ++pos;
      }
    } else {
      // many equal keys around the boundary: an exact radix select over the
      // keys (12 + 10 + 10-bit digits), then ordered compaction
      sel_sync();   // the peers have read this CTA's bucket histogram
      for (int i = tid; i < kBins0; i += kCalThreads) hist[i] = 0;
      __syncthreads();
      for (int i = tid; i < nr; i += kCalThreads) atomicAdd(&hist[keys[i] >> 20], 1);
      sel_sync();
      {
        int4 h = sum_peers_v4(hist + 4 * tid, r_lo, r_hi);
        const int sum = (h.x + h.y) + (h.z + h.w);
        const int excl = block_excl_scan(sum, sh.scan, nullptr);
        const int rank = B - 1;
        if (rank >= excl && rank < excl + sum) {
          int c = excl, d = 0;
          if (rank >= c + h.x) { c += h.x; d = 1; }
          if (d == 1 && rank >= c + h.y) { c += h.y; d = 2; }
          if (d == 2 && rank >= c + h.z) { c += h.z; d = 3; }
          sh.tprefix = static_cast<uint32_t>(tid * 4 + d) << 20;
          sh.trank = rank - c;
        }
      }
      __syncthreads();
      // digits 2 and 3: histogram B (past the digit-1 bins), then histogram A
      // again (every CTA has read the peers' digit-1 bins before the barrier)
      for (int pass = 1; pass <= 2; ++pass) {
        const int shift = pass == 1 ? 10 : 0;
        int* hp = pass == 1 ? hist + kBins0 : hist;
        const uint32_t P = sh.tprefix;
        const int rk = sh.trank;
        hp[tid] = 0;
        __syncthreads();
        for (int i = tid; i < nr; i += kCalThreads) {
          const uint32_t u = keys[i];
          if (((u ^ P) >> (shift + 10)) == 0) atomicAdd(&hp[(u >> shift) & 1023], 1);
        }
        sel_sync();
        int v = 0;
        {
          int q[kMaxCluster];
#pragma unroll
          for (int r = 0; r < kMaxCluster; ++r)
            if (r < r_hi - r_lo) q[r] = dsmem_ld_s32(dsmem_map(hp + tid, r_lo + r));
#pragma unroll
          for (int r = 0; r < kMaxCluster; ++r)
            if (r < r_hi - r_lo) v += q[r];
        }
        const int excl = block_excl_scan(v, sh.scan, nullptr);
        if (rk >= excl && rk < excl + v) {
          sh.tprefix = P | (static_cast<uint32_t>(tid) << shift);
          sh.trank = rk - excl;
        }
        __syncthreads();
      }
      // kept: key < P, or key == P and among the first rk + 1 equal keys in
      // position order; contiguous spans per thread keep position order
      const uint32_t P = sh.tprefix;
      const int rk = sh.trank;
      int nlt = 0, neq = 0;
      for (int i = i0; i < i1; ++i) {
        const uint32_t u = keys[i];
        nlt += u < P;
        neq += u == P;
      }
      int tot_lt, tot_eq;
      int lt_b = block_excl_scan(nlt, sh.scan, &tot_lt);
      int eq_b = block_excl_scan(neq, sh.scan, &tot_eq);
      if (tid == 0) {
        sh.nlt = tot_lt;
        sh.neq = tot_eq;
      }
      sel_sync();
      for (int r = r_lo; r < rank; ++r) {
        lt_b += dsmem_ld_s32(dsmem_map(&sh.nlt, r));
        eq_b += dsmem_ld_s32(dsmem_map(&sh.neq, r));
      }
      for (int i = i0; i < i1; ++i) {
        const uint32_t u = keys[i];
        int pos = -1;
        if (u < P) {
          pos = lt_b + min(eq_b, rk + 1);
          ++lt_b;
        } else if (u == P) {
          if (eq_b <= rk) pos = lt_b + eq_b;
          ++eq_b;
        }
        if (pos >= B) atomicOr(st.err, kErrIndex);   // cannot happen for a correct select
        else if (pos >= 0) idx[pos] = ta + i;
      }
    }
  }
  // the peers' shared memory stays valid until every remote read is done
  if (done_remote) cluster_wait();
  else cluster_sync();
}

int calibrate_capacity(int K, int M, int R, int C) {
  const size_t fixed = fixed_bytes(K, M, R, C);
  if (fixed >= kSmemMax) return 0;
  return static_cast<int>(((kSmemMax - fixed) / kBytesPerToken) & ~size_t(15));
}

cudaError_t select_configure() {
  const int bytes = static_cast<int>(kSmemMax);
  cudaError_t e = cudaFuncSetAttribute(k_calibrate<true, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(k_calibrate<true, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(k_calibrate<false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_calibrate<false, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

cudaError_t calibrate_launch(const SeqBatch& b, const KParams& kp, const DevState& st, bool from_raw, int lp_max,
                             cudaStream_t stream) {
  const int cap = calibrate_capacity(kp.K, kp.M, kp.R, kp.C);
  const int capl = std::min(cap, (lp_max + 15) & ~15);
  const size_t smem = fixed_bytes(kp.K, kp.M, kp.R, kp.C) + static_cast<size_t>(capl) * kBytesPerToken;
  cudaLaunchConfig_t cfg = {};
  const int ncta = std::min(kp.G, kMaxCluster);   // the per-KV-head mode has G <= kMaxCluster
  cfg.gridDim = dim3(ncta, b.nlayers, b.nseq);
  cfg.blockDim = dim3(kCalThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = ncta;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // set-up under the previous kernel's tail
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  const bool multi = kp.G > kMaxCluster;
  if (from_raw) return multi ? cudaLaunchKernelEx(&cfg, k_calibrate<true, true>, b, kp, st, capl)
                             : cudaLaunchKernelEx(&cfg, k_calibrate<true, false>, b, kp, st, capl);
  return multi ? cudaLaunchKernelEx(&cfg, k_calibrate<false, true>, b, kp, st, capl)
               : cudaLaunchKernelEx(&cfg, k_calibrate<false, false>, b, kp, st, capl);
}

}  // namespace starkv
