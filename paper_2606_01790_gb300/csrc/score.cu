// Window-query x key scoring of Sec. 3.3 (Eqs. 2-4, Algorithm 1 first two
// steps) on tcgen05 tensor cores.
//
//   A_raw[h, t] = sum_{i<w} softmax_t(Q_{-i,h} . K_past[g(h), t] / sqrt(d))
//   S_raw[g, t] = sum_{h in g} A_raw[h, t]          (pooling + 1/(H/G) later)
//
// The softmax normaliser of a window row spans every past key, so the work is
// done in two passes over the same key tiles:
//   pass 1 (k_score_lse):   rows (query, head) on TMEM lanes, 128 keys per MMA
//                           column block; each thread keeps an online
//                           (max, sum-of-exp2) for its row over its key range
//                           and writes one partial per (row, piece).
//   pass 2 (k_score_accum): keys on TMEM lanes (M = 128), the group's window
//                           rows on columns (N <= 256); each thread sums
//                           exp2(z * log2e/sqrt(d) - lse2[col]) over its
//                           columns, so the per-key group sum needs no
//                           cross-thread reduction.  The score matrix never
//                           leaves the chip.
// Both passes split the flattened (seq, layer, group, key tile) space into one
// contiguous range per CTA (persistent grid <= #SMs), so a CTA reloads the
// group's queries only when its range crosses into a new (seq, layer, group)
// row.  Warp roles: warp 0 TMA producer, warp 1 MMA issuer (+ TMEM owner),
// warps 4..11 epilogue (two warpgroups).
#include "common.cuh"
#include "ptx.cuh"
#include "score.cuh"

namespace starkv {

namespace {

constexpr int kStages = 4;                    // K-tile pipeline depth
constexpr int kTileBytes = kTileKeys * 256;   // 128 keys x 128 bf16
constexpr int kHalfBytes = kTileKeys * 128;   // one 64-column swizzled half
constexpr int kTmemCols = 512;

struct TileCoord {
  int s, l, g, j;
};

__device__ __forceinline__ TileCoord decode(const ScoreParams& p, int64_t f) {
  int s = 0;
  while (s + 1 < p.nseq && p.seq[s + 1].tile_base <= f) ++s;
  const int nt = p.seq[s].nt;
  const int64_t u = f - p.seq[s].tile_base;
  const int per_layer = p.G * nt;
  TileCoord c;
  c.s = s;
  c.l = static_cast<int>(u / per_layer);
  const int rem = static_cast<int>(u - static_cast<int64_t>(c.l) * per_layer);
  c.g = rem / nt;
  c.j = rem - c.g * nt;
  return c;
}

// Flat index of the first tile of the (seq, layer, group) row holding `c`.
__device__ __forceinline__ int64_t row_first(const ScoreParams& p, const TileCoord& c) {
  return p.seq[c.s].tile_base + static_cast<int64_t>(c.l * p.G + c.g) * p.seq[c.s].nt;
}

__device__ __forceinline__ int64_t range_begin(int64_t T, int c, int P) { return T * c / P; }

struct SmemCtl {
  uint64_t k_full[kStages];
  uint64_t k_empty[kStages];
  uint64_t t_full[2];
  uint64_t t_empty[2];
  uint64_t q_full;
  uint64_t q_empty;
  uint64_t drain;
  uint32_t tmem_base;
  volatile int abort;
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

__device__ __forceinline__ void fail(SmemCtl* ctl, uint32_t* err) {
  ctl->abort = 1;
  atomicOr(err, kErrTimeout);
}

__device__ __forceinline__ void ctl_init(SmemCtl* ctl) {
  for (int i = 0; i < kStages; ++i) {
    mbar_init(&ctl->k_full[i], 1);
    mbar_init(&ctl->k_empty[i], 1);
  }
  for (int i = 0; i < 2; ++i) {
    mbar_init(&ctl->t_full[i], 1);
    mbar_init(&ctl->t_empty[i], 8);   // one arrival per epilogue warp
  }
  mbar_init(&ctl->q_full, 1);
  mbar_init(&ctl->q_empty, 1);
  mbar_init(&ctl->drain, 1);
  ctl->abort = 0;
  fence_mbar_init();
}

// TMA producer shared by both passes.  Q tile: `q_boxes` boxes of (64, q_box_rows)
// rows starting at row g*rows + b*q_box_rows, halves interleaved as the pass
// expects; K tile: 128 keys as two 64-column halves.
template <int PASS>
__device__ void producer_loop(const ScoreParams& p, SmemCtl* ctl, uint8_t* sQ, uint8_t* sK,
                              int64_t fb, int64_t fe) {
  const uint64_t pol_k = PASS == 1 ? policy_evict_last() : policy_evict_first();
  int it = 0, pc = 0;
  int64_t cur_row = -1;
  int last_q_pc = -1;
  int last_it[kStages];
  for (int i = 0; i < kStages; ++i) last_it[i] = -1;
  for (int64_t f = fb; f < fe; ++f) {
    if (ctl->abort) break;
    const TileCoord c = decode(p, f);
    const int64_t row = row_first(p, c);
    if (row != cur_row) {
      cur_row = row;
      if (!mbar_wait(&ctl->q_empty, (pc & 1) ^ 1, p.wait_ns)) { fail(ctl, p.err); break; }
      const int zq = p.layer0 + c.l;
      if (PASS == 1) {
        mbar_arrive_expect_tx(&ctl->q_full, p.n_mtiles * kTileBytes);
        for (int mt = 0; mt < p.n_mtiles; ++mt)
          for (int h = 0; h < 2; ++h)
            tma_load_3d(sQ + mt * kTileBytes + h * kHalfBytes, &p.tmq1[c.s], &ctl->q_full, h * 64,
                        c.g * p.rows + mt * kTileKeys, zq);
      } else {
        mbar_arrive_expect_tx(&ctl->q_full, p.n2 * 256);
        for (int h = 0; h < 2; ++h)
          tma_load_3d(sQ + h * p.n2 * 128, &p.tmq2[c.s], &ctl->q_full, h * 64, c.g * p.rows, zq);
      }
      last_q_pc = pc;
      ++pc;
    }
    const int stage = it % kStages;
    const uint32_t ph = (it / kStages) & 1;
    if (!mbar_wait(&ctl->k_empty[stage], ph ^ 1, p.wait_ns)) { fail(ctl, p.err); break; }
    mbar_arrive_expect_tx(&ctl->k_full[stage], kTileBytes);
    const int zk = (p.layer0 + c.l) * p.G + c.g;
    for (int h = 0; h < 2; ++h)
      tma_load_3d_hint(sK + stage * kTileBytes + h * kHalfBytes, &p.tmk[c.s], &ctl->k_full[stage],
                       h * 64, c.j * kTileKeys, zk, pol_k);
    last_it[stage] = it;
    ++it;
  }
  if (ctl->abort) {
    // bring every issued copy to completion before the CTA can exit
    for (int i = 0; i < kStages; ++i)
      if (last_it[i] >= 0) mbar_wait(&ctl->k_full[i], (last_it[i] / kStages) & 1, p.wait_ns);
    if (last_q_pc >= 0) mbar_wait(&ctl->q_full, last_q_pc & 1, p.wait_ns);
  }
}

// MMA issuer shared by both passes.
template <int PASS>
__device__ void mma_loop(const ScoreParams& p, SmemCtl* ctl, const uint8_t* sQ, const uint8_t* sK,
                         uint32_t tmem, int64_t fb, int64_t fe) {
  const uint32_t idesc = PASS == 1 ? idesc_bf16(128, kTileKeys) : idesc_bf16(128, p.n2);
  const uint32_t q_addr = smem_u32(sQ), k_addr = smem_u32(sK);
  int it = 0, jt = 0, pc = 0;
  int64_t cur_row = -1;
  for (int64_t f = fb; f < fe; ++f) {
    if (ctl->abort) break;
    const TileCoord c = decode(p, f);
    const int64_t row = row_first(p, c);
    const bool last = (f + 1 == fe) || row_first(p, decode(p, f + 1)) != row;
    if (row != cur_row) {
      cur_row = row;
      if (!mbar_wait(&ctl->q_full, pc & 1, p.wait_ns)) { fail(ctl, p.err); break; }
      ++pc;
    }
    const int stage = it % kStages;
    const uint32_t ph = (it / kStages) & 1;
    const int ts = jt & 1;
    const uint32_t tph = (jt >> 1) & 1;
    if (!mbar_wait(&ctl->k_full[stage], ph, p.wait_ns)) { fail(ctl, p.err); break; }
    if (!mbar_wait(&ctl->t_empty[ts], tph ^ 1, p.wait_ns)) { fail(ctl, p.err); break; }
    tc_fence_after();
    const uint32_t kbase = k_addr + stage * kTileBytes;
    if (PASS == 1) {
      for (int mt = 0; mt < p.n_mtiles; ++mt) {
        const uint32_t d = tmem + ts * 256 + mt * kTileKeys;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t koff = (kk >> 2) * kHalfBytes + (kk & 3) * 32;
          mma_bf16(d, sdesc_k_sw128(q_addr + mt * kTileBytes + koff), sdesc_k_sw128(kbase + koff),
                   idesc, kk > 0);
        }
      }
    } else {
      const uint32_t d = tmem + ts * 256;
      const uint32_t qhalf = p.n2 * 128;
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint32_t koff = (kk >> 2) * kHalfBytes + (kk & 3) * 32;
        const uint32_t qoff = (kk >> 2) * qhalf + (kk & 3) * 32;
        mma_bf16(d, sdesc_k_sw128(kbase + koff), sdesc_k_sw128(q_addr + qoff), idesc, kk > 0);
      }
    }
    mma_commit(&ctl->k_empty[stage]);
    mma_commit(&ctl->t_full[ts]);
    if (last) mma_commit(&ctl->q_empty);
    ++it;
    ++jt;
  }
  // every MMA issued above must be complete before TMEM is released
  mma_commit(&ctl->drain);
  mbar_wait(&ctl->drain, 0, p.wait_ns);
}

// log2-domain log-sum-exp of window row `col` of the (seq, layer, group) row
// whose first flat tile is `r0`, from the pass-1 partials of every CTA piece
// that covered the row.
__device__ float combine_lse2(const ScoreParams& p, int64_t r0, int nt, int col) {
  const int64_t T = p.total_tiles;
  const int P = p.grid1;
  const int64_t r1 = r0 + nt - 1;
  const int c0 = static_cast<int>(((r0 + 1) * P - 1) / T);
  const int c1 = static_cast<int>(((r1 + 1) * P - 1) / T);
  float mx = -INFINITY;
  for (int c = c0; c <= c1; ++c) {
    const int64_t ps = max(range_begin(T, c, P), r0);
    mx = fmaxf(mx, p.partials[ps * kMaxRows + col].x);
  }
  float sum = 0.f;
  for (int c = c0; c <= c1; ++c) {
    const int64_t ps = max(range_begin(T, c, P), r0);
    const float2 v = p.partials[ps * kMaxRows + col];
    sum += v.y * exp2f(v.x - mx);
  }
  return mx + log2f(sum);
}

}  // namespace

__global__ void __launch_bounds__(kScoreThreads, 1) k_score_lse(const __grid_constant__ ScoreParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sQ = smem;                          // [2 M-tiles][2 halves][128][128 B]
  uint8_t* sK = smem + 2 * kTileBytes;         // [kStages][2 halves][128][128 B]
  SmemCtl* ctl = reinterpret_cast<SmemCtl*>(sK + kStages * kTileBytes);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) ctl_init(ctl);
  if (warp == 1) {
    tmem_alloc(&ctl->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctl->tmem_base;
  const int64_t T = p.total_tiles;
  const int64_t fb = range_begin(T, blockIdx.x, gridDim.x);
  const int64_t fe = range_begin(T, blockIdx.x + 1, gridDim.x);

  if (warp == 0) {
    if (lane == 0) producer_loop<1>(p, ctl, sQ, sK, fb, fe);
  } else if (warp == 1) {
    if (lane == 0) mma_loop<1>(p, ctl, sQ, sK, tmem, fb, fe);
  } else if (warp >= 4) {
    const int ew = warp - 4;
    const int mt = ew >> 2;                 // M-tile of this epilogue warpgroup
    const int quad = warp & 3;              // TMEM lane quadrant
    const int r = mt * kTileKeys + quad * 32 + lane;  // window row within the group
    const bool active = mt < p.n_mtiles;
    const float sc = p.scale2;
    float m = -INFINITY, s = 0.f;
    int jt = 0;
    int64_t cur_row = -1, piece_start = 0;
    for (int64_t f = fb; f < fe; ++f) {
      // every decision below is warp-uniform: tcgen05.ld is a .sync.aligned op
      if (__any_sync(0xffffffffu, ctl->abort != 0)) break;
      const TileCoord c = decode(p, f);
      const int64_t row = row_first(p, c);
      const bool last = (f + 1 == fe) || row_first(p, decode(p, f + 1)) != row;
      if (row != cur_row) {
        cur_row = row;
        piece_start = f;
        m = -INFINITY;
        s = 0.f;
      }
      const int ts = jt & 1;
      const uint32_t tph = (jt >> 1) & 1;
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&ctl->t_full[ts], tph, p.wait_ns));
      if (!ok) { fail(ctl, p.err); break; }
      tc_fence_after();
      if (active) {
        const int Lp = p.seq[c.s].Lp;
        const int key0 = c.j * kTileKeys;
        const uint32_t base = tmem + (static_cast<uint32_t>(quad * 32) << 16) + ts * 256 + mt * kTileKeys;
#pragma unroll 1
        for (int ch = 0; ch < 4; ++ch) {
          float v[32];
          tmem_ld32(base + ch * 32, v);
          const int kc = key0 + ch * 32;
          if (kc + 32 > Lp) {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (kc + i >= Lp) v[i] = -INFINITY;
          }
          float cm = v[0];
#pragma unroll
          for (int i = 1; i < 32; ++i) cm = fmaxf(cm, v[i]);
          const float mn = fmaxf(m, cm * sc);
          if (mn != -INFINITY) {
            s *= ex2_approx(m - mn);
            float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
            for (int i = 0; i < 32; i += 4) {
              a0 += ex2_approx(fmaf(v[i + 0], sc, -mn));
              a1 += ex2_approx(fmaf(v[i + 1], sc, -mn));
              a2 += ex2_approx(fmaf(v[i + 2], sc, -mn));
              a3 += ex2_approx(fmaf(v[i + 3], sc, -mn));
            }
            s += (a0 + a1) + (a2 + a3);
            m = mn;
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ctl->t_empty[ts]);
      if (last && active && r < p.rows)
        p.partials[piece_start * kMaxRows + r] = make_float2(m, s);
      ++jt;
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

__global__ void __launch_bounds__(kScoreThreads, 1) k_score_accum(const __grid_constant__ ScoreParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sQ = smem;                          // [2 halves][n2][128 B]  (<= 64 KB)
  uint8_t* sK = smem + 2 * kTileBytes;         // [kStages][2 halves][128][128 B]
  SmemCtl* ctl = reinterpret_cast<SmemCtl*>(sK + kStages * kTileBytes);
  float* lse2 = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(ctl) + 256);  // [256]
  float* red = lse2 + kMaxRows;                                                   // [2][128]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) ctl_init(ctl);
  if (warp == 1) {
    tmem_alloc(&ctl->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = ctl->tmem_base;
  const int64_t T = p.total_tiles;
  const int64_t fb = range_begin(T, blockIdx.x, gridDim.x);
  const int64_t fe = range_begin(T, blockIdx.x + 1, gridDim.x);

  if (warp == 0) {
    if (lane == 0) producer_loop<2>(p, ctl, sQ, sK, fb, fe);
  } else if (warp == 1) {
    if (lane == 0) mma_loop<2>(p, ctl, sQ, sK, tmem, fb, fe);
  } else if (warp >= 4) {
    const int et = threadIdx.x - 128;       // 0..255
    const int wg = (warp - 4) >> 2;         // column half
    const int quad = warp & 3;
    const int nch = p.n2 >> 4;              // 16-column chunks
    const int nch0 = (nch + 1) >> 1;
    const int ch_lo = wg == 0 ? 0 : nch0, ch_hi = wg == 0 ? nch0 : nch;
    const float sc = p.scale2;
    int jt = 0;
    int64_t cur_row = -1;
    // Decisions to stop are taken together by all 256 epilogue threads at the
    // per-tile named barrier, so no thread is left waiting at a barrier.
    for (int64_t f = fb; f < fe; ++f) {
      const TileCoord c = decode(p, f);
      const int64_t row = row_first(p, c);
      if (row != cur_row) {
        cur_row = row;
        named_bar_sync(1, 256);
        lse2[et] = et < p.rows ? combine_lse2(p, row, p.seq[c.s].nt, et) : INFINITY;
        named_bar_sync(1, 256);
      }
      const int ts = jt & 1;
      const uint32_t tph = (jt >> 1) & 1;
      const bool ok = __all_sync(0xffffffffu, mbar_wait(&ctl->t_full[ts], tph, p.wait_ns));
      tc_fence_after();
      const uint32_t base = tmem + (static_cast<uint32_t>(quad * 32) << 16) + ts * 256;
      float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll 1
      for (int ch = ok ? ch_lo : ch_hi; ch < ch_hi; ++ch) {
        float v[16];
        tmem_ld16(base + ch * 16, v);
        const float4* l4 = reinterpret_cast<const float4*>(lse2 + ch * 16);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float4 l = l4[i];
          a0 += ex2_approx(fmaf(v[4 * i + 0], sc, -l.x));
          a1 += ex2_approx(fmaf(v[4 * i + 1], sc, -l.y));
          a2 += ex2_approx(fmaf(v[4 * i + 2], sc, -l.z));
          a3 += ex2_approx(fmaf(v[4 * i + 3], sc, -l.w));
        }
      }
      tc_fence_before();
      __syncwarp();
      if (ok && lane == 0) mbar_arrive(&ctl->t_empty[ts]);
      const float acc = (a0 + a1) + (a2 + a3);
      const int kl = quad * 32 + lane;
      if (wg == 1) red[ts * 128 + kl] = acc;
      if (named_bar_any(2, 256, !ok || ctl->abort != 0)) {
        fail(ctl, p.err);
        break;
      }
      if (wg == 0) {
        const int key = c.j * kTileKeys + kl;
        const ScoreSeq& sq = p.seq[c.s];
        if (key < sq.Lp)
          sq.s_raw[static_cast<int64_t>(c.l * p.G + c.g) * sq.Lp + key] = acc + red[ts * 128 + kl];
      }
      ++jt;
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// S[g, t] = (G/H)(1/k) sum_{|j| <= k/2} S_raw[g, t + j]  (Eqs. 3-4; zero padding,
// divisor k).  grid: (ceil(Lp_max / 256), nlayers * G, nseq)
__global__ void k_pool(const __grid_constant__ SeqBatch b, int G, int H, int pool) {
  const SeqView& s = b.s[blockIdx.z];
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= s.Lp) return;
  const int lg = blockIdx.y;                  // launch-local layer * G + g
  const int layer = b.layer0 + lg / G, g = lg % G;
  const float* src = s.s_raw + static_cast<int64_t>(lg) * s.Lp;
  const int half = pool >> 1;
  float acc = 0.f;
  for (int j = -half; j <= half; ++j) {
    const int u = t + j;
    if (u >= 0 && u < s.Lp) acc += src[u];
  }
  const float scale = static_cast<float>(G) / static_cast<float>(H) / static_cast<float>(pool);
  s.S[(static_cast<int64_t>(layer) * G + g) * s.Lp + t] = acc * scale;
}

size_t score_smem_bytes() {
  return 1024 + 2 * kTileBytes + kStages * kTileBytes + 256 + (kMaxRows + 256) * sizeof(float);
}

cudaError_t score_configure() {
  const int bytes = static_cast<int>(score_smem_bytes());
  cudaError_t e = cudaFuncSetAttribute(k_score_lse, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_score_accum, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

cudaError_t score_lse_launch(const ScoreParams& p, int grid, cudaStream_t stream) {
  k_score_lse<<<grid, kScoreThreads, score_smem_bytes(), stream>>>(p);
  return cudaGetLastError();
}

cudaError_t score_accum_launch(const ScoreParams& p, int grid, cudaStream_t stream) {
  k_score_accum<<<grid, kScoreThreads, score_smem_bytes(), stream>>>(p);
  return cudaGetLastError();
}

cudaError_t pool_launch(const SeqBatch& b, int G, int H, int pool, int lp_max, cudaStream_t stream) {
  if (lp_max <= 0) return cudaSuccess;
  dim3 grid(ceil_div(lp_max, 256), b.nlayers * G, b.nseq);
  k_pool<<<grid, 256, 0, stream>>>(b, G, H, pool);
  return cudaGetLastError();
}

}  // namespace starkv
