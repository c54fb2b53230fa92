// Window-query x key scoring of Sec. 3.3 (Eqs. 2-4) on tcgen05 tensor cores.
//
//   A_raw[h, t] = sum_{i<w} softmax_t(Q_{-i,h} . K_past[g(h), t] / sqrt(d))
//   S_raw[g, t] = sum_{h in g} A_raw[h, t]          (pooling + 1/(H/G) later)
//
// The softmax normaliser of a window row spans every past key, so the work is
// done in two passes over the same key tiles:
//   pass 1 (k_score_lse):   rows (query, head) on TMEM lanes, 128 keys per MMA
//                           column block; each thread keeps a (reference,
//                           sum of exp2) pair for its row over its keys and
//                           one partial per (row, piece) is written.
//   pass 2 (k_score_accum): keys on TMEM lanes (M = 128), the group's window
//                           rows on columns (N <= 256); one extra K step adds
//                           -lse2[col] sqrt(d)/log2e to every logit (a ones
//                           operand against the rows' -lse as three bf16
//                           parts), and each thread sums exp2(acc log2e/sqrt(d))
//                           over its columns, so the per-key group sum needs
//                           no cross-lane reduction and no per-column operand.
//                           The score matrix never leaves the chip.
// Both passes split the flattened (seq, layer, group, key tile) space into one
// contiguous range per CTA (persistent grid <= #SMs), so a CTA reloads the
// group's queries only when its range crosses into a new (seq, layer, group)
// row ("piece").  Warp roles: warp 0 TMA producer, warps 1 and 2 MMA issuers
// (even / odd tiles; warp 1 also owns the TMEM allocation), warps 4..19
// epilogue: four warpgroups that all work on every tile, so the per-element
// exp2 and sums are spread over 16 warps.  Two 256-column TMEM accumulator
// stages let the MMA of tile i+1 run under the epilogue of tile i; TMEM is
// read in 16-column loads with the next load in flight under the arithmetic,
// which runs on packed fp32 pairs.  Each pass is bounded below by its K
// stream and, at nearly the same level, by the epilogue's per-tile cost.
#include <algorithm>
#include <utility>

#include "common.cuh"
#include "ptx.cuh"
#include "score.cuh"

namespace starkv {

namespace {

constexpr int kMaxStages = 4;                 // K-tile pipeline depth (at most; even, see score_kstages)
constexpr size_t kSmemLimit = 227 * 1024;
constexpr int kTileBytes = kTileKeys * 256;   // 128 keys x 128 bf16
constexpr int kHalfBytes = kTileKeys * 128;   // one 64-column swizzled half
constexpr int kTmemCols = 512;
constexpr int kMmaThreads = 2;                // MMA issuers (warps 1 and 2): even / odd tiles
constexpr int kEpiWarp0 = 4;                  // first epilogue warp (warpgroup aligned)
constexpr int kEpiWarps = 16;
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr uint32_t kFull = 0xffffffffu;
constexpr int kXOnesBytes = 256;              // pass 2: the ones operand (two 8 x 16 B core matrices)
constexpr int kXRowBytes = 32;                // pass 2: one window row of the -lse operand (16 bf16)
// Limit of the waits for copies and MMAs this CTA has already issued, before
// it exits or releases TMEM: those complete in microseconds, so the limit only
// guards against a broken memory system, whatever the configured wait limit.
constexpr uint64_t kDrainWaitNs = 2000000000ull;

__device__ __forceinline__ uint64_t drain_limit(uint64_t wait_ns) {
  return wait_ns > kDrainWaitNs ? wait_ns : kDrainWaitNs;
}

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


__device__ __forceinline__ int64_t range_begin(int64_t T, int c, int P) { return T * c / P; }

// Coordinates of consecutive flat tiles [f0, f1), advanced without divisions
// (one decode at the start).  A piece is a run of tiles of one (seq, layer,
// group) row inside the range.
struct TileIter {
  int s, l, g, j, nt;
  int64_t f, fe;
  __device__ void init(const ScoreParams& p, int64_t f0, int64_t f1) {
    f = f0;
    fe = f1;
    s = l = g = j = nt = 0;
    if (f >= fe) return;
    const TileCoord c = decode(p, f0);
    s = c.s;
    l = c.l;
    g = c.g;
    j = c.j;
    nt = p.seq[s].nt;
  }
  __device__ bool valid() const { return f < fe; }
  __device__ bool first(int64_t fb) const { return f == fb || j == 0; }
  __device__ bool last() const { return f + 1 == fe || j + 1 == nt; }
  __device__ void next(const ScoreParams& p) {
    ++f;
    if (f >= fe) return;
    if (++j < nt) return;
    j = 0;
    if (++g < p.G) return;
    g = 0;
    if (++l < p.nlayers) return;
    l = 0;
    do {
      ++s;
    } while (s + 1 < p.nseq && p.seq[s].nt == 0);
    nt = p.seq[s].nt;
  }
};

struct SmemCtl {
  uint64_t k_full[kMaxStages];
  uint64_t k_empty[kMaxStages];
  uint64_t t_full[2][2];   // [accumulator stage][M tile]: that M tile's tile product is done
  uint64_t t_empty[2];
  uint64_t q_full;
  uint64_t q_empty;
  uint64_t x_full[2];   // pass 2: a piece's -lse operand is in its buffer
  uint64_t drain;
  uint32_t tmem_base;
  volatile int abort;
};

static_assert(sizeof(SmemCtl) <= 256, "the control block has 256 bytes");

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

__device__ __forceinline__ void fail(SmemCtl* ctl, uint32_t* err) {
  ctl->abort = 1;
  atomicOr(err, kErrTimeout);
}

__device__ __forceinline__ void ctl_init(SmemCtl* ctl, int kstages) {
  for (int i = 0; i < kstages; ++i) {
    mbar_init(&ctl->k_full[i], 1);
    mbar_init(&ctl->k_empty[i], 1);
  }
  for (int i = 0; i < 2; ++i) {
    for (int m = 0; m < 2; ++m) mbar_init(&ctl->t_full[i][m], 1);
    mbar_init(&ctl->t_empty[i], kEpiWarps);   // one arrival per epilogue warp
  }
  mbar_init(&ctl->q_full, 1);
  mbar_init(&ctl->q_empty, kMmaThreads);   // each MMA thread commits once per piece
  for (int i = 0; i < 2; ++i) mbar_init(&ctl->x_full[i], 1);
  mbar_init(&ctl->drain, kMmaThreads);
  ctl->abort = 0;
  fence_mbar_init();
}

// TMA producer shared by both passes.  Q: [2 halves][q_rows][128 B]; pass 1
// loads the group's rows as a 128-row box and a (rows - 128)-row box per half,
// pass 2 one n2-row box per half.  K tile: 128 keys as two 64-column halves.
template <int PASS>
__device__ void producer_loop(const ScoreParams& p, SmemCtl* ctl, uint8_t* sQ, uint8_t* sK,
                              int64_t fb, int64_t fe) {
  const uint64_t pol_k = policy_evict_first();   // K streams through L2 once per pass
  const int qhalf = p.q_rows * 128;
  int stage = 0, phase = 0, pc = 0;
  int last_q_pc = -1;
  int last_ph[kMaxStages];
  for (int i = 0; i < kMaxStages; ++i) last_ph[i] = -1;
  TileIter c;
  for (c.init(p, fb, fe); c.valid(); c.next(p)) {
    if (ctl->abort) break;
    if (c.first(fb)) {
      if (!mbar_wait(&ctl->q_empty, (pc & 1) ^ 1, p.wait_ns)) { fail(ctl, p.err); break; }
      const int zq = p.layer0 + c.l, y = c.g * p.rows;
      if (PASS == 1) {
        mbar_arrive_expect_tx(&ctl->q_full, p.rows * 256);
        for (int h = 0; h < 2; ++h) {
          tma_load_3d(sQ + h * qhalf, &p.tmqa[c.s], &ctl->q_full, h * 64, y, zq);
          if (p.rows > kTileKeys)
            tma_load_3d(sQ + h * qhalf + kTileKeys * 128, &p.tmqb[c.s], &ctl->q_full, h * 64, y + kTileKeys, zq);
        }
      } else {
        mbar_arrive_expect_tx(&ctl->q_full, p.n2 * 256);
        for (int h = 0; h < 2; ++h) tma_load_3d(sQ + h * qhalf, &p.tmq2[c.s], &ctl->q_full, h * 64, y, zq);
      }
      last_q_pc = pc;
      ++pc;
    }
    if (!mbar_wait(&ctl->k_empty[stage], phase ^ 1, p.wait_ns)) { fail(ctl, p.err); break; }
    mbar_arrive_expect_tx(&ctl->k_full[stage], kTileBytes);
    const int zk = (p.layer0 + c.l) * p.G + c.g;
    for (int h = 0; h < 2; ++h)
      tma_load_3d_hint(sK + stage * kTileBytes + h * kHalfBytes, &p.tmk[c.s], &ctl->k_full[stage],
                       h * 64, c.j * kTileKeys, zk, pol_k);
    last_ph[stage] = phase;
    if (++stage == p.kstages) {
      stage = 0;
      phase ^= 1;
    }
  }
  if (ctl->abort) {
    // bring every issued copy to completion before the CTA can exit
    for (int i = 0; i < p.kstages; ++i)
      if (last_ph[i] >= 0) mbar_wait(&ctl->k_full[i], last_ph[i], drain_limit(p.wait_ns));
    if (last_q_pc >= 0) mbar_wait(&ctl->q_full, last_q_pc & 1, drain_limit(p.wait_ns));
  }
}

// MMA issuer shared by both passes.  Two issuing threads (warps 1 and 2)
// take the even and the odd tiles of the CTA's range, so the bookkeeping of
// one (barrier waits, commits, tile iteration) overlaps the other's MMAs: a
// single issuing thread leaves the tensor pipe idle for about that long every
// tile.  Issuer `who` owns TMEM accumulator stage `who`; both walk every tile
// to follow the piece boundaries and each commits the Q release of a piece
// for its own MMAs.
template <int PASS>
__device__ void mma_loop(const ScoreParams& p, SmemCtl* ctl, const uint8_t* sQ, const uint8_t* sK,
                         const uint8_t* sX, uint32_t tmem, int64_t fb, int64_t fe, int who) {
  const uint32_t idesc = PASS == 1 ? idesc_bf16(128, kTileKeys) : idesc_bf16(128, p.n2);
  // shared-memory descriptors are built once; an MMA only adds its operand's
  // offset (in 16-byte units) to the start-address field, which cannot carry
  // out of the field inside the 227 KB window
  const uint64_t dq0 = sdesc_k_sw128(smem_u32(sQ)), dk0 = sdesc_k_sw128(smem_u32(sK));
  const uint32_t qhalf16 = (p.q_rows * 128) >> 4;
  // pass 2, one more K step per tile: a constant operand of ones (every 8-key
  // group shares one core matrix) times each window row's -lse2 / scale as
  // three bf16 parts, so that the accumulator holds z - lse2 / scale
  const uint64_t dax = sdesc_k_none(smem_u32(sX), 128, 0);
  const uint64_t dbx0 = sdesc_k_none(smem_u32(sX) + kXOnesBytes, 128, 256);
  uint64_t dbx = dbx0;
  // K stage and phase of tile jt = who, who + 2, ...
  int stage = who % p.kstages, phase = 0, pc = 0, own = 0;
  const uint32_t d0 = tmem + who * 256;
  int64_t jt = 0;
  TileIter c;
  for (c.init(p, fb, fe); c.valid(); c.next(p), ++jt) {
    if (ctl->abort) break;
    if (c.first(fb)) {
      if (!mbar_wait(&ctl->q_full, pc & 1, p.wait_ns)) { fail(ctl, p.err); break; }
      if (PASS == 2) {
        if (!mbar_wait(&ctl->x_full[pc & 1], (pc >> 1) & 1, p.wait_ns)) { fail(ctl, p.err); break; }
        dbx = dbx0 + static_cast<uint64_t>((pc & 1) * ((p.q_rows * kXRowBytes) >> 4));
      }
      ++pc;
    }
    if ((jt & 1) == who) {
      if (!mbar_wait(&ctl->k_full[stage], phase, p.wait_ns)) { fail(ctl, p.err); break; }
      if (!mbar_wait(&ctl->t_empty[who], (own & 1) ^ 1, p.wait_ns)) { fail(ctl, p.err); break; }
      tc_fence_after();
      const uint64_t dk = dk0 + static_cast<uint64_t>(stage * (kTileBytes >> 4));
      if (PASS == 1) {
#pragma unroll
        for (int mt = 0; mt < 2; ++mt) {
          if (mt >= p.n_mtiles) break;
          const uint32_t d = d0 + mt * kTileKeys;
          // M tile 1 reads rows 128..255 of each Q half; rows past q_rows are
          // other shared memory and only feed accumulator rows that are dropped
          const uint64_t dq = dq0 + static_cast<uint64_t>(mt * ((kTileKeys * 128) >> 4));
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const uint32_t koff16 = (kk >> 2) * (kHalfBytes >> 4) + (kk & 3) * 2;
            const uint32_t qoff16 = (kk >> 2) * qhalf16 + (kk & 3) * 2;
            mma_bf16(d, dq + qoff16, dk + koff16, idesc, kk > 0);
          }
          mma_commit(&ctl->t_full[who][mt]);   // that M tile's epilogue starts without waiting for the next
        }
      } else {
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t koff16 = (kk >> 2) * (kHalfBytes >> 4) + (kk & 3) * 2;
          const uint32_t qoff16 = (kk >> 2) * qhalf16 + (kk & 3) * 2;
          mma_bf16(d0, dk + koff16, dq0 + qoff16, idesc, kk > 0);
        }
        mma_bf16(d0, dax, dbx, idesc, 1);
        mma_commit(&ctl->t_full[who][0]);
      }
      mma_commit(&ctl->k_empty[stage]);
      ++own;
      stage += 2;
      if (stage >= p.kstages) {
        stage -= p.kstages;
        phase ^= 1;
      }
    }
    if (c.last()) mma_commit(&ctl->q_empty);
  }
  // every MMA issued above must be complete before TMEM is released
  mma_commit(&ctl->drain);
  mbar_wait(&ctl->drain, 0, drain_limit(p.wait_ns));
}

// log2-domain log-sum-exp of window row `col` of the (seq, layer, group) row
// whose first flat tile is `r0`, from the pass-1 partials of every CTA piece
// that covered the row: one pass, eight partials loaded at a time, each batch
// merged into the running (maximum, sum).
__device__ float combine_lse2(const ScoreParams& p, int64_t r0, int nt, int col) {
  const int64_t T = p.total_tiles;
  const int P = p.grid1;
  const int64_t r1 = r0 + nt - 1;
  const int c0 = static_cast<int>(((r0 + 1) * P - 1) / T);
  const int c1 = static_cast<int>(((r1 + 1) * P - 1) / T);
  float mx = -INFINITY, sum = 0.f;
  for (int cb = c0; cb <= c1; cb += 8) {
    float2 v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      v[k] = make_float2(-INFINITY, 0.f);
      if (cb + k <= c1) v[k] = p.partials[max(range_begin(T, cb + k, P), r0) * kMaxRows + col];
    }
    float bm = mx;
#pragma unroll
    for (int k = 0; k < 8; ++k) bm = fmaxf(bm, v[k].x);
    if (bm == -INFINITY) continue;
    float bs = mx == -INFINITY ? 0.f : sum * exp2f(mx - bm);
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (v[k].x != -INFINITY) bs += v[k].y * exp2f(v[k].x - bm);
    mx = bm;
    sum = bs;
  }
  return mx + log2f(sum);
}

// Streams `n` 16-column chunks of this thread's TMEM lane from `base`, one
// load in flight under the arithmetic of the previous chunk.
template <typename F>
__device__ __forceinline__ void stream16(uint32_t base, int n, F&& consume) {
  uint32_t A[16], B[16];
  tmem_ld16_async(base, A);
  tmem_wait16(A);
  for (int ch = 0;; ch += 2) {
    const bool hb = ch + 1 < n;
    if (hb) tmem_ld16_async(base + (ch + 1) * 16, B);
    consume(A, ch);
    if (!hb) break;
    tmem_wait16(B);
    const bool ha = ch + 2 < n;
    if (ha) tmem_ld16_async(base + (ch + 2) * 16, A);
    consume(B, ch + 1);
    if (!ha) break;
    tmem_wait16(A);
  }
}

__device__ __forceinline__ float2 f2(uint32_t a, uint32_t b) { return make_float2(__uint_as_float(a), __uint_as_float(b)); }

// a0, a1 += exp2(z * sc - m) over 16 logits given as raw TMEM words (packed pairs)
__device__ __forceinline__ void exp2_acc16(const uint32_t (&r)[16], float2 sc2, float2 nm2, float2& a0, float2& a1) {
#pragma unroll
  for (int i = 0; i < 16; i += 4) {
    const float2 t0 = ffma2(f2(r[i], r[i + 1]), sc2, nm2);
    const float2 t1 = ffma2(f2(r[i + 2], r[i + 3]), sc2, nm2);
    a0 = fadd2(a0, make_float2(ex2_approx(t0.x), ex2_approx(t0.y)));
    a1 = fadd2(a1, make_float2(ex2_approx(t1.x), ex2_approx(t1.y)));
  }
}

// the same over the first `lim` logits only (the ragged last tile of a row)
__device__ __forceinline__ void exp2_acc16_masked(const uint32_t (&r)[16], int lim, float2 sc2, float2 nm2,
                                                  float2& a0, float2& a1) {
#pragma unroll
  for (int i = 0; i < 16; i += 2) {
    const float2 t = ffma2(f2(r[i], r[i + 1]), sc2, nm2);
    a0 = fadd2(a0, make_float2(i < lim ? ex2_approx(t.x) : 0.f, i + 1 < lim ? ex2_approx(t.y) : 0.f));
  }
}

// maximum over the first `lim` of 16 logits (-inf when none)
__device__ __forceinline__ float max16_masked(const uint32_t (&r)[16], int lim) {
  float mx = -INFINITY;
#pragma unroll
  for (int i = 0; i < 16; ++i)
    if (i < lim) mx = fmaxf(mx, __uint_as_float(r[i]));
  return mx;
}

// Slow path of lse_tile, taken by the whole warp (TMEM loads are
// warp-collective): the first tile of a piece (no reference yet), the ragged
// last tile of a row, or a tile with a logit more than 64 above the
// reference in some lane.  Each lane moves its reference to max(reference,
// its tile maximum), rescales its sum and adds the tile's valid keys.
__device__ __forceinline__ void lse_tile_slow(uint32_t base, int n, int lim, float sc, bool live, float& m, float& s) {
  float mx = -INFINITY;
  for (int ch = 0; ch < n; ++ch) {
    uint32_t r[16];
    tmem_ld16_async(base + ch * 16, r);
    tmem_wait16(r);
    mx = fmaxf(mx, max16_masked(r, lim - ch * 16));
  }
  const float mn = fmaxf(m, mx * sc);
  if (m != -INFINITY) s *= ex2_approx(m - mn);
  m = mn;
  const float2 sc2 = make_float2(sc, sc), nm2 = make_float2(-m, -m);
  float2 a0 = make_float2(0.f, 0.f), a1 = make_float2(0.f, 0.f);
  for (int ch = 0; ch < n; ++ch) {
    uint32_t r[16];
    tmem_ld16_async(base + ch * 16, r);
    tmem_wait16(r);
    exp2_acc16_masked(r, lim - ch * 16, sc2, nm2, a0, a1);
  }
  const float2 a = fadd2(a0, a1);
  if (live) s += a.x + a.y;   // a lane past the window rows holds garbage
}

// One row's running (reference m, sum s of exp2(z sc - m)) over this thread's
// `nch` 16-key chunks of one tile, `lim` of which keys are valid.  The
// reference is set on a piece's first tile and moves only when a tile's sum
// exceeds 2^64 (a logit more than 64 above it, or overflow); that tile is then
// redone.  Terms far below the reference underflow to zero, below the fp32
// resolution of the sum.  A lane that is not `live` (a row past the group's
// window rows) takes part in the warp-collective loads only.  The full-tile
// path is straight-line; everything else goes through the slow path.
__device__ __forceinline__ void lse_tile(uint32_t base, int nch, int lim, float sc, bool live, float& m, float& s) {
  if (lim <= 0) return;   // lim is the same in every lane
  if (lim < nch * 16 || __any_sync(kFull, m == -INFINITY)) {
    lse_tile_slow(base, min(nch, (lim + 15) >> 4), lim, sc, live, m, s);
    return;
  }
  const float2 sc2 = make_float2(sc, sc), nm2 = make_float2(-m, -m);
  float2 a0 = make_float2(0.f, 0.f), a1 = make_float2(0.f, 0.f);
  stream16(base, nch, [&](const uint32_t(&r)[16], int) { exp2_acc16(r, sc2, nm2, a0, a1); });
  const float2 a = fadd2(a0, a1);
  const float cs = a.x + a.y;
  if (__all_sync(kFull, !live || cs < 1.8446744e19f)) {   // below 2^64: the common case
    if (live) s += cs;
  } else {
    lse_tile_slow(base, nch, lim, sc, live, m, s);
  }
}

}  // namespace

// 20 warps share the register file: at most 96 registers a thread.
__global__ void __launch_bounds__(kScoreThreads, 1) k_score_lse(const __grid_constant__ ScoreParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sQ = smem;                          // [2 halves][q_rows][128 B]
  uint8_t* sK = smem + 2 * p.q_rows * 128;     // [kstages][2 halves][128][128 B]
  SmemCtl* ctl = reinterpret_cast<SmemCtl*>(sK + p.kstages * kTileBytes);
  float2* pbuf = reinterpret_cast<float2*>(reinterpret_cast<uint8_t*>(ctl) + 256);   // [4 wg][128]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) ctl_init(ctl, p.kstages);
  if (warp == 1) {
    tmem_alloc(&ctl->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // the set-up above overlaps the previous kernel's tail; its outputs are read below
  griddep_launch_dependents();
  griddep_wait();
  const uint32_t tmem = ctl->tmem_base;
  const int64_t T = p.total_tiles;
  const int64_t fb = range_begin(T, blockIdx.x, gridDim.x);
  const int64_t fe = range_begin(T, blockIdx.x + 1, gridDim.x);

  if (warp == 0) {
    if (lane == 0) producer_loop<1>(p, ctl, sQ, sK, fb, fe);
  } else if (warp == 1 || warp == 2) {
    if (lane == 0) mma_loop<1>(p, ctl, sQ, sK, nullptr, tmem, fb, fe, warp - 1);
  } else if (warp >= kEpiWarp0) {
    const int wg = (warp - kEpiWarp0) >> 2;  // epilogue warpgroup 0..3
    const int quad = warp & 3;              // TMEM lane quadrant
    const int q = quad * 32 + lane;         // TMEM lane
    // two M tiles: warpgroup (mt, half) owns 64 keys of M tile mt;
    // one M tile: the four warpgroups own 32 keys each
    const bool two = p.n_mtiles == 2;
    const int mt = two ? (wg >> 1) : 0;
    const int kofs = two ? (wg & 1) * 64 : wg * 32;
    const int nch = two ? 4 : 2;
    const int r = mt * kTileKeys + q;       // window row within the group
    const bool active = mt * kTileKeys + quad * 32 < p.rows;
    const uint32_t base0 = tmem + (static_cast<uint32_t>(quad * 32) << 16) + mt * kTileKeys + kofs;
    const float sc = p.scale2;
    float m = -INFINITY, s = 0.f;
    int jt = 0;
    bool dead = false;
    int64_t piece_start = 0;
    // Every epilogue warp walks every tile and meets the piece-end barrier in
    // the same order; a warp whose wait ran out keeps walking without waiting.
    TileIter c;
    for (c.init(p, fb, fe); c.valid(); c.next(p)) {
      const bool last = c.last();
      if (c.first(fb)) {
        piece_start = c.f;
        m = -INFINITY;
        s = 0.f;
      }
      const int ts = jt & 1;
      if (!dead) {
        if (!__all_sync(kFull, mbar_wait(&ctl->t_full[ts][mt], (jt >> 1) & 1, p.wait_ns))) {
          fail(ctl, p.err);
          dead = true;
        } else {
          tc_fence_after();
          if (active) lse_tile(base0 + ts * 256, nch, p.seq[c.s].Lp - (c.j * kTileKeys + kofs), sc, r < p.rows, m, s);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&ctl->t_empty[ts]);
        }
      }
      if (last) {
        // merge the key parts of each row, write the piece's partial
        pbuf[wg * 128 + q] = make_float2(m, s);
        named_bar_sync(1, kEpiThreads);
        const bool writer = two ? (wg & 1) == 0 : wg == 0;
        if (writer && r < p.rows && !dead) {
          const int n = two ? 2 : 4;
          const int w0 = two ? wg : 0;
          float mx = -INFINITY;
          for (int i = 0; i < n; ++i) mx = fmaxf(mx, pbuf[(w0 + i) * 128 + q].x);
          float sum = 0.f;
          if (mx != -INFINITY)
            for (int i = 0; i < n; ++i) {
              const float2 v = pbuf[(w0 + i) * 128 + q];
              if (v.x != -INFINITY) sum += v.y * ex2_approx(v.x - mx);
            }
          p.partials[piece_start * kMaxRows + r] = make_float2(mx, sum);
        }
        named_bar_sync(1, kEpiThreads);   // pbuf is reused by the next piece
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

__global__ void __launch_bounds__(kScoreThreads, 1) k_score_accum(const __grid_constant__ ScoreParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* sQ = smem;                          // [2 halves][q_rows][128 B]
  uint8_t* sK = smem + 2 * p.q_rows * 128;     // [kstages][2 halves][128][128 B]
  SmemCtl* ctl = reinterpret_cast<SmemCtl*>(sK + p.kstages * kTileBytes);
  // ones operand [256 B], then two buffers of the -lse operand [q_rows][32 B]
  uint8_t* sX = reinterpret_cast<uint8_t*>(ctl) + 256;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) ctl_init(ctl, p.kstages);
  if (warp == 1) {
    tmem_alloc(&ctl->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // the set-up above overlaps the previous kernel's tail; its outputs are read below
  griddep_launch_dependents();
  griddep_wait();
  const uint32_t tmem = ctl->tmem_base;
  const int64_t T = p.total_tiles;
  const int64_t fb = range_begin(T, blockIdx.x, gridDim.x);
  const int64_t fe = range_begin(T, blockIdx.x + 1, gridDim.x);

  if (warp == 0) {
    if (lane == 0) producer_loop<2>(p, ctl, sQ, sK, fb, fe);
  } else if (warp == 1 || warp == 2) {
    if (lane == 0) mma_loop<2>(p, ctl, sQ, sK, sX, tmem, fb, fe, warp - 1);
  } else if (warp >= kEpiWarp0) {
    const int et = threadIdx.x - 32 * kEpiWarp0;   // 0..511
    const int wg = et >> 7;                 // column quarter
    const int quad = warp & 3;
    const int q = quad * 32 + lane;         // key within the tile
    const int nc = p.n2 >> 4;               // 16-column chunks
    const int ch0 = wg * (nc >> 2) + min(wg, nc & 3);
    const int nch = (nc >> 2) + (wg < (nc & 3) ? 1 : 0);
    const uint32_t base0 = tmem + (static_cast<uint32_t>(quad * 32) << 16) + ch0 * 16;
    const float sc = p.scale2, isc = 1.f / p.scale2, sqd = sqrtf(static_cast<float>(kHeadDim));
    // the -lse operand of the piece `it` (whose row starts at flat tile r0),
    // into buffer `buf`: window row et holds x = -lse2 / scale (= -lse sqrt(d)
    // for a supplied natural-log normaliser) as three bf16 parts (x = hi + mid
    // + lo to about 2^-24 relative) in its K columns 0..2; rows past the
    // group's window rows get a large negative x (exp2 -> 0)
    auto write_x = [&](const TileIter& it, int64_t r0, int buf) {
      if (et < p.n2) {
        float x = -3.0e38f;
        if (et < p.rows) {
          const float* lse = p.seq[it.s].lse;
          x = lse ? -lse[(static_cast<int64_t>(p.layer0 + it.l) * p.G + it.g) * p.rows + et] * sqd
                  : -combine_lse2(p, r0, it.nt, et) * isc;
        }
        const __nv_bfloat16 hi = __float2bfloat16_rn(x);
        const float r1 = x - __bfloat162float(hi);
        const __nv_bfloat16 mid = __float2bfloat16_rn(r1);
        const __nv_bfloat16 lo = __float2bfloat16_rn(r1 - __bfloat162float(mid));
        uint8_t* row = sX + kXOnesBytes + buf * (p.q_rows * kXRowBytes) + (et >> 3) * 256 + (et & 7) * 16;
        *reinterpret_cast<uint4*>(row) =
            make_uint4(static_cast<uint32_t>(__bfloat16_as_ushort(hi)) | (static_cast<uint32_t>(__bfloat16_as_ushort(mid)) << 16),
                       static_cast<uint32_t>(__bfloat16_as_ushort(lo)), 0u, 0u);
        *reinterpret_cast<uint4*>(row + 128) = make_uint4(0u, 0u, 0u, 0u);
      }
      fence_proxy_async_smem();
      named_bar_sync(1, kEpiThreads);
      if (et == 0) mbar_arrive(&ctl->x_full[buf]);
    };
    int jt = 0, kp = 0;
    bool dead = false;
    float* dst = nullptr;   // this thread's copy of the piece's unpooled row
    int lp = 0;
    TileIter c;
    c.init(p, fb, fe);
    if (c.valid()) {
      // the ones operand: bf16 1.0 in K columns 0..2 of core matrix 0, zeros elsewhere
      if (et < 16) {
        *reinterpret_cast<uint4*>(sX + et * 16) =
            et < 8 ? make_uint4(0x3F803F80u, 0x00003F80u, 0u, 0u) : make_uint4(0u, 0u, 0u, 0u);
      }
      write_x(c, c.f - c.j, 0);
    }
    const float2 sc2 = make_float2(sc, sc), zero2 = make_float2(0.f, 0.f);
    for (; c.valid(); c.next(p)) {
      if (c.first(fb)) {
        // the next piece's operand goes to the other buffer now, one piece
        // ahead of its MMAs (this piece's buffer was written one piece earlier;
        // the other one's readers, the previous piece's MMAs, are done)
        const int64_t fn = c.f + (c.nt - c.j);
        if (fn < fe) {
          TileIter n;
          n.init(p, fn, fe);
          write_x(n, fn, (kp + 1) & 1);
        }
        ++kp;
        const ScoreSeq& sq = p.seq[c.s];
        lp = sq.Lp;
        dst = sq.s_raw + (static_cast<int64_t>(c.l * p.G + c.g) * kRawCopies + wg) * raw_stride(lp) + q;
      }
      const int ts = jt & 1;
      if (!dead) {
        if (!__all_sync(kFull, mbar_wait(&ctl->t_full[ts][0], (jt >> 1) & 1, p.wait_ns))) {
          fail(ctl, p.err);
          dead = true;
        } else {
          tc_fence_after();
          float2 a0 = make_float2(0.f, 0.f), a1 = make_float2(0.f, 0.f);
          if (nch > 0)
            stream16(base0 + ts * 256, nch, [&](const uint32_t(&v)[16], int) { exp2_acc16(v, sc2, zero2, a0, a1); });
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&ctl->t_empty[ts]);
          const int key0 = c.j * kTileKeys;
          const float2 a = fadd2(a0, a1);
          if (key0 + q < lp) dst[key0] = a.x + a.y;
        }
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
// divisor k), S_raw being the sum of its column-quarter copies.  grid: (ceil(Lp_max / 256), nlayers * G, nseq)
__global__ void k_pool(const __grid_constant__ SeqBatch b, int G, int H, int pool) {
  griddep_launch_dependents();
  griddep_wait();
  const SeqView& s = b.s[blockIdx.z];
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= s.Lp) return;
  const int lg = blockIdx.y;                  // launch-local layer * G + g
  const int layer = b.layer0 + lg / G, g = lg % G;
  const int rs = raw_stride(s.Lp);
  const float* src = s.s_raw + static_cast<int64_t>(lg) * kRawCopies * rs;
  const int half = pool >> 1;
  float acc = 0.f;
  for (int j = -half; j <= half; ++j) {
    const int u = t + j;
    if (u >= 0 && u < s.Lp) {
      float r = 0.f;
      for (int c = 0; c < kRawCopies; ++c) r += src[c * rs + u];
      acc += r;
    }
  }
  const float scale = static_cast<float>(G) / static_cast<float>(H) / static_cast<float>(pool);
  s.S[(static_cast<int64_t>(layer) * G + g) * s.Lp + t] = acc * scale;
}

// alignment slack + Q + K stages + control block + the larger of the pass-1
// merge buffer and the pass-2 -lse operands (ones + two row buffers)
size_t score_smem_bytes(int q_rows, int kstages) {
  const size_t aux = std::max<size_t>(4 * 128 * sizeof(float2), kXOnesBytes + 2 * static_cast<size_t>(q_rows) * kXRowBytes);
  return 1024 + static_cast<size_t>(2 * q_rows * 128) + static_cast<size_t>(kstages) * kTileBytes + 256 + aux;
}

// The K-stage count is even: MMA issuer `who` takes tiles who, who + 2, ..., so
// with an even count every stage belongs to one issuer, which consumes its
// phases in order.  With an odd count consecutive uses of a stage alternate
// between the issuers, and one can wait on the stage's next phase while the
// other's load of it is still in flight (the parity wait then passes early).
int score_kstages(int q_rows) {
  int k = kMaxStages & ~1;
  while (k > 0 && score_smem_bytes(q_rows, k) > kSmemLimit) k -= 2;
  return k;
}

cudaError_t score_configure() {
  const int bytes = static_cast<int>(kSmemLimit);
  cudaError_t e = cudaFuncSetAttribute(k_score_lse, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(k_score_accum, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

namespace {

// Launch with programmatic stream serialization: the kernel may start its
// set-up while the previous kernel of the stream drains (it waits in
// griddep_wait before reading that kernel's outputs).
template <typename... Args, typename... Act>
cudaError_t launch_pdl(void (*kernel)(Args...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                       Act&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Act>(args)...);
}

}  // namespace

cudaError_t score_lse_launch(const ScoreParams& p, int grid, cudaStream_t stream) {
  return launch_pdl(k_score_lse, dim3(grid), dim3(kScoreThreads), score_smem_bytes(p.q_rows, p.kstages), stream, p);
}

cudaError_t score_accum_launch(const ScoreParams& p, int grid, cudaStream_t stream) {
  return launch_pdl(k_score_accum, dim3(grid), dim3(kScoreThreads), score_smem_bytes(p.q_rows, p.kstages), stream, p);
}

cudaError_t pool_launch(const SeqBatch& b, int G, int H, int pool, int lp_max, cudaStream_t stream) {
  if (lp_max <= 0) return cudaSuccess;
  dim3 grid(ceil_div(lp_max, 256), b.nlayers * G, b.nseq);
  return launch_pdl(k_pool, grid, dim3(256), 0, stream, b, G, H, pool);
}

// Self-test of the failure path that every bounded wait above shares: one
// thread waits on a shared-memory barrier that nothing arrives on; the wait
// gives up after `limit_ns`, latches the timeout code and the kernel returns.
__global__ void k_wait_probe(uint32_t* err, uint64_t limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  fence_mbar_init();
  if (!mbar_wait(&bar, 0, limit_ns)) atomicOr(err, kErrTimeout);
}

cudaError_t wait_probe_launch(uint32_t* err, uint64_t limit_ns, cudaStream_t stream) {
  k_wait_probe<<<1, 32, 0, stream>>>(err, limit_ns);
  return cudaGetLastError();
}

}  // namespace starkv
