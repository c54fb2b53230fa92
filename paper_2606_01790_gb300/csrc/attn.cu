// Attention output and softmax normaliser of the window rows over the past
// keys: the part of a layer's own attention pass that computes the logits the
// compression scores (Sec. 3.3, Eq. 2; App. A.3 counts that Q K^T as shared
// with the attention).  For every (layer, group) row block of (H/G) w window
// rows r against the L_p past keys t (the window keys excluded, as in Eq. 2):
//   O[r]   = sum_t softmax_t(Q_r . K_t / sqrt(d)) V_t
//   lse[r] = log sum_t exp(Q_r . K_t / sqrt(d))       (natural log)
// lse is what starkv_seq.lse takes, so the compression can skip its first
// scoring pass (a whole read of K).  A model's causal attention for these
// rows adds the window keys' part by the usual log-sum-exp merge.
//
// Work split: the flat (seq, layer, group, 64-key unit) space in one
// contiguous range per CTA (persistent grid <= #SMs).  A run of units of one
// row inside a range is a piece; its partial (reference m, sum l, unnormalised
// O) goes to slot row + CTA (distinct for every piece: ranges and rows are
// both in flat order) and k_attn_combine merges the pieces of each row.
//
// Per unit on tcgen05, with two 128-row M tiles for up to 256 window rows:
//   S = Q K^T           M = 128 rows, N = 64 keys, K = d, bf16 -> fp32 in TMEM
//                       (two S stages, so the MMA of unit u+1 runs under the
//                       softmax of unit u);
//   softmax             rows on TMEM lanes, one thread per row: S read in two
//                       halves (the second half's loads under the first half's
//                       arithmetic), p = exp2(S c - m), l += p in fp32, P
//                       rounded to fp16 and written over the first 32 of the
//                       unit's 64 S columns (two fp16 per 32-bit column);
//   O += P V            M = 128, N = d = 128, K = 64 keys, fp16 -> fp32 in TMEM,
//                       A = P read from tensor memory;
//                       V arrives as bf16 and four warps convert it to fp16 in
//                       place (exact for |v| < 65504), read as the transposed
//                       (MN-major) operand.
// The row reference m is the piece's first unit's maximum and moves only when
// a unit's maximum exceeds it by more than 15 (fp16 holds P < 2^16); the move
// rescales that row's O in TMEM after the previous unit's P V is done (rare).
// Later units take no maximum unless their sum of P exceeds 2^15: below that
// no p can exceed 2^15, so no reference can have to move.
// An S stage holds P until the P V product of its unit is done, which frees
// it for S two units later.  Warp roles: warp 0 loads K (a four-stage ring,
// each stage free once S of its unit is done) and Q per piece, warp 3 loads V
// (a four-stage ring, free once the P V product is done), warp 1 issues S and
// owns TMEM, warp 2 issues P V, warps 4..11 softmax (warpgroup = M tile),
// warps 12..15 V conversion.
#include <algorithm>
#include <utility>

#include <cuda_fp16.h>

#include "attn.cuh"
#include "common.cuh"
#include "ptx.cuh"

namespace starkv {

namespace {

constexpr int kStages = 4;                        // largest depth of the K ring and of the V ring
constexpr int kUnitBytes = kAttnUnitKeys * 256;   // 64 keys x 128 bf16: 16 KB (K or V)
constexpr int kHalfBytes = kAttnUnitKeys * 128;   // one 64-column half of a unit: 8 KB
constexpr int kTmemCols = 512;                    // O [0, 256), S stage t at 256 + 128 t
constexpr int kSoftWarp0 = 4, kSoftWarps = 8;
constexpr int kConvWarp0 = 12, kConvWarps = 4;
constexpr uint32_t kFull = 0xffffffffu;
constexpr float kMoveThreshold = 15.f;            // log2 units: P stays below 2^16
constexpr uint64_t kDrainWaitNs = 2000000000ull;
constexpr size_t kSmemLimit = 227 * 1024;

__device__ __forceinline__ uint64_t drain_limit(uint64_t wait_ns) {
  return wait_ns > kDrainWaitNs ? wait_ns : kDrainWaitNs;
}

struct AttnCtl {
  uint64_t k_full[kStages], k_empty[kStages];
  uint64_t v_full[kStages], v_empty[kStages], v_ready[kStages];
  uint64_t s_full[2][2];   // [stage][M tile]: S of that M tile is in the stage
  uint64_t s_empty[2];      // the stage's P V products are done
  uint64_t p_full[2][2];    // [stage][M tile]: P of that M tile is written
  uint64_t q_full, q_empty, drain;
  uint32_t tmem_base;
  volatile int abort;
};

constexpr int kCtlBytes = 512;
static_assert(sizeof(AttnCtl) <= kCtlBytes, "the control block fits its bytes");

__device__ __forceinline__ void fail(AttnCtl* ctl, uint32_t* err) {
  ctl->abort = 1;
  atomicOr(err, kErrTimeout);
}

// Shared-memory descriptor of an MN-major operand in 128-byte swizzled rows
// (TMA SWIZZLE_128B of a [K][MN] tile, MN contiguous): 64-element MN groups
// `lbo` bytes apart, 8-row K groups `sbo` bytes apart.
__device__ __forceinline__ uint64_t sdesc_mn_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr >> 4) & 0x3FFFu);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
  d |= static_cast<uint64_t>(1) << 46;   // descriptor version (tcgen05)
  d |= static_cast<uint64_t>(2) << 61;   // swizzle mode: 128 B
  return d;
}

// Instruction descriptor of tcgen05.mma kind::f16 with fp16 A (K-major) and
// fp16 B (MN-major), fp32 accumulator, shape M x N.
__host__ __device__ constexpr uint32_t idesc_f16_bmn(int M, int N) {
  return (1u << 4)                                   // D format: f32
         | (1u << 16)                                // B major: MN
         | (static_cast<uint32_t>(N >> 3) << 17)
         | (static_cast<uint32_t>(M >> 4) << 24);
}

// D[tmem] (+)= A[tmem] * B[smem]: A with M = 128 rows on TMEM lanes and its
// K elements as fp16 pairs, lower index in the low half of each 32-bit column.
__device__ __forceinline__ void mma_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                           uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// 8 consecutive 32-bit columns of this warp's 32 TMEM lanes, stored.
__device__ __forceinline__ void tmem_st8(uint32_t taddr, const uint32_t (&r)[8]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};\n" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
      : "memory");
}

// 16 consecutive fp32 columns of this warp's 32 TMEM lanes, stored.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};\n" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

__device__ __forceinline__ uint32_t pack_half2(float a, float b) {
  const __half2 h = __floats2half2_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// bf16 pair (one 32-bit word) -> fp16 pair, exact for |x| < 65504
__device__ __forceinline__ uint32_t bf16x2_to_f16x2(uint32_t w) {
  return pack_half2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
}

// Coordinates of consecutive flat units [f0, f1), advanced without divisions.
struct UnitIter {
  int s, l, g, j, nu;
  int64_t f, fe;
  __device__ void init(const AttnParams& p, int64_t f0, int64_t f1) {
    f = f0;
    fe = f1;
    s = l = g = j = nu = 0;
    if (f >= fe) return;
    while (s + 1 < p.nseq && p.seq[s + 1].unit_base <= f0) ++s;
    nu = p.seq[s].nu;
    const int64_t u = f0 - p.seq[s].unit_base;
    const int per_layer = p.G * nu;
    l = static_cast<int>(u / per_layer);
    const int rem = static_cast<int>(u - static_cast<int64_t>(l) * per_layer);
    g = rem / nu;
    j = rem - g * nu;
  }
  __device__ bool valid() const { return f < fe; }
  __device__ bool first(int64_t fb) const { return f == fb || j == 0; }
  __device__ bool last() const { return f + 1 == fe || j + 1 == nu; }
  __device__ int row(const AttnParams& p) const { return (s * p.nlayers + l) * p.G + g; }
  __device__ void next(const AttnParams& p) {
    ++f;
    if (f >= fe) return;
    if (++j < nu) return;
    j = 0;
    if (++g < p.G) return;
    g = 0;
    if (++l < p.nlayers) return;
    l = 0;
    do {
      ++s;
    } while (s + 1 < p.nseq && p.seq[s].nu == 0);
    nu = p.seq[s].nu;
  }
};

__device__ __forceinline__ int64_t range_begin(int64_t T, int c, int P) { return T * c / P; }

// CTA whose range holds flat unit f
__host__ __device__ __forceinline__ int cta_of(int64_t f, int64_t T, int P) {
  return static_cast<int>(((f + 1) * P - 1) / T);
}

// K (and Q per piece) loader: a K stage is free once S of its unit is done,
// so K runs ahead of the products.
__device__ void k_loader(const AttnParams& p, AttnCtl* ctl, uint8_t* sQ, uint8_t* sK, int64_t fb, int64_t fe) {
  const uint64_t pol = policy_evict_first();   // K and V stream through L2 once
  const int qhalf = p.q_rows * 128;
  int stage = 0, phase = 0, pc = 0, last_q_pc = -1;
  int last_ph[kStages];
  for (int i = 0; i < kStages; ++i) last_ph[i] = -1;
  UnitIter c;
  for (c.init(p, fb, fe); c.valid(); c.next(p)) {
    if (ctl->abort) break;
    if (c.first(fb)) {
      if (!mbar_wait(&ctl->q_empty, (pc & 1) ^ 1, p.wait_ns)) { fail(ctl, p.err); break; }
      const int zq = p.layer0 + c.l, y = c.g * p.rows;
      mbar_arrive_expect_tx(&ctl->q_full, p.rows * 256);
      for (int h = 0; h < 2; ++h) {
        tma_load_3d(sQ + h * qhalf, &p.tmqa[c.s], &ctl->q_full, h * 64, y, zq);
        if (p.rows > 128) tma_load_3d(sQ + h * qhalf + 128 * 128, &p.tmqb[c.s], &ctl->q_full, h * 64, y + 128, zq);
      }
      last_q_pc = pc;
      ++pc;
    }
    if (!mbar_wait(&ctl->k_empty[stage], phase ^ 1, p.wait_ns)) { fail(ctl, p.err); break; }
    mbar_arrive_expect_tx(&ctl->k_full[stage], kUnitBytes);
    const int zk = (p.layer0 + c.l) * p.G + c.g, y = c.j * kAttnUnitKeys;
    for (int h = 0; h < 2; ++h)
      tma_load_3d_hint(sK + stage * kUnitBytes + h * kHalfBytes, &p.tmk[c.s], &ctl->k_full[stage], h * 64, y, zk, pol);
    last_ph[stage] = phase;
    if (++stage == p.kv_stages) {
      stage = 0;
      phase ^= 1;
    }
  }
  if (ctl->abort) {   // every issued copy completes before the CTA can exit
    for (int i = 0; i < kStages; ++i)
      if (last_ph[i] >= 0) mbar_wait(&ctl->k_full[i], last_ph[i], drain_limit(p.wait_ns));
    if (last_q_pc >= 0) mbar_wait(&ctl->q_full, last_q_pc & 1, drain_limit(p.wait_ns));
  }
}

// V loader: a V stage is free once the P V product of its unit is done.
__device__ void v_loader(const AttnParams& p, AttnCtl* ctl, uint8_t* sV, int64_t fb, int64_t fe) {
  const uint64_t pol = policy_evict_first();
  int stage = 0, phase = 0;
  int last_ph[kStages];
  for (int i = 0; i < kStages; ++i) last_ph[i] = -1;
  UnitIter c;
  for (c.init(p, fb, fe); c.valid(); c.next(p)) {
    if (ctl->abort) break;
    if (!mbar_wait(&ctl->v_empty[stage], phase ^ 1, p.wait_ns)) { fail(ctl, p.err); break; }
    mbar_arrive_expect_tx(&ctl->v_full[stage], kUnitBytes);
    const int zk = (p.layer0 + c.l) * p.G + c.g, y = c.j * kAttnUnitKeys;
    for (int h = 0; h < 2; ++h)
      tma_load_3d_hint(sV + stage * kUnitBytes + h * kHalfBytes, &p.tmv[c.s], &ctl->v_full[stage], h * 64, y, zk, pol);
    last_ph[stage] = phase;
    if (++stage == p.kv_stages) {
      stage = 0;
      phase ^= 1;
    }
  }
  if (ctl->abort)
    for (int i = 0; i < kStages; ++i)
      if (last_ph[i] >= 0) mbar_wait(&ctl->v_full[i], last_ph[i], drain_limit(p.wait_ns));
}

// Two MMA issuers walk the same units: warp 1 issues S(u) into S stage u & 1
// as soon as the stage is free and K(u) has landed, warp 2 issues
// O += P(u) V(u) once the softmax has written P(u) and V(u) is fp16, so that
// S of the next units runs ahead of the products.
__device__ void mma_s_loop(const AttnParams& p, AttnCtl* ctl, const uint8_t* sQ, const uint8_t* sK, uint32_t tmem,
                           int64_t fb, int64_t fe) {
  const uint32_t idesc_s = idesc_bf16(128, kAttnUnitKeys);
  const uint64_t dq0 = sdesc_k_sw128(smem_u32(sQ));
  const uint32_t qhalf16 = (p.q_rows * 128) >> 4;
  int stage = 0, kphase = 0, pc = 0;
  int64_t ui = 0;
  UnitIter c;
  for (c.init(p, fb, fe); c.valid(); c.next(p), ++ui) {
    if (ctl->abort) break;
    if (c.first(fb)) {
      if (!mbar_wait(&ctl->q_full, pc & 1, p.wait_ns)) { fail(ctl, p.err); break; }
      ++pc;
    }
    const int t = static_cast<int>(ui & 1);
    if (!mbar_wait(&ctl->k_full[stage], kphase, p.wait_ns)) { fail(ctl, p.err); break; }
    if (!mbar_wait(&ctl->s_empty[t], static_cast<uint32_t>(((ui >> 1) & 1) ^ 1), p.wait_ns)) { fail(ctl, p.err); break; }
    tc_fence_after();
    const uint64_t dk = sdesc_k_sw128(smem_u32(sK + stage * kUnitBytes));
#pragma unroll
    for (int mt = 0; mt < 2; ++mt) {
      if (mt >= p.n_mtiles) break;
      // M tile 1 reads rows 128..255 of each Q half; rows past q_rows feed
      // accumulator rows that no thread reads
      const uint64_t dq = dq0 + static_cast<uint64_t>(mt * ((128 * 128) >> 4));
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        const uint32_t koff16 = (kk >> 2) * (kHalfBytes >> 4) + (kk & 3) * 2;
        const uint32_t qoff16 = (kk >> 2) * qhalf16 + (kk & 3) * 2;
        mma_bf16(tmem + 256 + t * 128 + mt * kAttnUnitKeys, dq + qoff16, dk + koff16, idesc_s, kk > 0);
      }
      mma_commit(&ctl->s_full[t][mt]);   // that M tile's softmax starts without waiting for the next
    }
    mma_commit(&ctl->k_empty[stage]);
    if (c.last()) mma_commit(&ctl->q_empty);
    if (++stage == p.kv_stages) {
      stage = 0;
      kphase ^= 1;
    }
  }
  // every MMA issued above must be complete before TMEM is released
  mma_commit(&ctl->drain);
  mbar_wait(&ctl->drain, 0, drain_limit(p.wait_ns));
}

__device__ void mma_pv_loop(const AttnParams& p, AttnCtl* ctl, const uint8_t* sV, uint32_t tmem, int64_t fb,
                            int64_t fe) {
  const uint32_t idesc_o = idesc_f16_bmn(128, kHeadDim);
  int stage = 0, kphase = 0;
  int64_t ui = 0;
  UnitIter c;
  for (c.init(p, fb, fe); c.valid(); c.next(p), ++ui) {
    if (ctl->abort) break;
    const int t = static_cast<int>(ui & 1);
    if (!mbar_wait(&ctl->v_ready[stage], kphase, p.wait_ns)) { fail(ctl, p.err); break; }
    const bool first = c.first(fb);   // the piece's first product overwrites O
    const uint64_t dv = sdesc_mn_sw128(smem_u32(sV + stage * kUnitBytes), kHalfBytes, 1024);
    bool ok = true;
#pragma unroll
    for (int mt = 0; mt < 2; ++mt) {
      if (mt >= p.n_mtiles) break;
      // each M tile's product as soon as its P is written
      if (!mbar_wait(&ctl->p_full[t][mt], static_cast<uint32_t>((ui >> 1) & 1), p.wait_ns)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t ap = tmem + 256 + t * 128 + mt * kAttnUnitKeys;   // P of M tile mt over its S columns
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)   // 16 keys per step: +8 columns of P, +16 rows of V
        mma_f16_ts(tmem + mt * kHeadDim, ap + kk * 8, dv + static_cast<uint64_t>(kk * 128), idesc_o,
                   (!first || kk > 0) ? 1u : 0u);
    }
    if (!ok) {
      fail(ctl, p.err);
      break;
    }
    mma_commit(&ctl->v_empty[stage]);
    mma_commit(&ctl->s_empty[t]);   // S stage t (holding P) is free for S two units later
    if (++stage == p.kv_stages) {
      stage = 0;
      kphase ^= 1;
    }
  }
  mma_commit(&ctl->drain);
  mbar_wait(&ctl->drain, 0, drain_limit(p.wait_ns));
}

// Maximum raw logit of a thread's row over the unit's first `lim` keys.
__device__ __forceinline__ float unit_max(const uint32_t (&z)[4][16], int lim) {
  float pm[8];   // eight independent partial maxima (short dependency chains)
#pragma unroll
  for (int k = 0; k < 8; ++k) pm[k] = -INFINITY;
#pragma unroll
  for (int q = 0; q < 4; ++q)
#pragma unroll
    for (int i = 0; i < 16; ++i)
      if (q * 16 + i < lim) pm[i & 7] = fmaxf(pm[i & 7], __uint_as_float(z[q][i]));
  return fmaxf(fmaxf(fmaxf(pm[0], pm[1]), fmaxf(pm[2], pm[3])), fmaxf(fmaxf(pm[4], pm[5]), fmaxf(pm[6], pm[7])));
}

// exp2 and pack of one 16-key chunk (keys k0 .. k0 + 15)
__device__ __forceinline__ void exp_pack_chunk(const uint32_t (&z)[16], int k0, int lim, bool live, float2 sc2,
                                               float2 nm2, float2 (&acc)[4], uint32_t (&h)[8]) {
#pragma unroll
  for (int i = 0; i < 16; i += 2) {
    const float2 e = ffma2(make_float2(__uint_as_float(z[i]), __uint_as_float(z[i + 1])), sc2, nm2);
    const int k = k0 + i;
    const float p0 = (live && k < lim) ? ex2_approx(e.x) : 0.f;
    const float p1 = (live && k + 1 < lim) ? ex2_approx(e.y) : 0.f;
    acc[(i >> 1) & 3] = fadd2(acc[(i >> 1) & 3], make_float2(p0, p1));
    h[i >> 1] = pack_half2(p0, p1);
  }
}

// p = exp2(z c2 - m) of the unit's 64 keys (0 past `lim` and in a row that
// is not live) as fp16 pairs h[q][j] = (p[16 q + 2 j], p[16 q + 2 j + 1]), the
// lower key in the low half; returns the sum of the p.
__device__ __forceinline__ float exp_pack_p(const uint32_t (&z)[4][16], int lim, bool live, float c2, float m,
                                            uint32_t (&h)[4][8]) {
  const float2 sc2 = make_float2(c2, c2), nm2 = make_float2(-m, -m);
  float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                   make_float2(0.f, 0.f)};   // four independent running sums
#pragma unroll
  for (int q = 0; q < 4; ++q) exp_pack_chunk(z[q], 16 * q, lim, live, sc2, nm2, acc, h[q]);
  const float2 a01 = fadd2(acc[0], acc[1]), a23 = fadd2(acc[2], acc[3]);
  const float2 a = fadd2(a01, a23);
  return a.x + a.y;
}

// exp_pack_p reading S itself from `scol` in two halves, the second half's
// loads in flight under the first half's arithmetic (measured faster than
// waiting for all four loads first, and than one 16-column load ahead)
__device__ __forceinline__ float exp_pack_p_streamed(uint32_t scol, int lim, bool live, float c2, float m,
                                                     uint32_t (&h)[4][8]) {
  const float2 sc2 = make_float2(c2, c2), nm2 = make_float2(-m, -m);
  float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                   make_float2(0.f, 0.f)};   // four independent running sums
  uint32_t a0[16], a1[16], b0[16], b1[16];
  tmem_ld16_async(scol, a0);
  tmem_ld16_async(scol + 16, a1);
  tmem_wait16(a0);
  tmem_wait16(a1);
  tmem_ld16_async(scol + 32, b0);
  tmem_ld16_async(scol + 48, b1);
  exp_pack_chunk(a0, 0, lim, live, sc2, nm2, acc, h[0]);
  exp_pack_chunk(a1, 16, lim, live, sc2, nm2, acc, h[1]);
  tmem_wait16(b0);
  tmem_wait16(b1);
  exp_pack_chunk(b0, 32, lim, live, sc2, nm2, acc, h[2]);
  exp_pack_chunk(b1, 48, lim, live, sc2, nm2, acc, h[3]);
  const float2 a01 = fadd2(acc[0], acc[1]), a23 = fadd2(acc[2], acc[3]);
  const float2 a = fadd2(a01, a23);
  return a.x + a.y;
}

// The unit's 64 S columns of this warp's lanes from `scol`, waited for.
__device__ __forceinline__ void load_s(uint32_t scol, uint32_t (&z)[4][16]) {
#pragma unroll
  for (int q = 0; q < 4; ++q) tmem_ld16_async(scol + q * 16, z[q]);
#pragma unroll
  for (int q = 0; q < 4; ++q) tmem_wait16(z[q]);
}

// Rescales this warp's O rows by alpha (1 in lanes whose reference stays).
__device__ __forceinline__ void rescale_o(uint32_t o_addr, float alpha) {
#pragma unroll 1
  for (int ch = 0; ch < kHeadDim / 16; ++ch) {
    uint32_t o[16];
    tmem_ld16_async(o_addr + ch * 16, o);
    tmem_wait16(o);
#pragma unroll
    for (int i = 0; i < 16; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
    tmem_st16(o_addr + ch * 16, o);
  }
}

// One unit of a softmax warp (warp-uniform `wactive`; TMEM loads and stores
// are warp-collective): S at `scol` becomes P over its first 32 columns, and
// the reference m and sum l of the thread's row advance.  `fresh`: the
// piece's first unit, whose maximum sets the reference.  P is computed with
// the current reference; every p is below 2^15 unless the unit's sum exceeds
// it, and only then is the maximum taken (S is still in place, P is stored
// last): lanes where it lies more than 15 above the reference move it and
// rescale their O rows (at o_addr, once the product of the previous unit,
// phase `prev_par` of `prev_bar`, is done), and P is redone.  Returns false
// when that wait ran out.
__device__ __forceinline__ bool softmax_unit(const AttnParams& p, bool wactive, bool live, bool fresh, int lim,
                                             uint32_t scol, uint32_t o_addr, uint64_t* prev_bar, uint32_t prev_par,
                                             float& m, float& l) {
  const float c2 = p.scale2;
  if (fresh) l = 0.f;
  if (!wactive) {
    if (fresh) m = 0.f;   // a warp without rows keeps a finite reference
    return true;
  }
  uint32_t z[4][16];
  uint32_t h[4][8];
  float us;
  if (fresh) {
    load_s(scol, z);
    m = unit_max(z, lim) * c2;
    us = exp_pack_p(z, lim, live, c2, m, h);
  } else {
    us = exp_pack_p_streamed(scol, lim, live, c2, m, h);
  }
  if (__any_sync(kFull, live && us > 32768.f)) {   // rare
    load_s(scol, z);   // z again, so that it need not live across the first pass
    const float mx = unit_max(z, lim) * c2;
    const bool move = live && mx > m + kMoveThreshold;
    if (__any_sync(kFull, move)) {
      const float alpha = move ? ex2_approx(m - mx) : 1.f;
      if (move) m = mx;
      if (!__all_sync(kFull, mbar_wait(prev_bar, prev_par, p.wait_ns))) return false;
      tc_fence_after();
      rescale_o(o_addr, alpha);
      l *= alpha;
    }
    // P again in every lane (the same values where the reference stayed), so
    // that the first h need not live across the reload either
    us = exp_pack_p(z, lim, live, c2, m, h);
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) tmem_st8(scol + q * 8, h[q]);   // keys 16 q ..: columns 8 q ..
  l += us;
  return true;
}

constexpr int kSStages = 2;   // S stages in tensor memory

// Softmax warps: one thread per window row of M tile `mt` (TMEM lane
// quad * 32 + lane).  Unit u sits in S stage u mod kSStages; the S (then P)
// columns of stage t start at s_col0 + t s_stride and O at o_col.  A piece's
// partial goes to slot row + slot0.

__device__ void softmax_loop(const AttnParams& p, AttnCtl* ctl, uint32_t tmem, int mt, int quad, int lane,
                             uint32_t s_col0, uint32_t s_stride, uint32_t o_col, int slot0, int64_t fb, int64_t fe) {
  const int rho = quad * 32 + lane;   // row within the M tile (TMEM lane)
  const int r = mt * 128 + rho;       // window row within the group
  if (mt >= p.n_mtiles) return;   // no S is computed for this M tile, no P awaited from it
  const bool wactive = mt * 128 + quad * 32 < p.rows;
  const bool live = r < p.rows;
  const uint32_t lane_base = tmem + (static_cast<uint32_t>(quad * 32) << 16);
  float m = -INFINITY, l = 0.f;
  uint32_t ui = 0;
  UnitIter c;
  for (c.init(p, fb, fe); c.valid(); c.next(p), ++ui) {
    if (ctl->abort) break;
    const bool first = c.first(fb), last = c.last();
    const int t = static_cast<int>(ui % kSStages);
    const uint32_t par = (ui / kSStages) & 1u;
    const uint32_t scol = s_col0 + t * s_stride;   // this unit's S, then P, columns
    if (!__all_sync(kFull, mbar_wait(&ctl->s_full[t][mt], par, p.wait_ns))) {
      fail(ctl, p.err);
      break;
    }
    tc_fence_after();
    const int lim = p.seq[c.s].Lp - c.j * kAttnUnitKeys;   // valid keys of the unit (>= 1)
    const uint32_t up = ui - 1;   // the previous unit (a piece's first unit never moves)
    if (!softmax_unit(p, wactive, live, first, lim, lane_base + scol, lane_base + o_col,
                      &ctl->s_empty[up % kSStages], (up / kSStages) & 1u, m, l)) {
      fail(ctl, p.err);
      break;
    }
    tmem_wait_st();
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(&ctl->p_full[t][mt]);
    if (last) {
      // the piece's partial: (m, l) and the unnormalised O rows, once the
      // product of this last unit is done
      if (!__all_sync(kFull, mbar_wait(&ctl->s_empty[t], par, p.wait_ns))) {
        fail(ctl, p.err);
        break;
      }
      tc_fence_after();
      const int64_t slot = static_cast<int64_t>(c.row(p)) + slot0;
      if (wactive) {
        float* dst = p.part_o + (slot * kMaxRows + r) * kHeadDim;
#pragma unroll 1
        for (int ch = 0; ch < kHeadDim / 16; ++ch) {
          uint32_t o[16];
          tmem_ld16_async(lane_base + o_col + ch * 16, o);
          tmem_wait16(o);
          if (live)
#pragma unroll
            for (int i = 0; i < 16; i += 4)
              *reinterpret_cast<float4*>(dst + ch * 16 + i) =
                  make_float4(__uint_as_float(o[i]), __uint_as_float(o[i + 1]), __uint_as_float(o[i + 2]),
                              __uint_as_float(o[i + 3]));
        }
        if (live) p.part_ml[slot * kMaxRows + r] = make_float2(m, l);
      }
      tc_fence_before();
    }
  }
}

// V conversion warps (NW of them, thread ct of 32 NW): V of every unit to
// fp16 in place, then released to the P V product.
template <int NW>
__device__ void convert_loop(const AttnParams& p, AttnCtl* ctl, uint8_t* sV, int kv_stages, int ct, int lane, int64_t fb,
                             int64_t fe) {
  int stage = 0, phase = 0;
  for (int64_t f = fb; f < fe; ++f) {
    if (ctl->abort) break;
    if (!__all_sync(kFull, mbar_wait(&ctl->v_full[stage], phase, p.wait_ns))) {
      fail(ctl, p.err);
      break;
    }
    uint4* v4 = reinterpret_cast<uint4*>(sV + stage * kUnitBytes);
#pragma unroll
    for (int i = 0; i < kUnitBytes / 16 / (32 * NW); ++i) {
      uint4 x = v4[ct + i * 32 * NW];
      x.x = bf16x2_to_f16x2(x.x);
      x.y = bf16x2_to_f16x2(x.y);
      x.z = bf16x2_to_f16x2(x.z);
      x.w = bf16x2_to_f16x2(x.w);
      v4[ct + i * 32 * NW] = x;
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) mbar_arrive(&ctl->v_ready[stage]);
    if (++stage == kv_stages) {
      stage = 0;
      phase ^= 1;
    }
  }
}

}  // namespace

__global__ void __launch_bounds__(kAttnThreads, 1) k_window_attn(const __grid_constant__ AttnParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;                              // [2 halves][q_rows][128 B]
  uint8_t* sK = sQ + 2 * p.q_rows * 128;           // [kv_stages][2 halves][64 keys][128 B]
  uint8_t* sV = sK + p.kv_stages * kUnitBytes;     // [kv_stages][2 halves][64 keys][128 B]
  AttnCtl* ctl = reinterpret_cast<AttnCtl*>(sV + p.kv_stages * kUnitBytes);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&ctl->k_full[i], 1);
      mbar_init(&ctl->k_empty[i], 1);
      mbar_init(&ctl->v_full[i], 1);
      mbar_init(&ctl->v_empty[i], 1);
      mbar_init(&ctl->v_ready[i], kConvWarps);
    }
    for (int i = 0; i < 2; ++i) {
      for (int m = 0; m < 2; ++m) {
        mbar_init(&ctl->s_full[i][m], 1);
        mbar_init(&ctl->p_full[i][m], kSoftWarps / 2);   // the four warps of the M tile
      }
      mbar_init(&ctl->s_empty[i], 1);   // the P V issuer's commit
    }
    mbar_init(&ctl->q_full, 1);
    mbar_init(&ctl->q_empty, 1);
    mbar_init(&ctl->drain, 2);   // one commit per MMA issuer
    ctl->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&ctl->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  griddep_launch_dependents();
  griddep_wait();
  const uint32_t tmem = ctl->tmem_base;
  const int64_t T = p.total_units;
  const int64_t fb = range_begin(T, blockIdx.x, gridDim.x);
  const int64_t fe = range_begin(T, blockIdx.x + 1, gridDim.x);

  if (warp == 0) {
    if (lane == 0) k_loader(p, ctl, sQ, sK, fb, fe);
  } else if (warp == 3) {
    if (lane == 0) v_loader(p, ctl, sV, fb, fe);
  } else if (warp == 1) {
    if (lane == 0) mma_s_loop(p, ctl, sQ, sK, tmem, fb, fe);
  } else if (warp == 2) {
    if (lane == 0) mma_pv_loop(p, ctl, sV, tmem, fb, fe);
  } else if (warp >= kSoftWarp0 && warp < kSoftWarp0 + kSoftWarps) {
    const int mt = (warp - kSoftWarp0) >> 2;
    softmax_loop(p, ctl, tmem, mt, warp & 3, lane, 256 + mt * kAttnUnitKeys, 128, mt * kHeadDim, blockIdx.x, fb, fe);
  } else if (warp >= kConvWarp0) {
    convert_loop<kConvWarps>(p, ctl, sV, p.kv_stages, threadIdx.x - 32 * kConvWarp0, lane, fb, fe);
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// Merges the pieces of each (seq, layer, group) row: M = max m, L = sum
// 2^(m - M) l, O = sum 2^(m - M) O_piece / L, lse = (M + log2 L) ln 2.
// grid: (rows of the launch, ceil(window rows / 8)); one warp per window row,
// four output columns per lane, every piece's loads issued before the sums.
// Four pieces per batch of loads and six 256-thread blocks per SM (at most 40
// registers): more rows' loads in flight than eight pieces at three blocks.
constexpr int kMaxPieces = 4;   // pieces merged per batch of loads
__global__ void __launch_bounds__(256, 6) k_attn_combine(const __grid_constant__ AttnParams p) {
  griddep_launch_dependents();
  griddep_wait();
  const int R = blockIdx.x;
  const int per_seq = p.nlayers * p.G;
  const int s = R / per_seq, rem = R - s * per_seq, l = rem / p.G, g = rem - l * p.G;
  const AttnSeq& sq = p.seq[s];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.y * 8 + warp;
  if (r >= p.rows) return;
  const int64_t row0 = (static_cast<int64_t>(p.layer0 + l) * p.G + g) * p.rows;   // flat (h, i) row of r = 0
  int c0 = 0, c1 = -1;
  if (sq.nu > 0) {
    const int64_t f0 = sq.unit_base + static_cast<int64_t>(l * p.G + g) * sq.nu;
    c0 = cta_of(f0, p.total_units, p.grid);
    c1 = cta_of(f0 + sq.nu - 1, p.total_units, p.grid);
  }
  float M = -INFINITY, L = 0.f;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int cb = c0; cb <= c1; cb += kMaxPieces) {
    float2 ml[kMaxPieces];
    float4 o[kMaxPieces];
#pragma unroll
    for (int k = 0; k < kMaxPieces; ++k) {
      if (cb + k > c1) break;
      const int64_t slot = static_cast<int64_t>(R) + cb + k;
      ml[k] = p.part_ml[slot * kMaxRows + r];
      o[k] = reinterpret_cast<const float4*>(p.part_o + (slot * kMaxRows + r) * kHeadDim)[lane];
    }
    float bm = M;
#pragma unroll
    for (int k = 0; k < kMaxPieces; ++k)
      if (cb + k <= c1) bm = fmaxf(bm, ml[k].x);
    const float keep = M == -INFINITY ? 0.f : exp2f(M - bm);
    L *= keep;
    acc.x *= keep;
    acc.y *= keep;
    acc.z *= keep;
    acc.w *= keep;
#pragma unroll
    for (int k = 0; k < kMaxPieces; ++k) {
      if (cb + k > c1) break;
      const float wgt = exp2f(ml[k].x - bm);
      L += wgt * ml[k].y;
      acc.x += wgt * o[k].x;
      acc.y += wgt * o[k].y;
      acc.z += wgt * o[k].z;
      acc.w += wgt * o[k].w;
    }
    M = bm;
  }
  const float inv = L > 0.f ? 1.f / L : 0.f;
  if (sq.o)
    reinterpret_cast<float4*>(sq.o + (row0 + r) * kHeadDim)[lane] =
        make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
  if (lane == 0) sq.lse[row0 + r] = L > 0.f ? (M + log2f(L)) * 0.6931471805599453f : -INFINITY;
}

size_t attn_smem_bytes(int q_rows, int kv_stages) {
  return 1024 + static_cast<size_t>(2 * q_rows * 128) + 2 * static_cast<size_t>(kv_stages) * kUnitBytes + kCtlBytes;
}

int attn_kv_stages(int q_rows) {
  int k = kStages;
  while (k > 2 && attn_smem_bytes(q_rows, k) > kSmemLimit) --k;
  return k;
}

cudaError_t attn_configure() {
  return cudaFuncSetAttribute(k_window_attn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(kSmemLimit));
}

namespace {

cudaLaunchConfig_t pdl_config(cudaLaunchAttribute* attr, dim3 grid, dim3 block, size_t smem, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // set-up under the previous kernel's tail
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.stream = stream;
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  return cfg;
}

}  // namespace

cudaError_t attn_main_launch(const AttnParams& p, cudaStream_t stream) {
  if (p.total_units <= 0) return cudaSuccess;
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = pdl_config(attr, dim3(p.grid), dim3(kAttnThreads), attn_smem_bytes(p.q_rows, p.kv_stages), stream);
  return cudaLaunchKernelEx(&cfg, k_window_attn, p);
}

cudaError_t attn_combine_launch(const AttnParams& p, cudaStream_t stream) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = pdl_config(attr, dim3(p.nseq * p.nlayers * p.G, (p.rows + 7) / 8), dim3(256), 0, stream);
  return cudaLaunchKernelEx(&cfg, k_attn_combine, p);
}

}  // namespace starkv
