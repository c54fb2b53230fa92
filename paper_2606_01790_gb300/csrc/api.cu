// C ABI of the STaR-KV compression stage (include/starkv.h): argument
// validation, device state, workspace planning, TMA descriptors and launch
// sequencing.  All arithmetic of the method runs in the kernels of score.cu,
// select.cu and compact.cu.
#include <cudaTypedefs.h>
#include <nvtx3/nvToolsExt.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "attn.cuh"
#include "common.cuh"
#include "compact.cuh"
#include "score.cuh"
#include "select.cuh"

using namespace starkv;

struct starkv_state {
  starkv_config cfg;
  DevState dev;
  void* mem = nullptr;
  size_t mem_bytes = 0;
  int device = 0;
  int num_sms = 0;
  uint64_t wait_ns = 1000000000ull;
  // kernel timing (starkv_set_timing / starkv_kernel_times)
  bool timing = false;
  int64_t launches[STARKV_NUM_KERNELS] = {};
  struct Rec {
    int kind;
    cudaEvent_t a, b;
  };
  std::vector<Rec> recs;
  std::vector<cudaEvent_t> pool;
  // starkv_step_host: copy-in / copy-out streams and their ordering events
  cudaStream_t pipe_in = nullptr, pipe_out = nullptr;
  std::vector<cudaEvent_t> pipe_ev;
  // starkv_score_layer_noalloc: device address of the static scratch on this
  // state's device (looked up at init), or NULL with the reason kept
  void* noalloc_scratch = nullptr;
  std::string noalloc_error;
};

namespace {

thread_local std::string g_last_error;

starkv_status set_error(starkv_status s, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
starkv_status set_error(starkv_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

#define CUDA_TRY(expr)                                                                        \
  do {                                                                                        \
    cudaError_t e_ = (expr);                                                                  \
    if (e_ != cudaSuccess)                                                                    \
      return set_error(STARKV_ERR_CUDA, "%s failed: %s", #expr, cudaGetErrorString(e_));      \
  } while (0)

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;
cudaError_t g_encode_err = cudaSuccess;

starkv_status get_encoder() {
  std::call_once(g_encode_once, [] {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    g_encode_err = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                    cudaEnableDefault, &q);
    if (g_encode_err == cudaSuccess && q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  if (!g_encode)
    return set_error(STARKV_ERR_CUDA, "cuTensorMapEncodeTiled unavailable (%s)",
                     cudaGetErrorString(g_encode_err));
  return STARKV_OK;
}

// 3-D bf16 tensor map, 128-byte swizzle, box (64, box_rows, 1), zero fill out of bounds.
starkv_status encode_3d(CUtensorMap* map, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
                        uint32_t box_rows) {
  cuuint64_t dims[3] = {d0, d1, d2};
  cuuint64_t strides[2] = {d0 * 2, d0 * d1 * 2};
  cuuint32_t box[3] = {64, box_rows, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                        box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return set_error(STARKV_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
  return STARKV_OK;
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

cudaEvent_t take_event(starkv_state* st) {
  if (!st->pool.empty()) {
    cudaEvent_t e = st->pool.back();
    st->pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

// Launches one kernel kind through `fn`, counting it and, when timing is on,
// bracketing it with an event pair on `stream`.
// NVTX ranges name each host-side enqueue for a profiler's timeline (no cost
// unless a tool is attached; NVTX v3 is header-only).
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

const char* kernel_range_name(int kind) {
  switch (kind) {
    case STARKV_KERNEL_SCORE_LSE: return "starkv: scoring pass 1 (row LSE)";
    case STARKV_KERNEL_SCORE_ACCUM: return "starkv: scoring pass 2 (group sums)";
    case STARKV_KERNEL_POOL: return "starkv: pooling";
    case STARKV_KERNEL_CALIBRATE: return "starkv: calibration + top-B";
    case STARKV_KERNEL_COMPACT: return "starkv: compaction";
    case STARKV_KERNEL_ATTENTION: return "starkv: window attention (pieces)";
    case STARKV_KERNEL_ATTN_COMBINE: return "starkv: window attention (combine)";
    default: return "starkv: kernel";
  }
}

template <typename F>
cudaError_t launch(starkv_state* st, int kind, cudaStream_t stream, F&& fn) {
  NvtxRange range(kernel_range_name(kind));
  st->launches[kind] += 1;
  if (!st->timing) return fn();
  starkv_state::Rec r{kind, take_event(st), take_event(st)};
  cudaError_t e = cudaEventRecord(r.a, stream);
  if (e != cudaSuccess) return e;
  e = fn();
  if (e != cudaSuccess) return e;
  e = cudaEventRecord(r.b, stream);
  st->recs.push_back(r);
  return e;
}

// Scratch of starkv_score_layer_noalloc, the scoring call for callers that
// cannot allocate device memory: one static device array that every call on a
// device shares.  Host code may not hand the symbol itself to a kernel (on the
// host it names a stand-in, not device memory): starkv_init_state looks up its
// device address with the state's device current.
constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;   // 16 MiB per device
__device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

starkv_status validate_config(const starkv_config& c) {
  if (c.n_layers < 1 || c.n_heads < 1 || c.n_kv_heads < 1 || c.window < 1 || c.max_seqs < 1)
    return set_error(STARKV_ERR_INVALID_ARG, "config: n_layers, n_heads, n_kv_heads, window, max_seqs must be >= 1");
  if (c.head_dim != kHeadDim) return set_error(STARKV_ERR_UNSUPPORTED, "config: head_dim must be 128");
  if (c.n_heads % c.n_kv_heads) return set_error(STARKV_ERR_UNSUPPORTED, "config: n_heads %% n_kv_heads != 0");
  if (c.n_kv_heads > kMaxGroups) return set_error(STARKV_ERR_UNSUPPORTED, "config: n_kv_heads > 32");
  if ((c.n_heads / c.n_kv_heads) * c.window > kMaxRows)
    return set_error(STARKV_ERR_UNSUPPORTED, "config: (H/G)*w > 256");
  if (c.grid_rows < 1 || c.grid_cols < 1 || c.grid_rows > 1024 || c.grid_cols > 1024 ||
      c.grid_rows * c.grid_cols > kMaxGrid)
    return set_error(STARKV_ERR_UNSUPPORTED, "config: patch grid out of range");
  if (c.pool_kernel < 1 || c.pool_kernel > 31 || c.pool_kernel % 2 == 0)
    return set_error(STARKV_ERR_UNSUPPORTED, "config: pool_kernel must be odd, 1..31");
  if (c.mi_bins < 2 || c.mi_bins > 16 || c.mi_grid < 1 || c.mi_bins * c.mi_grid * c.mi_grid > kMaxHist)
    return set_error(STARKV_ERR_UNSUPPORTED, "config: mi_bins / mi_grid out of range");
  if (c.n_warmup < 0 || c.n_ramp < 0) return set_error(STARKV_ERR_INVALID_ARG, "config: negative schedule");
  if (!(c.t_min > 0.f) || !(c.t_max > 0.f) || !(c.tau > 0.f))
    return set_error(STARKV_ERR_INVALID_ARG, "config: t_min, t_max and tau must be > 0");
  if (c.decay_mode < 0 || c.decay_mode > 2 || c.aeb_mode < 0 || c.aeb_mode > 1 || c.mi_span < 0 || c.mi_span > 1)
    return set_error(STARKV_ERR_INVALID_ARG, "config: decay_mode in 0..2, aeb_mode and mi_span in 0..1");
  if (c.select_mode != STARKV_SELECT_GLOBAL && c.select_mode != STARKV_SELECT_PER_HEAD)
    return set_error(STARKV_ERR_INVALID_ARG, "config: select_mode must be 0 (global) or 1 (per KV head)");
  if (c.select_mode == STARKV_SELECT_PER_HEAD && c.n_kv_heads > kMaxCluster)
    return set_error(STARKV_ERR_UNSUPPORTED, "config: the per-KV-head mode takes n_kv_heads <= 8");
  if (!(c.rho_mi >= 0.f && c.rho_mi <= 1.f) || !(c.rho_t >= 0.f && c.rho_t <= 1.f) ||
      !(c.d_min >= 0.f && c.d_min <= 1.f) || !(c.eps >= 0.f) || !(c.eps_h >= 0.f) || !(c.delta >= 0.f))
    return set_error(STARKV_ERR_INVALID_ARG, "config: a rate or epsilon is out of range");
  return STARKV_OK;
}

enum Need : unsigned {
  kNeedK = 1, kNeedQ = 2, kNeedV = 4, kNeedMeta = 8, kNeedS = 16, kNeedIdx = 32, kNeedOut = 64
};

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }
bool aligned4(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 3) == 0; }

starkv_status validate_seqs(const starkv_state* st, const starkv_seq* seqs, int nseq, unsigned need) {
  if (!st) return set_error(STARKV_ERR_INVALID_ARG, "state is NULL");
  if (nseq < 0 || (nseq > 0 && !seqs)) return set_error(STARKV_ERR_INVALID_ARG, "bad sequence array");
  const starkv_config& c = st->cfg;
  std::vector<char> used(c.max_seqs, 0);
  for (int i = 0; i < nseq; ++i) {
    const starkv_seq& s = seqs[i];
    if (s.slot < 0 || s.slot >= c.max_seqs) return set_error(STARKV_ERR_INVALID_ARG, "seq %d: slot out of range", i);
    if (used[s.slot]) return set_error(STARKV_ERR_INVALID_ARG, "seq %d: slot %d used twice in one call", i, s.slot);
    used[s.slot] = 1;
    if (s.L < c.window) return set_error(STARKV_ERR_INVALID_ARG, "seq %d: L < window", i);
    if (s.L >= (1 << 24)) return set_error(STARKV_ERR_UNSUPPORTED, "seq %d: L >= 2^24", i);
    const int lp = s.L - c.window;
    if (s.budget < 0 || s.budget > lp) return set_error(STARKV_ERR_INVALID_ARG, "seq %d: budget outside [0, L - w]", i);
    if (s.cur_frame < 0 || s.cur_frame > 2047) return set_error(STARKV_ERR_INVALID_ARG, "seq %d: cur_frame outside [0, 2047]", i);
    if ((need & kNeedK) && (!s.k || !aligned16(s.k))) return set_error(STARKV_ERR_INVALID_ARG, "seq %d: k NULL or not 16-byte aligned", i);
    if ((need & kNeedQ) && (!s.q || !aligned16(s.q))) return set_error(STARKV_ERR_INVALID_ARG, "seq %d: q NULL or not 16-byte aligned", i);
    if ((need & kNeedV) && (!s.v || !aligned16(s.v))) return set_error(STARKV_ERR_INVALID_ARG, "seq %d: v NULL or not 16-byte aligned", i);
    if (need & kNeedMeta) {
      if (!s.meta) return set_error(STARKV_ERR_INVALID_ARG, "seq %d: meta is NULL", i);
      if (s.meta_group_stride != 0) {
        if (c.select_mode != STARKV_SELECT_PER_HEAD)
          return set_error(STARKV_ERR_INVALID_ARG, "seq %d: meta_group_stride must be 0 in the global selection mode", i);
        if (s.meta_group_stride < s.L)
          return set_error(STARKV_ERR_INVALID_ARG, "seq %d: meta_group_stride must be 0 or >= L", i);
      }
      const int64_t span = static_cast<int64_t>(c.n_kv_heads - 1) * s.meta_group_stride + s.L;
      if (s.meta_layer_stride != 0 && s.meta_layer_stride < span)
        return set_error(STARKV_ERR_INVALID_ARG, "seq %d: meta_layer_stride must be 0 or >= (G-1)*meta_group_stride + L", i);
    }
    // 4-byte words: a misaligned pointer is an argument error, not a device fault
    const void* words[] = {s.meta, s.meta_out, s.idx, s.S, s.score, s.stats, s.lse, s.attn_lse};
    for (const void* w : words)
      if (w && !aligned4(w)) return set_error(STARKV_ERR_INVALID_ARG, "seq %d: a 4-byte array is not 4-byte aligned", i);
    if (s.attn_o && !aligned16(s.attn_o)) return set_error(STARKV_ERR_INVALID_ARG, "seq %d: attn_o not 16-byte aligned", i);
    if ((need & kNeedS) && !s.S && lp > 0) return set_error(STARKV_ERR_INVALID_ARG, "seq %d: S is NULL", i);
    if ((need & kNeedIdx) && !s.idx && s.budget > 0) return set_error(STARKV_ERR_INVALID_ARG, "seq %d: idx is NULL", i);
    if (need & kNeedOut) {
      if (!s.k_out || !s.v_out || !s.meta_out || !aligned16(s.k_out) || !aligned16(s.v_out))
        return set_error(STARKV_ERR_INVALID_ARG, "seq %d: k_out / v_out / meta_out NULL or misaligned", i);
    }
  }
  return STARKV_OK;
}

KParams make_kparams(const starkv_state* st) {
  const starkv_config& c = st->cfg;
  KParams k;
  k.n_layers = c.n_layers; k.H = c.n_heads; k.G = c.n_kv_heads; k.w = c.window;
  k.R = c.grid_rows; k.C = c.grid_cols; k.pool = c.pool_kernel; k.K = c.mi_bins; k.M = c.mi_grid;
  k.n_warmup = c.n_warmup; k.n_ramp = c.n_ramp;
  k.lambda = c.lambda; k.tau = c.tau; k.rho_mi = c.rho_mi; k.rho_t = c.rho_t; k.delta = c.delta;
  k.d_min = c.d_min; k.t_min = c.t_min; k.t_max = c.t_max; k.eps = c.eps; k.eps_h = c.eps_h;
  k.per_head = c.select_mode == STARKV_SELECT_PER_HEAD;
  k.decay_mode = c.decay_mode;
  k.aeb_mode = c.aeb_mode;
  k.mi_span = c.mi_span;
  k.wait_ns = st->wait_ns;
  return k;
}

// Workspace regions of one call over layers [layer0, layer0 + nlayers).
struct WsPlan {
  size_t partials = 0, s_raw = 0, total = 0;
  std::vector<size_t> raw_off, S_off, score_off, vis_off;  // per seq, SIZE_MAX = not in workspace
};

int tiles_of(int lp) { return (lp + kTileKeys - 1) / kTileKeys; }

// Rows of idx, score and meta_out per layer: 1 (global selection) or G (per KV head).
size_t sel_rows(const starkv_config& c) {
  return c.select_mode == STARKV_SELECT_PER_HEAD ? static_cast<size_t>(c.n_kv_heads) : 1;
}

size_t stats_bytes(const starkv_config& c) { return static_cast<size_t>(STARKV_STATS_STRIDE(c.n_kv_heads)) * 4; }

// ws_score: the calibration kernel runs (fused score region; key/cell region
// of the rows longer than its shared-memory capacity).
void plan_ws(const starkv_state* st, const starkv_seq* seqs, int nseq, int nlayers, bool ws_S,
             bool ws_score, WsPlan* p) {
  const starkv_config& c = st->cfg;
  const int G = c.n_kv_heads;
  const int cap = calibrate_capacity(c.mi_bins, c.mi_grid, c.grid_rows, c.grid_cols);
  size_t off = 0;
  size_t tiles = 0;
  for (int i = 0; i < nseq; ++i) tiles += static_cast<size_t>(nlayers) * G * tiles_of(seqs[i].L - c.window);
  p->partials = off;
  off += align256(tiles * kMaxRows * sizeof(float2));
  p->raw_off.assign(nseq, SIZE_MAX);
  p->S_off.assign(nseq, SIZE_MAX);
  p->score_off.assign(nseq, SIZE_MAX);
  p->vis_off.assign(nseq, SIZE_MAX);
  for (int i = 0; i < nseq; ++i) {
    const size_t lp = seqs[i].L - c.window;
    if (ws_score && lp > static_cast<size_t>(cap)) {
      p->vis_off[i] = off;
      off += align256(static_cast<size_t>(nlayers) * G * lp * 3 * sizeof(uint32_t));
    }
    p->raw_off[i] = off;
    off += align256(static_cast<size_t>(nlayers) * G * kRawCopies * raw_stride(static_cast<int>(lp)) * sizeof(float));
    if (ws_S && !seqs[i].S) {
      p->S_off[i] = off;
      off += align256(static_cast<size_t>(c.n_layers) * G * lp * sizeof(float));
    }
    if (ws_score && !seqs[i].score) {
      p->score_off[i] = off;
      off += align256(static_cast<size_t>(c.n_layers) * sel_rows(c) * lp * sizeof(float));
    }
  }
  p->total = std::max<size_t>(off, 256);
}

SeqView make_view(const starkv_state* st, const starkv_seq& s, char* ws, const WsPlan& plan, int i) {
  const starkv_config& c = st->cfg;
  SeqView v;
  v.k = static_cast<const __nv_bfloat16*>(s.k);
  v.v = static_cast<const __nv_bfloat16*>(s.v);
  v.meta = s.meta;
  v.meta_layer_stride = s.meta_layer_stride;
  v.meta_group_stride = s.meta_group_stride;
  v.L = s.L;
  v.Lp = s.L - c.window;
  v.cur_frame = s.cur_frame;
  v.budget = s.budget;
  v.slot = s.slot;
  v.pad_ = 0;
  v.k_out = static_cast<__nv_bfloat16*>(s.k_out);
  v.v_out = static_cast<__nv_bfloat16*>(s.v_out);
  v.meta_out = s.meta_out;
  v.idx = s.idx;
  v.S = plan.S_off[i] != SIZE_MAX ? reinterpret_cast<float*>(ws + plan.S_off[i]) : s.S;
  v.s_raw = reinterpret_cast<float*>(ws + plan.raw_off[i]);
  v.score = plan.score_off[i] != SIZE_MAX ? reinterpret_cast<float*>(ws + plan.score_off[i]) : s.score;
  v.stats = s.stats;
  v.vis = plan.vis_off[i] != SIZE_MAX ? reinterpret_cast<uint32_t*>(ws + plan.vis_off[i]) : nullptr;
  return v;
}

// Both scoring passes for sequences [i0, i1) over layers [layer0, layer0 + nlayers).
starkv_status run_score(starkv_state* st, const starkv_seq* seqs, int i0, int i1, int layer0, int nlayers,
                        char* ws, const WsPlan& plan, size_t* partial_cursor, cudaStream_t stream) {
  const starkv_config& c = st->cfg;
  const int G = c.n_kv_heads, H = c.n_heads, w = c.window;
  starkv_status s = get_encoder();
  if (s != STARKV_OK) return s;
  static thread_local ScoreParams p;   // ~13 KB: kept off the stack
  memset(&p, 0, sizeof(p));
  p.nseq = i1 - i0;
  p.layer0 = layer0;
  p.nlayers = nlayers;
  p.G = G;
  p.rows = (H / G) * w;
  p.n2 = (p.rows + 15) & ~15;
  p.n_mtiles = (p.rows + kTileKeys - 1) / kTileKeys;
  p.q_rows = p.n2;
  p.kstages = score_kstages(p.q_rows);
  if (p.kstages < 2) return set_error(STARKV_ERR_UNSUPPORTED, "window rows per group too large for shared memory");
  p.scale2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(kHeadDim)));
  int64_t tiles = 0;
  bool need_lse = false;   // the first pass runs unless every sequence supplies its normalisers
  for (int i = i0; i < i1; ++i) {
    const starkv_seq& q = seqs[i];
    const int lp = q.L - w;
    ScoreSeq& ss = p.seq[i - i0];
    ss.Lp = lp;
    ss.nt = tiles_of(lp);
    ss.tile_base = tiles;
    ss.s_raw = reinterpret_cast<float*>(ws + plan.raw_off[i]);
    ss.lse = q.lse;
    if (!q.lse && ss.nt > 0) need_lse = true;
    tiles += static_cast<int64_t>(nlayers) * G * ss.nt;
    if (ss.nt == 0) continue;
    if ((s = encode_3d(&p.tmk[i - i0], q.k, kHeadDim, q.L, static_cast<uint64_t>(c.n_layers) * G, kTileKeys)) != STARKV_OK) return s;
    const uint64_t qrows = static_cast<uint64_t>(H) * w;
    if ((s = encode_3d(&p.tmqa[i - i0], q.q, kHeadDim, qrows, c.n_layers, std::min(p.rows, kTileKeys))) != STARKV_OK)
      return s;
    if (p.rows > kTileKeys &&
        (s = encode_3d(&p.tmqb[i - i0], q.q, kHeadDim, qrows, c.n_layers, p.rows - kTileKeys)) != STARKV_OK)
      return s;
    if ((s = encode_3d(&p.tmq2[i - i0], q.q, kHeadDim, static_cast<uint64_t>(H) * w, c.n_layers, p.n2)) != STARKV_OK) return s;
  }
  if (tiles == 0) return STARKV_OK;
  p.total_tiles = tiles;
  p.grid1 = static_cast<int>(std::min<int64_t>(tiles, st->num_sms));
  p.partials = reinterpret_cast<float2*>(ws + plan.partials) + *partial_cursor * kMaxRows;
  *partial_cursor += tiles;
  p.err = st->dev.err;
  p.wait_ns = st->wait_ns;
  if (need_lse)
    CUDA_TRY(launch(st, STARKV_KERNEL_SCORE_LSE, stream, [&] { return score_lse_launch(p, p.grid1, stream); }));
  CUDA_TRY(launch(st, STARKV_KERNEL_SCORE_ACCUM, stream, [&] { return score_accum_launch(p, p.grid1, stream); }));
  return STARKV_OK;
}

SeqBatch make_batch(const starkv_state* st, const starkv_seq* seqs, int i0, int i1, int layer0, int nlayers,
                    char* ws, const WsPlan& plan) {
  SeqBatch b;
  memset(&b, 0, sizeof(b));
  b.nseq = i1 - i0;
  b.layer0 = layer0;
  b.nlayers = nlayers;
  for (int i = i0; i < i1; ++i) b.s[i - i0] = make_view(st, seqs[i], ws, plan, i);
  return b;
}

starkv_status check_ws(const starkv_state* st, void* ws, size_t bytes, size_t need) {
  (void)st;
  if (need > 0 && (!ws || bytes < need))
    return set_error(STARKV_ERR_INVALID_ARG, "workspace too small: %zu bytes given, %zu needed", bytes, need);
  if (reinterpret_cast<uintptr_t>(ws) & 255) return set_error(STARKV_ERR_INVALID_ARG, "workspace not 256-byte aligned");
  return STARKV_OK;
}

starkv_status check_device(const starkv_state* st) {
  int dev = -1;
  CUDA_TRY(cudaGetDevice(&dev));
  if (dev != st->device)
    return set_error(STARKV_ERR_INVALID_ARG, "state lives on device %d, current device is %d", st->device, dev);
  return STARKV_OK;
}

// Stages of the step (per-layer calls use a one-layer range).
enum Stage : unsigned { kScore = 1, kPool = 2, kStatsRaw = 4, kStatsPooled = 8, kSelect = 16, kCompact = 32 };

starkv_status run_stages(starkv_state* st, const starkv_seq* seqs, int nseq, int layer0, int nlayers,
                         unsigned stages, void* workspace, size_t ws_bytes, cudaStream_t stream) {
  const starkv_config& c = st->cfg;
  WsPlan plan;
  const bool ws_S = (stages & kStatsRaw) != 0;
  const bool ws_score = (stages & kSelect) != 0;
  plan_ws(st, seqs, nseq, nlayers, ws_S, ws_score, &plan);
  starkv_status s = check_ws(st, workspace, ws_bytes, plan.total);
  if (s != STARKV_OK) return s;
  char* ws = static_cast<char*>(workspace);
  const KParams kp = make_kparams(st);
  size_t partial_cursor = 0;
  for (int i0 = 0; i0 < nseq; i0 += kMaxBatch) {
    const int i1 = std::min(nseq, i0 + kMaxBatch);
    int lp_max = 0, rows_out_max = 0;
    for (int i = i0; i < i1; ++i) {
      lp_max = std::max(lp_max, seqs[i].L - c.window);
      rows_out_max = std::max(rows_out_max, seqs[i].budget + c.window);
    }
    const SeqBatch b = make_batch(st, seqs, i0, i1, layer0, nlayers, ws, plan);
    if (stages & kScore) {
      s = run_score(st, seqs, i0, i1, layer0, nlayers, ws, plan, &partial_cursor, stream);
      if (s != STARKV_OK) return s;
    }
    if ((stages & kPool) && lp_max > 0)
      CUDA_TRY(launch(st, STARKV_KERNEL_POOL, stream, [&] {
        return pool_launch(b, c.n_kv_heads, c.n_heads, c.pool_kernel, lp_max, stream);
      }));
    if (stages & kSelect)
      CUDA_TRY(launch(st, STARKV_KERNEL_CALIBRATE, stream, [&] {
        return calibrate_launch(b, kp, st->dev, (stages & kStatsRaw) != 0, lp_max, stream);
      }));
    if ((stages & kCompact) && rows_out_max > 0)
      CUDA_TRY(launch(st, STARKV_KERNEL_COMPACT, stream, [&] {
        return compact_launch(b, c.n_kv_heads, c.window, kp.per_head, rows_out_max, st->dev.err, stream);
      }));
  }
  return STARKV_OK;
}

// Elements of a metadata buffer over `nl` layers (one layer if it is shared).
size_t meta_elems(const starkv_config& c, const starkv_seq& s, int nl) {
  if (s.meta_layer_stride) return static_cast<size_t>(nl) * s.meta_layer_stride;
  return static_cast<size_t>(c.n_kv_heads - 1) * s.meta_group_stride + s.L;
}

size_t seq_bytes_in(const starkv_config& c, const starkv_seq& s) {
  const size_t kv = static_cast<size_t>(c.n_layers) * c.n_kv_heads * s.L * kHeadDim * 2;
  const size_t q = static_cast<size_t>(c.n_layers) * c.n_heads * c.window * kHeadDim * 2;
  const size_t meta = meta_elems(c, s, c.n_layers) * 4;
  const size_t lse = s.lse ? align256(static_cast<size_t>(c.n_layers) * c.n_heads * c.window * 4) : 0;
  return align256(kv) * 2 + align256(q) + align256(meta) + lse;
}

size_t seq_bytes_out(const starkv_config& c, const starkv_seq& s) {
  const size_t ro = s.budget + c.window, lp = s.L - c.window;
  size_t b = align256(static_cast<size_t>(c.n_layers) * c.n_kv_heads * ro * kHeadDim * 2) * 2;
  const size_t P = sel_rows(c);
  b += align256(static_cast<size_t>(c.n_layers) * P * ro * 4);
  b += align256(static_cast<size_t>(c.n_layers) * P * s.budget * 4);
  if (s.S) b += align256(static_cast<size_t>(c.n_layers) * c.n_kv_heads * lp * 4);
  if (s.score) b += align256(static_cast<size_t>(c.n_layers) * P * lp * 4);
  if (s.stats) b += align256(static_cast<size_t>(c.n_layers) * stats_bytes(c));
  return b;
}

// ---- window attention (attn.cu): workspace and launches

int64_t attn_units(const starkv_config& c, const starkv_seq* seqs, int i0, int i1) {
  int64_t u = 0;
  for (int i = i0; i < i1; ++i)
    u += static_cast<int64_t>(c.n_layers) * c.n_kv_heads * ((seqs[i].L - c.window + kAttnUnitKeys - 1) / kAttnUnitKeys);
  return u;
}

// Piece partials of one launch batch: (m, l) and the unnormalised output per slot.
void attn_regions(const starkv_state* st, int nrows, int64_t units, int* grid, size_t* ml_bytes, size_t* o_bytes) {
  *grid = units > 0 ? static_cast<int>(std::min<int64_t>(units, st->num_sms)) : 0;
  const size_t slots = static_cast<size_t>(attn_slots(nrows, *grid));
  *ml_bytes = align256(slots * kMaxRows * sizeof(float2));
  *o_bytes = align256(slots * kMaxRows * kHeadDim * sizeof(float));
}

size_t attn_ws_bytes(const starkv_state* st, const starkv_seq* seqs, int nseq) {
  const starkv_config& c = st->cfg;
  size_t best = 0;
  for (int i0 = 0; i0 < nseq; i0 += kMaxBatch) {
    const int i1 = std::min(nseq, i0 + kMaxBatch);
    int grid;
    size_t ml, o;
    attn_regions(st, (i1 - i0) * c.n_layers * c.n_kv_heads, attn_units(c, seqs, i0, i1), &grid, &ml, &o);
    best = std::max(best, ml + o);
  }
  return best;
}

starkv_status run_attention(starkv_state* st, const starkv_seq* seqs, int nseq, void* workspace, size_t ws_bytes,
                            cudaStream_t stream) {
  const starkv_config& c = st->cfg;
  const int G = c.n_kv_heads, H = c.n_heads, w = c.window;
  starkv_status s = check_ws(st, workspace, ws_bytes, attn_ws_bytes(st, seqs, nseq));
  if (s != STARKV_OK) return s;
  if ((s = get_encoder()) != STARKV_OK) return s;
  static thread_local AttnParams p;   // ~17 KB: kept off the stack
  char* ws = static_cast<char*>(workspace);
  for (int i0 = 0; i0 < nseq; i0 += kMaxBatch) {
    const int i1 = std::min(nseq, i0 + kMaxBatch);
    memset(&p, 0, sizeof(p));
    p.nseq = i1 - i0;
    p.layer0 = 0;
    p.nlayers = c.n_layers;
    p.G = G;
    p.rows = (H / G) * w;
    p.n_mtiles = (p.rows + 127) / 128;
    p.q_rows = (p.rows + 15) & ~15;
    p.kv_stages = attn_kv_stages(p.q_rows);
    p.scale2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(kHeadDim)));
    int64_t units = 0;
    for (int i = i0; i < i1; ++i) {
      const starkv_seq& q = seqs[i];
      AttnSeq& a = p.seq[i - i0];
      a.Lp = q.L - w;
      a.nu = (a.Lp + kAttnUnitKeys - 1) / kAttnUnitKeys;
      a.unit_base = units;
      a.o = q.attn_o;
      a.lse = q.attn_lse;
      units += static_cast<int64_t>(c.n_layers) * G * a.nu;
      if (a.nu == 0) continue;
      const uint64_t zkv = static_cast<uint64_t>(c.n_layers) * G, qrows = static_cast<uint64_t>(H) * w;
      if ((s = encode_3d(&p.tmk[i - i0], q.k, kHeadDim, q.L, zkv, kAttnUnitKeys)) != STARKV_OK) return s;
      if ((s = encode_3d(&p.tmv[i - i0], q.v, kHeadDim, q.L, zkv, kAttnUnitKeys)) != STARKV_OK) return s;
      if ((s = encode_3d(&p.tmqa[i - i0], q.q, kHeadDim, qrows, c.n_layers, std::min(p.rows, 128))) != STARKV_OK)
        return s;
      if (p.rows > 128 &&
          (s = encode_3d(&p.tmqb[i - i0], q.q, kHeadDim, qrows, c.n_layers, p.rows - 128)) != STARKV_OK)
        return s;
    }
    size_t ml_bytes, o_bytes;
    attn_regions(st, p.nseq * c.n_layers * G, units, &p.grid, &ml_bytes, &o_bytes);
    p.total_units = units;
    p.part_ml = reinterpret_cast<float2*>(ws);
    p.part_o = reinterpret_cast<float*>(ws + ml_bytes);
    p.err = st->dev.err;
    p.wait_ns = st->wait_ns;
    if (units > 0)
      CUDA_TRY(launch(st, STARKV_KERNEL_ATTENTION, stream, [&] { return attn_main_launch(p, stream); }));
    CUDA_TRY(launch(st, STARKV_KERNEL_ATTN_COMBINE, stream, [&] { return attn_combine_launch(p, stream); }));
  }
  return STARKV_OK;
}

}  // namespace

extern "C" {

void starkv_default_config(starkv_config* c) {
  if (!c) return;
  memset(c, 0, sizeof(*c));
  c->n_layers = 28;
  c->n_heads = 28;
  c->n_kv_heads = 4;
  c->head_dim = 128;
  c->window = 32;
  c->grid_rows = 52;
  c->grid_cols = 52;
  c->pool_kernel = 5;
  c->mi_bins = 8;
  c->mi_grid = 8;
  c->n_warmup = 5;
  c->n_ramp = 10;
  c->max_seqs = 1;
  c->lambda = 0.5f;
  c->tau = 1.0f;
  c->rho_mi = 0.9f;
  c->rho_t = 0.9f;
  c->delta = 0.2f;
  c->d_min = 0.1f;
  c->t_min = 0.95f;
  c->t_max = 1.05f;
  c->eps = 1e-6f;
  c->eps_h = 1e-12f;
  c->select_mode = STARKV_SELECT_GLOBAL;
}

starkv_status starkv_init_state(const starkv_config* cfg, starkv_state** out, void* stream) {
  if (!cfg || !out) return set_error(STARKV_ERR_INVALID_ARG, "NULL config or output pointer");
  *out = nullptr;
  starkv_status s = validate_config(*cfg);
  if (s != STARKV_OK) return s;
  starkv_state* st = new (std::nothrow) starkv_state();
  if (!st) return set_error(STARKV_ERR_NOMEM, "host allocation failed");
  st->cfg = *cfg;
  cudaError_t e = cudaGetDevice(&st->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&st->num_sms, cudaDevAttrMultiProcessorCount, st->device);
  if (e == cudaSuccess) e = score_configure();
  if (e == cudaSuccess) e = select_configure();
  if (e == cudaSuccess) e = attn_configure();
  if (e != cudaSuccess) {
    delete st;
    return set_error(STARKV_ERR_CUDA, "device setup failed: %s", cudaGetErrorString(e));
  }
  // The no-allocation scoring call's scratch on this device.  Under lazy module
  // loading this lookup loads the module that holds the array, so its 16 MiB
  // are reserved here, where the library allocates anyway, and not inside a
  // call that promises to allocate nothing.  A failure only disables that call.
  e = cudaGetSymbolAddress(&st->noalloc_scratch, g_noalloc_scratch);
  if (e != cudaSuccess || !st->noalloc_scratch) {
    st->noalloc_scratch = nullptr;
    st->noalloc_error = cudaGetErrorString(e);
    cudaGetLastError();   // the failure is recorded, not left for the next call
  }
  const size_t SL = static_cast<size_t>(cfg->max_seqs) * cfg->n_layers;
  const size_t G = cfg->n_kv_heads, RC = static_cast<size_t>(cfg->grid_rows) * cfg->grid_cols;
  const size_t o_n = 0;
  const size_t o_mibar = o_n + align256(SL * sizeof(int32_t));
  const size_t o_micur = o_mibar + align256(SL * G * sizeof(double));
  const size_t o_phi = o_micur + align256(SL * G * sizeof(double));
  const size_t o_m = o_phi + align256(SL * G * sizeof(float));
  const size_t o_err = o_m + align256(SL * G * RC * sizeof(float));
  st->mem_bytes = o_err + 256;
  e = cudaMalloc(&st->mem, st->mem_bytes);
  if (e != cudaSuccess) {
    delete st;
    return set_error(STARKV_ERR_NOMEM, "state allocation of %zu bytes failed: %s", st->mem_bytes, cudaGetErrorString(e));
  }
  char* m = static_cast<char*>(st->mem);
  st->dev.n = reinterpret_cast<int32_t*>(m + o_n);
  st->dev.mi_bar = reinterpret_cast<double*>(m + o_mibar);
  st->dev.mi_cur = reinterpret_cast<double*>(m + o_micur);
  st->dev.phi_cur = reinterpret_cast<float*>(m + o_phi);
  st->dev.m = reinterpret_cast<float*>(m + o_m);
  st->dev.err = reinterpret_cast<uint32_t*>(m + o_err);
  e = cudaMemsetAsync(st->mem, 0, st->mem_bytes, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) {
    cudaFree(st->mem);
    delete st;
    return set_error(STARKV_ERR_CUDA, "state clear failed: %s", cudaGetErrorString(e));
  }
  *out = st;
  return STARKV_OK;
}

starkv_status starkv_reset_seq(starkv_state* st, int32_t slot, void* stream) {
  if (!st) return set_error(STARKV_ERR_INVALID_ARG, "state is NULL");
  const starkv_config& c = st->cfg;
  if (slot < 0 || slot >= c.max_seqs) return set_error(STARKV_ERR_INVALID_ARG, "slot out of range");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t L = c.n_layers, G = c.n_kv_heads, RC = static_cast<size_t>(c.grid_rows) * c.grid_cols;
  CUDA_TRY(cudaMemsetAsync(st->dev.n + slot * L, 0, L * sizeof(int32_t), s));
  CUDA_TRY(cudaMemsetAsync(st->dev.mi_bar + slot * L * G, 0, L * G * sizeof(double), s));
  CUDA_TRY(cudaMemsetAsync(st->dev.m + slot * L * G * RC, 0, L * G * RC * sizeof(float), s));
  return STARKV_OK;
}

starkv_status starkv_destroy_state(starkv_state* st) {
  if (!st) return STARKV_OK;
  cudaError_t e = cudaDeviceSynchronize();
  for (auto& r : st->recs) {
    cudaEventDestroy(r.a);
    cudaEventDestroy(r.b);
  }
  for (auto ev : st->pool) cudaEventDestroy(ev);
  for (auto ev : st->pipe_ev) cudaEventDestroy(ev);
  if (st->pipe_in) cudaStreamDestroy(st->pipe_in);
  if (st->pipe_out) cudaStreamDestroy(st->pipe_out);
  if (e == cudaSuccess) e = cudaFree(st->mem);
  delete st;
  if (e != cudaSuccess) return set_error(STARKV_ERR_CUDA, "destroy failed: %s", cudaGetErrorString(e));
  return STARKV_OK;
}

starkv_status starkv_slot_state_bytes(const starkv_state* st, size_t* bytes) {
  if (!st || !bytes) return set_error(STARKV_ERR_INVALID_ARG, "NULL state or output pointer");
  const starkv_config& c = st->cfg;
  *bytes = STARKV_SLOT_STATE_BYTES(c.n_layers, c.n_kv_heads, static_cast<size_t>(c.grid_rows) * c.grid_cols);
  return STARKV_OK;
}

namespace {

// Offsets of the three arrays of one slot in an exported buffer, and their
// sources in the device state.
struct SlotLayout {
  size_t o_n, o_mi, o_m, n_bytes, mi_bytes, m_bytes;
  int32_t* dn;
  double* dmi;
  float* dm;
};

SlotLayout slot_layout(const starkv_state* st, int slot) {
  const starkv_config& c = st->cfg;
  const size_t L = c.n_layers, G = c.n_kv_heads, RC = static_cast<size_t>(c.grid_rows) * c.grid_cols;
  SlotLayout s;
  s.n_bytes = L * sizeof(int32_t);
  s.mi_bytes = L * G * sizeof(double);
  s.m_bytes = L * G * RC * sizeof(float);
  s.o_n = sizeof(starkv_slot_header);
  s.o_mi = s.o_n + ((s.n_bytes + 7) & ~static_cast<size_t>(7));
  s.o_m = s.o_mi + s.mi_bytes;
  s.dn = st->dev.n + slot * L;
  s.dmi = st->dev.mi_bar + slot * L * G;
  s.dm = st->dev.m + slot * L * G * RC;
  return s;
}

starkv_status check_slot_buffer(const starkv_state* st, int slot, const void* host, size_t bytes) {
  if (!st) return set_error(STARKV_ERR_INVALID_ARG, "state is NULL");
  if (!host) return set_error(STARKV_ERR_INVALID_ARG, "host buffer is NULL");
  if (slot < 0 || slot >= st->cfg.max_seqs) return set_error(STARKV_ERR_INVALID_ARG, "slot out of range");
  size_t need = 0;
  starkv_slot_state_bytes(st, &need);
  if (bytes < need) return set_error(STARKV_ERR_INVALID_ARG, "slot buffer of %zu bytes, %zu needed", bytes, need);
  if (reinterpret_cast<uintptr_t>(host) & 7) return set_error(STARKV_ERR_INVALID_ARG, "slot buffer not 8-byte aligned");
  return STARKV_OK;
}

}  // namespace

starkv_status starkv_export_slot(starkv_state* st, int32_t slot, void* host, size_t bytes, void* stream) {
  starkv_status s = check_slot_buffer(st, slot, host, bytes);
  if (s != STARKV_OK) return s;
  if ((s = check_device(st)) != STARKV_OK) return s;
  const starkv_config& c = st->cfg;
  starkv_slot_header h;
  memset(&h, 0, sizeof(h));
  h.magic = STARKV_SLOT_MAGIC;
  h.version = 1;
  h.n_layers = c.n_layers;
  h.n_kv_heads = c.n_kv_heads;
  h.grid_rows = c.grid_rows;
  h.grid_cols = c.grid_cols;
  char* b = static_cast<char*>(host);
  memcpy(b, &h, sizeof(h));
  const SlotLayout l = slot_layout(st, slot);
  memset(b + l.o_n + l.n_bytes, 0, l.o_mi - l.o_n - l.n_bytes);   // padding
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  CUDA_TRY(cudaMemcpyAsync(b + l.o_n, l.dn, l.n_bytes, cudaMemcpyDeviceToHost, cs));
  CUDA_TRY(cudaMemcpyAsync(b + l.o_mi, l.dmi, l.mi_bytes, cudaMemcpyDeviceToHost, cs));
  CUDA_TRY(cudaMemcpyAsync(b + l.o_m, l.dm, l.m_bytes, cudaMemcpyDeviceToHost, cs));
  return STARKV_OK;
}

starkv_status starkv_import_slot(starkv_state* st, int32_t slot, const void* host, size_t bytes, void* stream) {
  starkv_status s = check_slot_buffer(st, slot, host, bytes);
  if (s != STARKV_OK) return s;
  if ((s = check_device(st)) != STARKV_OK) return s;
  const starkv_config& c = st->cfg;
  starkv_slot_header h;
  memcpy(&h, host, sizeof(h));
  if (h.magic != STARKV_SLOT_MAGIC || h.version != 1)
    return set_error(STARKV_ERR_INVALID_ARG, "not an exported slot state (magic / version)");
  if (h.n_layers != c.n_layers || h.n_kv_heads != c.n_kv_heads || h.grid_rows != c.grid_rows ||
      h.grid_cols != c.grid_cols)
    return set_error(STARKV_ERR_INVALID_ARG, "slot state of shape (layers %d, G %d, grid %d x %d), state has (%d, %d, %d x %d)",
                     h.n_layers, h.n_kv_heads, h.grid_rows, h.grid_cols, c.n_layers, c.n_kv_heads, c.grid_rows,
                     c.grid_cols);
  const char* b = static_cast<const char*>(host);
  const SlotLayout l = slot_layout(st, slot);
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  CUDA_TRY(cudaMemcpyAsync(l.dn, b + l.o_n, l.n_bytes, cudaMemcpyHostToDevice, cs));
  CUDA_TRY(cudaMemcpyAsync(l.dmi, b + l.o_mi, l.mi_bytes, cudaMemcpyHostToDevice, cs));
  CUDA_TRY(cudaMemcpyAsync(l.dm, b + l.o_m, l.m_bytes, cudaMemcpyHostToDevice, cs));
  return STARKV_OK;
}

starkv_status starkv_get_config(const starkv_state* st, starkv_config* out) {
  if (!st || !out) return set_error(STARKV_ERR_INVALID_ARG, "NULL argument");
  *out = st->cfg;
  return STARKV_OK;
}

starkv_status starkv_set_wait_limit(starkv_state* st, uint64_t limit_ns) {
  if (!st) return set_error(STARKV_ERR_INVALID_ARG, "state is NULL");
  st->wait_ns = limit_ns;
  return STARKV_OK;
}

starkv_status starkv_workspace_bytes(const starkv_state* st, const starkv_seq* seqs, int32_t nseq, int32_t host,
                                     size_t* bytes) {
  if (!bytes) return set_error(STARKV_ERR_INVALID_ARG, "bytes is NULL");
  starkv_status s = validate_seqs(st, seqs, nseq, 0);
  if (s != STARKV_OK) return s;
  WsPlan a, b, c1;
  plan_ws(st, seqs, nseq, st->cfg.n_layers, true, true, &a);   // starkv_step
  plan_ws(st, seqs, nseq, 1, false, false, &b);                 // starkv_score_layer, starkv_compact
  plan_ws(st, seqs, nseq, 1, false, true, &c1);                 // starkv_select
  size_t total = std::max(std::max(a.total, attn_ws_bytes(st, seqs, nseq)), std::max(b.total, c1.total));
  if (host) {
    std::vector<starkv_seq> dev(seqs, seqs + nseq);
    size_t staged = 0;
    for (int i = 0; i < nseq; ++i) {
      staged += seq_bytes_in(st->cfg, seqs[i]) + seq_bytes_out(st->cfg, seqs[i]);
      dev[i].S = nullptr;  // step keeps S in the workspace unless asked for it
    }
    WsPlan c;
    plan_ws(st, dev.data(), nseq, st->cfg.n_layers, true, true, &c);
    total = staged + c.total;
  }
  *bytes = total;
  return STARKV_OK;
}

starkv_status starkv_score_layer(starkv_state* st, int32_t layer, const starkv_seq* seqs, int32_t nseq,
                                 void* workspace, size_t workspace_bytes, void* stream) {
  starkv_status s = validate_seqs(st, seqs, nseq, kNeedK | kNeedQ | kNeedS);
  if (s != STARKV_OK) return s;
  if (layer < 0 || layer >= st->cfg.n_layers) return set_error(STARKV_ERR_INVALID_ARG, "layer out of range");
  if ((s = check_device(st)) != STARKV_OK) return s;
  return run_stages(st, seqs, nseq, layer, 1, kScore | kPool, workspace, workspace_bytes,
                    static_cast<cudaStream_t>(stream));
}

starkv_status starkv_select(starkv_state* st, int32_t layer, const starkv_seq* seqs, int32_t nseq,
                            void* workspace, size_t workspace_bytes, void* stream) {
  starkv_status s = validate_seqs(st, seqs, nseq, kNeedMeta | kNeedS | kNeedIdx);
  if (s != STARKV_OK) return s;
  if (layer < 0 || layer >= st->cfg.n_layers) return set_error(STARKV_ERR_INVALID_ARG, "layer out of range");
  if ((s = check_device(st)) != STARKV_OK) return s;
  return run_stages(st, seqs, nseq, layer, 1, kStatsPooled | kSelect, workspace, workspace_bytes,
                    static_cast<cudaStream_t>(stream));
}

starkv_status starkv_compact(starkv_state* st, int32_t layer, const starkv_seq* seqs, int32_t nseq,
                             void* workspace, size_t workspace_bytes, void* stream) {
  starkv_status s = validate_seqs(st, seqs, nseq, kNeedK | kNeedV | kNeedMeta | kNeedIdx | kNeedOut);
  if (s != STARKV_OK) return s;
  if (layer < 0 || layer >= st->cfg.n_layers) return set_error(STARKV_ERR_INVALID_ARG, "layer out of range");
  if ((s = check_device(st)) != STARKV_OK) return s;
  return run_stages(st, seqs, nseq, layer, 1, kCompact, workspace, workspace_bytes,
                    static_cast<cudaStream_t>(stream));
}

starkv_status starkv_step(starkv_state* st, const starkv_seq* seqs, int32_t nseq, void* workspace,
                          size_t workspace_bytes, void* stream) {
  NvtxRange range("starkv_step");
  starkv_status s = validate_seqs(st, seqs, nseq, kNeedK | kNeedQ | kNeedV | kNeedMeta | kNeedIdx | kNeedOut);
  if (s != STARKV_OK) return s;
  if ((s = check_device(st)) != STARKV_OK) return s;
  return run_stages(st, seqs, nseq, 0, st->cfg.n_layers, kScore | kStatsRaw | kSelect | kCompact, workspace,
                    workspace_bytes, static_cast<cudaStream_t>(stream));
}

starkv_status starkv_window_attention(starkv_state* st, const starkv_seq* seqs, int32_t nseq, void* workspace,
                                      size_t workspace_bytes, void* stream) {
  NvtxRange range("starkv_window_attention");
  starkv_status s = validate_seqs(st, seqs, nseq, kNeedK | kNeedQ | kNeedV);
  if (s != STARKV_OK) return s;
  for (int i = 0; i < nseq; ++i)
    if (!seqs[i].attn_lse) return set_error(STARKV_ERR_INVALID_ARG, "seq %d: attn_lse is NULL", i);
  if ((s = check_device(st)) != STARKV_OK) return s;
  return run_attention(st, seqs, nseq, workspace, workspace_bytes, static_cast<cudaStream_t>(stream));
}

starkv_status starkv_step_host(starkv_state* st, const starkv_seq* seqs, int32_t nseq, void* workspace,
                               size_t workspace_bytes, void* stream) {
  NvtxRange range("starkv_step_host");
  starkv_status s = validate_seqs(st, seqs, nseq, kNeedK | kNeedQ | kNeedV | kNeedMeta | kNeedIdx | kNeedOut);
  if (s != STARKV_OK) return s;
  if ((s = check_device(st)) != STARKV_OK) return s;
  size_t need = 0;
  if ((s = starkv_workspace_bytes(st, seqs, nseq, 1, &need)) != STARKV_OK) return s;
  if ((s = check_ws(st, workspace, workspace_bytes, need)) != STARKV_OK) return s;
  const starkv_config& c = st->cfg;
  const int G = c.n_kv_heads, NL = c.n_layers;
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  if (!st->pipe_in) {
    CUDA_TRY(cudaStreamCreateWithFlags(&st->pipe_in, cudaStreamNonBlocking));
    CUDA_TRY(cudaStreamCreateWithFlags(&st->pipe_out, cudaStreamNonBlocking));
  }
  // layers are independent: the step runs in chunks of layers so that the
  // upload of chunk i+1 and the download of chunk i-1 overlap the compute of
  // chunk i (the host link carries both directions at once).  Chunks of four
  // layers, the last ones halving (4 layers as 2 + 1 + 1): what follows the
  // last upload (that chunk's compute and download) is then one layer's
  std::vector<int> chunk_l0;
  for (int l0 = 0; l0 < NL;) {
    const int rem = NL - l0;
    chunk_l0.push_back(l0);
    l0 += rem > 4 ? 4 : (rem + 1) / 2;
  }
  chunk_l0.push_back(NL);
  const int nchunk = static_cast<int>(chunk_l0.size()) - 1;
  const size_t n_ev = 2 + 2 * static_cast<size_t>(nchunk);
  while (st->pipe_ev.size() < n_ev) {
    cudaEvent_t e = nullptr;
    CUDA_TRY(cudaEventCreateWithFlags(&e, cudaEventDisableTiming));
    st->pipe_ev.push_back(e);
  }
  cudaEvent_t* ev = st->pipe_ev.data();
  char* cur = static_cast<char*>(workspace);
  auto take = [&](size_t bytes) {
    char* p = cur;
    cur += align256(bytes);
    return p;
  };
  struct Rows { size_t kv_layer, q_layer, lse_layer, meta_layer, out_layer, sel_layer, meta_out_layer, lp; bool v_in_place; };
  const size_t P = sel_rows(c);
  std::vector<starkv_seq> dev(seqs, seqs + nseq);
  std::vector<Rows> rows(nseq);
  for (int i = 0; i < nseq; ++i) {
    const starkv_seq& h = seqs[i];
    starkv_seq& d = dev[i];
    Rows& r = rows[i];
    r.kv_layer = static_cast<size_t>(G) * h.L * kHeadDim * 2;
    r.q_layer = static_cast<size_t>(c.n_heads) * c.window * kHeadDim * 2;
    r.lse_layer = static_cast<size_t>(c.n_heads) * c.window * 4;
    r.meta_layer = static_cast<size_t>(h.meta_layer_stride) * 4;
    r.lp = static_cast<size_t>(h.L - c.window);
    r.out_layer = static_cast<size_t>(h.budget + c.window);
    r.sel_layer = P * h.budget;
    r.meta_out_layer = P * r.out_layer;
    const size_t mb = meta_elems(c, h, NL) * 4;
    d.k = take(NL * r.kv_layer);
    // V is read only at the kept rows: from page-locked host memory the gather
    // reads them in place instead of uploading all of V
    cudaPointerAttributes pa;
    r.v_in_place = cudaPointerGetAttributes(&pa, h.v) == cudaSuccess && pa.type == cudaMemoryTypeHost &&
                   pa.devicePointer != nullptr;
    if (!r.v_in_place) cudaGetLastError();
    d.v = r.v_in_place ? static_cast<const void*>(pa.devicePointer) : take(NL * r.kv_layer);
    d.q = take(NL * r.q_layer);
    d.meta = reinterpret_cast<const uint32_t*>(take(mb));
    d.k_out = take(NL * static_cast<size_t>(G) * r.out_layer * kHeadDim * 2);
    d.v_out = take(NL * static_cast<size_t>(G) * r.out_layer * kHeadDim * 2);
    d.meta_out = reinterpret_cast<uint32_t*>(take(NL * r.meta_out_layer * 4));
    d.idx = reinterpret_cast<int32_t*>(take(NL * r.sel_layer * 4));
    d.S = h.S ? reinterpret_cast<float*>(take(NL * static_cast<size_t>(G) * r.lp * 4)) : nullptr;
    d.score = h.score ? reinterpret_cast<float*>(take(NL * P * r.lp * 4)) : nullptr;
    d.stats = h.stats ? reinterpret_cast<float*>(take(static_cast<size_t>(NL) * stats_bytes(c))) : nullptr;
    d.lse = h.lse ? reinterpret_cast<const float*>(take(NL * r.lse_layer)) : nullptr;
  }
  const size_t used = static_cast<size_t>(cur - static_cast<char*>(workspace));
  // the uploads may start once earlier work on the caller's stream (which may
  // still read these staging buffers) is done
  CUDA_TRY(cudaEventRecord(ev[0], cs));
  CUDA_TRY(cudaStreamWaitEvent(st->pipe_in, ev[0], 0));
  auto h2d = [&](const void* dst, const void* src, size_t off, size_t bytes) {
    return cudaMemcpyAsync(static_cast<char*>(const_cast<void*>(dst)) + off, static_cast<const char*>(src) + off,
                           bytes, cudaMemcpyHostToDevice, st->pipe_in);
  };
  auto d2h = [&](void* dst, const void* src, size_t off, size_t bytes) {
    return cudaMemcpyAsync(static_cast<char*>(dst) + off, static_cast<const char*>(src) + off, bytes,
                           cudaMemcpyDeviceToHost, st->pipe_out);
  };
  for (int k = 0; k < nchunk; ++k) {
    const int l0 = chunk_l0[k], nl = chunk_l0[k + 1] - l0;
    for (int i = 0; i < nseq; ++i) {
      const starkv_seq& h = seqs[i];
      const starkv_seq& d = dev[i];
      const Rows& r = rows[i];
      CUDA_TRY(h2d(d.k, h.k, l0 * r.kv_layer, nl * r.kv_layer));
      if (!r.v_in_place) CUDA_TRY(h2d(d.v, h.v, l0 * r.kv_layer, nl * r.kv_layer));
      CUDA_TRY(h2d(d.q, h.q, l0 * r.q_layer, nl * r.q_layer));
      if (h.lse) CUDA_TRY(h2d(d.lse, h.lse, l0 * r.lse_layer, nl * r.lse_layer));
      if (h.meta_layer_stride) CUDA_TRY(h2d(d.meta, h.meta, l0 * r.meta_layer, nl * r.meta_layer));
      else if (k == 0) CUDA_TRY(h2d(d.meta, h.meta, 0, meta_elems(c, h, NL) * 4));
    }
    CUDA_TRY(cudaEventRecord(ev[2 + 2 * k], st->pipe_in));
    CUDA_TRY(cudaStreamWaitEvent(cs, ev[2 + 2 * k], 0));
    s = run_stages(st, dev.data(), nseq, l0, nl, kScore | kStatsRaw | kSelect | kCompact, cur,
                   workspace_bytes - used, cs);
    if (s != STARKV_OK) return s;
    CUDA_TRY(cudaEventRecord(ev[3 + 2 * k], cs));
    CUDA_TRY(cudaStreamWaitEvent(st->pipe_out, ev[3 + 2 * k], 0));
    for (int i = 0; i < nseq; ++i) {
      const starkv_seq& h = seqs[i];
      const starkv_seq& d = dev[i];
      const Rows& r = rows[i];
      const size_t kvo = static_cast<size_t>(G) * r.out_layer * kHeadDim * 2;
      CUDA_TRY(d2h(h.k_out, d.k_out, l0 * kvo, nl * kvo));
      CUDA_TRY(d2h(h.v_out, d.v_out, l0 * kvo, nl * kvo));
      CUDA_TRY(d2h(h.meta_out, d.meta_out, l0 * r.meta_out_layer * 4, nl * r.meta_out_layer * 4));
      if (h.budget > 0) CUDA_TRY(d2h(h.idx, d.idx, l0 * r.sel_layer * 4, nl * r.sel_layer * 4));
      if (h.S && r.lp > 0) CUDA_TRY(d2h(h.S, d.S, l0 * G * r.lp * 4, nl * G * r.lp * 4));
      if (h.score && r.lp > 0) CUDA_TRY(d2h(h.score, d.score, l0 * P * r.lp * 4, nl * P * r.lp * 4));
      if (h.stats) {
        const size_t sb = stats_bytes(c);
        CUDA_TRY(d2h(h.stats, d.stats, l0 * sb, nl * sb));
      }
    }
  }
  // the call's results are in host memory when the caller's stream reaches here
  CUDA_TRY(cudaEventRecord(ev[1], st->pipe_out));
  CUDA_TRY(cudaStreamWaitEvent(cs, ev[1], 0));
  return STARKV_OK;
}

starkv_status starkv_check_device_error(starkv_state* st, void* stream) {
  if (!st) return set_error(STARKV_ERR_INVALID_ARG, "state is NULL");
  uint32_t h = 0;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  CUDA_TRY(cudaMemcpyAsync(&h, st->dev.err, sizeof(h), cudaMemcpyDeviceToHost, s));
  CUDA_TRY(cudaStreamSynchronize(s));
  CUDA_TRY(cudaMemsetAsync(st->dev.err, 0, sizeof(uint32_t), s));
  if (h & kErrTimeout) return set_error(STARKV_ERR_TIMEOUT, "a bounded device wait ran out");
  if (h & kErrMeta) return set_error(STARKV_ERR_DEVICE, "token metadata outside the patch grid");
  if (h & kErrIndex) return set_error(STARKV_ERR_DEVICE, "a kept index outside the past tokens reached the gather");
  return STARKV_OK;
}

starkv_status starkv_selftest_wait(starkv_state* st, uint64_t limit_ns, void* stream) {
  if (!st) return set_error(STARKV_ERR_INVALID_ARG, "state is NULL");
  if (limit_ns < 1000ull || limit_ns > 1000000000ull)
    return set_error(STARKV_ERR_INVALID_ARG, "limit_ns must be in [1 us, 1 s]");
  starkv_status s = check_device(st);
  if (s != STARKV_OK) return s;
  CUDA_TRY(wait_probe_launch(st->dev.err, limit_ns, static_cast<cudaStream_t>(stream)));
  return STARKV_OK;
}

starkv_status starkv_set_timing(starkv_state* st, int32_t on) {
  if (!st) return set_error(STARKV_ERR_INVALID_ARG, "state is NULL");
  st->timing = on != 0;
  return STARKV_OK;
}

starkv_status starkv_kernel_times(starkv_state* st, int64_t* launches, float* total_ms) {
  if (!st) return set_error(STARKV_ERR_INVALID_ARG, "state is NULL");
  float ms[STARKV_NUM_KERNELS] = {};
  starkv_status status = STARKV_OK;
  for (auto& r : st->recs) {
    float t = 0.f;
    cudaError_t e = cudaEventSynchronize(r.b);
    if (e == cudaSuccess) e = cudaEventElapsedTime(&t, r.a, r.b);
    if (e != cudaSuccess && status == STARKV_OK)
      status = set_error(STARKV_ERR_CUDA, "event timing failed: %s", cudaGetErrorString(e));
    ms[r.kind] += t;
    st->pool.push_back(r.a);
    st->pool.push_back(r.b);
  }
  st->recs.clear();
  for (int k = 0; k < STARKV_NUM_KERNELS; ++k) {
    if (launches) launches[k] = st->launches[k];
    if (total_ms) total_ms[k] = ms[k];
    st->launches[k] = 0;
  }
  return status;
}

const char* starkv_last_error(void) { return g_last_error.c_str(); }

}  // extern "C"

// ---------------------------------------------------------------------------
// starkv_score_layer_noalloc: the scoring call for callers that cannot
// allocate device memory (see include/starkv.h).  Its scratch is the static
// device array above, whose address starkv_init_state looked up.

extern "C" starkv_status starkv_score_layer_noalloc(starkv_state* st, int32_t layer, const starkv_seq* seqs,
                                                    int32_t nseq, void* stream) {
  starkv_status s = validate_seqs(st, seqs, nseq, kNeedK | kNeedQ | kNeedS);
  if (s != STARKV_OK) return s;
  if (layer < 0 || layer >= st->cfg.n_layers) return set_error(STARKV_ERR_INVALID_ARG, "layer out of range");
  if (st->timing)
    return set_error(STARKV_ERR_INVALID_ARG, "kernel timing creates CUDA events: turn it off for this call");
  if ((s = check_device(st)) != STARKV_OK) return s;
  if (!st->noalloc_scratch)
    return set_error(STARKV_ERR_CUDA, "the static scratch is unavailable on device %d: %s", st->device,
                     st->noalloc_error.c_str());
  WsPlan plan;
  plan_ws(st, seqs, nseq, 1, false, false, &plan);
  if (plan.total > kNoAllocScratchBytes)
    return set_error(STARKV_ERR_UNSUPPORTED,
                     "this call needs %zu bytes of scratch; the static scratch holds %zu bytes: "
                     "split the batch or use starkv_score_layer with a workspace",
                     plan.total, kNoAllocScratchBytes);
  return run_stages(st, seqs, nseq, layer, 1, kScore | kPool, st->noalloc_scratch, kNoAllocScratchBytes,
                    static_cast<cudaStream_t>(stream));
}
