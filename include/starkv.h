/*
 * starkv.h -- C ABI of the STaR-KV compression stage on one GB300 (sm_103a).
 *
 * STaR-KV (Spatio-Temporal Adaptive Re-weighting) compresses the KV cache of a
 * GUI vision-language model per layer (Algorithm 1, App. A.2):
 *   1. score the last w window queries against every past key over the GQA
 *      groups, pool along tokens and average inside each group  (Sec. 3.3);
 *   2. re-weight by a per-group prior from the online spatial mutual
 *      information of each group's scores with the screen-patch grid (Sec. 3.4);
 *   3. discount stale visual tokens by the temporal stability of their
 *      governing group (Sec. 3.5);
 *   4. reshape by an entropy-derived temperature (Sec. 3.6);
 *   5. keep the global top-B historical tokens plus the recent window and
 *      gather them into a new contiguous cache (Sec. 3.7).
 * An optional per-KV-head selection mode (select_mode = STARKV_SELECT_PER_HEAD,
 * the head-wise top-K of App. A.3 with the STaR-KV factors) lets each group g
 * keep its own B tokens: it ranks s_{g,t} = max(S[g,t] beta_g D_{g,t}, 0)^(1/T_g)
 * with beta_g = (1 - lambda) + lambda G w_g, D_{g,t} of Eq. (9) with phi_g and
 * T_g from the entropy of S[g, .] (Sec. 3.6 on that row).  beta_g is one factor
 * per row, so in this mode the MI prior scales the scores without changing
 * any group's set.
 *
 * Conventions shared by every call
 * --------------------------------
 * - Pointers inside starkv_seq are DEVICE pointers (cudaMalloc / torch CUDA
 *   memory), except for starkv_step_host, where they are HOST pointers.
 *   The caller owns every input and output buffer; the library owns only the
 *   state created by starkv_init_state.
 * - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *   Calls are asynchronous and stream-ordered; none synchronises the stream.
 * - `workspace` is caller-owned device scratch of at least
 *   starkv_workspace_bytes(...) bytes, 256-byte aligned.  Its contents are
 *   undefined on entry and on exit.  Concurrent calls must not share it.
 * - Layouts (all row-major, contiguous):
 *     k, v        bf16  [n_layers][G][L][d]
 *     q           bf16  [n_layers][H][w][d]   post-RoPE queries of the last w tokens
 *     meta        u32   [n_layers][L]  or [L] shared (meta_layer_stride = 0);
 *                       per-KV-head mode: optionally one row per group,
 *                       [n_layers][G][L] (meta_group_stride = L, see below)
 *     S           f32   [n_layers][G][L_p]     group score map, L_p = L - w
 *     score       f32   [n_layers][P][L_p]     fused score s_t (s_{g,t})
 *     idx         i32   [n_layers][P][B]       kept historical positions, ascending
 *     k_out,v_out bf16  [n_layers][G][B + w][d]
 *     meta_out    u32   [n_layers][P][B + w]
 *   where P = 1 in the global selection mode and P = G in the per-KV-head mode
 *   (row g of idx / meta_out belongs to group g of k_out / v_out).
 *     stats       f32   [n_layers][STARKV_STATS_STRIDE(G)]
 *   Token metadata word: bit 31 = visual, bits 20..30 = frame id f(t),
 *   bits 10..19 = patch row r_t, bits 0..9 = patch column c_t (Sec. 3.1).
 *   Text tokens only need bit 31 clear.
 * - Errors: a call that returns non-OK has launched nothing unless the code is
 *   STARKV_ERR_CUDA (a launch or copy failed part-way).  Invalid arguments are
 *   caught on the host before any launch.  Device-side checks (metadata out of
 *   range, a bounded wait that ran out) latch a code in the state's device
 *   error word, which starkv_check_device_error reads.  starkv_last_error
 *   returns a thread-local message for the last non-OK status.
 * - Supported shapes: d = 128; w >= 1; H % G == 0; (H / G) * w <= 256;
 *   G <= 32 in the global selection mode (G = H is the MHA-head granularity of
 *   the ablation in Sec. 4.2: each group's key/value replicated for each of its
 *   query heads), G <= 8 in the per-KV-head mode; L >= w (L_p = L - w >= 0;
 *   L_p = 0 keeps only the window);
 *   0 <= B <= L_p; L < 2^24; 1 <= R, C <= 1024; R * C <= 16384;
 *   2 <= mi_bins <= 16; mi_bins * mi_grid^2 <= 4096; odd pool_kernel <= 31;
 *   frame ids 0..2047.  Other shapes return STARKV_ERR_UNSUPPORTED.
 *   k, v, q, k_out and v_out must be 16-byte aligned, every other array
 *   4-byte aligned (STARKV_ERR_INVALID_ARG otherwise).
 */
#ifndef STARKV_H
#define STARKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  STARKV_OK = 0,
  STARKV_ERR_INVALID_ARG = 1,  /* a pointer, size or index is invalid          */
  STARKV_ERR_UNSUPPORTED = 2,  /* valid but outside the supported shapes       */
  STARKV_ERR_CUDA = 3,         /* a CUDA runtime call failed                   */
  STARKV_ERR_TIMEOUT = 4,      /* a bounded device-side wait ran out           */
  STARKV_ERR_NOMEM = 5,        /* state allocation failed                      */
  STARKV_ERR_DEVICE = 6        /* a device-side input check failed             */
} starkv_status;

/* Hyper-parameters.  starkv_default_config fills the paper's defaults
 * (App. A.1, Table 7 AgentNetBench / UI-TARS) and this library's readings of
 * the values the paper leaves open (pool_kernel, mi_bins, mi_grid, eps, eps_h). */
typedef struct {
  int32_t n_layers;
  int32_t n_heads;      /* H query heads                                           */
  int32_t n_kv_heads;   /* G KV groups ("subspaces", Sec. 3.1)                     */
  int32_t head_dim;     /* d, must be 128                                          */
  int32_t window;       /* w: observation window = recent window W_rec (Sec. 3.1)  */
  int32_t grid_rows;    /* R: patch rows of one screenshot                         */
  int32_t grid_cols;    /* C: patch columns of one screenshot                      */
  int32_t pool_kernel;  /* AvgPool1D kernel (odd), stride 1, zero padding (Sec 3.3)*/
  int32_t mi_bins;      /* K equal-frequency rank bins (Sec. 3.4)                  */
  int32_t mi_grid;      /* M: SpatialBin grid is M x M (Sec. 3.4)                  */
  int32_t n_warmup;     /* lambda is 0 for the first n_warmup steps (App. A.1)     */
  int32_t n_ramp;       /* then ramps linearly to lambda over n_ramp steps         */
  int32_t max_seqs;     /* number of state slots (independent trajectories)        */
  float lambda;         /* MI prior strength (Eq. final_score)                     */
  float tau;            /* prior softmax temperature (Eq. 7)                       */
  float rho_mi;         /* MI EMA decay (Eq. 6)                                    */
  float rho_t;          /* temporal EMA decay (Eq. 8)                              */
  float delta;          /* temporal decay rate (Eq. 9)                             */
  float d_min;          /* minimum temporal factor D_min (Eq. 9)                   */
  float t_min, t_max;   /* AEB temperature range (Sec. 3.6)                        */
  float eps;            /* epsilon of the min-max prior (Eq. 7)                    */
  float eps_h;          /* epsilon of the AEB entropy (Algorithm 1)                */
  int32_t select_mode;  /* STARKV_SELECT_GLOBAL (the paper's, default) or
                           STARKV_SELECT_PER_HEAD (one top-B set per KV group)     */
  /* Variants of the paper's ablations (Table 3, the AEB ablation), 0 = the
   * method as defined.  The paper names them without a formula; this
   * library's readings, with x = Delta_f phi:
   *   decay_mode 1 (linear):    D = D_min + (1 - D_min) max(0, 1 - delta x)
   *   decay_mode 2 (power law): D = D_min + (1 - D_min) (1 + x)^(-delta)
   *   aeb_mode 1 (confidence):  T = T_min + (T_max - T_min)(1 - p_max), with
   *                             p_max = max_t s_bar_t / (sum_t s_bar_t + eps_h)
   *   mi_span 1:                the MI of Sec. 3.4 over the newest frame's
   *                             visual tokens only                              */
  int32_t decay_mode;
  int32_t aeb_mode;
  int32_t mi_span;
} starkv_config;

/* Values of starkv_config.select_mode. */
enum { STARKV_SELECT_GLOBAL = 0, STARKV_SELECT_PER_HEAD = 1 };

/* One sequence (trajectory) of a batch: inputs and caller-owned outputs.  For
 * per-layer calls (score_layer / select / compact) the `layer` argument picks
 * the [layer] slice of every [n_layers][...] buffer below. */
typedef struct {
  const void* k;                /* bf16 [n_layers][G][L][d]                         */
  const void* v;                /* bf16 [n_layers][G][L][d]                         */
  const void* q;                /* bf16 [n_layers][H][w][d]                         */
  const uint32_t* meta;         /* u32  [n_layers][L] (or [L] if stride is 0)       */
  int64_t meta_layer_stride;    /* elements between layers of meta: 0 or >= L       */
  int32_t L;                    /* cache length, including the w recent tokens      */
  int32_t cur_frame;            /* F: frame id of the current (newest) screenshot   */
  int32_t budget;               /* B: kept historical tokens, 0 <= B <= L - w       */
  int32_t slot;                 /* state slot in [0, max_seqs)                      */
  void* k_out;                  /* bf16 [n_layers][G][B + w][d]       (compact)    */
  void* v_out;                  /* bf16 [n_layers][G][B + w][d]       (compact)    */
  uint32_t* meta_out;           /* u32  [n_layers][P][B + w]          (compact)    */
  int32_t* idx;                 /* i32  [n_layers][P][B]   select writes, compact reads */
  float* S;                     /* f32  [n_layers][G][L_p] score_layer writes, select
                                   reads; may be NULL for starkv_step (workspace)   */
  float* score;                 /* f32  [n_layers][P][L_p] fused s_t, optional (NULL) */
  float* stats;                 /* f32  [n_layers][STARKV_STATS_STRIDE(G)], optional */
  int64_t meta_group_stride;    /* elements between the metadata rows of groups g
                                   and g + 1 of one layer: 0 = every group shares
                                   one row (required in the global mode), else >= L
                                   (per-KV-head mode, where each group's cache holds
                                   its own tokens after a compaction); with a
                                   nonzero meta_layer_stride it must be
                                   >= (G - 1) * meta_group_stride + L                */
  const float* lse;             /* f32 [n_layers][H][w], optional: the softmax
                                   normaliser of each window row (Eq. 2), as the
                                   natural-log log-sum-exp over the past keys t < L_p
                                   of z = Q_{-i,h} . K[g(h), t] / sqrt(d) (the window
                                   keys excluded), e.g. from the layer's own prefill
                                   attention pass, which computes these logits.  When
                                   every sequence of a call gives it, the first
                                   scoring pass (a whole read of K) is skipped.
                                   NULL = computed.                                 */
  float* attn_o;                /* f32 [n_layers][H][w][d], optional: written by
                                   starkv_window_attention (the window rows'
                                   attention output over the past keys); 16-byte
                                   aligned                                          */
  float* attn_lse;              /* f32 [n_layers][H][w]: written by
                                   starkv_window_attention, each window row's
                                   natural-log normaliser over the past keys, the
                                   value `lse` takes                                */
} starkv_seq;

/* Per-layer diagnostics written to starkv_seq.stats (floats):
 *   [0] H_hat (p_max with aeb_mode 1)  [1] T  [2] lambda_n  [3] n (steps seen before this one)
 *   [4] sum_t s_bar_t  [5] visual tokens in L_p  [6] kept count  [7] 0
 *   [8 + g]       MI_g of this step            (Eq. 5)
 *   [8 + G + g]   MI_bar_g after the EMA       (Eq. 6)
 *   [8 + 2G + g]  w_g                          (Eq. 7)
 *   [8 + 3G + g]  phi_g                        (Eq. 8)
 *   [8 + 4G + g]  H_hat of the row group g ranks: s_bar (global mode, the same
 *                 for every g) or S[g, .] (per-KV-head mode)
 *   [8 + 5G + g]  its temperature T
 * In the per-KV-head mode [0] and [1] are the means of [8 + 4G ..] and
 * [8 + 5G ..] over g.                                                         */
#define STARKV_STATS_STRIDE(G) (8 + 6 * (G))

typedef struct starkv_state starkv_state;

/* Fills `cfg` with the defaults for the UI-TARS-1.5-7B GQA shape (H = 28,
 * G = 4, d = 128, w = 32, 52 x 52 patches, 28 layers, 1 slot). */
void starkv_default_config(starkv_config* cfg);

/* Allocates the device-resident per-(slot, layer) state: step counter n, MI EMA
 * MI_bar[G] (Eq. 6), temporal EMA m_g[R*C] per group (Eq. 8), all zero (fresh).
 * The state lives on the current CUDA device; use it only there.
 * Errors: INVALID_ARG / UNSUPPORTED for a bad config, NOMEM, CUDA. */
starkv_status starkv_init_state(const starkv_config* cfg, starkv_state** out, void* stream);

/* Trajectory-level reset of one slot (App. A.4: states are reset per
 * trajectory): zeroes n, MI_bar and m_g of every layer, stream-ordered. */
starkv_status starkv_reset_seq(starkv_state* st, int32_t slot, void* stream);

/* Frees the state (synchronises the device first).  NULL is accepted. */
starkv_status starkv_destroy_state(starkv_state* st);

/* Checkpoint / resume of one slot's carried state (the step counters n, the
 * MI EMAs MI_bar of Eq. 6 and the temporal EMAs m_g of Eq. 8 of every layer),
 * e.g. to continue a trajectory in another process or on another device.
 * Host buffer layout, STARKV_SLOT_STATE_BYTES(n_layers, G, R*C) bytes:
 *   starkv_slot_header (32 B), then
 *   int32  n[n_layers]                 padded to a multiple of 8 bytes
 *   f64    mi_bar[n_layers][G]
 *   f32    m[n_layers][G][R*C]
 * The header records the shape; an import whose header does not match the
 * state's (magic, version, n_layers, G, R, C) or whose buffer is too small is
 * rejected with STARKV_ERR_INVALID_ARG before any copy. */
typedef struct {
  uint32_t magic;       /* STARKV_SLOT_MAGIC */
  uint32_t version;     /* 1 */
  int32_t n_layers, n_kv_heads, grid_rows, grid_cols;
  uint32_t reserved[2]; /* zero */
} starkv_slot_header;

#define STARKV_SLOT_MAGIC 0x31564B53u   /* "SKV1" */
#define STARKV_SLOT_STATE_BYTES(n_layers, G, RC)                              \
  (sizeof(starkv_slot_header) + (((size_t)(n_layers) * 4 + 7) & ~(size_t)7) + \
   (size_t)(n_layers) * (G) * 8 + (size_t)(n_layers) * (G) * (RC) * 4)

/* Bytes of one slot's exported state for this state's shape. */
starkv_status starkv_slot_state_bytes(const starkv_state* st, size_t* bytes);

/* Writes slot `slot`'s state into the HOST buffer `host` (>= the size above):
 * the header at once, the arrays by stream-ordered copies (valid after the
 * stream is synchronised; page-locked memory keeps them asynchronous). */
starkv_status starkv_export_slot(starkv_state* st, int32_t slot, void* host, size_t bytes, void* stream);

/* Replaces slot `slot`'s state with the one in the HOST buffer `host`, written
 * by starkv_export_slot for the same shape (stream-ordered copies; the buffer
 * may be reused once the stream has passed them). */
starkv_status starkv_import_slot(starkv_state* st, int32_t slot, const void* host, size_t bytes, void* stream);

/* Copies the config the state was created with. */
starkv_status starkv_get_config(const starkv_state* st, starkv_config* out);

/* Bytes of device workspace that starkv_score_layer, starkv_select,
 * starkv_compact, starkv_step and starkv_window_attention need for this batch
 * (the maximum of the five).
 * With host != 0: the bytes starkv_step_host needs (adds staging copies). */
starkv_status starkv_workspace_bytes(const starkv_state* st, const starkv_seq* seqs, int32_t nseq,
                                     int32_t host, size_t* bytes);

/* Sec. 3.3, Eqs. (2)-(4): for layer `layer` of
 * every sequence, writes S[g][t] = (G/H) * sum_{h in g} AvgPool1D(
 * sum_{i<w} softmax_t(Q_{-i,h} K_past[g]^T / sqrt(d)))[t]  for t < L_p,
 * softmax over K_past only.  Reads k, q; writes S.  Uses tcgen05 tensor cores
 * (bf16 in, fp32 accumulate) in two passes (log-sum-exp, then normalised sums);
 * the first is skipped when every sequence supplies `lse`. */
starkv_status starkv_score_layer(starkv_state* st, int32_t layer, const starkv_seq* seqs,
                                 int32_t nseq, void* workspace, size_t workspace_bytes,
                                 void* stream);

/* starkv_score_layer for callers that cannot allocate device memory: for
 * example code running where cudaMalloc is forbidden or unavailable, such as a
 * host that hands out only pre-registered buffers, or a plugin inside another
 * runtime that owns every device allocation.  The paper has no counterpart;
 * this is a deployment aid.  Same arguments and results as starkv_score_layer,
 * minus the workspace: the scratch (pass-1 partials and unpooled sums) is one
 * static device array of 16 MiB per device.  The array is reserved on a device
 * when this library's device code is loaded there: at context creation under
 * eager module loading, else (CUDA's default lazy loading) in
 * starkv_init_state, which looks up the array's device address
 * (cudaGetSymbolAddress) with the state's device current; it stays reserved
 * until the process exits.  The call itself allocates no device memory (no
 * cudaMalloc / cudaFree, no allocating library routine).  Every call on a
 * device shares the one array and leaves its last contents there (nothing in
 * it has to start at zero): calls that may overlap on the GPU (different
 * streams, or threads without ordering) race on it and must not be issued.  A
 * batch whose scratch would exceed 16 MiB is rejected with
 * STARKV_ERR_UNSUPPORTED before any launch (about 1.8 MB per sequence at the
 * 5-screenshot UI-TARS shape); kernel timing must be off (it creates CUDA
 * events).  STARKV_ERR_CUDA if the array could not be reserved when the state
 * was created. */
starkv_status starkv_score_layer_noalloc(starkv_state* st, int32_t layer, const starkv_seq* seqs,
                                         int32_t nseq, void* stream);

/* The attention pass whose logits Eq. (2) scores (Sec. 3.3; App. A.3 counts the
 * compression's Q K^T as shared with the model's attention): for every layer of
 * every sequence and every window row r = (h, i),
 *   attn_o[r]   = sum_{t < L_p} softmax_t(Q_{-i,h} . K[g(h), t] / sqrt(d)) V[g(h), t]
 *   attn_lse[r] = log sum_{t < L_p} exp(Q_{-i,h} . K[g(h), t] / sqrt(d))
 * over the past keys only (the window keys excluded, as in Eq. 2; a model's
 * causal attention for these rows merges in the window keys' part by the
 * usual log-sum-exp rule).  attn_lse is exactly what `lse` takes, so a caller
 * that runs this pass (or its own attention kernel with the same output)
 * lets starkv_step skip its first scoring pass.  Reads k, v, q; writes attn_o
 * (skipped when NULL) and attn_lse (required; -inf and a zero output when
 * L_p = 0).  Tensor cores: Q K^T in bf16, P V with P rounded to fp16 and V
 * converted to fp16 (|v| must stay below 65504), fp32 accumulation, so
 * |attn_o - O| <= 2^-11 sum_t p_t |V_t| + fp32 rounding, and attn_lse carries
 * the fp32 accuracy of the scoring passes.  Workspace from
 * starkv_workspace_bytes. */
starkv_status starkv_window_attention(starkv_state* st, const starkv_seq* seqs, int32_t nseq,
                                      void* workspace, size_t workspace_bytes, void* stream);

/* Sec. 3.3 - 3.7 after the group score map (Eq. 4 to Eq. 10): from
 * S of layer `layer`: s_bar, g*, online MI per group (Eq. 5) -> EMA (Eq. 6) ->
 * prior w (Eq. 7) -> beta; phi_g and the m_g update (Eq. 8) -> D_t (Eq. 9);
 * H_hat and T (Sec. 3.6); s_t = max(s_bar beta D, 0)^(1/T); global top-B with
 * ties to the lower index -> idx ascending (per-KV-head mode: each group's own
 * scores and top-B, see the top of this file).  Writes idx, and score / stats
 * when non-NULL.  Advances this layer's state by one step (n += 1 and both
 * EMAs). */
starkv_status starkv_select(starkv_state* st, int32_t layer, const starkv_seq* seqs,
                            int32_t nseq, void* workspace, size_t workspace_bytes, void* stream);

/* Sec. 3.7, Eq. (11): K' = [K_past[I]; K_rec], V' = [V_past[I]; V_rec] and the
 * same gather of meta, for layer `layer`, from idx.  Bit copies.  In the
 * per-KV-head mode group g gathers its own rows idx[g] (and meta_out[g]). */
starkv_status starkv_compact(starkv_state* st, int32_t layer, const starkv_seq* seqs,
                             int32_t nseq, void* workspace, size_t workspace_bytes, void* stream);

/* Whole compression step of every layer of every sequence (Algorithm 1 for all
 * layers): score, select, compact.  S may be NULL (workspace is used).
 * Equivalent to calling the three per-layer calls for each layer in order. */
starkv_status starkv_step(starkv_state* st, const starkv_seq* seqs, int32_t nseq,
                          void* workspace, size_t workspace_bytes, void* stream);

/* starkv_step with every pointer in `seqs` a HOST pointer (page-locked memory
 * gives asynchronous copies): copies k, v, q, meta to device staging inside
 * `workspace` (size from starkv_workspace_bytes(..., host = 1, ...)), runs the
 * step, and copies k_out, v_out, meta_out, idx (and score / stats / S when
 * non-NULL) back.  Stream-ordered: the host outputs are valid after the stream
 * is synchronised. */
starkv_status starkv_step_host(starkv_state* st, const starkv_seq* seqs, int32_t nseq,
                               void* workspace, size_t workspace_bytes, void* stream);

/* Reads and clears the state's device error word (synchronises `stream`).
 * Returns STARKV_OK, STARKV_ERR_DEVICE or STARKV_ERR_TIMEOUT. */
starkv_status starkv_check_device_error(starkv_state* st, void* stream);

/* Limit, in nanoseconds, of every bounded device-side wait of this state's
 * kernels (default 1e9).  A wait that runs out stops its kernel early and
 * latches STARKV_ERR_TIMEOUT in the device error word; before it exits or
 * releases tensor memory the kernel still waits for the copies and MMAs it
 * has already issued, for max(limit, 2 s). */
starkv_status starkv_set_wait_limit(starkv_state* st, uint64_t limit_ns);

/* Self-test of the failure path that every bounded device wait shares: one
 * thread of a one-block kernel waits on a shared-memory barrier that nothing
 * completes; after `limit_ns` (1e3 .. 1e9) the wait gives up, latches
 * STARKV_ERR_TIMEOUT in the state's device error word and the kernel
 * returns, so the context stays usable.  Stream-ordered; the next
 * starkv_check_device_error reports STARKV_ERR_TIMEOUT (and clears it).
 * STARKV_ERR_INVALID_ARG for a NULL state or a limit out of range. */
starkv_status starkv_selftest_wait(starkv_state* st, uint64_t limit_ns, void* stream);

/* Kernels of the library, for starkv_kernel_times. */
enum {
  STARKV_KERNEL_SCORE_LSE = 0,    /* scoring pass 1: per-row log-sum-exp (Sec. 3.3)        */
  STARKV_KERNEL_SCORE_ACCUM = 1,  /* scoring pass 2: normalised group sums (Eqs. 2-4)      */
  STARKV_KERNEL_POOL = 2,         /* AvgPool1D + group mean (Eqs. 3-4), per-layer calls    */
  STARKV_KERNEL_CALIBRATE = 3,    /* MI, phi, prior, temperature, fused score, top-B
                                     (Sec. 3.4-3.7): one cluster of min(G, 8) CTAs per
                                     layer                                                 */
  STARKV_KERNEL_COMPACT = 4,      /* KV gather (Eq. 11)                                    */
  STARKV_KERNEL_ATTENTION = 5,    /* window-row attention over the past keys (pieces)      */
  STARKV_KERNEL_ATTN_COMBINE = 6, /* merge of its pieces into attn_o / attn_lse            */
  STARKV_NUM_KERNELS = 7
};

/* Kernel timing, a profiling aid.  While `on` is non-zero every kernel launch
 * made for this state is bracketed by a CUDA event pair on its stream. */
starkv_status starkv_set_timing(starkv_state* st, int32_t on);

/* Per kernel kind (arrays of STARKV_NUM_KERNELS): launches made and, while
 * timing was on, their summed device time in milliseconds, since the last
 * call.  Waits for the recorded events.  Launch counts are kept with timing
 * off too (total_ms then stays 0).  Either array may be NULL. */
starkv_status starkv_kernel_times(starkv_state* st, int64_t* launches, float* total_ms);

/* Thread-local message describing the last non-OK status on this thread. */
const char* starkv_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* STARKV_H */
