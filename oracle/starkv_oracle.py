"""STaR-KV compression stage: plain, slow, fp64 CPU oracle.

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
module.  It shares no code with the CUDA library and imports nothing from it.

It is organised by the equations it restates: Sec. 3.3 Eqs. 2-4 (window
attention, pooling, group scores), Sec. 3.4 Eqs. 5-7 (spatial MI, its EMA and
the group prior), Sec. 3.5 Eqs. 8-9 (temporal stability and decay), Sec. 3.6
(entropy temperature), Sec. 3.7 Eqs. 10-11 (top-B and compaction); the layer
functions at the end compose them as the paper's Algorithm 1 does as a whole.
Everything runs in float64 from bf16-rounded inputs (upcast exactly).  Library
primitives used as single steps: numpy matmul, exp/log, lexsort, bincount.

Readings of points the paper leaves open (each is a keyword argument or a
parameter with the stated default):

* AvgPool1D (Sec. 3.3): kernel ``pool_kernel`` (odd, default 5), stride 1,
  zero padding of ``pool_kernel // 2`` on both sides, divisor = kernel size.
* The softmax of Sec. 3.3 runs over K_past only (the ``w`` window keys are
  neither scored nor in the normaliser).
* Entropy normaliser ``log L`` of Sec. 3.6 uses L = L_past, so that
  0 <= H <= 1; with L_past <= 1 the entropy is defined as 0.
* RankBin (Sec. 3.4): visual tokens ordered by (S ascending, index ascending),
  rank rho in 0..N-1, bin floor(rho K / N).  SpatialBin: cell
  (floor(r M / R), floor(c M / C)).  The visual span is every historical
  visual token.  Natural logarithm.  No visual tokens: MI = 0.
* The MI EMA starts at the first value (fresh state: MI_bar = MI).
* lambda schedule (Sec. 3.4 last paragraph, App. A.1): n = number of earlier
  steps of this (sequence, layer); lambda_n = 0 for n < n_warmup, then linear
  to lambda over n_ramp steps; n_ramp = 0 jumps to lambda at n_warmup.
* Temporal EMA m_g (Sec. 3.5) lives on the R x C patch grid; the current row
  s_g^(c) is S[g, .] over the visual tokens of the current frame F, summed per
  cell.  Fresh (||m_g|| = 0): phi_g = 0 and m_g <- s_g^(c).  A current frame
  with no visual tokens: phi_g = 0 and m_g unchanged.
* Top-B (Sec. 3.7, Eq. 10): one global token-level set per layer, ties to
  the lower index, returned ascending (the paper sorts the kept indices).
* Method variants of the ablations (Table 3 and the AEB ablation), off by
  default; the paper names them but prints no formula, so each is a reading:
  decay_mode 1 "linear": D = D_min + (1 - D_min) max(0, 1 - delta Df phi);
  decay_mode 2 "gamma" (power law): D = D_min + (1 - D_min) (1 + Df phi)^(-delta)
  (at the defaults it keeps more of old frames than Eq. 9, linear less, as the
  ablation describes them); aeb_mode 1 "confidence": T = T_min + (T_max -
  T_min)(1 - p_max) with p_max = max_t p_t, the peak attention mass;
  mi_span 1: the MI of Sec. 3.4 over the newest frame's visual tokens only.
* Per-KV-head selection (an optional mode; the paper's method is the global
  set above; App. A.3 names head-wise top-K as the SnapKV-style alternative):
  each group g ranks its own row s_{g,t} = max(S[g,t] beta_g D_{g,t}, 0)^(1/T_g)
  with beta_g = (1 - lambda) + lambda G w_g, D_{g,t} from Eq. (9) with phi_g,
  and T_g from the entropy of S[g, .] (Sec. 3.6 on that row); it keeps its own
  B tokens (ties to the lower index), and the compressed cache of group g is
  [X_g[I_g]; X_g,rec] with the metadata gathered per group.  beta_g is one
  factor per row, so in this mode the MI prior scales the scores without
  changing any set; only D changes the ranking.

MI, MI_bar and w of a layer are pinned end to end against scikit-learn and
scipy on small layers, and phi against scipy's cosine; that these are the
paper's values rests on the readings above, which the paper fixes with no
worked example (parity unpinned in that sense only).
"""
from __future__ import annotations

import dataclasses
import math
from dataclasses import dataclass, field
from typing import Dict, List, Optional

import numpy as np


@dataclass
class Params:
    """Hyper-parameters; defaults from App. A.1 and Table 7 (AgentNetBench,
    UI-TARS) unless marked as a reading."""

    lam: float = 0.5          # MI prior strength lambda
    tau: float = 1.0          # prior softmax temperature tau
    rho_mi: float = 0.9       # MI EMA decay rho
    n_warmup: int = 5         # online profiling steps
    n_ramp: int = 10          # lambda ramp steps
    delta: float = 0.2        # temporal decay rate delta
    d_min: float = 0.1        # D_min
    rho_t: float = 0.9        # temporal EMA decay rho_t
    t_min: float = 0.95       # AEB T range
    t_max: float = 1.05
    pool_kernel: int = 5      # reading
    mi_bins: int = 8          # K, reading
    mi_grid: int = 8          # M, reading
    eps: float = 1e-6         # epsilon of the min-max prior, reading
    eps_h: float = 1e-12      # epsilon of the AEB entropy, reading
    decay_mode: int = 0       # 0 exponential (Eq. 9), 1 linear, 2 power law (readings)
    aeb_mode: int = 0         # 0 entropy (Sec. 3.6), 1 peak confidence (reading)
    mi_span: int = 0          # 0 every historical visual token, 1 the newest frame's


# ---------------------------------------------------------------- Sec. 3.1

def head_group(h: int, n_heads: int, n_kv_heads: int) -> int:
    """Sec. 3.1, Eq. (1): query head h attends KV group g(h) = 1 + floor((h-1)G/H)
    (1-indexed), i.e. floor(h G / H) with 0-indexed h and g: contiguous blocks
    of H/G heads (the head range of Eq. (4))."""
    return (h * n_kv_heads) // n_heads


# ---------------------------------------------------------------- Sec. 3.3

def window_lse(q: np.ndarray, k: np.ndarray, window: int) -> np.ndarray:
    """Sec. 3.3, Eq. (2): the softmax normaliser of each window row, as the
    natural-log log-sum-exp of z = Q_{-i,h} . K_past[g(h), t] / sqrt(d) over
    the L_past past keys.  [H][w]; -inf when L_past = 0."""
    H, w, d = q.shape
    G, L, _ = k.shape
    assert w == window
    lp = L - w
    out = np.full((H, w), -np.inf)
    if lp == 0:
        return out
    for h in range(H):
        g = head_group(h, H, G)
        z = (q[h].astype(np.float64) @ k[g, :lp].astype(np.float64).T) / math.sqrt(d)
        m = z.max(axis=1)
        out[h] = m + np.log(np.exp(z - m[:, None]).sum(axis=1))
    return out


def window_attention_given_lse(q: np.ndarray, k: np.ndarray, window: int, lse: np.ndarray) -> np.ndarray:
    """Eq. (2) with the softmax normaliser supplied (the log-sum-exp of each
    window row over K_past, as the layer's own prefill attention pass produces
    it): A_raw[h, t] = sum_i exp(z_{h,i,t} - lse[h, i])."""
    H, w, d = q.shape
    G, L, _ = k.shape
    assert w == window
    lp = L - w
    a_raw = np.zeros((H, lp), np.float64)
    if lp == 0:
        return a_raw
    for h in range(H):
        g = head_group(h, H, G)
        z = (q[h].astype(np.float64) @ k[g, :lp].astype(np.float64).T) / math.sqrt(d)
        a_raw[h] = np.exp(z - lse[h][:, None]).sum(axis=0)
    return a_raw


def window_attention_output(q: np.ndarray, k: np.ndarray, v: np.ndarray, window: int) -> np.ndarray:
    """The attention output of the w window rows over the past keys, the part of
    the layer's own attention pass that computes the logits Eq. (2) scores
    (App. A.3 counts that Q K^T as shared with the attention):
    O[h, i] = sum_t softmax_t(Q_{-i,h} . K_past[g(h), t] / sqrt(d)) V_past[g(h), t]
    over t < L_past, the window keys excluded as in Eq. (2).  [H][w][d]; zeros
    when L_past = 0.  Its softmax normaliser is ``window_lse``."""
    H, w, d = q.shape
    G, L, _ = k.shape
    assert w == window and v.shape == k.shape
    lp = L - w
    out = np.zeros((H, w, d), np.float64)
    if lp == 0:
        return out
    for h in range(H):
        g = head_group(h, H, G)
        z = (q[h].astype(np.float64) @ k[g, :lp].astype(np.float64).T) / math.sqrt(d)   # [w][lp]
        z = z - z.max(axis=1, keepdims=True)
        p = np.exp(z)
        p = p / p.sum(axis=1, keepdims=True)
        out[h] = p @ v[g, :lp].astype(np.float64)
    return out


def window_attention(q: np.ndarray, k: np.ndarray, window: int) -> np.ndarray:
    """Sec. 3.3, Eq. (2): A_raw[h, t] = sum over the w
    window queries of softmax_t(Q_{-i,h} . K_past[g(h), t] / sqrt(d)).

    q: [H][w][d] window queries; k: [G][L][d] keys of the whole cache.
    Returns A_raw [H][L_past] with L_past = L - w.
    """
    H, w, d = q.shape
    G, L, _ = k.shape
    assert w == window
    lp = L - w
    a_raw = np.zeros((H, lp), np.float64)
    if lp == 0:
        return a_raw
    for h in range(H):
        g = head_group(h, H, G)
        z = (q[h].astype(np.float64) @ k[g, :lp].astype(np.float64).T) / math.sqrt(d)  # [w][lp]
        z = z - z.max(axis=1, keepdims=True)
        p = np.exp(z)
        p = p / p.sum(axis=1, keepdims=True)
        a_raw[h] = p.sum(axis=0)
    return a_raw


def avg_pool(a_raw: np.ndarray, kernel: int) -> np.ndarray:
    """Sec. 3.3, Eq. (3): A = AvgPool1D(A_raw) along tokens, per row: stride 1,
    zero padding kernel//2, divisor = kernel (padding counted)."""
    assert kernel >= 1 and kernel % 2 == 1
    rows, lp = a_raw.shape
    half = kernel // 2
    out = np.zeros_like(a_raw)
    for t in range(lp):
        lo, hi = max(0, t - half), min(lp, t + half + 1)
        out[:, t] = a_raw[:, lo:hi].sum(axis=1) / kernel
    return out


def group_scores(a: np.ndarray, n_kv_heads: int) -> np.ndarray:
    """Sec. 3.3, Eq. (4): S[g, t] = (G/H) sum of
    A[h, t] over the H/G heads of group g."""
    H, lp = a.shape
    G = n_kv_heads
    s = np.zeros((G, lp), np.float64)
    for h in range(H):
        s[head_group(h, H, G)] += a[h]
    return s * (G / H)


def base_score(s: np.ndarray) -> np.ndarray:
    """Sec. 3.3, Eq. (4): s_bar_t = (1/G) sum_g S[g, t]."""
    return s.mean(axis=0)


def governing_group(s: np.ndarray) -> np.ndarray:
    """Sec. 3.4: g*(t) = argmax_g S[g, t] (lowest g on exact ties)."""
    return np.argmax(s, axis=0)


# ---------------------------------------------------------------- Sec. 3.6

def entropy_temperature(sbar: np.ndarray, t_min: float, t_max: float,
                        eps_h: float) -> tuple:
    """Sec. 3.6, with the epsilons placed as the paper's Algorithm 1 places
    them: p_t = s_bar_t / (sum s_bar + eps), H = -sum p_t log(p_t + eps) / log L,
    T = T_min + (T_max - T_min) H."""
    lp = sbar.shape[0]
    if lp <= 1:
        h = 0.0
    else:
        z = sbar.sum()
        p = sbar / (z + eps_h)
        h = float(-(p * np.log(p + eps_h)).sum() / math.log(lp))
    return h, t_min + (t_max - t_min) * h


# ---------------------------------------------------------------- Sec. 3.4

def confidence_temperature(sbar: np.ndarray, t_min: float, t_max: float, eps_h: float) -> tuple:
    """The AEB ablation's confidence variant (reading): p_t = s_bar_t /
    (sum s_bar + eps), p_max = max_t p_t, T = T_min + (T_max - T_min)(1 - p_max).
    Returns (p_max, T); no tokens gives p_max = 0."""
    if sbar.shape[0] == 0:
        return 0.0, t_max
    pmax = float(sbar.max() / (sbar.sum() + eps_h))
    return pmax, t_min + (t_max - t_min) * (1.0 - pmax)


def layer_temperature(s: np.ndarray, p: "Params") -> tuple:
    """(H or p_max, T) of one score row by the configured AEB mode."""
    if p.aeb_mode == 1:
        return confidence_temperature(s, p.t_min, p.t_max, p.eps_h)
    return entropy_temperature(s, p.t_min, p.t_max, p.eps_h)


def rank_bins(values: np.ndarray, n_bins: int) -> np.ndarray:
    """Sec. 3.4 RankBin: K equal-frequency bins of the values; ties in value
    broken by position; bin(rho) = floor(rho K / N)."""
    n = values.shape[0]
    order = np.lexsort((np.arange(n), values))      # by value, then position
    rank = np.empty(n, np.int64)
    rank[order] = np.arange(n)
    return (rank * n_bins) // max(n, 1)


def spatial_cells(row: np.ndarray, col: np.ndarray, R: int, C: int, M: int) -> np.ndarray:
    """Sec. 3.4 SpatialBin: patch (r, c) of an R x C grid onto an M x M grid,
    cell index (floor(r M / R)) * M + floor(c M / C)."""
    return (row.astype(np.int64) * M // R) * M + (col.astype(np.int64) * M // C)


def mutual_information(bins: np.ndarray, cells: np.ndarray, n_bins: int, n_cells: int) -> float:
    """Sec. 3.4, Eq. (5): plug-in MI = sum_{b,r,c} p(b,r,c) log(p(b,r,c) / (p(b) p(r,c)))
    from the joint histogram of (bin, cell), natural log."""
    n = bins.shape[0]
    if n == 0:
        return 0.0
    joint = np.bincount(bins * n_cells + cells, minlength=n_bins * n_cells)
    joint = joint.reshape(n_bins, n_cells).astype(np.float64)
    pb = joint.sum(axis=1) / n
    pc = joint.sum(axis=0) / n
    mi = 0.0
    for b in range(n_bins):
        for c in range(n_cells):
            if joint[b, c] > 0:
                p = joint[b, c] / n
                mi += p * math.log(p / (pb[b] * pc[c]))
    return mi


def mi_ema(prev: np.ndarray, mi: np.ndarray, rho: float, fresh: bool) -> np.ndarray:
    """Sec. 3.4, Eq. (6): MI_bar <- rho MI_bar + (1 - rho) MI; fresh state starts at MI."""
    return mi.copy() if fresh else rho * prev + (1.0 - rho) * mi


def subspace_prior(mi_bar: np.ndarray, eps: float, tau: float) -> np.ndarray:
    """Sec. 3.4, Eq. (7): m_g = (MI_bar_g - min) / (max - min + eps), w = softmax(m / tau)."""
    delta = mi_bar - mi_bar.min()
    m = delta / (delta.max() + eps)
    e = np.exp(m / tau - (m / tau).max())
    return e / e.sum()


def lambda_at(n: int, lam: float, n_warmup: int, n_ramp: int) -> float:
    """Sec. 3.4 last paragraph with App. A.1: lambda annealed linearly from 0
    to lambda over the first n_warmup + n_ramp frames (0 during warm-up)."""
    if n < n_warmup:
        return 0.0
    if n_ramp <= 0:
        return lam
    return lam * min(1.0, (n - n_warmup) / n_ramp)


def mi_weight(gstar: np.ndarray, w: np.ndarray, lam_n: float) -> np.ndarray:
    """Eq. (final_score), beta_t = (1 - lambda) + lambda G w_{g*(t)}."""
    G = w.shape[0]
    return (1.0 - lam_n) + lam_n * G * w[gstar]


# ---------------------------------------------------------------- Sec. 3.5

def current_row(s_g: np.ndarray, is_visual: np.ndarray, frame: np.ndarray, row: np.ndarray,
                col: np.ndarray, cur_frame: int, R: int, C: int) -> np.ndarray:
    """Sec. 3.5: s_g^(c), the current-frame part of S[g, .] on the R x C grid."""
    out = np.zeros(R * C, np.float64)
    sel = (is_visual != 0) & (frame == cur_frame)
    np.add.at(out, row[sel].astype(np.int64) * C + col[sel].astype(np.int64), s_g[sel])
    return out


def temporal_stability(cur: np.ndarray, m: np.ndarray, rho_t: float) -> tuple:
    """Sec. 3.5, Eq. (8): phi_g = cos(s_g^(c), m_g), then m_g <- rho_t m_g + (1 - rho_t) s_g^(c).
    Returns (phi, new m)."""
    ncur = math.sqrt(float(cur @ cur))
    nm = math.sqrt(float(m @ m))
    if ncur == 0.0:
        return 0.0, m.copy()
    if nm == 0.0:
        return 0.0, cur.copy()
    phi = float(cur @ m) / (ncur * nm)
    return phi, rho_t * m + (1.0 - rho_t) * cur


def temporal_decay(is_visual: np.ndarray, frame: np.ndarray, cur_frame: int,
                   phi_gstar: np.ndarray, delta: float, d_min: float, mode: int = 0) -> np.ndarray:
    """Sec. 3.5, Eq. (9): D_t = D_min + (1 - D_min) exp(-delta Delta_f(t) phi_{g*(t)})
    for visual t with Delta_f = F - f(t); D_t = 1 for non-visual tokens.
    mode 1 / 2: the linear and power-law readings of Table 3's variants."""
    dist = (cur_frame - frame).astype(np.float64)
    x = dist * phi_gstar
    if mode == 1:
        shape = np.maximum(0.0, 1.0 - delta * x)
    elif mode == 2:
        shape = (1.0 + x) ** (-delta)
    else:
        shape = np.exp(-delta * x)
    d = d_min + (1.0 - d_min) * shape
    return np.where(is_visual != 0, d, 1.0)


# ---------------------------------------------------------------- Eq. final_score, Sec. 3.7

def final_score(sbar: np.ndarray, beta: np.ndarray, d: np.ndarray, temp: float) -> np.ndarray:
    """Eq. (final_score) with Sec. 3.6: s_t = max(s_bar_t beta_t D_t, 0)^(1/T)
    (D_t is already 1 for non-visual tokens)."""
    return np.maximum(sbar * beta * d, 0.0) ** (1.0 / temp)


def top_b(score: np.ndarray, b: int) -> np.ndarray:
    """Sec. 3.7, Eq. (10): the b largest scores,
    ties to the lower index, returned in ascending index order."""
    n = score.shape[0]
    order = np.lexsort((np.arange(n), -score))
    return np.sort(order[:b])


def compact(x: np.ndarray, idx: np.ndarray, window: int) -> np.ndarray:
    """Sec. 3.7, Eq. (11): X' = [X_past[I]; X_rec] along the token axis (axis -2
    for [G][L][d] caches, axis -1 for per-token metadata [L])."""
    if x.ndim == 1:
        lp = x.shape[0] - window
        return np.concatenate([x[idx], x[lp:]])
    lp = x.shape[-2] - window
    return np.concatenate([x[..., idx, :], x[..., lp:, :]], axis=-2)


# ---------------------------------------------------------------- per-layer pipeline

@dataclass
class LayerState:
    """State carried across steps of one trajectory for one layer (reset per
    trajectory, App. A.4)."""

    n: int
    mi_bar: np.ndarray      # [G]
    m: np.ndarray           # [G][R*C]

    @staticmethod
    def fresh(G: int, R: int, C: int) -> "LayerState":
        return LayerState(0, np.zeros(G), np.zeros((G, R * C)))

    def copy(self) -> "LayerState":
        return LayerState(self.n, self.mi_bar.copy(), self.m.copy())


def score_layer(q: np.ndarray, k: np.ndarray, window: int, p: Params,
                lse: Optional[np.ndarray] = None) -> np.ndarray:
    """Sec. 3.3, Eqs. (2)-(4) composed:
    S = group-mean of Pool(sum_i softmax(Q_{-i} K^T / sqrt d)).
    ``lse`` [H][w], when given, is the softmax normaliser of each window row."""
    a_raw = window_attention(q, k, window) if lse is None else window_attention_given_lse(q, k, window, lse)
    a = avg_pool(a_raw, p.pool_kernel)
    return group_scores(a, k.shape[0])


def _group_meta(a: np.ndarray, g: int) -> np.ndarray:
    """Metadata array of group g: a shared [L] array, or row g of a per-group
    [G][L] array (per-KV-head mode after a per-group compaction)."""
    return a[g] if a.ndim == 2 else a


def calibrate_layer(s: np.ndarray, is_visual: np.ndarray, frame: np.ndarray, row: np.ndarray,
                    col: np.ndarray, cur_frame: int, R: int, C: int, st: LayerState,
                    p: Params) -> Dict:
    """The per-group calibration of Sec. 3.4-3.5 (Eqs. 5-8), shared by both
    selection modes:
    MI_g (Eq. 5) -> MI EMA (Eq. 6) -> prior w (Eq. 7) and lambda_n (Sec. 3.4);
    phi_g and the m_g update (Eq. 8).  The metadata arrays are [L] (shared) or
    [G][L] (one row per group).  Does not modify ``st``; returns the new EMAs
    as ``mi_bar`` and ``m_new``."""
    G, lp = s.shape
    n_cells = p.mi_grid * p.mi_grid
    mi = np.zeros(G)
    phi = np.zeros(G)
    m_new = st.m.copy()
    for g in range(G):
        vis_g, fr_g, row_g, col_g = (_group_meta(a, g)[:lp] for a in (is_visual, frame, row, col))
        vis = vis_g != 0
        if p.mi_span == 1:   # the newest frame's visual tokens only
            vis = vis & (fr_g == cur_frame)
        cells = spatial_cells(row_g[vis], col_g[vis], R, C, p.mi_grid)
        mi[g] = mutual_information(rank_bins(s[g][vis], p.mi_bins), cells, p.mi_bins, n_cells)
        cur = current_row(s[g], vis_g, fr_g, row_g, col_g, cur_frame, R, C)
        phi[g], m_new[g] = temporal_stability(cur, st.m[g], p.rho_t)
    mi_bar = mi_ema(st.mi_bar, mi, p.rho_mi, st.n == 0)
    w = subspace_prior(mi_bar, p.eps, p.tau)
    lam_n = lambda_at(st.n, p.lam, p.n_warmup, p.n_ramp)
    return dict(mi=mi, mi_bar=mi_bar, w=w, lam=lam_n, phi=phi, m_new=m_new)


def _advance(st: LayerState, cal: Dict) -> None:
    st.mi_bar, st.m, st.n = cal["mi_bar"], cal["m_new"], st.n + 1


def select_layer(s: np.ndarray, is_visual: np.ndarray, frame: np.ndarray, row: np.ndarray,
                 col: np.ndarray, cur_frame: int, budget: int, R: int, C: int,
                 st: LayerState, p: Params, gstar_override: Optional[np.ndarray] = None) -> Dict:
    """Sec. 3.3 Eq. 4 to Sec. 3.7 Eq. 10 for one layer: from the group score
    map to the index set.

    ``s`` is the group score map S [G][L_past]; the metadata arrays cover the
    L_past historical tokens.  ``st`` is updated in place (MI EMA, m_g, n).
    ``gstar_override`` replaces argmax_g S (for tests of near-tie tokens).
    """
    G, lp = s.shape
    assert is_visual.ndim == 1, "the global mode ranks tokens shared by every group"
    sbar = base_score(s)
    gstar = governing_group(s) if gstar_override is None else gstar_override
    cal = calibrate_layer(s, is_visual, frame, row, col, cur_frame, R, C, st, p)
    # online MI prior (Sec. 3.4)
    beta = mi_weight(gstar, cal["w"], cal["lam"])
    # temporal discount (Sec. 3.5)
    d = temporal_decay(is_visual[:lp], frame[:lp], cur_frame, cal["phi"][gstar], p.delta, p.d_min,
                       p.decay_mode)
    # entropy temperature (Sec. 3.6) and fused score
    h, temp = layer_temperature(sbar, p)
    score = final_score(sbar, beta, d, temp)
    idx = top_b(score, budget)
    _advance(st, cal)
    return dict(sbar=sbar, gstar=gstar, mi=cal["mi"], mi_bar=cal["mi_bar"], w=cal["w"],
                lam=cal["lam"], beta=beta, phi=cal["phi"], D=d, H=h, T=temp, score=score, idx=idx)


def select_layer_per_head(s: np.ndarray, is_visual: np.ndarray, frame: np.ndarray,
                          row: np.ndarray, col: np.ndarray, cur_frame: int, budget: int, R: int,
                          C: int, st: LayerState, p: Params) -> Dict:
    """Per-KV-head selection mode (the SnapKV-style head-wise top-K of App. A.3,
    with the STaR-KV factors of group g): score [G][L_past], idx [G][B], one
    temperature per group.  The metadata arrays are [L] or [G][L] (each group's
    own tokens).  ``st`` is updated in place as in select_layer."""
    G, lp = s.shape
    cal = calibrate_layer(s, is_visual, frame, row, col, cur_frame, R, C, st, p)
    own = np.arange(G)
    beta = mi_weight(own, cal["w"], cal["lam"])                       # [G]
    d = np.stack([temporal_decay(_group_meta(is_visual, g)[:lp], _group_meta(frame, g)[:lp], cur_frame,
                                 np.full(lp, cal["phi"][g]), p.delta, p.d_min, p.decay_mode)
                  for g in range(G)])                                  # [G][L_past]
    ht = [layer_temperature(s[g], p) for g in range(G)]
    h = np.array([x[0] for x in ht])
    temp = np.array([x[1] for x in ht])
    score = np.stack([final_score(s[g], beta[g], d[g], temp[g]) for g in range(G)])
    idx = np.stack([top_b(score[g], budget) for g in range(G)]) if G else np.zeros((0, budget), np.int64)
    _advance(st, cal)
    return dict(mi=cal["mi"], mi_bar=cal["mi_bar"], w=cal["w"], lam=cal["lam"], beta=beta,
                phi=cal["phi"], D=d, H=h, T=temp, score=score, idx=idx)


def compact_per_head(x: np.ndarray, idx: np.ndarray, window: int) -> np.ndarray:
    """Eq. (11) per group: X'[g] = [X[g, I_g]; X[g, L_past:]] for [G][L][d]
    caches, and [G][B + w] metadata gathered per group for [L] or [G][L] arrays."""
    if x.ndim == 1:
        return np.stack([compact(x, idx[g], window) for g in range(idx.shape[0])])
    if x.ndim == 2:   # [G][L] metadata, one row per group
        return np.stack([compact(x[g], idx[g], window) for g in range(idx.shape[0])])
    return np.stack([compact(x[g], idx[g], window) for g in range(x.shape[0])])


def step_layer(q: np.ndarray, k: np.ndarray, v: np.ndarray, is_visual: np.ndarray,
               frame: np.ndarray, row: np.ndarray, col: np.ndarray, cur_frame: int,
               budget: int, window: int, R: int, C: int, st: LayerState, p: Params,
               per_head: bool = False) -> Dict:
    """The whole method for one layer (the paper's Algorithm 1 as a whole):
    scores, calibration, selection and the compressed cache (K', V', metadata'); ``per_head`` picks the per-KV-head
    selection mode (idx [G][B], metadata' [G][B + w])."""
    s = score_layer(q, k, window, p)
    meta = (is_visual, frame, row, col)
    if per_head:
        out = select_layer_per_head(s, *meta, cur_frame, budget, R, C, st, p)
        gather = compact_per_head
    else:
        out = select_layer(s, *meta, cur_frame, budget, R, C, st, p)
        gather = compact
    idx = out["idx"]
    out["S"] = s
    out["k_out"] = gather(k, idx, window)
    out["v_out"] = gather(v, idx, window)
    out["meta_out"] = tuple(gather(a, idx, window) for a in meta)
    return out
