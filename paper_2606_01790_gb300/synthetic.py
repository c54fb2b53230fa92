"""Seeded synthetic GUI-trajectory workloads for the STaR-KV compression stage.

This module is the one piece shared by the CUDA path's callers (tests,
``bench.py``) and the fp64 oracle: it draws inputs and nothing else.  It holds
none of the compression method's arithmetic (no attention, pooling, mutual
information, temporal decay, entropy or selection).

What the inputs look like (the paper runs UI-TARS-1.5-7B on GUI benchmarks,
Sec. 4.1; none of those datasets or weights exist here, so these draws stand in
for them):

* GQA shape of UI-TARS-1.5-7B: H = 28 query heads, G = 4 KV heads, d = 128,
  bf16 (Sec. 3.1, App. A.1).
* Token stream (Sec. 3.1): text runs interleaved with screenshots,
  ``[txt_0, shot_0, txt_1, ..., shot_{n-1}, txt_n]``; the last text run is at
  least ``w`` long so that the last ``w`` tokens (the observation window and
  recent window) are text.  Visual tokens of a screenshot are row-major over an
  R x C merged-patch grid; frame ids are absolute.
* Values: Q, K, V ~ N(0, 1).  For each (layer, KV group) there is a random unit
  key direction ``u`` and a Gaussian "spatial bump" centred at a random patch
  (distinct centres per group); visual keys get
  ``K += A * exp(-dist^2 / (2 sigma^2)) * u`` with sigma = 3 patches, A = 2.
  Window queries of heads in group g get ``Q += sqrt(d) * u`` so that the bump
  lifts logits by about A at its centre.
* fp32 draws are rounded to bf16 with round-to-nearest-even (torch).

Random streams are keyed by ``SeedSequence([seed, cfg_id, seq, layer, tag])``
so that any single (sequence, layer) can be regenerated on its own.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass, field
from typing import Dict, List, Optional, Tuple

import numpy as np
import torch

# stream tags (arbitrary distinct integers)
_TAG_DIR = 0xD1
_TAG_CENTRE = 0xCE
_TAG_AMP = 0xA3
_TAG_SEQ = 0x5E


@dataclass(frozen=True)
class Workload:
    """Shape of one synthetic workload (all sequences share the model shape)."""

    name: str
    cfg_id: int
    n_layers: int
    n_heads: int = 28
    n_kv_heads: int = 4
    head_dim: int = 128
    window: int = 32
    grid_rows: int = 52
    grid_cols: int = 52
    n_shots: int = 5
    n_text: int = 512
    budget_pct: int = 20
    amp: float = 2.0
    amp_range: Optional[Tuple[float, float]] = None   # per-frame U[a, b] amplitude
    sigma: float = 3.0
    n_seqs: int = 1
    steps: int = 1                 # trajectory steps (config 3)
    step_text: int = 64            # text tokens appended per trajectory step
    ragged: bool = False           # per-sequence shots / text / budget draws (config 5)
    shots_range: Tuple[int, int] = (1, 12)
    text_range: Tuple[int, int] = (128, 1024)
    pct_choices: Tuple[int, ...] = (10, 20, 30)
    # MHA-head granularity on a GQA model (the ablation of the MI prior's
    # granularity in Sec. 4.2): keys and values are drawn for this many groups and each
    # group's rows are replicated for its n_kv_heads / kv_source_groups query
    # heads, so that every query head has its own KV head (0: no replication)
    kv_source_groups: int = 0

    @property
    def visual_per_shot(self) -> int:
        return self.grid_rows * self.grid_cols


# The five workloads of the benchmark definition plus the per-step bench shape.
WORKLOADS: Dict[str, Workload] = {
    # 1 layer, 64 text + 2 x 16x16 screenshots, w = 8, B = 20% of 512 visual = 102.
    "tiny": Workload("tiny", 1, n_layers=1, window=8, grid_rows=16, grid_cols=16,
                     n_shots=2, n_text=64),
    # 1 layer, 5 x 2704 (52x52) + 512 text, w = 32, B = 2704.
    "uitars_layer": Workload("uitars_layer", 2, n_layers=1),
    # 28 layers x the 5-screenshot shape, 10 steps, +1 screenshot + 64 text per step.
    "trajectory": Workload("trajectory", 3, n_layers=28, steps=10),
    # 28 layers, 20 screenshots + 2048 text (L_p = 56,096), amplitude U[0.5, 4] per frame.
    "long": Workload("long", 4, n_layers=28, n_shots=20, n_text=2048,
                     amp_range=(0.5, 4.0)),
    # one layer of the long shape (parity case for rows longer than the
    # calibration kernel keeps on chip)
    "long_layer": Workload("long_layer", 7, n_layers=1, n_shots=20, n_text=2048,
                           amp_range=(0.5, 4.0)),
    # 16 ragged trajectories, 28 layers.
    "ragged": Workload("ragged", 5, n_layers=28, n_seqs=16, ragged=True),
    # the timed per-step workload: 28 layers of the 5-screenshot UI-TARS shape
    "uitars_5shot_28l": Workload("uitars_5shot_28l", 6, n_layers=28),
    # the same step at MHA-head granularity: the 4 groups' keys and values
    # replicated for each of the 28 query heads (G = H = 28)
    "uitars_5shot_28l_mha": Workload("uitars_5shot_28l_mha", 6, n_layers=28, n_kv_heads=28,
                                     kv_source_groups=4),
    # one layer of that shape, and the tiny case at MHA-head granularity
    "uitars_layer_mha": Workload("uitars_layer_mha", 2, n_layers=1, n_kv_heads=28, kv_source_groups=4),
    "tiny_mha": Workload("tiny_mha", 1, n_layers=1, window=8, grid_rows=16, grid_cols=16,
                         n_shots=2, n_text=64, n_kv_heads=28, kv_source_groups=4),
}


@dataclass
class TokenLayout:
    """Per-token metadata of one cache (unpacked)."""

    is_visual: np.ndarray   # int32 0/1 [L]
    frame: np.ndarray       # int32 [L]  (absolute frame id; 0 for text)
    row: np.ndarray         # int32 [L]
    col: np.ndarray         # int32 [L]

    @property
    def L(self) -> int:
        return int(self.is_visual.shape[0])

    def take(self, idx: np.ndarray) -> "TokenLayout":
        return TokenLayout(self.is_visual[idx], self.frame[idx], self.row[idx], self.col[idx])

    @staticmethod
    def concat(parts: List["TokenLayout"]) -> "TokenLayout":
        return TokenLayout(*[np.concatenate([getattr(p, f) for p in parts]).astype(np.int32)
                             for f in ("is_visual", "frame", "row", "col")])


def text_runs(n_text: int, n_shots: int, window: int) -> List[int]:
    """Split ``n_text`` text tokens into ``n_shots + 1`` runs, last run >= window."""
    if n_text < window:
        raise ValueError(f"need at least window={window} text tokens, got {n_text}")
    runs = [n_text // (n_shots + 1)] * (n_shots + 1)
    runs[-1] += n_text - sum(runs)
    deficit = window - runs[-1]
    i = 0
    while deficit > 0:
        take = min(deficit, runs[i])
        runs[i] -= take
        runs[-1] += take
        deficit -= take
        i += 1
    return runs


def token_layout(n_shots: int, n_text: int, R: int, C: int, window: int,
                 frame0: int = 0) -> TokenLayout:
    runs = text_runs(n_text, n_shots, window)
    parts = []
    j = np.arange(R * C, dtype=np.int32)
    for s in range(n_shots + 1):
        n = runs[s]
        z = np.zeros(n, np.int32)
        parts.append(TokenLayout(z, z, z, z))
        if s < n_shots:
            parts.append(TokenLayout(np.ones(R * C, np.int32),
                                     np.full(R * C, frame0 + s, np.int32),
                                     (j // C).astype(np.int32), (j % C).astype(np.int32)))
    return TokenLayout.concat(parts)


def _rng(*key: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(k) for k in key])))


def to_bf16(x: np.ndarray) -> torch.Tensor:
    """fp32 -> bf16, round-to-nearest-even."""
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)


def directions(seed: int, wl: Workload, seq: int, layer: int) -> np.ndarray:
    """Unit key directions u[g] for one (sequence, layer): [G][d] fp32."""
    r = _rng(seed, wl.cfg_id, seq, layer, _TAG_DIR)
    u = r.standard_normal((wl.n_kv_heads, wl.head_dim)).astype(np.float64)
    u /= np.linalg.norm(u, axis=1, keepdims=True)
    return u.astype(np.float32)


def centres(seed: int, wl: Workload, seq: int, layer: int, step: int) -> np.ndarray:
    """Bump centres [G][2] (row, col) at trajectory step ``step``.

    Step 0 centres are uniform on the grid and distinct per group; each later
    step moves every centre by a random {-1, 0, 1} patch in row and column,
    clamped to the grid.
    """
    r = _rng(seed, wl.cfg_id, seq, layer, _TAG_CENTRE)
    R, C = wl.grid_rows, wl.grid_cols
    cs: List[Tuple[int, int]] = []
    while len(cs) < wl.n_kv_heads:
        c = (int(r.integers(0, R)), int(r.integers(0, C)))
        if c not in cs or len(cs) >= R * C:
            cs.append(c)
    out = np.array(cs, np.int64)
    for _ in range(step):
        out = out + r.integers(-1, 2, size=out.shape)
        out[:, 0] = np.clip(out[:, 0], 0, R - 1)
        out[:, 1] = np.clip(out[:, 1], 0, C - 1)
    return out


def frame_amplitude(seed: int, wl: Workload, seq: int, frame: int) -> float:
    if wl.amp_range is None:
        return float(wl.amp)
    r = _rng(seed, wl.cfg_id, seq, frame, _TAG_AMP)
    return float(r.uniform(*wl.amp_range))


@dataclass
class SeqShape:
    """Per-sequence shape (ragged batches draw these per sequence)."""

    n_shots: int
    n_text: int
    budget_pct: int


def seq_shape(seed: int, wl: Workload, seq: int) -> SeqShape:
    if not wl.ragged:
        return SeqShape(wl.n_shots, wl.n_text, wl.budget_pct)
    r = _rng(seed, wl.cfg_id, seq, _TAG_SEQ)
    return SeqShape(int(r.integers(wl.shots_range[0], wl.shots_range[1] + 1)),
                    int(r.integers(wl.text_range[0], wl.text_range[1] + 1)),
                    int(r.choice(np.array(wl.pct_choices))))


def budget(pct: int, n_visual_history: int, l_past: int) -> int:
    """Historical-token budget B: an integer ``pct`` percent of the visual tokens
    the uncompressed history holds, capped at the number of scoreable tokens."""
    return min((pct * n_visual_history) // 100, l_past)


@dataclass
class SeqInput:
    """One sequence's inputs for one compression call (all layers)."""

    q: torch.Tensor            # bf16 [n_layers][H][w][d]
    k: torch.Tensor            # bf16 [n_layers][G][L][d]
    v: torch.Tensor            # bf16 [n_layers][G][L][d]
    layout: list               # per layer: a TokenLayout (identical for a fresh
                               # sequence), or G of them, one per KV group, after
                               # a per-KV-head compaction
    cur_frame: int
    budget: int
    n_visual_history: int

    @property
    def L(self) -> int:
        return int(self.k.shape[2])


def _keys_for(seed: int, wl: Workload, seq: int, layer: int, step: int,
              lay: TokenLayout, r: np.random.Generator) -> Tuple[np.ndarray, np.ndarray]:
    G, d = wl.n_kv_heads, wl.head_dim
    L = lay.L
    k = r.standard_normal((G, L, d), dtype=np.float32)
    v = r.standard_normal((G, L, d), dtype=np.float32)
    vis = lay.is_visual.astype(bool)
    if vis.any():
        u = directions(seed, wl, seq, layer)
        cen = centres(seed, wl, seq, layer, step)
        rows = lay.row[vis].astype(np.float32)
        cols = lay.col[vis].astype(np.float32)
        frames = lay.frame[vis]
        uniq, inv = np.unique(frames, return_inverse=True)
        amp = np.array([frame_amplitude(seed, wl, seq, int(f)) for f in uniq], np.float32)
        a = amp[inv]
        where = np.nonzero(vis)[0]
        for g in range(G):
            dist2 = (rows - cen[g, 0]) ** 2 + (cols - cen[g, 1]) ** 2
            bump = a * np.exp(-dist2 / (2.0 * wl.sigma ** 2)).astype(np.float32)
            k[g, where] += bump[:, None] * u[g][None, :]
    return k, v


def _queries_for(seed: int, wl: Workload, seq: int, layer: int,
                 r: np.random.Generator) -> np.ndarray:
    H, G, w, d = wl.n_heads, wl.n_kv_heads, wl.window, wl.head_dim
    q = r.standard_normal((H, w, d), dtype=np.float32)
    u = directions(seed, wl, seq, layer)
    heads_per_group = H // G
    for h in range(H):
        q[h] += np.sqrt(d) * u[h // heads_per_group][None, :]
    return q


def _parallel(fn, items):
    """Run ``fn`` over ``items`` on a thread pool (numpy releases the GIL while
    drawing; every item owns its own seeded stream, so results do not depend
    on the thread count)."""
    import concurrent.futures as cf
    import os
    n = min(len(items), os.cpu_count() or 1)
    if n <= 1:
        return [fn(i) for i in items]
    with cf.ThreadPoolExecutor(n) as ex:
        return list(ex.map(fn, items))


def make_sequence(wl: Workload, seq: int = 0, seed: int = 0,
                  layers: Optional[List[int]] = None) -> SeqInput:
    """Fresh (step 0) input of sequence ``seq``: the uncompressed history.

    ``layers`` restricts generation to a subset (the result is then stacked in
    that order); by default all ``wl.n_layers`` layers are drawn.
    """
    if wl.kv_source_groups:
        # draw the GQA model's keys and values, then give every query head its own copy
        src = dataclasses.replace(wl, n_kv_heads=wl.kv_source_groups, kv_source_groups=0)
        si = make_sequence(src, seq=seq, seed=seed, layers=layers)
        rep = wl.n_kv_heads // wl.kv_source_groups
        si.k = si.k.repeat_interleave(rep, dim=1)
        si.v = si.v.repeat_interleave(rep, dim=1)
        return si
    sh = seq_shape(seed, wl, seq)
    lay = token_layout(sh.n_shots, sh.n_text, wl.grid_rows, wl.grid_cols, wl.window)
    layers = list(range(wl.n_layers)) if layers is None else list(layers)
    nl, G, H, w, d, L = len(layers), wl.n_kv_heads, wl.n_heads, wl.window, wl.head_dim, lay.L
    q_out = torch.empty((nl, H, w, d), dtype=torch.bfloat16)
    k_out = torch.empty((nl, G, L, d), dtype=torch.bfloat16)
    v_out = torch.empty((nl, G, L, d), dtype=torch.bfloat16)

    def one(i):
        l = layers[i]
        r = _rng(seed, wl.cfg_id, seq, l, 0)
        k, v = _keys_for(seed, wl, seq, l, 0, lay, r)
        q = _queries_for(seed, wl, seq, l, r)
        k_out[i].copy_(to_bf16(k)); v_out[i].copy_(to_bf16(v)); q_out[i].copy_(to_bf16(q))

    _parallel(one, list(range(nl)))
    n_vis = sh.n_shots * wl.visual_per_shot
    l_past = lay.L - wl.window
    return SeqInput(q=q_out, k=k_out, v=v_out, layout=[lay] * nl, cur_frame=max(sh.n_shots - 1, 0),
                    budget=budget(sh.budget_pct, n_vis, l_past), n_visual_history=n_vis)


def append_step(wl: Workload, prev_k: torch.Tensor, prev_v: torch.Tensor,
                prev_layout: List[TokenLayout], step: int, n_visual_history: int,
                seq: int = 0, seed: int = 0, budget_pct: Optional[int] = None,
                layers: Optional[List[int]] = None) -> SeqInput:
    """Trajectory step ``step`` >= 1: append one screenshot (frame = previous
    newest frame + 1) and ``wl.step_text`` text tokens to each layer's compressed
    cache ``prev_k``/``prev_v`` ([n_layers][G][B+w][d]) and draw fresh window
    queries.  Bump centres drift by one random patch per step.  A layer whose
    ``prev_layout`` is a list of per-group layouts keeps one per group."""
    layers = list(range(wl.n_layers)) if layers is None else list(layers)
    flat = [x for lay in prev_layout for x in (lay if isinstance(lay, list) else [lay])]
    newest = max(int(lay.frame[lay.is_visual.astype(bool)].max()) if lay.is_visual.any() else -1
                 for lay in flat)
    frame = newest + 1
    R, C = wl.grid_rows, wl.grid_cols
    j = np.arange(R * C, dtype=np.int32)
    z = np.zeros(wl.step_text, np.int32)
    new_lay = TokenLayout.concat([
        TokenLayout(np.ones(R * C, np.int32), np.full(R * C, frame, np.int32),
                    (j // C).astype(np.int32), (j % C).astype(np.int32)),
        TokenLayout(z, z, z, z)])
    qs, ks, vs, lays = [], [], [], []
    for i, l in enumerate(layers):
        r = _rng(seed, wl.cfg_id, seq, l, step)
        k_new, v_new = _keys_for(seed, wl, seq, l, step, new_lay, r)
        q = _queries_for(seed, wl, seq, l, r)
        qs.append(q)
        ks.append(torch.cat([prev_k[i], to_bf16(k_new)], dim=1))
        vs.append(torch.cat([prev_v[i], to_bf16(v_new)], dim=1))
        prev = prev_layout[i]
        if isinstance(prev, list):
            lays.append([TokenLayout.concat([pg, new_lay]) for pg in prev])
        else:
            lays.append(TokenLayout.concat([prev, new_lay]))
    n_vis = n_visual_history + R * C
    pct = wl.budget_pct if budget_pct is None else budget_pct
    l_past = ks[0].shape[1] - wl.window
    return SeqInput(q=to_bf16(np.stack(qs)), k=torch.stack(ks), v=torch.stack(vs), layout=lays,
                    cur_frame=frame, budget=budget(pct, n_vis, l_past), n_visual_history=n_vis)


def flush_size_bytes() -> int:
    """Bytes of a buffer larger than the 129 MB L2 of the target GPU."""
    return 256 << 20
