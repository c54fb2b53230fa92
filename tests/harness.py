"""Shared test helpers: hyper-parameters for both sides, device inputs, the
oracle per layer, and the comparison rules (fused scores within 1e-3
relative, index sets equal except ties inside that band, compaction bit-exact).
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Dict, List, Optional

import numpy as np
import torch

from oracle import starkv_oracle as O
from paper_2606_01790_gb300 import starkv as sk
from paper_2606_01790_gb300 import synthetic as syn

RTOL = 1e-3          # fused scores, relative (fp32 accumulation from bf16 inputs)
FLOOR = 1e-6         # absolute floor, times max |score|
GSTAR_TIE = 1e-5     # tokens whose top-two S[g, t] are this close may take either g*


def hyper(**over) -> Dict:
    """One set of hyper-parameters, given to both sides explicitly."""
    h = dict(lam=0.5, tau=1.0, rho_mi=0.9, n_warmup=5, n_ramp=10, delta=0.2, d_min=0.1,
             rho_t=0.9, t_min=0.95, t_max=1.05, pool_kernel=5, mi_bins=8, mi_grid=8,
             eps=1e-6, eps_h=1e-12, decay_mode=0, aeb_mode=0, mi_span=0)
    h.update(over)
    return h


def oracle_params(h: Dict) -> O.Params:
    return O.Params(**h)


def gpu_config(wl: syn.Workload, h: Dict, n_layers: Optional[int] = None, max_seqs: int = 1,
               per_head: bool = False) -> sk.Config:
    return sk.Config(n_layers=n_layers or wl.n_layers, n_heads=wl.n_heads, n_kv_heads=wl.n_kv_heads,
                     head_dim=wl.head_dim, window=wl.window, grid_rows=wl.grid_rows,
                     grid_cols=wl.grid_cols, pool_kernel=h["pool_kernel"], mi_bins=h["mi_bins"],
                     mi_grid=h["mi_grid"], n_warmup=h["n_warmup"], n_ramp=h["n_ramp"],
                     max_seqs=max_seqs, lambda_=h["lam"], tau=h["tau"], rho_mi=h["rho_mi"],
                     rho_t=h["rho_t"], delta=h["delta"], d_min=h["d_min"], t_min=h["t_min"],
                     t_max=h["t_max"], eps=h["eps"], eps_h=h["eps_h"], decay_mode=h["decay_mode"],
                     aeb_mode=h["aeb_mode"], mi_span=h["mi_span"],
                     select_mode=sk.SELECT_PER_HEAD if per_head else sk.SELECT_GLOBAL)


@dataclass
class DevSeq:
    seq: sk.Seq
    si: syn.SeqInput


def _words(lay) -> np.ndarray:
    """Metadata words of one layer: [L], or [G][L] for per-group layouts."""
    if isinstance(lay, list):
        return np.stack([_words(x) for x in lay])
    return sk.pack_meta(lay.is_visual, lay.frame, lay.row, lay.col)


def layer_meta(lay, field: str) -> np.ndarray:
    """One metadata field of a layer: [L] or [G][L]."""
    if isinstance(lay, list):
        return np.stack([getattr(x, field) for x in lay])
    return getattr(lay, field)


def device_seq(si: syn.SeqInput, wl: syn.Workload, slot: int = 0, dev="cuda",
               with_S: bool = True, with_score: bool = True, with_stats: bool = True,
               per_head: bool = False) -> DevSeq:
    """Device buffers of one sequence; per_head sizes idx / score / meta_out with
    one row per KV group.  Per-group layouts give [n_layers][G][L] metadata."""
    nl, G, w, d = si.k.shape[0], wl.n_kv_heads, wl.window, wl.head_dim
    L, B = si.L, si.budget
    lp = L - w
    P = G if per_head else 1
    words = np.stack([_words(l) for l in si.layout])
    grouped = words.ndim == 3
    if grouped and not per_head:
        raise ValueError("per-group metadata needs the per-KV-head mode")
    seq = sk.Seq(k=si.k.to(dev), v=si.v.to(dev), q=si.q.to(dev),
                 meta=sk.meta_tensor(words).to(dev), meta_layer_stride=(G * L if grouped else L),
                 meta_group_stride=(L if grouped else 0), L=L,
                 cur_frame=si.cur_frame, budget=B, slot=slot,
                 k_out=torch.empty((nl, G, B + w, d), dtype=torch.bfloat16, device=dev),
                 v_out=torch.empty((nl, G, B + w, d), dtype=torch.bfloat16, device=dev),
                 meta_out=torch.empty((nl, P, B + w) if per_head else (nl, B + w), dtype=torch.int32,
                                      device=dev),
                 idx=torch.empty((nl, P, max(B, 0)) if per_head else (nl, max(B, 0)), dtype=torch.int32,
                                 device=dev),
                 S=torch.empty((nl, G, lp), dtype=torch.float32, device=dev) if with_S else None,
                 score=torch.empty((nl, P, lp) if per_head else (nl, lp), dtype=torch.float32, device=dev)
                 if with_score else None,
                 stats=torch.empty((nl, sk.stats_stride(G)), dtype=torch.float32, device=dev)
                 if with_stats else None)
    return DevSeq(seq, si)


def oracle_layer(si: syn.SeqInput, layer: int, wl: syn.Workload, st: O.LayerState, p: O.Params,
                 S_override: Optional[np.ndarray] = None, per_head: bool = False) -> Dict:
    """Algorithm 1 for one layer of one sequence; ``S_override`` skips scoring
    and feeds the given group score map to the calibration/selection steps."""
    lay = si.layout[layer]
    lp = si.L - wl.window
    if S_override is None:
        S = O.score_layer(si.q[layer].double().numpy(), si.k[layer].double().numpy(), wl.window, p)
    else:
        S = S_override
    meta = tuple(layer_meta(lay, f) for f in ("is_visual", "frame", "row", "col"))
    sel = O.select_layer_per_head if per_head else O.select_layer
    out = sel(S, *meta, si.cur_frame, si.budget, wl.grid_rows, wl.grid_cols, st, p)
    out["S"] = S
    out["lp"] = lp
    return out


def near_tie_tokens(S: np.ndarray, tol: float = GSTAR_TIE) -> np.ndarray:
    """Tokens whose two largest group scores are within ``tol`` relative."""
    if S.shape[0] < 2:
        return np.zeros(S.shape[1], bool)
    top2 = np.sort(S, axis=0)[-2:]
    return (top2[1] - top2[0]) <= tol * np.abs(top2[1])


def score_tolerance_ok(gpu: np.ndarray, ref: np.ndarray, rtol: float = RTOL) -> np.ndarray:
    floor = FLOOR * np.abs(ref).max() if ref.size else 0.0
    return np.abs(gpu - ref) <= rtol * np.abs(ref) + floor


def alt_scores(out: Dict, S: np.ndarray, si: syn.SeqInput, layer: int, wl: syn.Workload,
               p: O.Params) -> np.ndarray:
    """Oracle fused score with g* taken as the second-best group (for near ties)."""
    lay = si.layout[layer]
    lp = S.shape[1]
    gs2 = np.argsort(S, axis=0, kind="stable")[-2]
    beta = O.mi_weight(gs2, out["w"], out["lam"])
    d = O.temporal_decay(lay.is_visual[:lp], lay.frame[:lp], si.cur_frame, out["phi"][gs2],
                         p.delta, p.d_min)
    return O.final_score(out["sbar"], beta, d, out["T"])


def check_scores(gpu: np.ndarray, out: Dict, S_ref: np.ndarray, si, layer, wl, p,
                 rtol: float = RTOL) -> Dict:
    ref = out["score"]
    ok = score_tolerance_ok(gpu, ref, rtol)
    ties = near_tie_tokens(S_ref)
    if (~ok & ties).any():
        ok |= ties & score_tolerance_ok(gpu, alt_scores(out, S_ref, si, layer, wl, p), rtol)
    bad = np.nonzero(~ok)[0]
    rel = np.abs(gpu - ref) / np.maximum(np.abs(ref), 1e-30)
    return dict(ok=len(bad) == 0, bad=bad, max_rel=float(rel[ok].max()) if ok.any() else 0.0,
                n_tie_exempt=int((ties & ~score_tolerance_ok(gpu, ref, rtol)).sum()))


def check_index_set(gpu_idx: np.ndarray, ref: Dict, B: int, rtol: float = RTOL) -> Dict:
    """Index sets equal except tokens whose oracle score lies within ``rtol``
    relative of the oracle's B-th largest score."""
    ref_idx = ref["idx"]
    assert gpu_idx.shape[0] == B
    assert np.all(np.diff(gpu_idx) > 0), "indices must be strictly ascending"
    if B == 0:
        return dict(ok=True, n_diff=0)
    score = ref["score"]
    kth = np.sort(score)[::-1][B - 1]
    diff = np.setxor1d(gpu_idx, ref_idx)
    bad = [t for t in diff if abs(score[t] - kth) > rtol * abs(kth)]
    return dict(ok=not bad, n_diff=len(diff), bad=bad)


def check_compaction(seq: sk.Seq, si: syn.SeqInput, layer: int, w: int) -> None:
    """K', V', meta' are bit copies of the rows the GPU's own index set names."""
    idx = seq.idx[layer].cpu().long()
    lp = si.L - w
    rows = torch.cat([idx, torch.arange(lp, si.L)])
    k_ref = si.k[layer].index_select(1, rows)
    v_ref = si.v[layer].index_select(1, rows)
    assert torch.equal(seq.k_out[layer].cpu(), k_ref), "K' is not a bit copy"
    assert torch.equal(seq.v_out[layer].cpu(), v_ref), "V' is not a bit copy"
    lay = si.layout[layer]
    words = sk.pack_meta(lay.is_visual, lay.frame, lay.row, lay.col)[rows.numpy()]
    got = seq.meta_out[layer].cpu().numpy().view(np.uint32)
    assert np.array_equal(got, words), "meta' is not a bit copy"


def check_per_head(seq: sk.Seq, si: syn.SeqInput, layer: int, wl: syn.Workload, ref: Dict,
                   rtol: float = RTOL) -> Dict:
    """Per-KV-head mode: each group's fused scores within ``rtol`` relative, its
    index set equal except ties inside that band, and K', V', meta' of group g
    bit copies of the rows its own index set names."""
    G, w, B = wl.n_kv_heads, wl.window, si.budget
    lp = si.L - w
    out = dict(max_rel=0.0, n_diff=0)
    words = _words(si.layout[layer])
    if words.ndim == 1:
        words = np.tile(words, (G, 1))
    score = seq.score[layer].double().cpu().numpy() if seq.score is not None else None
    for g in range(G):
        if score is not None:
            ok = score_tolerance_ok(score[g], ref["score"][g], rtol)
            assert ok.all(), (layer, g, np.nonzero(~ok)[0][:10])
            rel = np.abs(score[g] - ref["score"][g]) / np.maximum(np.abs(ref["score"][g]), 1e-30)
            out["max_rel"] = max(out["max_rel"], float(rel.max()) if rel.size else 0.0)
        gi = seq.idx[layer][g].cpu().numpy()
        ix = check_index_set(gi, dict(idx=ref["idx"][g], score=ref["score"][g]), B, rtol)
        assert ix["ok"], (layer, g, ix)
        out["n_diff"] += ix["n_diff"]
        rows = torch.cat([torch.from_numpy(gi.astype(np.int64)), torch.arange(lp, si.L)])
        assert torch.equal(seq.k_out[layer][g].cpu(), si.k[layer][g].index_select(0, rows)), "K' group copy"
        assert torch.equal(seq.v_out[layer][g].cpu(), si.v[layer][g].index_select(0, rows)), "V' group copy"
        got = seq.meta_out[layer][g].cpu().numpy().view(np.uint32)
        assert np.array_equal(got, words[g][rows.numpy()]), "meta' group copy"
    return out
