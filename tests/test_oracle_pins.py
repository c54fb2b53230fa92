"""Pins of the fp64 oracle against facts fixed outside it: library routines the
oracle does not call (torch, scipy, scikit-learn), closed forms, invariants the
paper states, and brute force on tiny inputs.  CPU only."""
import math

import numpy as np
import pytest
import scipy.special
import scipy.stats
import torch
import torch.nn.functional as F

from oracle import starkv_oracle as O


def _rng(seed=0):
    return np.random.default_rng(seed)


# ------------------------------------------------------------------ Sec. 3.1

def test_head_group_matches_one_indexed_formula_and_block_ranges():
    for H, G in [(28, 4), (8, 8), (8, 1), (32, 8)]:
        for h1 in range(1, H + 1):  # Eq. (1), 1-indexed
            assert O.head_group(h1 - 1, H, G) == (1 + ((h1 - 1) * G) // H) - 1
        # Eq. (4): group g (1-indexed) owns heads (g-1)H/G .. gH/G - 1
        for g1 in range(1, G + 1):
            heads = [h for h in range(H) if O.head_group(h, H, G) == g1 - 1]
            assert heads == list(range((g1 - 1) * H // G, g1 * H // G))


# ------------------------------------------------------------------ Sec. 3.3

def _torch_window_attention(q, k, w):
    H, G = q.shape[0], k.shape[0]
    lp = k.shape[1] - w
    kk = torch.from_numpy(k[:, :lp]).repeat_interleave(H // G, dim=0)      # [H][lp][d]
    logits = torch.einsum("hid,htd->hit", torch.from_numpy(q), kk) / math.sqrt(q.shape[-1])
    return torch.softmax(logits, dim=-1).sum(dim=1).numpy()


@pytest.mark.parametrize("H,G,w,L", [(28, 4, 8, 100), (4, 4, 3, 20), (6, 1, 5, 40)])
def test_window_attention_vs_torch_softmax(H, G, w, L):
    r = _rng(1)
    q = r.standard_normal((H, w, 16))
    k = r.standard_normal((G, L, 16))
    a = O.window_attention(q, k, w)
    np.testing.assert_allclose(a, _torch_window_attention(q, k, w), rtol=1e-12, atol=1e-14)
    # each of the w softmax rows sums to 1 over K_past
    np.testing.assert_allclose(a.sum(axis=1), w, rtol=1e-12)


def test_window_attention_excludes_window_keys_and_uniform_keys():
    r = _rng(2)
    q = r.standard_normal((4, 3, 8))
    k = r.standard_normal((2, 30, 8))
    a = O.window_attention(q, k, 3)
    k2 = k.copy()
    k2[:, 27:] = 100.0  # window keys are neither scored nor normalised over
    np.testing.assert_array_equal(O.window_attention(q, k2, 3), a)
    k3 = np.repeat(r.standard_normal((2, 1, 8)), 30, axis=1)  # identical keys
    np.testing.assert_allclose(O.window_attention(q, k3, 3), 3.0 / 27.0, rtol=1e-12)


@pytest.mark.parametrize("kernel", [1, 3, 5, 7])
def test_avg_pool_vs_torch(kernel):
    x = _rng(3).random((5, 37))
    ref = F.avg_pool1d(torch.from_numpy(x)[None], kernel, stride=1, padding=kernel // 2,
                       count_include_pad=True)[0].numpy()
    np.testing.assert_allclose(O.avg_pool(x, kernel), ref, rtol=1e-13, atol=1e-15)


def test_group_scores_is_group_mean_and_mha_identity():
    a = _rng(4).random((28, 50))
    np.testing.assert_allclose(O.group_scores(a, 4), a.reshape(4, 7, 50).mean(axis=1), rtol=1e-13)
    np.testing.assert_allclose(O.group_scores(a, 28), a, rtol=1e-13)  # MHA: G = H


def test_base_score_and_governing_group():
    s = np.array([[1.0, 2.0, 3.0, 5.0], [4.0, 2.0, 1.0, 5.0]])
    np.testing.assert_allclose(O.base_score(s), [2.5, 2.0, 2.0, 5.0])
    assert O.governing_group(s).tolist() == [1, 0, 0, 0]  # ties -> lowest group


# ------------------------------------------------------------------ Sec. 3.6

def test_entropy_bounds_and_limits():
    L = 1000
    h, t = O.entropy_temperature(np.full(L, 0.3), 0.75, 1.25, 1e-12)
    assert abs(h - 1.0) < 1e-9 and abs(t - 1.25) < 1e-9          # uniform -> H = 1
    onehot = np.zeros(L); onehot[17] = 2.0
    h, t = O.entropy_temperature(onehot, 0.75, 1.25, 1e-12)
    assert abs(h) < 1e-9 and abs(t - 0.75) < 1e-9                # one-hot -> H = 0 (up to eps)
    for seed in range(5):
        x = _rng(seed).random(L) ** 4
        h, t = O.entropy_temperature(x, 0.95, 1.05, 1e-12)
        assert -1e-12 <= h <= 1.0 + 1e-12
        ref = scipy.stats.entropy(x / x.sum()) / math.log(L)
        assert abs(h - ref) < 1e-9
        assert abs(t - (0.95 + 0.1 * ref)) < 1e-9


# ------------------------------------------------------------------ Sec. 3.4

def test_rank_bins_vs_scipy_ordinal_ranks_and_equal_frequency():
    r = _rng(5)
    for n, K in [(100, 8), (13, 4), (64, 8), (1000, 7)]:
        v = np.round(r.random(n) * 20) / 20  # many ties
        ref = (scipy.stats.rankdata(v, method="ordinal").astype(np.int64) - 1) * K // n
        b = O.rank_bins(v, K)
        np.testing.assert_array_equal(b, ref)
        counts = np.bincount(b, minlength=K)
        assert counts.max() - counts.min() <= 1 and counts.sum() == n
        order = np.argsort(v, kind="stable")
        assert np.all(np.diff(b[order]) >= 0)  # monotone in value


def test_spatial_cells():
    r, c = np.meshgrid(np.arange(52), np.arange(52), indexing="ij")
    cells = O.spatial_cells(r.ravel(), c.ravel(), 52, 52, 8)
    counts = np.bincount(cells, minlength=64)
    assert counts.sum() == 52 * 52 and set(np.unique(counts)) <= {36, 42, 49}
    r, c = np.meshgrid(np.arange(8), np.arange(8), indexing="ij")
    np.testing.assert_array_equal(O.spatial_cells(r.ravel(), c.ravel(), 8, 8, 8), np.arange(64))


def test_mutual_information_vs_sklearn():
    metrics = pytest.importorskip("sklearn.metrics")
    r = _rng(6)
    for n in [10, 200, 3000]:
        bins = r.integers(0, 8, n)
        cells = (bins * 3 + r.integers(0, 5, n)) % 64  # dependent
        mi = O.mutual_information(bins, cells, 8, 64)
        assert abs(mi - metrics.mutual_info_score(bins, cells)) < 1e-12


def test_mutual_information_closed_forms_and_bounds():
    K, cells_n = 8, 64
    # every cell holds one token of each bin -> independent -> MI = 0
    bins = np.tile(np.arange(K), cells_n)
    cells = np.repeat(np.arange(cells_n), K)
    assert abs(O.mutual_information(bins, cells, K, cells_n)) < 1e-12
    # each cell maps to one bin, equal mass -> MI = H(B) = log K
    cells = np.arange(cells_n).repeat(5)
    bins = cells % K
    assert abs(O.mutual_information(bins, cells, K, cells_n) - math.log(K)) < 1e-12
    # entropy decomposition MI = H(B) + H(C) - H(B, C), and 0 <= MI <= log K
    r = _rng(7)
    for _ in range(5):
        b = r.integers(0, K, 500)
        c = (b + r.integers(0, 3, 500)) % cells_n
        mi = O.mutual_information(b, c, K, cells_n)
        hb = scipy.stats.entropy(np.bincount(b))
        hc = scipy.stats.entropy(np.bincount(c))
        hbc = scipy.stats.entropy(np.bincount(b * cells_n + c))
        assert abs(mi - (hb + hc - hbc)) < 1e-12
        assert -1e-12 <= mi <= math.log(K) + 1e-12


def test_mi_ema_fixed_point_and_geometric_decay():
    prev = np.array([1.0, 0.0])
    np.testing.assert_allclose(O.mi_ema(prev, np.array([0.0, 1.0]), 0.9, False), [0.9, 0.1])
    np.testing.assert_array_equal(O.mi_ema(prev, np.array([0.3, 0.7]), 0.9, True), [0.3, 0.7])
    m = np.array([2.0])
    for n in range(1, 20):
        m = O.mi_ema(m, np.array([1.0]), 0.9, False)
        assert abs((m[0] - 1.0) - 0.9 ** n) < 1e-12


def test_subspace_prior_vs_scipy_softmax_and_invariances():
    mi = np.array([0.1, 0.4, 0.25, 0.05])
    dm = mi - mi.min()
    ref = scipy.special.softmax((dm / (dm.max() + 1e-6)) / 0.7)
    np.testing.assert_allclose(O.subspace_prior(mi, 1e-6, 0.7), ref, rtol=1e-13)
    # min-max normalisation: invariant to shifting all MI values
    np.testing.assert_allclose(O.subspace_prior(mi + 3.0, 1e-6, 1.0),
                               O.subspace_prior(mi, 1e-6, 1.0), rtol=1e-9)
    # equal MI -> uniform prior -> beta == 1 (Sec. 3.4: G w averages to 1)
    w = O.subspace_prior(np.full(4, 0.3), 1e-6, 1.0)
    np.testing.assert_allclose(w, 0.25)
    gstar = _rng(8).integers(0, 4, 50)
    np.testing.assert_allclose(O.mi_weight(gstar, w, 0.5), 1.0)


def test_lambda_schedule():
    lam = [O.lambda_at(n, 0.5, 5, 10) for n in range(20)]
    assert lam[:6] == [0.0] * 6
    assert abs(lam[10] - 0.25) < 1e-15 and lam[15] == 0.5 and lam[19] == 0.5
    assert all(b >= a for a, b in zip(lam, lam[1:]))
    assert O.lambda_at(0, 0.5, 0, 0) == 0.5 and O.lambda_at(2, 0.5, 3, 0) == 0.0


# ------------------------------------------------------------------ Sec. 3.5

def test_temporal_stability_vs_scipy_cosine_and_fresh_state():
    import scipy.spatial.distance as dist
    r = _rng(9)
    cur, m = r.random(30), r.random(30)
    phi, m2 = O.temporal_stability(cur, m, 0.9)
    assert abs(phi - (1.0 - dist.cosine(cur, m))) < 1e-12 and 0.0 <= phi <= 1.0
    np.testing.assert_allclose(m2, 0.9 * m + 0.1 * cur)
    phi, m2 = O.temporal_stability(cur, np.zeros(30), 0.9)  # fresh
    assert phi == 0.0 and np.array_equal(m2, cur)
    phi, _ = O.temporal_stability(2.5 * m, m, 0.9)          # same direction
    assert abs(phi - 1.0) < 1e-12


def test_current_row_places_newest_frame_on_grid():
    R, C = 3, 4
    vis = np.array([0, 1, 1, 1, 1, 0])
    frame = np.array([0, 1, 2, 2, 2, 0])
    row = np.array([0, 0, 0, 2, 1, 0])
    col = np.array([0, 1, 3, 0, 2, 0])
    s = np.array([9.0, 8.0, 1.0, 2.0, 3.0, 7.0])
    out = O.current_row(s, vis, frame, row, col, 2, R, C)
    ref = np.zeros(R * C); ref[3] = 1.0; ref[8] = 2.0; ref[6] = 3.0
    np.testing.assert_array_equal(out, ref)


def test_temporal_decay_limits():
    vis = np.array([1, 1, 1, 0, 1])
    frame = np.array([3, 0, 0, 0, 3])
    phi = np.array([0.7, 0.0, 1.0, 1.0, 1.0])
    d = O.temporal_decay(vis, frame, 3, phi, 0.2, 0.1)
    assert d[0] == 1.0 and d[1] == 1.0 and d[3] == 1.0 and d[4] == 1.0  # Delta_f = 0, phi = 0, text
    assert abs(d[2] - (0.1 + 0.9 * math.exp(-0.6))) < 1e-15
    far = O.temporal_decay(np.array([1]), np.array([0]), 10 ** 6, np.array([1.0]), 0.2, 0.1)
    assert abs(far[0] - 0.1) < 1e-12                                     # D -> D_min
    x = O.temporal_decay(np.ones(100), _rng(10).integers(0, 5, 100), 5, _rng(11).random(100), 0.2, 0.1)
    assert np.all((x >= 0.1) & (x <= 1.0))


# ------------------------------------------------------------------ Sec. 3.7

def test_top_b_vs_brute_force_definition():
    r = _rng(12)
    for n, b in [(1, 0), (1, 1), (20, 7), (50, 50), (64, 10)]:
        s = np.round(r.random(n) * 5) / 5  # ties
        idx = O.top_b(s, b)
        brute = [t for t in range(n)
                 if sum(1 for u in range(n) if s[u] > s[t] or (s[u] == s[t] and u < t)) < b]
        assert idx.tolist() == brute


def test_top_b_vs_torch_topk_distinct():
    s = _rng(13).random(500)
    _, ref = torch.topk(torch.from_numpy(s), 123)
    assert O.top_b(s, 123).tolist() == sorted(ref.tolist())


def test_compact_vs_index_select():
    r = _rng(14)
    k = r.standard_normal((4, 40, 8))
    idx = np.array([0, 3, 9, 31])
    ref = torch.cat([torch.from_numpy(k[:, :32]).index_select(1, torch.from_numpy(idx)),
                     torch.from_numpy(k[:, 32:])], dim=1).numpy()
    np.testing.assert_array_equal(O.compact(k, idx, 8), ref)
    meta = np.arange(40)
    np.testing.assert_array_equal(O.compact(meta, idx, 8), np.r_[idx, np.arange(32, 40)])


def test_final_score_temperature_one_and_rank_preservation():
    r = _rng(15)
    sbar, beta, d = r.random(200), 0.5 + r.random(200), 0.1 + 0.9 * r.random(200)
    np.testing.assert_allclose(O.final_score(sbar, beta, d, 1.0), sbar * beta * d)
    base = O.top_b(O.final_score(sbar, beta, d, 1.0), 40)
    for temp in [0.75, 0.95, 1.05, 1.25]:
        assert np.array_equal(O.top_b(O.final_score(sbar, beta, d, temp), 40), base)


# ------------------------------------------------------------------ whole layer

def _small_case(seed, H=8, G=2, w=4, R=4, C=5, shots=3, n_text=20, d=16):
    r = _rng(seed)
    layout_vis, layout_frame, layout_row, layout_col = [], [], [], []
    per = n_text // (shots + 1)
    for s in range(shots + 1):
        n = per if s < shots else n_text - per * shots
        layout_vis += [0] * n; layout_frame += [0] * n; layout_row += [0] * n; layout_col += [0] * n
        if s < shots:
            j = np.arange(R * C)
            layout_vis += [1] * (R * C); layout_frame += [s] * (R * C)
            layout_row += (j // C).tolist(); layout_col += (j % C).tolist()
    L = len(layout_vis)
    meta = tuple(np.array(a, np.int64) for a in (layout_vis, layout_frame, layout_row, layout_col))
    q = r.standard_normal((H, w, d))
    k = r.standard_normal((G, L, d))
    return q, k, meta, shots - 1


def test_base_configuration_equals_topb_of_pooled_gqa_attention():
    """Table 2 "Base": lambda = 0, no temporal term, T = 1 gives global top-B of
    the pooled, group-averaged window attention (computed here with torch)."""
    q, k, meta, F_ = _small_case(20)
    w = q.shape[1]
    p = O.Params(lam=0.0, delta=0.0, t_min=1.0, t_max=1.0, pool_kernel=3)
    st = O.LayerState.fresh(k.shape[0], 4, 5)
    out = O.select_layer(O.score_layer(q, k, w, p), *meta, F_, 17, 4, 5, st, p)
    a = torch.from_numpy(_torch_window_attention(q, k, w))
    a = F.avg_pool1d(a[None], 3, stride=1, padding=1, count_include_pad=True)[0]
    sbar = a.reshape(k.shape[0], -1, a.shape[-1]).mean(dim=1).mean(dim=0)
    _, ref = torch.topk(sbar, 17)
    assert out["idx"].tolist() == sorted(ref.tolist())


def test_selection_invariant_to_token_permutation():
    q, k, meta, F_ = _small_case(21)
    w = q.shape[1]
    L = k.shape[1]
    lp = L - w
    p = O.Params(pool_kernel=1, n_warmup=0, n_ramp=0)
    st0 = O.LayerState.fresh(k.shape[0], 4, 5)
    st0.n, st0.mi_bar, st0.m = 3, np.array([0.2, 0.5]), _rng(3).random((2, 20))
    perm = np.r_[_rng(22).permutation(lp), np.arange(lp, L)]
    outs = []
    for pm in (np.arange(L), perm):
        st = st0.copy()
        s = O.score_layer(q, k[:, pm], w, p)
        o = O.select_layer(s, *(a[pm] for a in meta), F_, 19, 4, 5, st, p)
        outs.append(set(pm[o["idx"]].tolist()))
    assert outs[0] == outs[1]


def test_selection_invariant_to_temperature_range():
    q, k, meta, F_ = _small_case(23)
    sets = []
    for tmin, tmax in [(1.0, 1.0), (0.75, 1.25), (0.95, 1.05), (0.5, 3.0)]:
        p = O.Params(t_min=tmin, t_max=tmax, n_warmup=0, n_ramp=0)
        st = O.LayerState.fresh(k.shape[0], 4, 5)
        o = O.select_layer(O.score_layer(q, k, q.shape[1], p), *meta, F_, 21, 4, 5, st, p)
        sets.append(o["idx"].tolist())
    assert all(s == sets[0] for s in sets)


def test_single_frame_has_no_temporal_discount_and_mha_case():
    q, k, meta, F_ = _small_case(24, H=4, G=4, shots=1)
    p = O.Params(n_warmup=0, n_ramp=0)
    st = O.LayerState.fresh(4, 4, 5)
    st.m = _rng(5).random((4, 20)); st.n = 2
    o = O.select_layer(O.score_layer(q, k, q.shape[1], p), *meta, F_, 9, 4, 5, st, p)
    np.testing.assert_array_equal(o["D"], 1.0)  # App. A.1: single image -> D_t = 1
    a = O.avg_pool(O.window_attention(q, k, q.shape[1]), p.pool_kernel)
    np.testing.assert_allclose(O.score_layer(q, k, q.shape[1], p), a, rtol=1e-13)  # G = H


def test_single_group_prior_is_neutral():
    q, k, meta, F_ = _small_case(25, H=4, G=1)
    p = O.Params(n_warmup=0, n_ramp=0)
    st = O.LayerState.fresh(1, 4, 5)
    o = O.select_layer(O.score_layer(q, k, q.shape[1], p), *meta, F_, 9, 4, 5, st, p)
    np.testing.assert_allclose(o["beta"], 1.0)
    assert st.n == 1 and o["w"].tolist() == [1.0]


# ------------------------------------------------------------------ per-KV-head selection mode

def _headwise_topk(s_row, b):
    """Head-wise top-K by a plain sort (values descending, then lower index first)."""
    order = sorted(range(len(s_row)), key=lambda i: (-float(s_row[i]), i))
    return sorted(order[:b])


def test_per_head_base_configuration_equals_headwise_topk_of_pooled_attention():
    """lambda = 0, no temporal term, T = 1: each group keeps the top-B of its own
    pooled, group-averaged window attention (SnapKV-style head-wise top-K,
    App. A.3), computed here with torch."""
    q, k, meta, F_ = _small_case(40, G=4)
    w = q.shape[1]
    p = O.Params(lam=0.0, delta=0.0, t_min=1.0, t_max=1.0, pool_kernel=3)
    st = O.LayerState.fresh(4, 4, 5)
    out = O.select_layer_per_head(O.score_layer(q, k, w, p), *meta, F_, 13, 4, 5, st, p)
    a = torch.from_numpy(_torch_window_attention(q, k, w))
    a = F.avg_pool1d(a[None], 3, stride=1, padding=1, count_include_pad=True)[0]
    s = a.reshape(4, -1, a.shape[-1]).mean(dim=1).numpy()
    assert out["idx"].shape == (4, 13)
    for g in range(4):
        assert out["idx"][g].tolist() == _headwise_topk(s[g], 13)
    assert len({tuple(r) for r in out["idx"].tolist()}) > 1   # the groups really differ


def test_per_head_single_group_equals_global_mode():
    q, k, meta, F_ = _small_case(41, H=4, G=1)
    p = O.Params(n_warmup=0, n_ramp=0)
    s = O.score_layer(q, k, q.shape[1], p)
    st0 = O.LayerState.fresh(1, 4, 5)
    st0.n, st0.mi_bar, st0.m = 2, np.array([0.3]), _rng(6).random((1, 20))
    st1 = st0.copy()
    g = O.select_layer(s, *meta, F_, 11, 4, 5, st0, p)
    h = O.select_layer_per_head(s, *meta, F_, 11, 4, 5, st1, p)
    np.testing.assert_allclose(h["score"][0], g["score"], rtol=1e-14)
    assert h["idx"][0].tolist() == g["idx"].tolist()
    assert h["T"][0] == g["T"] and st0.n == st1.n == 3
    np.testing.assert_allclose(st1.m, st0.m, rtol=0)


def test_per_head_temperature_is_each_rows_own():
    """Sec. 3.6 per row: a uniform row has H = 1 (T = T_max), a one-hot row H = 0
    (T = T_min); a third row lies in between."""
    lp = 64
    s = np.stack([np.full(lp, 0.5), np.eye(lp)[7] * 3.0, _rng(7).random(lp)])
    z = np.zeros(lp, np.int64)
    p = O.Params(t_min=0.9, t_max=1.1)
    o = O.select_layer_per_head(s, z, z, z, z, 0, 5, 4, 5, O.LayerState.fresh(3, 4, 5), p)
    np.testing.assert_allclose(o["H"][:2], [1.0, 0.0], atol=1e-9)
    np.testing.assert_allclose(o["T"][:2], [1.1, 0.9], atol=1e-9)
    assert 0.0 < o["H"][2] < 1.0
    assert 7 in o["idx"][1].tolist()


def test_per_head_sets_invariant_to_prior_and_temperature():
    """beta_g is one factor per row and x -> x^(1/T) is increasing, so neither
    lambda, tau nor the temperature range changes any group's set."""
    q, k, meta, F_ = _small_case(42, G=4)
    s = O.score_layer(q, k, q.shape[1], O.Params())
    st0 = O.LayerState.fresh(4, 4, 5)
    st0.n, st0.mi_bar, st0.m = 6, np.array([0.1, 0.7, 0.3, 0.2]), _rng(8).random((4, 20))
    sets = []
    for lam, tau, tmin, tmax in [(0.0, 1.0, 1.0, 1.0), (0.5, 1.0, 0.95, 1.05), (1.0, 0.1, 0.5, 3.0)]:
        p = O.Params(lam=lam, tau=tau, t_min=tmin, t_max=tmax, n_warmup=0, n_ramp=0, delta=0.7)
        sets.append(O.select_layer_per_head(s, *meta, F_, 15, 4, 5, st0.copy(), p)["idx"].tolist())
    assert all(x == sets[0] for x in sets)


def test_per_head_temporal_discount_uses_each_groups_own_phi():
    """Group 0's m equals its current-frame row (phi_0 = 1), group 1's m is
    orthogonal to its row (phi_1 = 0), and group 1 governs every token
    (S[1] > S[0]).  With D_min = 0 and a steep delta, group 0 keeps only text
    and current-frame tokens (its B largest among them), group 1 is
    undiscounted (plain top-B of its row)."""
    q, k, meta, F_ = _small_case(43, G=2, shots=3, n_text=40)
    is_vis, frame, row, col = meta
    lp = k.shape[1] - q.shape[1]
    r = _rng(11)
    s0 = 0.01 + r.random(lp)
    s = np.stack([s0, 1.5 * s0 + 0.5 * r.random(lp)])
    R, C = 4, 5
    cur = np.zeros((2, R * C))
    for t in range(lp):
        if is_vis[t] and frame[t] == F_:
            cur[:, row[t] * C + col[t]] = s[:, t]
    m1 = r.standard_normal(R * C)
    m1 -= (m1 @ cur[1]) / (cur[1] @ cur[1]) * cur[1]
    st = O.LayerState.fresh(2, R, C)
    st.n, st.mi_bar, st.m = 3, np.array([0.2, 0.4]), np.stack([cur[0], m1])
    p = O.Params(delta=200.0, d_min=0.0, n_warmup=0, n_ramp=0)
    B = 10
    o = O.select_layer_per_head(s, *meta, F_, B, R, C, st, p)
    np.testing.assert_allclose(o["phi"], [1.0, 0.0], atol=1e-12)
    fresh = np.array([(not is_vis[t]) or frame[t] == F_ for t in range(lp)])
    assert fresh.sum() >= B
    keep0 = sorted(sorted(np.nonzero(fresh)[0], key=lambda t: (-s[0, t], t))[:B])
    assert o["idx"][0].tolist() == keep0
    assert o["idx"][0].tolist() != _headwise_topk(s[0], B)   # the discount took part
    assert o["idx"][1].tolist() == _headwise_topk(s[1], B)


def test_per_head_selection_invariant_to_token_permutation():
    q, k, meta, F_ = _small_case(44, G=4)
    w = q.shape[1]
    L = k.shape[1]
    lp = L - w
    p = O.Params(pool_kernel=1, n_warmup=0, n_ramp=0)
    st0 = O.LayerState.fresh(4, 4, 5)
    st0.n, st0.mi_bar, st0.m = 3, np.array([0.2, 0.5, 0.1, 0.9]), _rng(10).random((4, 20))
    perm = np.r_[_rng(45).permutation(lp), np.arange(lp, L)]
    outs = []
    for pm in (np.arange(L), perm):
        o = O.select_layer_per_head(O.score_layer(q, k[:, pm], w, p), *(a[pm] for a in meta), F_, 9,
                                    4, 5, st0.copy(), p)
        outs.append([set(pm[r].tolist()) for r in o["idx"]])
    assert outs[0] == outs[1]


def test_compact_per_head_vs_index_select():
    r = _rng(46)
    G, L, d, w, B = 3, 30, 8, 4, 6
    x = r.standard_normal((G, L, d))
    meta = r.integers(0, 1 << 20, L)
    idx = np.stack([np.sort(r.choice(L - w, B, replace=False)) for _ in range(G)])
    got = O.compact_per_head(x, idx, w)
    got_m = O.compact_per_head(meta, idx, w)
    for g in range(G):
        rows = torch.cat([torch.from_numpy(idx[g]), torch.arange(L - w, L)])
        ref = torch.from_numpy(x[g]).index_select(0, rows)
        assert torch.equal(torch.from_numpy(got[g]), ref)
        assert torch.equal(torch.from_numpy(got_m[g]), torch.from_numpy(meta).index_select(0, rows))


def test_per_head_per_group_metadata_follows_each_groups_tokens():
    """Per-group metadata rows: shuffling group g's tokens (its S row and its
    metadata row together, each group with its own permutation) maps every
    group's kept set and every group statistic through that permutation; a row
    of metadata equal for all groups gives the shared-metadata result."""
    q, k, meta, F_ = _small_case(47, G=3, shots=3, n_text=30)
    lp = k.shape[1] - q.shape[1]
    s = O.score_layer(q, k, q.shape[1], O.Params(pool_kernel=1))
    p = O.Params(n_warmup=0, n_ramp=0, delta=0.5)
    st0 = O.LayerState.fresh(3, 4, 5)
    st0.n, st0.mi_bar, st0.m = 4, np.array([0.3, 0.1, 0.6]), _rng(12).random((3, 20))
    shared = O.select_layer_per_head(s, *meta, F_, 12, 4, 5, st0.copy(), p)
    tiled = O.select_layer_per_head(s, *(np.tile(a[:lp], (3, 1)) for a in meta), F_, 12, 4, 5,
                                    st0.copy(), p)
    assert shared["idx"].tolist() == tiled["idx"].tolist()
    perms = [_rng(48 + g).permutation(lp) for g in range(3)]
    s_p = np.stack([s[g][perms[g]] for g in range(3)])
    meta_p = tuple(np.stack([a[:lp][perms[g]] for g in range(3)]) for a in meta)
    o = O.select_layer_per_head(s_p, *meta_p, F_, 12, 4, 5, st0.copy(), p)
    for g in range(3):
        assert sorted(perms[g][o["idx"][g]].tolist()) == shared["idx"][g].tolist()
    np.testing.assert_allclose(o["mi"], shared["mi"], rtol=1e-12)
    np.testing.assert_allclose(o["phi"], shared["phi"], rtol=1e-12)


# ------------------------------------------------------------------ normaliser supplied by the prefill pass

def test_window_lse_vs_torch_logsumexp():
    r = _rng(60)
    H, G, w, L, d = 8, 2, 4, 50, 16
    q = r.standard_normal((H, w, d)) * 3
    k = r.standard_normal((G, L, d))
    got = O.window_lse(q, k, w)
    kk = torch.from_numpy(k[:, :L - w]).repeat_interleave(H // G, dim=0)
    z = torch.einsum("hid,htd->hit", torch.from_numpy(q), kk) / math.sqrt(d)
    np.testing.assert_allclose(got, torch.logsumexp(z, dim=-1).numpy(), rtol=1e-13, atol=1e-13)
    assert np.all(O.window_lse(q, k[:, :w], w) == -np.inf)   # no past keys


def test_attention_with_the_exact_normaliser_is_the_softmax_sum():
    r = _rng(61)
    q = r.standard_normal((6, 5, 16))
    k = r.standard_normal((3, 40, 16))
    lse = O.window_lse(q, k, 5)
    np.testing.assert_allclose(O.window_attention_given_lse(q, k, 5, lse), O.window_attention(q, k, 5),
                               rtol=1e-12, atol=1e-15)
    # a normaliser larger by c scales every row's contribution by exp(-c)
    shifted = O.window_attention_given_lse(q, k, 5, lse + 0.5)
    np.testing.assert_allclose(shifted, O.window_attention(q, k, 5) * math.exp(-0.5), rtol=1e-12)


def test_window_attention_output_vs_torch_sdpa():
    """The attention output of the window rows over the past keys against
    torch's scaled_dot_product_attention in float64 (GQA by repeating each
    group's keys and values for its heads)."""
    r = _rng(62)
    H, G, w, L, d = 8, 2, 4, 70, 16
    q, k, v = r.standard_normal((H, w, d)) * 2, r.standard_normal((G, L, d)), r.standard_normal((G, L, d))
    got = O.window_attention_output(q, k, v, w)
    kk = torch.from_numpy(k[:, :L - w]).repeat_interleave(H // G, dim=0)
    vv = torch.from_numpy(v[:, :L - w]).repeat_interleave(H // G, dim=0)
    ref = F.scaled_dot_product_attention(torch.from_numpy(q), kk, vv)
    np.testing.assert_allclose(got, ref.numpy(), rtol=1e-12, atol=1e-13)
    # the window's own keys and values take no part
    k2, v2 = k.copy(), v.copy()
    k2[:, L - w:] = 100.0
    v2[:, L - w:] = -7.0
    np.testing.assert_allclose(O.window_attention_output(q, k2, v2, w), got, rtol=1e-13)
    assert np.all(O.window_attention_output(q, k[:, :w], v[:, :w], w) == 0.0)   # no past keys


def test_window_attention_output_limits_and_normaliser():
    """Zero queries give the mean of the past values; a query aligned with one
    key far above the rest gives that key's value; exp(lse) O is the
    unnormalised sum of exp(z) V."""
    r = _rng(63)
    H, G, w, L, d = 4, 2, 3, 40, 8
    k, v = r.standard_normal((G, L, d)), r.standard_normal((G, L, d))
    lp = L - w
    out = O.window_attention_output(np.zeros((H, w, d)), k, v, w)
    for h in range(H):
        np.testing.assert_allclose(out[h], np.broadcast_to(v[h * G // H, :lp].mean(axis=0), (w, d)), rtol=1e-12)
    kb = k.copy()
    kb[:, 11] *= 10.0 / np.linalg.norm(kb[:, 11], axis=1, keepdims=True)   # key 11: length 10
    q = np.zeros((H, w, d))
    for h in range(H):
        q[h] = 2.0 * kb[h * G // H, 11]    # logit 200 / sqrt(d) at key 11, far below elsewhere
    out = O.window_attention_output(q, kb, v, w)
    for h in range(H):
        np.testing.assert_allclose(out[h], np.broadcast_to(v[h * G // H, 11], (w, d)), atol=1e-6)
    q = r.standard_normal((H, w, d))
    out, lse = O.window_attention_output(q, k, v, w), O.window_lse(q, k, w)
    for h in range(H):
        g = h * G // H
        z = q[h] @ k[g, :lp].T / math.sqrt(d)
        np.testing.assert_allclose(np.exp(lse[h])[:, None] * out[h], np.exp(z) @ v[g, :lp], rtol=1e-12)


# ------------------------------------------------------------------ ablation variants (readings)

def test_decay_variants_limits_and_ordering():
    """All three shapes give D = 1 at Delta_f phi = 0 and for text tokens; the
    linear one reaches D_min at delta Delta_f phi = 1 and stays there; at the
    defaults linear < exponential < power law for old frames (the order in
    which the ablation says they keep history); each decreases with age."""
    dist = np.arange(0, 12)
    vis = np.ones_like(dist)
    cur = 11
    frame = cur - dist
    phi = np.full(dist.shape, 0.8)
    ds = [O.temporal_decay(vis, frame, cur, phi, 0.2, 0.1, m) for m in (0, 1, 2)]
    for d in ds:
        assert d[0] == 1.0 and np.all(np.diff(d) <= 0)
        np.testing.assert_array_equal(O.temporal_decay(vis * 0, frame, cur, phi, 0.2, 0.1), 1.0)
        np.testing.assert_array_equal(O.temporal_decay(vis, frame, cur, phi * 0, 0.2, 0.1), 1.0)
    lin = ds[1]
    floor = dist * 0.8 * 0.2 >= 1.0
    assert floor.any() and np.all(lin[floor] == 0.1) and np.all(lin[~floor] > 0.1)
    old = dist >= 2
    assert np.all(ds[1][old] < ds[0][old]) and np.all(ds[0][old] < ds[2][old])


def test_confidence_temperature_closed_forms_and_rank_preservation():
    L = 50
    pm, t = O.confidence_temperature(np.full(L, 0.3), 0.75, 1.25, 1e-12)
    assert abs(pm - 1 / L) < 1e-12 and abs(t - (0.75 + 0.5 * (1 - 1 / L))) < 1e-12
    pm, t = O.confidence_temperature(np.eye(L)[3] * 2.0, 0.75, 1.25, 1e-12)
    assert abs(pm - 1.0) < 1e-12 and abs(t - 0.75) < 1e-12
    q, k, meta, F_ = _small_case(62)
    sets = []
    for mode in (0, 1):
        p = O.Params(aeb_mode=mode, n_warmup=0, n_ramp=0, t_min=0.5, t_max=2.0)
        o = O.select_layer(O.score_layer(q, k, q.shape[1], p), *meta, F_, 17, 4, 5,
                           O.LayerState.fresh(k.shape[0], 4, 5), p)
        sets.append(o["idx"].tolist())
    assert sets[0] == sets[1]


def test_mi_over_the_newest_frame_vs_sklearn():
    """mi_span = 1: MI_g from the newest frame's visual tokens alone, checked
    against scikit-learn's mutual_info_score on that subset (scipy ordinal ranks
    for the rank bins)."""
    metrics = pytest.importorskip("sklearn.metrics")
    q, k, meta, F_ = _small_case(63, G=2, shots=3, n_text=20)
    is_vis, frame, row, col = meta
    p = O.Params(mi_span=1, n_warmup=0, n_ramp=0, pool_kernel=1, mi_bins=4, mi_grid=2)
    s = O.score_layer(q, k, q.shape[1], p)
    lp = s.shape[1]
    o = O.select_layer(s, *meta, F_, 9, 4, 5, O.LayerState.fresh(2, 4, 5), p)
    sel = (is_vis[:lp] != 0) & (frame[:lp] == F_)
    cells = (row[:lp][sel] * 2 // 4) * 2 + (col[:lp][sel] * 2 // 5)
    for g in range(2):
        v = s[g][sel]
        bins = (scipy.stats.rankdata(v, method="ordinal").astype(np.int64) - 1) * 4 // v.size
        assert abs(o["mi"][g] - metrics.mutual_info_score(bins, cells)) < 1e-12
    full = O.select_layer(s, *meta, F_, 9, 4, 5, O.LayerState.fresh(2, 4, 5),
                          O.Params(n_warmup=0, n_ramp=0, pool_kernel=1, mi_bins=4, mi_grid=2))
    assert not np.allclose(full["mi"], o["mi"])   # the span matters


def test_mi_prior_of_a_layer_end_to_end_vs_sklearn_and_scipy():
    """The default span: MI_g of every group over all visual tokens of the
    layer (equal-frequency rank bins of the pooled score, scipy ordinal ranks;
    patch cells on the M x M grid) against scikit-learn's mutual_info_score,
    the prior w = softmax(min-max(MI_bar) / tau) against scipy's softmax, and
    the EMA carried into a second step with new scores."""
    metrics = pytest.importorskip("sklearn.metrics")
    K, M, R, C = 4, 2, 4, 5
    p = O.Params(n_warmup=0, n_ramp=0, pool_kernel=3, mi_bins=K, mi_grid=M, tau=0.7, rho_mi=0.8)
    st = O.LayerState.fresh(3, R, C)
    mi_bar = None
    for step, seed in enumerate((71, 72)):
        q, k, meta, F_ = _small_case(seed, G=3, shots=3, n_text=20)
        is_vis, frame, row, col = meta
        s = O.score_layer(q, k, q.shape[1], p)
        lp = s.shape[1]
        o = O.select_layer(s, *meta, F_, 9, R, C, st, p)
        sel = is_vis[:lp] != 0
        cells = (row[:lp][sel] * M // R) * M + (col[:lp][sel] * M // C)
        mi = np.empty(3)
        for g in range(3):
            v = s[g][sel]
            bins = (scipy.stats.rankdata(v, method="ordinal").astype(np.int64) - 1) * K // v.size
            mi[g] = metrics.mutual_info_score(bins, cells)
        np.testing.assert_allclose(o["mi"], mi, rtol=0, atol=1e-12)
        mi_bar = mi.copy() if step == 0 else p.rho_mi * mi_bar + (1 - p.rho_mi) * mi
        np.testing.assert_allclose(o["mi_bar"], mi_bar, rtol=0, atol=1e-12)
        m = (mi_bar - mi_bar.min()) / (mi_bar.max() - mi_bar.min() + p.eps)
        np.testing.assert_allclose(o["w"], scipy.special.softmax(m / p.tau), rtol=0, atol=1e-12)


def test_mha_granularity_by_replicated_kv_keeps_s_bar():
    """The paper's MHA-head ablation on a GQA model: every group's keys
    replicated for each of its query heads (G' = H).  Each head's row of S is
    then that head's pooled attention, the mean of a group's head rows is the
    GQA row S[g], so s_bar is unchanged; with lambda = 0, no temporal term and
    T = 1 the fused score is s_bar and the selected set equals the GQA one.
    The MI prior, now over H groups, is what the granularity changes."""
    q, k, meta, F_ = _small_case(31, H=8, G=2)
    w, H, G = q.shape[1], q.shape[0], k.shape[0]
    k_mha = np.repeat(k, H // G, axis=0)
    p = O.Params()
    S = O.score_layer(q, k, w, p)
    S_mha = O.score_layer(q, k_mha, w, p)
    np.testing.assert_allclose(S_mha, O.avg_pool(O.window_attention(q, k_mha, w), p.pool_kernel), rtol=1e-13)
    np.testing.assert_allclose(S_mha.reshape(G, H // G, -1).mean(axis=1), S, rtol=1e-12)
    np.testing.assert_allclose(S_mha.mean(axis=0), S.mean(axis=0), rtol=1e-12)
    base = O.Params(lam=0.0, delta=0.0, t_min=1.0, t_max=1.0)
    outs = []
    for S_, g in ((S, G), (S_mha, H)):
        st = O.LayerState.fresh(g, 4, 5)
        outs.append(O.select_layer(S_, *meta, F_, 17, 4, 5, st, base))
    np.testing.assert_array_equal(outs[0]["idx"], outs[1]["idx"])
    st = O.LayerState.fresh(H, 4, 5)
    o = O.select_layer(S_mha, *meta, F_, 17, 4, 5, st, O.Params(n_warmup=0, n_ramp=0))
    assert o["w"].shape == (H,) and abs(o["w"].sum() - 1.0) < 1e-12
