"""GPU parity: the CUDA path through the C ABI against the fp64 oracle on the
same seeded inputs.  Fused scores within 1e-3 relative, index sets equal
except ties inside that band, compacted K/V/metadata bit-exact."""
import numpy as np
import pytest
import torch

from oracle import starkv_oracle as O
from paper_2606_01790_gb300 import starkv as sk
from paper_2606_01790_gb300 import synthetic as syn

import harness as H

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA device", allow_module_level=True)


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()


def _run_step(wl, si, h, n_layers=None, calls=1, state=None):
    cfg = H.gpu_config(wl, h, n_layers=n_layers or si.k.shape[0])
    st = state or sk.init_state(cfg)
    ds = H.device_seq(si, wl)
    ws = sk.workspace(st, [ds.seq])
    for _ in range(calls):
        sk.step(st, [ds.seq], ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)
    return st, ds


@pytest.mark.parametrize("name", ["tiny", "uitars_layer"])
def test_score_layer_matches_oracle(name):
    wl = syn.WORKLOADS[name]
    si = syn.make_sequence(wl)
    h = H.hyper()
    st = sk.init_state(H.gpu_config(wl, h))
    ds = H.device_seq(si, wl)
    ws = sk.workspace(st, [ds.seq])
    sk.score_layer(st, 0, [ds.seq], ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)
    S_gpu = ds.seq.S[0].double().cpu().numpy()
    S_ref = O.score_layer(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window, H.oracle_params(h))
    rel = np.abs(S_gpu - S_ref) / np.abs(S_ref)
    assert rel.max() < 1e-3, rel.max()
    # each window row's softmax sums to 1 over K_past: sum_t S_raw = w * H / G, pooled mass
    # differs only at the two ends
    assert abs(S_gpu.sum(axis=1).mean() - S_ref.sum(axis=1).mean()) < 1e-4 * S_ref.sum(axis=1).mean()


def test_score_layer_with_wide_logits():
    """Queries scaled by 32 (exact in bf16): a row's logits span far more than
    2^64 in exp2 units, so the running reference of pass 1 has to move after
    its first chunk (the rescale path)."""
    wl = syn.WORKLOADS["uitars_layer"]
    si = syn.make_sequence(wl)
    si.q = si.q * 32
    h = H.hyper()
    st = sk.init_state(H.gpu_config(wl, h))
    ds = H.device_seq(si, wl)
    ws = sk.workspace(st, [ds.seq])
    sk.score_layer(st, 0, [ds.seq], ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)
    S_gpu = ds.seq.S[0].double().cpu().numpy()
    S_ref = O.score_layer(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window, H.oracle_params(h))
    # fp32 exp2 flushes terms below 2^-126 of a row's reference: an absolute
    # floor far below any score that can matter
    err = np.abs(S_gpu - S_ref)
    assert np.all(err <= 1e-3 * np.abs(S_ref) + 1e-9 * S_ref.max()), float((err / np.abs(S_ref)).max())
    assert abs(S_gpu.sum() - S_ref.sum()) < 1e-4 * S_ref.sum()


@pytest.mark.parametrize("name", ["tiny", "uitars_layer"])
@pytest.mark.parametrize("sched", ["paper", "prior_on"])
def test_step_matches_oracle(name, sched):
    wl = syn.WORKLOADS[name]
    si = syn.make_sequence(wl)
    h = H.hyper() if sched == "paper" else H.hyper(n_warmup=0, n_ramp=0, t_min=0.75, t_max=1.25)
    p = H.oracle_params(h)
    st, ds = _run_step(wl, si, h)
    ost = O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols)
    ref = H.oracle_layer(si, 0, wl, ost, p)
    S_gpu = ds.seq.S[0].double().cpu().numpy()
    assert (np.abs(S_gpu - ref["S"]) / np.abs(ref["S"])).max() < 1e-3
    sc = H.check_scores(ds.seq.score[0].double().cpu().numpy(), ref, ref["S"], si, 0, wl, p)
    assert sc["ok"], sc
    ix = H.check_index_set(ds.seq.idx[0].cpu().numpy(), ref, si.budget)
    assert ix["ok"], ix
    H.check_compaction(ds.seq, si, 0, wl.window)
    stats = ds.seq.stats[0].double().cpu().numpy()
    G = wl.n_kv_heads
    assert abs(stats[0] - ref["H"]) < 1e-5 and abs(stats[1] - ref["T"]) < 1e-5
    assert np.all(stats[8 + 4 * G:8 + 5 * G] == stats[0]) and np.all(stats[8 + 5 * G:8 + 6 * G] == stats[1])
    np.testing.assert_allclose(stats[8:8 + G], ref["mi"], rtol=2e-3, atol=2e-4)
    np.testing.assert_allclose(stats[8 + 2 * G:8 + 3 * G], ref["w"], rtol=2e-3)
    # No visual token in the rank-bin tie band (the GPU's S puts every visual
    # token in the same equal-frequency bin as the oracle's S): MI and the prior
    # then differ by arithmetic alone, and w is held to 1e-4.
    if _same_rank_bins(S_gpu, ref["S"], si.layout[0], p):
        np.testing.assert_allclose(stats[8:8 + G], ref["mi"], rtol=1e-5, atol=1e-7)
        np.testing.assert_allclose(stats[8 + 2 * G:8 + 3 * G], ref["w"], rtol=1e-4)


def _same_rank_bins(S_gpu, S_ref, lay, p):
    """Every group's visual tokens fall in the same rank bins (Sec. 3.4) under
    the GPU's and the oracle's group score maps."""
    lp = S_ref.shape[1]
    vis = lay.is_visual[:lp] != 0
    return all(np.array_equal(O.rank_bins(S_gpu[g][vis], p.mi_bins), O.rank_bins(S_ref[g][vis], p.mi_bins))
               for g in range(S_ref.shape[0]))


def test_select_stage_isolated_on_oracle_scores():
    """The oracle's own S (rounded to fp32) fed to starkv_select: rank bins,
    argmax and thresholds see identical inputs on both sides."""
    wl = syn.WORKLOADS["uitars_layer"]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    S32 = O.score_layer(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window, p).astype(np.float32)
    st = sk.init_state(H.gpu_config(wl, h))
    ds = H.device_seq(si, wl)
    ds.seq.S.copy_(torch.from_numpy(S32)[None])
    ws = sk.workspace(st, [ds.seq])
    sk.select(st, 0, [ds.seq], ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)
    ref = H.oracle_layer(si, 0, wl, O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols), p,
                         S_override=S32.astype(np.float64))
    stats = ds.seq.stats[0].double().cpu().numpy()
    G = wl.n_kv_heads
    np.testing.assert_allclose(stats[8:8 + G], ref["mi"], rtol=1e-6)     # same bins -> same MI
    np.testing.assert_allclose(stats[8 + 2 * G:8 + 3 * G], ref["w"], rtol=1e-5)
    np.testing.assert_allclose(stats[8 + 3 * G:8 + 4 * G], ref["phi"], atol=1e-6)
    sc = H.check_scores(ds.seq.score[0].double().cpu().numpy(), ref, ref["S"], si, 0, wl, p, rtol=1e-5)
    assert sc["ok"], sc
    ix = H.check_index_set(ds.seq.idx[0].cpu().numpy(), ref, si.budget, rtol=1e-5)
    assert ix["ok"], ix


def _select_on_given_scores(wl, si, S32, h):
    p = H.oracle_params(h)
    st = sk.init_state(H.gpu_config(wl, h))
    ds = H.device_seq(si, wl)
    ds.seq.S.copy_(torch.from_numpy(S32)[None])
    ws = sk.workspace(st, [ds.seq])
    sk.select(st, 0, [ds.seq], ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)
    ref = H.oracle_layer(si, 0, wl, O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols), p,
                         S_override=S32.astype(np.float64))
    return ds, ref, p


def test_select_with_heavy_score_ties():
    """Scores quantised to 8 levels per group: thousands of equal keys at each
    rank-bin boundary, ordered by position (the radix fallback of the rank
    bins), and equal fused scores at the top-B threshold (lower index wins)."""
    wl = syn.WORKLOADS["uitars_layer"]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    S = O.score_layer(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window, p)
    top = S.max(axis=1, keepdims=True)
    S32 = (np.floor(S / top * 8.0) / 8.0 * top).astype(np.float32)
    ds, ref, p = _select_on_given_scores(wl, si, S32, h)
    stats = ds.seq.stats[0].double().cpu().numpy()
    G = wl.n_kv_heads
    np.testing.assert_allclose(stats[8:8 + G], ref["mi"], rtol=1e-6)     # same bins -> same MI
    sc = H.check_scores(ds.seq.score[0].double().cpu().numpy(), ref, ref["S"], si, 0, wl, p, rtol=1e-5)
    assert sc["ok"], sc
    ix = H.check_index_set(ds.seq.idx[0].cpu().numpy(), ref, si.budget, rtol=1e-5)
    assert ix["ok"], ix


def test_select_on_a_row_longer_than_shared_memory():
    """20 screenshots (L_p = 56,096): the calibration kernel keeps the row's
    keys in the workspace instead of shared memory."""
    wl = syn.WORKLOADS["long_layer"]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    S32 = O.score_layer(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window, p).astype(np.float32)
    ds, ref, p = _select_on_given_scores(wl, si, S32, h)
    stats = ds.seq.stats[0].double().cpu().numpy()
    G = wl.n_kv_heads
    np.testing.assert_allclose(stats[8:8 + G], ref["mi"], rtol=1e-5)
    np.testing.assert_allclose(stats[8 + 3 * G:8 + 4 * G], ref["phi"], atol=1e-6)
    sc = H.check_scores(ds.seq.score[0].double().cpu().numpy(), ref, ref["S"], si, 0, wl, p, rtol=1e-5)
    assert sc["ok"], sc
    ix = H.check_index_set(ds.seq.idx[0].cpu().numpy(), ref, si.budget, rtol=1e-5)
    assert ix["ok"], ix


def test_carried_state_over_two_steps():
    """Second call sees a non-fresh state: MI EMA and the temporal EMA m_g act."""
    wl = syn.WORKLOADS["tiny"]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    st, ds = _run_step(wl, si, h, calls=2)
    ost = O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols)
    H.oracle_layer(si, 0, wl, ost, p)
    ref = H.oracle_layer(si, 0, wl, ost, p)
    assert np.any(ref["phi"] > 0.5)           # the discount is active on the second step
    sc = H.check_scores(ds.seq.score[0].double().cpu().numpy(), ref, ref["S"], si, 0, wl, p)
    assert sc["ok"], sc
    ix = H.check_index_set(ds.seq.idx[0].cpu().numpy(), ref, si.budget)
    assert ix["ok"], ix
    stats = ds.seq.stats[0].double().cpu().numpy()
    G = wl.n_kv_heads
    assert stats[3] == 1.0
    np.testing.assert_allclose(stats[8 + 3 * G:8 + 4 * G], ref["phi"], atol=1e-4)


@pytest.mark.parametrize("budget", ["zero", "all", "one"])
def test_budget_edges(budget):
    wl = syn.WORKLOADS["tiny"]
    si = syn.make_sequence(wl)
    lp = si.L - wl.window
    si.budget = {"zero": 0, "all": lp, "one": 1}[budget]
    h = H.hyper()
    p = H.oracle_params(h)
    st, ds = _run_step(wl, si, h)
    ref = H.oracle_layer(si, 0, wl, O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols), p)
    ix = H.check_index_set(ds.seq.idx[0].cpu().numpy(), ref, si.budget)
    assert ix["ok"], ix
    if budget == "all":
        assert ds.seq.idx[0].cpu().tolist() == list(range(lp))
    H.check_compaction(ds.seq, si, 0, wl.window)


def test_ragged_batch_and_short_caches():
    """Several sequences of different lengths in one call, including caches
    shorter than one key tile and one with no historical token."""
    base = syn.WORKLOADS["tiny"]
    shapes = [(2, 64), (1, 40), (0, 20), (3, 300), (0, 8)]   # (screenshots, text tokens)
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    cfg = H.gpu_config(base, h, n_layers=1, max_seqs=len(shapes))
    st = sk.init_state(cfg)
    sis, dss = [], []
    for i, (shots, text) in enumerate(shapes):
        wl = syn.Workload(f"r{i}", 100 + i, n_layers=1, window=8, grid_rows=16, grid_cols=16,
                          n_shots=shots, n_text=text)
        si = syn.make_sequence(wl)
        si.budget = min(si.budget, si.L - 8)
        sis.append(si)
        dss.append(H.device_seq(si, wl, slot=i))
    seqs = [d.seq for d in dss]
    ws = sk.workspace(st, seqs)
    sk.step(st, seqs, ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)
    for i, (si, ds) in enumerate(zip(sis, dss)):
        wl = syn.Workload(f"r{i}", 100 + i, n_layers=1, window=8, grid_rows=16, grid_cols=16,
                          n_shots=shapes[i][0], n_text=shapes[i][1])
        ref = H.oracle_layer(si, 0, wl, O.LayerState.fresh(4, 16, 16), p)
        if ref["lp"] > 0:
            sc = H.check_scores(ds.seq.score[0].double().cpu().numpy(), ref, ref["S"], si, 0, wl, p)
            assert sc["ok"], (i, sc)
        ix = H.check_index_set(ds.seq.idx[0].cpu().numpy(), ref, si.budget)
        assert ix["ok"], (i, ix)
        H.check_compaction(ds.seq, si, 0, 8)


def test_invalid_arguments_rejected():
    wl = syn.WORKLOADS["tiny"]
    si = syn.make_sequence(wl)
    st = sk.init_state(H.gpu_config(wl, H.hyper(), max_seqs=2))
    ds = H.device_seq(si, wl)
    ws = sk.workspace(st, [ds.seq])
    bad = H.device_seq(si, wl).seq
    bad.budget = si.L - wl.window + 1
    with pytest.raises(sk.StarkvError) as e:
        sk.step(st, [bad], ws)
    assert e.value.status == sk.ERR_INVALID_ARG
    with pytest.raises(sk.StarkvError):
        sk.step(st, [ds.seq, ds.seq], ws)          # one slot twice
    with pytest.raises(sk.StarkvError):
        sk.step(st, [ds.seq], ws[:1024])           # workspace too small
    with pytest.raises(sk.StarkvError):
        sk.score_layer(st, 5, [ds.seq], ws)        # layer out of range
    # a 4-byte array at an odd address is refused before any launch
    mis = H.device_seq(si, wl).seq
    raw = torch.zeros(mis.meta.numel() * 4 + 4, dtype=torch.uint8, device="cuda")
    mis.meta = raw[2:2 + mis.meta.numel() * 4]
    with pytest.raises(sk.StarkvError) as e:
        sk.step(st, [mis], ws)
    assert e.value.status == sk.ERR_INVALID_ARG


def test_gather_reports_a_kept_index_past_the_history():
    """A kept index must name a past token (< L_p): the gather reports one that
    names a window row (in bounds of the cache, so nothing faults) through the
    device error word instead of copying the window row into the kept part."""
    wl = syn.WORKLOADS["tiny"]
    si = syn.make_sequence(wl)
    st = sk.init_state(H.gpu_config(wl, H.hyper()))
    ds = H.device_seq(si, wl)
    ws = sk.workspace(st, [ds.seq])
    lp = si.L - wl.window
    good = torch.arange(si.budget, dtype=torch.int32, device="cuda")[None]
    ds.seq.idx.copy_(good)
    sk.compact(st, 0, [ds.seq], ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)             # indices below L_p: no report
    H.check_compaction(ds.seq, si, 0, wl.window)
    bad = good.clone()
    bad[0, -1] = lp                       # the first window row
    ds.seq.idx.copy_(bad)
    sk.compact(st, 0, [ds.seq], ws)
    torch.cuda.synchronize()
    assert sk.device_error_status(st) == sk.ERR_DEVICE
    sk.check_device_error(st)             # the read cleared the word
    st.close()
