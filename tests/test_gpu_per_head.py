"""GPU parity of the per-KV-head selection mode (select_mode = 1) through the C
ABI against the oracle's select_layer_per_head: each group's fused scores
within 1e-3 relative, each group's index set equal except ties inside that
band, and every group's K', V', meta' bit copies of its own selection."""
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


def _fresh(wl):
    return O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols)


def _step(st, dss):
    ws = sk.workspace(st, [d.seq for d in dss])
    sk.step(st, [d.seq for d in dss], ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)


def _check_stats(seq, layer, ref, G, atol=1e-5):
    stats = seq.stats[layer].double().cpu().numpy()
    np.testing.assert_allclose(stats[8 + 4 * G:8 + 5 * G], ref["H"], atol=atol)
    np.testing.assert_allclose(stats[8 + 5 * G:8 + 6 * G], ref["T"], atol=atol)
    assert abs(stats[0] - np.mean(ref["H"])) < atol and abs(stats[1] - np.mean(ref["T"])) < atol
    np.testing.assert_allclose(stats[8 + 2 * G:8 + 3 * G], ref["w"], rtol=2e-3)


@pytest.mark.parametrize("name", ["tiny", "uitars_layer"])
@pytest.mark.parametrize("budget", ["zero", "pct", "all"])
def test_per_head_step_matches_oracle(name, budget):
    wl = syn.WORKLOADS[name]
    si = syn.make_sequence(wl)
    lp = si.L - wl.window
    si.budget = {"zero": 0, "pct": si.budget, "all": lp}[budget]
    h = H.hyper(n_warmup=0, n_ramp=0, t_min=0.75, t_max=1.25)
    p = H.oracle_params(h)
    st = sk.init_state(H.gpu_config(wl, h, per_head=True))
    ds = H.device_seq(si, wl, per_head=True)
    _step(st, [ds])
    ref = H.oracle_layer(si, 0, wl, _fresh(wl), p, per_head=True)
    H.check_per_head(ds.seq, si, 0, wl, ref)
    _check_stats(ds.seq, 0, ref, wl.n_kv_heads)
    if budget == "pct":   # the groups keep different tokens
        idx = ds.seq.idx[0].cpu().numpy()
        assert len({tuple(r) for r in idx.tolist()}) > 1


def test_per_head_select_isolated_on_oracle_scores():
    """The oracle's S (rounded to fp32) fed to starkv_select: both sides see the
    same rows, so scores agree to 1e-5 and sets up to ties inside that band."""
    wl = syn.WORKLOADS["uitars_layer"]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    S32 = O.score_layer(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window, p).astype(np.float32)
    st = sk.init_state(H.gpu_config(wl, h, per_head=True))
    ds = H.device_seq(si, wl, per_head=True)
    ds.seq.S.copy_(torch.from_numpy(S32)[None])
    ws = sk.workspace(st, [ds.seq])
    sk.select(st, 0, [ds.seq], ws)
    sk.compact(st, 0, [ds.seq], ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)
    ref = H.oracle_layer(si, 0, wl, _fresh(wl), p, S_override=S32.astype(np.float64), per_head=True)
    H.check_per_head(ds.seq, si, 0, wl, ref, rtol=1e-5)
    _check_stats(ds.seq, 0, ref, wl.n_kv_heads, atol=1e-6)


def test_per_head_28_layer_step_at_the_benchmark_shape():
    wl = syn.WORKLOADS["uitars_5shot_28l"]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    st = sk.init_state(H.gpu_config(wl, h, per_head=True))
    ds = H.device_seq(si, wl, per_head=True)
    _step(st, [ds])
    for layer in (0, 13, 27):
        ref = H.oracle_layer(si, layer, wl, _fresh(wl), p, per_head=True)
        H.check_per_head(ds.seq, si, layer, wl, ref)


def test_per_head_long_rows_beyond_shared_memory():
    """20 screenshots + 2,048 text tokens (L_p = 56,096): the calibration keeps
    its per-token arrays in the workspace instead of shared memory."""
    wl = syn.WORKLOADS["long_layer"]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    st = sk.init_state(H.gpu_config(wl, h, per_head=True))
    ds = H.device_seq(si, wl, per_head=True)
    _step(st, [ds])
    ref = H.oracle_layer(si, 0, wl, _fresh(wl), p, per_head=True)
    H.check_per_head(ds.seq, si, 0, wl, ref)


def test_per_head_trajectory_with_per_group_metadata():
    """Four steps of a 28-layer trajectory in the per-KV-head mode: after the
    first compaction every group's cache holds its own tokens, so the next
    step's metadata has one row per group (meta_group_stride = L).  The MI and
    temporal EMAs are carried on both sides."""
    wl = syn.WORKLOADS["trajectory"]
    h = H.hyper(n_warmup=1, n_ramp=2)
    p = H.oracle_params(h)
    st = sk.init_state(H.gpu_config(wl, h, per_head=True))
    sampled = (2, 19)
    ost = {l: _fresh(wl) for l in sampled}
    si = syn.make_sequence(wl)
    G = wl.n_kv_heads
    phis = []
    for step in range(4):
        ds = H.device_seq(si, wl, per_head=True)
        _step(st, [ds])
        for l in sampled:
            ref = H.oracle_layer(si, l, wl, ost[l], p, per_head=True)
            H.check_per_head(ds.seq, si, l, wl, ref)
            phis.append(float(np.max(ref["phi"])))
        lp = si.L - wl.window
        layouts = []
        for l in range(wl.n_layers):
            idx = ds.seq.idx[l].cpu().numpy()
            lay = si.layout[l]
            per_g = lay if isinstance(lay, list) else [lay] * G
            layouts.append([per_g[g].take(np.concatenate([idx[g], np.arange(lp, si.L)])) for g in range(G)])
        si = syn.append_step(wl, ds.seq.k_out.cpu(), ds.seq.v_out.cpu(), layouts, step + 1,
                             si.n_visual_history)
    assert max(phis) > 0.0


def test_meta_group_stride_needs_the_per_head_mode():
    wl = syn.WORKLOADS["tiny"]
    si = syn.make_sequence(wl)
    h = H.hyper()
    st = sk.init_state(H.gpu_config(wl, h))
    ds = H.device_seq(si, wl)
    ds.seq.meta_group_stride = si.L
    with pytest.raises(sk.StarkvError) as e:
        sk.step(st, [ds.seq], sk.workspace(st, [ds.seq]))
    assert e.value.status == sk.ERR_INVALID_ARG


def test_per_head_with_supplied_normalisers():
    """Per-KV-head selection on top of the supplied-normaliser path (first
    scoring pass skipped)."""
    wl = syn.WORKLOADS["uitars_layer"]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    lse = O.window_lse(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window)
    st = sk.init_state(H.gpu_config(wl, h, per_head=True))
    ds = H.device_seq(si, wl, per_head=True)
    ds.seq.lse = torch.from_numpy(lse.astype(np.float32))[None].cuda()
    sk.kernel_times(st)
    _step(st, [ds])
    assert sk.kernel_times(st)["score_lse"][0] == 0
    S = O.score_layer(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window, p,
                      lse=lse.astype(np.float32).astype(np.float64))
    ref = H.oracle_layer(si, 0, wl, _fresh(wl), p, S_override=S, per_head=True)
    H.check_per_head(ds.seq, si, 0, wl, ref)


def test_per_head_sixteen_ragged_trajectories():
    """16 independent sequences of different lengths and budgets in one
    batched per-KV-head step over 28 layers; sampled (sequence, layer) pairs."""
    wl = syn.WORKLOADS["ragged"]
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    sis = [syn.make_sequence(wl, seq=i) for i in range(wl.n_seqs)]
    st = sk.init_state(H.gpu_config(wl, h, max_seqs=wl.n_seqs, per_head=True))
    dss = [H.device_seq(si, wl, slot=i, per_head=True) for i, si in enumerate(sis)]
    _step(st, dss)
    lens = [si.L for si in sis]
    for i, layer in ((int(np.argmin(lens)), 5), (int(np.argmax(lens)), 22)):
        ref = H.oracle_layer(sis[i], layer, wl, _fresh(wl), p, per_head=True)
        H.check_per_head(dss[i].seq, sis[i], layer, wl, ref)
