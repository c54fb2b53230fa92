"""GPU parity at the full sizes of the five workload configs, through the C ABI
in the launch configuration the benchmark times: one starkv_step over every
layer of every sequence.  The layers and sequences of a step are independent
(Algorithm 1 runs per layer), so the fp64 oracle checks sampled layers /
sequences exactly as the single-layer tests do: fused scores within 1e-3
relative, index sets equal except ties inside that band, compacted K/V/meta
bit copies of the GPU's own selection."""
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


def _step(st, dss):
    ws = sk.workspace(st, [d.seq for d in dss])
    sk.step(st, [d.seq for d in dss], ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)


def _check(ds, si, layer, wl, ost, p, S=None):
    ref = H.oracle_layer(si, layer, wl, ost, p, S_override=S)
    sc = H.check_scores(ds.seq.score[layer].double().cpu().numpy(), ref, ref["S"], si, layer, wl, p)
    assert sc["ok"], (layer, sc)
    ix = H.check_index_set(ds.seq.idx[layer].cpu().numpy(), ref, si.budget)
    assert ix["ok"], (layer, ix)
    H.check_compaction(ds.seq, si, layer, wl.window)
    return ref


@pytest.mark.parametrize("sched", ["paper", "prior_on"])
def test_28_layer_step_at_the_benchmark_shape(sched):
    """Config 2 over the 28-layer stack (the benchmark's workload)."""
    wl = syn.WORKLOADS["uitars_5shot_28l"]
    si = syn.make_sequence(wl)
    h = H.hyper() if sched == "paper" else H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    st = sk.init_state(H.gpu_config(wl, h))
    ds = H.device_seq(si, wl)
    _step(st, [ds])
    for layer in (0, 13, 27):
        _check(ds, si, layer, wl, O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols), p)


def test_ten_step_trajectory_carries_the_state():
    """Config 3: 28 layers, 10 steps; each step appends a screenshot and 64 text
    tokens to the compressed cache and re-compresses, with the MI and temporal
    EMAs carried.  Both sides see the same cache each step (the GPU's
    compaction, which is checked bit-exact)."""
    wl = syn.WORKLOADS["trajectory"]
    h = H.hyper(n_warmup=2, n_ramp=3)
    p = H.oracle_params(h)
    st = sk.init_state(H.gpu_config(wl, h))
    sampled = (4, 21)
    ost = {l: O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols) for l in sampled}
    si = syn.make_sequence(wl)
    phis = []
    for step in range(wl.steps):
        ds = H.device_seq(si, wl)
        _step(st, [ds])
        for l in sampled:
            ref = _check(ds, si, l, wl, ost[l], p)
            phis.append(float(np.max(ref["phi"])))
        if step + 1 == wl.steps:
            break
        lp = si.L - wl.window
        layouts = []
        for l in range(wl.n_layers):
            rows = np.concatenate([ds.seq.idx[l].cpu().numpy(), np.arange(lp, si.L)])
            layouts.append(si.layout[l].take(rows))
        si = syn.append_step(wl, ds.seq.k_out.cpu(), ds.seq.v_out.cpu(), layouts, step + 1,
                             si.n_visual_history)
    assert max(phis) > 0.0   # the temporal discount took part


@pytest.mark.parametrize("pct", [10, 20, 40])
def test_long_cache_budget_sweep(pct, long_input):
    """Config 4: 20 screenshots + 2,048 text tokens (L_p = 56,096) on 28 layers,
    per-frame bump amplitude in [0.5, 4], budgets 10 / 20 / 40 %."""
    wl, si, S7 = long_input
    si.budget = syn.budget(pct, si.n_visual_history, si.L - wl.window)
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    st = sk.init_state(H.gpu_config(wl, h))
    ds = H.device_seq(si, wl)
    _step(st, [ds])
    _check(ds, si, 7, wl, O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols), p, S=S7)


@pytest.fixture(scope="module")
def long_input():
    wl = syn.WORKLOADS["long"]
    si = syn.make_sequence(wl)
    p = H.oracle_params(H.hyper())
    S7 = O.score_layer(si.q[7].double().numpy(), si.k[7].double().numpy(), wl.window, p)
    return wl, si, S7


def test_sixteen_ragged_trajectories():
    """Config 5: 16 independent sequences (1-12 screenshots, 128-1,024 text
    tokens, budgets 10/20/30 %) in one batched step over 28 layers."""
    wl = syn.WORKLOADS["ragged"]
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    sis = [syn.make_sequence(wl, seq=i) for i in range(wl.n_seqs)]
    st = sk.init_state(H.gpu_config(wl, h, max_seqs=wl.n_seqs))
    dss = [H.device_seq(si, wl, slot=i) for i, si in enumerate(sis)]
    _step(st, dss)
    lens = [si.L for si in sis]
    for i, layer in ((int(np.argmin(lens)), 3), (int(np.argmax(lens)), 26), (5, 14)):
        _check(dss[i], sis[i], layer, wl, O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols), p)
