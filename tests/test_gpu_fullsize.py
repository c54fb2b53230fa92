"""GPU parity at the full sizes of the five workload configs, through the C ABI
in the launch configuration the benchmark times: one starkv_step over every
layer of every sequence.  The fp64 oracle (run on a pool of spawned worker
processes, one layer per job) checks every layer of the 28-layer benchmark
step, every layer of the first and last steps of the 10-step trajectory (the
oracle carries every layer's state through all ten), one layer of each of the
16 ragged sequences (the layer rotating over the stack) and a deep layer of
the long cache at each budget, with the single-layer rules: fused scores
within 1e-3 relative, index sets equal except ties inside that band,
compacted K/V/meta bit copies of the GPU's own selection."""
import numpy as np
import pytest
import torch

from oracle import starkv_oracle as O
from paper_2606_01790_gb300 import starkv as sk
from paper_2606_01790_gb300 import synthetic as syn

import harness as H
import oracle_pool as OP

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


@pytest.fixture(scope="module")
def pool():
    pl = OP.OraclePool()
    yield pl
    pl.close()


def _check(ds, si, layer, wl, ost, p, S=None, ref=None):
    if ref is None:
        ref = H.oracle_layer(si, layer, wl, ost, p, S_override=S)
    sc = H.check_scores(ds.seq.score[layer].double().cpu().numpy(), ref, ref["S"], si, layer, wl, p)
    assert sc["ok"], (layer, sc)
    ix = H.check_index_set(ds.seq.idx[layer].cpu().numpy(), ref, si.budget)
    assert ix["ok"], (layer, ix)
    H.check_compaction(ds.seq, si, layer, wl.window)
    return ref


@pytest.mark.parametrize("sched", ["paper", "prior_on"])
def test_28_layer_step_at_the_benchmark_shape(sched, pool):
    """Config 2 over the 28-layer stack (the benchmark's workload): every layer."""
    wl = syn.WORKLOADS["uitars_5shot_28l"]
    si = syn.make_sequence(wl)
    h = H.hyper() if sched == "paper" else H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    st = sk.init_state(H.gpu_config(wl, h))
    ds = H.device_seq(si, wl)
    _step(st, [ds])
    fresh = lambda: O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols)
    refs = pool.map([OP.layer_job(si, l, wl, fresh(), p) for l in range(wl.n_layers)])
    for layer, (ref, _) in enumerate(refs):
        _check(ds, si, layer, wl, None, p, ref=ref)


def test_ten_step_trajectory_carries_the_state(pool):
    """Config 3: 28 layers, 10 steps; each step appends a screenshot and 64 text
    tokens to the compressed cache and re-compresses, with the MI and temporal
    EMAs carried.  Both sides see the same cache each step (the GPU's
    compaction, which is checked bit-exact); the oracle carries every layer's
    state and every layer is checked on the first and the last step."""
    wl = syn.WORKLOADS["trajectory"]
    h = H.hyper(n_warmup=2, n_ramp=3)
    p = H.oracle_params(h)
    st = sk.init_state(H.gpu_config(wl, h))
    ost = [O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols) for _ in range(wl.n_layers)]
    si = syn.make_sequence(wl)
    phis, checked = [], 0
    for step in range(wl.steps):
        ds = H.device_seq(si, wl)
        _step(st, [ds])
        res = pool.map([OP.layer_job(si, l, wl, ost[l], p) for l in range(wl.n_layers)])
        for l, (ref, st_l) in enumerate(res):
            ost[l] = st_l
            phis.append(float(np.max(ref["phi"])))
            if step in (0, wl.steps - 1):
                _check(ds, si, l, wl, None, p, ref=ref)
                checked += 1
        if step + 1 == wl.steps:
            break
        lp = si.L - wl.window
        layouts = []
        for l in range(wl.n_layers):
            rows = np.concatenate([ds.seq.idx[l].cpu().numpy(), np.arange(lp, si.L)])
            layouts.append(si.layout[l].take(rows))
        si = syn.append_step(wl, ds.seq.k_out.cpu(), ds.seq.v_out.cpu(), layouts, step + 1,
                             si.n_visual_history)
    assert checked == 2 * wl.n_layers
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


def test_sixteen_ragged_trajectories(pool):
    """Config 5: 16 independent sequences (1-12 screenshots, 128-1,024 text
    tokens, budgets 10/20/30 %) in one batched step over 28 layers; one layer
    of every sequence is checked, the layer rotating over the stack."""
    wl = syn.WORKLOADS["ragged"]
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    sis = [syn.make_sequence(wl, seq=i) for i in range(wl.n_seqs)]
    st = sk.init_state(H.gpu_config(wl, h, max_seqs=wl.n_seqs))
    dss = [H.device_seq(si, wl, slot=i) for i, si in enumerate(sis)]
    _step(st, dss)
    fresh = lambda: O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols)
    layers = [(11 * i) % wl.n_layers for i in range(wl.n_seqs)]
    refs = pool.map([OP.layer_job(si, l, wl, fresh(), p) for si, l in zip(sis, layers)])
    for i, (l, (ref, _)) in enumerate(zip(layers, refs)):
        _check(dss[i], sis[i], l, wl, None, p, ref=ref)
