"""GPU parity of the supplied-normaliser path: when every sequence gives the
log-sum-exp of each window row over the past keys (what the layer's own
prefill attention computes), the first scoring pass is skipped and the second
uses the given normalisers.  Checked against the oracle fed the same
normalisers, against the full GPU path, and for actually using the input."""
import math

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


def _oracle_lse(si, wl, layers):
    """[n_layers][H][w] fp32 from the fp64 oracle (layers not listed: zeros)."""
    nl = si.k.shape[0]
    out = np.zeros((nl, wl.n_heads, wl.window), np.float32)
    for l in layers:
        out[l] = O.window_lse(si.q[l].double().numpy(), si.k[l].double().numpy(), wl.window)
    return torch.from_numpy(out)


def _run(st, ds, lse=None):
    if lse is not None:
        ds.seq.lse = lse.cuda()
    sk.kernel_times(st)
    sk.step(st, [ds.seq], sk.workspace(st, [ds.seq]))
    torch.cuda.synchronize()
    sk.check_device_error(st)
    return sk.kernel_times(st)


@pytest.mark.parametrize("name", ["tiny", "uitars_layer"])
def test_step_with_supplied_normalisers_matches_oracle(name):
    wl = syn.WORKLOADS[name]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    lse = _oracle_lse(si, wl, range(si.k.shape[0]))
    st = sk.init_state(H.gpu_config(wl, h))
    ds = H.device_seq(si, wl)
    kt = _run(st, ds, lse)
    assert kt["score_lse"][0] == 0 and kt["score_accum"][0] == 1   # the first pass is skipped
    S = O.score_layer(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window, p,
                      lse=lse[0].double().numpy())
    ref = H.oracle_layer(si, 0, wl, O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols), p,
                         S_override=S)
    S_gpu = ds.seq.S[0].double().cpu().numpy()
    assert (np.abs(S_gpu - S) / np.abs(S)).max() < 1e-3
    sc = H.check_scores(ds.seq.score[0].double().cpu().numpy(), ref, S, si, 0, wl, p)
    assert sc["ok"], sc
    assert H.check_index_set(ds.seq.idx[0].cpu().numpy(), ref, si.budget)["ok"]
    H.check_compaction(ds.seq, si, 0, wl.window)


def test_supplied_normalisers_agree_with_the_computed_ones_at_the_benchmark_shape():
    """28 layers: the step with the oracle's normalisers against the full GPU
    step (S within 1e-5 relative: the same second pass, normalisers that agree
    to fp32 rounding), and sampled layers against the oracle."""
    wl = syn.WORKLOADS["uitars_5shot_28l"]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    lse = _oracle_lse(si, wl, range(wl.n_layers))
    st_a = sk.init_state(H.gpu_config(wl, h))
    full = H.device_seq(si, wl)
    _run(st_a, full)
    st_b = sk.init_state(H.gpu_config(wl, h))
    given = H.device_seq(si, wl)
    kt = _run(st_b, given, lse)
    assert kt["score_lse"][0] == 0
    Sa, Sb = full.seq.S.double().cpu().numpy(), given.seq.S.double().cpu().numpy()
    assert (np.abs(Sb - Sa) / np.abs(Sa)).max() < 1e-5
    for layer in (0, 27):
        ref = H.oracle_layer(si, layer, wl, O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols), p)
        sc = H.check_scores(given.seq.score[layer].double().cpu().numpy(), ref, ref["S"], si, layer, wl, p)
        assert sc["ok"], (layer, sc)
        assert H.check_index_set(given.seq.idx[layer].cpu().numpy(), ref, si.budget)["ok"]
        H.check_compaction(given.seq, si, layer, wl.window)


def test_the_supplied_normalisers_are_used():
    """Normalisers larger by ln 2 halve every row's contribution, so S halves."""
    wl = syn.WORKLOADS["uitars_layer"]
    si = syn.make_sequence(wl)
    h = H.hyper()
    lse = _oracle_lse(si, wl, [0])
    out = []
    for shift in (0.0, math.log(2.0)):
        st = sk.init_state(H.gpu_config(wl, h))
        ds = H.device_seq(si, wl)
        _run(st, ds, lse + shift)
        out.append(ds.seq.S[0].double().cpu().numpy())
    np.testing.assert_allclose(out[1], out[0] / 2, rtol=1e-5)


def test_host_buffer_step_with_supplied_normalisers():
    wl = syn.WORKLOADS["uitars_layer"]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0)
    lse = _oracle_lse(si, wl, [0])
    st_d = sk.init_state(H.gpu_config(wl, h))
    ds = H.device_seq(si, wl)
    _run(st_d, ds, lse)
    d = ds.seq

    def host(t):
        o = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
        o.copy_(t.cpu())
        return o

    hs = sk.Seq(k=host(d.k), v=host(d.v), q=host(d.q), meta=host(d.meta), meta_layer_stride=d.meta_layer_stride,
                L=d.L, cur_frame=d.cur_frame, budget=d.budget, slot=0, lse=host(lse),
                k_out=torch.empty(d.k_out.shape, dtype=d.k_out.dtype, pin_memory=True),
                v_out=torch.empty(d.v_out.shape, dtype=d.v_out.dtype, pin_memory=True),
                meta_out=torch.empty(d.meta_out.shape, dtype=d.meta_out.dtype, pin_memory=True),
                idx=torch.empty(d.idx.shape, dtype=d.idx.dtype, pin_memory=True),
                S=torch.empty(d.S.shape, dtype=d.S.dtype, pin_memory=True))
    st_h = sk.init_state(H.gpu_config(wl, h))
    sk.kernel_times(st_h)
    sk.step_host(st_h, [hs], sk.workspace(st_h, [hs], host=True))
    torch.cuda.synchronize()
    sk.check_device_error(st_h)
    assert sk.kernel_times(st_h)["score_lse"][0] == 0
    np.testing.assert_allclose(hs.S.numpy(), d.S.cpu().numpy(), rtol=1e-5, atol=0)
    assert torch.equal(hs.idx, d.idx.cpu())
    assert torch.equal(hs.k_out, d.k_out.cpu()) and torch.equal(hs.v_out, d.v_out.cpu())
