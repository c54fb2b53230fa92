"""GPU parity at attention shapes other than the benchmark's 28 query / 4 KV
heads: other GQA ratios (one KV head, eight KV heads, one query head per KV
head), window lengths whose group row count is not a multiple of 16, and a
group of exactly 256 window rows.  Each shape runs the scoring passes with
one or two M tiles, pass-2 MMA widths from 16 to 256, and calibration
clusters of 1, 2, 4 or 8 CTAs.  Same bars as the benchmark-shape tests:
fused scores within 1e-3 relative of the oracle, index sets equal except ties
inside that band, compacted K/V/metadata bit copies."""
import dataclasses

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


# (query heads H, KV heads G, window w): group rows (H/G)*w
SHAPES = [
    (32, 8, 16),    # 64 rows, clusters of 8
    (16, 2, 32),    # 256 rows: two full M tiles, pass-2 N = 256
    (8, 8, 16),     # one query head per KV head: 16 rows, pass-2 N = 16
    (12, 1, 16),    # one KV head (cluster of 1), 192 rows
    (28, 4, 24),    # 168 rows, padded to 176 columns in pass 2
    (40, 8, 8),     # 40 rows, padded to 48
    (6, 2, 8),      # 24 rows, padded to 32
]


def _workload(Hq, G, w):
    return dataclasses.replace(syn.WORKLOADS["tiny"], n_heads=Hq, n_kv_heads=G, window=w)


@pytest.mark.parametrize("shape", SHAPES, ids=[f"H{a}_G{b}_w{c}" for a, b, c in SHAPES])
def test_global_step_matches_oracle(shape):
    wl = _workload(*shape)
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0, t_min=0.75, t_max=1.25)
    p = H.oracle_params(h)
    st = sk.init_state(H.gpu_config(wl, h))
    ds = H.device_seq(si, wl)
    sk.step(st, [ds.seq], sk.workspace(st, [ds.seq]))
    torch.cuda.synchronize()
    sk.check_device_error(st)
    ref = H.oracle_layer(si, 0, wl, O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols), p)
    S_gpu = ds.seq.S[0].double().cpu().numpy()
    assert (np.abs(S_gpu - ref["S"]) / np.abs(ref["S"])).max() < 1e-3
    sc = H.check_scores(ds.seq.score[0].double().cpu().numpy(), ref, ref["S"], si, 0, wl, p)
    assert sc["ok"], sc
    ix = H.check_index_set(ds.seq.idx[0].cpu().numpy(), ref, si.budget)
    assert ix["ok"], ix
    H.check_compaction(ds.seq, si, 0, wl.window)
    G = wl.n_kv_heads
    stats = ds.seq.stats[0].double().cpu().numpy()
    assert abs(stats[0] - ref["H"]) < 1e-5 and abs(stats[1] - ref["T"]) < 1e-5
    np.testing.assert_allclose(stats[8:8 + G], ref["mi"], rtol=2e-3, atol=2e-4)
    np.testing.assert_allclose(stats[8 + 2 * G:8 + 3 * G], ref["w"], rtol=2e-3)


@pytest.mark.parametrize("shape", SHAPES, ids=[f"H{a}_G{b}_w{c}" for a, b, c in SHAPES])
def test_per_head_step_matches_oracle(shape):
    wl = _workload(*shape)
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0, t_min=0.75, t_max=1.25)
    p = H.oracle_params(h)
    st = sk.init_state(H.gpu_config(wl, h, per_head=True))
    ds = H.device_seq(si, wl, per_head=True)
    sk.step(st, [ds.seq], sk.workspace(st, [ds.seq]))
    torch.cuda.synchronize()
    sk.check_device_error(st)
    ref = H.oracle_layer(si, 0, wl, O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols), p,
                         per_head=True)
    H.check_per_head(ds.seq, si, 0, wl, ref)


def test_supplied_normalisers_at_an_odd_shape():
    """The supplied-normaliser path with 168 rows per group (pass-2 columns
    padded past the group's rows) against the oracle fed the same values."""
    wl = _workload(28, 4, 24)
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    lse = O.window_lse(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window).astype(np.float32)
    st = sk.init_state(H.gpu_config(wl, h))
    ds = H.device_seq(si, wl)
    ds.seq.lse = torch.from_numpy(lse)[None].cuda()
    sk.kernel_times(st)
    sk.step(st, [ds.seq], sk.workspace(st, [ds.seq]))
    torch.cuda.synchronize()
    sk.check_device_error(st)
    assert sk.kernel_times(st)["score_lse"][0] == 0
    S = O.score_layer(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window, p, lse=lse.astype(np.float64))
    S_gpu = ds.seq.S[0].double().cpu().numpy()
    assert (np.abs(S_gpu - S) / np.abs(S)).max() < 1e-3


def test_forty_sequences_span_two_launch_batches():
    """40 ragged sequences in one step: a launch carries at most 32 sequences,
    so the call runs two batches of every kernel (the second with its own
    tensor maps, partial-sum offsets and state slots).  Sampled sequences on
    both sides of the batch boundary against the oracle, in both layers."""
    wl = dataclasses.replace(syn.WORKLOADS["tiny"], n_layers=2, n_seqs=40, ragged=True,
                             shots_range=(1, 3), text_range=(16, 160))
    h = H.hyper(n_warmup=0, n_ramp=0, t_min=0.75, t_max=1.25)
    p = H.oracle_params(h)
    sis = [syn.make_sequence(wl, seq=i) for i in range(wl.n_seqs)]
    assert len({si.L for si in sis}) > 10
    st = sk.init_state(H.gpu_config(wl, h, max_seqs=wl.n_seqs))
    dss = [H.device_seq(si, wl, slot=i) for i, si in enumerate(sis)]
    sk.step(st, [d.seq for d in dss], sk.workspace(st, [d.seq for d in dss]))
    torch.cuda.synchronize()
    sk.check_device_error(st)
    for i in (0, 31, 32, 39):
        for layer in (0, 1):
            ref = H.oracle_layer(sis[i], layer, wl,
                                 O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols), p)
            sc = H.check_scores(dss[i].seq.score[layer].double().cpu().numpy(), ref, ref["S"], sis[i], layer, wl, p)
            assert sc["ok"], (i, layer, sc)
            ix = H.check_index_set(dss[i].seq.idx[layer].cpu().numpy(), ref, sis[i].budget)
            assert ix["ok"], (i, layer, ix)
            H.check_compaction(dss[i].seq, sis[i], layer, wl.window)
