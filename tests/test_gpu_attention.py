"""GPU parity of the window-attention producer (starkv_window_attention): the
attention output of the w window rows over the past keys and its normaliser,
the pass whose logits Eq. (2) scores (App. A.3: Q K^T shared with the
attention).  Checked against the fp64 oracle (``window_attention_output``,
``window_lse``):

* lse within 1e-5 + 1e-6 |lse| (natural log; fp32 resolves a normaliser of
  size |lse| to about 1e-7 |lse|, and the wide-logit case reaches |lse| ~ 200);
* every output element within the bound its arithmetic gives: P is rounded to
  fp16 (unit roundoff 2^-11) before the P V product, so
  |O_gpu - O| <= 2^-11 sum_t p_t |V_t| plus fp32 slack; and every row within
  1e-3 in relative norm;
* the compression step fed this normaliser matches the oracle as the
  supplied-normaliser path does, and matches the step that computes its own.
"""
import dataclasses
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

U_P = 2.0 ** -11     # unit roundoff of the fp16 P
LSE_TOL = 1e-5      # absolute, plus LSE_REL |lse|
LSE_REL = 1e-6


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()


def _outputs(si, wl, dev="cuda"):
    nl, H_, w = si.k.shape[0], wl.n_heads, wl.window
    return (torch.full((nl, H_, w, wl.head_dim), float("nan"), dtype=torch.float32, device=dev),
            torch.full((nl, H_, w), float("nan"), dtype=torch.float32, device=dev))


def _run_attention(st, dss):
    ws = sk.workspace(st, [d.seq for d in dss])
    sk.kernel_times(st)
    sk.window_attention(st, [d.seq for d in dss], ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)
    return sk.kernel_times(st)


def _attach(ds, si, wl):
    ds.seq.attn_o, ds.seq.attn_lse = _outputs(si, wl)
    return ds


def check_layer(ds, si, wl, layer):
    """The layer's output and normaliser against the oracle; returns the
    largest element error as a fraction of its bound and the largest row
    relative error."""
    q, k, v = (x[layer].double().numpy() for x in (si.q, si.k, si.v))
    w, d = wl.window, wl.head_dim
    lp = si.L - w
    ref_o = O.window_attention_output(q, k, v, w)
    ref_lse = O.window_lse(q, k, w)
    got_o = ds.seq.attn_o[layer].double().cpu().numpy()
    got_lse = ds.seq.attn_lse[layer].double().cpu().numpy()
    if lp == 0:
        assert np.all(got_lse == -np.inf) and np.all(got_o == 0.0)
        return 0.0, 0.0
    np.testing.assert_allclose(got_lse, ref_lse, rtol=LSE_REL, atol=LSE_TOL)
    G = k.shape[0]
    worst_bound, worst_row = 0.0, 0.0
    for h in range(wl.n_heads):
        g = h * G // wl.n_heads
        z = q[h] @ k[g, :lp].T / math.sqrt(d)
        pz = np.exp(z - ref_lse[h][:, None])                     # softmax weights
        bound = U_P * (pz @ np.abs(v[g, :lp])) + 1e-6 * (pz @ np.abs(v[g, :lp])) + 1e-7
        err = np.abs(got_o[h] - ref_o[h])
        worst_bound = max(worst_bound, float((err / bound).max()))
        row = np.linalg.norm(got_o[h] - ref_o[h], axis=1) / np.maximum(np.linalg.norm(ref_o[h], axis=1), 1e-30)
        worst_row = max(worst_row, float(row.max()))
    assert worst_bound <= 1.0, (layer, worst_bound)
    assert worst_row <= 1e-3, (layer, worst_row)
    return worst_bound, worst_row


@pytest.mark.parametrize("name", ["tiny", "uitars_layer"])
def test_attention_matches_oracle(name):
    wl = syn.WORKLOADS[name]
    si = syn.make_sequence(wl)
    st = sk.init_state(H.gpu_config(wl, H.hyper()))
    ds = _attach(H.device_seq(si, wl), si, wl)
    kt = _run_attention(st, [ds])
    assert kt["attention"][0] == 1 and kt["attn_combine"][0] == 1
    check_layer(ds, si, wl, 0)
    st.close()


def test_attention_without_output_buffer_writes_the_normaliser_only():
    wl = syn.WORKLOADS["tiny"]
    si = syn.make_sequence(wl)
    st = sk.init_state(H.gpu_config(wl, H.hyper()))
    ds = _attach(H.device_seq(si, wl), si, wl)
    ds.seq.attn_o = None
    _run_attention(st, [ds])
    ref = O.window_lse(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window)
    np.testing.assert_allclose(ds.seq.attn_lse[0].double().cpu().numpy(), ref, rtol=LSE_REL, atol=LSE_TOL)
    st.close()


def test_attention_with_wide_logits_moves_the_reference():
    """Queries scaled by 32: logits spread over hundreds of log2 units, so the
    row references move often (each move rescales O in tensor memory) and the
    pieces of a row merge from very different references."""
    wl = syn.WORKLOADS["uitars_layer"]
    si = syn.make_sequence(wl)
    si.q = (si.q.float() * 32).to(torch.bfloat16)
    st = sk.init_state(H.gpu_config(wl, H.hyper()))
    ds = _attach(H.device_seq(si, wl), si, wl)
    _run_attention(st, [ds])
    check_layer(ds, si, wl, 0)
    st.close()


def test_attention_at_the_28_layer_benchmark_shape():
    wl = syn.WORKLOADS["uitars_5shot_28l"]
    si = syn.make_sequence(wl)
    st = sk.init_state(H.gpu_config(wl, H.hyper()))
    ds = _attach(H.device_seq(si, wl), si, wl)
    _run_attention(st, [ds])
    for layer in (0, 13, 27):
        check_layer(ds, si, wl, layer)
    # every layer's normaliser
    for layer in range(wl.n_layers):
        ref = O.window_lse(si.q[layer].double().numpy(), si.k[layer].double().numpy(), wl.window)
        np.testing.assert_allclose(ds.seq.attn_lse[layer].double().cpu().numpy(), ref, rtol=LSE_REL, atol=LSE_TOL)
    st.close()


def test_attention_ragged_batch_with_short_and_empty_histories():
    """Sequences with L_p = 0, L_p below one 64-key unit, ragged last units,
    one long row: pieces of many rows inside one CTA's range and rows split
    over several CTAs."""
    base = syn.WORKLOADS["tiny"]
    shapes = [(0, 8), (0, 20), (1, 8), (2, 64), (1, 200), (3, 17)]   # (screenshots, text tokens)
    sis, dss = [], []
    st = sk.init_state(H.gpu_config(base, H.hyper(), max_seqs=len(shapes)))
    for i, (shots, text) in enumerate(shapes):
        wl = dataclasses.replace(base, name=f"r{i}", cfg_id=200 + i, n_shots=shots, n_text=text)
        si = syn.make_sequence(wl)
        sis.append((si, wl))
        dss.append(_attach(H.device_seq(si, wl, slot=i), si, wl))
    _run_attention(st, dss)
    for (si, wl), ds in zip(sis, dss):
        check_layer(ds, si, wl, 0)
    st.close()


@pytest.mark.parametrize("shape", [(16, 2, 32), (8, 8, 16), (12, 1, 16), (28, 4, 24), (40, 8, 8)],
                         ids=["rows256", "rows16", "rows192", "rows168", "rows40"])
def test_attention_at_other_shapes(shape):
    Hq, G, w = shape
    wl = dataclasses.replace(syn.WORKLOADS["tiny"], n_heads=Hq, n_kv_heads=G, window=w)
    si = syn.make_sequence(wl)
    st = sk.init_state(H.gpu_config(wl, H.hyper()))
    ds = _attach(H.device_seq(si, wl), si, wl)
    _run_attention(st, [ds])
    check_layer(ds, si, wl, 0)
    st.close()


def test_attention_on_a_56k_token_row():
    """The long-cache shape (L_p = 56,096): about 880 units per row, so a
    piece runs over hundreds of units and the references can move late."""
    wl = syn.WORKLOADS["long_layer"]
    si = syn.make_sequence(wl)
    st = sk.init_state(H.gpu_config(wl, H.hyper()))
    ds = _attach(H.device_seq(si, wl), si, wl)
    _run_attention(st, [ds])
    check_layer(ds, si, wl, 0)
    st.close()


def test_attention_at_mha_head_granularity():
    """G = H = 28 (each group's keys and values replicated for its query head):
    32 rows per group, one M tile, 28 groups per layer."""
    wl = syn.WORKLOADS["uitars_layer_mha"]
    si = syn.make_sequence(wl)
    st = sk.init_state(H.gpu_config(wl, H.hyper()))
    ds = _attach(H.device_seq(si, wl), si, wl)
    _run_attention(st, [ds])
    check_layer(ds, si, wl, 0)
    st.close()


def _lifted_keys(si, wl, lift_of_key, seed=7):
    """Queries along one axis and past keys whose logit along it is
    lift_of_key(t) log2 units, the other dimensions small noise."""
    d, lp = wl.head_dim, si.L - wl.window
    g = torch.Generator().manual_seed(seed)
    beta = 8.0
    q = 0.05 * torch.randn(si.q.shape, generator=g)
    q[..., 0] = beta
    k = si.k.float().clone()
    k[..., :lp, :] = 0.05 * torch.randn(k[..., :lp, :].shape, generator=g)
    lift = torch.tensor([lift_of_key(t) for t in range(lp)], dtype=torch.float32)
    k[..., :lp, 0] = lift / (beta / math.sqrt(d) * math.log2(math.e))   # q.k / sqrt(d) = lift / log2(e)
    si.q = q.to(torch.bfloat16)
    si.k = k.to(torch.bfloat16)


@pytest.mark.parametrize("pattern", ["sum_over_guard", "reference_moves"])
def test_attention_keys_far_above_the_reference(pattern):
    """Logits that force the softmax off its fast path, against the fp64
    oracle at the usual bounds.  sum_over_guard: every other 128-key block 10
    log2 units up, so that after a low block the 64 p of a half sum to about
    2^16 although none exceeds 2^15: the maximum is taken and the reference
    stays.  reference_moves: a sawtooth rising 20 log2 units every 64 keys
    (eight steps, then down again), so that references move in the middle of
    pieces, in the first half of a unit (O and the row sum rescaled) and in
    the second (the first half's stored P rescaled too)."""
    wl = syn.WORKLOADS["uitars_layer"]
    si = syn.make_sequence(wl)
    if pattern == "sum_over_guard":
        _lifted_keys(si, wl, lambda t: 10.0 * ((t // 128) % 2))
    else:
        _lifted_keys(si, wl, lambda t: 20.0 * ((t // 64) % 8))
    st = sk.init_state(H.gpu_config(wl, H.hyper()))
    ds = _attach(H.device_seq(si, wl), si, wl)
    _run_attention(st, [ds])
    check_layer(ds, si, wl, 0)
    st.close()


def test_attention_on_sixteen_ragged_sequences():
    """Config 5's batch (16 sequences of 1-12 screenshots and 128-1,024 text
    tokens) in one launch over 28 layers: every sequence's output against the
    oracle on one layer, rotating over the stack, and its normaliser on two
    more."""
    wl = syn.WORKLOADS["ragged"]
    sis = [syn.make_sequence(wl, seq=i) for i in range(wl.n_seqs)]
    st = sk.init_state(H.gpu_config(wl, H.hyper(), max_seqs=wl.n_seqs))
    dss = [_attach(H.device_seq(si, wl, slot=i), si, wl) for i, si in enumerate(sis)]
    kt = _run_attention(st, dss)
    assert kt["attention"][0] == 1   # one launch for the whole batch
    for i, (si, ds) in enumerate(zip(sis, dss)):
        layer = (11 * i) % wl.n_layers
        check_layer(ds, si, wl, layer)
        for extra in ((layer + 9) % wl.n_layers, (layer + 19) % wl.n_layers):
            ref = O.window_lse(si.q[extra].double().numpy(), si.k[extra].double().numpy(), wl.window)
            np.testing.assert_allclose(ds.seq.attn_lse[extra].double().cpu().numpy(), ref, rtol=LSE_REL,
                                       atol=LSE_TOL)
    st.close()


@pytest.mark.parametrize("name", ["tiny", "uitars_layer"])
def test_step_fed_by_the_attention_pass_matches_oracle(name):
    """The compression step with lse = attn_lse: pass 1 skipped, the group
    score map equal to the computing path's to 1e-5, and scores, sets and
    compaction held to the oracle's bars."""
    wl = syn.WORKLOADS[name]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0)
    p = H.oracle_params(h)
    st = sk.init_state(H.gpu_config(wl, h))
    ds = _attach(H.device_seq(si, wl), si, wl)
    _run_attention(st, [ds])
    ds.seq.lse = ds.seq.attn_lse
    ws = sk.workspace(st, [ds.seq])
    sk.kernel_times(st)
    sk.step(st, [ds.seq], ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)
    kt = sk.kernel_times(st)
    assert kt["score_lse"][0] == 0 and kt["score_accum"][0] == 1
    S_fed = ds.seq.S.clone()
    ref = H.oracle_layer(si, 0, wl, O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols), p)
    sc = H.check_scores(ds.seq.score[0].double().cpu().numpy(), ref, ref["S"], si, 0, wl, p)
    assert sc["ok"], sc
    ix = H.check_index_set(ds.seq.idx[0].cpu().numpy(), ref, si.budget)
    assert ix["ok"], ix
    H.check_compaction(ds.seq, si, 0, wl.window)
    # the same inputs through the path that computes its own normalisers
    st2 = sk.init_state(H.gpu_config(wl, h))
    ds2 = H.device_seq(si, wl)
    sk.step(st2, [ds2.seq], sk.workspace(st2, [ds2.seq]))
    torch.cuda.synchronize()
    rel = ((S_fed - ds2.seq.S).abs() / ds2.seq.S.abs().clamp_min(1e-30)).max().item()
    assert rel <= 1e-5, rel
    st.close()
    st2.close()
