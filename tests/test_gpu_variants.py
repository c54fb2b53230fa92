"""GPU parity of the ablation variants (linear and power-law temporal decay,
peak-confidence temperature, MI over the newest frame) against the oracle's
same readings.  Two calls on the same cache, so that the second has a
temporal state (phi > 0) and the decay shape matters."""
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


@pytest.mark.parametrize("variant", [dict(decay_mode=1), dict(decay_mode=2), dict(aeb_mode=1),
                                     dict(mi_span=1), dict(decay_mode=2, aeb_mode=1, mi_span=1)])
@pytest.mark.parametrize("per_head", [False, True])
def test_variant_matches_oracle_over_two_calls(variant, per_head):
    wl = syn.WORKLOADS["uitars_layer"]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0, t_min=0.75, t_max=1.25, **variant)
    p = H.oracle_params(h)
    st = sk.init_state(H.gpu_config(wl, h, per_head=per_head))
    ost = O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols)
    G = wl.n_kv_heads
    for call in range(2):
        ds = H.device_seq(si, wl, per_head=per_head)
        sk.step(st, [ds.seq], sk.workspace(st, [ds.seq]))
        torch.cuda.synchronize()
        sk.check_device_error(st)
        ref = H.oracle_layer(si, 0, wl, ost, p, per_head=per_head)
        stats = ds.seq.stats[0].double().cpu().numpy()
        if per_head:
            H.check_per_head(ds.seq, si, 0, wl, ref)
            np.testing.assert_allclose(stats[8 + 4 * G:8 + 5 * G], ref["H"], rtol=1e-4, atol=1e-6)
        else:
            sc = H.check_scores(ds.seq.score[0].double().cpu().numpy(), ref, ref["S"], si, 0, wl, p)
            assert sc["ok"], (call, sc)
            assert H.check_index_set(ds.seq.idx[0].cpu().numpy(), ref, si.budget)["ok"]
            H.check_compaction(ds.seq, si, 0, wl.window)
            assert abs(stats[0] - ref["H"]) < 1e-4 * max(1.0, abs(ref["H"])) and abs(stats[1] - ref["T"]) < 1e-4
        np.testing.assert_allclose(stats[8:8 + G], ref["mi"], rtol=2e-3, atol=2e-4)
        np.testing.assert_allclose(stats[8 + 3 * G:8 + 4 * G], ref["phi"], atol=1e-4)
    assert np.max(ref["phi"]) > 0.0   # the second call has a temporal state
    if "decay_mode" in variant:
        d = ref["D"]
        assert np.ptp(d) > 1e-3        # the decay shape took part


def test_variants_on_a_row_longer_than_shared_memory():
    """20 screenshots + 2,048 text tokens (L_p = 56,096): the calibration keeps
    its per-token arrays in the workspace; the decay and MI-span switches on
    that path, over two calls."""
    wl = syn.WORKLOADS["long_layer"]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0, decay_mode=1, mi_span=1, aeb_mode=1)
    p = H.oracle_params(h)
    S = O.score_layer(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window, p)
    st = sk.init_state(H.gpu_config(wl, h))
    ost = O.LayerState.fresh(wl.n_kv_heads, wl.grid_rows, wl.grid_cols)
    for call in range(2):
        ds = H.device_seq(si, wl)
        sk.step(st, [ds.seq], sk.workspace(st, [ds.seq]))
        torch.cuda.synchronize()
        sk.check_device_error(st)
        ref = H.oracle_layer(si, 0, wl, ost, p, S_override=S)
        sc = H.check_scores(ds.seq.score[0].double().cpu().numpy(), ref, S, si, 0, wl, p)
        assert sc["ok"], (call, sc)
        assert H.check_index_set(ds.seq.idx[0].cpu().numpy(), ref, si.budget)["ok"]
        H.check_compaction(ds.seq, si, 0, wl.window)
    assert np.max(ref["phi"]) > 0.0
