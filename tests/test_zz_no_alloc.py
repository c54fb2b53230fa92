"""The scoring call for callers that cannot allocate device memory
(starkv_score_layer_noalloc): some callers run where cudaMalloc is forbidden
or unavailable, for example inside another runtime that owns every device
allocation.  This call must give the same group score map as the regular call
with a caller workspace, bit for bit (the scoring path is deterministic), call
after call, with the window normalisers computed or supplied; it must leave the
device's free memory unchanged, and it must refuse batches larger than its
static scratch.  Collected last on purpose: it must pass alone in a fresh
process and after every other test."""
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


def _noalloc_twice_against(st, ds, ref):
    """Two no-allocation calls in a row, each bit-identical to ``ref``; the
    first one (after a synchronize) must change neither the device's free
    memory nor torch's allocated bytes."""
    for i in range(2):
        ds.seq.S.fill_(float("nan"))
        torch.cuda.synchronize()
        free0, alloc0 = torch.cuda.mem_get_info()[0], torch.cuda.memory_allocated()
        sk.score_layer_noalloc(st, 0, [ds.seq])
        torch.cuda.synchronize()
        if i == 0:
            assert torch.cuda.mem_get_info()[0] == free0, "the call allocated device memory"
            assert torch.cuda.memory_allocated() == alloc0
        sk.check_device_error(st)
        assert torch.equal(ds.seq.S, ref), "differs from the workspace call"


def test_noalloc_scoring_matches_workspace_call_on_two_calls_in_a_row():
    wl = syn.WORKLOADS["uitars_layer"]
    si = syn.make_sequence(wl)
    st = sk.init_state(H.gpu_config(wl, H.hyper()))
    ds = H.device_seq(si, wl)
    ws = sk.workspace(st, [ds.seq])
    sk.score_layer(st, 0, [ds.seq], ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)
    ref = ds.seq.S.clone()
    assert torch.isfinite(ref).all()
    _noalloc_twice_against(st, ds, ref)
    st.close()


def test_noalloc_scoring_with_supplied_normalisers():
    """With the window rows' normalisers supplied (the prefill pass's
    log-sum-exp; here the oracle's), the first scoring pass is skipped and only
    the unpooled sums live in the static scratch."""
    wl = syn.WORKLOADS["uitars_layer"]
    si = syn.make_sequence(wl)
    st = sk.init_state(H.gpu_config(wl, H.hyper()))
    ds = H.device_seq(si, wl)
    lse = O.window_lse(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window)
    ds.seq.lse = torch.from_numpy(lse.astype(np.float32))[None].cuda()
    ws = sk.workspace(st, [ds.seq])
    sk.kernel_times(st)   # reset the launch counters
    sk.score_layer(st, 0, [ds.seq], ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)
    assert sk.kernel_times(st)["score_lse"][0] == 0, "pass 1 ran although the normalisers were given"
    ref = ds.seq.S.clone()
    assert torch.isfinite(ref).all()
    _noalloc_twice_against(st, ds, ref)
    assert sk.kernel_times(st)["score_lse"][0] == 0
    st.close()


def test_noalloc_rejects_a_batch_beyond_its_static_scratch():
    wl = syn.WORKLOADS["uitars_layer"]
    si = syn.make_sequence(wl)
    n = 16  # ~1.8 MB of scratch each at this shape: more than 16 MiB together
    st = sk.init_state(H.gpu_config(wl, H.hyper(), max_seqs=n))
    seqs = [H.device_seq(si, wl, slot=i, with_score=False, with_stats=False).seq for i in range(n)]
    with pytest.raises(sk.StarkvError) as e:
        sk.score_layer_noalloc(st, 0, seqs)
    assert e.value.status == sk.ERR_UNSUPPORTED
    assert "static scratch" in str(e.value)
    st.close()
