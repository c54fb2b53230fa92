"""The scoring call for callers that cannot allocate device memory
(starkv_score_layer_noalloc) gives the same group score map as the regular
call with a caller workspace, call after call, and refuses batches larger than
its static scratch.  Collected last on purpose: it must pass alone in a fresh
process and after every other test."""
import numpy as np
import pytest
import torch

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


def test_noalloc_scoring_matches_workspace_call_on_two_calls_in_a_row():
    wl = syn.WORKLOADS["uitars_layer"]
    si = syn.make_sequence(wl)
    st = sk.init_state(H.gpu_config(wl, H.hyper()))
    ds = H.device_seq(si, wl)
    ws = sk.workspace(st, [ds.seq])
    sk.score_layer(st, 0, [ds.seq], ws)
    torch.cuda.synchronize()
    ref = ds.seq.S.clone()
    for _ in range(2):
        ds.seq.S.fill_(float("nan"))
        sk.score_layer_noalloc(st, 0, [ds.seq])
        torch.cuda.synchronize()
        sk.check_device_error(st)
        got = ds.seq.S
        assert torch.isfinite(got).all()
        rel = ((got - ref).abs() / ref.abs()).max().item()
        assert rel <= H.RTOL, rel
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
