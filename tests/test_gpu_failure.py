"""Failure detection on the GPU without a fault: every bounded device wait of
the kernels shares one failure path (give up after the state's limit, latch
STARKV_ERR_TIMEOUT in the device error word, return).  starkv_selftest_wait
runs that path on a barrier that nothing completes; the host reads the status,
and the same context then runs a normal step that matches the oracle."""
import time

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


def test_a_wait_that_runs_out_reports_timeout_and_the_context_stays_usable():
    wl = syn.WORKLOADS["tiny"]
    si = syn.make_sequence(wl)
    h = H.hyper()
    st = sk.init_state(H.gpu_config(wl, h))
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    sk.selftest_wait(st, 2_000_000)   # 2 ms
    with pytest.raises(sk.StarkvError) as e:
        sk.check_device_error(st)
    dt = time.perf_counter() - t0
    assert e.value.status == sk.ERR_TIMEOUT
    assert 0.002 <= dt < 1.0          # gave up after its limit, not at once and not hung
    sk.check_device_error(st)         # reading the word cleared it
    ds = H.device_seq(si, wl)
    sk.step(st, [ds.seq], sk.workspace(st, [ds.seq]))
    torch.cuda.synchronize()
    sk.check_device_error(st)
    S_ref = O.score_layer(si.q[0].double().numpy(), si.k[0].double().numpy(), wl.window, H.oracle_params(h))
    S_gpu = ds.seq.S[0].double().cpu().numpy()
    assert (np.abs(S_gpu - S_ref) / np.abs(S_ref)).max() < 1e-3


def test_wait_selftest_limit_out_of_range_is_rejected():
    st = sk.init_state(H.gpu_config(syn.WORKLOADS["tiny"], H.hyper()))
    for bad in (10, 2_000_000_000):
        with pytest.raises(sk.StarkvError) as e:
            sk.selftest_wait(st, bad)
        assert e.value.status == sk.ERR_INVALID_ARG
