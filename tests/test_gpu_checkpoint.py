"""Checkpoint / resume of a trajectory slot: the carried state (step counters,
MI EMAs, temporal EMAs m_g) exported from one state and imported into a slot
of another continues the trajectory with bit-identical results; mismatched or
damaged buffers are rejected before any copy."""
import dataclasses

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


OUTPUTS = ("S", "score", "idx", "k_out", "v_out", "meta_out", "stats")
WL = dataclasses.replace(syn.WORKLOADS["uitars_5shot_28l"], n_layers=4)
HYP = H.hyper(n_warmup=1, n_ramp=2)   # lambda moves with the step counter


def _call(st, ds, ws):
    sk.step(st, [ds.seq], ws)
    torch.cuda.synchronize()
    sk.check_device_error(st)
    return {n: getattr(ds.seq, n).clone() for n in OUTPUTS}


def test_a_resumed_slot_continues_the_trajectory_bit_for_bit():
    si = syn.make_sequence(WL)
    st_a = sk.init_state(H.gpu_config(WL, HYP))
    a = H.device_seq(si, WL)
    ws_a = sk.workspace(st_a, [a.seq])
    for _ in range(2):
        _call(st_a, a, ws_a)
    buf = sk.export_slot(st_a, 0)
    torch.cuda.synchronize()
    hdr = sk.CSlotHeader.from_buffer_copy(buf.numpy().tobytes()[:32])
    assert (hdr.magic, hdr.version, hdr.n_layers, hdr.n_kv_heads, hdr.grid_rows, hdr.grid_cols) == \
        (sk.SLOT_MAGIC, 1, WL.n_layers, WL.n_kv_heads, WL.grid_rows, WL.grid_cols)
    n = np.frombuffer(buf.numpy().tobytes()[32:32 + 4 * WL.n_layers], dtype=np.int32)
    assert np.all(n == 2)                      # two steps seen by every layer
    # resume in slot 1 of another state; a fresh slot 0 there shows the state matters
    st_b = sk.init_state(H.gpu_config(WL, HYP, max_seqs=2))
    sk.import_slot(st_b, 1, buf)
    b = H.device_seq(si, WL, slot=1)
    fresh = H.device_seq(si, WL, slot=0)
    ws_b = sk.workspace(st_b, [b.seq])
    want = _call(st_a, a, ws_a)
    got = _call(st_b, b, ws_b)
    for k in OUTPUTS:
        assert torch.equal(want[k], got[k]), k
    other = _call(st_b, fresh, ws_b)
    assert not torch.equal(other["score"], want["score"])
    # the resumed slot's state moved on exactly as the original's
    again_a, again_b = sk.export_slot(st_a, 0), sk.export_slot(st_b, 1)
    torch.cuda.synchronize()
    assert torch.equal(again_a, again_b)


def test_mismatched_or_damaged_slot_buffers_are_rejected():
    st = sk.init_state(H.gpu_config(WL, HYP))
    buf = sk.export_slot(st, 0)
    torch.cuda.synchronize()
    other_shape = dataclasses.replace(WL, grid_rows=26, grid_cols=26)
    st2 = sk.init_state(H.gpu_config(other_shape, HYP))
    bad = [(st2, buf)]                                    # another patch grid
    damaged = buf.clone()
    damaged[0] ^= 0xFF                                    # magic
    bad.append((st, damaged))
    bad.append((st, buf[: buf.numel() - 8].clone()))       # too short
    for s, b in bad:
        with pytest.raises(sk.StarkvError) as e:
            sk.import_slot(s, 0, b)
        assert e.value.status == sk.ERR_INVALID_ARG
    with pytest.raises(sk.StarkvError) as e:
        sk.import_slot(st, 1, buf)                        # slot out of range
    assert e.value.status == sk.ERR_INVALID_ARG
