"""starkv_step_host (every buffer in host memory) against starkv_step on
device buffers: the same kernels on the same inputs, run in layer chunks with
the uploads, the compute and the downloads overlapped.  The scoring launches
then split the key tiles over the CTAs differently, which changes the order in
which the log-sum-exp partials combine, so S and the fused scores agree to
fp32 rounding (1e-5 relative) rather than bit for bit; the index sets agree
except at near ties, and the compacted rows are bit copies of the host run's
own selection.  With V in page-locked memory the gather reads the kept rows in
place; with pageable V it is uploaded."""
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


def _host(t, pin):
    o = torch.empty(t.shape, dtype=t.dtype, pin_memory=pin)
    o.copy_(t)
    return o


@pytest.mark.parametrize("v_pinned", [True, False])
def test_host_buffer_step_matches_device_step(v_pinned):
    wl = syn.WORKLOADS["uitars_5shot_28l"]
    si = syn.make_sequence(wl)
    h = H.hyper(n_warmup=0, n_ramp=0)
    cfg = H.gpu_config(wl, h)
    st_d = sk.init_state(cfg)
    ds = H.device_seq(si, wl)
    sk.step(st_d, [ds.seq], sk.workspace(st_d, [ds.seq]))
    torch.cuda.synchronize()
    sk.check_device_error(st_d)

    d = ds.seq
    hs = sk.Seq(k=_host(d.k.cpu(), True), v=_host(d.v.cpu(), v_pinned), q=_host(d.q.cpu(), True),
                meta=_host(d.meta.cpu(), True), meta_layer_stride=d.meta_layer_stride, L=d.L,
                cur_frame=d.cur_frame, budget=d.budget, slot=0,
                k_out=torch.empty(d.k_out.shape, dtype=d.k_out.dtype, pin_memory=True),
                v_out=torch.empty(d.v_out.shape, dtype=d.v_out.dtype, pin_memory=True),
                meta_out=torch.empty(d.meta_out.shape, dtype=d.meta_out.dtype, pin_memory=True),
                idx=torch.empty(d.idx.shape, dtype=d.idx.dtype, pin_memory=True),
                S=torch.empty(d.S.shape, dtype=d.S.dtype, pin_memory=True),
                score=torch.empty(d.score.shape, dtype=d.score.dtype, pin_memory=True),
                stats=torch.empty(d.stats.shape, dtype=d.stats.dtype, pin_memory=True))
    st_h = sk.init_state(cfg)
    hws = sk.workspace(st_h, [hs], host=True)
    for _ in range(2):   # the second call reuses the staging buffers of the first
        sk.reset_seq(st_h, 0)
        sk.step_host(st_h, [hs], hws)
        torch.cuda.synchronize()
        sk.check_device_error(st_h)
        np.testing.assert_allclose(hs.S.numpy(), d.S.cpu().numpy(), rtol=1e-5, atol=0)
        score_d = d.score.cpu().numpy()
        np.testing.assert_allclose(hs.score.numpy(), score_d, rtol=1e-5, atol=1e-7 * score_d.max())
        np.testing.assert_allclose(hs.stats.numpy(), d.stats.cpu().numpy(), rtol=1e-4, atol=1e-6)
        lp = si.L - wl.window
        for layer in range(wl.n_layers):
            got, ref = hs.idx[layer].numpy(), d.idx[layer].cpu().numpy()
            kth = np.sort(score_d[layer])[::-1][si.budget - 1]
            diff = np.setxor1d(got, ref)
            assert all(abs(score_d[layer][t] - kth) <= 1e-5 * kth for t in diff), layer
            rows = torch.cat([torch.from_numpy(got).long(), torch.arange(lp, si.L)])
            assert torch.equal(hs.k_out[layer], si.k[layer].index_select(1, rows)), layer
            assert torch.equal(hs.v_out[layer], si.v[layer].index_select(1, rows)), layer


def test_host_buffer_step_per_head_with_per_group_metadata():
    """Per-KV-head mode through starkv_step_host with one metadata row per group
    shared by every layer ([G][L], meta_layer_stride = 0, meta_group_stride = L),
    against starkv_step on device buffers with [n_layers][G][L] metadata."""
    wl = syn.WORKLOADS["uitars_5shot_28l"]
    si = syn.make_sequence(wl)
    G = wl.n_kv_heads
    si.layout = [[lay] * G for lay in si.layout]
    h = H.hyper(n_warmup=0, n_ramp=0)
    cfg = H.gpu_config(wl, h, per_head=True)
    st_d = sk.init_state(cfg)
    ds = H.device_seq(si, wl, per_head=True)
    sk.step(st_d, [ds.seq], sk.workspace(st_d, [ds.seq]))
    torch.cuda.synchronize()
    sk.check_device_error(st_d)

    d = ds.seq
    meta0 = d.meta.cpu().reshape(wl.n_layers, G, d.L)[0]
    hs = sk.Seq(k=_host(d.k.cpu(), True), v=_host(d.v.cpu(), True), q=_host(d.q.cpu(), True),
                meta=_host(meta0, True), meta_layer_stride=0, meta_group_stride=d.L, L=d.L,
                cur_frame=d.cur_frame, budget=d.budget, slot=0,
                k_out=torch.empty(d.k_out.shape, dtype=d.k_out.dtype, pin_memory=True),
                v_out=torch.empty(d.v_out.shape, dtype=d.v_out.dtype, pin_memory=True),
                meta_out=torch.empty(d.meta_out.shape, dtype=d.meta_out.dtype, pin_memory=True),
                idx=torch.empty(d.idx.shape, dtype=d.idx.dtype, pin_memory=True),
                score=torch.empty(d.score.shape, dtype=d.score.dtype, pin_memory=True),
                stats=torch.empty(d.stats.shape, dtype=d.stats.dtype, pin_memory=True))
    st_h = sk.init_state(cfg)
    sk.step_host(st_h, [hs], sk.workspace(st_h, [hs], host=True))
    torch.cuda.synchronize()
    sk.check_device_error(st_h)
    score_d = d.score.cpu().numpy()
    np.testing.assert_allclose(hs.score.numpy(), score_d, rtol=1e-5, atol=1e-7 * score_d.max())
    np.testing.assert_allclose(hs.stats.numpy(), d.stats.cpu().numpy(), rtol=1e-4, atol=1e-6)
    lp = si.L - wl.window
    words = meta0.numpy().view(np.uint32)
    for layer in range(wl.n_layers):
        for g in range(G):
            got, ref = hs.idx[layer][g].numpy(), d.idx[layer][g].cpu().numpy()
            kth = np.sort(score_d[layer][g])[::-1][si.budget - 1]
            diff = np.setxor1d(got, ref)
            assert all(abs(score_d[layer][g][t] - kth) <= 1e-5 * kth for t in diff), (layer, g)
            rows = torch.cat([torch.from_numpy(got).long(), torch.arange(lp, si.L)])
            assert torch.equal(hs.k_out[layer][g], si.k[layer][g].index_select(0, rows)), (layer, g)
            assert torch.equal(hs.v_out[layer][g], si.v[layer][g].index_select(0, rows)), (layer, g)
            assert np.array_equal(hs.meta_out[layer][g].numpy().view(np.uint32), words[g][rows.numpy()])
