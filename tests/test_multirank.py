"""Host logic of the multi-GPU benchmark path, on CPU with gloo and two ranks:
each rank draws its own trajectories, the job time is the slowest rank's, the
whole-job throughput counts every rank's tokens, and only rank 0 reports.
(The data path shards into independent (sequence, layer) units: there is no
collective besides the timing reduction.)"""
import json
import os
import subprocess
import sys

import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    w, r, _ = bench.rank_env()
    ms = 10.0 + 5.0 * r                      # rank 1 is the slow one
    ms_max = bench.max_over_ranks(ms, dist, "cpu")
    seeds = bench.rank_seeds(r, 3)
    gathered = [None] * world
    dist.all_gather_object(gathered, seeds)
    out[r] = (w, ms_max, bench.job_throughput(1000, w, 4, ms_max), gathered)
    dist.destroy_process_group()


def _free_port():
    import socket
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_two_gloo_ranks_reduce_the_job_time_and_draw_distinct_inputs():
    world = 2
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(world, _free_port(), out), nprocs=world, join=True)
        res = dict(out)
    for r in range(world):
        w, ms_max, thr, seeds = res[r]
        assert w == world
        assert ms_max == 15.0                          # max over ranks, seen by every rank
        assert abs(thr - 1000 * 2 * 4 / 0.015) < 1e-6  # all ranks' tokens over the slowest time
        flat = [s for per in seeds for s in per]
        assert len(set(flat)) == len(flat)             # weak scaling: independent trajectories


def test_reference_arm_prints_on_rank_zero_only():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "0"], env=env, capture_output=True, text=True,
                       timeout=120)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == ""


def test_reference_arm_line_keeps_the_contract():
    """The reference arm (the fp64 oracle on the host cores) on the tiny
    workload: one JSON line with the contract's keys, the metric's unit and
    direction, a cpu_baseline describing the run and an e2e object that moves
    no bytes over the host link."""
    env = dict(os.environ)
    for v in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        env.pop(v, None)
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny",
                        "--steps", "1", "--warmup", "0"], env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["impl"] == "reference" and d["unit"] == "tokens/s" and d["higher_is_better"] is True
    assert d["value"] > 0 and d["ms_per_step"] > 0 and d["steps"] == 1
    assert d["config"]["workload"] == "tiny"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_recorded_traffic_follows_the_kernel_code_not_its_comments():
    """The DRAM bytes a committed ncu capture recorded are reported only for
    the code they were measured on: the key ignores comments and layout, and
    changes with any code token."""
    a = "int f(int x) {\n  return x + 1;  // one more\n}\n/* note */\n"
    b = "int f(int x) {   return x + 1; }\n// another note\n"
    c = "int f(int x) {\n  return x + 2;\n}\n"
    assert bench.code_only(a) == bench.code_only(b) != bench.code_only(c)
    assert bench.code_only('s = "a // b"; // tail') == 's = "a // b";'
    tree = {f: open(os.path.join(ROOT, "paper_2606_01790_gb300", "csrc", f)).read()
            for f in ("score.cu", "ptx.cuh", "common.cuh")}
    edited = dict(tree, **{"score.cu": "// a new comment line\n" + tree["score.cu"]})
    changed = dict(tree, **{"score.cu": tree["score.cu"] + "\nstatic int extra_symbol;\n"})
    h = bench.kernel_src_hash("score_lse", tree.__getitem__)
    assert bench.kernel_src_hash("score_lse", edited.__getitem__) == h
    assert bench.kernel_src_hash("score_lse", changed.__getitem__) != h


def test_algorithmic_bytes_match_the_tensors_of_the_step():
    """The roofline's algorithmic bytes for the 28-layer 5-screenshot step,
    rebuilt from the byte sizes of the tensors the step must touch once (torch
    meta tensors with the ABI's layouts): the past keys and the window queries
    read, the group score map written and read, and every kept K/V row and
    metadata word read and written."""
    from paper_2606_01790_gb300 import synthetic as syn
    wl = syn.WORKLOADS["uitars_5shot_28l"]
    lay = syn.token_layout(wl.n_shots, wl.n_text, wl.grid_rows, wl.grid_cols, wl.window)
    L, nl, G, H, w, d = lay.L, wl.n_layers, wl.n_kv_heads, wl.n_heads, wl.window, wl.head_dim
    B = syn.budget(wl.budget_pct, wl.n_shots * wl.visual_per_shot, L - w)
    meta = dict(device="meta")
    nbytes = lambda t: t.numel() * t.element_size()
    k_past = torch.empty((nl, G, L - w, d), dtype=torch.bfloat16, **meta)
    q = torch.empty((nl, H, w, d), dtype=torch.bfloat16, **meta)
    S = torch.empty((nl, G, L - w), dtype=torch.float32, **meta)
    kv_out = torch.empty((2, nl, G, B + w, d), dtype=torch.bfloat16, **meta)
    meta_out = torch.empty((nl, B + w), dtype=torch.int32, **meta)
    want = nbytes(k_past) + nbytes(q) + 2 * nbytes(S) + 2 * nbytes(kv_out) + 2 * nbytes(meta_out)
    work = bench.work_per_step(wl, [dict(L=L, B=B)])
    assert work["step_bytes"] == want
    assert work["qk_flops"] == 2 * H * w * d * nl * (L - w)
    peaks = dict(hbm=6698.5, tc=1903.3, tc_sus=1721.9)
    assert bench.kernel_work("score_lse", work, peaks)[0] == "hbm"   # 224 flop/B, below the ridge
